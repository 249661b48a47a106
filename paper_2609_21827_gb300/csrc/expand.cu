// expand.cu -- one expansion call of the draft tree (Sec. 2.1, Sec. 3.2, App. C.1).
//
// Grid (chunks, B*F).  Each CTA streams one 32 KiB chunk of one draft row into
// registers and produces
//   * the chunk's (max, sum exp(l - max)) at T = 1 (untempered, Sec. 5.4),
//   * the chunk's exact top-S keys under (logit desc, id asc).
// The last CTA of a row (arrival counter, no waiting) merges the chunk lists
// into the row's sorted support, draws Y from the tempered tail by Gumbel-max
// and writes the K+1 children with their proxies and path scores.  The last
// row of a request selects the next frontier.
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {

namespace {

struct E2Smem {
    unsigned long long sel[kMaxSupport];
    unsigned long long sorted[kMaxSupport];
    int32_t id[kMaxSupport];
    float l[kMaxSupport];
    float lq0[kMaxSupport];
    float q[kMaxSupport];
    float lp;
    int sel_count;
    int best;
    float lse1;
    int bad;
};

}  // namespace

template <int DT, bool ALIGNED>
__global__ void __launch_bounds__(kThreads) expand_kernel(const ExpandArgs a) {
    using E = Elem<DT>;
    constexpr int VEC = E::VEC;
    constexpr int CH = E::CHUNK;
    extern __shared__ unsigned long long keys[];
    __shared__ BlockScratch bs;
    __shared__ E2Smem e2;
    __shared__ int s_count;

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const int r = blockIdx.y;
    const int b = r / a.F, f = r % a.F;
    const int V = n.V, S = n.S;
    const char* row = a.logits + (int64_t)r * a.row_stride_bytes;
    const int64_t e_lo = (int64_t)k * CH;
    int parity = 0;

    // ---- stream the chunk ----------------------------------------------------
    uint4 v[kNV];
#pragma unroll
    for (int j = 0; j < kNV; ++j) v[j] = load_vec<DT, ALIGNED>(row, e_lo + (int64_t)(j * kThreads + tid) * VEC, V);

    float mu = -INFINITY;
#pragma unroll
    for (int j = 0; j < kNV; ++j)
#pragma unroll
        for (int i = 0; i < VEC; ++i) mu = fmaxf(mu, E::value(E::raw(v[j], i)));
    float s = 0.0f;
    if (mu != -INFINITY) {
        const float c = 1.4426950408889634f;
        const float mc = mu * c;
#pragma unroll
        for (int j = 0; j < kNV; ++j)
#pragma unroll
            for (int i = 0; i < VEC; ++i) s += fast_exp2(fmaf(E::value(E::raw(v[j], i)), c, -mc));
    }
    float Mc;
    double Sc;
    block_max_sum(mu, (double)s, bs, Mc, Sc);
    const int64_t ck = (int64_t)r * n.chunks + k;
    if (tid == 0) {
        a.chunk_mu[ck] = Mc;
        a.chunk_sum[ck] = Sc;
        if (isnan(Sc) || Mc == INFINITY) atomicOr(a.status, kStBadLogit);
    }

    // ---- exact top-S of the chunk --------------------------------------------
    const int n_valid = (int)min((int64_t)CH, (int64_t)V - e_lo);
    const int target = min(S, n_valid);
    const bool have = e_lo + (int64_t)tid * VEC < V;
    const uint32_t kmax = have ? E::key(DT == 0 ? __float_as_uint(mu) : (__float_as_uint(mu) >> 16)) : 0u;
    const int n_thr = (int)min((int64_t)kThreads, ((int64_t)n_valid + VEC - 1) / VEC);

    // lower bound L on the chunk's S-th key: the S-th largest thread maximum
    uint32_t L = 0;
    if (n_valid > S && n_thr >= S) {
        const unsigned long long mk = have ? ((unsigned long long)kmax << 32) : 0ull;
        const unsigned long long aand = block_and_or_u64(have ? mk : ~0ull, false, bs);
        const unsigned long long aor = block_and_or_u64(mk, true, bs);
        const unsigned long long t = block_select(
            [&](unsigned long long x) { return (have && mk >= x) ? 1 : 0; }, S, aand, aor, bs, parity);
        L = (uint32_t)(t >> 32);
    }

    if (tid == 0) s_count = 0;
    __syncthreads();
    if (have && kmax >= L) {
#pragma unroll
        for (int j = 0; j < kNV; ++j)
#pragma unroll
            for (int i = 0; i < VEC; ++i) {
                const int64_t e = e_lo + (int64_t)(j * kThreads + tid) * VEC + i;
                const uint32_t kk = E::key(E::raw(v[j], i));
                if (e < V && kk >= L) {
                    const int pos = atomicAdd(&s_count, 1);
                    if (pos < kCandCap) keys[pos] = ((unsigned long long)kk << 32) | (0xFFFFFFFFu - (uint32_t)e);
                }
            }
    }
    __syncthreads();
    const int ncand = s_count;
    const bool overflow = ncand > kCandCap;
    unsigned long long thr = 1ull;
    if (ncand > target) {
        if (!overflow) {
            unsigned long long aand = ~0ull, aor = 0ull;
            for (int i = tid; i < ncand; i += kThreads) { aand &= keys[i]; aor |= keys[i]; }
            aand = block_and_or_u64(aand, false, bs);
            aor = block_and_or_u64(aor, true, bs);
            thr = block_select(
                [&](unsigned long long x) {
                    int c = 0;
                    for (int i = tid; i < ncand; i += kThreads) c += keys[i] >= x;
                    return c;
                },
                target, aand, aor, bs, parity);
        } else {
            // many ties at the boundary: select directly over the registers
            auto key_at = [&](int j, int i, int64_t& e) -> unsigned long long {
                e = e_lo + (int64_t)(j * kThreads + tid) * VEC + i;
                return ((unsigned long long)E::key(E::raw(v[j], i)) << 32) | (0xFFFFFFFFu - (uint32_t)e);
            };
            unsigned long long aand = ~0ull, aor = 0ull;
#pragma unroll
            for (int j = 0; j < kNV; ++j)
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    int64_t e;
                    const unsigned long long x = key_at(j, i, e);
                    if (e < V) { aand &= x; aor |= x; }
                }
            aand = block_and_or_u64(aand, false, bs);
            aor = block_and_or_u64(aor, true, bs);
            thr = block_select(
                [&](unsigned long long t) {
                    int c = 0;
#pragma unroll
                    for (int j = 0; j < kNV; ++j)
#pragma unroll
                        for (int i = 0; i < VEC; ++i) {
                            int64_t e;
                            const unsigned long long x = key_at(j, i, e);
                            c += (e < V && x >= t);
                        }
                    return c;
                },
                target, aand, aor, bs, parity);
        }
    }
    // write the chunk list (unsorted), padded with 0 keys
    unsigned long long* out = a.chunk_keys + ck * S;
    __syncthreads();
    if (tid == 0) s_count = 0;
    __syncthreads();
    if (!overflow) {
        for (int i = tid; i < ncand; i += kThreads) {
            const unsigned long long x = keys[i];
            if (x >= thr) {
                const int pos = atomicAdd(&s_count, 1);
                if (pos < S) out[pos] = x;
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < kNV; ++j)
#pragma unroll
            for (int i = 0; i < VEC; ++i) {
                const int64_t e = e_lo + (int64_t)(j * kThreads + tid) * VEC + i;
                const unsigned long long x =
                    ((unsigned long long)E::key(E::raw(v[j], i)) << 32) | (0xFFFFFFFFu - (uint32_t)e);
                if (e < V && x >= thr) {
                    const int pos = atomicAdd(&s_count, 1);
                    if (pos < S) out[pos] = x;
                }
            }
    }
    __syncthreads();
    const int written = s_count;
    if (tid == 0 && written != target) atomicOr(a.status, kStInternal);
    for (int i = written + tid; i < S; i += kThreads) out[i] = 0ull;

    // ---- last CTA of the row: support, tail sample, pool ----------------------
    if (!arrive_last(a.row_ticket + r, (unsigned)n.chunks, bs)) return;

    const int nkeys = n.chunks * S;
    const unsigned long long* rk = a.chunk_keys + (int64_t)r * n.chunks * S;
    for (int i = tid; i < nkeys; i += kThreads) keys[i] = __ldcg(rk + i);
    if (tid == 0) e2.sel_count = 0;
    __syncthreads();
    {
        unsigned long long aand = ~0ull, aor = 0ull;
        int nz = 0;
        for (int i = tid; i < nkeys; i += kThreads) {
            const unsigned long long x = keys[i];
            if (x) { aand &= x; aor |= x; ++nz; }
        }
        nz = block_sum_int(nz, bs, parity);
        aand = block_and_or_u64(aand, false, bs);
        aor = block_and_or_u64(aor, true, bs);
        unsigned long long rthr = 1ull;
        if (nz > S)
            rthr = block_select(
                [&](unsigned long long x) {
                    int c = 0;
                    for (int i = tid; i < nkeys; i += kThreads) c += keys[i] >= x;
                    return c;
                },
                S, aand, aor, bs, parity);
        for (int i = tid; i < nkeys; i += kThreads) {
            const unsigned long long x = keys[i];
            if (x && x >= rthr) {
                const int pos = atomicAdd(&e2.sel_count, 1);
                if (pos < S) e2.sel[pos] = x;
            }
        }
    }
    __syncthreads();
    if (tid < S) {
        const unsigned long long x = e2.sel[tid];
        int rank = 0;
        for (int j = 0; j < S; ++j) rank += e2.sel[j] > x;
        e2.sorted[rank] = x;
    }
    // log-partition of the whole row (fp64 merge of the chunk partials)
    if (tid < 32) {
        float m = -INFINITY;
        for (int c = tid; c < n.chunks; c += 32) m = fmaxf(m, __ldcg(a.chunk_mu + (int64_t)r * n.chunks + c));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
        double t = 0.0;
        for (int c = tid; c < n.chunks; c += 32) {
            const double sc = __ldcg(a.chunk_sum + (int64_t)r * n.chunks + c);
            if (sc != 0.0) t += sc * exp((double)__ldcg(a.chunk_mu + (int64_t)r * n.chunks + c) - (double)m);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
        if (tid == 0) {
            e2.lse1 = (float)((double)m + log(t));
            e2.bad = (e2.sel_count != S) ? 1 : 0;
        }
    }
    __syncthreads();
    const float lse1 = e2.lse1;
    if (tid < S) {
        const unsigned long long x = e2.sorted[tid];
        e2.id[tid] = (int32_t)(0xFFFFFFFFu - (uint32_t)x);
        const float l = E::value_of_key((uint32_t)(x >> 32));
        e2.l[tid] = l;
        e2.lq0[tid] = __fsub_rn(l, lse1);
    }
    __syncthreads();

    const int m = n.m, K = n.K, TL = n.TL;
    const float T = a.T[b];
    const uint64_t seed = a.seed[b], off = a.offset[b];
    const int64_t nb = (int64_t)b * n.G1;
    int64_t par = (a.d == 1) ? 0 : (int64_t)a.tree.frontier[(int64_t)b * K + f];
    if (par < 0 || par >= n.G1) {  // frontier never written for this tree
        if (tid == 0) atomicOr(a.status, kStInternal);
        par = 0;
    }
    const int64_t eidx = (a.d == 1) ? 0 : 1 + (int64_t)(a.d - 2) * K + f;
    const int64_t g0 = depth_base(K, a.d) + (int64_t)f * (K + 1);

    // tempered tail q~ = softmax(l / T) over support ranks m+1..S; Y by Gumbel-max
    const float tau = (tid < TL) ? __fdiv_rn(e2.l[m + tid], T) : -INFINITY;
    float mt;
    double st;
    block_max_sum(tau, (tid < TL) ? 1.0 : 0.0, bs, mt, st);
    const double lse_tail = (double)mt + log(st);
    unsigned long long pack = 0ull;
    if (tid < TL) {
        e2.q[tid] = (float)exp((double)tau - lse_tail);
        const float g = gumbel(uniform(seed, off, kTagSample, (int)par, (uint64_t)tid));
        const float key = __fadd_rn(tau, g);
        if (key > -INFINITY) pack = ((unsigned long long)ord_f32(key) << 32) | (0xFFFFFFFFu - (uint32_t)tid);
    }
    const unsigned long long bestp = block_max_u64(pack, bs);
    if (tid == 0) {
        e2.best = bestp ? (int)(0xFFFFFFFFu - (uint32_t)bestp) : 0;
        if (e2.bad) atomicOr(a.status, kStInternal);
        if (!bestp || !(e2.l[m] > -INFINITY)) atomicOr(a.status, kStEmptyRow);
        if (!(T > 0.0f) || isinf(T)) atomicOr(a.status, kStBadTemperature);
        // construction probability of Y (Sec. 3.2): min{q0(x_m), z}, never below q0(x_{m+1});
        // m = 0: min(1, q0(x_1) + eps)
        float lp;
        if (m >= 1) {
            double zs = 0.0;
            for (int i = 0; i < m; ++i) zs += exp((double)e2.lq0[i]);
            if (zs > 1.0) zs = 1.0;
            const float lz = (float)log1p(-zs);
            lp = fminf(e2.lq0[m - 1], lz);
            lp = fmaxf(lp, e2.lq0[m]);
        } else {
            double pr = exp((double)e2.lq0[0]) + (double)n.eps;
            if (pr > 1.0) pr = 1.0;
            lp = (float)log(pr);
        }
        e2.lp = lp;
        if (a.d == 1) {
            a.tree.token[nb] = -1;
            a.tree.parent[nb] = -1;
            a.tree.log_proxy[nb] = 0.0f;
            a.tree.score[nb] = 0.0f;
            a.tree.qtilde[nb] = 0.0f;
            a.tree.slot[nb] = kSlotRoot;
        }
    }
    __syncthreads();

    // children in slot order: leads, Y, fills (highest remaining ranks, Y skipped)
    const int best = e2.best;
    if (tid <= K) {
        const int j = tid;
        int rank;
        float lpj, qv = 0.0f;
        uint8_t st8;
        if (j < m) {
            rank = j; lpj = e2.lq0[j]; st8 = kSlotLead;
        } else if (j == m) {
            rank = m + best; lpj = e2.lp; st8 = kSlotSampled; qv = e2.q[best];
        } else {
            const int qf = j - m - 1;
            rank = m + qf + (qf >= best ? 1 : 0); lpj = e2.lq0[rank]; st8 = kSlotFill;
        }
        const float ps = (a.d == 1) ? 0.0f : a.tree.score[nb + par];
        const int64_t g = nb + g0 + j;
        a.tree.token[g] = e2.id[rank];
        a.tree.parent[g] = (int32_t)par;
        a.tree.log_proxy[g] = lpj;
        a.tree.score[g] = __fadd_rn(ps, lpj);
        a.tree.qtilde[g] = qv;
        a.tree.slot[g] = st8;
    }
    if (tid < TL) {
        const int64_t t0 = ((int64_t)b * n.E + eidx) * TL;
        a.tree.tail_ids[t0 + tid] = e2.id[m + tid];
        a.tree.tail_q[t0 + tid] = e2.q[tid];
    }
    if (tid == 0) a.tree.lse1[(int64_t)b * n.E + eidx] = lse1;

    // ---- last row of the request: the K best depth-d nodes become the frontier ----
    if (!arrive_last(a.req_ticket + b, (unsigned)a.F, bs)) return;
    if (a.d == n.D) return;
    {
        const int nn = a.F * (K + 1);
        const int64_t base = depth_base(K, a.d);
        auto key_of = [&](int i) -> unsigned long long {
            const float sc = __ldcg(a.tree.score + nb + base + i);
            return ((unsigned long long)ord_f32(sc) << 32) | (0xFFFFFFFFu - (uint32_t)(base + i));
        };
        unsigned long long aand = ~0ull, aor = 0ull;
        for (int i = tid; i < nn; i += kThreads) {
            const unsigned long long x = key_of(i);
            aand &= x;
            aor |= x;
        }
        aand = block_and_or_u64(aand, false, bs);
        aor = block_and_or_u64(aor, true, bs);
        const unsigned long long fthr = block_select(
            [&](unsigned long long t) {
                int c = 0;
                for (int i = tid; i < nn; i += kThreads) c += key_of(i) >= t;
                return c;
            },
            K, aand, aor, bs, parity);
        const int per = (nn + kThreads - 1) / kThreads;
        const int lo = min(nn, tid * per), hi = min(nn, lo + per);
        int cnt = 0;
        for (int i = lo; i < hi; ++i) cnt += key_of(i) >= fthr;
        int total;
        int pos = block_exclusive_scan(cnt, total, bs);
        for (int i = lo; i < hi; ++i)
            if (key_of(i) >= fthr) {
                if (pos < K) a.tree.frontier[(int64_t)b * K + pos] = (int32_t)(base + i);
                ++pos;
            }
        if (tid == 0 && total != K) atomicOr(a.status, kStInternal);
    }
}

cudaError_t launch_expand(const ExpandArgs& a, int dtype, bool aligned, dim3 grid, size_t smem, cudaStream_t s) {
    if (dtype == 1) {
        if (aligned) expand_kernel<1, true><<<grid, kThreads, smem, s>>>(a);
        else expand_kernel<1, false><<<grid, kThreads, smem, s>>>(a);
    } else {
        if (aligned) expand_kernel<0, true><<<grid, kThreads, smem, s>>>(a);
        else expand_kernel<0, false><<<grid, kThreads, smem, s>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace rheo
