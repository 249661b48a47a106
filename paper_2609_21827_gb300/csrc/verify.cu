// verify.cu -- RheoVerification (Algorithm 1) applied layer by layer (Theorem 1).
//
// verify_stream_kernel, grid (chunks, B*(N+1)): each CTA streams one chunk of
// one target row, producing the chunk's (max, sum exp((l - max) / T)), and
// picks out of its chunk the logits of the row's surviving children and, when
// the row's sampled child survived, of the tail support that child was drawn
// from.  The last CTA of a request walks the tree from the root with
// Algorithm 1 and leaves a residual descriptor for the stopping node.
//
// residual_kernel, grid (chunks, B): the final draw u* ~ r over V minus the
// candidate set by Gumbel-max over the stopping row; chunk maxima meet through
// 64-bit atomicMax and the last CTA of a request writes the bonus token.
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {

namespace {

struct WalkSmem {
    float rhat[kMaxSupport];
    int32_t tid[kMaxSupport];
    int32_t cpos[kMaxSupport];
};

// log sum_v exp(l_v / T) of one row from its chunk partials (warp-wide, fp64)
__device__ __forceinline__ double row_lse(const VerifyArgs& a, int64_t rowg, float T) {
    const int lane = threadIdx.x & 31;
    const int C = a.n.chunks;
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, __ldcg(a.row_mu + rowg * C + c));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    double t = 0.0;
    for (int c = lane; c < C; c += 32) {
        const double sc = __ldcg(a.row_sum + rowg * C + c);
        if (sc != 0.0) t += sc * exp(((double)__ldcg(a.row_mu + rowg * C + c) - (double)m) / (double)T);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
    return (double)m / (double)T + log(t);
}

// expansion index of the parent of child gen id g, clamped into [0, E)
__device__ __forceinline__ int64_t expansion_of_child(int K, int64_t g, int64_t G1, int64_t E) {
    g = min(max(g, (int64_t)1), G1 - 1);
    return min(parent_expansion_of(K, g), E - 1);
}

// a pruned row's child range lies inside the pruned tree
__device__ __forceinline__ bool pruned_row_ok(int nc, int fc, int sc, int K, int N) {
    if (nc < 0 || nc > K + 1) return false;
    if (nc > 0 && (fc < 1 || fc + nc > N + 1)) return false;
    if (sc != -1 && (nc == 0 || sc < fc || sc >= fc + nc)) return false;
    return true;
}

__device__ __forceinline__ float p_of(float l, float T, double lse) {
    return (float)exp((double)l / (double)T - lse);
}

}  // namespace

template <int DT, bool ALIGNED>
__global__ void __launch_bounds__(kThreads) verify_stream_kernel(const VerifyArgs a) {
    using E = Elem<DT>;
    constexpr int VEC = E::VEC;
    constexpr int CH = E::CHUNK;
    __shared__ BlockScratch bs;
    __shared__ WalkSmem ws;

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const int64_t r = blockIdx.y;
    const int NP = n.N + 1;
    const int b = (int)(r / NP);
    const int V = n.V, K = n.K, TL = n.TL;
    const char* row = a.logits + r * a.row_stride_bytes;
    const int64_t e_lo = (int64_t)k * CH;
    const float T = a.T[b];

    // ---- stream: (max, sum exp((l - max)/T)) of the chunk ---------------------
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
        const float c = 1.4426950408889634f / T;
        const float mc = mu * c;
#pragma unroll
        for (int j = 0; j < kNV; ++j)
#pragma unroll
            for (int i = 0; i < VEC; ++i) s += fast_exp2(fmaf(E::value(E::raw(v[j], i)), c, -mc));
    }
    float Mc;
    double Sc;
    block_max_sum(mu, (double)s, bs, Mc, Sc);
    if (tid == 0) {
        a.row_mu[r * n.chunks + k] = Mc;
        a.row_sum[r * n.chunks + k] = Sc;
        if (isnan(Sc) || Mc == INFINITY) atomicOr(a.status, kStBadLogit);
        if (k == 0 && (!(T > 0.0f) || isinf(T))) atomicOr(a.status, kStBadTemperature);
    }

    // ---- gathers: children tokens and, if the sampled child survived, its tail
    {
        int nc = a.pr.n_child[r], fc = a.pr.first_child[r], sc = a.pr.sampled_child[r];
        if (!pruned_row_ok(nc, fc, sc, K, n.N)) nc = 0, sc = -1;
        const int32_t* tids = nullptr;
        if (sc >= 0) {
            const int64_t e = expansion_of_child(K, a.pr.gen_id[(int64_t)b * NP + sc], n.G1, n.E);
            tids = a.tree.tail_ids + ((int64_t)b * n.E + e) * TL;
        }
        for (int i = tid; i < n.GW; i += kThreads) {
            int tok = -1;
            if (i < nc) tok = a.pr.token[(int64_t)b * NP + fc + i];
            else if (i > K && tids) tok = tids[i - (K + 1)];
            if (tok >= 0 && tok >= e_lo && tok < e_lo + CH && tok < V)
                a.gather[r * n.GW + i] = E::value(E::load_scalar(row, tok));
        }
    }

    // ---- last CTA of the request: Algorithm 1 from the root --------------------
    if (!arrive_last(a.req_ticket + b, (unsigned)(n.chunks * NP), bs)) return;

    if (a.row_lse) {
        // every row's log-partition (reported for parity checks)
        for (int u = tid >> 5; u < NP; u += kWarps) {
            const double l = row_lse(a, (int64_t)b * NP + u, T);
            if ((tid & 31) == 0) a.row_lse[(int64_t)b * NP + u] = (float)l;
        }
    }
    if (tid >= 32) return;
    const int lane = tid;
    const uint64_t seed = a.seed[b], off = a.offset[b];
    const int64_t pb = (int64_t)b * NP, nb = (int64_t)b * n.G1;
    int u = 0, len = 0;
    for (;;) {
        const int64_t rowg = pb + u;
        const double lse = row_lse(a, rowg, T);
        if (!(lse > -INFINITY) && lane == 0) atomicOr(a.status, kStEmptyRow);
        int nc = a.pr.n_child[rowg], fc = a.pr.first_child[rowg], sc = a.pr.sampled_child[rowg];
        if (!pruned_row_ok(nc, fc, sc, K, n.N) || (nc > 0 && len >= n.D)) {
            if (lane == 0) atomicOr(a.status, kStInternal);
            nc = 0, sc = -1;
        }
        const int gen_u = a.pr.gen_id[rowg];
        const float* gth = a.gather + rowg * n.GW;
        double M = 1.0;
        int use_tail = 0, e = 0, acc = -1;
        if (nc > 0 && sc >= 0) {
            // stochastic first: accept u_s with probability min(1, p / q~)
            const int64_t gs = min(max((int64_t)a.pr.gen_id[pb + sc], (int64_t)1), n.G1 - 1);
            const float eta0 = uniform(seed, off, kTagVerify, gen_u, 0);
            const float qv = a.tree.qtilde[nb + gs];
            const float pv = p_of(__ldcg(gth + (sc - fc)), T, lse);
            if (__fmul_rn(eta0, qv) <= pv) {
                acc = sc;
            } else {
                // r = norm(max(0, p - q~)): unnormalised r^ with mass M
                e = (int)expansion_of_child(K, gs, n.G1, n.E);
                const int64_t t0 = ((int64_t)b * n.E + e) * TL;
                double ov = 0.0;
                for (int i = lane; i < TL; i += 32) {
                    const float pt = p_of(__ldcg(gth + K + 1 + i), T, lse);
                    const float qi = a.tree.tail_q[t0 + i];
                    const float d = __fsub_rn(pt, qi);
                    ws.rhat[i] = d > 0.0f ? d : 0.0f;
                    ws.tid[i] = a.tree.tail_ids[t0 + i];
                    ov += (double)fminf(pt, qi);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) ov += __shfl_xor_sync(0xFFFFFFFFu, ov, o);
                M = 1.0 - ov;
                use_tail = 1;
                __syncwarp();
                for (int c = 0; c < nc; ++c) {
                    const int tok = a.pr.token[pb + fc + c];
                    int pos = -1;
                    for (int i = lane; i < TL; i += 32)
                        if (ws.tid[i] == tok) pos = i;
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) pos = max(pos, __shfl_xor_sync(0xFFFFFFFFu, pos, o));
                    if (lane == 0) ws.cpos[c] = pos;
                }
                __syncwarp();
            }
        }
        if (acc < 0 && nc > 0) {
            // recursive rejection over the remaining candidates, in slot order
            for (int c = 0; c < nc; ++c) {
                const int vv = fc + c;
                if (vv == sc) continue;
                const int gv = a.pr.gen_id[pb + vv];
                const float eta = uniform(seed, off, kTagVerify, gen_u, (uint64_t)(1 + slot_of(K, gv)));
                const int cp = use_tail ? ws.cpos[c] : -1;
                const float rv = (cp >= 0) ? ws.rhat[cp] : p_of(__ldcg(gth + c), T, lse);
                if ((double)eta * M <= (double)rv) {
                    acc = vv;
                    break;
                }
                M -= (double)rv;
                __syncwarp();
                if (cp >= 0 && lane == 0) ws.rhat[cp] = 0.0f;
                __syncwarp();
            }
        }
        if (acc >= 0) {
            if (lane == 0) {
                a.accepted_tokens[(int64_t)b * n.D + len] = a.pr.token[pb + acc];
                a.accepted_nodes[(int64_t)b * n.D + len] = acc;
            }
            ++len;
            u = acc;
            continue;
        }
        // stop here: describe the residual for the final draw
        if (lane == 0) {
            int32_t* d = a.desc + (int64_t)b * 8;
            d[0] = u;
            d[1] = gen_u;
            d[2] = __float_as_int((float)lse);
            d[3] = use_tail;
            d[4] = nc;
            d[5] = e;
            d[6] = __float_as_int((float)M);
            d[7] = 0;
            for (int c = 0; c < 3; ++c) a.res_best[(int64_t)b * 3 + c] = 0ull;
        }
        for (int c = lane; c < nc; c += 32) a.excl[(int64_t)b * (K + 1) + c] = a.pr.token[pb + fc + c];
        if (use_tail)
            for (int i = lane; i < TL; i += 32) a.rhat[(int64_t)b * TL + i] = ws.rhat[i];
        break;
    }
    if (lane == 0) a.accepted_len[b] = len;
    for (int i = len + lane; i < n.D; i += 32) {
        a.accepted_tokens[(int64_t)b * n.D + i] = -1;
        a.accepted_nodes[(int64_t)b * n.D + i] = -1;
    }
}

template <int DT, bool ALIGNED>
__global__ void __launch_bounds__(kThreads) residual_kernel(const VerifyArgs a) {
    using E = Elem<DT>;
    constexpr int VEC = E::VEC;
    constexpr int CH = E::CHUNK;
    __shared__ BlockScratch bs;
    __shared__ uint32_t excl_bits[CH / 32];
    __shared__ uint32_t tail_bits[CH / 32];

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const int b = blockIdx.y;
    const int V = n.V, K = n.K, TL = n.TL, NP = n.N + 1;
    const int32_t* d = a.desc + (int64_t)b * 8;
    // descriptor written by the walk; clamped so that a stale one cannot index out of range
    const int u = min(max(d[0], 0), n.N), gen_u = d[1], use_tail = d[3];
    const int nexcl = min(max(d[4], 0), K + 1);
    const int e = (int)min(max((int64_t)d[5], (int64_t)0), n.E - 1);
    const float lse = __int_as_float(d[2]);
    const float T = a.T[b];
    const uint64_t seed = a.seed[b], off = a.offset[b];
    const char* row = a.logits + ((int64_t)b * NP + u) * a.row_stride_bytes;
    const int64_t e_lo = (int64_t)k * CH;
    const int32_t* tids = a.tree.tail_ids + ((int64_t)b * n.E + e) * TL;

    for (int i = tid; i < CH / 32; i += kThreads) { excl_bits[i] = 0u; tail_bits[i] = 0u; }
    __syncthreads();
    for (int c = tid; c < nexcl; c += kThreads) {
        const int tok = a.excl[(int64_t)b * (K + 1) + c];
        if (tok >= e_lo && tok < e_lo + CH) atomicOr(&excl_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
    }
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = tids[i];
            if (tok >= e_lo && tok < e_lo + CH) atomicOr(&tail_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
        }
    __syncthreads();

    // keys: 0 -> r^ over V minus the candidates; 1 -> p over V minus the
    // candidates; 2 -> p over V (1 and 2 only matter after rounding dead ends)
    unsigned long long best[3] = {0ull, 0ull, 0ull};
    auto offer = [&](int w, float key, int64_t id) {
        if (key > -INFINITY) {
            const unsigned long long pk = ((unsigned long long)ord_f32(key) << 32) | (0xFFFFFFFFu - (uint32_t)id);
            best[w] = pk > best[w] ? pk : best[w];
        }
    };
#pragma unroll 1
    for (int j = 0; j < kNV; ++j) {
        const int64_t e0 = e_lo + (int64_t)(j * kThreads + tid) * VEC;
        if (e0 >= V) break;
        const uint4 raw = load_vec<DT, ALIGNED>(row, e0, V);
        uint4 rnd[VEC / 4];
#pragma unroll
        for (int q = 0; q < VEC / 4; ++q) rnd[q] = philox_block(seed, off, kTagResidual, gen_u, (uint64_t)(e0 >> 2) + q);
#pragma unroll
        for (int i = 0; i < VEC; ++i) {
            const int64_t id = e0 + i;
            if (id >= V) break;
            const float x = E::value(E::raw(raw, i));
            const float g = gumbel(u01(word_of(rnd[i >> 2], i & 3)));
            const float tv = __fdiv_rn(x, T);
            const float fb = __fadd_rn(tv, g);
            offer(2, fb, id);
            const int li = (int)(id - e_lo);
            const bool ex = (excl_bits[li >> 5] >> (li & 31)) & 1u;
            if (ex) continue;
            offer(1, fb, id);
            const bool tl = (tail_bits[li >> 5] >> (li & 31)) & 1u;
            if (!tl) offer(0, __fadd_rn(__fsub_rn(tv, lse), g), id);
        }
    }
    // tail entries use log r^ (zero mass after a rejection: no key)
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = tids[i];
            if (tok < e_lo || tok >= e_lo + CH) continue;
            const int li = tok - (int)e_lo;
            if ((excl_bits[li >> 5] >> (li & 31)) & 1u) continue;
            const float rv = a.rhat[(int64_t)b * TL + i];
            if (!(rv > 0.0f)) continue;
            const float g = gumbel(uniform(seed, off, kTagResidual, gen_u, (uint64_t)tok));
            offer(0, __fadd_rn(logf(rv), g), tok);
        }
    for (int w = 0; w < 3; ++w) {
        const unsigned long long m = block_max_u64(best[w], bs);
        if (tid == 0 && m) atomicMax(a.res_best + (int64_t)b * 3 + w, m);
    }
    if (!arrive_last(a.res_ticket + b, (unsigned)n.chunks, bs)) return;
    if (tid == 0) {
        unsigned long long m = __ldcg(a.res_best + (int64_t)b * 3 + 0);
        if (!m) m = __ldcg(a.res_best + (int64_t)b * 3 + 1);
        if (!m) m = __ldcg(a.res_best + (int64_t)b * 3 + 2);
        a.bonus_token[b] = m ? (int32_t)(0xFFFFFFFFu - (uint32_t)m) : -1;
        if (!m) atomicOr(a.status, kStEmptyRow);
    }
}

cudaError_t launch_verify(const VerifyArgs& a, int dtype, bool aligned, dim3 g1, dim3 g2, cudaStream_t s) {
    if (dtype == 1) {
        if (aligned) {
            verify_stream_kernel<1, true><<<g1, kThreads, 0, s>>>(a);
            residual_kernel<1, true><<<g2, kThreads, 0, s>>>(a);
        } else {
            verify_stream_kernel<1, false><<<g1, kThreads, 0, s>>>(a);
            residual_kernel<1, false><<<g2, kThreads, 0, s>>>(a);
        }
    } else {
        if (aligned) {
            verify_stream_kernel<0, true><<<g1, kThreads, 0, s>>>(a);
            residual_kernel<0, true><<<g2, kThreads, 0, s>>>(a);
        } else {
            verify_stream_kernel<0, false><<<g1, kThreads, 0, s>>>(a);
            residual_kernel<0, false><<<g2, kThreads, 0, s>>>(a);
        }
    }
    return cudaGetLastError();
}

}  // namespace rheo
