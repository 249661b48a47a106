// verify.cu -- RheoVerification (Algorithm 1) applied layer by layer (Theorem 1).
//
// verify_stream_kernel: persistent CTAs stream the B*(N+1) target rows tile by
// tile (stream.cuh), keeping a running (max, sum exp((l - max) / T)) per
// thread over each row segment.  The CTA that ends the last segment of a row
// (arrival counter, never a wait) turns the row into its decision table:
// lse_T, p at the surviving children, and -- when the row's sampled child
// survived -- r^ = max(0, p - q~) over the tail that child was drawn from, the
// residual mass M = 1 - sum_tail min(p, q~), r^ at the children, plus the
// Philox coins of the node.  Every row is independent, so all tables are built
// in parallel while the stream is still running.
//
// residual_kernel, grid (chunks, B): each CTA stages its request's tables,
// replays the walk of Algorithm 1 from the root (a few comparisons per level),
// and takes part in the final draw u* ~ r over V minus the candidate set
// (Gumbel-max over the stopping row; chunk maxima meet through 64-bit
// atomicMax, the last CTA of the request writes the bonus token).
#include "rheo_device.cuh"
#include "rheo_kernels.h"
#include "stream.cuh"

namespace rheo {

namespace {

// decision table of one pruned row (floats):
//   0 M_hi, 1 M_lo (residual mass), 2 q~(sampled child), 3 lse_hi, 4 lse_lo,
//   5 use_tail (the sampled child survived and was rejected),
//   6 verdict: pruned index of the accepted child, -1 when the walk stops here,
//   7 .. 7+K+1        p at the children (slot order of the pruned row)
//   7+K+1 .. 7+2K+2   r^ at the children (p when the sampled child did not survive)
//   7+2K+2 .. +K+2    coins: draw 0 (sampled child), draw 1+slot (others)
// A row's verdict depends on nothing but the row itself (Algorithm 1 at one
// node), so every row gets it in parallel; the walk only follows verdicts.
constexpr int kTabP = 7;
__host__ __device__ __forceinline__ int table_width(int K) { return kTabP + 2 * (K + 1) + (K + 2); }

struct RowSmem {
    int32_t tok[kMaxSupport];    // children tokens
    int32_t cgen[kMaxSupport];   // children gen ids
    int32_t tids[kMaxSupport];   // tail ids
    float tq[kMaxSupport];       // tail q~
    float lval[2 * kMaxSupport]; // gathered logits: children, then tail
    int32_t cpos[kMaxSupport];   // tail position of each child (-1: off the tail)
    float pt[kMaxSupport];       // r^ over the tail
    float pc[kMaxSupport];       // p at the children
    float rc[kMaxSupport];       // r^ at the children
    float coin[kMaxSupport + 2]; // Philox coins of the node
    float qs;                    // q~ of the sampled child
    int nc, fc, sc, gen;
    int64_t e;
};

__device__ __forceinline__ bool pruned_row_ok(int nc, int fc, int sc, int K, int N) {
    if (nc < 0 || nc > K + 1) return false;
    if (nc > 0 && (fc < 1 || fc + nc > N + 1)) return false;
    if (sc != -1 && (nc == 0 || sc < fc || sc >= fc + nc)) return false;
    return true;
}

__device__ __forceinline__ int64_t expansion_of_child(int K, int64_t g, int64_t G1, int64_t E) {
    g = min(max(g, (int64_t)1), G1 - 1);
    return min((int64_t)parent_expansion_of(K, (int)g), E - 1);
}

// lse_T of a row from its segment partials (one warp; float-float accumulation)
__device__ __forceinline__ FF combine_lse(const float* mu, const float* sm, int nseg, float T) {
    const int lane = threadIdx.x & 31;
    float m = -INFINITY;
    for (int c = lane; c < nseg; c += 32) m = fmaxf(m, __ldcg(mu + c));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    FF t{0.0f, 0.0f};
    for (int c = lane; c < nseg; c += 32) {
        const FF sc{__ldcg(sm + 2 * c), __ldcg(sm + 2 * c + 1)};
        if (sc.hi != 0.0f) t = ff_add(t, ff_mul(expf(__fdiv_rn(__ldcg(mu + c) - m, T)), sc));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t = ff_add(t, ff_shfl_xor(t, o));
    return ff_add(ff_div(m, T), ff_log(t));  // m / T + log sum
}

}  // namespace

template <int DT, bool TMA>
__global__ void __launch_bounds__(kThreads, 2) verify_stream_kernel(const VerifyArgs a) {
    using E = Elem<DT>;
    using W = Vec<DT>;
    constexpr int VEC = E::VEC;
    constexpr int TE = kTileBytes / E::SIZE;
    constexpr int VPT = TE / VEC / kThreads;
    constexpr float kLog2e = 1.4426950408889634f;
    extern __shared__ __align__(128) unsigned char dsm[];
    unsigned char* ring = dsm;
    __shared__ __align__(8) uint64_t full[kStages];
    __shared__ BlockScratch bs;
    __shared__ RowSmem rs;

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int V = n.V, K = n.K, TL = n.TL, NP = n.N + 1;
    const int tpr = (V + TE - 1) / TE;
    const TileSplit sp{(int64_t)n.B * NP * tpr, (int)gridDim.x};
    const int64_t t0 = sp.begin(blockIdx.x), t1 = sp.begin(blockIdx.x + 1);
    const int TW = table_width(K);

    if (TMA && tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
        mbar_fence_init();
    }
    __syncthreads();
    auto issue = [&](int64_t t) {
        const int64_t r = t / tpr;
        const int64_t e0 = (t % tpr) * (int64_t)TE;
        const unsigned bytes = (unsigned)(min((int64_t)TE, (int64_t)V - e0) * E::SIZE);
        const int s = (int)((t - t0) % kStages);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_load(ring + s * kTileBytes, a.logits + r * a.row_stride_bytes + e0 * E::SIZE, bytes, &full[s]);
    };
    int64_t issued = t0;
    if (TMA && tid == 0)
        for (; issued < min(t1, t0 + kStages); ++issued) issue(issued);

    float mu = -INFINITY, sum = 0.0f;
    bool timed_out = false;
    int64_t t = t0;
    for (; t < t1; ++t) {
        const int64_t r = t / tpr;
        const int b = (int)(r / NP);
        const int tt = (int)(t % tpr);
        const bool seg_first = (t == t0) || (tt == 0);
        const bool seg_last = (t == t1 - 1) || (tt == tpr - 1);
        const int s = (int)((t - t0) % kStages);
        const int64_t e0 = (int64_t)tt * TE;
        const int ne = (int)min((int64_t)TE, (int64_t)V - e0);
        unsigned char* tile = ring + s * kTileBytes;
        const char* row = a.logits + r * a.row_stride_bytes;
        const float T = a.T[b];
        bool ok = true;
        if (TMA) {
            ok = mbar_wait(&full[s], (unsigned)(((t - t0) / kStages) & 1));
        } else {
            for (int e = tid; e < ne; e += kThreads) {
                const uint32_t w = E::load_scalar(row, e0 + e);
                if (DT == 0) reinterpret_cast<uint32_t*>(tile)[e] = w;
                else reinterpret_cast<uint16_t*>(tile)[e] = (uint16_t)w;
            }
            __syncthreads();
        }
        if (seg_first) {
            mu = -INFINITY;
            sum = 0.0f;
        }
        const bool fullt = (ne == TE);
        uint4 v[VPT];
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            v[j] = *reinterpret_cast<const uint4*>(tile + (size_t)(j * kThreads + tid) * 16);
            if (!fullt) v[j] = W::mask(v[j], ne - (j * kThreads + tid) * VEC);
        }
        // every thread has its values in registers: the stage can be refilled
        if (!__syncthreads_and(ok)) {
            timed_out = true;
            break;
        }
        if (TMA && tid == 0 && issued < t1) issue(issued++);
        const float tmax = fmaxf(fmaxf(W::vmax(v[0]), W::vmax(v[1])), fmaxf(W::vmax(v[2]), W::vmax(v[3])));
        const float c = kLog2e / T;
        if (tmax > mu) {
            if (mu != -INFINITY) sum *= fast_exp2((mu - tmax) * c);
            mu = tmax;
        }
        if (mu != -INFINITY) {
            const float mc = mu * c;
            sum += (W::vexp(v[0], c, mc) + W::vexp(v[1], c, mc)) + (W::vexp(v[2], c, mc) + W::vexp(v[3], c, mc));
        }
        if (!seg_last) continue;

        // ---- end of segment: partial sums to the workspace ----------------------
        const int first_owner = sp.owner(r * tpr);
        const int seg = (int)blockIdx.x - first_owner;
        const int nseg = sp.owner(r * tpr + tpr - 1) - first_owner + 1;
        const float Ms = block_max_f32(mu, bs);
        const FF Ss = block_sum_ff((mu != -INFINITY) ? sum * fast_exp2((mu - Ms) * c) : sum, bs);
        if (tid == 0) {
            a.seg_mu[r * tpr + seg] = Ms;
            a.seg_sum[2 * (r * tpr + seg)] = Ss.hi;
            a.seg_sum[2 * (r * tpr + seg) + 1] = Ss.lo;
            if (isnan(Ss.hi) || Ms == INFINITY) atomicOr(a.status, kStBadLogit);
            if (seg == 0 && (r % NP) == 0 && (!(T > 0.0f) || isinf(T))) atomicOr(a.status, kStBadTemperature);
        }
        if (!arrive_last(a.row_ticket + r, (unsigned)nseg, bs)) continue;

        // ---- last segment of row r: its decision table ----------------------------
        float* tab = a.table + r * TW;
        if (tid < 32) {
            const FF l2 = combine_lse(a.seg_mu + r * tpr, a.seg_sum + 2 * r * tpr, nseg, T);
            if (tid == 0) {
                tab[3] = l2.hi;
                tab[4] = l2.lo;
                if (a.row_lse) a.row_lse[r] = __fadd_rn(l2.hi, l2.lo);
                if (!(l2.hi > -INFINITY)) atomicOr(a.status, kStEmptyRow);
                int nc = a.pr.n_child[r], fc = a.pr.first_child[r], sc = a.pr.sampled_child[r];
                if (!pruned_row_ok(nc, fc, sc, K, n.N)) {
                    atomicOr(a.status, kStInternal);
                    nc = 0, sc = -1;
                }
                rs.nc = nc;
                rs.fc = fc;
                rs.sc = sc;
                rs.gen = a.pr.gen_id[r];
                rs.e = (sc >= 0) ? expansion_of_child(K, a.pr.gen_id[(int64_t)b * NP + sc], n.G1, n.E) : 0;
            }
        }
        __syncthreads();
        const int nc = rs.nc, fc = rs.fc, sc = rs.sc;
        const FF lse{tab[3], tab[4]};
        const int64_t q0 = ((int64_t)b * n.E + rs.e) * TL;
        // gather: children tokens, then (sampled child alive) the tail of its draw
        if (tid < nc) {
            rs.tok[tid] = a.pr.token[(int64_t)b * NP + fc + tid];
            rs.cgen[tid] = a.pr.gen_id[(int64_t)b * NP + fc + tid];
        }
        if (sc >= 0 && tid < TL) {
            rs.tids[tid] = a.tree.tail_ids[q0 + tid];
            rs.tq[tid] = a.tree.tail_q[q0 + tid];
        }
        __syncthreads();
        for (int i = tid; i < nc + (sc >= 0 ? TL : 0); i += kThreads) {
            const int tok = (i < nc) ? rs.tok[i] : rs.tids[i - nc];
            rs.lval[i] = (tok >= 0 && tok < V) ? E::value(E::load_scalar(row, tok)) : -INFINITY;
        }
        __syncthreads();
        const uint64_t seed = a.seed[b], off = a.offset[b];
        float ov = 0.0f;
        if (sc >= 0 && tid < TL) {
            const float pt = exp_scaled_minus(rs.lval[nc + tid], T, lse);
            const float qi = rs.tq[tid];
            const float d = __fsub_rn(pt, qi);
            const float rh = d > 0.0f ? d : 0.0f;
            rs.pt[tid] = rh;
            a.rhat_tail[r * TL + tid] = rh;
            ov = fminf(pt, qi);
        }
        if (tid < nc) {
            int pos = -1;
            if (sc >= 0)
                for (int i = 0; i < TL; ++i)
                    if (rs.tids[i] == rs.tok[tid]) pos = i;
            rs.cpos[tid] = pos;
        }
        const FF overlap = block_sum_ff(ov, bs);  // also orders the rs writes above
        if (tid < nc) {
            const float p = exp_scaled_minus(rs.lval[tid], T, lse);
            const float rh = (rs.cpos[tid] >= 0) ? rs.pt[rs.cpos[tid]] : p;
            rs.pc[tid] = p;
            rs.rc[tid] = rh;
            tab[kTabP + tid] = p;
            tab[kTabP + (K + 1) + tid] = rh;
        }
        if (tid < K + 2) {
            const float u = uniform(seed, off, kTagVerify, rs.gen, (uint64_t)tid);
            rs.coin[tid] = u;
            tab[kTabP + 2 * (K + 1) + tid] = u;
        }
        if (tid == kThreads - 1) rs.qs = (sc >= 0) ? a.tree.qtilde[(int64_t)b * n.G1 + rs.cgen[sc - fc]] : 0.0f;
        __syncthreads();
        if (tid == 0) {
            // Algorithm 1 at this node: stochastic first, then recursive rejection in slot order
            const float qs = rs.qs;
            FF M{1.0f, 0.0f};
            int acc = -1, use_tail = 0;
            if (sc >= 0) {
                if (__fmul_rn(rs.coin[0], qs) <= rs.pc[sc - fc]) {
                    acc = sc;
                } else {
                    M = ff_add(FF{1.0f, 0.0f}, ff_neg(overlap));
                    use_tail = 1;
                }
            }
            const FF M0 = M;
            if (acc < 0)
                for (int c2 = 0; c2 < nc; ++c2) {
                    if (fc + c2 == sc) continue;
                    const float eta = rs.coin[1 + slot_of(K, rs.cgen[c2])];
                    const float rv = use_tail ? rs.rc[c2] : rs.pc[c2];
                    if (ff_le(ff_mul(eta, M), rv)) {  // eta * M <= r^(u_i)
                        acc = fc + c2;
                        break;
                    }
                    M = ff_add(M, -rv);
                }
            tab[0] = M0.hi;
            tab[1] = M0.lo;
            tab[2] = qs;
            tab[5] = (float)use_tail;
            tab[6] = (float)acc;
        }
        __syncthreads();
    }

    if (timed_out) {
        if (tid == 0) {
            atomicOr(a.status, kStTimeout);
            for (int64_t u = t; u < issued; ++u)
                mbar_wait(&full[(int)((u - t0) % kStages)], (unsigned)(((u - t0) / kStages) & 1));
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// walk + final draw
// ---------------------------------------------------------------------------
constexpr int kResChunk = 2048;  // elements of the stopping row per residual CTA
constexpr int kStageRows = 1024; // pruned rows whose verdicts the walk stages in shared memory

template <int DT>
__global__ void __launch_bounds__(kThreads) residual_kernel(const VerifyArgs a) {
    using E = Elem<DT>;
    __shared__ BlockScratch bs;
    __shared__ uint32_t excl_bits[kResChunk / 32];
    __shared__ uint32_t tail_bits[kResChunk / 32];
    __shared__ int s_stop, s_len;
    __shared__ int s_path[64];
    __shared__ int s_verdict[kStageRows];

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const int b = blockIdx.y;
    const int V = n.V, K = n.K, TL = n.TL, NP = n.N + 1, D = n.D;
    const int TW = table_width(K);
    const int64_t pb = (int64_t)b * NP;
    // the walk follows the per-row verdicts from the root (staged when they fit)
    const bool staged = NP <= kStageRows;
    if (staged)
        for (int i = tid; i < NP; i += kThreads) s_verdict[i] = (int)__ldcg(a.table + (pb + i) * TW + 6);
    __syncthreads();
    if (tid == 0) {
        int u = 0, len = 0;
        for (;;) {
            const int acc = staged ? s_verdict[u] : (int)__ldcg(a.table + (pb + u) * TW + 6);
            if (acc < 0) break;
            if (acc > n.N || len >= D) {
                if (k == 0) atomicOr(a.status, kStInternal);
                break;
            }
            s_path[len++] = acc;
            u = acc;
        }
        s_stop = u;
        s_len = len;
    }
    __syncthreads();
    const int u = s_stop, len = s_len;
    if (k == 0) {
        if (tid == 0) a.accepted_len[b] = len;
        for (int i = tid; i < D; i += kThreads) {
            a.accepted_tokens[(int64_t)b * D + i] = (i < len) ? a.pr.token[pb + s_path[i]] : -1;
            a.accepted_nodes[(int64_t)b * D + i] = (i < len) ? s_path[i] : -1;
        }
    }
    const int64_t rowg = pb + u;
    const float* tu = a.table + rowg * TW;
    const int use_tail = (int)__ldcg(tu + 5);
    const float lse = __ldcg(tu + 3);
    const float T = a.T[b];
    const uint64_t seed = a.seed[b], off = a.offset[b];
    const int gen_u = a.pr.gen_id[rowg];
    const int nc = a.pr.n_child[rowg], fc = a.pr.first_child[rowg];
    const int nc_ok = (nc >= 0 && nc <= K + 1 && fc >= 0 && fc + nc <= NP) ? nc : 0;
    int64_t e = 0;
    if (use_tail) {
        const int sc = a.pr.sampled_child[rowg];
        e = expansion_of_child(K, (sc >= 0 && sc < NP) ? a.pr.gen_id[pb + sc] : 1, n.G1, n.E);
    }
    const int32_t* tids = a.tree.tail_ids + ((int64_t)b * n.E + e) * TL;
    const char* row = a.logits + rowg * a.row_stride_bytes;
    const int64_t e_lo = (int64_t)k * kResChunk;

    for (int i = tid; i < kResChunk / 32; i += kThreads) { excl_bits[i] = 0u; tail_bits[i] = 0u; }
    __syncthreads();
    for (int c = tid; c < nc_ok; c += kThreads) {
        const int tok = a.pr.token[pb + fc + c];
        if (tok >= e_lo && tok < e_lo + kResChunk)
            atomicOr(&excl_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
    }
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = tids[i];
            if (tok >= e_lo && tok < e_lo + kResChunk)
                atomicOr(&tail_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
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
    {
        // each thread: 8 consecutive elements, two Philox blocks
        const int64_t e0 = e_lo + (int64_t)tid * 8;
        if (e0 < V) {
            uint4 rnd[2];
            rnd[0] = philox_block(seed, off, kTagResidual, gen_u, (uint64_t)(e0 >> 2));
            rnd[1] = philox_block(seed, off, kTagResidual, gen_u, (uint64_t)(e0 >> 2) + 1);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int64_t id = e0 + i;
                if (id >= V) break;
                const float x = E::value(E::load_scalar(row, id));
                const float g = gumbel(u01(word_of(rnd[i >> 2], i & 3)));
                const float tv = __fdiv_rn(x, T);
                const float fb = __fadd_rn(tv, g);
                offer(2, fb, id);
                const int li = (int)(id - e_lo);
                if ((excl_bits[li >> 5] >> (li & 31)) & 1u) continue;
                offer(1, fb, id);
                if (!((tail_bits[li >> 5] >> (li & 31)) & 1u)) offer(0, __fadd_rn(__fsub_rn(tv, lse), g), id);
            }
        }
    }
    // tail entries use log r^ (zero mass after a rejection: no key)
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = tids[i];
            if (tok < e_lo || tok >= e_lo + kResChunk) continue;
            const int li = tok - (int)e_lo;
            if ((excl_bits[li >> 5] >> (li & 31)) & 1u) continue;
            const float rv = __ldcg(a.rhat_tail + rowg * TL + i);
            if (!(rv > 0.0f)) continue;
            const float g = gumbel(uniform(seed, off, kTagResidual, gen_u, (uint64_t)tok));
            offer(0, __fadd_rn(logf(rv), g), tok);
        }
    for (int w = 0; w < 3; ++w) {
        const unsigned long long m = block_max_u64(best[w], bs);
        if (tid == 0 && m) atomicMax(a.res_best + (int64_t)b * 3 + w, m);
    }
    if (!arrive_last(a.res_ticket + b, gridDim.x, bs)) return;
    if (tid == 0) {
        unsigned long long m = __ldcg(a.res_best + (int64_t)b * 3 + 0);
        if (!m) m = __ldcg(a.res_best + (int64_t)b * 3 + 1);
        if (!m) m = __ldcg(a.res_best + (int64_t)b * 3 + 2);
        a.bonus_token[b] = m ? (int32_t)(0xFFFFFFFFu - (uint32_t)m) : -1;
        if (!m) atomicOr(a.status, kStEmptyRow);
        for (int w = 0; w < 3; ++w) a.res_best[(int64_t)b * 3 + w] = 0ull;  // ready for the next call
    }
}

cudaError_t launch_verify(const VerifyArgs& a, int dtype, bool tma, int grid, size_t smem, cudaStream_t s) {
    auto go_stream = [&](auto kern) {
        cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        kern<<<grid, kThreads, smem, s>>>(a);
        return cudaGetLastError();
    };
    cudaError_t err;
    if (dtype == 1) err = tma ? go_stream(verify_stream_kernel<1, true>) : go_stream(verify_stream_kernel<1, false>);
    else err = tma ? go_stream(verify_stream_kernel<0, true>) : go_stream(verify_stream_kernel<0, false>);
    if (err != cudaSuccess) return err;
    const dim3 g2((a.n.V + kResChunk - 1) / kResChunk, a.n.B);
    auto go_res = [&](auto kern) {
        kern<<<g2, kThreads, 0, s>>>(a);
        return cudaGetLastError();
    };
    return dtype == 1 ? go_res(residual_kernel<1>) : go_res(residual_kernel<0>);
}

size_t verify_stream_smem_bytes() { return (size_t)kStages * kTileBytes; }
int verify_table_width(int K) { return table_width(K); }
int verify_tile_elems(int dtype) { return kTileBytes / (dtype == 1 ? 2 : 4); }

}  // namespace rheo
