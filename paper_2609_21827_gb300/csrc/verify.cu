// verify.cu -- RheoVerification (Algorithm 1) applied layer by layer (Theorem 1).
//
// Four launches on the caller's stream:
//
// verify_prep_kernel (beside the stream): one warp per pruned row gathers the
// row's record from the trees (children, tail list, l/T at those tokens, the
// node's Philox coins).
//
// verify_stream_kernel: the B*(N+1) target rows are cut into units of
// kUnitChunks 2 KB chunks (units never straddle rows); every warp takes units
// in row order from one of kStreamQueues counters (its first unit follows from
// its index; the next grab is in flight while it streams), loads 16 bytes a lane straight into registers with
// the next chunk in flight while the current one is summed, and writes one
// partial (max, sum exp((l - max) / T)) per unit.  Warps that run ahead take
// more units, so the launch ends when the work does.
//
// verify_table_kernel, one warp per pruned row after the stream: the row's
// decision table -- lse_T from the unit partials, p at the surviving children
// and, when the row's sampled child survived, r^ = max(0, p - q~) over the tail
// that child was drawn from, the residual mass M = 1 - sum_tail min(p, q~), r^
// at the children, the node's coins, and the verdict of Algorithm 1 at the
// node.  A row's verdict depends on nothing but the row itself.
//
// residual_kernel, grid (chunks, B): each CTA stages its request's verdicts,
// replays the walk from the root (a few comparisons per level), and takes part
// in the final draw u* ~ r over V minus the candidate set (Gumbel-max over the
// stopping row; chunk maxima meet through 64-bit atomicMax, the last CTA of the
// request writes the bonus token).
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
constexpr int kTabP = 7;
__host__ __device__ __forceinline__ int table_width(int K) { return kTabP + 2 * (K + 1) + (K + 2); }

constexpr int kCV = 4;                     // 16-byte vectors per lane per chunk
constexpr int kChunkBytesW = 32 * kCV * 16;  // bytes one warp takes per step
constexpr int kUnitChunks = 4;             // chunks of one row per stream unit
__host__ __device__ __forceinline__ int units_per_row(int cpr) { return (cpr + kUnitChunks - 1) / kUnitChunks; }

struct WarpRow {
    int32_t tok[kMaxSupport];   // children slots
    float pc[kMaxSupport];      // p at the children
    float rc[kMaxSupport];      // r^ at the children
    float pt[kMaxSupport];      // r^ over the tail
    float coin[kMaxSupport + 2];
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

// The first 64 unit partials of a row, two per lane, loaded with the row's
// record so that both arrive in one round trip (absent ones: max -inf, sum 0)
struct Partials {
    float mu[2];
    FF s[2];
};
__device__ __forceinline__ Partials load_partials(const float* mu, const float* sm, int nseg) {
    const int lane = threadIdx.x & 31;
    Partials p;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int c = lane + 32 * k;
        const bool ok = c < nseg;
        p.mu[k] = ok ? __ldcg(mu + c) : -INFINITY;
        p.s[k] = ok ? FF{__ldcg(sm + 2 * c), __ldcg(sm + 2 * c + 1)} : FF{0.0f, 0.0f};
    }
    return p;
}

// lse_T of a row from its unit partials (one warp; float-float accumulation):
// the preloaded first 64, the rest (rows of more than 64 units) read here
__device__ __forceinline__ FF combine_lse(const Partials& p, const float* mu, const float* sm, int nseg, float T) {
    const int lane = threadIdx.x & 31;
    float m = fmaxf(p.mu[0], p.mu[1]);
    for (int c = lane + 64; c < nseg; c += 32) m = fmaxf(m, __ldcg(mu + c));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    FF t{0.0f, 0.0f};
#pragma unroll
    for (int k = 0; k < 2; ++k)
        if (p.s[k].hi != 0.0f) t = ff_add(t, ff_mul(expf(__fdiv_rn(p.mu[k] - m, T)), p.s[k]));
    for (int c = lane + 64; c < nseg; c += 32) {
        const FF sc{__ldcg(sm + 2 * c), __ldcg(sm + 2 * c + 1)};
        if (sc.hi != 0.0f) t = ff_add(t, ff_mul(expf(__fdiv_rn(__ldcg(mu + c) - m, T)), sc));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t = ff_add(t, ff_shfl_xor(t, o));
    return ff_add(ff_div(m, T), ff_log(t));  // m / T + log sum
}

// one warp: (max, float-float sum of 2^((x - max) c)) of the lanes' (m, s)
__device__ __forceinline__ FF warp_partition(float m, float s, float c, float& M) {
    FF v{s, 0.0f};
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o);
        const FF v2 = ff_shfl_xor(v, o);
        const float mm = fmaxf(m, m2);
        const FF x = (m == -INFINITY) ? FF{0.0f, 0.0f} : ff_mul(fast_exp2((m - mm) * c), v);
        const FF y = (m2 == -INFINITY) ? FF{0.0f, 0.0f} : ff_mul(fast_exp2((m2 - mm) * c), v2);
        v = ff_add(x, y);
        m = mm;
    }
    M = m;
    return v;
}

template <int DT, bool ALIGNED>
__device__ __forceinline__ void load_chunk(uint4 (&v)[kCV], const char* row, int e0, int V) {
    using E = Elem<DT>;
    constexpr int CE = 32 * kCV * E::VEC;
    const int lane = threadIdx.x & 31;
    if (ALIGNED && e0 + CE <= V) {
#pragma unroll
        for (int j = 0; j < kCV; ++j) v[j] = ld_stream(row + ((int64_t)e0 + (j * 32 + lane) * E::VEC) * E::SIZE);
        return;
    }
#pragma unroll
    for (int j = 0; j < kCV; ++j) v[j] = load_vec<DT, ALIGNED>(row, (int64_t)e0 + (j * 32 + lane) * E::VEC, V);
}

}  // namespace

// Row records, built by verify_prep_kernel from the trees while the stream
// runs, so that a decision table needs two memory round trips (the record with
// the partials, then the gathers from the target row):
//   hdr[8]     n_child, first_child, sampled_child, gen id, q~(sampled child) bits
//   child[3]   per surviving child: token, tail position (-1: off the tail), slot
//   tids, tq   the tail list of the node's expansion (when its sampled child survived)
//   cx, tx     l / T as float-float at the children and at the tail tokens
//   coin       the node's K+2 Philox coins
constexpr int kHdr = 8;
// three stream CTAs of 256 threads per SM (more loads in flight per SM than
// two): 80 registers a thread at most
constexpr int kPrepThreads = 256;
constexpr int kStreamMaxRegs = 80;

// One warp per pruned row: the row's record.
template <int DT>
__device__ void prep_row(const VerifyArgs& a, int64_t r) {
    using E = Elem<DT>;
    const Dims& n = a.n;
    const int lane = threadIdx.x & 31;
    const int K = n.K, TL = n.TL, NP = n.N + 1, m = n.m;
    const int b = (int)(r / NP);
    const int64_t pb = (int64_t)b * NP, nb = (int64_t)b * n.G1;
    int nc = a.pr.n_child[r], fc = a.pr.first_child[r], sc = a.pr.sampled_child[r];
    if (!pruned_row_ok(nc, fc, sc, K, n.N)) {
        if (lane == 0) atomicOr(a.status, kStInternal);
        nc = 0;
        sc = -1;
    }
    const int gen = a.pr.gen_id[r];
    int* hdr = a.rec_hdr + r * kHdr;
    int* child = a.rec_child + r * (K + 1) * 3;
    // children: token, gen id (slot), and the sampled child's token
    int ctok[4], cslot[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = lane + 32 * q;
        ctok[q] = (i < nc) ? a.pr.token[pb + fc + i] : -1;
        cslot[q] = (i < nc) ? slot_of(K, min(max(a.pr.gen_id[pb + fc + i], 1), (int)n.G1 - 1)) : 0;
    }
    const int ytok = (sc >= 0) ? a.pr.token[pb + sc] : -1;
    const int ygen = (sc >= 0) ? a.pr.gen_id[pb + sc] : 1;
    float qs = 0.0f;
    int ypos = -1;
    if (sc >= 0) {
        qs = a.tree.qtilde[nb + min(max(ygen, 1), (int)n.G1 - 1)];
        const int64_t e = expansion_of_child(K, ygen, n.G1, n.E);
        const int64_t q0 = ((int64_t)b * n.E + e) * TL;
        for (int i0 = 0; i0 < TL; i0 += 32) {
            const int i = i0 + lane;
            int tok = -1;
            if (i < TL) {
                tok = a.tree.tail_ids[q0 + i];
                a.rec_tids[r * TL + i] = tok;
                a.rec_tq[r * TL + i] = a.tree.tail_q[q0 + i];
            }
            const unsigned hit = __ballot_sync(0xFFFFFFFFu, i < TL && tok == ytok);
            if (hit && ypos < 0) ypos = i0 + __ffs(hit) - 1;
        }
    }
    __syncwarp();  // the copied tail is read back below
    // tail positions: the sampled child at ypos, fills at the next ranks with
    // ypos skipped, leads off the tail; anything else is searched for
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = lane + 32 * q;
        if (i >= nc) continue;
        int pos = -1;
        if (sc >= 0) {
            const int j = cslot[q], qf = j - m - 1;
            pos = (j < m) ? -1 : (j == m) ? ypos : qf + (qf >= ypos ? 1 : 0);
            if (pos >= TL || (pos >= 0 && a.rec_tids[r * TL + pos] != ctok[q]) || (pos < 0 && j >= m)) {
                pos = -1;
                for (int t = 0; t < TL; ++t)
                    if (a.rec_tids[r * TL + t] == ctok[q]) pos = t;
            }
        }
        child[3 * i + 0] = ctok[q];
        child[3 * i + 1] = pos;
        child[3 * i + 2] = cslot[q];
    }
    // target logits at the children and at the tail, as l / T
    const float T = a.T[b];
    const char* row = a.logits + r * a.row_stride_bytes;
    auto scaled = [&](int tok) -> FF {
        const float l = (tok >= 0 && tok < n.V) ? E::value(E::load_scalar(row, tok)) : -INFINITY;
        return ff_div(l, T);
    };
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = lane + 32 * q;
        if (i < nc) {
            const FF x = scaled(ctok[q]);
            a.rec_cx[2 * (r * (K + 1) + i)] = x.hi;
            a.rec_cx[2 * (r * (K + 1) + i) + 1] = x.lo;
        }
        if (sc >= 0 && i < TL) {
            const FF x = scaled(a.rec_tids[r * TL + i]);
            a.rec_tx[2 * (r * TL + i)] = x.hi;
            a.rec_tx[2 * (r * TL + i) + 1] = x.lo;
        }
    }
    const uint64_t seed = a.seed[b], off = a.offset[b];
    for (int i = lane; i < K + 2; i += 32) a.rec_coin[r * (K + 2) + i] = uniform(seed, off, kTagVerify, gen, (uint64_t)i);
    if (lane == 0) {
        hdr[0] = nc;
        hdr[1] = fc;
        hdr[2] = sc;
        hdr[3] = gen;
        hdr[4] = __float_as_int(qs);
    }
}

// One warp per pruned row (the grid may be capped, each warp then taking rows in
// turn); it runs beside the stream launch, and the table launch reads its
// records after the stream launch (which waits for this grid before it ends).
template <int DT>
__global__ void __launch_bounds__(kPrepThreads) verify_prep_kernel(const VerifyArgs a) {
    grid_dependency_begin();
    const int64_t rows = (int64_t)a.n.B * (a.n.N + 1);
    const int w = threadIdx.x >> 5;
    for (int64_t r = (int64_t)blockIdx.x * (kPrepThreads / 32) + w; r < rows;
         r += (int64_t)gridDim.x * (kPrepThreads / 32))
        prep_row<DT>(a, r);
}

// exp(x - c) for x = l / T and c as float-float (the arithmetic of exp_scaled_minus)
__device__ __forceinline__ float exp_ff_minus(FF x, FF c) {
    if (!(x.hi > -INFINITY && x.hi < INFINITY)) return expf(x.hi - c.hi);
    return expf(__fsub_rn(x.hi, c.hi) + (x.lo - c.lo));
}

// The decision table of pruned row r (Algorithm 1 at the node), built by one
// warp from the row's unit partials and its record (verify_table_kernel).
// Vanilla verification of the node's children as a top-K pool (Sec. 2.2,
// App. A): every surviving child, the sampled one too, a one-hot candidate in
// slot order against r^ = p; coin draw 1+slot.  Lane 0.
__device__ void onehot_walk(const WarpRow& w, int nc, int fc, float* tab) {
    FF M{1.0f, 0.0f};
    int acc = -1;
    for (int c2 = 0; c2 < nc; ++c2) {
        const float eta = w.coin[1 + w.tok[c2]];
        if (ff_le(ff_mul(eta, M), w.pc[c2])) {
            acc = fc + c2;
            break;
        }
        M = ff_add(M, -w.pc[c2]);
    }
    tab[0] = 1.0f;
    tab[1] = 0.0f;
    tab[5] = 0.0f;
    tab[6] = (float)acc;
}

// Recursive rejection without replacement on the hybrid pool (App. D.2): the
// leads (slots < m) one-hot against p, then the sampled child against the
// renormalised residual p~ = r^ / M (accept iff fp32(eta q~) * M <= p), then on
// its rejection the tail residual becomes max(0, r^ - M q~) and the fills
// (slots > m) go one-hot against it.  Whole warp (the tail is spread over the
// lanes); coins: draw 0 for the sampled child, draw 1+slot otherwise.
__device__ void rrsw_walk(const VerifyArgs& a, int64_t r, WarpRow& w, int nc, int fc, int sc, float qs,
                          const int (&cpos)[4], const float (&tq)[4], const FF (&tx)[4], FF lse, float* tab) {
    const int lane = threadIdx.x & 31;
    const int m = a.n.m, TL = a.n.TL;
    FF M{1.0f, 0.0f};
    int acc = -1;
    if (lane == 0)
        for (int c2 = 0; c2 < nc; ++c2) {
            if (w.tok[c2] >= m) continue;  // leads only
            const float eta = w.coin[1 + w.tok[c2]];
            if (ff_le(ff_mul(eta, M), w.pc[c2])) {
                acc = fc + c2;
                break;
            }
            M = ff_add(M, -w.pc[c2]);
        }
    acc = __shfl_sync(0xFFFFFFFFu, acc, 0);
    M = FF{__shfl_sync(0xFFFFFFFFu, M.hi, 0), __shfl_sync(0xFFFFFFFFu, M.lo, 0)};
    int use_tail = 0;
    if (acc < 0 && sc >= 0) {
        if (lane == 0 && ff_le(ff_mul(__fmul_rn(w.coin[0], qs), M), w.pc[sc - fc])) acc = sc;
        acc = __shfl_sync(0xFFFFFFFFu, acc, 0);
        if (acc < 0) {
            FF ov{0.0f, 0.0f};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = lane + 32 * q;
                if (i >= TL) continue;
                const float pt = exp_ff_minus(tx[q], lse);
                const FF mq = ff_mul(tq[q], M);
                const FF d = ff_add(FF{pt, 0.0f}, ff_neg(mq));
                const float dv = __fadd_rn(d.hi, d.lo);
                const float rh = dv > 0.0f ? dv : 0.0f;
                w.pt[i] = rh;
                a.rhat_tail[r * TL + i] = rh;
                ov = ff_add(ov, (pt < __fadd_rn(mq.hi, mq.lo)) ? FF{pt, 0.0f} : mq);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) ov = ff_add(ov, ff_shfl_xor(ov, o));
            M = ff_add(M, ff_neg(ov));
            use_tail = 1;
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int i = lane + 32 * q;
                if (i < nc) w.rc[i] = (cpos[q] >= 0 && cpos[q] < TL) ? w.pt[cpos[q]] : w.pc[i];
            }
            __syncwarp();
        }
    }
    if (lane == 0) {
        const FF M0 = M;
        if (acc < 0)
            for (int c2 = 0; c2 < nc; ++c2) {
                if (w.tok[c2] <= m) continue;  // fills only
                const float eta = w.coin[1 + w.tok[c2]];
                const float rv = use_tail ? w.rc[c2] : w.pc[c2];
                if (ff_le(ff_mul(eta, M), rv)) {
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
}

template <int DT>
__device__ __noinline__ void finalize_row(const VerifyArgs& a, int64_t r, WarpRow& w) {
    const Dims& n = a.n;
    const int lane = threadIdx.x & 31;
    const int K = n.K, TL = n.TL, NP = n.N + 1;
    const int b = (int)(r / NP);
    const int cpr = n.chunks;
    const int TW = table_width(K);
    const int nseg = units_per_row(cpr);
    // one round trip: the record and the partials
    const Partials part = load_partials(a.seg_mu + r * cpr, a.seg_sum + 2 * r * cpr, nseg);
    const float T = a.T[b];
    const int* hdr = a.rec_hdr + r * kHdr;
    const int* child = a.rec_child + r * (K + 1) * 3;
    const int nc = __ldcg(hdr + 0), fc = __ldcg(hdr + 1), sc = __ldcg(hdr + 2);
    const float qs = __int_as_float(__ldcg(hdr + 4));
    int cpos[4], cslot[4];
    float tq[4];
    FF cx[4], tx[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = lane + 32 * q;
        const bool c_ok = i < K + 1, t_ok = i < TL;
        cpos[q] = c_ok ? __ldcg(child + 3 * i + 1) : -1;
        cslot[q] = c_ok ? __ldcg(child + 3 * i + 2) : 0;
        cx[q] = c_ok ? FF{__ldcg(a.rec_cx + 2 * (r * (K + 1) + i)), __ldcg(a.rec_cx + 2 * (r * (K + 1) + i) + 1)}
                     : FF{-INFINITY, 0.0f};
        tq[q] = t_ok ? __ldcg(a.rec_tq + r * TL + i) : 0.0f;
        tx[q] = t_ok ? FF{__ldcg(a.rec_tx + 2 * (r * TL + i)), __ldcg(a.rec_tx + 2 * (r * TL + i) + 1)}
                     : FF{-INFINITY, 0.0f};
    }
    const float coin_l = (lane < K + 2) ? __ldcg(a.rec_coin + r * (K + 2) + lane) : 0.0f;
    const FF lse = combine_lse(part, a.seg_mu + r * cpr, a.seg_sum + 2 * r * cpr, nseg, T);
    float* tab = a.table + r * TW;
    if (lane == 0) {
        tab[3] = lse.hi;
        tab[4] = lse.lo;
        if (a.row_lse) a.row_lse[r] = __fadd_rn(lse.hi, lse.lo);
        if (!(lse.hi > -INFINITY)) atomicOr(a.status, kStEmptyRow);
        if ((r % NP) == 0 && (!(T > 0.0f) || isinf(T))) atomicOr(a.status, kStBadTemperature);
    }
    // full support: q~ lives in the draft row; full_overlap_kernel decides such rows
    if (a.n.full && sc >= 0) return;
    // r^ over the tail and the overlap sum of min(p, q~) (sampled child survived)
    const int variant = a.variant;
    FF ov{0.0f, 0.0f};
    if (variant == kVerifyRheo && sc >= 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int i = lane + 32 * q;
            if (i >= TL) continue;
            const float pt = exp_ff_minus(tx[q], lse);
            const float d = __fsub_rn(pt, tq[q]);
            const float rh = d > 0.0f ? d : 0.0f;
            w.pt[i] = rh;
            a.rhat_tail[r * TL + i] = rh;
            ov = ff_add(ov, fminf(pt, tq[q]));
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ov = ff_add(ov, ff_shfl_xor(ov, o));
    for (int i = lane; i < K + 2; i += 32) {
        const float u = (i == lane) ? coin_l : __ldcg(a.rec_coin + r * (K + 2) + i);
        w.coin[i] = u;
        tab[kTabP + 2 * (K + 1) + i] = u;
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = lane + 32 * q;
        if (i >= nc) continue;
        const float p = exp_ff_minus(cx[q], lse);
        const float rh = (variant == kVerifyRheo && sc >= 0 && cpos[q] >= 0 && cpos[q] < TL) ? w.pt[cpos[q]] : p;
        w.pc[i] = p;
        w.rc[i] = rh;
        w.tok[i] = cslot[q];  // the slot decides the coin
        tab[kTabP + i] = p;
        tab[kTabP + (K + 1) + i] = rh;
    }
    __syncwarp();
    if (variant == kVerifyRrsw) {
        rrsw_walk(a, r, w, nc, fc, sc, qs, cpos, tq, tx, lse, tab);
        return;
    }
    if (variant == kVerifyOneHot) {
        if (lane == 0) onehot_walk(w, nc, fc, tab);
        return;
    }
    if (lane == 0) {
        // Algorithm 1 at this node: stochastic first, then recursive rejection in slot order
        FF M{1.0f, 0.0f};
        int acc = -1, use_tail = 0;
        if (sc >= 0) {
            if (__fmul_rn(w.coin[0], qs) <= w.pc[sc - fc]) {
                acc = sc;
            } else {
                M = ff_add(FF{1.0f, 0.0f}, ff_neg(ov));
                use_tail = 1;
            }
        }
        const FF M0 = M;
        if (acc < 0)
            for (int c2 = 0; c2 < nc; ++c2) {
                if (fc + c2 == sc) continue;
                const float eta = w.coin[1 + w.tok[c2]];
                const float rv = use_tail ? w.rc[c2] : w.pc[c2];
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
}

template <int DT, bool ALIGNED>
__global__ void __maxnreg__(kStreamMaxRegs) verify_stream_kernel(const VerifyArgs a) {
    // streaming needs nothing from the grids before this one: let the next grid
    // launch now; the wait at the end makes this grid's completion imply the
    // record launch's
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    using E = Elem<DT>;
    using W = Vec<DT>;
    constexpr int VEC = E::VEC;
    constexpr int CE = 32 * kCV * VEC;  // elements per chunk
    constexpr float kLog2e = 1.4426950408889634f;
    const Dims& n = a.n;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int V = n.V, NP = n.N + 1;
    const int cpr = n.chunks, upr = units_per_row(cpr);
    const int64_t total = (int64_t)n.B * NP * upr;
    const int64_t nw = (int64_t)gridDim.x * kWarps;
    // kStreamQueues counters on separate cache lines (one address alone caps the
    // grab rate): counter k hands out units k, k + Q, k + 2Q, ... (row order) to
    // the warps w = k mod Q; a warp's first unit is k + Q * (w / Q), its later
    // ones come from the counter, and every warp grabs until one grab finds no
    // unit, so counter k sees max(units, warps) grabs of its own in all
    // (Q = min(kStreamQueues, warps), so that every counter has warps)
    const int Q = nw < kStreamQueues ? (int)nw : kStreamQueues;
    const int w = blockIdx.x * kWarps + warp;
    const int qk = w % Q;
    unsigned* ctr = a.queue + qk * kStreamQueueStride;
    const int64_t nwk = (nw - qk + Q - 1) / Q;
    const int64_t tk = total > qk ? (total - qk + Q - 1) / Q : 0;
    const int64_t grabs = tk > nwk ? tk : nwk;
    unsigned ticket = 0u;  // lane 0: the grab in flight, read only when needed
    auto grab = [&]() {
        if (lane == 0) ticket = atomicAdd(ctr, 1u);
    };
    auto take = [&]() -> int64_t {  // the next unit, or total when the counter has none left
        const unsigned g = __shfl_sync(0xFFFFFFFFu, ticket, 0);
        if (lane == 0 && (int64_t)g == grabs - 1) atomicExch(ctr, 0u);  // its last grab: ready for the next call
        const int64_t i = nwk + (int64_t)g;
        return i < tk ? qk + (int64_t)Q * i : total;
    };
    int64_t q = qk + (int64_t)Q * (w / Q);
    grab();
    if (q >= total) {
        take();  // the one grab that finds no unit
    } else {
        int64_t r = q / upr;
        int j = (int)(q % upr);
        float c = kLog2e / a.T[r / NP];
        uint4 nxt[kCV];
        load_chunk<DT, ALIGNED>(nxt, a.logits + r * a.row_stride_bytes, j * kUnitChunks * CE, V);
        for (;;) {
            const int cc1 = min(cpr, (j + 1) * kUnitChunks);
            int64_t qn = total, rn = 0;
            int jn = 0;
            float cn = 1.0f;
            float mu = -INFINITY;
            unsigned long long sum2 = 0ull;  // the running sum as a pair of fp32 partial sums
            for (int cc = j * kUnitChunks; cc < cc1; ++cc) {
                uint4 v[kCV];
#pragma unroll
                for (int k = 0; k < kCV; ++k) v[k] = nxt[k];
                if (cc + 1 < cc1) {
                    load_chunk<DT, ALIGNED>(nxt, a.logits + r * a.row_stride_bytes, (cc + 1) * CE, V);
                } else {  // the unit's last chunk: the next unit's first chunk goes in flight
                    qn = take();
                    if (qn < total) {
                        rn = qn / upr;
                        jn = (int)(qn % upr);
                        load_chunk<DT, ALIGNED>(nxt, a.logits + rn * a.row_stride_bytes, jn * kUnitChunks * CE, V);
                        cn = kLog2e / a.T[rn / NP];
                    }
                }
                float tmax = W::vmax(v[0]);
#pragma unroll
                for (int k = 1; k < kCV; ++k) tmax = fmaxf(tmax, W::vmax(v[k]));
                if (tmax > mu) {
                    if (mu != -INFINITY) {
                        const float rs = fast_exp2((mu - tmax) * c);
                        sum2 = f2_mul(sum2, f2_pack(rs, rs));
                    }
                    mu = tmax;
                }
                if (mu != -INFINITY) {  // packed fp32x2 fma and add, one ex2 per element
                    const float mc = mu * c;
                    const unsigned long long c2 = f2_pack(c, c), n2 = f2_pack(-mc, -mc);
                    unsigned long long t = W::vexp2(v[0], c2, n2);
#pragma unroll
                    for (int k = 1; k < kCV; ++k) t = f2_add(t, W::vexp2(v[k], c2, n2));
                    sum2 = f2_add(sum2, t);
                }
            }
            // the unit's partial, read by the table launch after this grid
            float M;
            const FF Sw = warp_partition(mu, f2_fold(sum2), c, M);
            if (lane == 0) {
                const int64_t at = r * cpr + j;
                a.seg_mu[at] = M;
                a.seg_sum[2 * at] = Sw.hi;
                a.seg_sum[2 * at + 1] = Sw.lo;
                if (isnan(Sw.hi) || M == INFINITY) atomicOr(a.status, kStBadLogit);
            }
            if (qn >= total) break;
            r = rn;
            j = jn;
            c = cn;
            grab();
        }
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// One warp per pruned row, after the stream launch: the row's decision table.
template <int DT>
__global__ void __launch_bounds__(kThreads) verify_table_kernel(const VerifyArgs a) {
    // the residual launch may queue up now; the partials and records are read
    // after the wait
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    __shared__ WarpRow wrs[kWarps];
    const int64_t rows = (int64_t)a.n.B * (a.n.N + 1);
    const int warp = threadIdx.x >> 5;
    for (int64_t r = (int64_t)blockIdx.x * kWarps + warp; r < rows; r += (int64_t)gridDim.x * kWarps)
        finalize_row<DT>(a, r, wrs[warp]);
}

// ---------------------------------------------------------------------------
// walk + final draw
// ---------------------------------------------------------------------------
constexpr int kResChunk = 4096;  // elements of the stopping row per residual CTA
constexpr int kResPer = kResChunk / kThreads;  // consecutive elements per thread
constexpr int kStageRows = 1024; // pruned rows whose verdicts the walk stages in shared memory

__device__ __forceinline__ unsigned long long pack_key(float key, int64_t id) {
    return ((unsigned long long)ord_f32(key) << 32) | (0xFFFFFFFFu - (uint32_t)id);
}
__device__ __forceinline__ float key_of_pack(unsigned long long pk) { return Elem<0>::value_of_key((uint32_t)(pk >> 32)); }

// Full support (FULL): every token but the lead belongs to the tail, so after a
// rejection the key of each token outside the candidates is log r^ + g with
// r^ = max(0, p - q~), q~ = exp(l_d/T - lse_tail) read off the stopping node's
// draft row (DALIGNED: that row is 16-byte aligned); the lead keeps log p + g.
template <int DT, bool ALIGNED, bool FULL = false, bool DALIGNED = false>
__global__ void __launch_bounds__(kThreads) residual_kernel(const VerifyArgs a) {
    grid_dependency_begin();
    using E = Elem<DT>;
    static_assert(kResPer % 4 == 0, "whole Philox blocks per thread");
    __shared__ BlockScratch bs;
    __shared__ Red red;
    __shared__ uint32_t excl_bits[kResChunk / 32];
    __shared__ uint32_t tail_bits[kResChunk / 32];
    __shared__ int s_stop, s_len;
    __shared__ unsigned long long s_b0;  // the CTA's best exact key before the filter
    __shared__ int s_path[64];
    __shared__ int s_verdict[kStageRows];

    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const int b = blockIdx.y;
    const int V = n.V, K = n.K, TL = n.TL, NP = n.N + 1, D = n.D;
    const int TW = table_width(K);
    const int64_t pb = (int64_t)b * NP;
    int par = 0;
    // the walk follows the per-row verdicts from the root (staged when they fit)
    const bool staged = NP <= kStageRows;
    if (staged)
        for (int i = tid; i < NP; i += kThreads) s_verdict[i] = (int)__ldcg(a.table + (pb + i) * TW + 6);
    for (int i = tid; i < kResChunk / 32; i += kThreads) {
        excl_bits[i] = 0u;
        tail_bits[i] = 0u;
    }
    if (tid == 0) s_b0 = 0ull;
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
    const FF lse_ff{lse, __ldcg(tu + 4)};
    const float T = a.T[b];
    const uint64_t seed = a.seed[b], off = a.offset[b];
    // the stopping row's record: children and (after a rejection) its tail
    const int* hdr = a.rec_hdr + rowg * kHdr;
    const int nc = __ldcg(hdr + 0), gen_u = __ldcg(hdr + 3);
    const int nc_ok = (nc >= 0 && nc <= K + 1) ? nc : 0;
    const int* rchild = a.rec_child + rowg * (K + 1) * 3;
    const int32_t* tids = a.rec_tids + rowg * TL;
    const char* row = a.logits + rowg * a.row_stride_bytes;
    const int64_t e_lo = (int64_t)k * kResChunk;
    // full support after a rejection: the stopping node's draft row, tail
    // log-partition and lead
    const char* drow = nullptr;
    FF lt{0.0f, 0.0f};
    int lead = -1;
    if (FULL && use_tail) {
        const int sc = __ldcg(hdr + 2);
        const int gs = a.pr.gen_id[pb + (sc >= 0 ? sc : 0)];
        const int e = parent_expansion_of(K, gs);
        const int dd = (e == 0) ? 1 : 2 + (e - 1) / K, f = (e == 0) ? 0 : (e - 1) % K;
        drow = a.draft[dd - 1] + ((int64_t)b * (dd == 1 ? 1 : K) + f) * a.draft_row_stride_bytes;
        lt = FF{__ldcg(a.lse_tail_ff + 2 * ((int64_t)b * n.E + e)), __ldcg(a.lse_tail_ff + 2 * ((int64_t)b * n.E + e) + 1)};
        lead = (n.m == 1) ? a.tree.token[(int64_t)b * n.G1 + gs - 1] : -1;
    }

    // this thread's elements of the stopping row (and, with full support after
    // a rejection, of its draft row), requested before the candidates' records
    // so that both round trips overlap
    const int64_t e0 = e_lo + (int64_t)tid * kResPer;
    uint4 xv[kResPer / E::VEC];
    uint4 dv[kResPer / E::VEC];
#pragma unroll
    for (int j = 0; j < kResPer / E::VEC; ++j) {
        xv[j] = load_vec<DT, ALIGNED>(row, e0 + j * E::VEC, V);
        if (FULL && drow) dv[j] = load_vec<DT, DALIGNED>(drow, e0 + j * E::VEC, V);
    }
    for (int c = tid; c < nc_ok; c += kThreads) {
        const int tok = __ldcg(rchild + 3 * c);
        if (tok >= e_lo && tok < e_lo + kResChunk)
            atomicOr(&excl_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
    }
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = __ldcg(tids + i);
            if (tok >= e_lo && tok < e_lo + kResChunk)
                atomicOr(&tail_bits[(tok - e_lo) >> 5], 1u << ((tok - e_lo) & 31));
        }
    __syncthreads();

    // key of the draw from r: log r^ + g on the tail (after a rejection), log p + g
    // elsewhere, over V minus the candidates; with full support after a
    // rejection every token but the lead is tail, r^ = max(0, p - q~) (no key
    // where it is 0), and the lead keeps log p + g.
    // Exact filter: every key is at most lp + g, lp = fp32(l/T - lse) (log r^ <=
    // log p); the CTA's best exact key among each thread's highest-lp token is a
    // lower bound B0 of the winning key; g never exceeds kGumbelMax, so a token
    // with lp + kGumbelMax < B0 cannot win (no uniform drawn); otherwise it can
    // beat B0 only if u > exp(-exp(lp - B0)), tested with a 1e-4 margin; the
    // rest get the exact key.
    unsigned long long best = 0ull;
    {
        constexpr float kGumbelMax = 16.7f;  // -log(-log u) at the largest uniform is 16.636
        const bool fullr = FULL && drow;
        float lp[kResPer];
        int top = -1;
#pragma unroll
        for (int q = 0; q < kResPer; ++q) {
            const int64_t id = e0 + q;
            const int li = (int)(id - e_lo);
            const bool ok = id < V && !(((excl_bits[li >> 5] | tail_bits[li >> 5]) >> (li & 31)) & 1u);
            lp[q] = ok ? __fsub_rn(__fdiv_rn(E::value(E::raw(xv[q / E::VEC], q % E::VEC)), T), lse) : -INFINITY;
            if (lp[q] > -INFINITY && (top < 0 || lp[q] > lp[top])) top = q;
        }
        auto exact_key = [&](int q, float u) -> float {  // -inf: no key
            if (fullr && e0 + q != lead) {
                const float x = E::value(E::raw(xv[q / E::VEC], q % E::VEC));
                const float xd = E::value(E::raw(dv[q / E::VEC], q % E::VEC));
                const float pt = exp_ff_minus(ff_div(x, T), lse_ff);
                const float qt = expf(__fsub_rn(__fdiv_rn(xd, T), lt.hi) - lt.lo);
                const float rv = __fsub_rn(pt, qt);
                return (rv > 0.0f) ? __fadd_rn(logf(rv), gumbel(u)) : -INFINITY;
            }
            return __fadd_rn(lp[q], gumbel(u));
        };
        unsigned long long pk0 = 0ull;
        if (top >= 0) {
            const float u = u01(word_of(philox_block(seed, off, kTagResidual, gen_u, (uint64_t)((e0 + top) >> 2)),
                                        (int)((e0 + top) & 3)));
            const float k0 = exact_key(top, u);
            if (k0 > -INFINITY) pk0 = pack_key(k0, e0 + top);
        }
        best = pk0;
        const unsigned long long wb = warp_max_u64(pk0);
        if ((tid & 31) == 0 && wb) atomicMax(&s_b0, wb);
        __syncthreads();
        const float B0 = s_b0 ? key_of_pack(s_b0) : -INFINITY;
#pragma unroll
        for (int h = 0; h < kResPer / 4; ++h) {
            bool any = false;
#pragma unroll
            for (int i = 0; i < 4; ++i) any |= (lp[4 * h + i] > -INFINITY && lp[4 * h + i] + kGumbelMax >= B0);
            if (!any) continue;
            const uint4 rnd = philox_block(seed, off, kTagResidual, gen_u, (uint64_t)((e0 >> 2) + h));
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int q = 4 * h + i;
                if (!(lp[q] > -INFINITY) || q == top) continue;
                const float d = B0 - lp[q];
                const float u = u01(word_of(rnd, i));
                if (d > 0.0f) {
                    const float t = fast_exp2(-d * 1.4426950408889634f);          // exp(-d)
                    const float ub = fast_exp2(-t * 1.4426950408889634f);         // exp(-exp(-d))
                    if (u < ub * (1.0f - 1e-4f)) continue;                         // g < d: key below B0
                }
                const float key = exact_key(q, u);
                if (key > -INFINITY) {
                    const unsigned long long pk = pack_key(key, e0 + q);
                    best = pk > best ? pk : best;
                }
            }
        }
    }
    // tail entries use log r^ (zero mass after a rejection: no key)
    if (use_tail)
        for (int i = tid; i < TL; i += kThreads) {
            const int tok = __ldcg(tids + i);
            if (tok < e_lo || tok >= e_lo + kResChunk) continue;
            const int li = tok - (int)e_lo;
            if ((excl_bits[li >> 5] >> (li & 31)) & 1u) continue;
            const float rv = __ldcg(a.rhat_tail + rowg * TL + i);
            if (!(rv > 0.0f)) continue;
            const float g = gumbel(uniform(seed, off, kTagResidual, gen_u, (uint64_t)tok));
            const float key = __fadd_rn(logf(rv), g);
            if (key > -INFINITY) {
                const unsigned long long pk = pack_key(key, tok);
                best = pk > best ? pk : best;
            }
        }
    {
        const unsigned long long m = red_max_u64(best, red, par);
        if (tid == 0 && m) atomicMax(a.res_best + (int64_t)b * 3, m);
    }
    if (!arrive_last(a.res_ticket + b, gridDim.x * gridDim.z, bs)) return;
    unsigned long long m = __ldcg(a.res_best + (int64_t)b * 3);
    if (!m) {
        // rounding left no mass in r: draw from p over V minus the candidates, else
        // over V (one CTA sweeps the whole row; this only follows dead ends)
        unsigned long long b1 = 0ull, b2 = 0ull;
        for (int64_t id = tid; id < V; id += kThreads) {
            bool ex = false;
            for (int c = 0; c < nc_ok; ++c) ex |= (__ldcg(rchild + 3 * c) == id);
            const float x = E::value(E::load_scalar(row, id));
            const float g = gumbel(uniform(seed, off, kTagResidual, gen_u, (uint64_t)id));
            const float key = __fadd_rn(__fdiv_rn(x, T), g);
            if (key > -INFINITY) {
                const unsigned long long pk = pack_key(key, id);
                b2 = pk > b2 ? pk : b2;
                if (!ex) b1 = pk > b1 ? pk : b1;
            }
        }
        const unsigned long long m1 = red_max_u64(b1, red, par);
        const unsigned long long m2 = red_max_u64(b2, red, par);
        m = m1 ? m1 : m2;
    }
    if (tid == 0) {
        a.bonus_token[b] = m ? (int32_t)(0xFFFFFFFFu - (uint32_t)m) : -1;
        if (!m) atomicOr(a.status, kStEmptyRow);
        a.res_best[(int64_t)b * 3] = 0ull;  // ready for the next call
    }
}

// Full support, after the stream kernel: the rows whose sampled child
// survived.  One CTA per such row first decides the sampled child (coin
// against p(Y) / q~(Y)); only after a rejection does it stream the target row
// and its node's draft row side by side for M = 1 - sum min(p, q~) (p =
// softmax(l/T) with the log-partition from the stream kernel, q~ = exp(l_d/T -
// lse_tail) off the lead, 0 at the lead), then decides the other children in
// slot order against r^ = max(0, p - q~) (Algorithm 1), writing the row's table
// as the stream kernel does for other rows.
// While streaming, each exponent is formed in log2 units as (l - T*lse) *
// log2(e)/T, with T*lse and log2(e)/T held as float-float constants of the
// row: l - (T*lse).hi is exact near the terms that carry mass, so the
// exponent keeps fp32 relative accuracy however large l/T is, and the
// hardware exp2 gives p and q~; each thread sums eight min(p, q~) in fp32 and
// carries the running total as float-float.
constexpr int kOvThreads = 512;
constexpr int kOvWarps = kOvThreads / 32;
constexpr int kOvBatch = 4;  // vectors of each row in flight per thread

template <int DT, bool ALIGNED, bool DALIGNED>
__global__ void __launch_bounds__(kOvThreads) full_overlap_kernel(const VerifyArgs a) {
    grid_dependency_begin();
    using E = Elem<DT>;
    constexpr int VEC = E::VEC;
    __shared__ Red red;
    __shared__ float s_pc[kMaxSupport], s_rc[kMaxSupport], s_coin[kMaxSupport + 1];
    __shared__ int s_slot[kMaxSupport];
    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int64_t r = blockIdx.x;
    const int K = n.K, NP = n.N + 1, V = n.V;
    const int* hdr = a.rec_hdr + r * kHdr;
    const int sc = __ldcg(hdr + 2);
    if (sc < 0) return;  // decided by the stream kernel
    const int nc = __ldcg(hdr + 0), fc = __ldcg(hdr + 1);
    const float qs = __int_as_float(__ldcg(hdr + 4));
    const int b = (int)(r / NP);
    const int64_t pb = (int64_t)b * NP;
    float* tab = a.table + r * table_width(K);
    const FF lse{__ldcg(tab + 3), __ldcg(tab + 4)};
    const float T = a.T[b];
    const int gs = a.pr.gen_id[pb + sc];
    const int e = parent_expansion_of(K, gs);
    const FF lt{__ldcg(a.lse_tail_ff + 2 * ((int64_t)b * n.E + e)), __ldcg(a.lse_tail_ff + 2 * ((int64_t)b * n.E + e) + 1)};
    const int lead = (n.m == 1) ? a.tree.token[(int64_t)b * n.G1 + gs - 1] : -1;
    const int dd = (e == 0) ? 1 : 2 + (e - 1) / K, f = (e == 0) ? 0 : (e - 1) % K;
    const char* drow = a.draft[dd - 1] + ((int64_t)b * (dd == 1 ? 1 : K) + f) * a.draft_row_stride_bytes;
    const char* trow = a.logits + r * a.row_stride_bytes;
    int par = 0;

    // the children: p and r^ = max(0, p - q~) at each
    const int nc_ok = (nc >= 0 && nc <= K + 1) ? nc : 0;
    for (int c = tid; c < nc_ok; c += kOvThreads) {
        const int* ch = a.rec_child + (r * (K + 1) + c) * 3;
        const int tok = __ldcg(ch + 0);
        const float pt = exp_ff_minus(ff_div(E::value(E::load_scalar(trow, tok)), T), lse);
        const float qt = (tok == lead) ? 0.0f
                                       : expf(__fsub_rn(__fdiv_rn(E::value(E::load_scalar(drow, tok)), T), lt.hi) - lt.lo);
        const float dlt = __fsub_rn(pt, qt);
        s_pc[c] = pt;
        s_rc[c] = dlt > 0.0f ? dlt : 0.0f;
        s_slot[c] = __ldcg(ch + 2);
    }
    for (int i = tid; i < K + 2; i += kOvThreads) s_coin[i] = __ldcg(a.rec_coin + r * (K + 2) + i);
    __syncthreads();
    // the sampled child first: accepted iff eta * q~(Y) <= p(Y); M is then not needed
    const bool sampled_ok = sc - fc >= 0 && sc - fc < nc_ok && __fmul_rn(s_coin[0], qs) <= s_pc[sc - fc];

    FF ov{0.0f, 0.0f};
    if (!sampled_ok) {  // block-uniform
        const FF cp = ff_mul(T, lse), cq = ff_mul(T, lt);
        // log2(e)/T as float-float (log2(e) = 0x1.715476p+0 + 0x1.4ae0cp-26); the
        // high part rounded down, so the low part is positive and a logit of -inf
        // gives an exponent of -inf (never -inf + inf)
        const float l2h = 0x1.715476p+0f, l2l = 0x1.4ae0cp-26f;
        const float clh = __fdiv_rd(l2h, T);
        const float cll = __fdiv_rn(fmaf(-clh, T, l2h) + l2l, T);
        const int nvec = (V + VEC - 1) / VEC;
        // the next batch of both rows is in flight while this one is summed
        uint4 tn[kOvBatch], dn[kOvBatch];
#pragma unroll
        for (int u = 0; u < kOvBatch; ++u) {
            const int64_t e0 = (int64_t)(tid + u * kOvThreads) * VEC;
            tn[u] = load_vec<DT, ALIGNED>(trow, e0, V);  // past V: -inf, no mass
            dn[u] = load_vec<DT, DALIGNED>(drow, e0, V);
        }
        for (int v0 = tid; v0 < nvec; v0 += kOvBatch * kOvThreads) {
            uint4 tv[kOvBatch], dv[kOvBatch];
#pragma unroll
            for (int u = 0; u < kOvBatch; ++u) {
                tv[u] = tn[u];
                dv[u] = dn[u];
            }
            if (v0 + kOvBatch * kOvThreads < nvec) {
#pragma unroll
                for (int u = 0; u < kOvBatch; ++u) {
                    const int64_t e0 = (int64_t)(v0 + (kOvBatch + u) * kOvThreads) * VEC;
                    tn[u] = load_vec<DT, ALIGNED>(trow, e0, V);
                    dn[u] = load_vec<DT, DALIGNED>(drow, e0, V);
                }
            }
#pragma unroll
            for (int u = 0; u < kOvBatch; ++u) {
                const int e0 = (v0 + u * kOvThreads) * VEC;
                float s8 = 0.0f;
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    const float dpx = __fsub_rn(__fsub_rn(E::value(E::raw(tv[u], i)), cp.hi), cp.lo);
                    const float dqx = __fsub_rn(__fsub_rn(E::value(E::raw(dv[u], i)), cq.hi), cq.lo);
                    const float pt = fast_exp2(fmaf(dpx, clh, dpx * cll));
                    const float qt = fast_exp2(fmaf(dqx, clh, dqx * cll));
                    s8 += fminf(pt, qt);
                }
                if ((unsigned)(lead - e0) < (unsigned)VEC) {  // q~ is 0 at the lead: sum the vector again without it
                    s8 = 0.0f;
                    for (int i = 0; i < VEC; ++i) {
                        if (e0 + i == lead) continue;
                        const float dpx = __fsub_rn(__fsub_rn(E::value(E::raw(tv[u], i)), cp.hi), cp.lo);
                        const float dqx = __fsub_rn(__fsub_rn(E::value(E::raw(dv[u], i)), cq.hi), cq.lo);
                        s8 += fminf(fast_exp2(fmaf(dpx, clh, dpx * cll)), fast_exp2(fmaf(dqx, clh, dqx * cll)));
                    }
                }
                ov = ff_add(ov, s8);
            }
        }
        ov = red_sum_ff<kOvWarps>(ov, red, par);
    }
    if (tid == 0) {
        FF M{1.0f, 0.0f};
        int acc = -1, use_tail = 0;
        if (sampled_ok) {
            acc = sc;
        } else {
            M = ff_add(FF{1.0f, 0.0f}, ff_neg(ov));
            use_tail = 1;
        }
        const FF M0 = M;
        if (acc < 0)
            for (int c2 = 0; c2 < nc_ok; ++c2) {
                if (fc + c2 == sc) continue;
                const float eta = s_coin[1 + s_slot[c2]];
                if (ff_le(ff_mul(eta, M), s_rc[c2])) {
                    acc = fc + c2;
                    break;
                }
                M = ff_add(M, -s_rc[c2]);
            }
        tab[0] = M0.hi;
        tab[1] = M0.lo;
        tab[2] = qs;
        tab[5] = (float)use_tail;
        tab[6] = (float)acc;
    }
}

cudaError_t launch_verify_full(const VerifyArgs& a, int dtype, bool aligned, bool draft_aligned, int grid,
                               cudaStream_t s) {
    const int64_t rows = (int64_t)a.n.B * (a.n.N + 1);
    const int64_t prep_ctas = (rows + kPrepThreads / 32 - 1) / (kPrepThreads / 32);
    const dim3 gp((unsigned)(a.prep_grid > 0 && a.prep_grid < prep_ctas ? a.prep_grid : prep_ctas));
    cudaError_t err = (dtype == 1) ? launch_dependent(verify_prep_kernel<1>, gp, dim3(kPrepThreads), 0, s, a)
                                   : launch_dependent(verify_prep_kernel<0>, gp, dim3(kPrepThreads), 0, s, a);
    if (err != cudaSuccess) return err;
    auto go = [&](auto kern, dim3 g) { return launch_dependent(kern, g, dim3(kThreads), 0, s, a); };
    if (dtype == 1) err = aligned ? go(verify_stream_kernel<1, true>, dim3(grid)) : go(verify_stream_kernel<1, false>, dim3(grid));
    else err = aligned ? go(verify_stream_kernel<0, true>, dim3(grid)) : go(verify_stream_kernel<0, false>, dim3(grid));
    if (err != cudaSuccess) return err;
    const dim3 gt((unsigned)((rows + kWarps - 1) / kWarps));
    err = (dtype == 1) ? go(verify_table_kernel<1>, gt) : go(verify_table_kernel<0>, gt);
    if (err != cudaSuccess) return err;
    const dim3 go_rows((unsigned)rows);
    auto go_ov = [&](auto kern) { return launch_dependent(kern, go_rows, dim3(kOvThreads), 0, s, a); };
    if (dtype == 1) {
        if (aligned && draft_aligned) err = go_ov(full_overlap_kernel<1, true, true>);
        else err = go_ov(full_overlap_kernel<1, false, false>);
    } else {
        if (aligned && draft_aligned) err = go_ov(full_overlap_kernel<0, true, true>);
        else err = go_ov(full_overlap_kernel<0, false, false>);
    }
    if (err != cudaSuccess) return err;
    const dim3 g2((a.n.V + kResChunk - 1) / kResChunk, a.n.B);
    if (dtype == 1) {
        if (aligned && draft_aligned) return go(residual_kernel<1, true, true, true>, g2);
        return go(residual_kernel<1, false, true, false>, g2);
    }
    if (aligned && draft_aligned) return go(residual_kernel<0, true, true, true>, g2);
    return go(residual_kernel<0, false, true, false>, g2);
}

cudaError_t launch_verify(const VerifyArgs& a, int dtype, bool aligned, int grid, cudaStream_t s) {
    const int64_t rows = (int64_t)a.n.B * (a.n.N + 1);
    const int64_t prep_ctas = (rows + kPrepThreads / 32 - 1) / (kPrepThreads / 32);
    const dim3 gp((unsigned)(a.prep_grid > 0 && a.prep_grid < prep_ctas ? a.prep_grid : prep_ctas));
    cudaError_t e0 = (dtype == 1) ? launch_dependent(verify_prep_kernel<1>, gp, dim3(kPrepThreads), 0, s, a)
                                  : launch_dependent(verify_prep_kernel<0>, gp, dim3(kPrepThreads), 0, s, a);
    if (e0 != cudaSuccess) return e0;
    auto go_stream = [&](auto kern) {
        return launch_dependent(kern, dim3(grid), dim3(kThreads), 0, s, a);
    };
    cudaError_t err;
    if (dtype == 1) err = aligned ? go_stream(verify_stream_kernel<1, true>) : go_stream(verify_stream_kernel<1, false>);
    else err = aligned ? go_stream(verify_stream_kernel<0, true>) : go_stream(verify_stream_kernel<0, false>);
    if (err != cudaSuccess) return err;
    const dim3 gt((unsigned)((rows + kWarps - 1) / kWarps));
    err = (dtype == 1) ? launch_dependent(verify_table_kernel<1>, gt, dim3(kThreads), 0, s, a)
                       : launch_dependent(verify_table_kernel<0>, gt, dim3(kThreads), 0, s, a);
    if (err != cudaSuccess) return err;
    const dim3 g2((a.n.V + kResChunk - 1) / kResChunk, a.n.B);
    if (dtype == 1)
        return aligned ? launch_dependent(residual_kernel<1, true>, g2, dim3(kThreads), 0, s, a)
                       : launch_dependent(residual_kernel<1, false>, g2, dim3(kThreads), 0, s, a);
    return aligned ? launch_dependent(residual_kernel<0, true>, g2, dim3(kThreads), 0, s, a)
                   : launch_dependent(residual_kernel<0, false>, g2, dim3(kThreads), 0, s, a);
}

int verify_table_width(int K) { return table_width(K); }
int verify_chunks_per_row(int dtype, int V) {
    const int ce = kChunkBytesW / (dtype == 1 ? 2 : 4);
    return (V + ce - 1) / ce;
}
// stream grid: three CTAs per SM, no more CTAs than needed for one chunk per warp
int verify_stream_grid(int sms, int64_t chunks) {
    const int64_t g = 3 * (int64_t)sms;
    const int64_t need = (chunks + kWarps - 1) / kWarps;
    return (int)(g < need ? g : need);
}

}  // namespace rheo
