// expand.cu -- one expansion call of the draft tree (Sec. 2.1, Sec. 3.2, App. C.1).
//
// Persistent CTAs stream the B*F draft rows tile by tile (stream.cuh).  Over
// each row segment a CTA keeps
//   * a running (max, sum exp(l - max)) per thread at T = 1 (untempered, Sec. 5.4),
//   * the segment's exact top-S keys (ord(logit) << 32 | ~id): a shared-memory
//     candidate buffer filled with every element at or above a threshold theta
//     that is always a lower bound of the segment's S-th key.  theta starts as
//     a bound from the first tile (each warp's ceil(S/8)-th largest thread
//     maximum; their minimum has >= S elements above it) and is raised to the
//     exact S-th key whenever the buffer is compacted.
// At the end of a segment the list and the partial sums go to the workspace.
// The CTA that ends the last segment of a row (arrival counter, never a wait)
// merges the lists into the row's sorted support, draws Y from the tempered
// tail by Gumbel-max and writes the K+1 children; the last row of a request
// selects the next frontier.
#include "rheo_device.cuh"
#include "rheo_kernels.h"
#include "stream.cuh"

namespace rheo {

namespace {

constexpr int kCand = 1024;      // candidate buffer (keys) of a segment
constexpr int kCandHigh = 896;   // compact when the buffer holds more than this

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

__device__ __forceinline__ unsigned long long make_key(uint32_t k32, int64_t id) {
    return ((unsigned long long)k32 << 32) | (0xFFFFFFFFu - (uint32_t)id);
}

// k-th largest (1-based) of the 32 lanes' values, all lanes get it
__device__ __forceinline__ uint32_t warp_kth_largest(uint32_t x, int k) {
    const int lane = threadIdx.x & 31;
    int rank = 0;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        const uint32_t y = __shfl_sync(0xFFFFFFFFu, x, j);
        rank += (y > x) || (y == x && j < lane);
    }
    const unsigned who = __ballot_sync(0xFFFFFFFFu, rank == k - 1);
    return __shfl_sync(0xFFFFFFFFu, x, __ffs(who) - 1);
}

// Top-`keep` of the buffer: returns the threshold T (keys >= T are kept).
__device__ unsigned long long select_buffer(const unsigned long long* buf, int n, int keep, unsigned* hist,
                                            RadixScratch& rs) {
    if (n <= keep) return 1ull;
    return block_radix_threshold([&](int i) { return buf[i]; }, n, keep, hist, rs);
}

// Keep the buffer entries >= thr (the buffer holds at most kCand keys).
__device__ void compact_buffer(unsigned long long* buf, int n, unsigned long long thr, int* count) {
    const int tid = threadIdx.x;
    unsigned long long mine[kCand / kThreads];
#pragma unroll
    for (int j = 0; j < kCand / kThreads; ++j) {
        const int i = tid + j * kThreads;
        mine[j] = (i < n) ? buf[i] : 0ull;
    }
    __syncthreads();
    if (tid == 0) *count = 0;
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kCand / kThreads; ++j)
        if (mine[j] && mine[j] >= thr) buf[atomicAdd(count, 1)] = mine[j];
    __syncthreads();
}


// Overflow of the candidate buffer while adding one tile (massive ties, or a
// weak bound): exact S-th key of (buffer before this tile) U (tile elements >=
// theta), read again from the tile in shared memory; keeps exactly those keys.
template <int DT>
__device__ __noinline__ uint32_t tile_overflow(const unsigned char* tile, int ne, int64_t e0, uint32_t theta,
                                               unsigned long long* cand, int before, int S, int* count,
                                               unsigned* hist, RadixScratch& rs) {
    using E = Elem<DT>;
    const int tid = threadIdx.x;
    auto elem_key = [&](int e) -> uint32_t {
        const uint32_t raw = (DT == 0) ? reinterpret_cast<const uint32_t*>(tile)[e]
                                       : (uint32_t)reinterpret_cast<const uint16_t*>(tile)[e];
        return E::key(raw);
    };
    const unsigned long long thr = block_radix_threshold(
        [&](int i) -> unsigned long long {
            if (i < before) return cand[i];
            const int e = i - before;
            const uint32_t kk = elem_key(e);
            return kk >= theta ? make_key(kk, e0 + e) : 0ull;
        },
        before + ne, S, hist, rs);
    compact_buffer(cand, before, thr, count);
    for (int e = tid; e < ne; e += kThreads) {
        const uint32_t kk = elem_key(e);
        if (kk >= theta) {
            const unsigned long long x = make_key(kk, e0 + e);
            if (x >= thr) cand[atomicAdd(count, 1)] = x;
        }
    }
    __syncthreads();
    return (uint32_t)(thr >> 32);
}

}  // namespace

template <int DT, bool TMA>
__global__ void __launch_bounds__(kThreads, 2) expand_kernel(const ExpandArgs a) {
    using E = Elem<DT>;
    using W = Vec<DT>;
    constexpr int VEC = E::VEC;
    constexpr int TE = kTileBytes / E::SIZE;   // elements per tile
    constexpr int VPT = TE / VEC / kThreads;   // 16-byte vectors per thread per tile
    static_assert(VPT == 4, "tile layout");
    constexpr float kLog2e = 1.4426950408889634f;
    extern __shared__ __align__(128) unsigned char dsm[];
    unsigned char* ring = dsm;
    unsigned long long* cand = reinterpret_cast<unsigned long long*>(dsm + kStages * kTileBytes);
    unsigned long long* mkeys = cand + kCand;
    __shared__ __align__(8) uint64_t full[kStages];
    __shared__ BlockScratch bs;
    __shared__ E2Smem e2;
    __shared__ int s_count;
    __shared__ uint32_t s_wk[3][kWarps];
    __shared__ int s_wtot[2][kWarps];
    __shared__ unsigned s_hist[kRadixBins];
    __shared__ RadixScratch s_rad;

    const Dims& n = a.n;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int V = n.V, S = n.S, K = n.K, m = n.m, TL = n.TL;
    const int tpr = (V + TE - 1) / TE;
    const TileSplit sp{(int64_t)n.B * a.F * tpr, (int)gridDim.x};
    const int64_t t0 = sp.begin(blockIdx.x), t1 = sp.begin(blockIdx.x + 1);
    int parity = 0;

    if (tid == 0) {
        s_count = 0;
        if (TMA) {
            for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
            mbar_fence_init();
        }
    }
    __syncthreads();
    auto issue = [&](int64_t t) {  // thread 0: start the copy of tile t into its stage
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

    // per-segment state; theta, before and seg_valid are the same in every thread
    float mu = -INFINITY, sum = 0.0f;
    uint32_t theta = 0;
    int before = 0;
    int64_t seg_valid = 0;
    bool timed_out = false;
    int64_t t = t0;
    for (; t < t1; ++t) {
        const int64_t r = t / tpr;
        const int tt = (int)(t % tpr);
        const bool seg_first = (t == t0) || (tt == 0);
        const bool seg_last = (t == t1 - 1) || (tt == tpr - 1);
        const int s = (int)((t - t0) % kStages);
        const int64_t e0 = (int64_t)tt * TE;
        const int ne = (int)min((int64_t)TE, (int64_t)V - e0);
        unsigned char* tile = ring + s * kTileBytes;
        bool ok = true;
        if (TMA) {
            ok = mbar_wait(&full[s], (unsigned)(((t - t0) / kStages) & 1));
        } else {
            const char* row = a.logits + r * a.row_stride_bytes;
            for (int e = tid; e < ne; e += kThreads) {
                const uint32_t w = E::load_scalar(row, e0 + e);
                if (DT == 0) reinterpret_cast<uint32_t*>(tile)[e] = w;
                else reinterpret_cast<uint16_t*>(tile)[e] = (uint16_t)w;
            }
            __syncthreads();
        }
        const bool fullt = (ne == TE);
        uint4 v[VPT];
#pragma unroll
        for (int j = 0; j < VPT; ++j) {
            v[j] = *reinterpret_cast<const uint4*>(tile + (size_t)(j * kThreads + tid) * 16);
            if (!fullt) v[j] = W::mask(v[j], ne - (j * kThreads + tid) * VEC);
        }
        float vm[VPT];
#pragma unroll
        for (int j = 0; j < VPT; ++j) vm[j] = W::vmax(v[j]);
        const float tmax = fmaxf(fmaxf(vm[0], vm[1]), fmaxf(vm[2], vm[3]));

        if (seg_first) {
            mu = -INFINITY;
            sum = 0.0f;
            seg_valid = 0;
            before = 0;
            // bootstrap from this tile: every warp has >= kk thread maxima >= its kk-th largest
            const uint32_t kmax = (tid * VEC < ne) ? E::key_of_value(tmax) : 0u;
            const uint32_t w = warp_kth_largest(kmax, (S + kWarps - 1) / kWarps);
            if (lane == 0) s_wk[0][warp] = w;
            __syncthreads();
            uint32_t th = s_wk[0][0];
#pragma unroll
            for (int i = 1; i < kWarps; ++i) th = min(th, s_wk[0][i]);
            theta = th;
        }
        seg_valid += ne;

        // running partition sum at T = 1 (online max); mu is also the running maximum
        if (tmax > mu) {
            if (mu != -INFINITY) sum *= fast_exp2((mu - tmax) * kLog2e);
            mu = tmax;
        }
        if (mu != -INFINITY) {
            const float mc = mu * kLog2e;
            sum += (W::vexp(v[0], kLog2e, mc) + W::vexp(v[1], kLog2e, mc)) +
                   (W::vexp(v[2], kLog2e, mc) + W::vexp(v[3], kLog2e, mc));
        }

        // candidates: elements >= theta (float compare; the key order is the value order)
        const float thv = E::threshold_value(theta);
        uint32_t cmask = 0u;
#pragma unroll
        for (int j = 0; j < VPT; ++j)
            if (vm[j] >= thv)
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    const float x = E::value(E::raw(v[j], i));
                    cmask |= (x >= thv && (fullt || (j * kThreads + tid) * VEC + i < ne)) ? (1u << (j * VEC + i)) : 0u;
                }
        const int c = __popc(cmask);
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        // next lower bound of the segment's S-th key from the running thread maxima
        const uint32_t wk = warp_kth_largest((seg_valid > (int64_t)tid * VEC) ? E::key_of_value(mu) : 0u,
                                             (S + kWarps - 1) / kWarps);
        if (lane == 31) s_wtot[t & 1][warp] = incl;
        if (lane == 0) s_wk[1 + (t & 1)][warp] = wk;
        if (!__syncthreads_and(ok)) {  // also: every thread is done reading the stage
            timed_out = true;
            break;
        }
        int total = 0, woff = incl - c;
        uint32_t th_next = s_wk[1 + (t & 1)][0];
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const int x = s_wtot[t & 1][w];
            woff += (w < warp) ? x : 0;
            total += x;
            th_next = min(th_next, s_wk[1 + (t & 1)][w]);
        }
        if (before + total <= kCand) {
            int pos = before + woff;
            for (uint32_t mm = cmask; mm; mm &= mm - 1) {
                const int q = __ffs(mm) - 1;
                const int j = q / VEC, i = q % VEC;
                cand[pos++] = make_key(E::key(E::raw(v[j], i)), e0 + (j * kThreads + tid) * VEC + i);
            }
            before += total;
            if (TMA && tid == 0 && issued < t1) issue(issued++);
            if (before > kCandHigh) {
                __syncthreads();
                const unsigned long long thr = select_buffer(cand, before, S, s_hist, s_rad);
                compact_buffer(cand, before, thr, &s_count);
                before = s_count;
                theta = max(theta, (uint32_t)(thr >> 32));
                __syncthreads();
            }
        } else {
            // overflow (massive ties, or a weak bound): rebuild from the tile, which
            // stays in shared memory until this is done
            __syncthreads();
            theta = tile_overflow<DT>(tile, ne, e0, theta, cand, before, S, &s_count, s_hist, s_rad);
            before = s_count;
            __syncthreads();
            if (TMA && tid == 0 && issued < t1) issue(issued++);
        }
        theta = max(theta, th_next);

        if (!seg_last) continue;
        __syncthreads();  // the candidate writes of this tile are visible
        const int cnt = before;

        // ---- end of segment: exact top-S list and partial sums to the workspace ----
        const int target = (int)min((int64_t)S, seg_valid);
        const unsigned long long thr = select_buffer(cand, cnt, target, s_hist, s_rad);
        const int first_owner = sp.owner(r * tpr);
        const int seg = (int)blockIdx.x - first_owner;
        const int nseg = sp.owner(r * tpr + tpr - 1) - first_owner + 1;
        unsigned long long* out = a.seg_keys + ((int64_t)r * tpr + seg) * S;
        __syncthreads();
        if (tid == 0) e2.sel_count = 0;
        __syncthreads();
        for (int i = tid; i < cnt; i += kThreads)
            if (cand[i] >= thr) {
                const int pos = atomicAdd(&e2.sel_count, 1);
                if (pos < S) out[pos] = cand[i];
            }
        const float Ms = block_max_f32(mu, bs);
        const FF Ss = block_sum_ff((mu != -INFINITY) ? sum * fast_exp2((mu - Ms) * kLog2e) : sum, bs);
        const int written = e2.sel_count;
        for (int i = written + tid; i < S; i += kThreads) out[i] = 0ull;
        if (tid == 0) {
            a.seg_mu[(int64_t)r * tpr + seg] = Ms;
            a.seg_sum[2 * ((int64_t)r * tpr + seg)] = Ss.hi;
            a.seg_sum[2 * ((int64_t)r * tpr + seg) + 1] = Ss.lo;
            if (isnan(Ss.hi) || Ms == INFINITY) atomicOr(a.status, kStBadLogit);
            if (written != target) atomicOr(a.status, kStInternal);
        }
        if (!arrive_last(a.row_ticket + r, (unsigned)nseg, bs)) continue;

        // ---- last segment of row r: support, tail sample, pool ---------------------
        const int b = (int)(r / a.F), f = (int)(r % a.F);
        const int nkeys = nseg * S;
        const unsigned long long* rk = a.seg_keys + (int64_t)r * tpr * S;
        for (int i = tid; i < nkeys; i += kThreads) mkeys[i] = __ldcg(rk + i);
        __syncthreads();
        {
            int nz = 0;
            for (int i = tid; i < nkeys; i += kThreads) nz += mkeys[i] != 0ull;
            nz = block_sum_int(nz, bs, parity);
            unsigned long long rthr = 1ull;
            if (nz > S) rthr = block_radix_threshold([&](int i) { return mkeys[i]; }, nkeys, S, s_hist, s_rad);
            if (tid == 0) e2.sel_count = 0;
            __syncthreads();
            for (int i = tid; i < nkeys; i += kThreads) {
                const unsigned long long x = mkeys[i];
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
        if (tid < 32) {
            float mx = -INFINITY;
            for (int c = tid; c < nseg; c += 32) mx = fmaxf(mx, __ldcg(a.seg_mu + (int64_t)r * tpr + c));
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
            FF acc{0.0f, 0.0f};
            for (int c = tid; c < nseg; c += 32) {
                const int64_t q = (int64_t)r * tpr + c;
                const FF sc{__ldcg(a.seg_sum + 2 * q), __ldcg(a.seg_sum + 2 * q + 1)};
                if (sc.hi != 0.0f) acc = ff_add(acc, ff_mul(expf(__ldcg(a.seg_mu + q) - mx), sc));
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc = ff_add(acc, ff_shfl_xor(acc, o));
            if (tid == 0) {
                const FF l = ff_add(ff_log(acc), mx);
                e2.lse1 = __fadd_rn(l.hi, l.lo);
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
        const float mt = block_max_f32(tau, bs);
        const FF st = block_sum_ff((tid < TL && mt > -INFINITY) ? expf(tau - mt) : 0.0f, bs);
        const FF lse_tail = ff_add(ff_log(st), mt);
        unsigned long long pack = 0ull;
        if (tid < TL) {
            e2.q[tid] = expf(__fsub_rn(tau, lse_tail.hi) - lse_tail.lo);
            const float g = gumbel(uniform(seed, off, kTagSample, (int)par, (uint64_t)tid));
            const float key = __fadd_rn(tau, g);
            if (key > -INFINITY) pack = make_key(ord_f32(key), tid);
        }
        const unsigned long long bestp = block_max_u64(pack, bs);
        if (tid == 0) {
            e2.best = bestp ? (int)(0xFFFFFFFFu - (uint32_t)bestp) : 0;
            if (e2.bad) atomicOr(a.status, kStInternal);
            if (!bestp || !(e2.l[m] > -INFINITY)) atomicOr(a.status, kStEmptyRow);
            if (!(T > 0.0f) || isinf(T)) atomicOr(a.status, kStBadTemperature);
            // construction probability of Y (Sec. 3.2): min{q0(x_m), z}, never below
            // q0(x_{m+1}); m = 0: min(1, q0(x_1) + eps)
            float lp;
            if (m >= 1) {
                FF zs{0.0f, 0.0f};
                for (int i = 0; i < m; ++i) zs = ff_add(zs, expf(e2.lq0[i]));
                const FF z = ff_add(FF{1.0f, 0.0f}, ff_neg(zs));  // z = 1 - sum of the leads
                const float zf = __fadd_rn(z.hi, z.lo);
                const float lz = (zf > 0.0f) ? logf(zf) : -INFINITY;
                lp = fminf(e2.lq0[m - 1], lz);
                lp = fmaxf(lp, e2.lq0[m]);
            } else {
                const float pr = fminf(1.0f, __fadd_rn(expf(e2.lq0[0]), n.eps));
                lp = logf(pr);
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
            const int64_t q0 = ((int64_t)b * n.E + eidx) * TL;
            a.tree.tail_ids[q0 + tid] = e2.id[m + tid];
            a.tree.tail_q[q0 + tid] = e2.q[tid];
        }
        if (tid == 0) a.tree.lse1[(int64_t)b * n.E + eidx] = lse1;

        // ---- last row of the request: the K best depth-d nodes become the frontier ----
        if (!arrive_last(a.req_ticket + b, (unsigned)a.F, bs)) continue;
        if (a.d == n.D) continue;
        {
            const int nn = a.F * (K + 1);
            const int64_t base = depth_base(K, a.d);
            const bool staged = nn <= kCand;
            auto key_at = [&](int i) -> unsigned long long {
                return staged ? cand[i] : make_key(ord_f32(__ldcg(a.tree.score + nb + base + i)), base + i);
            };
            if (staged)
                for (int i = tid; i < nn; i += kThreads)
                    cand[i] = make_key(ord_f32(__ldcg(a.tree.score + nb + base + i)), base + i);
            __syncthreads();
            const unsigned long long fthr = block_radix_threshold([&](int i) { return key_at(i); }, nn, K, s_hist, s_rad);
            const int per = (nn + kThreads - 1) / kThreads;
            const int lo = min(nn, tid * per), hi = min(nn, lo + per);
            int c = 0;
            for (int i = lo; i < hi; ++i) c += key_at(i) >= fthr;
            int total;
            int pos = block_exclusive_scan(c, total, bs);
            for (int i = lo; i < hi; ++i)
                if (key_at(i) >= fthr) {
                    if (pos < K) a.tree.frontier[(int64_t)b * K + pos] = (int32_t)(base + i);
                    ++pos;
                }
            if (tid == 0 && total != K) atomicOr(a.status, kStInternal);
            __syncthreads();
        }
    }

    if (timed_out) {
        if (tid == 0) {
            atomicOr(a.status, kStTimeout);
            // let the copies still in flight land before the CTA leaves
            for (int64_t u = t; u < issued; ++u)
                mbar_wait(&full[(int)((u - t0) % kStages)], (unsigned)(((u - t0) / kStages) & 1));
        }
        __syncthreads();
    }
}

cudaError_t launch_expand(const ExpandArgs& a, int dtype, bool tma, int grid, size_t smem, cudaStream_t s) {
    auto go = [&](auto kern) {
        cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        kern<<<grid, kThreads, smem, s>>>(a);
        return cudaGetLastError();
    };
    if (dtype == 1) return tma ? go(expand_kernel<1, true>) : go(expand_kernel<1, false>);
    return tma ? go(expand_kernel<0, true>) : go(expand_kernel<0, false>);
}

size_t expand_smem_bytes(int max_segments, int support) {
    return (size_t)kStages * kTileBytes + sizeof(unsigned long long) * (kCand + (size_t)max_segments * support);
}

int expand_tile_elems(int dtype) { return kTileBytes / (dtype == 1 ? 2 : 4); }

}  // namespace rheo
