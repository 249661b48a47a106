// expand.cu -- one expansion call of the draft tree (Sec. 2.1, Sec. 3.2, App. C.1).
//
// Persistent CTAs stream the B*F draft rows in tiles of kTileBytes, each thread
// loading its four 16-byte vectors of a tile straight into registers while it
// still works on the previous tile; the warps never wait for one another while
// streaming.  Over each row segment a warp keeps
//   * a running (max, sum exp(l - max)) per thread at T = 1 (untempered, Sec. 5.4),
//   * its candidate keys (ord(logit) << 32 | ~id) in a region of shared memory:
//     every element whose key reaches theta, a lower bound of the segment's
//     S-th key.  At the first tile theta is the minimum over warps of each
//     warp's ceil(S/16)-th largest lane maximum; on every later tile one warp
//     in turn reads, off a shared two-level histogram of the keys inserted so
//     far (256 coarse bins of the top 8 key bits over 16384 fine bins of the
//     top 14), the fine bin holding the S-th key, whose lower edge becomes
//     theta.  A warp whose region fills up cuts it to its own S best keys,
//     which raises theta too.
// At the end of a segment the histogram locates the fine bin of the S-th key,
// and the keys at or above it are counting-sorted by fine bin and ranked
// within their bin.  A row held by one CTA goes straight on to
// its children; otherwise the lists and partial sums go to the workspace and
// the CTA that ends the last segment of a row (arrival counter, never a wait)
// merges them.  Then the row's sorted support gives Y from the tempered tail by
// Gumbel-max and the K+1 children; the last row of a request selects the next
// frontier.  With full support (the FULL template) each warp also sums the
// tempered terms of its 32*VEC-token groups while streaming, and the row's end
// draws Y in two Gumbel-max stages over 256-token blocks and then tokens.
#include "rheo_device.cuh"
#include "rheo_kernels.h"
#include "stream.cuh"

namespace rheo {

namespace {

constexpr int kXThreads = 512;  // one CTA of 16 warps per SM
constexpr int kXWarps = kXThreads / 32;
constexpr int kRegion = 256;    // candidate keys per warp
constexpr int kVPT = 4;         // 16-byte vectors per thread per tile
constexpr int kXTileBytes = kVPT * 16 * kXThreads;  // 32 KiB per tile
// staged vectors per warp: flushed once 32 are staged, so a list holding fewer
// than 32 always has room for a whole tile's worth
constexpr int kStageCap = 32 + 32 * kVPT;
// per-warp staging lists while streaming; the bin-ordered list of the top-S sort after
constexpr int kSpillBytes = kXWarps * kStageCap * (int)(sizeof(uint4) + sizeof(int));
// two-level histogram of candidate keys: 256 coarse bins (top 8 key bits, two
// octaves of value each) over 16384 fine bins (top 14 bits, 1/32 octave)
constexpr int kCoarseBins = 256, kCoarseShift = 56;
constexpr int kFineBins = 16384, kFineShift = 50;
constexpr int kFinePerCoarse = kFineBins / kCoarseBins;

struct E2Smem {
    unsigned long long sorted[kMaxSupport];
    int32_t id[kMaxSupport];
    float l[kMaxSupport];
    float lq0[kMaxSupport];
    float q[kMaxSupport];
    float lp;
    int best;    // sparse support: tail position of Y; full support: its support rank, or -1
    float lse1;
    int bad;
    float lse_tail;
    int yid;     // full support: the sampled token
    float qy;    // full support: q~(Y)
    float lead_sum;  // full support: the lead's group summed without the lead
};

struct HistSel {
    int bin, cbin, above, tie_n;
    int cbefore[kCoarseBins];  // keys in coarse bins above each coarse bin
};

__device__ __forceinline__ unsigned long long make_key(uint32_t k32, int64_t id) {
    return ((unsigned long long)k32 << 32) | (0xFFFFFFFFu - (uint32_t)id);
}

// Cut a warp's region down to its S best keys; returns the S-th key, a lower
// bound of the segment's S-th key.  cnt > S on entry.  The histogram loses the
// keys that go.
__device__ __noinline__ unsigned long long warp_cut_region(unsigned long long* region, int& cnt, int S,
                                                           unsigned* fine, unsigned* coarse) {
    const int lane = threadIdx.x & 31;
    unsigned long long x[kRegion / 32];
#pragma unroll
    for (int i = 0; i < kRegion / 32; ++i) {
        const int j = lane + 32 * i;
        x[i] = j < cnt ? region[j] : 0ull;
    }
    const unsigned long long thr = warp_kth_largest_of<kRegion / 32>(x, S);
    __syncwarp();
    int w = 0;
#pragma unroll
    for (int i = 0; i < kRegion / 32; ++i) {
        const bool keep = x[i] != 0ull && x[i] >= thr;
        if (x[i] != 0ull && !keep) {
            atomicSub(&fine[(unsigned)(x[i] >> kFineShift)], 1u);
            atomicSub(&coarse[(unsigned)(x[i] >> kCoarseShift)], 1u);
        }
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, keep);
        if (keep) region[w + __popc(bal & ((1u << lane) - 1u))] = x[i];
        w += __popc(bal);
    }
    __syncwarp();
    cnt = w;
    return thr;
}

// Asynchronous 4- and 8-byte copies global -> shared (no register held while
// they are in flight); cp_async_wait waits for the calling thread's copies.
__device__ __forceinline__ void cp_async(void* smem, const void* gmem, int bytes) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
    if (bytes == 8)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(sa), "l"(gmem) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Per-row values the end of a segment needs (request constants, the parent's
// gen id and path score), fetched while the row streams.
struct RowPre {
    unsigned long long seed, off;
    float T, ps;
    int par_g, stage;
};

// The tile's vectors of this thread: elements [e0 + (j*kXThreads + tid)*VEC, +VEC);
// positions at or past V read as -inf.
template <int DT, bool ALIGNED>
__device__ __forceinline__ void load_tile(uint4 (&v)[kVPT], const char* row, int e0, int V) {
    using E = Elem<DT>;
    constexpr int TE = kVPT * kXThreads * E::VEC;
    if (ALIGNED && e0 + TE <= V) {  // a whole tile: plain 16-byte loads
#pragma unroll
        for (int j = 0; j < kVPT; ++j)
            v[j] = ld_stream(row + ((int64_t)e0 + (j * kXThreads + (int)threadIdx.x) * E::VEC) * E::SIZE);
        return;
    }
#pragma unroll
    for (int j = 0; j < kVPT; ++j)
        v[j] = load_vec<DT, ALIGNED>(row, (int64_t)e0 + (j * kXThreads + (int)threadIdx.x) * E::VEC, V);
}

// Append the keys >= thr among get(i), i < n, to sel (at most cap of them);
// positions come from one shared counter, one atomic per warp and step.
template <class Get>
__device__ __forceinline__ void gather_at_least(Get get, int n, unsigned long long thr, unsigned long long* sel,
                                                int cap, int* counter) {
    const int lane = threadIdx.x & 31;
    for (int i0 = 0; i0 < n; i0 += kXThreads) {
        const int i = i0 + (int)threadIdx.x;
        const unsigned long long x = i < n ? get(i) : 0ull;
        const bool take = x != 0ull && x >= thr;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, take);
        int base = 0;
        if (lane == 0 && bal) base = atomicAdd(counter, __popc(bal));
        base = __shfl_sync(0xFFFFFFFFu, base, 0);
        const int pos = base + __popc(bal & ((1u << lane) - 1u));
        if (take && pos < cap) sel[pos] = x;
    }
}

// One warp: the fine bin holding the k-th largest key counted by the two-level
// histogram (coarse scan from the top, then the 64 fine bins of that coarse
// bin).  bin = -1 when fewer than k keys are counted; above = keys in higher
// fine bins.  Counts may change meanwhile (other warps insert or cut): a fine
// level that lags its coarse level yields the coarse bin's lowest fine bin.
__device__ __forceinline__ void warp_hist_find(const unsigned* coarse, const unsigned* fine, int k, int& bin,
                                               int& above) {
    const int lane = threadIdx.x & 31;
    int acc = 0;
    bin = -1;
    above = 0;
    for (int c0 = kCoarseBins - 1; c0 >= 0; c0 -= 32) {
        const int v = (int)*reinterpret_cast<const volatile unsigned*>(&coarse[c0 - lane]);
        int incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        const int tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
        if (acc + tot < k) {
            acc += tot;
            continue;
        }
        const int L = __ffs(__ballot_sync(0xFFFFFFFFu, acc + incl >= k)) - 1;
        const int cb = c0 - L;
        int acc2 = acc + __shfl_sync(0xFFFFFFFFu, incl - v, L);
        for (int f0 = cb * kFinePerCoarse + kFinePerCoarse - 1; f0 >= cb * kFinePerCoarse; f0 -= 32) {
            const int w = (int)*reinterpret_cast<const volatile unsigned*>(&fine[f0 - lane]);
            int inc2 = w;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, inc2, o);
                if (lane >= o) inc2 += y;
            }
            const int t2 = __shfl_sync(0xFFFFFFFFu, inc2, 31);
            if (acc2 + t2 >= k) {
                const int L2 = __ffs(__ballot_sync(0xFFFFFFFFu, acc2 + inc2 >= k)) - 1;
                bin = f0 - L2;
                above = acc2 + __shfl_sync(0xFFFFFFFFu, inc2 - w, L2);
                return;
            }
            acc2 += t2;
        }
        bin = cb * kFinePerCoarse;
        above = acc2;
        return;
    }
}

// Boundary of the k best keys counted by the two-level histogram: hs.bin = the
// fine bin holding the k-th key (-1 when fewer than k keys are counted) and
// hs.tie_n = 0.  Thread t scans coarse bin 255 - t (a block scan from the top),
// then one warp scans the 64 fine bins of the coarse bin found.
__device__ void hist_boundary(const unsigned* coarse, const unsigned* fine, int k, HistSel& hs, Red& red, int& par) {
    static_assert(kCoarseBins <= kXThreads, "one coarse bin per thread");
    const int tid = threadIdx.x, lane = tid & 31;
    const int cb = kCoarseBins - 1 - tid;  // negative: no bin
    const int c = cb >= 0 ? (int)coarse[cb] : 0;
    int total;
    const int before = red_scan<kXWarps>(c, total, red, par);
    if (cb >= 0) hs.cbefore[cb] = before;
    if (tid == 0) {
        hs.bin = -1;
        hs.tie_n = 0;
    }
    if (c > 0 && total >= k && before < k && before + c >= k) {
        hs.cbin = cb;
        hs.above = before;
    }
    __syncthreads();
    if (total >= k && tid < 32) {
        const int cbin = hs.cbin;
        int acc = hs.above;
        for (int f0 = cbin * kFinePerCoarse + kFinePerCoarse - 1; f0 >= cbin * kFinePerCoarse; f0 -= 32) {
            const int w = (int)fine[f0 - lane];
            int inc = w;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                if (lane >= o) inc += y;
            }
            const int t2 = __shfl_sync(0xFFFFFFFFu, inc, 31);
            if (acc + t2 >= k) {
                const int L2 = __ffs(__ballot_sync(0xFFFFFFFFu, acc + inc >= k)) - 1;
                const int above = acc + __shfl_sync(0xFFFFFFFFu, inc - w, L2);
                if (lane == 0) {
                    hs.bin = f0 - L2;
                    hs.above = above;  // keys in higher fine bins
                }
                break;
            }
            acc += t2;
        }
    }
    __syncthreads();
}

// The k best keys in descending order into sorted[0, k), by a counting sort on
// the fine histogram (after hist_boundary): every fine bin from the boundary bin
// up gets its offset (keys in higher bins) in place of its count, the keys of
// those bins are scattered (scatter(f): f(x) for each such key, called by all
// threads) into tmp in bin order, and each is ranked among the keys of its own
// bin.  Returns min(k, keys at or above the boundary).  The fine histogram is
// consumed.
template <class Scatter, class CoarseCount>
__device__ int hist_sort_top(Scatter scatter, CoarseCount coarse_count, int k, unsigned* fine,
                             unsigned long long* tmp, unsigned long long* sorted, HistSel& hs) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int bstar = hs.bin < 0 ? 0 : hs.bin;
    const int cstar = bstar / kFinePerCoarse;
    {
        // each warp converts the non-empty coarse bins of its lanes (lane t: coarse
        // bin 255 - t), the 64 fine bins two per lane with a warp scan, from the top
        static_assert(kFinePerCoarse == 64, "two fine bins per lane");
        const int cbl = kCoarseBins - 1 - tid;
        unsigned todo = __ballot_sync(0xFFFFFFFFu, cbl >= 0 && cbl >= cstar && coarse_count(cbl) > 0);
        while (todo) {
            const int L = __ffs(todo) - 1;
            todo &= todo - 1u;
            const int C = kCoarseBins - 1 - (warp * 32 + L);
            const int f0 = C * kFinePerCoarse + kFinePerCoarse - 1 - 2 * lane, f1 = f0 - 1;
            const int c0 = (int)fine[f0], c1 = (int)fine[f1];
            int incl = c0 + c1;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += y;
            }
            const int o0 = hs.cbefore[C] + incl - c0 - c1;
            fine[f0] = (unsigned)o0;
            fine[f1] = (unsigned)(o0 + c0);
            if (hs.bin >= 0 && f0 == bstar) hs.tie_n = o0 + c0;  // keys at or above the boundary bin
            if (hs.bin >= 0 && f1 == bstar) hs.tie_n = o0 + c0 + c1;
        }
        if (hs.bin < 0 && tid == 0) hs.tie_n = hs.cbefore[0] + coarse_count(0);  // fewer than k: all keys
    }
    __syncthreads();
    const int nsel = hs.tie_n;
    scatter([&](unsigned long long x) {
        const int f = (int)(x >> kFineShift);
        if (f >= bstar) tmp[atomicAdd(&fine[f], 1u)] = x;
    });
    __syncthreads();
    const int kk = nsel < k ? nsel : k;
    for (int p = tid; p < nsel; p += kXThreads) {
        const unsigned long long x = tmp[p];
        const int f = (int)(x >> kFineShift);
        const int start = (f % kFinePerCoarse == kFinePerCoarse - 1) ? hs.cbefore[f / kFinePerCoarse] : (int)fine[f + 1];
        const int end = (int)fine[f];
        int rank = start;
        for (int q = start; q < end; ++q) rank += tmp[q] > x;
        if (rank < kk) sorted[rank] = x;
    }
    __syncthreads();
    return kk;
}

// Block-wide: append the keys with fine bin >= bin among get(i), i < n.
template <class Get>
__device__ __forceinline__ void block_gather_bin(Get get, int n, int bin, unsigned long long* tmp, int cap,
                                                 HistSel& hs) {
    const int lane = threadIdx.x & 31;
    for (int i0 = 0; i0 < n; i0 += kXThreads) {
        const int i = i0 + (int)threadIdx.x;
        const unsigned long long x = i < n ? get(i) : 0ull;
        const bool take = x != 0ull && (int)(x >> kFineShift) >= bin;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, take);
        int base = 0;
        if (lane == 0 && bal) base = atomicAdd(&hs.tie_n, __popc(bal));
        base = __shfl_sync(0xFFFFFFFFu, base, 0);
        const int pos = base + __popc(bal & ((1u << lane) - 1u));
        if (take && pos < cap) tmp[pos] = x;
    }
}

// The gathered keys tmp[0, hs.tie_n) ranked: the k best in descending order into
// sorted[0, k); returns how many (min(k, gathered)).  Two threads rank each key.
__device__ int rank_gathered(const unsigned long long* tmp, int k, unsigned long long* sorted, HistSel& hs) {
    __syncthreads();
    const int nsel = hs.tie_n;
    const int kk = nsel < k ? nsel : k;
    for (int p0 = 0; p0 < nsel; p0 += kXThreads / 2) {
        const int p = p0 + ((int)threadIdx.x >> 1), h = threadIdx.x & 1;
        const unsigned long long x = p < nsel ? tmp[p] : 0ull;
        int rank = 0;
        if (p < nsel) {
            int r0 = 0, r1 = 0;
            int q = h;
            for (; q + 2 < nsel; q += 4) {
                r0 += tmp[q] > x;
                r1 += tmp[q + 2] > x;
            }
            for (; q < nsel; q += 2) r0 += tmp[q] > x;
            rank = r0 + r1;
        }
        rank += __shfl_xor_sync(0xFFFFFFFFu, rank, 1);
        if (p < nsel && h == 0 && rank < kk) sorted[rank] = x;
    }
    __syncthreads();
    return kk;
}

// Slow insertion path (pend: this lane's element bits of its vector vv, whose
// first element is eidx): one candidate per lane and round, keys below theta
// dropped, the region cut to its S best whenever it fills.
template <int DT>
__device__ __forceinline__ void insert_rounds(unsigned long long* region, int& cnt, uint32_t pend, uint4 vv, int eidx,
                                           unsigned long long& theta, int S, unsigned* fine, unsigned* coarse,
                                           unsigned long long* s_theta) {
    using E = Elem<DT>;
    const int lane = threadIdx.x & 31;
    while (__any_sync(0xFFFFFFFFu, pend != 0u)) {
        if (cnt > kRegion - 32) {
            const unsigned long long thr = warp_cut_region(region, cnt, S, fine, coarse);
            if (lane == 0) atomicMax(s_theta, thr);
            theta = thr > theta ? thr : theta;
        }
        unsigned long long x = 0ull;
        if (pend) {
            const int i = __ffs(pend) - 1;
            pend &= pend - 1u;
            x = make_key(E::key(E::raw(vv, i)), (int64_t)eidx + i);
            if (x < theta) x = 0ull;
        }
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, x != 0ull);
        if (x) {
            region[cnt + __popc(bal & ((1u << lane) - 1u))] = x;
            atomicAdd(&fine[(unsigned)(x >> kFineShift)], 1u);
            atomicAdd(&coarse[(unsigned)(x >> kCoarseShift)], 1u);
        }
        cnt += __popc(bal);
    }
}

// One warp inserts its staged vectors (sv[0, n), first elements si[]) into its
// candidate region: every element at or above theta (as it stands now) of
// the row's first V elements becomes a key, counted in both histograms; one
// vector per lane and round.
template <int DT>
__device__ __forceinline__ void stage_flush(unsigned long long* region, int& cnt, const uint4* sv, const int* si, int n,
                                         int V, unsigned long long& theta, int S, unsigned* fine, unsigned* coarse,
                                         unsigned long long* s_theta) {
    using E = Elem<DT>;
    using W = Vec<DT>;
    constexpr int VEC = E::VEC;
    const int lane = threadIdx.x & 31;
    for (int k0 = 0; k0 < n; k0 += 32) {
        const float thv = E::threshold_value((uint32_t)(theta >> 32));
        const uint32_t t2 = (DT == 0) ? __float_as_uint(thv)
                                      : ((__float_as_uint(thv) >> 16) | (__float_as_uint(thv) & 0xFFFF0000u));
        const int k = k0 + lane;
        uint4 vv = make_uint4(0u, 0u, 0u, 0u);
        int eidx = 0;
        uint32_t pend = 0u;
        if (k < n) {
            vv = sv[k];
            eidx = si[k];
            pend = W::ge_bits(vv, t2);
            const int left = V - eidx;  // elements of this vector inside the row
            if (left < VEC) pend &= (left > 0) ? ((1u << left) - 1u) : 0u;
        }
        const int c = __popc(pend);
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        const int total = __shfl_sync(0xFFFFFFFFu, incl, 31);
        if (cnt + total <= kRegion) {
            int pos = cnt + incl - c;
            for (uint32_t mm = pend; mm; mm &= mm - 1u) {
                const int i = __ffs(mm) - 1;
                const unsigned long long x = make_key(E::key(E::raw(vv, i)), (int64_t)eidx + i);
                region[pos++] = x;
                atomicAdd(&fine[(unsigned)(x >> kFineShift)], 1u);
                atomicAdd(&coarse[(unsigned)(x >> kCoarseShift)], 1u);
            }
            cnt += total;
        } else {
            insert_rounds<DT>(region, cnt, pend, vv, eidx, theta, S, fine, coarse, s_theta);
        }
    }
    __syncwarp();
}

}  // namespace

// Full support: the block of the two-stage draw of Y (token ids per block)
constexpr int kFullBlock = 256;

template <int DT, bool ALIGNED, bool FULL>
__global__ void __launch_bounds__(kXThreads, 1) expand_kernel(const ExpandArgs a) {
    grid_dependency_begin();
    using E = Elem<DT>;
    using W = Vec<DT>;
    constexpr int VEC = E::VEC;
    constexpr int TE = kXTileBytes / E::SIZE;  // elements per tile
    static_assert(TE == kVPT * VEC * kXThreads, "tile layout");
    constexpr float kLog2e = 1.4426950408889634f;
    extern __shared__ __align__(128) unsigned char dsm[];
    // per-warp candidate regions; after a segment's selection the same space
    // holds the merge keys of a row and the frontier candidates of a request
    unsigned long long* keys = reinterpret_cast<unsigned long long*>(dsm);
    // per-warp copy of the lanes' vectors of a tile that has candidates
    uint4* spill = reinterpret_cast<uint4*>(dsm + a.keys_bytes);
    unsigned* fine = reinterpret_cast<unsigned*>(dsm + a.keys_bytes + kSpillBytes);
    unsigned* coarse = fine + kFineBins;
    // the spill area doubles as the bin-ordered list of the top-S sort
    unsigned long long* tmpk = reinterpret_cast<unsigned long long*>(spill);
    constexpr int kTmpCap = kSpillBytes / (int)sizeof(unsigned long long);
    __shared__ unsigned long long s_theta;
    __shared__ uint32_t s_wb[kXWarps];
    __shared__ int s_rcount[kXWarps];
    __shared__ BlockScratch bs;
    __shared__ Red red;
    __shared__ E2Smem e2;
    __shared__ HistSel hs;
    __shared__ unsigned s_hist[kRadixBins];
    __shared__ SelScratch s_sel;
    __shared__ RowPre s_pre;

    const Dims& n = a.n;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int V = n.V, S = n.S, K = n.K, m = n.m, TL = n.TL;
    const int tpr = (V + TE - 1) / TE;
    const int kb = (S + kXWarps - 1) / kXWarps;  // per-warp share of S in the bounds
    const TileSplit sp{(int64_t)n.B * a.F * tpr, (int)gridDim.x};
    const int64_t t0 = sp.begin(blockIdx.x), t1 = sp.begin(blockIdx.x + 1);
    unsigned long long* region = keys + warp * kRegion;
    // per-warp staging list of vectors holding candidates (in the spill area)
    static_assert(kXWarps * kStageCap * (sizeof(uint4) + sizeof(int)) <= kSpillBytes, "staging fits the spill area");
    uint4* stage_v = spill + warp * kStageCap;
    int* stage_i = reinterpret_cast<int*>(spill + kXWarps * kStageCap) + warp * kStageCap;
    int scnt = 0;  // staged vectors of this warp (warp-uniform)
    int par = 0;

    if (tid == 0) s_theta = 0ull;

    // per-segment state; cnt, theta and seg_valid are warp-uniform
    float mu = -INFINITY;
    unsigned long long sum2 = 0ull;  // the running sum as a pair of fp32 partial sums
    float fT = 1.0f;  // full support: the row's temperature
    unsigned long long theta = 0ull;
    int cnt = 0, seg_tiles = 0;
    int64_t seg_valid = 0;

    // tid 0 starts the copies of the row's constants and, on the second tile, of
    // its parent's score (which needs the parent's gen id from the frontier)
    auto prefetch_row = [&](int64_t r) {
        if (tid != 0) return;
        const int b = (int)(r / a.F), f = (int)(r % a.F);
        cp_async(&s_pre.T, a.T + b, 4);
        cp_async(&s_pre.seed, a.seed + b, 8);
        cp_async(&s_pre.off, a.offset + b, 8);
        if (a.d > 1) {
            cp_async(&s_pre.par_g, a.tree.frontier + (int64_t)b * K + f, 4);
            s_pre.stage = 1;
        } else {  // the root: nothing to fetch
            s_pre.par_g = 0;
            s_pre.ps = 0.0f;
            s_pre.stage = 0;
        }
    };
    auto prefetch_parent = [&](int64_t r) {  // tid 0, after the frontier entry arrived
        cp_async_wait();
        if (s_pre.stage != 1) return;
        const int b = (int)(r / a.F);
        const int pg = s_pre.par_g;
        s_pre.stage = 2;
        if (pg >= 0 && pg < n.G1)
            cp_async(&s_pre.ps, a.tree.score + (int64_t)b * n.G1 + pg, 4);
        else
            s_pre.ps = 0.0f;  // reported as an internal error at the segment's end
    };
    auto seg_begin = [&](int64_t r) {
        mu = -INFINITY;
        sum2 = 0ull;
        if constexpr (FULL) fT = __ldg(a.T + r / a.F);
        seg_valid = 0;
        cnt = 0;
        for (int i = tid; i < (kFineBins + kCoarseBins) / 4; i += kXThreads)
            reinterpret_cast<uint4*>(fine)[i] = make_uint4(0u, 0u, 0u, 0u);
    };
    // running partition sum at T = 1 (online max); mu is also the running
    // maximum of this thread's elements
    auto tile_sum = [&](const uint4 (&v)[kVPT], float (&vm)[kVPT]) {
#pragma unroll
        for (int j = 0; j < kVPT; ++j) vm[j] = W::vmax(v[j]);
        float tmax = vm[0];
#pragma unroll
        for (int j = 1; j < kVPT; ++j) tmax = fmaxf(tmax, vm[j]);
        if (tmax > mu) {
            if (mu != -INFINITY) {
                const float rs = fast_exp2((mu - tmax) * kLog2e);
                sum2 = f2_mul(sum2, f2_pack(rs, rs));
            }
            mu = tmax;
        }
        if (mu != -INFINITY) {
            const float mc = mu * kLog2e;
            const unsigned long long c2 = f2_pack(kLog2e, kLog2e), n2 = f2_pack(-mc, -mc);
            unsigned long long t = W::vexp2(v[0], c2, n2);
#pragma unroll
            for (int j = 1; j < kVPT; ++j) t = f2_add(t, W::vexp2(v[j], c2, n2));
            sum2 = f2_add(sum2, t);
        }
    };
    // full support, per warp and vector row of a tile: the warp holds a group
    // of 32*VEC consecutive token ids; its tempered sum at the group's own
    // maximum (the reference) goes to the workspace for the row end's two-stage
    // draw of Y.  tau = l/T to within an ulp: q = l*(1/T) corrected by one
    // residual step (Markstein, IBM J. Res. Dev. 34(1), 1990); an infinite l
    // gives NaN, which the exponent's clamp turns into a zero term.
    auto tile_full = [&](const uint4 (&v)[kVPT], const float (&vm)[kVPT], int e0, int64_t r) {
        constexpr int GS = 32 * VEC;
        const int gpr = (V + GS - 1) / GS;
        const float rT = 1.0f / fT;
#pragma unroll
        for (int j = 0; j < kVPT; ++j) {
            const int g0 = e0 + (j * kXThreads + warp * 32) * VEC;  // the group's first token
            const float gmax = Elem<0>::value_of_key(__reduce_max_sync(0xFFFFFFFFu, ord_f32(vm[j])));
            const float ref = gmax * rT;
            const float nref = (ref > -INFINITY && ref < INFINITY) ? -ref * kLog2e : -INFINITY;
            float sg;
            if constexpr (DT == 1) {
                // bf16 pairs in packed fp32 (each lane rounded as the scalar
                // ops); -inf clamped to -1e30 first (bf16 0xF149), so every
                // step stays finite and its term is 0
                const unsigned long long rT2 = f2_pack(rT, rT), nT2 = f2_pack(-fT, -fT);
                const unsigned long long c2 = f2_pack(kLog2e, kLog2e), nr2 = f2_pack(nref, nref);
                const uint32_t wv[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
                unsigned long long acc = f2_pack(0.0f, 0.0f);
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    const uint32_t wc = bmax2(wv[h], 0xF149F149u);
                    const unsigned long long x2 = f2_pack(bf_lo(wc), bf_hi(wc));
                    const unsigned long long q2 = f2_mul(x2, rT2);
                    const unsigned long long t2 = f2_fma(f2_fma(q2, nT2, x2), rT2, q2);
                    acc = f2_add(acc, f2_exp2(f2_fma(t2, c2, nr2)));
                }
                sg = f2_fold(acc);
            } else {
                float s0 = 0.0f, s1 = 0.0f;
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    const float x = E::value(E::raw(v[j], i));
                    const float q0 = x * rT;
                    const float tq = fmaf(fmaf(-q0, fT, x), rT, q0);
                    const float tv = fast_exp2(fmaxf(fmaf(tq, kLog2e, nref), -200.0f));
                    if (i & 1) s1 += tv; else s0 += tv;
                }
                sg = s0 + s1;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sg += __shfl_xor_sync(0xFFFFFFFFu, sg, o);
            if (lane == 0 && g0 < V) {
                const int64_t q = r * gpr + g0 / GS;
                a.grp[2 * q] = ref;
                a.grp[2 * q + 1] = sg;
            }
        }
    };
    // The bound theta.  On the first step of a segment: every warp's kb-th
    // largest running maximum of its lanes (lanes with no element count as
    // absent) -- kb lanes hold an element at or above it, so at least S elements
    // reach the smallest of those bounds; the block synchronises on it.  On every
    // later step one warp in turn finds, in the histogram of the candidates so
    // far, the fine bin of the S-th key: at least S elements lie at or above
    // that bin's lower edge, which becomes the shared bound.
    auto refresh = [&](bool seg_first) {
        seg_tiles = seg_first ? 1 : seg_tiles + 1;
        if (seg_first) {
            const uint32_t lk = (mu > -INFINITY) ? E::key_of_value(mu) : 0u;
            int rank = 0;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const uint32_t y = __shfl_sync(0xFFFFFFFFu, lk, j);
                rank += (y > lk || (y == lk && j < lane)) ? 1 : 0;
            }
            const unsigned who = __ballot_sync(0xFFFFFFFFu, rank == kb - 1);
            const uint32_t wb = __shfl_sync(0xFFFFFFFFu, lk, __ffs(who) - 1);
            if (lane == 0) s_wb[warp] = wb;
            __syncthreads();
            uint32_t b = s_wb[0];
#pragma unroll
            for (int w = 1; w < kXWarps; ++w) b = min(b, s_wb[w]);
            theta = (unsigned long long)b << 32;
        } else if (seg_tiles % kXWarps == warp) {
            int bin, above;
            warp_hist_find(coarse, fine, S, bin, above);
            if (bin >= 0) {
                const unsigned long long hb = (unsigned long long)bin << kFineShift;
                if (lane == 0) atomicMax(&s_theta, hb);
                theta = hb > theta ? hb : theta;
            }
        }
        const unsigned long long ts = *reinterpret_cast<volatile unsigned long long*>(&s_theta);
        theta = ts > theta ? ts : theta;
    };
    // candidates of one tile: elements whose value reaches theta's (a superset
    // of the keys >= theta; the final selection is exact).  Every lane writes its
    // own at offsets from a warp scan.
    auto tile_candidates = [&](const uint4 (&v)[kVPT], const float (&vm)[kVPT], int e0) {
        const float thv = E::threshold_value((uint32_t)(theta >> 32));
        // a vector whose maximum reaches theta is staged as it is (its elements
        // are screened when the list is flushed): a vote per vector row of the
        // tile, one store per staged vector
        unsigned bal[kVPT];
        int total = 0;
#pragma unroll
        for (int j = 0; j < kVPT; ++j) {
            bal[j] = __ballot_sync(0xFFFFFFFFu, vm[j] >= thv);
            total += __popc(bal[j]);
        }
        if (total == 0) return;
#pragma unroll
        for (int j = 0; j < kVPT; ++j) {
            if ((bal[j] >> lane) & 1u) {
                const int p = scnt + __popc(bal[j] & ((1u << lane) - 1u));
                stage_v[p] = v[j];
                stage_i[p] = e0 + (j * kXThreads + tid) * VEC;
            }
            scnt += __popc(bal[j]);
        }
        if (scnt >= 32) {  // a full round of one vector per lane
            __syncwarp();
            stage_flush<DT>(region, cnt, stage_v, stage_i, scnt, V, theta, S, fine, coarse, &s_theta);
            scnt = 0;
        }
    };
    // end of the segment of row r that this CTA holds
    auto segment_end = [&](int64_t r) {
        // ---- end of segment: exact top-S keys ------------------------------------
        if (tid == 0) {  // the row's constants have landed (or land now)
            prefetch_parent(r);
            cp_async_wait();
        }
        if (scnt > 0) stage_flush<DT>(region, cnt, stage_v, stage_i, scnt, V, theta, S, fine, coarse, &s_theta);
        scnt = 0;
        if (lane == 0) s_rcount[warp] = cnt;
        float Ms;
        const FF Ss = red_partition<kXWarps>(mu, f2_fold(sum2), kLog2e, Ms, red, par);  // its barrier also publishes the counts
        if (tid == 0) s_theta = 0ull;  // every warp is past its last cut: ready for the next segment
        const int target = (int)min((int64_t)S, seg_valid);
        auto rkey = [&](int i) -> unsigned long long {
            return (i % kRegion) < s_rcount[i / kRegion] ? keys[i] : 0ull;
        };
        // the k best: all keys at or above the fine bin of the k-th, ranked
        hist_boundary(coarse, fine, target, hs, red, par);
        int written;
        if (hs.bin < 0 || hs.above + (int)fine[hs.bin] <= kTmpCap) {
            written = hist_sort_top(
                [&](auto put) {
                    for (int j = lane; j < cnt; j += 32) put(region[j]);
                },
                [&](int c) { return coarse[c]; }, target, fine, tmpk, e2.sorted, hs);
        } else {  // a tie class too large for the list
            const unsigned long long thr = block_kth_key<kXThreads>(rkey, kXWarps * kRegion, target, s_hist, s_sel);
            if (tid == 0) hs.tie_n = 0;
            __syncthreads();
            gather_at_least(rkey, kXWarps * kRegion, thr, tmpk, target, &hs.tie_n);
            written = rank_gathered(tmpk, target, e2.sorted, hs);
        }
        const int first_owner = sp.owner(r * tpr);
        const int seg = (int)blockIdx.x - first_owner;
        const int nseg = sp.owner(r * tpr + tpr - 1) - first_owner + 1;
        const int b = (int)(r / a.F), f = (int)(r % a.F);
        if (tid == 0) {
            if (isnan(Ss.hi) || Ms == INFINITY) atomicOr(a.status, kStBadLogit);
            if (written != target) atomicOr(a.status, kStInternal);
        }
        if (nseg == 1) {
            // the whole row is here: its support is e2.sorted, its partition sum Ss
            if (tid == 0) {
                const FF l = ff_add(ff_log(Ss), Ms);
                e2.lse1 = __fadd_rn(l.hi, l.lo);
                e2.bad = (written != S) ? 1 : 0;
            }
        } else {
            unsigned long long* out = a.seg_keys + ((int64_t)r * tpr + seg) * S;
            for (int i = tid; i < S; i += kXThreads) out[i] = i < written ? e2.sorted[i] : 0ull;
            if (tid == 0) {
                a.seg_mu[(int64_t)r * tpr + seg] = Ms;
                a.seg_sum[2 * ((int64_t)r * tpr + seg)] = Ss.hi;
                a.seg_sum[2 * ((int64_t)r * tpr + seg) + 1] = Ss.lo;
            }
            if (!arrive_last(a.row_ticket + r, (unsigned)nseg, bs)) return;

            // ---- last segment of row r: merge the segments' lists and sums ---------
            const int nkeys = nseg * S;
            const unsigned long long* rk = a.seg_keys + (int64_t)r * tpr * S;
            for (int i = tid; i < (kFineBins + kCoarseBins) / 4; i += kXThreads)
                reinterpret_cast<uint4*>(fine)[i] = make_uint4(0u, 0u, 0u, 0u);
            __syncthreads();
            for (int i = tid; i < nkeys; i += kXThreads) {
                const unsigned long long x = __ldcg(rk + i);
                keys[i] = x;
                if (x) {
                    atomicAdd(&fine[(unsigned)(x >> kFineShift)], 1u);
                    atomicAdd(&coarse[(unsigned)(x >> kCoarseShift)], 1u);
                }
            }
            __syncthreads();
            auto mkey = [&](int i) { return keys[i]; };
            hist_boundary(coarse, fine, S, hs, red, par);
            int got;
            if (hs.bin < 0 || hs.above + (int)fine[hs.bin] <= kTmpCap) {
                got = hist_sort_top(
                    [&](auto put) {
                        for (int i = tid; i < nkeys; i += kXThreads)
                            if (keys[i]) put(keys[i]);
                    },
                    [&](int c) { return coarse[c]; }, S, fine, tmpk, e2.sorted, hs);
            } else {
                const unsigned long long thr = block_kth_key<kXThreads>(mkey, nkeys, S, s_hist, s_sel);
                if (tid == 0) hs.tie_n = 0;
                __syncthreads();
                gather_at_least(mkey, nkeys, thr, tmpk, S, &hs.tie_n);
                got = rank_gathered(tmpk, S, e2.sorted, hs);
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
                }
            }
            __syncthreads();
            if (tid == 0) e2.bad = (got != S) ? 1 : 0;
        }
        __syncthreads();
        const float lse1 = e2.lse1;
        if (tid < S) {  // read by others only after the next barrier
            const unsigned long long x = e2.sorted[tid];
            e2.id[tid] = (int32_t)(0xFFFFFFFFu - (uint32_t)x);
            const float l = E::value_of_key((uint32_t)(x >> 32));
            e2.l[tid] = l;
            e2.lq0[tid] = __fsub_rn(l, lse1);
        }

        const float T = s_pre.T;
        const uint64_t seed = s_pre.seed, off = s_pre.off;
        const int64_t nb = (int64_t)b * n.G1;
        int64_t par_g = s_pre.par_g;
        if (par_g < 0 || par_g >= n.G1) {  // frontier never written for this tree
            if (tid == 0) atomicOr(a.status, kStInternal);
            par_g = 0;
        }
        const int64_t eidx = (a.d == 1) ? 0 : 1 + (int64_t)(a.d - 2) * K + f;
        const int64_t g0 = depth_base(K, a.d) + (int64_t)f * (K + 1);

        if constexpr (!FULL) {
            // tempered tail q~ = softmax(l / T) over support ranks m+1..S; Y by
            // Gumbel-max (the key needs no partition sum: one reduction for both)
            auto lof = [&](int i) { return E::value_of_key((uint32_t)(e2.sorted[i] >> 32)); };
            const float tau = (tid < TL) ? __fdiv_rn(lof(m + tid), T) : -INFINITY;
            const float mt = __fdiv_rn(lof(m), T);  // the support is sorted: rank m is the tail's maximum
            unsigned long long pack = 0ull;
            if (tid < TL) {
                const float g = gumbel(uniform(seed, off, kTagSample, (int)par_g, (uint64_t)tid));
                const float key = __fadd_rn(tau, g);
                if (key > -INFINITY) pack = make_key(ord_f32(key), tid);
            }
            FF st;
            unsigned long long bestp;
            red_sum_ff_max_u64<kXWarps>(FF{(tid < TL && mt > -INFINITY) ? expf(tau - mt) : 0.0f, 0.0f}, pack, red, par,
                                        st, bestp);
            const FF lse_tail = ff_add(ff_log(st), mt);
            if (tid < TL) e2.q[tid] = expf(__fsub_rn(tau, lse_tail.hi) - lse_tail.lo);
            if (tid == 0) {
                e2.best = bestp ? (int)(0xFFFFFFFFu - (uint32_t)bestp) : 0;
                e2.lse_tail = __fadd_rn(lse_tail.hi, lse_tail.lo);
                if (!bestp) atomicOr(a.status, kStEmptyRow);
            }
        } else {
            // full support: Y in two stages, each a Gumbel-max (exact: P(block) =
            // its mass / the tail's, then P(Y | block) = q~ / the block's mass):
            // a block of kFullBlock consecutive token ids by its tempered
            // log-mass fp32(reference + log sum) + g (draw V + block; ties keep
            // the lower block), then a token of that block by tau + g (tau
            // correctly rounded, draw = token id; ties keep the lower id).  The
            // masses come from the groups' sums written while streaming; the
            // lead's group (m = 1) is summed again without the lead.  The same
            // sums give the tail's partition.
            constexpr int GS = 32 * VEC;
            constexpr int GPB = kFullBlock / GS;
            static_assert(kFullBlock % GS == 0 && kFullBlock <= kXThreads, "groups tile a block");
            const int gpr = (V + GS - 1) / GS;
            const int nblk = (V + kFullBlock - 1) / kFullBlock;
            const float* grp = a.grp + 2 * r * gpr;
            const char* rowp = a.logits + r * a.row_stride_bytes;
            const float rT = 1.0f / T;
            __syncthreads();  // the support's ids are published
            const int lead_id = (m == 1) ? e2.id[0] : -1;
            const int lead_g = (lead_id >= 0) ? lead_id / GS : -1;
            if (warp == 0) {
                float sg = 0.0f;
                if (lead_g >= 0) {
                    const float ref = __ldcg(grp + 2 * lead_g);
                    const float nref = (ref > -INFINITY && ref < INFINITY) ? -ref * kLog2e : -INFINITY;
                    const int e = lead_g * GS + lane * VEC;
                    const uint4 vv = load_vec<DT, ALIGNED>(rowp, e, V);
#pragma unroll
                    for (int i = 0; i < VEC; ++i) {
                        if (e + i == lead_id) continue;
                        const float x = E::value(E::raw(vv, i));
                        const float q0 = x * rT;
                        const float tq = fmaf(fmaf(-q0, T, x), rT, q0);
                        sg += fast_exp2(fmaxf(fmaf(tq, kLog2e, nref), -200.0f));
                    }
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) sg += __shfl_xor_sync(0xFFFFFFFFu, sg, o);
                if (lane == 0) e2.lead_sum = sg;
            }
            __syncthreads();
            // this thread's blocks: the tail's partition (at this thread's
            // largest group reference) and the best block key
            float mth = -INFINITY, sth = 0.0f;
            unsigned long long kb = 0ull;
            for (int k = tid; k < nblk; k += kXThreads) {
                float rf[GPB], sm[GPB];
                float rm = -INFINITY;
#pragma unroll
                for (int q = 0; q < GPB; ++q) {
                    const int gi = k * GPB + q;
                    rf[q] = -INFINITY;
                    sm[q] = 0.0f;
                    if (gi < gpr) {
                        rf[q] = __ldcg(grp + 2 * gi);
                        sm[q] = (gi == lead_g) ? e2.lead_sum : __ldcg(grp + 2 * gi + 1);
                        if (sm[q] > 0.0f) rm = fmaxf(rm, rf[q]);
                    }
                }
                if (!(rm > -INFINITY)) continue;  // no mass in this block
                float bs = 0.0f;
#pragma unroll
                for (int q = 0; q < GPB; ++q)
                    if (sm[q] > 0.0f) bs += sm[q] * fast_exp2((rf[q] - rm) * kLog2e);
                if (rm > mth) {
                    sth = sth * fast_exp2((mth - rm) * kLog2e) + bs;
                    mth = rm;
                } else {
                    sth += bs * fast_exp2((rm - mth) * kLog2e);
                }
                const float lm = __fadd_rn(rm, logf(bs));
                const float key = __fadd_rn(lm, gumbel(uniform(seed, off, kTagSample, (int)par_g, (uint64_t)V + k)));
                if (key > -INFINITY) {
                    const unsigned long long pk = make_key(ord_f32(key), k);
                    kb = pk > kb ? pk : kb;
                }
            }
            float MT;
            const FF ST = red_partition<kXWarps>(mth, sth, kLog2e, MT, red, par);
            const unsigned long long bkey = red_max_u64<kXWarps>(kb, red, par);
            const int blk = bkey ? (int)(0xFFFFFFFFu - (uint32_t)bkey) : -1;
            unsigned long long tk = 0ull;
            if (blk >= 0 && tid < kFullBlock) {
                const int id = blk * kFullBlock + tid;
                if (id < V && id != lead_id) {
                    const float tau = __fdiv_rn(E::value(E::load_scalar(rowp, id)), T);
                    const float key = __fadd_rn(tau, gumbel(uniform(seed, off, kTagSample, (int)par_g, (uint64_t)id)));
                    if (key > -INFINITY) tk = make_key(ord_f32(key), id);
                }
            }
            const unsigned long long ykey = red_max_u64<kXWarps>(tk, red, par);
            if (tid == 0) {
                const int yid = ykey ? (int)(0xFFFFFFFFu - (uint32_t)ykey) : -1;
                const FF lse_tail = ff_add(ff_log(ST), MT);
                e2.lse_tail = __fadd_rn(lse_tail.hi, lse_tail.lo);
                const int64_t ei = (a.d == 1) ? 0 : 1 + (int64_t)(a.d - 2) * K + f;
                a.lse_tail_ff[2 * ((int64_t)b * n.E + ei)] = lse_tail.hi;
                a.lse_tail_ff[2 * ((int64_t)b * n.E + ei) + 1] = lse_tail.lo;
                e2.yid = yid;
                e2.best = -1;
                e2.qy = 0.0f;
                if (yid < 0) {
                    atomicOr(a.status, kStEmptyRow);
                } else {
                    const float tauy = __fdiv_rn(E::value(E::load_scalar(rowp, yid)), T);
                    e2.qy = expf(__fsub_rn(tauy, lse_tail.hi) - lse_tail.lo);
                    for (int j = m; j < S; ++j)
                        if (e2.id[j] == yid) e2.best = j;
                }
            }
        }
        if (tid == 0) {
            if (e2.bad) atomicOr(a.status, kStInternal);
            if (!(e2.l[m] > -INFINITY)) atomicOr(a.status, kStEmptyRow);
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
            int rank, tok;
            float lpj, qv = 0.0f;
            uint8_t st8;
            if (j < m) {
                rank = j; lpj = e2.lq0[j]; st8 = kSlotLead;
                tok = e2.id[rank];
            } else if (j == m) {
                lpj = e2.lp; st8 = kSlotSampled;
                if constexpr (FULL) {
                    tok = e2.yid; qv = e2.qy;
                } else {
                    rank = m + best; qv = e2.q[best]; tok = e2.id[rank];
                }
            } else {
                const int qf = j - m - 1;
                if constexpr (FULL)
                    rank = m + qf + ((best >= 0 && m + qf >= best) ? 1 : 0);
                else
                    rank = m + qf + (qf >= best ? 1 : 0);
                lpj = e2.lq0[rank]; st8 = kSlotFill;
                tok = e2.id[rank];
            }
            const float ps = s_pre.ps;
            const int64_t g = nb + g0 + j;
            a.tree.token[g] = tok;
            a.tree.parent[g] = (int32_t)par_g;
            a.tree.log_proxy[g] = lpj;
            a.tree.score[g] = __fadd_rn(ps, lpj);
            a.tree.qtilde[g] = qv;
            a.tree.slot[g] = st8;
        }
        // ---- last row of the request: the K best depth-d nodes become the frontier ----
        // (the arrival waits only for the children's writes: the tail lists, read
        // by no one before verification, are written after it)
        const bool last_row = arrive_last(a.req_ticket + b, (unsigned)a.F, bs);
        if (tid < TL) {
            const int64_t q0 = ((int64_t)b * n.E + eidx) * TL;
            a.tree.tail_ids[q0 + tid] = e2.id[m + tid];
            a.tree.tail_q[q0 + tid] = e2.q[tid];
        }
        if (tid == 0) {
            a.tree.lse1[(int64_t)b * n.E + eidx] = lse1;
            if (a.tree.lse_tail) a.tree.lse_tail[(int64_t)b * n.E + eidx] = e2.lse_tail;
        }
        if (!last_row) return;
        if (a.d == n.D) return;
        {
            const int nn = a.F * (K + 1);
            const int64_t base = depth_base(K, a.d);
            if (nn <= kXThreads) {
                // rank of every candidate; the K best, written in gen-id order
                const unsigned long long x =
                    tid < nn ? make_key(ord_f32(__ldcg(a.tree.score + nb + base + tid)), base + tid) : 0ull;
                if (tid < nn) keys[tid] = x;
                __syncthreads();
                int rank = 0;
                if (tid < nn)
                    for (int j = 0; j < nn; ++j) rank += keys[j] > x;
                const bool take = tid < nn && rank < K;
                int total;
                const int pos = red_scan<kXWarps>(take ? 1 : 0, total, red, par);
                if (take && pos < K) a.tree.frontier[(int64_t)b * K + pos] = (int32_t)(base + tid);
                if (tid == 0 && total != K) atomicOr(a.status, kStInternal);
            } else {
                auto key_at = [&](int i) -> unsigned long long {
                    return make_key(ord_f32(__ldcg(a.tree.score + nb + base + i)), base + i);
                };
                const unsigned long long fthr = block_kth_key<kXThreads>(key_at, nn, K, s_hist, s_sel);
                const int per = (nn + kXThreads - 1) / kXThreads;
                const int lo = min(nn, tid * per), hi = min(nn, lo + per);
                int c = 0;
                for (int i = lo; i < hi; ++i) c += key_at(i) >= fthr;
                int total;
                int pos = red_scan<kXWarps>(c, total, red, par);
                for (int i = lo; i < hi; ++i)
                    if (key_at(i) >= fthr) {
                        if (pos < K) a.tree.frontier[(int64_t)b * K + pos] = (int32_t)(base + i);
                        ++pos;
                    }
                if (tid == 0 && total != K) atomicOr(a.status, kStInternal);
            }
            __syncthreads();
        }
    };

    {
        // the CTA's tiles in order; segments end at row boundaries
        int64_t r = t0 / tpr;
        int tt = (int)(t0 % tpr);
        uint4 nxt[kVPT];
        if (t0 < t1) load_tile<DT, ALIGNED>(nxt, a.logits + r * a.row_stride_bytes, tt * TE, V);
        for (int64_t t = t0; t < t1; ++t, ++tt) {
            if (tt == tpr) {
                tt = 0;
                ++r;
            }
            const bool seg_first = (t == t0) || (tt == 0);
            const bool seg_last = (t == t1 - 1) || (tt == tpr - 1);
            const int e0 = tt * TE;
            const int ne = min(TE, V - e0);
            uint4 v[kVPT];
#pragma unroll
            for (int j = 0; j < kVPT; ++j) v[j] = nxt[j];
            if (t + 1 < t1) {  // the next tile is in flight while this one is worked on
                const bool wrap = (tt + 1 == tpr);
                load_tile<DT, ALIGNED>(nxt, a.logits + (r + (wrap ? 1 : 0)) * a.row_stride_bytes, wrap ? 0 : e0 + TE, V);
            }
            if (seg_first) {
                prefetch_row(r);
                seg_begin(r);
            } else if (tid == 0 && s_pre.stage == 1) {
                prefetch_parent(r);
            }
            float vm[kVPT];
            tile_sum(v, vm);
            if constexpr (FULL) tile_full(v, vm, e0, r);
            refresh(seg_first);
            seg_valid += ne;
            tile_candidates(v, vm, e0);
            if (seg_last) segment_end(r);
        }
    }
}

cudaError_t launch_expand(const ExpandArgs& a, int dtype, bool aligned, bool full, int grid, size_t smem,
                          cudaStream_t s) {
    auto go = [&](auto kern) {
        cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        return launch_dependent(kern, dim3(grid), dim3(kXThreads), smem, s, a);
    };
    if (full) {
        if (dtype == 1) return aligned ? go(expand_kernel<1, true, true>) : go(expand_kernel<1, false, true>);
        return aligned ? go(expand_kernel<0, true, true>) : go(expand_kernel<0, false, true>);
    }
    if (dtype == 1) return aligned ? go(expand_kernel<1, true, false>) : go(expand_kernel<1, false, false>);
    return aligned ? go(expand_kernel<0, true, false>) : go(expand_kernel<0, false, false>);
}

size_t expand_keys_bytes(int max_segments, int support) {
    size_t keys = (size_t)kXWarps * kRegion;
    if ((size_t)max_segments * support > keys) keys = (size_t)max_segments * support;
    return (sizeof(unsigned long long) * keys + 127) & ~(size_t)127;  // the spill area after it is 16-byte aligned
}

size_t expand_smem_bytes(int max_segments, int support) {
    return expand_keys_bytes(max_segments, support) + kSpillBytes +
           sizeof(unsigned) * (kFineBins + kCoarseBins);
}

int expand_tile_elems(int dtype) { return kXTileBytes / (dtype == 1 ? 2 : 4); }

int full_group_tokens(int dtype) { return 32 * (dtype == 1 ? Elem<1>::VEC : Elem<0>::VEC); }

}  // namespace rheo
