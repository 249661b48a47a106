// prune.cu -- global rerank/prune to the verification budget (App. C.1 "Path
// scores and global pruning"; Lemma 2 makes the result ancestor-closed).
//
// One CTA per request.  Keys (ord(score) << 32 | ~gen) order nodes by score
// descending, then gen id ascending (= shallower first, then left to right);
// the N-th largest key is found by bitwise selection, the survivors are
// compacted in gen-id order with a block scan, and parents are remapped
// through a gen -> pruned-index table in shared memory.
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {

__global__ void __launch_bounds__(kThreads) prune_kernel(const PruneArgs a) {
    extern __shared__ int32_t map[];  // [G1]
    __shared__ BlockScratch bs;
    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int b = blockIdx.x;
    const int N = n.N;
    const int64_t G1 = n.G1;
    const int64_t nb = (int64_t)b * G1, pb = (int64_t)b * (N + 1);
    int parity = 0;

    auto key_of = [&](int64_t g) -> unsigned long long {
        return ((unsigned long long)ord_f32(a.tree.score[nb + g]) << 32) | (0xFFFFFFFFu - (uint32_t)g);
    };

    // threshold: the N-th largest key among gen ids 1..G1-1
    unsigned long long thr = 1ull;
    if (G1 - 1 > N) {
        unsigned long long aand = ~0ull, aor = 0ull;
        for (int64_t g = 1 + tid; g < G1; g += kThreads) {
            const unsigned long long x = key_of(g);
            aand &= x;
            aor |= x;
        }
        aand = block_and_or_u64(aand, false, bs);
        aor = block_and_or_u64(aor, true, bs);
        thr = block_select(
            [&](unsigned long long t) {
                int c = 0;
                for (int64_t g = 1 + tid; g < G1; g += kThreads) c += key_of(g) >= t;
                return c;
            },
            N, aand, aor, bs, parity);
    }

    // compaction in gen-id order; the root is always kept
    const int per = (int)((G1 + kThreads - 1) / kThreads);
    const int64_t lo = min(G1, (int64_t)tid * per), hi = min(G1, lo + per);
    int cnt = 0;
    for (int64_t g = lo; g < hi; ++g) cnt += (g == 0 || key_of(g) >= thr);
    int total;
    int pos = block_exclusive_scan(cnt, total, bs);
    for (int64_t g = lo; g < hi; ++g) {
        if (g == 0 || key_of(g) >= thr) {
            map[g] = pos;
            if (pos <= N) {
                a.pr.gen_id[pb + pos] = (int32_t)g;
                a.pr.token[pb + pos] = a.tree.token[nb + g];
                a.pr.depth[pb + pos] = depth_of(n.K, g);
            }
            ++pos;
        } else {
            map[g] = -1;
        }
    }
    if (total != N + 1) {  // cannot happen with distinct keys; never index with a partial table
        if (tid == 0) atomicOr(a.status, kStInternal);
        return;
    }
    for (int i = tid; i <= N; i += kThreads) {
        a.pr.first_child[pb + i] = -1;
        a.pr.n_child[pb + i] = 0;
        a.pr.sampled_child[pb + i] = -1;
    }
    __syncthreads();

    // parents; children are contiguous in pruned order (gen-consecutive pools)
    for (int i = tid; i <= N; i += kThreads) {
        const int64_t g = a.pr.gen_id[pb + i];
        int32_t p = -1;
        if (g != 0) {
            const int32_t pg = a.tree.parent[nb + g];
            p = (pg >= 0 && pg < G1) ? map[pg] : -1;
            if (p < 0) atomicOr(a.status, kStInternal);  // not ancestor-closed (or tree never expanded)
        }
        a.pr.parent[pb + i] = p;
    }
    __syncthreads();
    for (int i = 1 + tid; i <= N; i += kThreads) {
        const int32_t p = a.pr.parent[pb + i];
        if (p < 0) continue;
        const bool first = (i == 1) || (a.pr.parent[pb + i - 1] != p);
        const bool last = (i == N) || (a.pr.parent[pb + i + 1] != p);
        if (first) a.pr.first_child[pb + p] = i;
        if (last) a.pr.n_child[pb + p] = i;  // index of the last child, turned into a count below
        if (a.tree.slot[nb + a.pr.gen_id[pb + i]] == kSlotSampled) a.pr.sampled_child[pb + p] = i;
    }
    __syncthreads();
    for (int i = tid; i <= N; i += kThreads) {
        const int fc = a.pr.first_child[pb + i];
        if (fc >= 0) a.pr.n_child[pb + i] = a.pr.n_child[pb + i] - fc + 1;
    }
}

cudaError_t launch_prune(const PruneArgs& a, int batch, size_t smem, cudaStream_t s) {
    if (smem > 48 * 1024) {
        const cudaError_t err = cudaFuncSetAttribute(prune_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
    }
    prune_kernel<<<batch, kThreads, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace rheo
