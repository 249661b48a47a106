// prune.cu -- global rerank/prune to the verification budget (App. C.1 "Path
// scores and global pruning"; Lemma 2 makes the result ancestor-closed).
//
// One CTA per request, everything staged in shared memory.  Keys
// (ord(score) << 32 | ~gen) order nodes by score descending, then gen id
// ascending (= shallower first, then left to right); the N-th largest key is
// found by bitwise selection, the survivors are compacted in gen-id order with
// a block scan, and parents are remapped through a gen -> pruned-index table.
// When they fit, the nodes' parent, token and slot are read together with the
// scores, so the kernel makes one round trip to the tree instead of three.
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {

__global__ void __launch_bounds__(kThreads) prune_kernel(const PruneArgs a) {
    grid_dependency_begin();
    extern __shared__ __align__(16) unsigned char psm[];
    __shared__ BlockScratch bs;
    __shared__ unsigned hist[kRadixBins];
    __shared__ RadixScratch rad;
    const Dims& n = a.n;
    const int tid = threadIdx.x;
    const int b = blockIdx.x;
    const int N = n.N, NP = n.N + 1;
    const int G1 = (int)n.G1;
    const int64_t nb = (int64_t)b * G1, pb = (int64_t)b * NP;

    unsigned long long* keys = reinterpret_cast<unsigned long long*>(psm);     // [G1]
    int32_t* map = reinterpret_cast<int32_t*>(keys + G1);                      // [G1] gen -> pruned index
    int32_t* pgen = map + G1;                                                  // [NP] pruned index -> gen
    int32_t* ppar = pgen + NP;                                                 // [NP] parent (pruned index)
    int32_t* pfc = ppar + NP;                                                  // [NP] first child
    int32_t* plc = pfc + NP;                                                   // [NP] last child
    int32_t* psc = plc + NP;                                                   // [NP] sampled child
    int32_t* tpar = psc + NP;                                                  // [G1] parent gen id (staged)
    int32_t* ttok = tpar + G1;                                                 // [G1] token (staged)
    uint8_t* tslot = reinterpret_cast<uint8_t*>(ttok + G1);                    // [G1] slot (staged)
    const bool staged = a.staged != 0;

    for (int g = tid; g < G1; g += kThreads) {
        keys[g] = ((unsigned long long)ord_f32(a.tree.score[nb + g]) << 32) | (0xFFFFFFFFu - (uint32_t)g);
        if (staged) {
            tpar[g] = a.tree.parent[nb + g];
            ttok[g] = a.tree.token[nb + g];
            tslot[g] = a.tree.slot[nb + g];
        }
    }
    for (int i = tid; i < NP; i += kThreads) { pfc[i] = -1; plc[i] = -1; psc[i] = -1; }
    __syncthreads();

    // threshold: the N-th largest key among gen ids 1..G1-1
    unsigned long long thr = 1ull;
    if (G1 - 1 > N) thr = block_radix_threshold([&](int i) { return keys[1 + i]; }, G1 - 1, N, hist, rad);

    // compaction in gen-id order; the root is always kept
    const int per = (G1 + kThreads - 1) / kThreads;
    const int lo = min(G1, tid * per), hi = min(G1, lo + per);
    int cnt = 0;
    for (int g = lo; g < hi; ++g) cnt += (g == 0 || keys[g] >= thr);
    int total;
    int pos = block_exclusive_scan(cnt, total, bs);
    if (total != NP) {  // cannot happen with distinct keys; never index with a partial table
        if (tid == 0) atomicOr(a.status, kStInternal);
        return;
    }
    for (int g = lo; g < hi; ++g) {
        if (g == 0 || keys[g] >= thr) {
            map[g] = pos;
            pgen[pos] = g;
            ++pos;
        } else {
            map[g] = -1;
        }
    }
    __syncthreads();

    // parents (one parallel round trip for the tree fields), then children ranges
    for (int i = tid; i < NP; i += kThreads) {
        const int g = pgen[i];
        int32_t p = -1;
        if (g != 0) {
            const int32_t pg = staged ? tpar[g] : a.tree.parent[nb + g];
            p = (pg >= 0 && pg < G1) ? map[pg] : -1;
            if (p < 0) atomicOr(a.status, kStInternal);  // not ancestor-closed (or tree never expanded)
        }
        ppar[i] = p;
        a.pr.gen_id[pb + i] = g;
        a.pr.token[pb + i] = staged ? ttok[g] : a.tree.token[nb + g];
        a.pr.depth[pb + i] = depth_of(n.K, g);
        a.pr.parent[pb + i] = p;
    }
    __syncthreads();
    for (int i = 1 + tid; i < NP; i += kThreads) {
        const int32_t p = ppar[i];
        if (p < 0) continue;
        if (i == 1 || ppar[i - 1] != p) pfc[p] = i;
        if (i == N || ppar[i + 1] != p) plc[p] = i;
        const int g = pgen[i];
        if ((staged ? tslot[g] : a.tree.slot[nb + g]) == kSlotSampled) psc[p] = i;
    }
    __syncthreads();
    for (int i = tid; i < NP; i += kThreads) {
        a.pr.first_child[pb + i] = pfc[i];
        a.pr.n_child[pb + i] = (pfc[i] >= 0) ? plc[i] - pfc[i] + 1 : 0;
        a.pr.sampled_child[pb + i] = psc[i];
    }
}

cudaError_t launch_prune(const PruneArgs& a, int batch, size_t smem, cudaStream_t s) {
    if (smem > 48 * 1024) {
        const cudaError_t err = cudaFuncSetAttribute(prune_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
    }
    const cudaError_t err = launch_dependent(prune_kernel, dim3(batch), dim3(kThreads), smem, s, a);
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
}

}  // namespace rheo
