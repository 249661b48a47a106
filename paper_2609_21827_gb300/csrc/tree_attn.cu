// tree_attn.cu -- inputs of the target forward over the pruned tree: the
// ancestor mask, the positions and the root-to-leaf paths.  The paper leaves
// these to its code base (Sec. 5.1); the definitions are stated with
// rheo_tree_attention in include/rheo.h.
//
// One CTA per request.  The pruned tree's parent, depth and child-count arrays
// are staged in shared memory; each warp builds a node's ancestor set as a
// bitmap by following parent pointers (at most depth + 1 steps) and writes that
// node's mask row from it, 32 bytes per store instruction; a block scan over
// the child counts numbers the leaves in ascending pruned index, and each leaf
// writes its path, root first, into its own row of the retrieve table.
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {

__global__ void __launch_bounds__(kThreads) tree_attn_kernel(const TreeAttnArgs a) {
    grid_dependency_begin();
    extern __shared__ __align__(16) int32_t tsm[];
    __shared__ BlockScratch bs;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int NP = a.n.N + 1, W = a.n.D + 1;
    const int words = (NP + 31) / 32;
    const int b = blockIdx.x;
    const int64_t pb = (int64_t)b * NP;
    int32_t* par = tsm;         // [NP]
    int32_t* dep = par + NP;    // [NP]
    int32_t* nch = dep + NP;    // [NP]
    unsigned* bits = reinterpret_cast<unsigned*>(nch + NP) + warp * words;  // this warp's bitmap

    for (int i = tid; i < NP; i += kThreads) {
        // in pruned order a parent precedes its children: anything else is not a tree
        int p = a.pr.parent[pb + i];
        if ((i == 0) ? (p != -1) : (p < 0 || p >= i)) {
            atomicOr(a.status, kStInternal);
            p = (i == 0) ? -1 : 0;
        }
        par[i] = p;
        dep[i] = a.pr.depth[pb + i];
        nch[i] = a.pr.n_child[pb + i];
    }
    __syncthreads();

    if (a.mask) {
        for (int i = warp; i < NP; i += kWarps) {
            for (int w = lane; w < words; w += 32) bits[w] = 0u;
            __syncwarp();
            if (lane == 0)  // parents strictly decrease, so the walk ends at the root
                for (int j = i; j >= 0; j = par[j]) bits[j >> 5] |= 1u << (j & 31);
            __syncwarp();
            uint8_t* row = a.mask + (pb + i) * NP;
            for (int j = lane; j < NP; j += 32) row[j] = (uint8_t)((bits[j >> 5] >> (j & 31)) & 1u);
            __syncwarp();
        }
    }
    if (a.position)
        for (int i = tid; i < NP; i += kThreads) a.position[pb + i] = dep[i];

    if (a.retrieve || a.n_leaves) {
        int before = 0;  // leaves in earlier chunks
        for (int i0 = 0; i0 < NP; i0 += kThreads) {
            const int i = i0 + tid;
            const bool leaf = i < NP && nch[i] == 0;
            int total;
            const int r = before + block_exclusive_scan(leaf ? 1 : 0, total, bs);
            if (leaf && a.retrieve) {
                int32_t* out = a.retrieve + (pb + r) * W;
                const int d = dep[i];
                if (d < 0 || d >= W) {
                    atomicOr(a.status, kStInternal);
                } else {
                    for (int k = d + 1; k < W; ++k) out[k] = -1;
                    int k = d;
                    for (int j = i; j >= 0 && k >= 0; j = par[j], --k) out[k] = j;
                    if (k != -1) atomicOr(a.status, kStInternal);  // depth and parent chain disagree
                }
            }
            before += total;
        }
        // rows past the last leaf
        if (a.retrieve)
            for (int64_t q = (int64_t)before * W + tid; q < (int64_t)NP * W; q += kThreads) a.retrieve[pb * W + q] = -1;
        if (a.n_leaves && tid == 0) a.n_leaves[b] = before;
    }
}

size_t tree_attn_smem_bytes(int budget) {
    const size_t NP = (size_t)budget + 1;
    return 3 * sizeof(int32_t) * NP + sizeof(unsigned) * kWarps * ((NP + 31) / 32);
}

cudaError_t launch_tree_attn(const TreeAttnArgs& a, int batch, size_t smem, cudaStream_t s) {
    cudaError_t err = cudaFuncSetAttribute(tree_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    return launch_dependent(tree_attn_kernel, dim3(batch), dim3(kThreads), smem, s, a);
}

}  // namespace rheo
