// rheo_kernels.h -- launch arguments shared by the C-ABI layer and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace rheo {

struct TreePtrs {
    int32_t* token;
    int32_t* parent;
    float* log_proxy;
    float* score;
    float* qtilde;
    uint8_t* slot;
    int32_t* frontier;
    int32_t* tail_ids;
    float* tail_q;
    float* lse1;
    float* lse_tail;   // [B, E] or null (sparse support); required with full support
};

struct PrunedPtrs {
    int32_t* gen_id;
    int32_t* token;
    int32_t* parent;
    int32_t* depth;
    int32_t* first_child;
    int32_t* n_child;
    int32_t* sampled_child;
};

struct Dims {
    int B = 0, V = 0, K = 0, m = 0, S = 0, D = 0, N = 0;
    int full = 0;    // full support: S = K+1 ranks selected, the sampled token drawn over V
    int TL = 0;      // S - m
    int GW = 0;      // gathered logits per verify row: (K+1) + TL
    int chunks = 0;  // chunks per row
    int64_t G1 = 0, E = 0;
    float eps = 0.0f;
};

struct ExpandArgs {
    Dims n;
    int d, F;
    size_t keys_bytes;              // dynamic shared memory for keys; the spill area follows
    const char* logits;
    int64_t row_stride_bytes;
    const float* T;
    const uint64_t* seed;
    const uint64_t* offset;
    TreePtrs tree;
    unsigned* status;
    unsigned* row_ticket;           // [B*F]
    unsigned* req_ticket;           // [B]
    float* seg_mu;                  // [B*F*tiles_per_row]
    float* seg_sum;                 // [B*F*tiles_per_row*2] float-float partition sums
    unsigned long long* seg_keys;   // [B*F*tiles_per_row*S]
    float* lse_tail_ff;             // [B*E*2] full support: the tail's log-partition as float-float
    // full support: per group of full_group_tokens consecutive token ids of a
    // row, its tempered sum at the group's reference (reference, sum)
    float* grp;                     // [B*F*groups_per_row*2]
};

struct PruneArgs {
    Dims n;
    TreePtrs tree;
    PrunedPtrs pr;
    unsigned* status;
    int staged;  // parent, token and slot of every node are read with the scores into shared memory
};

struct TreeAttnArgs {
    Dims n;
    PrunedPtrs pr;
    uint8_t* mask;       // [B, N+1, N+1] or null
    int32_t* position;   // [B, N+1] or null
    int32_t* retrieve;   // [B, N+1, D+1] or null
    int32_t* n_leaves;   // [B] or null
    unsigned* status;
};

enum : int { kVerifyRheo = 0, kVerifyRrsw = 1, kVerifyOneHot = 2 };
constexpr int kMaxFullDepth = 32;  // depth limit of full-support verification

// the verification stream's unit counters: kStreamQueues of them, 128 bytes apart
constexpr int kStreamQueues = 16;
constexpr int kStreamQueueStride = 32;

struct VerifyArgs {
    Dims n;                         // n.chunks: 2 KB chunks per target row
    int variant = kVerifyRheo;      // verification rule at every node (kVerify*)
    int prep_grid = 0;              // CTAs of the prep launch (0: one per two rows)
    const char* logits;
    int64_t row_stride_bytes;
    const float* T;
    const uint64_t* seed;
    const uint64_t* offset;
    TreePtrs tree;
    PrunedPtrs pr;
    int32_t* accepted_len;
    int32_t* accepted_tokens;
    int32_t* accepted_nodes;
    int32_t* bonus_token;
    float* row_lse;                 // may be null
    unsigned* status;
    float* seg_mu;                  // [B*(N+1)*chunks]
    float* seg_sum;                 // [B*(N+1)*chunks*2] float-float partition sums
    unsigned* queue;                // [kStreamQueues * kStreamQueueStride] unit counters (zero between calls)
    int* rec_hdr;                   // [B*(N+1)*8] row records (see verify.cu)
    int* rec_child;                 // [B*(N+1)*(K+1)*3]
    int* rec_tids;                  // [B*(N+1)*TL]
    float* rec_tq;                  // [B*(N+1)*TL]
    float* rec_cx;                  // [B*(N+1)*(K+1)*2]
    float* rec_tx;                  // [B*(N+1)*TL*2]
    float* rec_coin;                // [B*(N+1)*(K+2)]
    float* table;                   // [B*(N+1)*table_width(K)] decision tables
    float* rhat_tail;               // [B*(N+1)*TL]
    unsigned long long* res_best;   // [B*3]
    unsigned* res_ticket;           // [B]
    // full support: the draft rows of the expanded nodes (depth d: [B, F_d, V]
    // rows at draft[d-1] + (b*F_d + f) * draft_row_stride_bytes) and the tails'
    // log-partitions written by the expansions
    const char* draft[kMaxFullDepth] = {};
    int64_t draft_row_stride_bytes = 0;
    const float* lse_tail_ff = nullptr;  // [B*E*2]
};

// Launch with the programmatic stream serialization attribute: the kernel may
// start launching while the previous kernel on the stream finishes; kernels
// call grid_dependency_begin() before touching global memory.
template <class... P, class... A>
cudaError_t launch_dependent(void (*kern)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, A&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<A&&>(args)...);
}

// Host launchers, defined next to their kernels.  dtype: 0 fp32, 1 bf16;
// aligned: every row starts on a 16-byte boundary, so rows are read with
// 16-byte vector loads (a row's ragged end element-wise); otherwise element-wise.
// whole: every CTA's tiles lie in one row (the two halves are streamed side by side)
cudaError_t launch_expand(const ExpandArgs& a, int dtype, bool aligned, bool full, int grid, size_t smem,
                          cudaStream_t s);
cudaError_t launch_prune(const PruneArgs& a, int batch, size_t smem, cudaStream_t s);
cudaError_t launch_verify(const VerifyArgs& a, int dtype, bool aligned, int grid, cudaStream_t s);
cudaError_t launch_verify_full(const VerifyArgs& a, int dtype, bool aligned, bool draft_aligned, int grid,
                               cudaStream_t s);
size_t expand_keys_bytes(int max_segments, int support);
size_t expand_smem_bytes(int max_segments, int support);
int expand_tile_elems(int dtype);
int full_group_tokens(int dtype);
cudaError_t launch_tree_attn(const TreeAttnArgs& a, int batch, size_t smem, cudaStream_t s);
size_t tree_attn_smem_bytes(int budget);
int verify_table_width(int K);
int verify_chunks_per_row(int dtype, int V);
int verify_stream_grid(int sms, int64_t chunks);

}  // namespace rheo
