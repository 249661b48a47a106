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
    int B, V, K, m, S, D, N;
    int TL;      // S - m
    int GW;      // gathered logits per verify row: (K+1) + TL
    int chunks;  // chunks per row
    int64_t G1, E;
    float eps;
};

struct ExpandArgs {
    Dims n;
    int d, F;
    const char* logits;
    int64_t row_stride_bytes;
    const float* T;
    const uint64_t* seed;
    const uint64_t* offset;
    TreePtrs tree;
    unsigned* status;
    unsigned* row_ticket;          // [B*F]
    unsigned* req_ticket;          // [B]
    float* chunk_mu;               // [B*F*chunks]
    double* chunk_sum;             // [B*F*chunks]
    unsigned long long* chunk_keys;  // [B*F*chunks*S]
};

struct PruneArgs {
    Dims n;
    TreePtrs tree;
    PrunedPtrs pr;
    unsigned* status;
};

struct VerifyArgs {
    Dims n;
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
    float* row_lse;  // may be null
    unsigned* status;
    float* row_mu;           // [B*(N+1)*chunks]
    double* row_sum;         // [B*(N+1)*chunks]
    float* gather;           // [B*(N+1)*GW]
    unsigned* req_ticket;    // [B]
    int32_t* desc;           // [B*8]: stop row, gen, lse bits, use_tail, n_excl, expansion, M bits, -
    int32_t* excl;           // [B*(K+1)]
    float* rhat;             // [B*TL]
    unsigned long long* res_best;  // [B*3]
    unsigned* res_ticket;    // [B]
};

// Host launchers, defined next to their kernels.  dtype: 0 fp32, 1 bf16;
// aligned: rows start on 16-byte boundaries (128-bit loads).
cudaError_t launch_expand(const ExpandArgs& a, int dtype, bool aligned, dim3 grid, size_t smem, cudaStream_t s);
cudaError_t launch_prune(const PruneArgs& a, int batch, size_t smem, cudaStream_t s);
cudaError_t launch_verify(const VerifyArgs& a, int dtype, bool aligned, dim3 stream_grid, dim3 residual_grid,
                          cudaStream_t s);

}  // namespace rheo
