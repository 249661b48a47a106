/*
 * rheo.h -- C ABI of the RheoSampling draft-tree hot path on one GPU.
 *
 * One decoding cycle is:  rheo_expand(d = 1..D)  ->  rheo_prune  ->  rheo_verify.
 * Between expansion calls the caller runs its draft model on the frontier
 * nodes (tree.frontier, ascending gen id) and passes their logits to the next
 * call; after the prune it runs the target model on the pruned tree (root
 * first, ascending gen id) and passes those logits to rheo_verify.
 *
 * Paper: RheoSampling (arXiv 2609.21827).  Sec. 2.1 (expand-then-rerank),
 * Sec. 3.2 (hybrid pool, proxy / true probability, sparse top-128 draft),
 * Sec. 5.4 (untempered construction), App. C.1 (pool, path scores, global
 * prune and tie-break), Algorithm 1 (RheoVerification, applied layer by layer
 * as in Theorem 1).
 *
 * Ownership.  The caller allocates and owns every buffer (device memory unless
 * stated).  The library never allocates, keeps no global state (except the
 * static scratch array of rheo_verify_static), and runs asynchronously on the
 * caller's stream.  A workspace holds scratch state of
 * one cycle; it must be zeroed once by rheo_workspace_init (and again after any
 * call reported an error) and must not be shared by calls that may overlap in
 * time (use one workspace per stream).
 *
 * Errors.  Functions return RHEO_OK (0), RHEO_EINVAL (-1) for an argument the
 * host rejects before any launch, or RHEO_ELAUNCH (-2) for a failed launch.
 * Faults in the data (NaN or +inf logits, an all -inf row, a non-positive
 * temperature) set bits of a device status word; rheo_get_status reads it.
 * Outputs of a call whose status is non-zero are unspecified.
 *
 * Node numbering (per request).  gen id 0 is the root.  The K+1 children of
 * the root are 1..K+1 in slot order; at depth d >= 2 the child in slot j of the
 * f-th frontier node is base_d + f(K+1) + j, base_d = 1 + (K+1) + (d-2)K(K+1).
 * Slot order: m leads, the sampled token, K-m fills.  G1 = 1 + (K+1) +
 * (D-1)K(K+1) nodes; E = 1 + (D-1)K expanded nodes (root = 0, the f-th
 * frontier node chosen at depth d = 1 + (d-1)K + f).
 */
#ifndef RHEO_H
#define RHEO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without including CUDA headers; NULL is the legacy default stream */
typedef struct CUstream_st* rheo_stream_t;

enum { RHEO_F32 = 0, RHEO_BF16 = 1 };
enum { RHEO_OK = 0, RHEO_EINVAL = -1, RHEO_ELAUNCH = -2, RHEO_ETOOLARGE = -3 };

/* device status bits */
enum {
    RHEO_STATUS_BAD_LOGIT = 1,       /* NaN or +inf in a row                  */
    RHEO_STATUS_EMPTY_ROW = 2,       /* a row with fewer than m+1 (draft) or no (target) finite logits */
    RHEO_STATUS_BAD_TEMPERATURE = 4, /* T <= 0, inf or NaN                    */
    RHEO_STATUS_INTERNAL = 8         /* broken invariant (e.g. prune not ancestor-closed) */
};

/* Problem size.  K = deterministic slots per pool (pool = K+1), 0 <= m <= K,
 * K+1 <= support <= min(vocab, 128), depth >= 1 (depth 1 if K = 0),
 * 1 <= budget <= G1-1, G1 <= 16384, vocab <= 262144, eps > 0 when m = 0.
 * support = 0 selects full support (App. B, Table tab:sparse_support, row
 * Full): the sampled token is drawn from the tempered draft distribution over
 * the whole vocabulary minus the leads, in two Gumbel-max stages (a block of
 * 256 consecutive token ids by its tempered mass, Philox draw index V + block;
 * then the token within it, draw index = token id; sparse support: one stage,
 * draw index = tail position); requires m <= 1 and K+1 <= 128; no tail
 * lists are kept (tail_ids / tail_q unused, lse_tail required) and the tree is
 * verified by rheo_verify_full, which re-reads the expanded nodes' draft rows. */
typedef struct {
    int32_t batch;   /* B requests                                  */
    int32_t vocab;   /* V                                           */
    int32_t K;       /* deterministic slots (pool = K+1)            */
    int32_t m;       /* leads; the sampled token sits in slot m     */
    int32_t support; /* S, sparse draft support (top-S logits)      */
    int32_t depth;   /* D expansion layers                          */
    int32_t budget;  /* N non-root nodes kept by the prune          */
    float eps;       /* proxy offset when m = 0 (Sec. 3.2)          */
    int32_t dtype;   /* RHEO_F32 or RHEO_BF16, for all logits       */
} rheo_config;

/* Unpruned tree of every request, written by rheo_expand.  Row-major, request
 * major: [B, G1] for node fields, [B, K] frontier, [B, E, S-m] tail lists. */
typedef struct {
    int32_t* token;     /* [B,G1] token id; root -1                                    */
    int32_t* parent;    /* [B,G1] parent gen id; root -1                               */
    float* log_proxy;   /* [B,G1] log construction probability: log q0 (leads, fills,
                           untempered full-vocab softmax) or the log proxy (sampled)   */
    float* score;       /* [B,G1] path score, sum of log_proxy from the root (fp32)    */
    float* qtilde;      /* [B,G1] true sampling probability q~(Y) of sampled nodes, else 0 */
    uint8_t* slot;      /* [B,G1] 0 root, 1 lead, 2 sampled, 3 fill                    */
    int32_t* frontier;  /* [B,K] gen ids to expand next, ascending                     */
    int32_t* tail_ids;  /* [B,E,S-m] support ranks m+1..S of each expanded node        */
    float* tail_q;      /* [B,E,S-m] q~ over that tail: softmax(l/T) renormalised      */
    float* lse1;        /* [B,E] log sum_v exp(l_v) of each expanded draft row         */
    float* lse_tail;    /* [B,E] log of the tail's sum of exp(l/T) (ranks m+1..S, or V
                           minus the leads with full support); may be NULL with sparse
                           support, required with full support                          */
} rheo_tree;

/* Pruned tree, written by rheo_prune: [B, N+1], root first, ascending gen id. */
typedef struct {
    int32_t* gen_id;
    int32_t* token;
    int32_t* parent;        /* pruned index; root -1                       */
    int32_t* depth;
    int32_t* first_child;   /* pruned index of the first surviving child, -1 */
    int32_t* n_child;       /* surviving children (contiguous, slot order)  */
    int32_t* sampled_child; /* pruned index of the surviving sampled child, -1 */
} rheo_pruned;

/* Verification outputs (device memory). */
typedef struct {
    int32_t* accepted_len;    /* [B] accepted draft tokens, 0..D                 */
    int32_t* accepted_tokens; /* [B,D] -1 past accepted_len                      */
    int32_t* accepted_nodes;  /* [B,D] pruned indices, -1 past accepted_len      */
    int32_t* bonus_token;     /* [B] token drawn from the final residual (Alg. 1) */
    float* row_lse;           /* [B,N+1] optional (may be NULL): log sum exp(l/T) per row */
} rheo_verify_out;

/* Sizes for a configuration: nodes per request (G1), expanded nodes per
 * request (E) and workspace bytes.  Any output pointer may be NULL. */
int rheo_sizes(const rheo_config* cfg, int64_t* nodes_per_request, int64_t* expansions_per_request,
               size_t* workspace_bytes);

/* Zero a workspace of at least rheo_sizes() bytes (cudaMemsetAsync on stream). */
int rheo_workspace_init(const rheo_config* cfg, void* workspace, size_t bytes, rheo_stream_t stream);

/* Expansion at depth d (1..D).  Sec. 3.2 / App. C.1 / Sec. 2.1.
 * draft_logits: [B, F_d, V] of cfg.dtype, F_1 = 1 (the root) and F_d = K (the
 *   frontier chosen at depth d-1, in tree.frontier order); row r = b*F_d + f
 *   starts at element r*row_stride (row_stride >= V, in elements).
 * temperature, seed, offset: [B] device arrays (per-request T > 0; Philox key
 *   and counter offset).
 * For every row: support = top-S logits (logit desc, id asc); lse1 over all V
 *   at T = 1; Y ~ softmax(l/T) over support ranks m+1..S by Gumbel-max;
 *   children in slot order with log q0 = l - lse1 and the proxy of Y
 *   (min{q0(x_m), z}, z = 1 - sum_{i<=m} q0(x_i), never below q0(x_{m+1});
 *   min(1, q0(x_1) + eps) when m = 0); scores accumulate; if d < D, the K best
 *   depth-d nodes (score desc, gen id asc) become tree.frontier. */
int rheo_expand(const rheo_config* cfg, int32_t d, const void* draft_logits, int64_t row_stride,
                const float* temperature, const uint64_t* seed, const uint64_t* offset,
                const rheo_tree* tree, void* workspace, rheo_stream_t stream);

/* Global prune (App. C.1): keep the root and the N best of the G1-1 generated
 * nodes by (score desc, gen id asc); the result is ancestor-closed (Lemma 2). */
int rheo_prune(const rheo_config* cfg, const rheo_tree* tree, const rheo_pruned* pruned,
               void* workspace, rheo_stream_t stream);

/* RheoVerification (Algorithm 1) layer by layer from the root.
 * target_logits: [B, N+1, V] of cfg.dtype in pruned order, row stride in
 *   elements.  p = softmax(l/T).  At node u with surviving children C: if the
 *   sampled child s survived, accept it iff eta*q~(s) <= p(s); else r^ = max(0,
 *   p - q~) over u's tail (p elsewhere) with mass M = 1 - sum_tail min(p, q~);
 *   then each other child in slot order is accepted iff eta*M <= r^(c), else M
 *   -= r^(c) and r^(c) = 0.  When no child is accepted (or C is empty) the
 *   bonus token is drawn from r^ over V minus C by Gumbel-max.  Uniforms:
 *   Philox, tag 2 (coins) and 3 (residual), node = gen id of u. */
int rheo_verify(const rheo_config* cfg, const void* target_logits, int64_t row_stride,
                const float* temperature, const uint64_t* seed, const uint64_t* offset,
                const rheo_tree* tree, const rheo_pruned* pruned, const rheo_verify_out* out,
                void* workspace, rheo_stream_t stream);

/* Verification variants on the same kernels (App. A, App. D.2), for
 * comparisons of acceptance; all are lossless.  variant:
 *   RHEO_VERIFY_RHEO    Algorithm 1 (exactly rheo_verify);
 *   RHEO_VERIFY_RRSW    recursive rejection without replacement (App. D.2):
 *                       leads (slots < m) one-hot against p in slot order;
 *                       then the sampled child against the renormalised
 *                       residual p~ = r/M: accept iff fp32(eta*q~)*M <= r(Y);
 *                       on rejection the tail residual becomes max(0, r - M q~)
 *                       (mass M - sum_tail min(r, M q~)); then the fills
 *                       (slots > m) one-hot against it;
 *   RHEO_VERIFY_ONEHOT  vanilla verification of the pool as a top-K set
 *                       (Sec. 2.2, App. A): every surviving child, the sampled
 *                       one too, one-hot against r = p in slot order.
 * One-hot test of child c: accept iff eta*M <= r(c), else M -= r(c), r(c) = 0.
 * Coins: tag 2, draw 0 for the sampled child's test under RRSW, draw 1+slot for
 * every one-hot test.  The final draw after all rejections is u* ~ r over V
 * minus the surviving children, as in rheo_verify.  Other arguments, outputs
 * and errors as rheo_verify; an unknown variant returns RHEO_EINVAL. */
enum { RHEO_VERIFY_RHEO = 0, RHEO_VERIFY_RRSW = 1, RHEO_VERIFY_ONEHOT = 2 };
int rheo_verify_variant(const rheo_config* cfg, int32_t variant, const void* target_logits, int64_t row_stride,
                        const float* temperature, const uint64_t* seed, const uint64_t* offset,
                        const rheo_tree* tree, const rheo_pruned* pruned, const rheo_verify_out* out,
                        void* workspace, rheo_stream_t stream);

/* Verification of a tree built with full support (cfg.support = 0; App. B,
 * Table tab:sparse_support, row Full), Algorithm 1 as rheo_verify.  With no
 * tail lists, q~ over the whole vocabulary is re-derived from the draft rows:
 * draft_logits is a host array of cfg.depth device pointers, entry d-1 the
 * [B, F_d, V] draft logits passed to rheo_expand at depth d (row b*F_d + f at
 * element (b*F_d + f)*draft_row_stride); they must be unchanged since the
 * expansion, and the workspace must be the one the expansions used (it holds
 * the tails' log-partitions).  At a node whose sampled child survived:
 * q~(v) = exp(l_d(v)/T - lse_tail) off the lead, 0 at the lead,
 * M = 1 - sum_V min(p, q~), r^ = max(0, p - q~).  Requires depth <= 32.
 * Other arguments, outputs and errors as rheo_verify. */
int rheo_verify_full(const rheo_config* cfg, const void* target_logits, int64_t row_stride,
                     const void* const* draft_logits, int64_t draft_row_stride, const float* temperature,
                     const uint64_t* seed, const uint64_t* offset, const rheo_tree* tree, const rheo_pruned* pruned,
                     const rheo_verify_out* out, void* workspace, rheo_stream_t stream);

/* Verification for callers that cannot allocate device memory where they
 * verify (code handed only fixed input/output buffers by a host framework,
 * runtimes whose device memory is partitioned up front, loops that must not
 * pay cudaMalloc's implicit synchronisation).  The paper has no counterpart:
 * this is a deployment variant of rheo_verify, same arguments and results
 * minus the workspace.  Scratch state lives in a static device array of
 * RHEO_STATIC_SCRATCH_BYTES that every GPU loading the library holds until
 * exit; configurations needing more return RHEO_ETOOLARGE before any launch.
 * Every call looks the array up in the current context (the first call on a
 * device also loads it: make that call before any stream capture), so calls
 * after a cudaDeviceReset find the new context's array.  Calls share the
 * array: calls that overlap on the GPU race, so
 * serialise them.  status: optional device int32 that receives this call's
 * status word (the bits of rheo_get_status); may be NULL. */
#define RHEO_STATIC_SCRATCH_BYTES (8u << 20)
int rheo_verify_static(const rheo_config* cfg, const void* target_logits, int64_t row_stride,
                       const float* temperature, const uint64_t* seed, const uint64_t* offset,
                       const rheo_tree* tree, const rheo_pruned* pruned, const rheo_verify_out* out,
                       int32_t* status, rheo_stream_t stream);

/* Inputs of the target forward over the pruned tree (tree attention).  The
 * paper runs the target model on the tree inside its code base (Sec. 5.1) and
 * does not define these arrays; the definitions are ours:
 *   mask      [B, N+1, N+1] uint8: mask[b][i][j] = 1 iff pruned node j is
 *             node i or an ancestor of i (node i attends to j), else 0;
 *   position  [B, N+1] int32: depth of pruned node i (root 0); the caller adds
 *             its context length;
 *   retrieve  [B, N+1, D+1] int32: row r < n_leaves[b] holds the pruned
 *             indices of the path from the root to the r-th leaf (leaves =
 *             nodes without a surviving child, in ascending pruned index),
 *             position k = the node at depth k, -1 past the leaf's depth;
 *             rows r >= n_leaves[b] are all -1;
 *   n_leaves  [B] int32.
 * Any of the four pointers may be NULL (that output is skipped).  Requires
 * N+1 <= 4096 (RHEO_EINVAL otherwise).  A pruned tree whose parent of node i
 * is not in [0, i) (root: -1), or whose depths disagree with its parent
 * chain, sets RHEO_STATUS_INTERNAL.  The workspace carries the status word. */
typedef struct {
    uint8_t* mask;
    int32_t* position;
    int32_t* retrieve;
    int32_t* n_leaves;
} rheo_tree_attn;

int rheo_tree_attention(const rheo_config* cfg, const rheo_pruned* pruned, const rheo_tree_attn* out,
                        void* workspace, rheo_stream_t stream);

/* Synchronise the stream, return the device status word in *status (host
 * memory) and clear it.  Returns RHEO_ELAUNCH if the stream reported an error. */
int rheo_get_status(const rheo_config* cfg, void* workspace, rheo_stream_t stream, int32_t* status);

#ifdef __cplusplus
}
#endif
#endif /* RHEO_H */
