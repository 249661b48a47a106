/*
 * rheo_oracle.h -- plain CPU reference of the RheoSampling draft-tree hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may include, link,
 * load or call this code: only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / --impl reference legs of bench.py use it.  It shares no
 * source, header, table or helper with the CUDA library.
 *
 * Every routine follows the paper step by step, with full sorts, fp64 sums and
 * plain loops:
 *   - hybrid pool (top-m leads, one token sampled from the tail, fills),
 *     Sec. 3.2 "Hybrid sampling mechanism" and App. C.1 "Hybrid candidate pool";
 *   - dual identity (proxy min{q(x_m), z} for construction, q~(Y) = q(Y)/z for
 *     verification), Sec. 3.2 "Dual treatment of the sampled token";
 *   - sparse top-128 draft distribution, Sec. 3.2 "Efficient implementation";
 *   - untempered construction / tempered sampling and verification, Sec. 5.4;
 *   - path scores, frontier top-K and global prune with the depth / left-to-
 *     right tie-break, Sec. 2.1 and App. C.1 "Path scores and global pruning";
 *   - RheoVerification applied layer by layer, Algorithm 1 and Theorem 1.
 *
 * Conventions the paper leaves open (node numbering, Philox counter layout,
 * uniform conversion, tie-breaks, fp32 rounding points) are stated in the
 * comments of rheo_oracle.c; they are ours, so their parity is pinned only by
 * agreement between the two implementations ("parity unpinned" by the paper).
 */
#ifndef RHEO_ORACLE_H
#define RHEO_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_SLOT_ROOT = 0, ORC_SLOT_LEAD = 1, ORC_SLOT_SAMPLED = 2, ORC_SLOT_FILL = 3 };
enum { ORC_TAG_SAMPLE = 1, ORC_TAG_VERIFY = 2, ORC_TAG_RESIDUAL = 3, ORC_TAG_CONTINUE = 0 };

typedef struct {
    int32_t B;       /* requests */
    int32_t V;       /* vocabulary */
    int32_t K;       /* deterministic slots per pool; pool size K+1 */
    int32_t m;       /* lead tokens (the rheostat), 0 <= m <= K */
    int32_t S;       /* sparse support, K+1 <= S <= min(V,128); 0: the whole vocabulary
                        (full support: Y drawn in two Gumbel-max stages, a block of
                        256 token ids by its tail mass with draw V + block, then the
                        token within it with draw = token id) */
    int32_t D;       /* expansion depth */
    int32_t N;       /* prune budget (non-root nodes kept) */
    double eps;      /* proxy offset for m = 0 */
    int32_t proxy_mode;      /* 0: the paper's proxy. 1: fixed log-proxy (planted mistake for tests) */
    double fixed_log_proxy;  /* used only when proxy_mode == 1 */
    int32_t verify_mode;     /* ORC_VERIFY_*: the verification rule applied at every node */
    int32_t plant_mode;      /* ORC_PLANT_*: a mistake planted on purpose, for tests that must
                                reject it; 0 everywhere else */
} orc_cfg;

/* Planted mistakes in Algorithm 1 after the sampled child is rejected (test
 * infrastructure: each is a no-op when the support covers the vocabulary, so
 * only tests at S < V can tell them from the method):
 *  RESIDUAL_ON_SUPPORT  the final draw u* ~ r^ considers only the expansion's
 *                       support (its m leads and its tail), dropping r^ = p
 *                       off the support;
 *  MASS_ON_SUPPORT      the residual mass M is summed over the support only
 *                       (tail r^ plus p at the leads) instead of
 *                       1 - sum_tail min(p, q~).
 * And one in the full-support draw of Y (a no-op while the vocabulary fits in
 * one block):
 *  BLOCK_UNWEIGHTED     the block of the two-stage draw is chosen by g alone,
 *                       ignoring its mass. */
enum {
    ORC_PLANT_NONE = 0,
    ORC_PLANT_RESIDUAL_ON_SUPPORT = 1,
    ORC_PLANT_MASS_ON_SUPPORT = 2,
    ORC_PLANT_BLOCK_UNWEIGHTED = 3
};

/* Verification rules (all lossless):
 *  RHEO    Algorithm 1: the sampled child first (accept iff eta*q~ <= p), then
 *          the others in slot order against r = norm(max(0, p - q~));
 *  RRSW    recursive rejection, App. D.2: the leads in slot order by one-hot
 *          rejection under p, then the sampled child against the renormalised
 *          residual p~ (accept iff eta*q~ <= p~), then the fills against
 *          norm(max(0, p~ - q~));
 *  ONEHOT  vanilla verification of a top-K tree (Sec. 2.2, App. A): every child
 *          a one-hot candidate in slot order, residual from p. */
enum { ORC_VERIFY_RHEO = 0, ORC_VERIFY_RRSW = 1, ORC_VERIFY_ONEHOT = 2 };

typedef struct {
    int32_t* token;      /* [B*G1] token of each generated node; root -1 */
    int32_t* parent;     /* [B*G1] parent gen id; root -1 */
    float* log_proxy;    /* [B*G1] log of the construction probability (q0, or the proxy for Y) */
    float* score;        /* [B*G1] path score = sum of log proxies (fp32) */
    float* qtilde;       /* [B*G1] true sampling probability q~(Y) of sampled nodes, else 0 */
    uint8_t* slot;       /* [B*G1] ORC_SLOT_* */
    int32_t* frontier;   /* [B*K] gen ids selected for the next expansion, ascending */
    int32_t* tail_ids;   /* [B*E*(S-m)] support ranks m+1..S of every expanded node */
    float* tail_q;       /* [B*E*(S-m)] q~ over that tail (tempered, renormalised) */
    float* lse1;         /* [B*E] log-partition of the untempered draft row */
    double* gap_sample;  /* [B*E] relative gap of the two best Gumbel keys */
    double* gap_frontier;/* [B*D] relative gap at the frontier boundary of depth d (index d-1) */
    float* lse_tail;     /* [B*E] log sum over the tail of exp(l/T), or NULL */
} orc_tree;

typedef struct {
    int32_t* gen_id;        /* [B*(N+1)] pruned order = ascending gen id, root first */
    int32_t* token;
    int32_t* parent;        /* pruned index, root -1 */
    int32_t* depth;
    int32_t* first_child;   /* pruned index of first surviving child or -1 */
    int32_t* n_child;
    int32_t* sampled_child; /* pruned index of the surviving sampled child or -1 */
    double* gap_prune;      /* [B] relative gap at the prune boundary (1 if N == G) */
} orc_pruned;

typedef struct {
    int32_t* accepted_len;     /* [B] */
    int32_t* accepted_tokens;  /* [B*D] */
    int32_t* accepted_nodes;   /* [B*D] pruned indices */
    int32_t* bonus_token;      /* [B] */
    float* row_lse;            /* [B*(N+1)] log sum_v exp(l_v / T) of each target row */
    double* gap_level;         /* [B*(D+1)] smallest decision gap taken at walk level i */
    float* stop_mass;          /* [B] residual mass M when the walk stopped (1 if r = p) */
} orc_verify_out;

int orc_check_cfg(const orc_cfg* c);
int64_t orc_nodes_per_request(const orc_cfg* c);      /* G1 = 1 + (K+1) + (D-1)K(K+1) */
int64_t orc_expansions_per_request(const orc_cfg* c); /* E = 1 + (D-1)K */

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
float orc_uniform(uint64_t seed, uint64_t offset, int32_t tag, int32_t node, uint64_t draw);

/* top-S of one row under (logit desc, id asc); returns 0 or -1 */
int orc_topk_row(const float* row, int32_t V, int32_t S, int32_t* ids_out);

int orc_expand(const orc_cfg* c, int32_t d, const float* rows, const float* T,
               const uint64_t* seed, const uint64_t* offset, orc_tree* t);
int orc_prune(const orc_cfg* c, const orc_tree* t, orc_pruned* p);
int orc_verify(const orc_cfg* c, const float* target, const float* T, const uint64_t* seed,
               const uint64_t* offset, const orc_tree* t, const orc_pruned* p, orc_verify_out* o);

/* Whole decoding cycles against draft/target "language models" given as
 * tables indexed by token prefix (row of prefix x_1..x_j = sum_{i<j} V^i +
 * base-V value of the prefix).  Runs n_trials independent cycles (seed_b =
 * seed0 + b, offset 0), then extends each emitted stream autoregressively from
 * the target table to L tokens.  Used by the losslessness tests (Theorem 1). */
int orc_run_prefix_lm(const orc_cfg* c, const float* draft_table, const float* target_table,
                      int32_t table_depth, int64_t n_trials, float T, uint64_t seed0, int32_t L,
                      int32_t* streams, int32_t* acc_len);

/* Inputs of the target forward over the pruned tree (tree attention).  The
 * paper leaves them to its code base (Sec. 5.1); the definitions are ours:
 *   mask[b][i][j] = 1 iff pruned node j is node i or an ancestor of i, else 0
 *                   ([B][N+1][N+1] bytes);
 *   position[b][i] = depth of pruned node i (root 0);
 *   leaves = pruned nodes without a surviving child, in ascending pruned index;
 *   retrieve[b][r][k] = pruned index of the depth-k node on the path from the
 *                   root to the r-th leaf ([B][N+1][D+1]), -1 past the leaf's
 *                   depth and on every row r >= n_leaves[b].
 * Computed by following parent pointers.  Any output may be NULL. */
int orc_tree_attention(const orc_cfg* c, const orc_pruned* p, uint8_t* mask, int32_t* position,
                       int32_t* retrieve, int32_t* n_leaves);

/* Timing reports: OpenMP threads that ran an iteration of a parallel loop
 * since the last reset (reset != 0 clears the record), the team size for the
 * next parallel loops, and the current maximum team size (1 without OpenMP). */
int orc_threads_used(int32_t reset);
void orc_set_threads(int32_t n);
int orc_max_threads(void);

#ifdef __cplusplus
}
#endif
#endif
