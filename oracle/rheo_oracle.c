/*
 * rheo_oracle.c -- plain CPU reference of the RheoSampling hot path.
 *
 * TEST INFRASTRUCTURE ONLY (see rheo_oracle.h).  Slow on purpose: full sorts,
 * fp64 sums, one request or one row at a time.  The only parallelism is an
 * OpenMP loop over independent rows / requests, which does not change results.
 *
 * Conventions fixed here because the paper leaves them open (both this file
 * and the CUDA library implement them from their written description; there is
 * no shared code):
 *
 *  Node numbering.  gen id 0 is the root.  Depth-1 children are 1..K+1 in slot
 *  order.  At depth d >= 2 the child in slot j of the f-th frontier node has gen
 *  id base_d + f(K+1) + j with base_d = 1 + (K+1) + (d-2)K(K+1).  Frontier
 *  nodes are kept in ascending gen id, so gen-id order equals the left-to-right
 *  order of App. C.1 within every depth.  The expansion index of the root is 0
 *  and of the f-th frontier node chosen at depth d is 1 + (d-1)K + f.
 *
 *  Slot order.  Leads (ranks 1..m), then the sampled token Y, then the K-m
 *  fills (Sec. 3.2 "Hybrid sampling mechanism").
 *
 *  Random numbers.  Philox4x32-10 (Salmon et al., SC'11), key = (lo32 seed,
 *  hi32 seed), counter = (draw>>2, lo32 offset, 4*node + tag, hi32 offset),
 *  output word draw&3.  Uniform u = ((w>>9) + 0.5) * 2^-23, exact in fp32 and
 *  strictly inside (0,1).  Tags: 1 tail sample (node = expanded parent, draw =
 *  tail position), 2 verification coin (node = verified parent, draw 0 for the
 *  sampled child and 1+slot for the others), 3 residual draw (node = stopping
 *  node, draw = token id), 0 continuation (tests only).
 *
 *  Rounding points.  Values that decide an integer (Gumbel keys, path scores,
 *  acceptance tests) are formed in fp32 exactly as written below; sums are
 *  accumulated in fp64 and rounded once to fp32.
 */
#include "rheo_oracle.h"
#ifdef _OPENMP
#include <omp.h>
#endif

#include <math.h>
#include <stdlib.h>
#include <string.h>

#define ORC_MAX_NODES 16384 /* keeps 4*node + tag below 2^16 */

/* ------------------------------------------------------------------ */
/* configuration and numbering                                          */
/* ------------------------------------------------------------------ */

int64_t orc_nodes_per_request(const orc_cfg* c) {
    return 1 + (int64_t)(c->K + 1) + (int64_t)(c->D - 1) * c->K * (c->K + 1);
}

int64_t orc_expansions_per_request(const orc_cfg* c) { return 1 + (int64_t)(c->D - 1) * c->K; }

/* Thread accounting for timing reports: which OpenMP threads ran at least one
 * iteration of a parallel loop since the last reset. */
#define ORC_MAX_THREADS 1024
static volatile unsigned char g_thread_busy[ORC_MAX_THREADS];
static void note_thread(void) {
#ifdef _OPENMP
    const int t = omp_get_thread_num();
    if (t >= 0 && t < ORC_MAX_THREADS) g_thread_busy[t] = 1;
#else
    g_thread_busy[0] = 1;
#endif
}
int orc_threads_used(int32_t reset) {
    int n = 0;
    for (int i = 0; i < ORC_MAX_THREADS; ++i) {
        n += g_thread_busy[i] ? 1 : 0;
        if (reset) g_thread_busy[i] = 0;
    }
    return n;
}
void orc_set_threads(int32_t n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}
int orc_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

int orc_check_cfg(const orc_cfg* c) {
    if (!c) return -1;
    if (c->B < 1 || c->V < 1 || c->K < 0 || c->m < 0 || c->m > c->K) return -1;
    if (c->S != 0 && (c->S < c->K + 1 || c->S > c->V || c->S > 128)) return -1;
    if (c->S == 0 && c->V < c->K + 1) return -1;
    if (c->D < 1 || (c->K == 0 && c->D > 1)) return -1;
    int64_t G1 = orc_nodes_per_request(c);
    if (G1 > ORC_MAX_NODES) return -1;
    if (c->N < 1 || c->N > G1 - 1) return -1;
    if (c->m == 0 && !(c->eps > 0.0)) return -1;
    if (c->verify_mode < ORC_VERIFY_RHEO || c->verify_mode > ORC_VERIFY_ONEHOT) return -1;
    if (c->plant_mode < ORC_PLANT_NONE || c->plant_mode > ORC_PLANT_BLOCK_UNWEIGHTED) return -1;
    return 0;
}

/* Support size: S, or the whole vocabulary when S == 0 ("full support",
 * App. B Table tab:sparse_support, row Full).  In full support the tail draw
 * of token v uses draw index v (the token id) instead of its tail position,
 * after a first draw of the block of ORC_FULL_BLOCK token ids it lies in
 * (draw V + block index). */
#define ORC_FULL_BLOCK 256
static int support_of(const orc_cfg* c) { return c->S == 0 ? c->V : c->S; }

static int64_t depth_base(const orc_cfg* c, int d) {
    return d == 1 ? 1 : 1 + (int64_t)(c->K + 1) + (int64_t)(d - 2) * c->K * (c->K + 1);
}

static int rows_at_depth(const orc_cfg* c, int d) { return d == 1 ? 1 : c->K; }

static int depth_of(const orc_cfg* c, int64_t g) {
    if (g == 0) return 0;
    if (g <= c->K + 1) return 1;
    return 2 + (int)((g - (c->K + 2)) / ((int64_t)c->K * (c->K + 1)));
}

/* slot index j of a non-root node inside its pool */
static int slot_of(const orc_cfg* c, int64_t g) {
    if (g <= c->K + 1) return (int)(g - 1);
    return (int)((g - (c->K + 2)) % (c->K + 1));
}

/* expansion index of the parent of non-root node g */
static int64_t parent_expansion_of(const orc_cfg* c, int64_t g) {
    if (g <= c->K + 1) return 0;
    int64_t w = g - (c->K + 2);
    int64_t per_depth = (int64_t)c->K * (c->K + 1);
    int64_t d = 2 + w / per_depth;
    int64_t f = (w % per_depth) / (c->K + 1);
    return 1 + (d - 2) * c->K + f;
}

static double rel_gap(double a, double b) {
    if (isinf(a) || isinf(b)) return (a == b) ? 0.0 : INFINITY;
    double s = fabs(a) > fabs(b) ? fabs(a) : fabs(b);
    if (s < 1.0) s = 1.0;
    return fabs(a - b) / s;
}

/* ------------------------------------------------------------------ */
/* Philox4x32-10 and uniforms                                           */
/* ------------------------------------------------------------------ */

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        uint32_t n1 = (uint32_t)p1;
        uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        uint32_t n3 = (uint32_t)p0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

float orc_uniform(uint64_t seed, uint64_t offset, int32_t tag, int32_t node, uint64_t draw) {
    uint32_t ctr[4] = {(uint32_t)(draw >> 2), (uint32_t)offset, (uint32_t)(4 * node + tag),
                       (uint32_t)(offset >> 32)};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    orc_philox4x32_10(ctr, key, out);
    uint32_t w = out[draw & 3u];
    return ((float)(w >> 9) + 0.5f) * (1.0f / 8388608.0f);
}

/* standard Gumbel variate -log(-log u), correctly rounded to fp32 */
static float gumbel(float u) { return (float)(-log(-log((double)u))); }

/* ------------------------------------------------------------------ */
/* top-S under (logit desc, id asc)                                     */
/* ------------------------------------------------------------------ */

typedef struct {
    float l;
    int32_t id;
} orc_entry;

static int cmp_entry(const void* a, const void* b) {
    const orc_entry* x = (const orc_entry*)a;
    const orc_entry* y = (const orc_entry*)b;
    if (x->l > y->l) return -1;
    if (x->l < y->l) return 1;
    return (x->id < y->id) ? -1 : (x->id > y->id);
}

int orc_topk_row(const float* row, int32_t V, int32_t S, int32_t* ids_out) {
    if (S < 1 || S > V) return -1;
    orc_entry* e = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)V);
    if (!e) return -1;
    for (int32_t v = 0; v < V; ++v) {
        if (isnan(row[v])) { free(e); return -1; }
        e[v].l = row[v];
        e[v].id = v;
    }
    qsort(e, (size_t)V, sizeof(orc_entry), cmp_entry);
    for (int32_t i = 0; i < S; ++i) ids_out[i] = e[i].id;
    free(e);
    return 0;
}

/* ------------------------------------------------------------------ */
/* expansion: sparse draft, hybrid pool, proxy, path scores             */
/* ------------------------------------------------------------------ */

/* Expand one parent row.  Returns 0, or -2 for a row the method cannot use
 * (NaN / +inf entry, or fewer than m+1 finite logits). */
static int expand_row(const orc_cfg* c, int d, int b, int f, const float* l, float T, uint64_t seed,
                      uint64_t offset, orc_tree* t) {
    const int K = c->K, m = c->m, S = support_of(c), V = c->V, TL = S - m;
    const int64_t G1 = orc_nodes_per_request(c), E = orc_expansions_per_request(c);
    const int64_t par = (d == 1) ? 0 : t->frontier[(int64_t)b * K + f];
    const int64_t e = (d == 1) ? 0 : 1 + (int64_t)(d - 2) * K + f;
    const int64_t g0 = depth_base(c, d) + (int64_t)f * (K + 1);
    const int64_t nb = (int64_t)b * G1;

    int nfinite = 0;
    for (int v = 0; v < V; ++v) {
        if (isnan(l[v]) || (isinf(l[v]) && l[v] > 0)) return -2;
        if (isfinite(l[v])) ++nfinite;
    }
    if (nfinite < m + 1) return -2;

    /* untempered full-vocabulary log-partition (Sec. 5.4: construction uses
     * the original draft probabilities; App. B: the sparse truncation leaves
     * the deterministic candidates untouched) */
    double mx = -INFINITY;
    for (int v = 0; v < V; ++v) if (l[v] > mx) mx = l[v];
    double s = 0.0;
    for (int v = 0; v < V; ++v) s += exp((double)l[v] - mx);
    const float lse1 = (float)(mx + log(s));

    /* sparse support: the S largest logits (Sec. 3.2, top-128 before softmax) */
    orc_entry* srt = (orc_entry*)malloc(sizeof(orc_entry) * (size_t)V);
    if (!srt) return -2;
    for (int v = 0; v < V; ++v) { srt[v].l = l[v]; srt[v].id = v; }
    qsort(srt, (size_t)V, sizeof(orc_entry), cmp_entry);

    float* lq0 = (float*)malloc(sizeof(float) * (size_t)S * 3);
    if (!lq0) { free(srt); return -2; }
    float* tau = lq0 + S;
    float* qt = tau + S;
    for (int i = 0; i < S; ++i) lq0[i] = srt[i].l - lse1; /* fp32 */

    /* tempered tail q~ over support ranks m+1..S (App. C.1: q~ = q / z on the
     * complement of the leads; Sec. 5.4: temperature applies to sampling) */
    double mt = -INFINITY;
    for (int i = 0; i < TL; ++i) {
        tau[i] = srt[m + i].l / T; /* fp32 division */
        if (tau[i] > mt) mt = tau[i];
    }
    double st = 0.0;
    for (int i = 0; i < TL; ++i) st += exp((double)tau[i] - mt);
    const double lse_tail = mt + log(st);
    for (int i = 0; i < TL; ++i) qt[i] = (float)exp((double)tau[i] - lse_tail);
    if (t->lse_tail) t->lse_tail[(int64_t)b * E + e] = (float)lse_tail;

    /* Y ~ q~ by Gumbel-max; ties keep the earlier tail position (full support:
     * the lower token id).  Full support draws in two stages, each a
     * Gumbel-max and so exact (P(block) = its mass / the tail's, then
     * P(Y | block) = q~ / the block's mass): first a block of ORC_FULL_BLOCK
     * consecutive token ids by its tempered log-mass, fp32(mt + log mass) + g
     * (draw V + block index; ties keep the lower block), then the token within
     * that block by tau + g (draw = token id). */
    int best = -1;
    float bk = -INFINITY, second = -INFINITY;
    double gap_block = INFINITY;
    int blk = -1;
    if (c->S == 0) {
        const int nblk = (V + ORC_FULL_BLOCK - 1) / ORC_FULL_BLOCK;
        double* mass = (double*)calloc((size_t)nblk, sizeof(double));
        if (!mass) { free(srt); free(lq0); return -2; }
        for (int i = 0; i < TL; ++i) mass[srt[m + i].id / ORC_FULL_BLOCK] += exp((double)tau[i] - mt);
        float kb = -INFINITY, kb2 = -INFINITY;
        for (int k = 0; k < nblk; ++k) {
            if (!(mass[k] > 0.0)) continue; /* no tail token with mass here */
            const float lm = (c->plant_mode == ORC_PLANT_BLOCK_UNWEIGHTED) ? 0.0f : (float)(mt + log(mass[k]));
            const float key = lm + gumbel(orc_uniform(seed, offset, ORC_TAG_SAMPLE, (int32_t)par, (uint64_t)V + k));
            if (key > kb) {
                kb2 = kb;
                kb = key;
                blk = k;
            } else if (key > kb2) kb2 = key;
        }
        free(mass);
        gap_block = rel_gap(kb, kb2);
    }
    for (int i = 0; i < TL; ++i) {
        if (c->S == 0 && srt[m + i].id / ORC_FULL_BLOCK != blk) continue;
        const uint64_t draw = (c->S == 0) ? (uint64_t)srt[m + i].id : (uint64_t)i;
        float g = gumbel(orc_uniform(seed, offset, ORC_TAG_SAMPLE, (int32_t)par, draw));
        float key = tau[i] + g;
        if (key > bk || (c->S == 0 && key == bk && best >= 0 && srt[m + i].id < srt[m + best].id)) {
            second = bk;
            bk = key;
            best = i;
        } else if (key > second) second = key;
    }
    if (best < 0) { free(srt); free(lq0); return -2; }

    /* construction probability of Y (Sec. 3.2; App. C.1):
     *   m >= 1: min{q(x_m), z}, z = 1 - sum_{i<=m} q(x_i); never below
     *           q(x_{m+1}) (Lemma 1 holds in exact arithmetic; the max() keeps
     *           it true after rounding);
     *   m == 0: q(x_1) + eps, capped at 1 so that Lemma 2 keeps holding. */
    float lp;
    if (c->proxy_mode == 1) {
        lp = (float)c->fixed_log_proxy;
    } else if (m >= 1) {
        double zs = 0.0;
        for (int i = 0; i < m; ++i) zs += exp((double)lq0[i]);
        if (zs > 1.0) zs = 1.0;
        float lz = (float)log1p(-zs);
        lp = lq0[m - 1] < lz ? lq0[m - 1] : lz;
        if (lp < lq0[m]) lp = lq0[m];
    } else {
        double pr = exp((double)lq0[0]) + c->eps;
        if (pr > 1.0) pr = 1.0;
        lp = (float)log(pr);
    }

    const float ps = t->score[nb + par];
    for (int j = 0; j <= K; ++j) {
        int64_t g = nb + g0 + j;
        int rank;
        float lpj;
        uint8_t st8;
        float qv = 0.0f;
        if (j < m) {
            rank = j; lpj = lq0[j]; st8 = ORC_SLOT_LEAD;
        } else if (j == m) {
            rank = m + best; lpj = lp; st8 = ORC_SLOT_SAMPLED; qv = qt[best];
        } else {
            rank = -1; lpj = 0; st8 = ORC_SLOT_FILL; /* assigned below */
        }
        if (j <= m) {
            t->token[g] = srt[rank].id;
            t->log_proxy[g] = lpj;
            t->score[g] = ps + lpj; /* fp32 */
            t->qtilde[g] = qv;
            t->slot[g] = st8;
            t->parent[g] = (int32_t)par;
        }
    }
    /* fills: highest remaining support ranks, skipping Y */
    int r = m;
    for (int j = m + 1; j <= K; ++j) {
        if (r == m + best) ++r;
        int64_t g = nb + g0 + j;
        t->token[g] = srt[r].id;
        t->log_proxy[g] = lq0[r];
        t->score[g] = ps + lq0[r];
        t->qtilde[g] = 0.0f;
        t->slot[g] = ORC_SLOT_FILL;
        t->parent[g] = (int32_t)par;
        ++r;
    }

    for (int i = 0; i < TL; ++i) {
        t->tail_ids[((int64_t)b * E + e) * TL + i] = srt[m + i].id;
        t->tail_q[((int64_t)b * E + e) * TL + i] = qt[i];
    }
    t->lse1[(int64_t)b * E + e] = lse1;
    {
        const double gt = rel_gap(bk, second);
        t->gap_sample[(int64_t)b * E + e] = gt < gap_block ? gt : gap_block;
    }
    free(srt);
    free(lq0);
    return 0;
}

typedef struct {
    float s;
    int32_t g;
} orc_scored;

/* (score desc, gen id asc): depth first then left to right, App. C.1 */
static int cmp_scored(const void* a, const void* b) {
    const orc_scored* x = (const orc_scored*)a;
    const orc_scored* y = (const orc_scored*)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    return (x->g < y->g) ? -1 : (x->g > y->g);
}

static int cmp_int32(const void* a, const void* b) {
    int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
    return (x < y) ? -1 : (x > y);
}

int orc_expand(const orc_cfg* c, int32_t d, const float* rows, const float* T, const uint64_t* seed,
               const uint64_t* offset, orc_tree* t) {
    if (orc_check_cfg(c) || d < 1 || d > c->D) return -1;
    const int F = rows_at_depth(c, d);
    const int64_t G1 = orc_nodes_per_request(c);
    if (d == 1) {
        for (int b = 0; b < c->B; ++b) {
            int64_t nb = (int64_t)b * G1;
            t->token[nb] = -1; t->parent[nb] = -1; t->log_proxy[nb] = 0.0f;
            t->score[nb] = 0.0f; t->qtilde[nb] = 0.0f; t->slot[nb] = ORC_SLOT_ROOT;
        }
    }
    for (int b = 0; b < c->B; ++b)
        if (!(T[b] > 0.0f) || isinf(T[b])) return -2;
    int err = 0;
    const int64_t nrows = (int64_t)c->B * F;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (int64_t rr = 0; rr < nrows; ++rr) {
        int b = (int)(rr / F), f = (int)(rr % F);
        const float* l = rows + rr * (int64_t)c->V;
        note_thread();
        if (expand_row(c, d, b, f, l, T[b], seed[b], offset[b], t)) err |= 1;
    }
    if (err) return -2;

    /* next frontier: the K best depth-d nodes (Sec. 2.1 expand-then-rerank) */
    if (d < c->D) {
        const int n = F * (c->K + 1);
        orc_scored* cand = (orc_scored*)malloc(sizeof(orc_scored) * (size_t)n);
        if (!cand) return -2;
        for (int b = 0; b < c->B; ++b) {
            int64_t nb = (int64_t)b * G1, base = depth_base(c, d);
            for (int i = 0; i < n; ++i) {
                cand[i].s = t->score[nb + base + i];
                cand[i].g = (int32_t)(base + i);
            }
            qsort(cand, (size_t)n, sizeof(orc_scored), cmp_scored);
            int32_t* fr = t->frontier + (int64_t)b * c->K;
            for (int k = 0; k < c->K; ++k) fr[k] = cand[k].g;
            qsort(fr, (size_t)c->K, sizeof(int32_t), cmp_int32);
            t->gap_frontier[(int64_t)b * c->D + (d - 1)] =
                (n > c->K) ? rel_gap(cand[c->K - 1].s, cand[c->K].s) : INFINITY;
        }
        free(cand);
    } else {
        for (int b = 0; b < c->B; ++b) t->gap_frontier[(int64_t)b * c->D + (d - 1)] = INFINITY;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* global prune (App. C.1 "Path scores and global pruning")             */
/* ------------------------------------------------------------------ */

int orc_prune(const orc_cfg* c, const orc_tree* t, orc_pruned* p) {
    if (orc_check_cfg(c)) return -1;
    const int64_t G1 = orc_nodes_per_request(c);
    const int N = c->N;
    const int64_t G = G1 - 1;
    orc_scored* cand = (orc_scored*)malloc(sizeof(orc_scored) * (size_t)G);
    int32_t* map = (int32_t*)malloc(sizeof(int32_t) * (size_t)G1);
    uint8_t* keep = (uint8_t*)malloc((size_t)G1);
    if (!cand || !map || !keep) { free(cand); free(map); free(keep); return -2; }
    int rc = 0;
    for (int b = 0; b < c->B && !rc; ++b) {
        const int64_t nb = (int64_t)b * G1, pb = (int64_t)b * (N + 1);
        for (int64_t i = 0; i < G; ++i) { cand[i].s = t->score[nb + 1 + i]; cand[i].g = (int32_t)(1 + i); }
        qsort(cand, (size_t)G, sizeof(orc_scored), cmp_scored);
        memset(keep, 0, (size_t)G1);
        keep[0] = 1;
        for (int i = 0; i < N; ++i) keep[cand[i].g] = 1;
        p->gap_prune[b] = (N < G) ? rel_gap(cand[N - 1].s, cand[N].s) : INFINITY;
        int k = 0;
        for (int64_t g = 0; g < G1; ++g) {
            map[g] = keep[g] ? k : -1;
            if (keep[g]) {
                p->gen_id[pb + k] = (int32_t)g;
                p->token[pb + k] = t->token[nb + g];
                p->depth[pb + k] = depth_of(c, g);
                p->first_child[pb + k] = -1;
                p->n_child[pb + k] = 0;
                p->sampled_child[pb + k] = -1;
                ++k;
            }
        }
        for (int i = 0; i <= N; ++i) {
            int64_t g = p->gen_id[pb + i];
            if (g == 0) { p->parent[pb + i] = -1; continue; }
            int32_t par = map[t->parent[nb + g]];
            if (par < 0) { rc = -3; break; } /* not ancestor-closed: Lemma 2 violated */
            p->parent[pb + i] = par;
            if (p->first_child[pb + par] < 0) p->first_child[pb + par] = i;
            else if (p->first_child[pb + par] + p->n_child[pb + par] != i) { rc = -3; break; }
            p->n_child[pb + par] += 1;
            if (t->slot[nb + g] == ORC_SLOT_SAMPLED) p->sampled_child[pb + par] = i;
        }
    }
    free(cand); free(map); free(keep);
    return rc;
}

/* ------------------------------------------------------------------ */
/* Tree attention inputs for the target forward (our definitions; the  */
/* paper defers them to its code base, Sec. 5.1)                        */
/* ------------------------------------------------------------------ */

int orc_tree_attention(const orc_cfg* c, const orc_pruned* p, uint8_t* mask, int32_t* position,
                       int32_t* retrieve, int32_t* n_leaves) {
    if (orc_check_cfg(c)) return -1;
    const int NP = c->N + 1, W = c->D + 1;
    for (int b = 0; b < c->B; ++b) {
        const int64_t pb = (int64_t)b * NP;
        const int32_t* par = p->parent + pb;
        /* node i attends to itself and to every ancestor: follow the parents */
        if (mask) {
            uint8_t* mb = mask + (int64_t)b * NP * NP;
            memset(mb, 0, (size_t)NP * (size_t)NP);
            for (int i = 0; i < NP; ++i) {
                int steps = 0;
                for (int j = i; j >= 0; j = par[j]) {
                    if (j >= NP || ++steps > NP) return -3; /* not a tree */
                    mb[(int64_t)i * NP + j] = 1;
                }
            }
        }
        if (position)
            for (int i = 0; i < NP; ++i) position[pb + i] = p->depth[pb + i];
        /* leaves in ascending pruned index; the path of each, root first */
        int nl = 0;
        if (retrieve)
            for (int64_t q = 0; q < (int64_t)NP * W; ++q) retrieve[pb * W + q] = -1;
        for (int i = 0; i < NP; ++i) {
            if (p->n_child[pb + i] != 0) continue;
            if (retrieve) {
                const int dep = p->depth[pb + i];
                if (dep < 0 || dep >= W) return -3;
                int k = dep;
                for (int j = i; j >= 0; j = par[j]) {
                    if (k < 0) return -3; /* depth disagrees with the parent chain */
                    retrieve[(pb + nl) * W + k] = j;
                    --k;
                }
                if (k != -1) return -3;
            }
            ++nl;
        }
        if (n_leaves) n_leaves[b] = nl;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* RheoVerification, layer by layer (Algorithm 1, Theorem 1)            */
/* ------------------------------------------------------------------ */

/* The verification variants at one node u (target row l, log-partition lu):
 * returns the accepted pruned index or -1, and leaves the residual mass in *M,
 * and, when the sampled child was rejected, the tail residual in rhat (indexed
 * through tail_pos) with *use_tail = 1.  The rules are those of orc_cfg's
 * verify_mode.  Coins: draw 0 for the sampled child under RRSW, draw 1+slot
 * for every one-hot candidate (the sampled child too under ONEHOT). */
static int verify_variant(const orc_cfg* c, int b, const float* l, double lu, float T, uint64_t seed,
                          uint64_t offset, const orc_tree* t, const orc_pruned* p, int u, double* gap_out,
                          float* rhat, int32_t* tail_pos, const int32_t** tids_out, double* M_out,
                          int* use_tail_out) {
    const int N = c->N, TL = support_of(c) - c->m;
    const int64_t G1 = orc_nodes_per_request(c), E = orc_expansions_per_request(c);
    const int64_t nb = (int64_t)b * G1, pb = (int64_t)b * (N + 1);
    const int fc = p->first_child[pb + u], nc = p->n_child[pb + u], sc = p->sampled_child[pb + u];
    const int64_t gu = p->gen_id[pb + u];
    double M = 1.0;
    int use_tail = 0;
#define P_OF(tok) ((float)exp((double)l[(tok)] / (double)T - lu))
    /* one-hot rejection of child v against the current residual (mass M) */
#define ONE_HOT(v)                                                                                        \
    do {                                                                                                  \
        const int64_t gv_ = p->gen_id[pb + (v)];                                                         \
        const int tok_ = p->token[pb + (v)];                                                             \
        const float eta_ = orc_uniform(seed, offset, ORC_TAG_VERIFY, (int32_t)gu,                        \
                                       (uint64_t)(1 + slot_of(c, gv_)));                                 \
        float rv_;                                                                                       \
        if (use_tail && tail_pos[tok_] >= 0) rv_ = rhat[tail_pos[tok_]];                                 \
        else rv_ = P_OF(tok_);                                                                           \
        const double lhs_ = (double)eta_ * M;                                                            \
        const double gap_ = rel_gap(lhs_, rv_);                                                          \
        if (gap_ < *gap_out) *gap_out = gap_;                                                            \
        if (lhs_ <= (double)rv_) { accepted = (v); goto done; }                                          \
        M -= (double)rv_;                                                                                \
        if (use_tail && tail_pos[tok_] >= 0) rhat[tail_pos[tok_]] = 0.0f;                                \
    } while (0)
    int accepted = -1;
    if (c->verify_mode == ORC_VERIFY_ONEHOT) {
        for (int k = 0; k < nc; ++k) ONE_HOT(fc + k);
        goto done;
    }
    /* RRSw: the leads under p */
    for (int k = 0; k < nc; ++k)
        if (t->slot[nb + p->gen_id[pb + fc + k]] == ORC_SLOT_LEAD) ONE_HOT(fc + k);
    if (sc >= 0) {
        /* the sampled child against p~ = r / M: accept iff eta*q~ <= r(Y) / M */
        const int64_t gs = p->gen_id[pb + sc];
        const float eta0 = orc_uniform(seed, offset, ORC_TAG_VERIFY, (int32_t)gu, 0);
        const float qv = t->qtilde[nb + gs];
        const float pv = P_OF(p->token[pb + sc]);
        const double lhs = (double)(eta0 * qv) * M; /* fp32(eta*q~), then times M */
        const double gap = rel_gap(lhs, pv);
        if (gap < *gap_out) *gap_out = gap;
        if (lhs <= (double)pv) { accepted = sc; goto done; }
        /* residual M * norm(max(0, p~ - q~)) = max(0, r - M q~) on the tail */
        const int64_t e = parent_expansion_of(c, gs);
        const int32_t* tids = t->tail_ids + ((int64_t)b * E + e) * TL;
        const float* tq = t->tail_q + ((int64_t)b * E + e) * TL;
        double overlap = 0.0;
        for (int i = 0; i < TL; ++i) {
            const float pt = P_OF(tids[i]);
            const double mq = M * (double)tq[i];
            const double d = (double)pt - mq;
            rhat[i] = d > 0.0 ? (float)d : 0.0f;
            overlap += (double)pt < mq ? (double)pt : mq;
            tail_pos[tids[i]] = i;
        }
        M -= overlap;
        use_tail = 1;
        *tids_out = tids;
    }
    /* the fills against the residual */
    for (int k = 0; k < nc; ++k)
        if (t->slot[nb + p->gen_id[pb + fc + k]] == ORC_SLOT_FILL) ONE_HOT(fc + k);
done:
#undef ONE_HOT
#undef P_OF
    *M_out = M;
    *use_tail_out = use_tail;
    return accepted;
}

static int verify_request(const orc_cfg* c, int b, const float* target, float T, uint64_t seed,
                          uint64_t offset, const orc_tree* t, const orc_pruned* p, orc_verify_out* o) {
    const int V = c->V, N = c->N, D = c->D, K = c->K, TL = support_of(c) - c->m;
    const int64_t G1 = orc_nodes_per_request(c), E = orc_expansions_per_request(c);
    const int64_t nb = (int64_t)b * G1, pb = (int64_t)b * (N + 1);
    const float* rows = target + pb * V;

    double* lse = (double*)malloc(sizeof(double) * (size_t)(N + 1));
    int32_t* tail_pos = (int32_t*)malloc(sizeof(int32_t) * (size_t)V);
    float* rhat = (float*)malloc(sizeof(float) * (size_t)(TL > 0 ? TL : 1));
    if (!lse || !tail_pos || !rhat) { free(lse); free(tail_pos); free(rhat); return -2; }

    /* target distribution p = softmax(l / T) of every pruned node's row */
    for (int u = 0; u <= N; ++u) {
        const float* l = rows + (int64_t)u * V;
        double mx = -INFINITY;
        for (int v = 0; v < V; ++v) {
            if (isnan(l[v]) || (isinf(l[v]) && l[v] > 0)) { free(lse); free(tail_pos); free(rhat); return -2; }
            double x = (double)l[v] / (double)T;
            if (x > mx) mx = x;
        }
        if (isinf(mx)) { free(lse); free(tail_pos); free(rhat); return -2; }
        double s = 0.0;
        for (int v = 0; v < V; ++v) s += exp((double)l[v] / (double)T - mx);
        lse[u] = mx + log(s);
        o->row_lse[pb + u] = (float)lse[u];
    }
    for (int v = 0; v < V; ++v) tail_pos[v] = -1;

    double* gl = o->gap_level + (int64_t)b * (D + 1);
    for (int i = 0; i <= D; ++i) gl[i] = INFINITY;

    int u = 0, len = 0;
    for (;;) {
        const float* l = rows + (int64_t)u * V;
        const double lu = lse[u];
        const float lsef = (float)lu;
        const int fc = p->first_child[pb + u], nc = p->n_child[pb + u], sc = p->sampled_child[pb + u];
        const int64_t gu = p->gen_id[pb + u];
#define P_OF(tok) ((float)exp((double)l[(tok)] / (double)T - lu))
        double M = 1.0;
        int use_tail = 0;
        const int32_t* tids = NULL;
        int64_t pool0 = -1; /* gen id of slot 0 in the pool of u's sampled child (after its rejection) */
        int accepted = -1;
        if (c->verify_mode != ORC_VERIFY_RHEO) {
            accepted = verify_variant(c, b, l, lu, T, seed, offset, t, p, u, gl + len, rhat, tail_pos, &tids,
                                      &M, &use_tail);
        } else {
            if (nc > 0 && sc >= 0) {
                /* stochastic-first: accept u_s with probability min(1, p/q~) */
                const int64_t gs = p->gen_id[pb + sc];
                const float eta0 = orc_uniform(seed, offset, ORC_TAG_VERIFY, (int32_t)gu, 0);
                const float qv = t->qtilde[nb + gs];
                const float pv = P_OF(p->token[pb + sc]);
                const float lhs = eta0 * qv; /* fp32 */
                double gap = rel_gap(lhs, pv);
                if (gap < gl[len]) gl[len] = gap;
                if (lhs <= pv) {
                    accepted = sc;
                } else {
                    /* residual r = norm(max(0, p - q~)), kept unnormalised with mass M */
                    const int64_t e = parent_expansion_of(c, gs);
                    tids = t->tail_ids + ((int64_t)b * E + e) * TL;
                    const float* tq = t->tail_q + ((int64_t)b * E + e) * TL;
                    double overlap = 0.0;
                    for (int i = 0; i < TL; ++i) {
                        float pt = P_OF(tids[i]);
                        rhat[i] = pt - tq[i] > 0.0f ? pt - tq[i] : 0.0f;
                        overlap += (double)(pt < tq[i] ? pt : tq[i]);
                        tail_pos[tids[i]] = i;
                    }
                    M = 1.0 - overlap;
                    use_tail = 1;
                    pool0 = gs - c->m;
                    if (c->plant_mode == ORC_PLANT_MASS_ON_SUPPORT) {
                        M = 0.0;
                        for (int i = 0; i < TL; ++i) M += (double)rhat[i];
                        for (int j = 0; j < c->m; ++j) M += (double)P_OF(t->token[nb + pool0 + j]);
                    }
                }
            }
            if (accepted < 0 && nc > 0) {
                /* recursive rejection over the remaining candidates in slot order */
                for (int k = 0; k < nc; ++k) {
                    const int v = fc + k;
                    if (v == sc) continue;
                    const int64_t gv = p->gen_id[pb + v];
                    const int tok = p->token[pb + v];
                    const float eta = orc_uniform(seed, offset, ORC_TAG_VERIFY, (int32_t)gu,
                                                  (uint64_t)(1 + slot_of(c, gv)));
                    float rv;
                    if (use_tail && tail_pos[tok] >= 0) rv = rhat[tail_pos[tok]];
                    else rv = P_OF(tok);
                    const double lhs = (double)eta * M;
                    double gap = rel_gap(lhs, rv);
                    if (gap < gl[len]) gl[len] = gap;
                    if (lhs <= (double)rv) { accepted = v; break; }
                    M -= (double)rv;
                    if (use_tail && tail_pos[tok] >= 0) rhat[tail_pos[tok]] = 0.0f;
                }
            }
        }
        if (accepted >= 0) {
            if (use_tail) for (int i = 0; i < TL; ++i) tail_pos[tids[i]] = -1;
            o->accepted_tokens[(int64_t)b * D + len] = p->token[pb + accepted];
            o->accepted_nodes[(int64_t)b * D + len] = accepted;
            ++len;
            u = accepted;
            continue;
        }
        /* final draw u* ~ r over tokens outside the candidate set (Gumbel-max) */
        int best = -1;
        float bk = -INFINITY, second = -INFINITY;
        for (int pass = 0; pass < 3 && best < 0; ++pass) {
            bk = -INFINITY; second = -INFINITY;
            for (int v = 0; v < V; ++v) {
                int excluded = 0;
                for (int k = 0; k < nc && pass < 2; ++k)
                    if (p->token[pb + fc + k] == v) { excluded = 1; break; }
                if (excluded) continue;
                if (pass == 0 && use_tail && c->plant_mode == ORC_PLANT_RESIDUAL_ON_SUPPORT && tail_pos[v] < 0) {
                    int lead = 0;
                    for (int j = 0; j < c->m; ++j) lead |= (t->token[nb + pool0 + j] == v);
                    if (!lead) continue;
                }
                const float g = gumbel(orc_uniform(seed, offset, ORC_TAG_RESIDUAL, (int32_t)gu, (uint64_t)v));
                const float tv = l[v] / T;
                float key;
                if (pass == 0 && use_tail && tail_pos[v] >= 0) {
                    const float rv = rhat[tail_pos[v]];
                    if (!(rv > 0.0f)) continue;
                    key = (float)log((double)rv) + g;
                } else if (pass == 0) {
                    key = (tv - lsef) + g;
                } else {
                    key = tv + g; /* rounding-only fallback: draw from p */
                }
                if (key > bk) { second = bk; bk = key; best = v; }
                else if (key > second) second = key;
            }
        }
        {
            double gap = rel_gap(bk, second);
            if (gap < gl[len]) gl[len] = gap;
        }
        if (use_tail) for (int i = 0; i < TL; ++i) tail_pos[tids[i]] = -1;
        o->bonus_token[b] = best;
        o->stop_mass[b] = (float)M;
#undef P_OF
        break;
    }
    o->accepted_len[b] = len;
    for (int i = len; i < D; ++i) {
        o->accepted_tokens[(int64_t)b * D + i] = -1;
        o->accepted_nodes[(int64_t)b * D + i] = -1;
    }
    free(lse); free(tail_pos); free(rhat);
    (void)K;
    return 0;
}

int orc_verify(const orc_cfg* c, const float* target, const float* T, const uint64_t* seed,
               const uint64_t* offset, const orc_tree* t, const orc_pruned* p, orc_verify_out* o) {
    if (orc_check_cfg(c)) return -1;
    for (int b = 0; b < c->B; ++b)
        if (!(T[b] > 0.0f) || isinf(T[b])) return -2;
    int err = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (int b = 0; b < c->B; ++b) {
        note_thread();
        if (verify_request(c, b, target, T[b], seed[b], offset[b], t, p, o)) err |= 1;
    }
    return err ? -2 : 0;
}

/* ------------------------------------------------------------------ */
/* whole cycles against prefix-indexed tables (Theorem 1 tests)         */
/* ------------------------------------------------------------------ */

static int64_t prefix_row(const int32_t* toks, int len, int V) {
    int64_t base = 0, pw = 1, val = 0;
    for (int i = 0; i < len; ++i) { base += pw; pw *= V; }
    for (int i = 0; i < len; ++i) val = val * V + toks[i];
    return base + val;
}

/* tokens on the path root -> node g (excluding the root) */
static int path_tokens(const orc_cfg* c, const orc_tree* t, int64_t g, int32_t* out) {
    int32_t rev[64];
    int n = 0;
    while (g != 0 && n < 64) { rev[n++] = t->token[g]; g = t->parent[g]; }
    for (int i = 0; i < n; ++i) out[i] = rev[n - 1 - i];
    (void)c;
    return n;
}

int orc_run_prefix_lm(const orc_cfg* c0, const float* draft_table, const float* target_table,
                      int32_t table_depth, int64_t n_trials, float T, uint64_t seed0, int32_t L,
                      int32_t* streams, int32_t* acc_len) {
    orc_cfg c = *c0;
    c.B = 1;
    if (orc_check_cfg(&c) || table_depth < c.D || table_depth < L - 1 || L < 1) return -1;
    const int V = c.V, K = c.K, D = c.D, N = c.N, TL = support_of(&c) - c.m;
    const int64_t G1 = orc_nodes_per_request(&c), E = orc_expansions_per_request(&c);
    int err = 0;
#pragma omp parallel for schedule(static) reduction(| : err)
    for (int64_t trial = 0; trial < n_trials; ++trial) {
        if (err) continue;
        orc_tree t;
        orc_pruned p;
        orc_verify_out o;
        t.token = (int32_t*)malloc(sizeof(int32_t) * G1);
        t.parent = (int32_t*)malloc(sizeof(int32_t) * G1);
        t.log_proxy = (float*)malloc(sizeof(float) * G1);
        t.score = (float*)malloc(sizeof(float) * G1);
        t.qtilde = (float*)malloc(sizeof(float) * G1);
        t.slot = (uint8_t*)malloc(G1);
        t.frontier = (int32_t*)malloc(sizeof(int32_t) * (K > 0 ? K : 1));
        t.tail_ids = (int32_t*)malloc(sizeof(int32_t) * E * TL);
        t.tail_q = (float*)malloc(sizeof(float) * E * TL);
        t.lse1 = (float*)malloc(sizeof(float) * E);
        t.gap_sample = (double*)malloc(sizeof(double) * E);
        t.gap_frontier = (double*)malloc(sizeof(double) * D);
        t.lse_tail = NULL;
        int32_t* pbuf = (int32_t*)malloc(sizeof(int32_t) * 7 * (N + 1));
        p.gen_id = pbuf; p.token = pbuf + (N + 1); p.parent = pbuf + 2 * (N + 1);
        p.depth = pbuf + 3 * (N + 1); p.first_child = pbuf + 4 * (N + 1);
        p.n_child = pbuf + 5 * (N + 1); p.sampled_child = pbuf + 6 * (N + 1);
        double gp;
        p.gap_prune = &gp;
        int32_t alen, bonus;
        int32_t* atok = (int32_t*)malloc(sizeof(int32_t) * D);
        int32_t* anode = (int32_t*)malloc(sizeof(int32_t) * D);
        float* rlse = (float*)malloc(sizeof(float) * (N + 1));
        double* glv = (double*)malloc(sizeof(double) * (D + 1));
        float smass;
        o.accepted_len = &alen; o.accepted_tokens = atok; o.accepted_nodes = anode;
        o.bonus_token = &bonus; o.row_lse = rlse; o.gap_level = glv; o.stop_mass = &smass;
        float* rows = (float*)malloc(sizeof(float) * (size_t)(K > 0 ? K : 1) * V);
        float* trows = (float*)malloc(sizeof(float) * (size_t)(N + 1) * V);
        int32_t path[64];
        const uint64_t seed = seed0 + (uint64_t)trial, off = 0;
        int rc = 0;
        for (int d = 1; d <= D && !rc; ++d) {
            int F = rows_at_depth(&c, d);
            for (int f = 0; f < F; ++f) {
                int64_t g = (d == 1) ? 0 : t.frontier[f];
                int n = path_tokens(&c, &t, g, path);
                memcpy(rows + (int64_t)f * V, draft_table + prefix_row(path, n, V) * V, sizeof(float) * V);
            }
            rc = orc_expand(&c, d, rows, &T, &seed, &off, &t);
        }
        if (!rc) rc = orc_prune(&c, &t, &p);
        if (!rc) {
            for (int u = 0; u <= N; ++u) {
                int n = path_tokens(&c, &t, p.gen_id[u], path);
                memcpy(trows + (int64_t)u * V, target_table + prefix_row(path, n, V) * V, sizeof(float) * V);
            }
            rc = orc_verify(&c, trows, &T, &seed, &off, &t, &p, &o);
        }
        if (!rc) {
            int32_t* st = streams + trial * L;
            int n = 0;
            for (int i = 0; i < alen && n < L; ++i) st[n++] = atok[i];
            if (n < L) st[n++] = bonus;
            while (n < L) {
                const float* row = target_table + prefix_row(st, n, V) * V;
                int best = -1;
                float bk = -INFINITY;
                for (int v = 0; v < V; ++v) {
                    float key = row[v] / T + gumbel(orc_uniform(seed, off, ORC_TAG_CONTINUE, n, (uint64_t)v));
                    if (key > bk) { bk = key; best = v; }
                }
                st[n++] = best;
            }
            acc_len[trial] = alen;
        } else {
            err |= 1;
        }
        free(t.token); free(t.parent); free(t.log_proxy); free(t.score); free(t.qtilde); free(t.slot);
        free(t.frontier); free(t.tail_ids); free(t.tail_q); free(t.lse1); free(t.gap_sample);
        free(t.gap_frontier); free(pbuf); free(atok); free(anode); free(rlse); free(glv);
        free(rows); free(trows);
    }
    return err ? -2 : 0;
}
