// api.cu -- the extern "C" entry points declared in include/rheo.h.
//
// Host side only: argument validation, the workspace layout, kernel selection
// (dtype x 16-byte alignment) and launches on the caller's stream.  No
// allocation, no synchronisation except in rheo_get_status.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>

#include "config_dims.h"
#include "rheo.h"
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {
namespace {

int64_t nodes_per_request(const rheo_config& c) {
    return 1 + (int64_t)(c.K + 1) + (int64_t)(c.depth - 1) * c.K * (c.K + 1);
}
int64_t expansions_per_request(const rheo_config& c) { return 1 + (int64_t)(c.depth - 1) * c.K; }
int elem_size(const rheo_config& c) { return c.dtype == RHEO_BF16 ? 2 : 4; }
int tiles_per_row(const rheo_config& c) {
    const int te = expand_tile_elems(c.dtype == RHEO_BF16 ? 1 : 0);
    return (c.vocab + te - 1) / te;
}

bool valid(const rheo_config* c) {
    if (!c) return false;
    if (c->dtype != RHEO_F32 && c->dtype != RHEO_BF16) return false;
    if (c->batch < 1 || c->vocab < 1 || c->vocab > kMaxVocab) return false;
    if (c->K < 0 || c->m < 0 || c->m > c->K) return false;
    if (c->support == 0) {  // full support: the sampled token over the whole vocabulary
        if (c->K + 1 > c->vocab || c->K + 1 > kMaxSupport || c->m > 1) return false;
    } else if (c->support < c->K + 1 || c->support > c->vocab || c->support > kMaxSupport) {
        return false;
    }
    if (c->depth < 1 || (c->K == 0 && c->depth > 1)) return false;
    const int64_t G1 = nodes_per_request(*c);
    if (G1 > kMaxNodes) return false;
    if (c->budget < 1 || c->budget > G1 - 1) return false;
    if (c->m == 0 && !(c->eps > 0.0f && c->eps < 1.0f)) return false;
    const int64_t F = c->K > 0 ? c->K : 1;
    if ((int64_t)c->batch * F > 65535 || (int64_t)c->batch * (c->budget + 1) > 65535) return false;
    return true;
}

struct Layout {
    size_t status, ex_row_ticket, ex_req_ticket, ex_mu, ex_sum, ex_keys, ex_ltail, ex_grp;
    size_t v_mu, v_sum, v_queue, v_hdr, v_child, v_tids, v_tq, v_cx, v_tx, v_coin, v_table, v_rhat, r_best,
        r_ticket;
    size_t total;
};

size_t up(size_t x) { return (x + 255) & ~(size_t)255; }

Layout layout(const rheo_config& c) {
    const int64_t B = c.batch, F = c.K > 0 ? c.K : 1, P = tiles_per_row(c), S = c.support == 0 ? c.K + 1 : c.support;
    const int64_t NP = c.budget + 1, TL = c.support == 0 ? 0 : c.support - c.m;
    const int64_t VC = verify_chunks_per_row(c.dtype == RHEO_BF16 ? 1 : 0, c.vocab);
    Layout L{};
    size_t o = 0;
    auto take = [&](size_t bytes) { size_t at = o; o = up(o + bytes); return at; };
    L.status = take(sizeof(unsigned));
    L.ex_row_ticket = take(sizeof(unsigned) * B * F);
    L.ex_req_ticket = take(sizeof(unsigned) * B);
    L.ex_mu = take(sizeof(float) * B * F * P);
    L.ex_sum = take(2 * sizeof(float) * B * F * P);
    L.ex_keys = take(sizeof(unsigned long long) * B * F * P * S);
    L.ex_ltail = take(2 * sizeof(float) * B * expansions_per_request(c));
    const int64_t GT = full_group_tokens(c.dtype == RHEO_BF16 ? 1 : 0);
    const int64_t FG = c.support == 0 ? B * F * ((c.vocab + GT - 1) / GT) : 0;  // full support's group sums
    L.ex_grp = take(2 * sizeof(float) * FG);
    L.v_mu = take(sizeof(float) * B * NP * VC);
    L.v_sum = take(2 * sizeof(float) * B * NP * VC);
    L.v_queue = take(sizeof(unsigned) * kStreamQueues * kStreamQueueStride);
    L.v_hdr = take(sizeof(int) * B * NP * 8);
    L.v_child = take(sizeof(int) * B * NP * (c.K + 1) * 3);
    L.v_tids = take(sizeof(int) * B * NP * TL);
    L.v_tq = take(sizeof(float) * B * NP * TL);
    L.v_cx = take(2 * sizeof(float) * B * NP * (c.K + 1));
    L.v_tx = take(2 * sizeof(float) * B * NP * TL);
    L.v_coin = take(sizeof(float) * B * NP * (c.K + 2));
    L.v_table = take(sizeof(float) * B * NP * verify_table_width(c.K));
    L.v_rhat = take(sizeof(float) * B * NP * TL);
    L.r_best = take(sizeof(unsigned long long) * B * 3);
    L.r_ticket = take(sizeof(unsigned) * B);
    L.total = o;
    return L;
}

int sm_count() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                   cudaSuccess || sms < 1)
        return 1;
    return sms;
}

// largest number of segments any row is cut into by the tile split
int max_segments(int64_t rows, int tpr, int grid) {
    const int64_t total = rows * tpr;
    auto owner = [&](int64_t t) { return (int)((t * grid + grid - 1) / total); };
    int best = 1;
    for (int64_t r = 0; r < rows; ++r) {
        const int s = owner(r * tpr + tpr - 1) - owner(r * tpr) + 1;
        best = s > best ? s : best;
    }
    return best;
}

// rows start on 16-byte boundaries (16-byte vector loads; a row's ragged end is read element-wise)
bool rows_aligned(const void* p, int64_t row_stride, const rheo_config& c) {
    return ((uintptr_t)p % 16 == 0) && ((row_stride * elem_size(c)) % 16 == 0);
}


}  // namespace

Dims config_dims(const rheo_config& c) {
    Dims n;
    n.B = c.batch; n.V = c.vocab; n.K = c.K; n.m = c.m; n.S = c.support; n.D = c.depth; n.N = c.budget;
    n.full = c.support == 0 ? 1 : 0;
    if (n.full) n.S = c.K + 1;  // ranks selected: the leads and the fill candidates
    n.TL = n.full ? 0 : c.support - c.m;
    n.GW = (c.K + 1) + n.TL;
    n.chunks = tiles_per_row(c);
    n.G1 = nodes_per_request(c);
    n.E = expansions_per_request(c);
    n.eps = c.eps;
    return n;
}

TreePtrs tree_ptrs(const rheo_tree* t) {
    return TreePtrs{t->token, t->parent, t->log_proxy, t->score, t->qtilde, t->slot,
                    t->frontier, t->tail_ids, t->tail_q, t->lse1, t->lse_tail};
}
PrunedPtrs pruned_ptrs(const rheo_pruned* p) {
    return PrunedPtrs{p->gen_id, p->token, p->parent, p->depth, p->first_child, p->n_child, p->sampled_child};
}

namespace {

bool tree_ok(const rheo_tree* t, const rheo_config& c) {
    if (!(t && t->token && t->parent && t->log_proxy && t->score && t->qtilde && t->slot && t->frontier && t->lse1))
        return false;
    return c.support == 0 ? t->lse_tail != nullptr : (t->tail_ids && t->tail_q);
}
bool pruned_ok(const rheo_pruned* p) {
    return p && p->gen_id && p->token && p->parent && p->depth && p->first_child && p->n_child && p->sampled_child;
}

template <class T> T* at(void* ws, size_t off) { return reinterpret_cast<T*>(static_cast<char*>(ws) + off); }

}  // namespace
}  // namespace rheo

using namespace rheo;

extern "C" int rheo_sizes(const rheo_config* cfg, int64_t* nodes, int64_t* expansions, size_t* ws_bytes) {
    if (!valid(cfg)) return RHEO_EINVAL;
    if (nodes) *nodes = nodes_per_request(*cfg);
    if (expansions) *expansions = expansions_per_request(*cfg);
    if (ws_bytes) *ws_bytes = layout(*cfg).total;
    return RHEO_OK;
}

extern "C" int rheo_workspace_init(const rheo_config* cfg, void* ws, size_t bytes, rheo_stream_t stream) {
    if (!valid(cfg) || !ws || bytes < layout(*cfg).total) return RHEO_EINVAL;
    return cudaMemsetAsync(ws, 0, layout(*cfg).total, (cudaStream_t)stream) == cudaSuccess ? RHEO_OK : RHEO_ELAUNCH;
}

extern "C" int rheo_expand(const rheo_config* cfg, int32_t d, const void* logits, int64_t row_stride,
                           const float* temperature, const uint64_t* seed, const uint64_t* offset,
                           const rheo_tree* tree, void* ws, rheo_stream_t stream) {
    if (!valid(cfg) || d < 1 || d > cfg->depth || !logits || row_stride < cfg->vocab || !temperature || !seed ||
        !offset || !tree_ok(tree, *cfg) || !ws)
        return RHEO_EINVAL;
    const Layout L = layout(*cfg);
    ExpandArgs a;
    a.n = config_dims(*cfg);
    a.d = d;
    a.F = (d == 1) ? 1 : cfg->K;
    a.logits = static_cast<const char*>(logits);
    a.row_stride_bytes = row_stride * elem_size(*cfg);
    a.T = temperature;
    a.seed = seed;
    a.offset = offset;
    a.tree = tree_ptrs(tree);
    a.status = at<unsigned>(ws, L.status);
    a.row_ticket = at<unsigned>(ws, L.ex_row_ticket);
    a.req_ticket = at<unsigned>(ws, L.ex_req_ticket);
    a.seg_mu = at<float>(ws, L.ex_mu);
    a.seg_sum = at<float>(ws, L.ex_sum);
    a.seg_keys = at<unsigned long long>(ws, L.ex_keys);
    a.lse_tail_ff = at<float>(ws, L.ex_ltail);
    a.grp = at<float>(ws, L.ex_grp);
    const int tpr = tiles_per_row(*cfg);
    const int64_t rows = (int64_t)cfg->batch * a.F;
    const int sms = sm_count();
    // Launch shape: one CTA of 16 warps per SM.  Up to one row per SM: every
    // row is cut into P equal segments (P CTAs, P = SMs / rows), so a CTA holds
    // one segment and P = 1 needs no merge.  More rows: one CTA per SM, rows
    // cut where the even split of the tiles falls.
    int grid;
    if (rows <= sms) {
        const int64_t P = std::max<int64_t>(1, std::min<int64_t>(tpr, sms / rows));
        grid = (int)(rows * P);
    } else {
        grid = (int)std::min<int64_t>(rows * tpr, (int64_t)sms);
    }
    const int segs = max_segments(rows, tpr, grid);
    a.keys_bytes = expand_keys_bytes(segs, a.n.S);
    const size_t smem = expand_smem_bytes(segs, a.n.S);
    if (smem + 8 * 1024 > 227 * 1024) return RHEO_EINVAL;
    return launch_expand(a, cfg->dtype, rows_aligned(logits, row_stride, *cfg), cfg->support == 0, grid, smem,
                         (cudaStream_t)stream) ==
                   cudaSuccess
               ? RHEO_OK
               : RHEO_ELAUNCH;
}

extern "C" int rheo_prune(const rheo_config* cfg, const rheo_tree* tree, const rheo_pruned* pruned, void* ws,
                          rheo_stream_t stream) {
    if (!valid(cfg) || !tree_ok(tree, *cfg) || !pruned_ok(pruned) || !ws) return RHEO_EINVAL;
    const Layout L = layout(*cfg);
    PruneArgs a;
    a.n = config_dims(*cfg);
    a.tree = tree_ptrs(tree);
    a.pr = pruned_ptrs(pruned);
    a.status = at<unsigned>(ws, L.status);
    size_t smem = (sizeof(int32_t) + sizeof(unsigned long long)) * (size_t)a.n.G1 +
                  5 * sizeof(int32_t) * (size_t)(cfg->budget + 1);
    // the nodes' parent, token and slot beside the keys when that still fits
    const size_t staged = smem + (2 * sizeof(int32_t) + sizeof(uint8_t)) * (size_t)a.n.G1;
    a.staged = staged <= 160 * 1024 ? 1 : 0;
    if (a.staged) smem = staged;
    return launch_prune(a, cfg->batch, smem, (cudaStream_t)stream) == cudaSuccess ? RHEO_OK : RHEO_ELAUNCH;
}

extern "C" int rheo_tree_attention(const rheo_config* cfg, const rheo_pruned* pruned, const rheo_tree_attn* out,
                                   void* ws, rheo_stream_t stream) {
    if (!valid(cfg) || !pruned || !pruned->parent || !pruned->depth || !pruned->n_child || !out || !ws ||
        cfg->budget + 1 > 4096)
        return RHEO_EINVAL;
    if (!out->mask && !out->position && !out->retrieve && !out->n_leaves) return RHEO_OK;
    const Layout L = layout(*cfg);
    TreeAttnArgs a;
    a.n = config_dims(*cfg);
    a.pr = pruned_ptrs(pruned);
    a.mask = out->mask;
    a.position = out->position;
    a.retrieve = out->retrieve;
    a.n_leaves = out->n_leaves;
    a.status = at<unsigned>(ws, L.status);
    return launch_tree_attn(a, cfg->batch, tree_attn_smem_bytes(cfg->budget), (cudaStream_t)stream) == cudaSuccess
               ? RHEO_OK
               : RHEO_ELAUNCH;
}

extern "C" int rheo_verify_variant(const rheo_config* cfg, int32_t variant, const void* logits, int64_t row_stride,
                                   const float* temperature, const uint64_t* seed, const uint64_t* offset,
                                   const rheo_tree* tree, const rheo_pruned* pruned, const rheo_verify_out* out,
                                   void* ws, rheo_stream_t stream) {
    if (variant != RHEO_VERIFY_RHEO && variant != RHEO_VERIFY_RRSW && variant != RHEO_VERIFY_ONEHOT) return RHEO_EINVAL;
    if (cfg && cfg->support == 0) return RHEO_EINVAL;  // full support verifies through rheo_verify_full
    if (!valid(cfg) || !logits || row_stride < cfg->vocab || !temperature || !seed || !offset || !tree_ok(tree, *cfg) ||
        !pruned_ok(pruned) || !out || !out->accepted_len || !out->accepted_tokens || !out->accepted_nodes ||
        !out->bonus_token || !ws)
        return RHEO_EINVAL;
    const Layout L = layout(*cfg);
    VerifyArgs a;
    a.n = config_dims(*cfg);
    a.variant = variant == RHEO_VERIFY_RRSW ? kVerifyRrsw : variant == RHEO_VERIFY_ONEHOT ? kVerifyOneHot : kVerifyRheo;
    a.logits = static_cast<const char*>(logits);
    a.row_stride_bytes = row_stride * elem_size(*cfg);
    a.T = temperature;
    a.seed = seed;
    a.offset = offset;
    a.tree = tree_ptrs(tree);
    a.pr = pruned_ptrs(pruned);
    a.accepted_len = out->accepted_len;
    a.accepted_tokens = out->accepted_tokens;
    a.accepted_nodes = out->accepted_nodes;
    a.bonus_token = out->bonus_token;
    a.row_lse = out->row_lse;
    a.status = at<unsigned>(ws, L.status);
    a.seg_mu = at<float>(ws, L.v_mu);
    a.seg_sum = at<float>(ws, L.v_sum);
    a.queue = at<unsigned>(ws, L.v_queue);
    a.rec_hdr = at<int>(ws, L.v_hdr);
    a.rec_child = at<int>(ws, L.v_child);
    a.rec_tids = at<int>(ws, L.v_tids);
    a.rec_tq = at<float>(ws, L.v_tq);
    a.rec_cx = at<float>(ws, L.v_cx);
    a.rec_tx = at<float>(ws, L.v_tx);
    a.rec_coin = at<float>(ws, L.v_coin);
    a.table = at<float>(ws, L.v_table);
    a.rhat_tail = at<float>(ws, L.v_rhat);
    a.res_best = at<unsigned long long>(ws, L.r_best);
    a.res_ticket = at<unsigned>(ws, L.r_ticket);
    const int64_t NP = cfg->budget + 1;
    a.n.chunks = verify_chunks_per_row(cfg->dtype == RHEO_BF16 ? 1 : 0, cfg->vocab);
    const int64_t chunks = (int64_t)cfg->batch * NP * a.n.chunks;
    const int grid = verify_stream_grid(sm_count(), chunks);
    return launch_verify(a, cfg->dtype, rows_aligned(logits, row_stride, *cfg), grid, (cudaStream_t)stream) ==
                   cudaSuccess
               ? RHEO_OK
               : RHEO_ELAUNCH;
}

extern "C" int rheo_verify_full(const rheo_config* cfg, const void* logits, int64_t row_stride,
                                const void* const* draft_logits, int64_t draft_row_stride, const float* temperature,
                                const uint64_t* seed, const uint64_t* offset, const rheo_tree* tree,
                                const rheo_pruned* pruned, const rheo_verify_out* out, void* ws, rheo_stream_t stream) {
    if (!cfg || cfg->support != 0 || cfg->depth > kMaxFullDepth || !draft_logits || draft_row_stride < cfg->vocab)
        return RHEO_EINVAL;
    for (int d = 0; d < cfg->depth; ++d)
        if (!draft_logits[d]) return RHEO_EINVAL;
    if (!valid(cfg) || !logits || row_stride < cfg->vocab || !temperature || !seed || !offset || !tree_ok(tree, *cfg) ||
        !pruned_ok(pruned) || !out || !out->accepted_len || !out->accepted_tokens || !out->accepted_nodes ||
        !out->bonus_token || !ws)
        return RHEO_EINVAL;
    const Layout L = layout(*cfg);
    VerifyArgs a;
    a.n = config_dims(*cfg);
    a.variant = kVerifyRheo;
    bool draft_aligned = (draft_row_stride * elem_size(*cfg)) % 16 == 0;
    for (int d = 0; d < cfg->depth; ++d) {
        a.draft[d] = static_cast<const char*>(draft_logits[d]);
        draft_aligned = draft_aligned && (reinterpret_cast<uintptr_t>(draft_logits[d]) % 16 == 0);
    }
    a.draft_row_stride_bytes = draft_row_stride * elem_size(*cfg);
    a.lse_tail_ff = at<float>(ws, L.ex_ltail);
    a.logits = static_cast<const char*>(logits);
    a.row_stride_bytes = row_stride * elem_size(*cfg);
    a.T = temperature;
    a.seed = seed;
    a.offset = offset;
    a.tree = tree_ptrs(tree);
    a.pr = pruned_ptrs(pruned);
    a.accepted_len = out->accepted_len;
    a.accepted_tokens = out->accepted_tokens;
    a.accepted_nodes = out->accepted_nodes;
    a.bonus_token = out->bonus_token;
    a.row_lse = out->row_lse;
    a.status = at<unsigned>(ws, L.status);
    a.seg_mu = at<float>(ws, L.v_mu);
    a.seg_sum = at<float>(ws, L.v_sum);
    a.queue = at<unsigned>(ws, L.v_queue);
    a.rec_hdr = at<int>(ws, L.v_hdr);
    a.rec_child = at<int>(ws, L.v_child);
    a.rec_tids = at<int>(ws, L.v_tids);
    a.rec_tq = at<float>(ws, L.v_tq);
    a.rec_cx = at<float>(ws, L.v_cx);
    a.rec_tx = at<float>(ws, L.v_tx);
    a.rec_coin = at<float>(ws, L.v_coin);
    a.table = at<float>(ws, L.v_table);
    a.rhat_tail = at<float>(ws, L.v_rhat);
    a.res_best = at<unsigned long long>(ws, L.r_best);
    a.res_ticket = at<unsigned>(ws, L.r_ticket);
    const int64_t NP = cfg->budget + 1;
    a.n.chunks = verify_chunks_per_row(cfg->dtype == RHEO_BF16 ? 1 : 0, cfg->vocab);
    const int64_t chunks = (int64_t)cfg->batch * NP * a.n.chunks;
    const int grid = verify_stream_grid(sm_count(), chunks);
    return launch_verify_full(a, cfg->dtype, rows_aligned(logits, row_stride, *cfg), draft_aligned, grid,
                              (cudaStream_t)stream) ==
                   cudaSuccess
               ? RHEO_OK
               : RHEO_ELAUNCH;
}

extern "C" int rheo_verify(const rheo_config* cfg, const void* logits, int64_t row_stride, const float* temperature,
                           const uint64_t* seed, const uint64_t* offset, const rheo_tree* tree,
                           const rheo_pruned* pruned, const rheo_verify_out* out, void* ws, rheo_stream_t stream) {
    return rheo_verify_variant(cfg, RHEO_VERIFY_RHEO, logits, row_stride, temperature, seed, offset, tree, pruned, out,
                               ws, stream);
}

extern "C" int rheo_get_status(const rheo_config* cfg, void* ws, rheo_stream_t stream, int32_t* status) {
    if (!valid(cfg) || !ws || !status) return RHEO_EINVAL;
    const Layout L = layout(*cfg);
    cudaStream_t s = (cudaStream_t)stream;
    unsigned host = 0;
    if (cudaMemcpyAsync(&host, at<unsigned>(ws, L.status), sizeof(unsigned), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return RHEO_ELAUNCH;
    if (cudaMemsetAsync(at<unsigned>(ws, L.status), 0, sizeof(unsigned), s) != cudaSuccess) return RHEO_ELAUNCH;
    if (cudaStreamSynchronize(s) != cudaSuccess) return RHEO_ELAUNCH;
    *status = (int32_t)host;
    return RHEO_OK;
}
