// noalloc.cu -- rheo_verify_static: verification without a caller workspace.
//
// Some callers cannot allocate device memory at the point where they verify:
// code handed only pre-sized input and output buffers by a host framework
// (an inference-engine plugin, a custom operator), runtimes whose device memory
// is fully partitioned up front, or latency-critical loops that must not hit
// the implicit synchronisation of cudaMalloc.  This entry point runs exactly
// the kernels of rheo_verify, with their scratch state in the file-scope array
// below instead of a workspace.  It allocates nothing.
//
// The array is a static device variable: every GPU that loads this library
// holds its kStaticScratchBytes until the process exits.  Its device address is
// looked up once per device, by the first call made on that device (with that
// device current); make that first call before any stream capture.  The address
// is cached for the life of the process: it does not survive a
// cudaDeviceReset (or any other teardown of the device's primary context), after
// which this entry point must not be called again in the same process.  All calls
// share the array and it keeps the last call's contents, so calls whose work
// overlaps on the GPU (other streams, other threads) race on it: serialise them.
#include <cuda_runtime.h>

#include <cstdint>

#include "config_dims.h"
#include "rheo.h"
#include "rheo_device.cuh"
#include "rheo_kernels.h"

namespace rheo {
namespace {

constexpr size_t kStaticScratchBytes = RHEO_STATIC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// device address of the array in the current context, looked up on every call
// (a runtime lookup, no allocation): an address kept across calls would go
// stale after the context is torn down and made again (cudaDeviceReset)
void* scratch_address() {
    void* ptr = nullptr;
    return cudaGetSymbolAddress(&ptr, g_static_scratch) == cudaSuccess ? ptr : nullptr;
}

size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

// the verification part of the workspace layout, laid out in the static array
struct StaticLayout {
    size_t status, mu, sum, queue, hdr, child, tids, tq, cx, tx, coin, table, rhat, best, res_ticket, total,
        clear_end;
};

StaticLayout static_layout(const rheo_config& c) {
    const int64_t B = c.batch, NP = c.budget + 1, TL = c.support - c.m;
    const int64_t P = verify_chunks_per_row(c.dtype == RHEO_BF16 ? 1 : 0, c.vocab);
    StaticLayout L{};
    size_t o = 0;
    auto take = [&](size_t bytes) { size_t at = o; o = up256(o + bytes); return at; };
    // everything that must start at zero first, so one memset clears it
    L.status = take(sizeof(unsigned));
    L.queue = take(sizeof(unsigned) * kStreamQueues * kStreamQueueStride);
    L.best = take(sizeof(unsigned long long) * B * 3);
    L.res_ticket = take(sizeof(unsigned) * B);
    L.clear_end = o;
    L.mu = take(sizeof(float) * B * NP * P);
    L.sum = take(2 * sizeof(float) * B * NP * P);
    L.table = take(sizeof(float) * B * NP * verify_table_width(c.K));
    L.rhat = take(sizeof(float) * B * NP * TL);
    L.hdr = take(sizeof(int) * B * NP * 8);
    L.child = take(sizeof(int) * B * NP * (c.K + 1) * 3);
    L.tids = take(sizeof(int) * B * NP * TL);
    L.tq = take(sizeof(float) * B * NP * TL);
    L.cx = take(2 * sizeof(float) * B * NP * (c.K + 1));
    L.tx = take(2 * sizeof(float) * B * NP * TL);
    L.coin = take(sizeof(float) * B * NP * (c.K + 2));
    L.total = o;
    return L;
}

bool config_ok(const rheo_config* c) {
    size_t ws = 0;
    return rheo_sizes(c, nullptr, nullptr, &ws) == RHEO_OK;
}

bool buffers_ok(const rheo_tree* t, const rheo_pruned* p, const rheo_verify_out* o) {
    return t && t->token && t->parent && t->log_proxy && t->score && t->qtilde && t->slot && t->frontier &&
           t->tail_ids && t->tail_q && t->lse1 && p && p->gen_id && p->token && p->parent && p->depth &&
           p->first_child && p->n_child && p->sampled_child && o && o->accepted_len && o->accepted_tokens &&
           o->accepted_nodes && o->bonus_token;
}

}  // namespace
}  // namespace rheo

using namespace rheo;

extern "C" int rheo_verify_static(const rheo_config* cfg, const void* logits, int64_t row_stride,
                                  const float* temperature, const uint64_t* seed, const uint64_t* offset,
                                  const rheo_tree* tree, const rheo_pruned* pruned, const rheo_verify_out* out,
                                  int32_t* status, rheo_stream_t stream) {
    if (!config_ok(cfg) || cfg->support == 0 || !logits || row_stride < cfg->vocab || !temperature || !seed ||
        !offset || !buffers_ok(tree, pruned, out))
        return RHEO_EINVAL;
    const StaticLayout L = static_layout(*cfg);
    if (L.total > kStaticScratchBytes) return RHEO_ETOOLARGE;
    unsigned char* base = static_cast<unsigned char*>(scratch_address());
    if (!base) return RHEO_ELAUNCH;
    cudaStream_t s = (cudaStream_t)stream;
    // the previous call's counters and status must not leak into this one
    if (cudaMemsetAsync(base, 0, L.clear_end, s) != cudaSuccess) return RHEO_ELAUNCH;

    VerifyArgs a;
    a.n = config_dims(*cfg);  // the same dimensions as every other entry point
    a.n.chunks = verify_chunks_per_row(cfg->dtype == RHEO_BF16 ? 1 : 0, cfg->vocab);
    const int es = cfg->dtype == RHEO_BF16 ? 2 : 4;
    a.logits = static_cast<const char*>(logits);
    a.row_stride_bytes = row_stride * es;
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
    a.status = reinterpret_cast<unsigned*>(base + L.status);
    a.seg_mu = reinterpret_cast<float*>(base + L.mu);
    a.seg_sum = reinterpret_cast<float*>(base + L.sum);
    a.queue = reinterpret_cast<unsigned*>(base + L.queue);
    a.rec_hdr = reinterpret_cast<int*>(base + L.hdr);
    a.rec_child = reinterpret_cast<int*>(base + L.child);
    a.rec_tids = reinterpret_cast<int*>(base + L.tids);
    a.rec_tq = reinterpret_cast<float*>(base + L.tq);
    a.rec_cx = reinterpret_cast<float*>(base + L.cx);
    a.rec_tx = reinterpret_cast<float*>(base + L.tx);
    a.rec_coin = reinterpret_cast<float*>(base + L.coin);
    a.table = reinterpret_cast<float*>(base + L.table);
    a.rhat_tail = reinterpret_cast<float*>(base + L.rhat);
    a.res_best = reinterpret_cast<unsigned long long*>(base + L.best);
    a.res_ticket = reinterpret_cast<unsigned*>(base + L.res_ticket);
    int sms = 1, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return RHEO_ELAUNCH;
    const int64_t chunks = (int64_t)cfg->batch * (cfg->budget + 1) * a.n.chunks;
    const int grid = verify_stream_grid(sms, chunks);
    const bool aligned = ((uintptr_t)logits % 16 == 0) && ((row_stride * es) % 16 == 0);
    if (launch_verify(a, cfg->dtype, aligned, grid, s) != cudaSuccess) return RHEO_ELAUNCH;
    if (status && cudaMemcpyAsync(status, base + L.status, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return RHEO_ELAUNCH;
    return RHEO_OK;
}
