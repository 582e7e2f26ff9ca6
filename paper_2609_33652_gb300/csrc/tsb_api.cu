// C ABI of libtsb (include/tsb.h): argument validation, workspace layout and kernel
// launches on the caller's stream. Nothing is launched unless every check passes.
#include <math.h>
#include <stdint.h>


#include "../../include/tsb.h"
#include "tsb_launch.h"

namespace {

constexpr size_t kStatusBytes = tsb::kWsStatusBytes;  // status word region at the start of the workspace

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int64_t max_nodes(int K, int L) {
    int64_t total = 0, level = 1;
    for (int d = 1; d <= L; ++d) {
        level *= K;
        total += level;
        if (total > (int64_t)1 << 40) break;
    }
    return total;
}

tsb_status check_cfg(const tsb_cfg *c) {
    if (!c) return TSB_ERR_ARG;
    if (!(c->temperature > 0.0f) || !isfinite(c->temperature)) return TSB_ERR_ARG;
    if (c->B < 1 || c->B > TSB_MAX_B || c->L < 1 || c->L > TSB_MAX_L || c->K < 1 || c->K > TSB_MAX_K ||
        c->N < 1 || c->N > TSB_MAX_N || c->V < 1 || c->V > TSB_MAX_V || c->K > c->V)
        return TSB_ERR_SHAPE;
    if ((int64_t)c->N > max_nodes(c->K, c->L)) return TSB_ERR_SHAPE;
    return TSB_OK;
}

// rows must hold at least B trees x R rows x V logits, 16-byte aligned rows
tsb_status check_logits(const tsb_logits *t, int B, int R_min, int V) {
    if (!t || !t->data) return TSB_ERR_ARG;
    if (t->dtype != TSB_F32 && t->dtype != TSB_BF16) return TSB_ERR_DTYPE;
    if (t->B != B || t->V != V || t->R < R_min || t->R < 1 || t->row_stride < t->V || t->batch_stride < 0)
        return TSB_ERR_SHAPE;
    const int64_t es = t->dtype == TSB_BF16 ? 2 : 4;
    if (!aligned(t->data, 16) || (t->row_stride * es) % 16 != 0 || (t->batch_stride * es) % 16 != 0)
        return TSB_ERR_ALIGN;
    return TSB_OK;
}

tsb::RowsDesc rows_of(const tsb_logits *t) {
    tsb::RowsDesc r;
    r.data = t->data;
    r.dtype = t->dtype;
    r.B = t->B;
    r.R = t->R;
    r.V = t->V;
    r.batch_stride = t->batch_stride;
    r.row_stride = t->row_stride;
    return r;
}

tsb::TreeDesc tree_of(const tsb_tree *t) {
    tsb::TreeDesc d;
    d.parent = t->parent;
    d.depth = t->depth;
    d.rank = t->rank;
    d.plan_token = t->plan_token;
    d.score = t->score;
    d.child_off = t->child_off;
    d.child_ids = t->child_ids;
    return d;
}

size_t ws_bytes_for(const tsb_cfg *c) { return tsb::workspace_bytes(c->B, c->N, c->L, c->K); }

tsb_status check_ws(void *ws, size_t ws_bytes, size_t need) {
    if (!ws) return TSB_ERR_ARG;
    if (!aligned(ws, 256) || ws_bytes < need) return TSB_ERR_WORKSPACE;
    return TSB_OK;
}

tsb_status check_stats(const void *stats, size_t bytes, int B, int R, int V) {
    if (!stats) return TSB_ERR_ARG;
    if (!aligned(stats, 16) || bytes < tsb_stats_bytes(B, R, V)) return TSB_ERR_WORKSPACE;
    return TSB_OK;
}

tsb_status cuda_status(cudaError_t e) { return e == cudaSuccess ? TSB_OK : TSB_ERR_CUDA; }

float inv_temperature(float T) { return 1.0f / T; }

// expand-then-prune: width in range, between N and kEptMaxCandidates candidates generated
tsb_status check_width(const tsb_cfg *c, int32_t width) {
    if (width < 1 || width > TSB_MAX_WIDTH) return TSB_ERR_SHAPE;
    const int64_t G = tsb::ept_layer_start(c->L + 1, c->K, width);
    if (G < c->N || G > tsb::kEptMaxCandidates) return TSB_ERR_SHAPE;
    return TSB_OK;
}

tsb_status plan_expand_common(const tsb_cfg *cfg, int32_t width, const tsb_logits *draft, const void *stats_in,
                              void *stats_out, size_t stats_bytes, const tsb_tree *out, void *ws, size_t ws_bytes,
                              tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_width(cfg, width);
    if (st != TSB_OK) return st;
    st = check_logits(draft, cfg->B, cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(stats_in ? stats_in : stats_out, stats_bytes, cfg->B, draft->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!out || !out->parent || !out->depth || !out->rank || !out->plan_token || !out->score || !out->child_off ||
        !out->child_ids)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_plan_expand(rows_of(draft), static_cast<const float2 *>(stats_in),
                                               static_cast<float2 *>(stats_out), cfg->L, cfg->N, cfg->K, width,
                                               inv_temperature(cfg->temperature), tree_of(out), ws,
                                               (cudaStream_t)stream));
}

// pooled draft laws: K <= P <= TSB_MAX_POOL, P <= V
tsb_status check_pool(const tsb_cfg *c, int32_t P) {
    if (P < c->K || P > TSB_MAX_POOL || P > c->V) return TSB_ERR_SHAPE;
    return TSB_OK;
}

tsb_status replay_common(bool mixed, const tsb_cfg *cfg, const tsb_logits *qrows, const void *qstats,
                         size_t stats_bytes, const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed,
                         int32_t *token, void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_logits(qrows, cfg->B, qrow_of_node ? 1 : cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(qstats, stats_bytes, cfg->B, qrows->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!tree || !tree->child_off || !tree->child_ids || (!qrow_of_node && !tree->depth) || !token)
        return TSB_ERR_ARG;
    const auto launch = mixed ? tsb::launch_replay_mixed : tsb::launch_replay;
    return cuda_status(launch(rows_of(qrows), static_cast<const float2 *>(qstats), qrow_of_node, cfg->B, cfg->N,
                              cfg->K, tree_of(tree), inv_temperature(cfg->temperature), seed, token,
                              static_cast<uint32_t *>(ws), (cudaStream_t)stream));
}

}  // namespace

extern "C" {

tsb_status tsb_plan_expand(const tsb_cfg *cfg, int32_t width, const tsb_logits *draft, const void *draft_stats,
                           size_t stats_bytes, const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream) {
    if (!draft_stats) return TSB_ERR_ARG;
    return plan_expand_common(cfg, width, draft, draft_stats, nullptr, stats_bytes, out, ws, ws_bytes, stream);
}

tsb_status tsb_plan_rows_expand(const tsb_cfg *cfg, int32_t width, const tsb_logits *draft, void *draft_stats,
                                size_t stats_bytes, const tsb_tree *out, void *ws, size_t ws_bytes,
                                tsb_stream stream) {
    if (!draft_stats) return TSB_ERR_ARG;
    return plan_expand_common(cfg, width, draft, nullptr, draft_stats, stats_bytes, out, ws, ws_bytes, stream);
}

tsb_status tsb_plan_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *draft, const void *draft_stats,
                           size_t stats_bytes, int32_t *pool_ids, const tsb_tree *out, void *ws, size_t ws_bytes,
                           tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st == TSB_OK) st = check_pool(cfg, P);
    if (st != TSB_OK) return st;
    st = check_logits(draft, cfg->B, cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(draft_stats, stats_bytes, cfg->B, draft->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!pool_ids || !out || !out->parent || !out->depth || !out->rank || !out->plan_token || !out->score ||
        !out->child_off || !out->child_ids)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_plan_pooled(rows_of(draft), static_cast<const float2 *>(draft_stats), cfg->L,
                                               cfg->N, cfg->K, P, inv_temperature(cfg->temperature), pool_ids,
                                               tree_of(out), ws, (cudaStream_t)stream));
}

tsb_status tsb_replay_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *qrows, const int32_t *qrow_of_node,
                             const int32_t *pool_ids, const tsb_tree *tree, uint64_t seed, int32_t *token, void *ws,
                             size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st == TSB_OK) st = check_pool(cfg, P);
    if (st != TSB_OK) return st;
    st = check_logits(qrows, cfg->B, qrow_of_node ? 1 : cfg->L, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!pool_ids || !tree || !tree->child_off || !tree->child_ids || !tree->depth || !token) return TSB_ERR_ARG;
    return cuda_status(tsb::launch_replay_pooled(rows_of(qrows), qrow_of_node, cfg->B, cfg->N, cfg->L, P,
                                                 tree_of(tree), pool_ids, inv_temperature(cfg->temperature), seed,
                                                 token, static_cast<uint32_t *>(ws), (cudaStream_t)stream));
}

tsb_status tsb_verify_pooled(const tsb_cfg *cfg, int32_t P, const tsb_logits *target, const tsb_logits *qrows,
                             const int32_t *qrow_of_node, const int32_t *pool_ids, const tsb_tree *tree,
                             const int32_t *token, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                             int32_t *out_len, void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st == TSB_OK) st = check_pool(cfg, P);
    if (st != TSB_OK) return st;
    st = check_logits(target, cfg->B, cfg->N + 1, cfg->V);
    if (st == TSB_OK) st = check_logits(qrows, cfg->B, qrow_of_node ? 1 : cfg->L, cfg->V);
    if (st == TSB_OK && target->dtype != qrows->dtype) st = TSB_ERR_DTYPE;
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!pool_ids || !tree || !tree->child_off || !tree->child_ids || !tree->depth || !token || !out_tokens ||
        !out_nodes || !out_len)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_verify_pooled(rows_of(target), rows_of(qrows), qrow_of_node, cfg->B, cfg->N,
                                                 cfg->L, P, tree_of(tree), pool_ids, token,
                                                 inv_temperature(cfg->temperature), seed, out_tokens, out_nodes,
                                                 out_len, static_cast<uint32_t *>(ws), (cudaStream_t)stream));
}

tsb_status tsb_replay_mixed(const tsb_cfg *cfg, const tsb_logits *qrows, const void *qstats, size_t stats_bytes,
                            const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed, int32_t *token,
                            void *ws, size_t ws_bytes, tsb_stream stream) {
    return replay_common(true, cfg, qrows, qstats, stats_bytes, qrow_of_node, tree, seed, token, ws, ws_bytes,
                         stream);
}

int32_t tsb_version(void) { return 200; }

const char *tsb_status_str(tsb_status s) {
    switch (s) {
        case TSB_OK: return "ok";
        case TSB_ERR_ARG: return "invalid argument";
        case TSB_ERR_SHAPE: return "shape out of range or inconsistent";
        case TSB_ERR_DTYPE: return "unsupported dtype";
        case TSB_ERR_ALIGN: return "row not 16-byte aligned";
        case TSB_ERR_WORKSPACE: return "workspace or stats buffer too small or misaligned";
        case TSB_ERR_CUDA: return "CUDA error";
        case TSB_ERR_DEVICE: return "device status bits set";
    }
    return "unknown status";
}

size_t tsb_stats_bytes(int32_t B, int32_t R, int32_t V) {
    if (B < 1 || R < 1 || V < 1 || V > TSB_MAX_V) return 0;
    return (size_t)B * (size_t)R * (size_t)tsb::num_chunks(V) * sizeof(float2);
}

size_t tsb_workspace_bytes(const tsb_cfg *cfg) {
    if (!cfg || check_cfg(cfg) != TSB_OK) return 0;
    return ws_bytes_for(cfg);
}

tsb_status tsb_workspace_init(void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_ws(ws, ws_bytes, kStatusBytes);
    if (st != TSB_OK) return st;
    return cuda_status(cudaMemsetAsync(ws, 0, sizeof(uint32_t), (cudaStream_t)stream));
}

tsb_status tsb_device_status(void *ws, tsb_stream stream, uint32_t *bits) {
    if (!ws || !bits) return TSB_ERR_ARG;
    uint32_t host = 0;
    cudaError_t e = cudaMemcpyAsync(&host, ws, sizeof host, cudaMemcpyDeviceToHost, (cudaStream_t)stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e == cudaSuccess && host) {
        e = cudaMemsetAsync(ws, 0, sizeof(uint32_t), (cudaStream_t)stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
    }
    *bits = host;
    if (e != cudaSuccess) return TSB_ERR_CUDA;
    return host ? TSB_ERR_DEVICE : TSB_OK;
}

tsb_status tsb_row_stats(const tsb_logits *rows, float temperature, void *stats, size_t stats_bytes, void *ws,
                         size_t ws_bytes, tsb_stream stream) {
    if (!rows) return TSB_ERR_ARG;
    if (!(temperature > 0.0f) || !isfinite(temperature)) return TSB_ERR_ARG;
    if (rows->B < 1 || rows->B > TSB_MAX_B || rows->V < 1 || rows->V > TSB_MAX_V) return TSB_ERR_SHAPE;
    tsb_status st = check_logits(rows, rows->B, 1, rows->V);
    if (st == TSB_OK) st = check_stats(stats, stats_bytes, rows->B, rows->R, rows->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, kStatusBytes);
    if (st != TSB_OK) return st;
    return cuda_status(tsb::launch_row_stats(rows_of(rows), inv_temperature(temperature),
                                             static_cast<float2 *>(stats), static_cast<uint32_t *>(ws),
                                             (cudaStream_t)stream));
}

tsb_status tsb_plan(const tsb_cfg *cfg, const tsb_logits *draft, const void *draft_stats, size_t stats_bytes,
                    const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_logits(draft, cfg->B, cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(draft_stats, stats_bytes, cfg->B, draft->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!out || !out->parent || !out->depth || !out->rank || !out->plan_token || !out->score || !out->child_off ||
        !out->child_ids)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_plan(rows_of(draft), static_cast<const float2 *>(draft_stats), cfg->L, cfg->N,
                                        cfg->K, inv_temperature(cfg->temperature), tree_of(out), ws,
                                        (cudaStream_t)stream));
}

tsb_status tsb_plan_rows(const tsb_cfg *cfg, const tsb_logits *draft, void *draft_stats, size_t stats_bytes,
                         const tsb_tree *out, void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_logits(draft, cfg->B, cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(draft_stats, stats_bytes, cfg->B, draft->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!out || !out->parent || !out->depth || !out->rank || !out->plan_token || !out->score || !out->child_off ||
        !out->child_ids)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_plan_rows(rows_of(draft), static_cast<float2 *>(draft_stats), cfg->L, cfg->N,
                                             cfg->K, inv_temperature(cfg->temperature), tree_of(out), ws,
                                             (cudaStream_t)stream));
}

tsb_status tsb_replay(const tsb_cfg *cfg, const tsb_logits *qrows, const void *qstats, size_t stats_bytes,
                      const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed, int32_t *token, void *ws,
                      size_t ws_bytes, tsb_stream stream) {
    return replay_common(false, cfg, qrows, qstats, stats_bytes, qrow_of_node, tree, seed, token, ws, ws_bytes,
                         stream);
}

tsb_status tsb_verify(const tsb_cfg *cfg, int32_t mode, const tsb_logits *target, const tsb_logits *qrows,
                      const void *qstats, size_t stats_bytes, const int32_t *qrow_of_node, const tsb_tree *tree,
                      const int32_t *token, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                      int32_t *out_len, void *ws, size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    if (mode != TSB_VERIFY_RRS && mode != TSB_VERIFY_BLOCK && mode != TSB_VERIFY_NAIVE &&
        mode != TSB_VERIFY_TRAVERSAL)
        return TSB_ERR_ARG;
    if (mode == TSB_VERIFY_BLOCK && cfg->N > cfg->L) return TSB_ERR_SHAPE;
    st = check_logits(target, cfg->B, cfg->N + 1, cfg->V);
    if (mode == TSB_VERIFY_NAIVE) {  // no draft rows: only the target and the tree
        if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
        if (st != TSB_OK) return st;
        if (!tree || !tree->child_off || !tree->child_ids || !token || !out_tokens || !out_nodes || !out_len)
            return TSB_ERR_ARG;
        return cuda_status(tsb::launch_verify_naive(rows_of(target), cfg->B, cfg->N, cfg->L, tree_of(tree), token,
                                                    inv_temperature(cfg->temperature), seed, out_tokens,
                                                    out_nodes, out_len, static_cast<uint32_t *>(ws),
                                                    (cudaStream_t)stream));
    }
    if (st == TSB_OK) st = check_logits(qrows, cfg->B, qrow_of_node ? 1 : cfg->L, cfg->V);
    if (st == TSB_OK && target->dtype != qrows->dtype) st = TSB_ERR_DTYPE;
    if (st == TSB_OK) st = check_stats(qstats, stats_bytes, cfg->B, qrows->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!tree || !tree->child_off || !tree->child_ids || (!qrow_of_node && !tree->depth) || !token ||
        !out_tokens || !out_nodes || !out_len)
        return TSB_ERR_ARG;
    const float invT = inv_temperature(cfg->temperature);
    cudaError_t e;
    if (mode == TSB_VERIFY_TRAVERSAL)
        e = tsb::launch_verify_traversal(rows_of(target), rows_of(qrows), static_cast<const float2 *>(qstats),
                                         qrow_of_node, cfg->B, cfg->N, cfg->L, tree_of(tree), token, invT, seed,
                                         out_tokens, out_nodes, out_len, static_cast<uint32_t *>(ws),
                                         (cudaStream_t)stream);
    else if (mode == TSB_VERIFY_RRS)
        e = tsb::launch_verify_rrs(rows_of(target), rows_of(qrows), static_cast<const float2 *>(qstats),
                                   qrow_of_node, cfg->B, cfg->N, cfg->L, tree_of(tree), token, invT, seed,
                                   out_tokens, out_nodes, out_len, static_cast<uint32_t *>(ws),
                                   (cudaStream_t)stream);
    else
        e = tsb::launch_verify_block(rows_of(target), rows_of(qrows), static_cast<const float2 *>(qstats),
                                     qrow_of_node, cfg->B, cfg->N, cfg->L, tree_of(tree), token, invT, seed,
                                     out_tokens, out_nodes, out_len, static_cast<uint32_t *>(ws),
                                     (cudaStream_t)stream);
    return cuda_status(e);
}

tsb_status tsb_replay_verify(const tsb_cfg *cfg, const tsb_logits *target, const tsb_logits *qrows, const void *qstats,
                             size_t stats_bytes, const int32_t *qrow_of_node, const tsb_tree *tree, uint64_t seed,
                             int32_t *token, int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, void *ws,
                             size_t ws_bytes, tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_logits(target, cfg->B, cfg->N + 1, cfg->V);
    if (st == TSB_OK) st = check_logits(qrows, cfg->B, qrow_of_node ? 1 : cfg->L, cfg->V);
    if (st == TSB_OK && target->dtype != qrows->dtype) st = TSB_ERR_DTYPE;
    if (st == TSB_OK) st = check_stats(qstats, stats_bytes, cfg->B, qrows->R, cfg->V);
    if (st == TSB_OK) st = check_ws(ws, ws_bytes, ws_bytes_for(cfg));
    if (st != TSB_OK) return st;
    if (!tree || !tree->child_off || !tree->child_ids || (!qrow_of_node && !tree->depth) || !token ||
        !out_tokens || !out_nodes || !out_len)
        return TSB_ERR_ARG;
    return cuda_status(tsb::launch_replay_verify(rows_of(target), rows_of(qrows), static_cast<const float2 *>(qstats),
                                                 qrow_of_node, cfg->B, cfg->N, cfg->L, cfg->K, tree_of(tree), token,
                                                 inv_temperature(cfg->temperature), seed, out_tokens, out_nodes,
                                                 out_len, static_cast<uint32_t *>(ws), (cudaStream_t)stream));
}

}  // extern "C"

// ---------------------------------------------------------------------------------------
// tsb_plan_noalloc: the first pass for callers that may not allocate device memory.
//
// Its scratch (the first pass's per-draft-row log-normaliser and top-K list, plus a status
// word used when the caller gives none) lives in one file-scope device array of
// TSB_NOALLOC_SCRATCH_BYTES. Every device that loads this library holds the array until the
// process exits, and every call on that device shares it.
namespace {

constexpr size_t kNoallocBytes = TSB_NOALLOC_SCRATCH_BYTES;
static_assert(kNoallocBytes % 256 == 0 && kNoallocBytes > kStatusBytes, "scratch size");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocBytes];

// In host code g_noalloc_scratch names a host-side shadow, not device memory: its device
// address on the current device is looked up with cudaGetSymbolAddress. The lookup is made
// on every call rather than cached, so the address stays right after a cudaDeviceReset (which
// unloads the module) or under another context on the same device; once the module is
// loaded on the device the lookup is a table read in the runtime.
tsb_status noalloc_scratch(unsigned char **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return TSB_ERR_CUDA;
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return TSB_ERR_CUDA;
    *out = static_cast<unsigned char *>(p);
    return TSB_OK;
}

// Bytes of the scratch one configuration uses: status word, then per draft row a float2
// log-normaliser, K floats and K int32 (the same per-row record as the workspace's).
size_t noalloc_need(const tsb_cfg *c) {
    const size_t rows = (size_t)c->B * (size_t)c->L;
    return kStatusBytes + rows * sizeof(float2) + rows * (size_t)c->K * (sizeof(float) + sizeof(int32_t));
}

}  // namespace

extern "C" tsb_status tsb_plan_noalloc(const tsb_cfg *cfg, const tsb_logits *draft, const void *draft_stats,
                                       size_t stats_bytes, const tsb_tree *out, uint32_t *dev_status,
                                       tsb_stream stream) {
    tsb_status st = check_cfg(cfg);
    if (st != TSB_OK) return st;
    st = check_logits(draft, cfg->B, cfg->L, cfg->V);
    if (st == TSB_OK) st = check_stats(draft_stats, stats_bytes, cfg->B, draft->R, cfg->V);
    if (st != TSB_OK) return st;
    if (!out || !out->parent || !out->depth || !out->rank || !out->plan_token || !out->score || !out->child_off ||
        !out->child_ids)
        return TSB_ERR_ARG;
    if (dev_status && !aligned(dev_status, sizeof(uint32_t))) return TSB_ERR_ARG;
    if (noalloc_need(cfg) > kNoallocBytes) return TSB_ERR_SHAPE;
    unsigned char *base = nullptr;
    st = noalloc_scratch(&base);
    if (st != TSB_OK) return st;
    uint32_t *status = dev_status;
    if (!status) {
        // bits nobody reads, but the word is OR-ed into: start it at zero on every call
        status = reinterpret_cast<uint32_t *>(base);
        if (cudaMemsetAsync(status, 0, sizeof(uint32_t), (cudaStream_t)stream) != cudaSuccess) return TSB_ERR_CUDA;
    }
    // The top-K launch writes every (lse, x, id) entry the frontier launch reads, so the
    // rest of the scratch needs no clearing.
    const size_t rows = (size_t)cfg->B * (size_t)cfg->L;
    tsb::PlanScratch sc;
    sc.lse = reinterpret_cast<float2 *>(base + kStatusBytes);
    sc.topk_x = reinterpret_cast<float *>(base + kStatusBytes + rows * sizeof(float2));
    sc.topk_id = reinterpret_cast<int32_t *>(base + kStatusBytes + rows * sizeof(float2) +
                                             rows * (size_t)cfg->K * sizeof(float));
    return cuda_status(tsb::launch_plan_scratch(rows_of(draft), static_cast<const float2 *>(draft_stats), cfg->L,
                                                cfg->N, cfg->K, inv_temperature(cfg->temperature), tree_of(out), sc,
                                                status, (cudaStream_t)stream));
}
