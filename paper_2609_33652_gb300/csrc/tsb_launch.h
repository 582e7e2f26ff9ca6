// Host-side launchers of the libtsb kernels (internal; the public ABI is include/tsb.h).
// Arguments are validated by the ABI layer before any of these is called.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace tsb {

struct RowsDesc {
    const void *data;
    int dtype;  // 0 fp32, 1 bf16
    int B, R, V;
    int64_t batch_stride, row_stride;
};

struct TreeDesc {
    int32_t *parent, *depth, *rank, *plan_token;
    float *score;
    int32_t *child_off, *child_ids;
};

inline int num_chunks(int V) { return (V + 255) / 256; }

// Launch with the programmatic-stream-serialisation attribute (the kernel must begin with
// pdl_begin()), optionally as clusters of cluster_x CTAs.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, int cluster_x,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    int n = 1;
    if (cluster_x > 0) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = (unsigned)cluster_x;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        n = 2;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

// Workspace layout (caller-owned, 256-byte aligned):
//   [0, 256)                       sticky status word
//   B*(N+1) x 32 bytes             per-(tree, node) scalars: block verification's per-position
//                                  values, or the verifier pre-pass's log-normalisers
//   B x 1024 bytes                 per tree, the recursive-rejection pre-pass's partial
//                                  normalisers (up to 8 chain nodes x 8 row parts x 16 bytes)
//   B*L float2, B*L*K floats,      per-draft-row log-normaliser (float-float) and top-K
//   B*L*K int32                    (x, id) of the first pass
constexpr size_t kWsStatusBytes = 256;
constexpr size_t kWsBvRowBytes = 32;
constexpr size_t kWsPrePartBytes = 1024;

inline size_t ws_pre_part_offset(int B, int N) { return kWsStatusBytes + (size_t)B * ((size_t)N + 1) * kWsBvRowBytes; }
inline size_t ws_plan_offset(int B, int N) { return ws_pre_part_offset(B, N) + (size_t)B * kWsPrePartBytes; }

inline size_t workspace_bytes(int B, int N, int L, int K) {
    return ws_plan_offset(B, N) + (size_t)B * L * 2 * sizeof(float) + (size_t)B * L * K * (sizeof(float) + sizeof(int32_t));
}

// Expand-then-prune first pass: layer d holds n_d candidates, n_1 = K and
// n_{d+1} = min(W, n_d) * K; ept_layer_start(d) = n_1 + ... + n_{d-1}, so
// ept_layer_start(L + 1) is the number of candidates generated. The planner keeps them all in
// shared memory, at most kEptMaxCandidates.
constexpr int kEptMaxCandidates = 8192;
__host__ __device__ inline int64_t ept_layer_start(int d, int K, int W) {
    int64_t start = 0, n = K;
    for (int e = 1; e < d; ++e) {
        start += n;
        n = (n < W ? n : W) * (int64_t)K;
        if (start > ((int64_t)1 << 40)) break;
    }
    return start;
}

struct PlanScratch {
    float2 *lse;
    float *topk_x;
    int32_t *topk_id;
};
PlanScratch plan_scratch(void *ws, int B, int N, int L, int K);

cudaError_t launch_row_stats(const RowsDesc &rows, float invT, float2 *stats, uint32_t *status, cudaStream_t s);

cudaError_t launch_plan(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                        const TreeDesc &tree, void *ws, cudaStream_t s);
cudaError_t launch_plan_rows(const RowsDesc &draft, float2 *stats_out, int L, int N, int K, float invT,
                             const TreeDesc &tree, void *ws, cudaStream_t s);
cudaError_t launch_plan_scratch(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                                const TreeDesc &tree, const PlanScratch &sc, uint32_t *status, cudaStream_t s);

cudaError_t launch_plan_expand(const RowsDesc &draft, const float2 *stats, float2 *stats_out, int L, int N, int K,
                               int W, float invT, const TreeDesc &tree, void *ws, cudaStream_t s);

cudaError_t launch_plan_pooled(const RowsDesc &draft, const float2 *stats, int L, int N, int K, int P, float invT,
                               int32_t *pool_ids, const TreeDesc &tree, void *ws, cudaStream_t s);
cudaError_t launch_pool_finish(const RowsDesc &draft, int L, int K, int P, float invT, const int32_t *pool_ids,
                               float2 *lse, float *topk_x, int32_t *topk_id, uint32_t *status, cudaStream_t s);
cudaError_t launch_pool_select(const RowsDesc &draft, const float2 *stats, int L, int P, float invT,
                               int32_t *pool_ids, cudaStream_t s);

cudaError_t launch_replay_pooled(const RowsDesc &q, const int32_t *qrow_of_node, int B, int N, int L, int P,
                                 const TreeDesc &tree, const int32_t *pool_ids, float invT, uint64_t seed,
                                 int32_t *token, uint32_t *status, cudaStream_t s);
cudaError_t launch_verify_pooled(const RowsDesc &target, const RowsDesc &q, const int32_t *qrow_of_node, int B,
                                 int N, int L, int P, const TreeDesc &tree, const int32_t *pool_ids,
                                 const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                 int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s);

cudaError_t launch_replay(const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node, int B, int N,
                          int K, const TreeDesc &tree, float invT, uint64_t seed, int32_t *token, uint32_t *status,
                          cudaStream_t s);

cudaError_t launch_replay_mixed(const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node, int B, int N,
                                int K, const TreeDesc &tree, float invT, uint64_t seed, int32_t *token,
                                uint32_t *status, cudaStream_t s);

// tsb_replay followed by tsb_verify (recursive rejection sampling) in two launches: the replay
// CTAs and the verifier's pre-pass CTAs in one grid (the pre-pass reads only the tree and the
// target rows), then the walk.
cudaError_t launch_replay_verify(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                 const int32_t *qrow_of_node, int B, int N, int L, int K, const TreeDesc &tree,
                                 int32_t *token, float invT, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                                 int32_t *out_len, uint32_t *status, cudaStream_t s);

cudaError_t launch_verify_naive(const RowsDesc &target, int B, int N, int L, const TreeDesc &tree,
                                const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s);

cudaError_t launch_verify_rrs(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                              const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                              const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                              int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s);

cudaError_t launch_verify_traversal(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                    const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                                    const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                    int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s);

cudaError_t launch_verify_block(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                                const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s);

}  // namespace tsb
