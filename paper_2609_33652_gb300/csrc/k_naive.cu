// Verification by target-sample matching ("Naive" in Table 2; Sec. 2.3): at the current node
// u a token y is drawn from the target law p_u; the first child of u that carries y is accepted
// and the walk continues there, otherwise y is the final token. At a leaf y is the bonus
// token. The draw is the two-level Gumbel-max of the bonus token: chunk keys
// A_c + G(U[final chunk, u, c]) with A_c = log sum_{v in c} exp(x_v), the best chunk by
// (key desc, c asc), then x_v + G(U[final, u, v]) inside it by (key desc, v asc).
//
// Every node's draw depends only on its own target row and its own uniforms, so the draws of
// all (tree, node) rows are computed at once, one cluster per row, streaming each row once
// (k_naive_draw); the walk is then a pointer chase over the drawn tokens in shared memory, one
// CTA per tree (k_naive_walk). This reads every target row, where a sequential walk would read
// only the visited ones, in exchange for one fully parallel streaming pass.
#include <cooperative_groups.h>

#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

namespace cg = cooperative_groups;

// A row is split over a cluster of kSplit CTAs of kDrawWarps warps, so even a few hundred rows
// keep every SM streaming.
constexpr int kSplit = 4;
constexpr int kDrawWarps = 4;
constexpr int kDrawThreads = kDrawWarps * 32;
// chunks per warp iteration: eight (bf16) or four (fp32) 16-byte loads in flight per lane
template <typename T>
struct Unit {
    static constexpr int n = sizeof(T) == 2 ? 8 : 4;
};
constexpr int kWalkThreads = 128;

struct NaiveArgs {
    const void *target;
    int64_t bstride, rstride;
    int V, C, B, N, L;
    float invT;
    uint64_t seed;
    const int32_t *child_off, *child_ids, *token;
    int32_t *draw;  // [B][N+1] drawn token per node (workspace)
    int32_t *out_tokens, *out_nodes, *out_len;
    uint32_t *status;
};

// One cluster of kSplit CTAs per (tree, node) row; CTA r takes the r-th quarter of the row's
// chunks. Chunk log-masses with one warp per chunk (lane l holds logits 8l..8l+7), a unit of U
// chunks per warp iteration with all U loads issued first and the U sums reduced together;
// each CTA publishes its best chunk key, CTA 0 reads the others through distributed shared
// memory and one of its warps draws the token inside the best chunk.
template <typename T>
__global__ void __launch_bounds__(kDrawThreads, 8) k_naive_draw(NaiveArgs a) {
    pdl_begin();
    constexpr int U = Unit<T>::n;
    __shared__ uint64_t s_best[kDrawWarps];
    __shared__ uint64_t s_part;  // this CTA's best chunk key
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int rid = blockIdx.x / kSplit;
    const int b = rid / NN, u = rid - (rid / NN) * NN;
    const T *row = static_cast<const T *>(a.target) + (int64_t)b * a.bstride + (int64_t)u * a.rstride;
    const uint32_t ub = (uint32_t)b, un = (uint32_t)u;
    const int per = (a.C + kSplit - 1) / kSplit;
    const int c_lo = rank * per, c_hi = min(a.C, c_lo + per);
    const int units = c_hi > c_lo ? (c_hi - c_lo + U - 1) / U : 0;
    uint64_t best = 0ull;
    bool bad = false;
    for (int un0 = warp; un0 < units; un0 += kDrawWarps) {  // uniform over the warp
        const int cu = c_lo + un0 * U;
        RawGroup<T> raw[U];
#pragma unroll
        for (int k = 0; k < U; ++k)
            if (cu + k < c_hi) raw[k].load(row, (cu + k) * kChunk + lane * 8, a.V);
        float mcs[U], part[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            mcs[k] = -INFINITY;
            part[k] = 0.f;
            if (cu + k >= c_hi) continue;  // uniform over the warp
            float z[8];
            raw[k].unpack(z);  // padding past V is -inf
            float zm = z[0];
#pragma unroll
            for (int i = 1; i < 8; ++i) zm = fmaxf(zm, z[i]);
            mcs[k] = __fmul_rn(warp_max(zm), a.invT);
            const float2 offs = exp_offset(mcs[k]);
#pragma unroll
            for (int i = 0; i < 8; ++i) part[k] += chunk_term(z[i], a.invT, offs.x);
            part[k] = chunk_sum_fix(part[k], offs.y);
        }
        // the U chunk sums at once; the lane holding a chunk's sum keys that chunk
        const float tot = warp_multi_sum<U>(part);
        const int ch = multi_sum_index<U>(lane), c = cu + ch;
        if (lane % (32 / U) == 0 && c < c_hi) {
            float mc = mcs[0];
#pragma unroll
            for (int k = 1; k < U; ++k) mc = ch == k ? mcs[k] : mc;
            bad |= !(tot == tot) || isinf(mc);
            const uint32_t w = draw_word(a.seed, kFinalChunk, ub, un, (uint32_t)c);
            const uint64_t k = pack_key(__fadd_rn(__fadd_rn(mc, logf(tot)), gumbel_of(w)), (uint32_t)c);
            best = k > best ? k : best;
        }
    }
    if (__any_sync(kFull, bad) && lane == 0) raise_status(a.status, kDevNonFinite);
    best = warp_max_u64(best);
    if (lane == 0) s_best[warp] = best;
    __syncthreads();
    if (warp == 0) {
        const uint64_t v = warp_max_u64(lane < kDrawWarps ? s_best[lane] : 0ull);
        if (lane == 0) s_part = v;
    }
    cluster.sync();  // every CTA's best chunk key is published
    uint64_t cb = 0ull;
    if (rank == 0 && warp == 0) cb = warp_max_u64(lane < kSplit ? *cluster.map_shared_rank(&s_part, lane) : 0ull);
    cluster.sync();  // CTA 0 has read the others; they may leave
    if (rank != 0 || warp != 0) return;
    if (cb == 0ull) {  // non-finite row (status already raised)
        if (lane == 0) a.draw[(int64_t)b * NN + u] = -1;
        return;
    }
    const int c = (int)key_id(cb);
    const int v0 = c * kChunk + lane * 8;
    float x[8];
    Logit<T>::load8(row, v0, a.V, x);
    const Words4 w0 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2));
    const Words4 w1 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2) + 1u);
    uint64_t tk = 0ull;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        if (v0 + i < a.V) {
            const uint32_t wi = i < 4 ? w0.w[i] : w1.w[i - 4];
            const uint64_t k = pack_key(__fadd_rn(__fmul_rn(x[i], a.invT), gumbel_of(wi)), (uint32_t)(v0 + i));
            tk = k > tk ? k : tk;
        }
    }
    tk = warp_max_u64(tk);
    if (lane == 0) a.draw[(int64_t)b * NN + u] = tk == 0ull ? -1 : (int32_t)key_id(tk);
}

// One CTA per tree: the tree's drawn tokens, child lists and tokens are copied to shared
// memory with coalesced loads, then thread 0 follows the drawn tokens from the root.
__global__ void __launch_bounds__(kWalkThreads) k_naive_walk(NaiveArgs a) {
    pdl_begin();
    extern __shared__ int32_t wsm[];  // draws [NN], child_off [NN+1], child_ids [N], tokens [NN]
    const int b = blockIdx.x;
    const int NN = a.N + 1;
    int32_t *dr = wsm, *off = dr + NN, *ids = off + NN + 1, *tok = ids + a.N;
    for (int i = threadIdx.x; i < NN; i += kWalkThreads) {
        dr[i] = a.draw[(int64_t)b * NN + i];
        tok[i] = a.token[(int64_t)b * NN + i];
    }
    for (int i = threadIdx.x; i <= NN; i += kWalkThreads) off[i] = a.child_off[(int64_t)b * (NN + 1) + i];
    for (int i = threadIdx.x; i < a.N; i += kWalkThreads) ids[i] = a.child_ids[(int64_t)b * a.N + i];
    __syncthreads();
    if (threadIdx.x != 0) return;
    int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1), *onode = a.out_nodes + (int64_t)b * a.L;
    int u = 0, nacc = 0, y = -1;
    uint32_t bits = 0;
    for (;;) {
        y = dr[u];
        if (y < 0) {
            bits |= kDevNonFinite;
            break;
        }
        const int o = off[u], m = off[u + 1] - o;
        if (o < 0 || m < 0 || o + m > a.N) {
            bits |= kDevBadTree;
            break;
        }
        int next = -1;
        for (int i = 0; i < m; ++i) {
            const int c = ids[o + i];
            if (c < 1 || c > a.N) {
                bits |= kDevBadIndex;
                break;
            }
            if (tok[c] == y) {
                next = c;
                break;
            }
        }
        if (next < 0 || nacc >= a.L) break;
        otok[nacc] = y;
        onode[nacc] = next;
        ++nacc;
        u = next;
    }
    if (bits) raise_status(a.status, bits);
    otok[nacc] = y;
    for (int k = nacc + 1; k <= a.L; ++k) otok[k] = -1;
    for (int k = nacc; k < a.L; ++k) onode[k] = -1;
    a.out_len[b] = nacc + 1;
}

template <typename T>
cudaError_t launch_naive_t(const NaiveArgs &a, cudaStream_t s) {
    const int64_t blocks = (int64_t)a.B * (a.N + 1) * kSplit;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    cudaError_t e = launch_pdl(k_naive_draw<T>, dim3((unsigned)blocks), dim3(kDrawThreads), 0, s, kSplit, a);
    if (e != cudaSuccess) return e;
    const size_t smem = (size_t)(3 * (a.N + 1) + 1 + a.N) * sizeof(int32_t);
    return launch_pdl(k_naive_walk, dim3((unsigned)a.B), dim3(kWalkThreads), smem, s, 0, a);
}

}  // namespace

cudaError_t launch_verify_naive(const RowsDesc &target, int B, int N, int L, const TreeDesc &tree,
                                const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                int32_t *out_nodes, int32_t *out_len, void *ws, cudaStream_t s) {
    NaiveArgs a;
    a.target = target.data;
    a.bstride = target.batch_stride;
    a.rstride = target.row_stride;
    a.V = target.V;
    a.C = num_chunks(target.V);
    a.B = B;
    a.N = N;
    a.L = L;
    a.invT = invT;
    a.seed = seed;
    a.child_off = tree.child_off;
    a.child_ids = tree.child_ids;
    a.token = token;
    // the per-(tree, node) region of the workspace holds the drawn tokens
    a.draw = reinterpret_cast<int32_t *>(static_cast<unsigned char *>(ws) + kWsStatusBytes);
    a.out_tokens = out_tokens;
    a.out_nodes = out_nodes;
    a.out_len = out_len;
    a.status = static_cast<uint32_t *>(ws);
    return target.dtype == 1 ? launch_naive_t<__nv_bfloat16>(a, s) : launch_naive_t<float>(a, s);
}

}  // namespace tsb
