// Second pass with mixed sampling (Sec. 3.2 and App. A: the greedy draft sampling of Hu et al.
// 2025, which the paper pairs with its tree verifiers).
//
// For a parent u with m_u children, child slots 0..m_u-2 take the m_u-1 most probable tokens
// of q_u in order, by (x desc, id asc), and slot m_u-1 takes one draw from q_u renormalised over
// the other tokens. The draw is the largest Gumbel key among the remaining tokens, with the keys
// of the top-down construction the WoR sampler uses (chunk keys K_c from the chunk statistics,
// element keys shifted to their chunk's maximum): the keys are jointly i.i.d. Gumbel(x_v), so
// the largest over a fixed token set follows q restricted to that set. A chunk without an
// excluded token has its chunk key as its largest key (held by its largest raw element key),
// so element keys are needed only in the chunks holding an excluded token and in the best
// clean chunk; of each, only its best non-excluded raw key is shifted. With m_u = 1 nothing is
// excluded and the draw is the WoR sampler's single draw, bit for bit.
//
// One CTA of 4 warps per (tree, node), nodes without children return at once:
//   1. every chunk key goes to shared memory (four chunks per Philox block); for m_u > 1 each
//      thread also keeps its largest chunk maxima;
//   2. (m_u > 1) tau = the (m_u-1)-th largest chunk maximum bounds the (m_u-1)-th largest logit
//      from below; the chunks whose maximum reaches tau are re-read (one warp per chunk) and
//      their logits >= tau go through per-lane sorted lists, then warp and CTA merges;
//   3. the best clean chunk by (K_c desc, c asc); one warp per expanded chunk computes its
//      candidate key; the largest candidate is the sampled slot.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;

struct MixedArgs {
    const void *q;
    int64_t bstride, rstride;
    int R, V, C;
    const float2 *stats;
    const int32_t *qrow_of_node, *depth, *child_off, *child_ids;
    int B, N;
    float invT;
    uint64_t seed;
    int32_t *token;
    uint32_t *status;
};

// The top n keys of a warp's lanes' lists into dst[0..n) (lane 0 writes; zeros once the lists
// are empty).
template <int CAP>
__device__ __forceinline__ void warp_top_n(TopList<CAP> &list, int n, uint64_t *dst) {
    for (int j = 0; j < n; ++j) {
        const uint64_t best = warp_pop_max(list);
        if ((threadIdx.x & 31) == 0) dst[j] = best;
    }
}

// Warp 0 only: the top n keys of the warps' lists cand[0..kWarps)[0..n) into out[0..n).
template <int CAP>
__device__ __forceinline__ void merge_warp_lists(const uint64_t (*cand)[CAP], int n, uint64_t *out) {
    TopList<CAP> t;
    t.clear();
    for (int e = threadIdx.x & 31; e < kWarps * n; e += 32) t.insert(cand[e / n][e % n]);
    warp_top_n(t, n, out);
}

template <int KCAP, typename T>
__global__ void __launch_bounds__(kThreads, KCAP <= 8 ? 8 : 2) k_replay_mixed(MixedArgs a) {
    pdl_begin();
    __shared__ uint64_t cand[kWarps][KCAP];
    __shared__ uint64_t sel[KCAP];        // the deterministic tokens' (x, id) keys, in order
    __shared__ uint64_t pick[KCAP + 1];   // candidate key of each expanded chunk
    __shared__ uint64_t s_best[kWarps];
    __shared__ int s_dirty[KCAP];         // chunks holding a deterministic token
    __shared__ int s_ndirty, s_ncand;
    extern __shared__ __align__(16) float ckey[];  // [C] chunk keys, then [C] candidate chunks
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int b = blockIdx.x / NN, u = blockIdx.x - (blockIdx.x / NN) * NN;
    if (u == 0 && threadIdx.x == 0) a.token[(int64_t)b * NN] = -1;
    const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
    const int o = off[u], m = off[u + 1] - o;
    if (m <= 0) return;  // uniform over the CTA
    if (m > KCAP || o < 0 || o + m > a.N || m > a.V) {
        if (threadIdx.x == 0) raise_status(a.status, kDevBadTree);
        return;
    }
    const int r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : a.depth[(int64_t)b * NN + u];
    if (r < 0 || r >= a.R) {
        if (threadIdx.x == 0) raise_status(a.status, kDevBadIndex);
        return;
    }
    const int32_t *kids = a.child_ids + (int64_t)b * a.N + o;
    const float2 *st = a.stats + ((int64_t)b * a.R + r) * a.C;
    const T *row = static_cast<const T *>(a.q) + (int64_t)b * a.bstride + (int64_t)r * a.rstride;
    const uint32_t ub = (uint32_t)b, un = (uint32_t)u;
    const int nd = m - 1;  // deterministic slots (uniform over the CTA)
    int *clist = reinterpret_cast<int *>(ckey + a.C);
    if (threadIdx.x == 0) {
        s_ndirty = 0;
        s_ncand = 0;
    }

    // 1. chunk keys (the WoR sampler's arithmetic) and each thread's largest chunk maxima
    TopList<KCAP> cl;
    cl.clear();
    for (int c4 = threadIdx.x * 4; c4 < a.C; c4 += 4 * kThreads) {
        const Words4 w = draw_block(a.seed, kReplayChunk, ub, un, (uint32_t)(c4 >> 2));
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int c = c4 + i;
            if (c < a.C) {
                const float2 s = st[c];
                ckey[c] = (s.x + logf(s.y)) + gumbel_of(w.w[i]);
                if (nd > 0) cl.insert(pack_key(s.x, (uint32_t)c));
            }
        }
    }
    if (nd > 0) {
        // 2a. tau = the nd-th largest chunk maximum (-inf when there are fewer chunks)
        warp_top_n(cl, nd, cand[warp]);
        __syncthreads();
        if (warp == 0) merge_warp_lists<KCAP>(cand, nd, sel);
        __syncthreads();
        const uint64_t tk = sel[nd - 1];
        const float tau = tk == 0ull ? -INFINITY : key_value(tk);
        // 2b. the chunks whose maximum reaches tau
        for (int c = threadIdx.x; c < a.C; c += kThreads)
            if (st[c].x >= tau) {
                const int pos = atomicAdd(&s_ncand, 1);
                if (in_bounds(pos, a.C, a.status)) clist[pos] = c;
            }
        __syncthreads();
        // 2c. their logits >= tau, one warp per chunk, into per-lane lists
        const int nc = s_ncand;
        TopList<KCAP> el;
        el.clear();
        for (int i = warp; i < nc; i += kWarps) {
            const int v0 = clist[i] * kChunk + lane * 8;
            float z[8];
            Logit<T>::load8(row, v0, a.V, z);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float x = __fmul_rn(z[k], a.invT);
                if (v0 + k < a.V && x >= tau) el.insert(pack_key(x, (uint32_t)(v0 + k)));
            }
        }
        warp_top_n(el, nd, cand[warp]);
        __syncthreads();
        if (warp == 0) {
            merge_warp_lists<KCAP>(cand, nd, sel);
            __syncwarp();
            if (lane < nd) {
                const int child = kids[lane];
                if (child > 0 && child < NN)
                    a.token[(int64_t)b * NN + child] = (int32_t)key_id(sel[lane]);
                else
                    raise_status(a.status, kDevBadTree);
            }
            if (lane == 0) {  // distinct chunks of the deterministic tokens
                int n = 0;
                for (int j = 0; j < nd; ++j) {
                    const int c = (int)(key_id(sel[j]) / kChunk);
                    bool seen = false;
                    for (int e = 0; e < n; ++e) seen |= s_dirty[e] == c;
                    if (!seen) s_dirty[n++] = c;
                }
                s_ndirty = n;
            }
        }
    }
    __syncthreads();

    // 3a. the best clean chunk by (K_c desc, c asc)
    const int ndirty = s_ndirty;
    {
        uint64_t best = 0ull;
        for (int c = threadIdx.x; c < a.C; c += kThreads) {
            bool dirty = false;
            for (int e = 0; e < ndirty; ++e) dirty |= s_dirty[e] == c;
            if (!dirty) {
                const uint64_t k = pack_key(ckey[c], (uint32_t)c);
                best = k > best ? k : best;
            }
        }
        best = warp_max_u64(best);
        if (lane == 0) s_best[warp] = best;
    }
    __syncthreads();
    uint64_t clean = 0ull;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) clean = s_best[w] > clean ? s_best[w] : clean;
    const int nexp = ndirty + (clean != 0ull ? 1 : 0);

    // 3b. one warp per expanded chunk: the dirty chunks, then the best clean chunk
    for (int e = warp; e < nexp; e += kWarps) {
        const bool dirty = e < ndirty;
        const int c = dirty ? s_dirty[e] : (int)key_id(clean);
        const float Tc = ckey[c];
        const int v0 = c * kChunk + lane * 8;
        float x[8];
        Logit<T>::load8(row, v0, a.V, x);
        const Words4 w0 = draw_block(a.seed, kReplayElem, ub, un, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kReplayElem, ub, un, (uint32_t)(v0 >> 2) + 1u);
        uint64_t zk = 0ull, gk = 0ull;  // the chunk's largest raw key; the largest kept one
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            if (v0 + i < a.V) {
                const uint32_t wi = i < 4 ? w0.w[i] : w1.w[i - 4];
                const float g = __fadd_rn(__fmul_rn(x[i], a.invT), gumbel_of(wi));
                const uint64_t k = pack_key(g, (uint32_t)(v0 + i));
                zk = k > zk ? k : zk;
                bool excluded = false;
                if (dirty)
                    for (int j = 0; j < nd; ++j) excluded |= key_id(sel[j]) == (uint32_t)(v0 + i);
                if (!excluded) gk = k > gk ? k : gk;
            }
        }
        zk = warp_max_u64(zk);
        gk = warp_max_u64(gk);
        if (lane == 0) {
            uint64_t p = 0ull;
            if (gk != 0ull) {
                const float k = key_id(gk) == key_id(zk) ? Tc : shifted_gumbel_key(Tc, key_value(zk), key_value(gk));
                p = pack_key(k, key_id(gk));
            }
            pick[e] = p;
        }
    }
    __syncthreads();

    // 3c. the sampled slot: the largest candidate key
    if (threadIdx.x == 0) {
        uint64_t best = 0ull;
        for (int e = 0; e < nexp; ++e) best = pick[e] > best ? pick[e] : best;
        const int child = kids[m - 1];
        if (best != 0ull && child > 0 && child < NN)
            a.token[(int64_t)b * NN + child] = (int32_t)key_id(best);
        else
            raise_status(a.status, kDevBadTree);
    }
}

template <int KCAP, typename T>
cudaError_t launch_mixed_t(const MixedArgs &a, cudaStream_t s) {
    const int64_t blocks = (int64_t)a.B * (a.N + 1);
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const size_t smem = (size_t)a.C * (sizeof(float) + sizeof(int));
    cudaError_t e =
        cudaFuncSetAttribute(k_replay_mixed<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_replay_mixed<KCAP, T>, dim3((unsigned)blocks), dim3(kThreads), smem, s, 0, a);
}

}  // namespace

cudaError_t launch_replay_mixed(const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node, int B, int N,
                                int K, const TreeDesc &tree, float invT, uint64_t seed, int32_t *token,
                                uint32_t *status, cudaStream_t s) {
    MixedArgs a;
    a.q = q.data;
    a.bstride = q.batch_stride;
    a.rstride = q.row_stride;
    a.R = q.R;
    a.V = q.V;
    a.C = num_chunks(q.V);
    a.stats = qstats;
    a.qrow_of_node = qrow_of_node;
    a.depth = tree.depth;
    a.child_off = tree.child_off;
    a.child_ids = tree.child_ids;
    a.B = B;
    a.N = N;
    a.invT = invT;
    a.seed = seed;
    a.token = token;
    a.status = status;
    if (q.dtype == 1)
        return K <= 8 ? launch_mixed_t<8, __nv_bfloat16>(a, s) : launch_mixed_t<32, __nv_bfloat16>(a, s);
    return K <= 8 ? launch_mixed_t<8, float>(a, s) : launch_mixed_t<32, float>(a, s);
}

}  // namespace tsb
