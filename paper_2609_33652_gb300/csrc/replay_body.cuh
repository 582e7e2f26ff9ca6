// The second pass's per-parent draws as a device function of one CTA, shared by the replay
// kernel and by the launch that runs replay beside the verifier's pre-pass (the algorithm is
// described in k_replay.cu).
#pragma once
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {


constexpr int kRpWarps = 4;
constexpr int kRpThreads = kRpWarps * 32;
// 4 warps and at most 64 registers: eight CTAs per SM, so a batch's B*(N+1) CTAs (1,040 at
// B=16, N=64) are resident in one wave (leaf nodes' CTAs exit at once).
constexpr int kRpMinBlocks = 8;

struct ReplayArgs {
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

// Merge per-warp lists: each warp writes its top n keys to cand[warp][0..n).
template <int CAP>
__device__ __forceinline__ void warp_top_to(TopList<CAP> &list, int n, uint64_t *dst) {
    const int lane = threadIdx.x & 31;
    for (int j = 0; j < n; ++j) {
        const uint64_t best = warp_pop_max(list);
        if (lane == 0) dst[j] = best;
    }
}

// Warp 0: the top n keys of cand[0..kRpWarps)[0..n) into out[0..n).
template <int CAP>
__device__ __forceinline__ void merge_warps(const uint64_t (*cand)[CAP], int n, uint64_t *out) {
    const int lane = threadIdx.x & 31;
    TopList<CAP> t;
    t.clear();
    for (int e = lane; e < kRpWarps * n; e += 32) t.insert(cand[e / n][e % n]);
    warp_top_to(t, n, out);
}

// Shared-memory key buffer: every chunk key (C), then the chunk keys that reach the lower bound
// (at most C) or up to max(C, kElemBuf) element keys.
constexpr int kElemBuf = 512;
__host__ __device__ inline int key_buf_len(int C) { return C + (C > kElemBuf ? C : kElemBuf); }

// The draws of CTA `blk`: parent u = blk mod (N+1) of tree b = blk / (N+1). Every thread of a
// kRpThreads-thread CTA calls it (after the grid dependency wait); it may return early.
template <int KCAP, typename T>
__device__ __forceinline__ void replay_node(const ReplayArgs &a, int blk) {
    __shared__ uint64_t cand[kRpWarps][KCAP];
    __shared__ uint64_t sel[KCAP];
    __shared__ uint64_t s_lb;
    __shared__ int s_n, s_n2;
    extern __shared__ uint64_t kbuf[];  // [key_buf_len(C)]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int b = blk / NN, u = blk - (blk / NN) * NN;
    if (u == 0 && threadIdx.x == 0) a.token[(int64_t)b * NN] = -1;
    const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
    // the child count and the q row index in one round of loads (a leaf reads its row index too)
    const int o = off[u], o1 = off[u + 1];
    const int r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : a.depth[(int64_t)b * NN + u];
    const int m = o1 - o;
    if (m <= 0) return;  // uniform over the CTA
    if (m > KCAP || o < 0 || o + m > a.N) {
        if (threadIdx.x == 0) raise_status(a.status, kDevBadTree);
        return;
    }
    if (r < 0 || r >= a.R) {
        if (threadIdx.x == 0) raise_status(a.status, kDevBadIndex);
        return;
    }
    const int32_t *kids = a.child_ids + (int64_t)b * a.N + o;
    const float2 *st = a.stats + ((int64_t)b * a.R + r) * a.C;
    const T *row = static_cast<const T *>(a.q) + (int64_t)b * a.bstride + (int64_t)r * a.rstride;
    const uint32_t ub = (uint32_t)b, un = (uint32_t)u;
    const int msel = min(m, a.C);
    // One child: the draw is the Gumbel-max token, i.e. the top chunk by K_c and inside it the
    // token with the largest raw key g_v (its shifted key is K_c itself and every other key of
    // the chunk lies below K_c), so running maxima replace the lists and no key is shifted.
    // The same loops serve both cases (one copy of the key arithmetic).
    const bool single = m == 1;  // uniform over the CTA

    // 1. chunk keys: thread t takes chunks 4t..4t+3 (+1024k), one Philox block each; every key
    //    goes to ckeys[c], each thread keeps its RR largest
    constexpr int RR = KCAP / kRpWarps;  // >= rr = ceil(msel / kRpWarps): each warp's share below
    uint64_t *ckeys = kbuf, *ebuf = kbuf + a.C;
    const int ecap = key_buf_len(a.C) - a.C;
    {
        TopList<RR> cl;
        cl.clear();
        uint64_t best = 0ull;
        for (int c4 = threadIdx.x * 4; c4 < a.C; c4 += 4 * kRpThreads) {
            const Words4 w = draw_block(a.seed, kReplayChunk, ub, un, (uint32_t)(c4 >> 2));
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int c = c4 + i;
                if (c < a.C) {
                    const float2 s = st[c];
                    const float Kc = (s.x + logf(s.y)) + gumbel_of(w.w[i]);
                    const uint64_t k = pack_key(Kc, (uint32_t)c);
                    if (single) {
                        best = k > best ? k : best;
                    } else {
                        ckeys[c] = k;
                        cl.insert(k);
                    }
                }
            }
        }
        // the top msel chunk keys by rank among those that reach a lower bound: the msel-th
        // largest of the warps' rr largest keys (every key when the warps hold fewer)
        const int rr = (msel + kRpWarps - 1) / kRpWarps;  // kRpWarps * rr <= 32
        if (single) {
            best = warp_max_u64(best);
            if (lane == 0) cand[warp][0] = best;
        } else {
            for (int j = 0; j < rr; ++j) {
                const uint64_t k = warp_pop_max(cl);
                if (lane == 0) cand[warp][j] = k;
            }
        }
        __syncthreads();
        if (warp == 0) {
            if (single) {
                const uint64_t v = warp_max_u64(lane < kRpWarps ? cand[lane][0] : 0ull);
                if (lane == 0) sel[0] = v;
            } else {
                __syncwarp();  // converged before the shuffles (the warp reductions' note)
                const uint64_t v = lane < kRpWarps * rr ? cand[lane / rr][lane - (lane / rr) * rr] : 0ull;
                int rk = 0, nz = 0;
                for (int j = 0; j < kRpWarps * rr; ++j) {
                    const uint64_t w = __shfl_sync(kFull, v, j);
                    rk += w > v ? 1 : 0;
                    nz += w != 0ull ? 1 : 0;
                }
                if (nz < msel) {
                    if (lane == 0) s_lb = 0ull;  // every key
                } else if (v != 0ull && rk == msel - 1) {
                    s_lb = v;
                }
                if (lane == 0) {
                    s_n = 0;
                    s_n2 = 0;
                }
            }
        }
        __syncthreads();
        if (!single) {  // the chunk keys that reach the bound, then the top msel by rank
            const uint64_t lb = s_lb;
            for (int c = threadIdx.x; c < a.C; c += kRpThreads)
                if (ckeys[c] >= lb) {
                    const int pos = atomicAdd(&s_n, 1);
                    if (in_bounds(pos, ecap, a.status)) ebuf[pos] = ckeys[c];
                }
            __syncthreads();
            const int n = s_n;
            for (int i = threadIdx.x; i < n; i += kRpThreads) {
                const uint64_t v = ebuf[i];
                const int rk = rank_among(ebuf, n, v);
                if (rk < msel) sel[rk] = v;
            }
        }
    }
    __syncthreads();

    // 2. element keys of each kept chunk (one warp per chunk), shifted to the chunk key
    {
        // K*, the smallest kept chunk key, bounds the drawn keys from below when m chunks are
        // kept (m <= C)
        const float kstar = msel == m ? key_value(sel[msel - 1]) : -INFINITY;
        TopList<KCAP> el;
        el.clear();
        for (int s = warp; s < msel; s += kRpWarps) {
            const uint64_t kk = sel[s];
            const int c = (int)key_id(kk);
            const float Tc = key_value(kk);
            const int v0 = c * kChunk + lane * 8;
            float x[8];
            Logit<T>::load8(row, v0, a.V, x);
            const Words4 w0 = draw_block(a.seed, kReplayElem, ub, un, (uint32_t)(v0 >> 2));
            const Words4 w1 = draw_block(a.seed, kReplayElem, ub, un, (uint32_t)(v0 >> 2) + 1u);
            float g[8];
            uint64_t zk = 0;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                g[i] = -INFINITY;
                if (v0 + i < a.V) {
                    const uint32_t wi = i < 4 ? w0.w[i] : w1.w[i - 4];
                    g[i] = __fadd_rn(__fmul_rn(x[i], a.invT), gumbel_of(wi));
                    const uint64_t k = pack_key(g[i], (uint32_t)(v0 + i));
                    zk = k > zk ? k : zk;
                }
            }
            zk = warp_max_u64(zk);
            if (single) {  // warp 0 only (msel = 1)
                const int child = kids[0];
                if (lane == 0) {
                    if (child > 0 && child < NN)
                        a.token[(int64_t)b * NN + child] = (int32_t)key_id(zk);
                    else
                        raise_status(a.status, kDevBadTree);
                }
                continue;
            }
            const float Z = key_value(zk);
            const uint32_t jmax = key_id(zk);
            // The m kept chunks' maxima hold keys K_c >= K* (the m-th chunk key), so a key below
            // K* is never drawn. The shifted key grows with g, and k_v >= K* exactly when
            //   g_v >= g* = Z - softplus((Z - K*) + log(-expm1(K* - T_c))),
            // so only elements with g_v >= g* - margin (rounding of g* and of the keys) get a
            // shifted key and a list entry.
            float gmin = -INFINITY;
            if (kstar != -INFINITY) {
                const float w = __fadd_rn(__fsub_rn(Z, kstar), logf(-expm1f(__fsub_rn(kstar, Tc))));
                const float sp = w == -INFINITY ? 0.f : fmaxf(w, 0.f) + log1pf(expf(-fabsf(w)));
                gmin = __fsub_rn(__fsub_rn(Z, sp), 1e-3f * (1.f + fabsf(Z)));
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (v0 + i >= a.V || !(g[i] >= gmin)) continue;
                const float k = ((uint32_t)(v0 + i) == jmax) ? Tc : shifted_gumbel_key(Tc, Z, g[i]);
                const uint64_t key = pack_key(k, (uint32_t)(v0 + i));
                el.insert(key);
                const int idx = atomicAdd(&s_n2, 1);
                if (idx < ecap) ebuf[idx] = key;
            }
        }
        if (single) return;  // uniform over the CTA
        __syncthreads();     // the chunk lists in cand[] are no longer needed
        const int n2 = s_n2;
        if (n2 <= ecap) {  // 3. the top-m keys by rank are the ordered draws
            int32_t *tok = a.token + (int64_t)b * NN;
            for (int i = threadIdx.x; i < n2; i += kRpThreads) {
                const uint64_t v = ebuf[i];
                const int rk = rank_among(ebuf, n2, v);
                if (rk < m) {
                    const int child = kids[rk];
                    if (child > 0 && child < NN)
                        tok[child] = (int32_t)key_id(v);
                    else
                        raise_status(a.status, kDevBadTree);
                }
            }
            return;
        }
        warp_top_to(el, m, cand[warp]);  // more element keys than the buffer holds
    }
    __syncthreads();

    // 3. the top-m keys are the ordered draws; draw j fills child slot j
    if (warp == 0) {
        merge_warps<KCAP>(cand, m, sel);
        __syncwarp();
        int32_t *tok = a.token + (int64_t)b * NN;
        if (lane < m) {
            const int child = kids[lane];
            if (child > 0 && child < NN)
                tok[child] = (int32_t)key_id(sel[lane]);
            else
                raise_status(a.status, kDevBadTree);
        }
    }
}

inline ReplayArgs replay_args(const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node, int B, int N,
                              const TreeDesc &tree, float invT, uint64_t seed, int32_t *token, uint32_t *status) {
    ReplayArgs a;
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
    return a;
}

}  // namespace
}  // namespace tsb
