// First pass (Sec. 3.1; max-heap expansion as in DDTree, Sec. 2.2 / App. B.3), two kernels.
//
// k_row_topk, one 4-warp CTA per draft row (every row of the batch in parallel): the row's
//   chunk statistics are staged in shared memory (one round of loads), merged into the
//   log-normaliser LSE_d, and give tau = the K-th largest chunk maximum, a lower bound on the
//   K-th largest logit (K distinct chunk maxima reach it). Only chunks whose maximum reaches
//   tau are re-read, spread over the warps; their logits >= tau go through per-lane sorted
//   lists, and warp then CTA merges yield the top-K by (x desc, id asc). Results go to the
//   workspace.
// k_plan_select, one CTA per tree: the best-first expansion's N nodes. A candidate at depth d
//   holds the sum Sx of its path's logits (exact, in 64-bit fixed point) and the key
//   Sx - CL[d], CL[d] = LSE_1 + ... + LSE_d (its draft path log-probability). Pop order:
//   (key desc, depth asc, parent asc, rank asc), compared as integers. Popping (p, r) at depth d
//   pushes the next sibling (p, r+1) and, below the depth cap, the first child (i, 0). Keys never
//   increase along these links, so the N pops are the N first paths of that order: the kernel
//   bounds the N-th key, enumerates the paths that reach the bound and numbers them by counting
//   (the serial pops remain as the fallback). Siblings are popped in rank order, so the children
//   of u occupy child_ids[child_off[u] + rank] directly.
//
// Both are latency-bound: the draft rows were streamed once by the statistics kernel and only
// the few candidate chunks per row are read again.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kTopkThreads = 128;
constexpr int kRowPlanThreads = 512;
constexpr int kHeapThreads = 256;

struct TopkArgs {
    const void *draft;
    int64_t bstride, rstride;
    int B, R, V, C, L, K;
    const float2 *stats;
    float2 *stats_out;  // k_row_stats_topk: the statistics it writes ([B][R][C])
    uint32_t *status;
    float invT;
    float2 *lse;       // [B*L] row log-normalisers as float-float (hi, lo)
    float *topk_x;     // [B*L*K]
    int32_t *topk_id;  // [B*L*K]
};

// Top n keys of a warp's lanes' lists into dst[0..n) (lane 0 writes; zeros once the lists
// are empty, without further pops).
template <int CAP>
__device__ __forceinline__ void warp_top_to(TopList<CAP> &list, int n, uint64_t *dst) {
    int j = 0;
    for (; j < n; ++j) {
        const uint64_t best = warp_pop_max(list);
        if ((threadIdx.x & 31) == 0) dst[j] = best;
        if (best == 0ull) break;  // uniform over the warp
    }
    if ((threadIdx.x & 31) == 0)
        for (++j; j < n; ++j) dst[j] = 0ull;
}

// The top-K pass of one draft row from its chunk statistics st[0..C) in shared memory (all NT
// threads of the CTA call it, after a barrier that follows the last write of st; cand has room
// for C keys): the float-float log-normaliser; tau = the K-th largest chunk maximum (a lower
// bound on the K-th largest logit, since K distinct chunk maxima reach it), found by rank
// among the chunk keys that reach a cheap lower bound (the K-th largest of the warps' top
// keys); the logits >= tau of the chunks whose maximum reaches tau (a chunk goes to the warp
// that scans it, four chunks' loads per batch), ranked in shared memory (per-warp lists and
// merges when more than C logits reach tau). Writes lse[row], topk_x / topk_id [row][K].
template <int KCAP, int NT, typename T>
__device__ void topk_from_stats(const TopkArgs &a, int row, const float2 *st, uint64_t *cand) {
    constexpr int NW = NT / 32;
    static_assert(NW >= 2, "warps 0 and 1 work in parallel");
    constexpr int kLseThreads = 128, kLseWarps = kLseThreads / 32;
    static_assert(NT >= kLseThreads, "the partition needs kLseThreads threads");
    constexpr int kLseWarp0 = NW - kLseWarps;  // the log-normaliser runs on the last four warps
    __shared__ uint64_t wl[NW][KCAP];
    __shared__ float wm[4], wsh[4], wsl[4];
    __shared__ float s_tau;
    __shared__ uint64_t s_lb;
    __shared__ int s_n, s_n2;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const int C = a.C, K = a.K;
    const int r = (K + NW - 1) / NW;  // each warp's share of the lower bound (NW * r <= 32)
    // 1. per-thread list of chunk keys; log-normaliser partials over a fixed partition of
    //    kLseThreads threads (the same for every caller, so every caller sums in one order)
    TopList<KCAP> cl;
    cl.clear();
    for (int c = threadIdx.x; c < C; c += NT) cl.insert(pack_key(st[c].x, (uint32_t)c));
    if (warp >= kLseWarp0) {
        const int t = threadIdx.x - kLseWarp0 * 32;
        float m = -INFINITY;
        for (int c = t; c < C; c += kLseThreads) m = fmaxf(m, st[c].x);
        KahanF acc;
        if (m != -INFINITY)
            for (int c = t; c < C; c += kLseThreads) acc.add(__fmul_rn(st[c].y, expf(__fsub_rn(st[c].x, m))));
        const MaxSum ms = warp_maxsum(MaxSum{m, acc.ff()});
        if (lane == 0) {
            wm[warp - kLseWarp0] = ms.m;
            wsh[warp - kLseWarp0] = ms.s.hi;
            wsl[warp - kLseWarp0] = ms.s.lo;
        }
    }
    // 2. each warp's r largest chunk keys
    for (int j = 0; j < r; ++j) {
        const uint64_t best = warp_pop_max(cl);
        if (lane == 0) wl[warp][j] = best;
    }
    __syncthreads();
    if (warp == 0) {
        // 3. lower bound of tau (= the K-th largest chunk key): the K-th largest of the warps'
        //    keys (K distinct chunk keys reach it), or 0 when they hold fewer than K keys
        __syncwarp();  // converged before the shuffles (the warp reductions' note)
        const uint64_t v = lane < NW * r ? wl[lane / r][lane - (lane / r) * r] : 0ull;
        int rk = 0, nz = 0;
        for (int j = 0; j < 32; ++j) {
            const uint64_t w = __shfl_sync(kFull, v, j);
            rk += w > v ? 1 : 0;
            nz += w != 0ull ? 1 : 0;
        }
        if (nz < K) {
            if (lane == 0) s_lb = 0ull;
        } else if (v != 0ull && rk == K - 1) {
            s_lb = v;
        }
        if (lane == 0) {
            s_tau = -INFINITY;  // fewer than K chunks
            s_n = 0;
            s_n2 = 0;
        }
    } else if (warp == 1) {  // in parallel with warp 0
        MaxSum v = lane < kLseWarps ? MaxSum{wm[lane], FF{wsh[lane], wsl[lane]}} : MaxSum{-INFINITY, FF{0.f, 0.f}};
        v = warp_maxsum(v);
        if (lane == 0) {
            const FF l = maxsum_lse(v);
            a.lse[row] = make_float2(l.hi, l.lo);
        }
    }
    __syncthreads();
    // 4. the chunk keys at or above the bound, then tau by rank among them
    const uint64_t lb = s_lb;
    for (int c = threadIdx.x; c < C; c += NT) {
        const uint64_t k = pack_key(st[c].x, (uint32_t)c);
        if (k >= lb) {
            const int pos = atomicAdd(&s_n, 1);
            if (in_bounds(pos, C, a.status)) cand[pos] = k;
        }
    }
    __syncthreads();
    if (C >= K) {
        const int n = s_n;
        for (int i = threadIdx.x; i < n; i += NT) {
            const uint64_t v = cand[i];
            if (rank_among(cand, n, v) == K - 1) s_tau = key_value(v);
        }
    }
    __syncthreads();
    const float tau = s_tau;
    // 5. the logits >= tau of the chunks whose maximum reaches tau: into cand (up to C of them)
    //    and into per-lane lists for the case of more
    const T *rowp = static_cast<const T *>(a.draft) + (int64_t)b * a.bstride + (int64_t)d * a.rstride;
    TopList<KCAP> el;
    el.clear();
    for (int cb = warp * 32; cb < C; cb += NT) {
        const int c = cb + lane;
        __syncwarp();
        unsigned mask = __ballot_sync(kFull, c < C && st[c].x >= tau);
        while (mask) {
            int cs[4];
            int nb = 0;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                cs[k] = -1;
                if (mask) {
                    cs[k] = cb + __ffs(mask) - 1;
                    mask &= mask - 1;
                    ++nb;
                }
            }
            float x[4][8];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (k < nb) Logit<T>::load8(rowp, cs[k] * kChunk + lane * 8, a.V, x[k]);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                if (k >= nb) break;
                const int v0 = cs[k] * kChunk + lane * 8;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (v0 + i >= a.V) continue;
                    const float xi = __fmul_rn(x[k][i], a.invT);
                    if (xi >= tau) {
                        const uint64_t key = pack_key(xi, (uint32_t)(v0 + i));
                        el.insert(key);
                        const int idx = atomicAdd(&s_n2, 1);
                        if (idx < C) cand[idx] = key;
                    }
                }
            }
        }
    }
    __syncthreads();
    const int n2 = s_n2;
    if (n2 <= C) {  // 6. the top K by rank (at least K logits reach tau)
        for (int i = threadIdx.x; i < n2; i += NT) {
            const uint64_t v = cand[i];
            const int rk = rank_among(cand, n2, v);
            if (rk < K) {
                a.topk_id[(int64_t)row * K + rk] = (int32_t)key_id(v);
                if (a.topk_x) a.topk_x[(int64_t)row * K + rk] = key_value(v);
            }
        }
        return;
    }
    // 6'. more than C logits reach tau (ties, flat rows): per warp top-K, then the CTA's
    warp_top_to(el, K, wl[warp]);  // wl was last read before the barriers above
    __syncthreads();
    if (warp == 0) {
        TopList<KCAP> t;
        t.clear();
        for (int e = lane; e < NW * K; e += 32) t.insert(wl[e / K][e % K]);
        for (int j = 0; j < K; ++j) {
            const uint64_t best = warp_pop_max(t);
            if (lane == 0) {
                a.topk_id[(int64_t)row * K + j] = (int32_t)key_id(best);
                if (a.topk_x) a.topk_x[(int64_t)row * K + j] = key_value(best);
            }
        }
    }
}

// One 4-warp CTA per draft row: stage the row's chunk statistics (one round of loads), then
// the top-K pass.
template <int KCAP, typename T>
__global__ void __launch_bounds__(kTopkThreads) k_row_topk(TopkArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) float2 st[];  // [C] the row's chunk statistics
    const int row = blockIdx.x;
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const int C = a.C;
    const float2 *gst = a.stats + ((int64_t)b * a.R + d) * C;
    for (int c0 = threadIdx.x; c0 < C; c0 += kTopkThreads * 8) {  // eight loads in flight per thread
        float2 v[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int c = c0 + kTopkThreads * e;
            v[e] = c < C ? __ldg(&gst[c]) : make_float2(-INFINITY, 0.f);
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int c = c0 + kTopkThreads * e;
            if (c < C) st[c] = v[e];
        }
    }
    __syncthreads();
    topk_from_stats<KCAP, kTopkThreads, T>(a, row, st, reinterpret_cast<uint64_t *>(st + C));
}

// One 16-warp CTA per draft row, streaming the row once: the chunk statistics exactly as
// k_row_stats computes them (same per-chunk code, so the same bits), written to the caller's
// statistics buffer and kept in shared memory, then the top-K pass, whose candidate chunks
// are then still in L2. Two CTAs per SM (K <= 8), so up to 2 rows per SM run in one wave.
template <int KCAP, typename T>
__global__ void __launch_bounds__(kRowPlanThreads, KCAP <= 8 ? 2 : 1) k_row_stats_topk(TopkArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) float2 st[];  // [C]
    constexpr int NW = kRowPlanThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, g = lane & 7, q = lane >> 3;
    const int row = blockIdx.x;
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const int C = a.C;
    const T *rp = static_cast<const T *>(a.draft) + (int64_t)b * a.bstride + (int64_t)d * a.rstride;
    float2 *gst = a.stats_out + ((int64_t)b * a.R + d) * C;
    const int units = (C + 3) / 4;  // four chunks (eight lanes each) per warp unit
    constexpr int kU = sizeof(T) == 2 ? 2 : 1;  // units in flight per warp (register budget)
    bool bad = false;
    for (int u0 = warp; u0 < units; u0 += kU * NW) {  // uniform over the warp
        RawGroup<T> raw[kU][4];
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * NW) * 4 + q;
            if (u0 + e * NW < units && c < C)
#pragma unroll
                for (int k = 0; k < 4; ++k) raw[e][k].load(rp, c * kChunk + k * 64 + g * 8, a.V);
        }
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * NW) * 4 + q;
            const bool live = u0 + e * NW < units && c < C;
            float mc, sc;
            chunk_stats8<T>(raw[e], live, a.invT, &mc, &sc);
            if (live && g == 0) {
                const float2 v = make_float2(mc, sc);
                gst[c] = v;
                st[c] = v;
                bad |= !(sc == sc) || isinf(mc);
            }
        }
    }
    if (bad) raise_status(a.status, kDevNonFinite);
    __syncthreads();
    topk_from_stats<KCAP, kRowPlanThreads, T>(a, row, st, reinterpret_cast<uint64_t *>(st + C));
}

struct HeapArgs {
    int L, N, K;
    const float2 *lse;
    const float *topk_x;
    const int32_t *topk_id;
    TreeDesc tree;
    uint32_t *status;
};

// Path sums are kept in 64-bit fixed point with 2^-30 resolution: a logit x converts exactly
// when |x| >= 2^-7 (its fp32 ulp is then a multiple of 2^-30), and sums stay exact up to
// |Sx| < 2^33, so equal real path sums give equal integers and the expansion needs only
// integer additions. The key of a candidate at depth d is Sx - CL[d], CL[d] rounded to the
// same grid once per depth.
// A frontier candidate is a 96-bit integer, larger = pops first:
//   okey = key with its sign bit flipped (order-preserving as unsigned);
//   w3   = (255 - depth) << 24 | (65535 - parent) << 8 | (255 - rank)
// so the order is (key desc, depth asc, parent asc, rank asc); an empty slot is (0, 0).
constexpr float kFixScale = 1073741824.0f;  // 2^30
constexpr float kFixInv = 9.313225746154785e-10f;  // 2^-30

__device__ __forceinline__ unsigned w3_of(int depth, int parent, int rank) {
    return ((unsigned)(255 - depth) << 24) | ((unsigned)(65535 - parent) << 8) | (unsigned)(255 - rank);
}
__device__ __forceinline__ bool key_better(unsigned long long ka, unsigned wa, unsigned long long kb, unsigned wb) {
    return ka > kb || (ka == kb && wa > wb);
}
__device__ __forceinline__ unsigned long long okey_of(long long key) {
    return (unsigned long long)key ^ 0x8000000000000000ull;
}
__device__ __forceinline__ long long key_of_okey(unsigned long long o) { return (long long)(o ^ 0x8000000000000000ull); }
__device__ __forceinline__ long long fix_of(float x) { return __float2ll_rn(__fmul_rn(x, kFixScale)); }

// CL[d] = LSE_1 + ... + LSE_d (d = 0..L) of one tree's draft rows, summed in float-float in
// depth order and rounded onto the fixed grid once per depth. Called by one whole warp; lane 0
// writes CL[0..L].
__device__ __forceinline__ void depth_prefix_fixed(const float2 *lse, int L, long long *CL) {
    __syncwarp();
    const int lane = threadIdx.x & 31;
    FF l0 = FF{0.f, 0.f}, l1 = FF{0.f, 0.f};
    if (lane < L) {
        const float2 v = lse[lane];
        l0 = FF{v.x, v.y};
    }
    if (lane + 32 < L) {
        const float2 v = lse[lane + 32];
        l1 = FF{v.x, v.y};
    }
    FF acc = FF{0.f, 0.f};
    for (int d = 0; d < L; ++d) {  // prefix sums in depth order (every lane, same values)
        const FF l = d < 32 ? FF{__shfl_sync(kFull, l0.hi, d), __shfl_sync(kFull, l0.lo, d)}
                            : FF{__shfl_sync(kFull, l1.hi, d - 32), __shfl_sync(kFull, l1.lo, d - 32)};
        acc = ff_add(acc, l);
        if (lane == 0) CL[d + 1] = fix_of(acc.hi) + fix_of(acc.lo);
    }
    if (lane == 0) CL[0] = 0;
}

// The tree's outputs from per-node arrays in shared memory (node 0 the root, nodes 1..N with
// parent < node and siblings holding ranks 0..m-1): child lists by counting, an exclusive scan
// (warp 0) and placement by rank, then the per-node arrays. n_count must hold zeros; it is
// reused for the child-list starts. All NT threads of the CTA call it after a barrier.
template <int NT>
__device__ void emit_tree(int b, int N, const int32_t *n_parent, const int32_t *n_depth, const int32_t *n_rank,
                          const int32_t *n_token, int32_t *n_count, const float *n_score, const TreeDesc &tree,
                          uint32_t *status) {
    const int NN = N + 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = 1 + threadIdx.x; i <= N; i += NT)
        if (in_bounds(n_parent[i], NN, status)) atomicAdd(&n_count[n_parent[i]], 1);
    __syncthreads();
    int32_t *off = tree.child_off + (int64_t)b * (NN + 1);
    if (warp == 0) {
        __syncwarp();
        const int per = (NN + 31) / 32;
        const int lo = min(NN, lane * per), hi = min(NN, lo + per);
        int s = 0;
        for (int u = lo; u < hi; ++u) s += n_count[u];
        int incl = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += y;
        }
        int run = incl - s;
        for (int u = lo; u < hi; ++u) {
            const int c = n_count[u];
            n_count[u] = run;  // now the start of u's children
            off[u] = run;
            run += c;
        }
        if (lane == 31) off[NN] = incl;
    }
    __syncthreads();
    int32_t *ids = tree.child_ids + (int64_t)b * N;
    for (int i = 1 + threadIdx.x; i <= N; i += NT) {
        const int slot = n_count[n_parent[i]] + n_rank[i];
        if (slot >= 0 && slot < N) ids[slot] = i;  // always, unless a tree check already failed
    }
    int32_t *par = tree.parent + (int64_t)b * NN, *dep = tree.depth + (int64_t)b * NN;
    int32_t *rk = tree.rank + (int64_t)b * NN, *tok = tree.plan_token + (int64_t)b * NN;
    float *sc = tree.score + (int64_t)b * NN;
    for (int i = threadIdx.x; i < NN; i += NT) {
        par[i] = n_parent[i];
        dep[i] = n_depth[i];
        rk[i] = n_rank[i];
        tok[i] = n_token[i];
        sc[i] = n_score[i];
    }
}

// A 32-bit image of an okey, monotone non-decreasing: keys in [-2^41, 2^41) (|log-probability|
// below 2048) at 2^-20 resolution, clamped outside; an empty slot (0) maps to 0. Equal images
// are resolved on the full key.
__device__ __forceinline__ unsigned coarse_of(unsigned long long okey) {
    constexpr unsigned long long kBase = 0x8000000000000000ull - (1ull << 41);
    if (okey < kBase) return 0u;
    const unsigned long long c = (okey - kBase) >> 10;
    return c > 0xffffffffull ? 0xffffffffu : (unsigned)c;
}

template <int S>
struct Slots {
    unsigned long long k[S];  // okey
    unsigned w[S];            // tie word
    long long x[S];           // the candidate's path sum Sx (fixed point)
    unsigned long long bk;    // the lane's best
    unsigned bw;
    long long bx;
    int bs;
    __device__ __forceinline__ void clear() {
#pragma unroll
        for (int s = 0; s < S; ++s) {
            k[s] = 0ull;
            w[s] = 0u;
            x[s] = 0;
        }
        bk = 0ull;
        bw = 0u;
        bx = 0;
        bs = 0;
    }
    // Predicated writes of slot `slot` (every lane runs the same instructions).
    __device__ __forceinline__ void put_if(bool p, int slot, unsigned long long kk, unsigned ww, long long xx) {
#pragma unroll
        for (int s = 0; s < S; ++s) {
            const bool hit = p && s == slot;
            k[s] = hit ? kk : k[s];
            w[s] = hit ? ww : w[s];
            x[s] = hit ? xx : x[s];
        }
    }
    __device__ __forceinline__ void rescan() {
        bk = 0ull;
        bw = 0u;
        bx = 0;
        bs = 0;
#pragma unroll
        for (int s = 0; s < S; ++s) {
            const bool better = key_better(k[s], w[s], bk, bw);
            bk = better ? k[s] : bk;
            bw = better ? w[s] : bw;
            bx = better ? x[s] : bx;
            bs = better ? s : bs;
        }
    }
};

// ---------------------------------------------------------------------------------------
// Best-first expansion by selection. Keys never increase along a path's links: a first child's
// key is its parent's plus x - (CL[d] - CL[d-1]) <= 0 (checked per tree), a sibling's is at
// most its left neighbour's (the top-K lists are sorted). Then every candidate's predecessor
// precedes it in the global order (key desc, depth asc, parent asc, rank asc), so the max-heap's
// N pops are exactly the N first paths of that order, and the kernel finds them in parallel:
//   1. a lower bound tau on the N-th key: the top-1 chain of each length and every path that
//      leaves it once (rank r >= 1 at depth i, then rank 0 down to depth d) are real paths, so
//      the N-th largest key among them (family F0) is at most the N-th largest overall; two
//      histogram rounds over their keys (64 power-of-two bins of hi - key, then 64 sub-bins of
//      the bin holding the N-th) give a bin edge with at least N keys of F0 at or above it;
//   2. every path with key >= tau, as chains: the top-1 chain as far as it reaches tau, then
//      level by level every rank >= 1 child (reaching tau) of a node found in the level before
//      (first the root and the top-1 chain), each with its rank-0 continuation as far as it
//      reaches tau (a binary search over the chain keys). More than `cap` paths: the N-th
//      largest key among `cap` of them is a tighter bound, and the enumeration restarts;
//   3. each path's position by counting the paths before it. Parents' positions decide only
//      between equal keys at equal depths (frequent with bf16 logits): there the ancestors' keys
//      are compared upwards, then the ranks below the common ancestor. Positions 0..N-1 are
//      nodes 1..N.
// Trees whose first-child keys would rise (a rounding of the normaliser prefix above a logit),
// or whose bound does not tighten, take the serial expansion below (one warp popping the
// frontier), which gives the same tree by definition.
constexpr int kSelLevels = 64;   // chain levels (deviations from the top-1 chain) per enumeration
constexpr int kMaxDepth = 64;    // depth cap L <= 64
constexpr int kSelAttempts = 4;  // enumerations before the serial expansion takes over

__device__ __forceinline__ int sel_cap(int N) { return 4 * N + 64; }

size_t select_smem_bytes(int L, int N, int K) {
    const size_t NN = (size_t)N + 1, cap = (size_t)4 * N + 64;
    return (size_t)(L + 1) * 8 + NN * 8 + (size_t)L * K * 8 + 6 * NN * 4 + (size_t)L * K * 4 + 8 +  // heap layout
           (size_t)(L + 1) * 8 + (size_t)(L + 1) * K * 8 + cap * 8 + 4 * cap * 4;
}

struct SelShared {
    long long tau, lo;
    int hist[64];
    int nent, ovf, alo, ahi, root, mono, fast, jstar, cum, kstar, nkept;
};

// A bin edge t <= the N-th largest of a set of keys (all in [lo, hi], at least N of them) with
// at least N of them >= t: 64 power-of-two bins of hi - key, then 64 sub-bins of the bin holding
// the N-th. fill(s1, s2, jb, hist) adds every key's bin to hist: (hi - key) >> s1 for jb < 0,
// else, for the keys with (hi - key) >> s1 == jb, ((hi - key) >> s2) - (jb << (s1 - s2)).
// Every thread of the CTA calls it; ends synchronised.
template <typename F>
__device__ long long nth_bound(SelShared &ss, int N, long long hi, long long lo, F fill) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int bits = 64 - __clzll(hi - lo);  // hi - lo >= 0
    const int s1 = bits > 6 ? bits - 6 : 0;  // (hi - lo) >> s1 < 64
    const int s2 = s1 > 6 ? s1 - 6 : 0;
    for (int round = 0; round < 2; ++round) {
        if (threadIdx.x < 64) ss.hist[threadIdx.x] = 0;
        __syncthreads();
        fill(s1, s2, round == 0 ? -1 : ss.jstar, ss.hist);
        __syncthreads();
        if (warp == 0) {  // the first bin whose inclusive prefix reaches N (two bins per lane)
            __syncwarp();
            const int base = round == 0 ? 0 : ss.cum;
            const int h0 = ss.hist[2 * lane], h1 = ss.hist[2 * lane + 1];
            int incl = h0 + h1;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += y;
            }
            const int excl = base + incl - h0 - h1;
            const bool in0 = excl + h0 >= N, in1 = excl + h0 + h1 >= N;
            const unsigned m = __ballot_sync(kFull, in1);
            const int first = m ? __ffs(m) - 1 : 31;
            if (lane == first) {
                const int j = in0 ? 2 * lane : 2 * lane + 1;
                if (round == 0) {
                    ss.jstar = j;
                    ss.cum = in0 ? excl : excl + h0;
                } else {
                    ss.kstar = j;
                }
            }
        }
        __syncthreads();
    }
    const long long idx = ((long long)ss.jstar << (s1 - s2)) + ss.kstar;
    return hi - ((idx + 1) << s2) + 1;
}

// The bin of key k in a round of nth_bound (-1: outside the round's bin).
__device__ __forceinline__ int bound_bin(long long hi, long long k, int s1, int s2, int jb) {
    const unsigned long long dv = (unsigned long long)(hi - k);
    if (jb < 0) return (int)(dv >> s1);
    return (int)(dv >> s1) == jb ? (int)((dv >> s2) - ((unsigned long long)jb << (s1 - s2))) : -1;
}

// Positions in the global order (key desc, depth asc, parent's position asc, rank asc) of the
// MK enumerated paths ekept[0..MK) (with COMPACT; else paths 0..MK), by counting the paths
// before each one, four lanes per path: between equal keys at equal depths with different
// parents, the ancestors' keys compared upwards until they differ, else (equal up to the common
// ancestor) the ranks of its two children on the paths. All threads of the CTA call it.
template <bool COMPACT>
__device__ __forceinline__ void count_positions(const long long *ekey, const int32_t *einfo, const int32_t *epar,
                                                const int32_t *ekept, int MK, int32_t *epos) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int x0 = warp * 8; x0 < MK; x0 += kHeapThreads / 4) {  // uniform over the warp; four lanes per path
        const int xi = x0 + (lane >> 2), sub = lane & 3;
        const int x = xi < MK ? (COMPACT ? ekept[xi] : xi) : 0;
        int n = 0;
        if (xi < MK) {
            const long long kx = ekey[x];
            const int dx = einfo[x] & 255, rx = einfo[x] >> 8, px = epar[x];
            for (int yi = sub; yi < MK; yi += 4) {
                const int y = COMPACT ? ekept[yi] : yi;
                const long long ky = ekey[y];
                int add = ky > kx ? 1 : 0;
                if (ky == kx && y != x) {
                    const int iy = einfo[y], dy = iy & 255;
                    if (dy < dx) {
                        add = 1;
                    } else if (dy == dx) {
                        const int py = epar[y];
                        if (py == px) {
                            add = (iy >> 8) < rx ? 1 : 0;
                        } else {  // both at depth >= 2: walk up to the first difference
                            int cx = x, cy = y, ax = px, ay = py, before = -1;
                            for (int up = 0; up < kMaxDepth && before < 0; ++up) {
                                if (ax == ay) {
                                    before = (einfo[cy] >> 8) < (einfo[cx] >> 8) ? 1 : 0;
                                } else if (ekey[ax] != ekey[ay]) {
                                    before = ekey[ay] > ekey[ax] ? 1 : 0;
                                } else {
                                    cx = ax;
                                    cy = ay;
                                    ax = epar[ax];
                                    ay = epar[ay];
                                }
                            }
                            add = before > 0 ? 1 : 0;
                        }
                    }
                }
                n += add;
            }
        }
        __syncwarp();  // after the lanes' ancestor walks
        n += __shfl_xor_sync(kFull, n, 1);
        n += __shfl_xor_sync(kFull, n, 2);
        if (xi < MK && sub == 0) epos[x] = n;
    }
}

// Max-heap expansion by selection (steps 1-3 above), with the serial expansion as fallback.
// Each pop of the serial expansion: a warp maximum of the lanes' best keys, one
// __reduce_max_sync on a 32-bit monotone image of the key, refined on the full key (high word,
// low word, tie word) only among lanes whose images tie; the popped candidate's slot takes its
// next sibling; its first child goes to the next round-robin slot (children are numbered in
// creation order, lane = c % 32, slot = c / 32).
template <int S>
__global__ void __launch_bounds__(kHeapThreads) k_plan_select(HeapArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ SelShared ss;
    const int L = a.L, N = a.N, K = a.K, NN = N + 1;
    long long *CL = reinterpret_cast<long long *>(smem);           // [L+1] fixed point
    long long *n_sx = CL + (L + 1);                                // [NN] raw pop keys
    long long *fx = n_sx + NN;                                     // [L*K] candidate logits
    int32_t *n_parent = reinterpret_cast<int32_t *>(fx + L * K);   // [NN]
    int32_t *n_depth = n_parent + NN;
    int32_t *n_rank = n_depth + NN;
    int32_t *n_token = n_rank + NN;
    int32_t *n_count = n_token + NN;                               // [NN]
    float *n_score = reinterpret_cast<float *>(n_count + NN);      // [NN]
    int32_t *tk_id = reinterpret_cast<int32_t *>(n_score + NN);    // [L*K]
    const int cap = sel_cap(N);
    long long *Bk = reinterpret_cast<long long *>(smem + ((size_t)(L + 1) * 8 + (size_t)NN * 8 + (size_t)L * K * 8 +
                                                          6 * (size_t)NN * 4 + (size_t)L * K * 4 + 7) / 8 * 8);
    long long *dl = Bk + (L + 1);             // [(L+1)*K] key step of rank r at depth d: dl[d*K + r]
    long long *ekey = dl + (size_t)(L + 1) * K;  // [cap] enumerated paths
    int32_t *einfo = reinterpret_cast<int32_t *>(ekey + cap);  // depth | rank << 8
    int32_t *epar = einfo + cap;                               // parent entry (-1: the root)
    int32_t *epos = epar + cap;                                // position in the global order
    int32_t *ekept = epos + cap;                               // the entries that get a position

    const int b = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < L * K; i += kHeapThreads) {
        tk_id[i] = a.topk_id[(int64_t)b * L * K + i];
        fx[i] = fix_of(a.topk_x[(int64_t)b * L * K + i]);
    }
    for (int i = threadIdx.x; i < NN; i += kHeapThreads) {  // defined even if the expansion stops early
        n_count[i] = 0;
        n_parent[i] = 0;
        n_depth[i] = 0;
        n_rank[i] = 0;
        n_token[i] = -1;
        n_score[i] = 0.f;
        n_sx[i] = 0;
    }
    if (warp == 0) depth_prefix_fixed(a.lse + (int64_t)b * L, L, CL);
    __syncthreads();

    // ---- 1. key steps, the top-1 chain keys Bk[d], monotonicity, the bound from F0
    for (int i = threadIdx.x; i < L * K; i += kHeapThreads) {
        const int d = i / K + 1;
        dl[d * K + i % K] = fx[i] - (CL[d] - CL[d - 1]);
    }
    __syncthreads();
    if (warp == 0) {  // Bk[d] = dl[1][0] + ... + dl[d][0] by a warp scan (depths lane + 1, lane + 33)
        __syncwarp();
        const long long a0 = lane < L ? dl[(lane + 1) * K] : 0, a1 = lane + 32 < L ? dl[(lane + 33) * K] : 0;
        long long c0 = lane < L ? dl[(lane + 1) * K] - dl[(lane + 1) * K + K - 1] : 0;
        const long long c1 = lane + 32 < L ? dl[(lane + 33) * K] - dl[(lane + 33) * K + K - 1] : 0;
        long long s0 = a0, s1 = a1;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const long long y0 = __shfl_up_sync(kFull, s0, o), y1 = __shfl_up_sync(kFull, s1, o);
            if (lane >= o) {
                s0 += y0;
                s1 += y1;
            }
        }
        s1 += __shfl_sync(kFull, s0, 31);
        if (lane < L) Bk[lane + 1] = s0;
        if (lane + 32 < L) Bk[lane + 33] = s1;
        c0 = c0 > c1 ? c0 : c1;  // the largest step off the chain at any depth: lo = Bk[L] - that
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const long long y = __shfl_xor_sync(kFull, c0, o);
            c0 = y > c0 ? y : c0;
        }
        const int bad = __ballot_sync(kFull, a0 > 0 || a1 > 0) != 0u;
        const long long bkl = __shfl_sync(kFull, L <= 32 ? s0 : s1, (L - 1) & 31);
        if (lane == 0) {
            Bk[0] = 0;
            ss.mono = !bad;
            ss.fast = !bad;
            ss.lo = bkl - c0;
        }
    }
    __syncthreads();
    long long tau = -(1ll << 62);
    const long long hi = Bk[1];
    if (ss.fast) {
        const long long nF0 = (long long)L + (long long)(K - 1) * L * (L + 1) / 2;
        if (nF0 >= N) {
            const long long lo = ss.lo;
            // F0 as sorted sequences: q = 0 the top-1 chain Bk[1..L]; q = 1 + (i - 1) (K - 1) + r - 1
            // the paths leaving it at depth i with rank r, Bk[d] - c (d = i..L). Bins grow along a
            // sequence, so each thread adds runs of equal bins.
            const int nq = 1 + L * (K - 1);
            tau = nth_bound(ss, N, hi, lo, [&](int s1, int s2, int jb, int *hist) {
                for (int q = threadIdx.x; q < nq; q += kHeapThreads) {
                    int d0 = 1;
                    long long c = 0;
                    if (q > 0) {
                        const int i = 1 + (q - 1) / (K - 1), r = 1 + (q - 1) % (K - 1);
                        d0 = i;
                        c = dl[i * K] - dl[i * K + r];
                    }
                    int run_bin = -1, run = 0;
                    for (int d = d0; d <= L; ++d) {
                        const int bin = bound_bin(hi, Bk[d] - c, s1, s2, jb);
                        if (bin != run_bin) {
                            if (run_bin >= 0) atomicAdd(&hist[run_bin], run);
                            run_bin = bin;
                            run = 0;
                        }
                        ++run;
                    }
                    if (run_bin >= 0) atomicAdd(&hist[run_bin], run);
                }
            });
        }
    }

    // ---- 2. every path with key >= tau, as chains
    bool fast = ss.fast != 0;
    int M = 0;
    for (int attempt = 0; fast && attempt < kSelAttempts; ++attempt) {
        if (threadIdx.x == 0) {  // the top-1 chain: a prefix of depths (Bk decreases)
            int l0 = 0, h0 = L;  // the last depth whose chain key reaches tau
            while (l0 < h0) {
                const int mid = (l0 + h0 + 1) >> 1;
                if (Bk[mid] >= tau)
                    l0 = mid;
                else
                    h0 = mid - 1;
            }
            ss.nent = min(l0, cap);
            ss.ovf = l0 > cap;
            ss.alo = 0;
            ss.ahi = min(l0, cap);
            ss.root = 1;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < ss.ahi; e += kHeapThreads) {
            ekey[e] = Bk[e + 1];
            einfo[e] = e + 1;
            epar[e] = e - 1;
        }
        __syncthreads();
        for (int lev = 0; lev < kSelLevels && !ss.ovf; ++lev) {  // uniform: read after a barrier
            const int alo = ss.alo, ahi = ss.ahi, root = ss.root;
            const int na = root + (ahi - alo);
            if (na == 0) break;
            const int nc = na * (K - 1);
            for (int c = threadIdx.x; c < nc; c += kHeapThreads) {
                const int ai = c / (K - 1), r = 1 + c % (K - 1);
                int ae = -1, da = 0;
                long long ka = 0;
                if (!(root && ai == 0)) {
                    ae = alo + ai - root;
                    da = einfo[ae] & 255;
                    ka = ekey[ae];
                }
                const int d = da + 1;
                if (d > L) continue;
                const long long key = ka + dl[d * K + r];
                if (key < tau) continue;
                int lo2 = d, hi2 = L;  // the last depth whose rank-0 continuation reaches tau
                while (lo2 < hi2) {
                    const int mid = (lo2 + hi2 + 1) >> 1;
                    if (key + Bk[mid] - Bk[d] >= tau)
                        lo2 = mid;
                    else
                        hi2 = mid - 1;
                }
                const int n = 1 + lo2 - d;
                const int base = atomicAdd(&ss.nent, n);
                if (base + n > cap) ss.ovf = 1;
                for (int j = 0; j < n && base + j < cap; ++j) {
                    ekey[base + j] = j == 0 ? key : key + Bk[d + j] - Bk[d];
                    einfo[base + j] = (d + j) | ((j == 0 ? r : 0) << 8);
                    epar[base + j] = j == 0 ? ae : base + j - 1;
                }
            }
            __syncthreads();
            if (threadIdx.x == 0) {
                ss.alo = ahi;
                ss.ahi = min(ss.nent, cap);
                ss.root = 0;
            }
            __syncthreads();
        }
        M = min(ss.nent, cap);
        if (!ss.ovf) break;
        const long long t2 = nth_bound(ss, N, hi, tau, [&](int s1, int s2, int jb, int *hist) {
            for (int f = threadIdx.x; f < cap; f += kHeapThreads) {
                const int bin = bound_bin(hi, ekey[f], s1, s2, jb);
                if (bin >= 0) atomicAdd(&hist[bin], 1);
            }
        });
        if (t2 <= tau || attempt + 1 == kSelAttempts) {
            fast = false;
            break;
        }
        tau = t2;
        __syncthreads();
    }
    if (fast && M < N) fast = false;

    if (fast) {
        // ---- 3. positions by counting, among the paths whose key reaches t: with many more
        //      paths than N, t is a second bound from the enumerated keys (at least N of them reach
        //      it); a path's predecessors in the order all have keys >= its own, so they all
        //      reach t and the counts among these paths are the global positions, and a parent
        //      (key >= its child's) reaches t with its child. Between equal keys at equal depths
        //      with different parents the order is that of the parents, recursively: ancestors'
        //      keys compared upwards until they differ, else (equal up to the common ancestor)
        //      the ranks of its two children on the paths.
        const bool compact = M > N + (N >> 3);  // uniform: M from shared memory after a barrier
        int MK = M;
        if (compact) {
            const long long t = nth_bound(ss, N, hi, tau, [&](int s1, int s2, int jb, int *hist) {
                for (int f = threadIdx.x; f < M; f += kHeapThreads) {
                    const int bin = bound_bin(hi, ekey[f], s1, s2, jb);
                    if (bin >= 0) atomicAdd(&hist[bin], 1);
                }
            });
            if (threadIdx.x == 0) ss.nkept = 0;
            __syncthreads();
            for (int x = threadIdx.x; x < M; x += kHeapThreads) {
                epos[x] = -1;
                if (ekey[x] >= t) {
                    const int p = atomicAdd(&ss.nkept, 1);
                    if (in_bounds(p, cap, a.status)) ekept[p] = x;
                }
            }
            __syncthreads();
            MK = min(ss.nkept, cap);
        }
        if (compact)
            count_positions<true>(ekey, einfo, epar, ekept, MK, epos);
        else
            count_positions<false>(ekey, einfo, epar, ekept, MK, epos);
        __syncthreads();
        bool bad = false;
        for (int x = threadIdx.x; x < M; x += kHeapThreads) {
            const int pos = epos[x];
            if (pos < 0 || pos >= N) continue;
            const int i = pos + 1, d = einfo[x] & 255, r = einfo[x] >> 8;
            if (epar[x] >= 0 && !in_bounds(epar[x], M, a.status)) continue;
            if (!in_bounds(d - 1, L, a.status) || !in_bounds(r, K, a.status)) continue;
            const int par = epar[x] < 0 ? 0 : epos[epar[x]] + 1;
            if (par >= i) bad = true;
            n_parent[i] = par;
            n_depth[i] = d;
            n_rank[i] = r;
            n_token[i] = tk_id[(d - 1) * K + r];
            n_score[i] = __fmul_rn(__ll2float_rn(ekey[x]), kFixInv);
        }
        if (bad) raise_status(a.status, kDevBadTree);
        if (threadIdx.x == 0) {
            n_parent[0] = -1;
            n_depth[0] = 0;
            n_rank[0] = -1;
            n_token[0] = -1;
            n_score[0] = 0.f;
        }
        __syncthreads();
        emit_tree<kHeapThreads>(b, N, n_parent, n_depth, n_rank, n_token, n_count, n_score, a.tree, a.status);
        return;
    }
    // The expansion (warp 0). Per pop the critical path is the warp maximum, three shuffles,
    // the decode, independent shared loads of the candidate logits and depth normalisers, and
    // predicated slot updates: no dependent load of the parent's path sum (each slot carries
    // its own) and no divergent branch. Each pop's tie word and key are stored raw and
    // decoded after the loop by all threads.
    unsigned *rec_w = reinterpret_cast<unsigned *>(n_rank);  // [NN], 0 = not popped
    long long *rec_k = n_sx;                                  // [NN]
    if (warp == 0) {
        Slots<S> fr;
        fr.clear();
        // the root's first child (depth 1, rank 0) is child number 0: lane 0, slot 0
        fr.put_if(lane == 0, 0, okey_of(fx[0] - CL[1]), w3_of(1, 0, 0), fx[0]);
        fr.rescan();
        int nchild = 1;
        for (int i = 1; i <= N; ++i) {
            __syncwarp();
            const unsigned ck = coarse_of(fr.bk);
            const unsigned m0 = __reduce_max_sync(kFull, ck);
            unsigned c = __ballot_sync(kFull, ck == m0);
            if (__popc(c) > 1) {  // coarse keys tie: the full key (high word, low word), then w3
                const unsigned hk = (unsigned)(fr.bk >> 32);
                const unsigned m1 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? hk : 0u);
                c &= __ballot_sync(kFull, hk == m1);
                const unsigned lk = (unsigned)fr.bk;
                const unsigned m2 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? lk : 0u);
                c &= __ballot_sync(kFull, lk == m2);
                if (__popc(c) > 1) {
                    const unsigned m3 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? fr.bw : 0u);
                    c &= __ballot_sync(kFull, fr.bw == m3);
                }
            }
            const int winner = __ffs(c) - 1;
            const unsigned ww = __shfl_sync(kFull, fr.bw, winner);
            const long long wx = __shfl_sync(kFull, fr.bx, winner);
            if (ww == 0u) {  // frontier exhausted: only with N above the tree's capacity
                if (lane == 0) raise_status(a.status, kDevBadTree);
                break;
            }
            if (lane == winner) {  // the pop's record, before its slot is overwritten
                rec_w[i] = ww;
                rec_k[i] = (long long)fr.bk;
            }
            const int depth = 255 - (int)(ww >> 24);
            const int parent = 65535 - (int)((ww >> 8) & 0xffffu);
            const int rank = 255 - (int)(ww & 0xffu);
            const bool sib = rank + 1 < K, kid = depth < L;
            const long long fr0 = fx[(depth - 1) * K + rank];
            const long long fn = sib ? fx[(depth - 1) * K + rank + 1] : 0;
            const long long f0 = kid ? fx[depth * K] : 0;
            const long long cd = CL[depth], cd1 = kid ? CL[depth + 1] : 0;
            const long long xs = wx - fr0 + fn, xc = wx + f0;  // sibling's and first child's Sx
            // the next sibling takes the popped slot; the first child the next round-robin slot
            fr.put_if(lane == winner, fr.bs, sib ? okey_of(xs - cd) : 0ull, sib ? w3_of(depth, parent, rank + 1) : 0u,
                      xs);
            fr.put_if(kid && lane == (nchild & 31), nchild >> 5, okey_of(xc - cd1), w3_of(depth + 1, i, 0), xc);
            fr.rescan();
            nchild += kid ? 1 : 0;
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < NN; i += kHeapThreads) {  // decode the records
        if (i == 0) {
            n_parent[0] = -1;
            n_depth[0] = 0;
            n_rank[0] = -1;
            n_token[0] = -1;
            n_score[0] = 0.f;
            continue;
        }
        const unsigned ww = rec_w[i];
        if (ww == 0u) continue;  // not popped (the expansion stopped early)
        const int depth = 255 - (int)(ww >> 24);
        const int rank = 255 - (int)(ww & 0xffu);
        n_parent[i] = 65535 - (int)((ww >> 8) & 0xffffu);
        n_depth[i] = depth;
        n_rank[i] = rank;
        n_token[i] = tk_id[(depth - 1) * K + rank];
        n_score[i] = __fmul_rn(__ll2float_rn(key_of_okey((unsigned long long)rec_k[i])), kFixInv);
    }
    __syncthreads();

    emit_tree<kHeapThreads>(b, N, n_parent, n_depth, n_rank, n_token, n_count, n_score, a.tree, a.status);
}

// ---------------------------------------------------------------------------------------
// Expand-then-prune first pass (the EAGLE-2-style planner of Sec. 3.1 and App. B.3), one CTA
// per tree. Layer 1 is the root's K children; layer d+1 holds the K children of each of the W
// best candidates of layer d (its frontier), so layers stay at most W*K wide and L layers
// deep. Every layer is kept sorted by (key desc, parent's position asc, rank asc): a layer of at
// most kEptSmallLayer candidates by counting, for each candidate, the ones before it (several
// threads per candidate); a wider one by binary search: candidate (f, r) of layer d+1 has sum
// Sx = Sx_f + x_{d,r}, the candidates of frontier entry f' that precede it are those whose logit
// exceeds Sx - Sx_f' (or reaches it when f' < f), a prefix of the depth's sorted top-K logits,
// and its position is r plus those counts.
// After the last layer, one warp merges the sorted layers in the global order (key desc, depth
// asc, parent's position asc, rank asc): the N first are the nodes, numbered in that order.
// Keys are the 64-bit fixed-point path sums of the max-heap planner, so same-depth comparisons
// are exact and a frontier holding N candidates gives the heap's tree bit for bit.
constexpr int kEptThreads = 512;
constexpr int kEptSmallLayer = 512;  // layers up to this size are ranked by counting

struct EptArgs {
    int L, N, K, W;
    const float2 *lse;
    const float *topk_x;
    const int32_t *topk_id;
    TreeDesc tree;
    uint32_t *status;
};

size_t ept_smem_bytes(int L, int N, int K, int G) {
    const size_t NN = (size_t)N + 1;
    return (size_t)(L + 1) * 8 + (size_t)L * K * 8 + (size_t)G * 8 + (size_t)L * K * 4 + (size_t)G * 8 +
           (size_t)(L + 2) * 4 + 6 * NN * 4;
}

__global__ void __launch_bounds__(kEptThreads) k_plan_ept(EptArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) unsigned char smem[];
    const int L = a.L, N = a.N, K = a.K, W = a.W, NN = N + 1;
    const int G = (int)ept_layer_start(L + 1, K, W);
    long long *CL = reinterpret_cast<long long *>(smem);          // [L+1]
    long long *fx = CL + (L + 1);                                 // [L*K] candidate logits, fixed point
    long long *skey = fx + L * K;                                 // [G] keys, each layer sorted
    int32_t *tk_id = reinterpret_cast<int32_t *>(skey + G);       // [L*K]
    int32_t *smeta = tk_id + L * K;                               // [G] (parent position << 8) | rank
    int32_t *node_of = smeta + G;                                 // [G] node number, 0 if not kept
    int32_t *lstart = node_of + G;                                // [L+2]
    int32_t *n_parent = lstart + (L + 2);                         // [NN] each
    int32_t *n_depth = n_parent + NN;
    int32_t *n_rank = n_depth + NN;
    int32_t *n_token = n_rank + NN;
    int32_t *n_count = n_token + NN;
    float *n_score = reinterpret_cast<float *>(n_count + NN);

    const int b = blockIdx.x;
    const int warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < L * K; i += kEptThreads) {
        tk_id[i] = a.topk_id[(int64_t)b * L * K + i];
        fx[i] = fix_of(a.topk_x[(int64_t)b * L * K + i]);
    }
    for (int i = threadIdx.x; i < NN; i += kEptThreads) {
        n_count[i] = 0;
        n_parent[i] = i == 0 ? -1 : 0;
        n_depth[i] = 0;
        n_rank[i] = i == 0 ? -1 : 0;
        n_token[i] = -1;
        n_score[i] = 0.f;
    }
    for (int d = 1 + threadIdx.x; d <= L + 1; d += kEptThreads) lstart[d] = (int)ept_layer_start(d, K, W);
    if (warp == 0) depth_prefix_fixed(a.lse + (int64_t)b * L, L, CL);
    __syncthreads();

    // 1. layer 1 is sorted as built (the draft row's logits do not increase with rank)
    for (int j = threadIdx.x; j < K; j += kEptThreads) {
        skey[j] = fx[j] - CL[1];
        smeta[j] = j;
    }
    __syncthreads();
    // 2. layers 2..L, each placed at its sorted positions: a layer of at most kEptSmallLayer
    //    candidates by counting the candidates before each, a wider one by binary searches over
    //    the depth's sorted logits
    __shared__ long long tkey[kEptSmallLayer];
    __shared__ int tpos[kEptSmallLayer];
    int kbits = 0;  // steps of the binary search over a depth's K logits
    while ((1 << kbits) <= K) ++kbits;
    for (int d = 1; d < L; ++d) {
        const int prev = lstart[d], nf = min(W, lstart[d + 1] - prev), base = lstart[d + 1];
        const long long cd = CL[d], cd1 = CL[d + 1];
        const long long *row = fx + d * K;  // logits of depth d+1, non-increasing in rank
        if (nf * K <= kEptSmallLayer) {  // uniform over the CTA
            const int n = nf * K;
            for (int j = threadIdx.x; j < n; j += kEptThreads) {
                const int f = j / K, r = j - f * K;
                tkey[j] = skey[prev + f] + cd + row[r] - cd1;
                tpos[j] = 0;
            }
            __syncthreads();
            // candidate j's position = the candidates before it (larger key, or the same key and a
            // smaller index: index order j = f*K + r is the order of equal keys), counted by
            // S threads per candidate over slices of the layer
            const int S = max(1, kEptThreads / n), per = (n + S - 1) / S;
            for (int t = threadIdx.x; t < n * S; t += kEptThreads) {
                const int j = t / S, part = t - j * S;
                const long long key = tkey[j];
                const int lo = part * per, hi = min(n, lo + per);
                int cnt = 0;
#pragma unroll 4
                for (int i2 = lo; i2 < hi; ++i2) {
                    const long long k2 = tkey[i2];
                    cnt += (k2 > key || (k2 == key && i2 < j)) ? 1 : 0;
                }
                if (cnt) atomicAdd(&tpos[j], cnt);
            }
            __syncthreads();
            for (int j = threadIdx.x; j < n; j += kEptThreads) {
                const int f = j / K, r = j - f * K;
                skey[base + tpos[j]] = tkey[j];
                smeta[base + tpos[j]] = (f << 8) | r;
            }
            __syncthreads();  // before the next layer reads skey and rewrites tkey
            continue;
        }
        for (int j = threadIdx.x; j < nf * K; j += kEptThreads) {
            const int f = j / K, r = j - f * K;
            const long long sx = skey[prev + f] + cd + row[r];
            int pos = r;
            for (int f2 = 0; f2 < nf; ++f2) {
                if (f2 == f) continue;
                const long long t = sx - (skey[prev + f2] + cd);
                const bool incl = f2 < f;
                int c = 0;  // logits of the depth above t (at or above t when incl)
                for (int step = 1 << (kbits - 1); step > 0; step >>= 1)
                    if (c + step <= K && (incl ? row[c + step - 1] >= t : row[c + step - 1] > t)) c += step;
                pos += c;
            }
            skey[base + pos] = sx - cd1;
            smeta[base + pos] = (f << 8) | r;
        }
        __syncthreads();
    }
    // 3. the first N of the global order, merged from the sorted layers by one warp: lane l
    //    holds the heads of layers l+1 and l+33; each step takes the largest head by (key desc,
    //    depth asc), the 32-bit monotone image of the key first, the full key and the depth
    //    only among lanes that tie on it
    for (int idx = threadIdx.x; idx < G; idx += kEptThreads) node_of[idx] = 0;
    __syncthreads();
    if (warp == 0) {
        const int lane = threadIdx.x & 31;
        const int dA = lane + 1, dB = lane + 33;
        const int sA = dA <= L ? lstart[dA] : 0, nA = dA <= L ? lstart[dA + 1] - sA : 0;
        const int sB = dB <= L ? lstart[dB] : 0, nB = dB <= L ? lstart[dB + 1] - sB : 0;
        int pA = 0, pB = 0;
        unsigned long long kA = nA > 0 ? okey_of(skey[sA]) : 0ull;
        unsigned long long kB = nB > 0 ? okey_of(skey[sB]) : 0ull;
        for (int i = 1; i <= N; ++i) {
            __syncwarp();
            const bool useB = kB > kA;  // equal keys: the shallower layer A first
            const unsigned long long kb = useB ? kB : kA;
            const unsigned wd = 255u - (unsigned)(useB ? dB : dA);
            const unsigned ck = coarse_of(kb);
            const unsigned m0 = __reduce_max_sync(kFull, ck);
            unsigned c = __ballot_sync(kFull, ck == m0);
            if (__popc(c) > 1) {
                const unsigned hk = (unsigned)(kb >> 32);
                const unsigned m1 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? hk : 0u);
                c &= __ballot_sync(kFull, hk == m1);
                const unsigned lk = (unsigned)kb;
                const unsigned m2 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? lk : 0u);
                c &= __ballot_sync(kFull, lk == m2);
                const unsigned m3 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? wd : 0u);
                c &= __ballot_sync(kFull, wd == m3);
            }
            const int owner = __ffs(c) - 1;
            if (__shfl_sync(kFull, kb, owner) == 0ull) {  // every layer used up (N > G: rejected on the host)
                if (lane == 0) raise_status(a.status, kDevBadTree);
                break;
            }
            if (lane == owner) {
                if (useB) {
                    node_of[sB + pB] = i;
                    ++pB;
                    kB = pB < nB ? okey_of(skey[sB + pB]) : 0ull;
                } else {
                    node_of[sA + pA] = i;
                    ++pA;
                    kA = pA < nA ? okey_of(skey[sA + pA]) : 0ull;
                }
            }
        }
    }
    __syncthreads();
    bool bad = false;
    for (int idx = threadIdx.x; idx < G; idx += kEptThreads) {
        const int i = node_of[idx];
        if (i == 0) continue;
        int d = 1;
        while (lstart[d + 1] <= idx) ++d;
        const int meta = smeta[idx], f = meta >> 8, r = meta & 255;
        int par = d == 1 ? 0 : node_of[lstart[d - 1] + f];
        if (d > 1 && (par == 0 || par >= i)) {  // a child's key rounded above its parent's
            bad = true;
            par = 0;
        }
        n_parent[i] = par;
        n_depth[i] = d;
        n_rank[i] = r;
        n_token[i] = tk_id[(d - 1) * K + r];
        n_score[i] = __fmul_rn(__ll2float_rn(skey[idx]), kFixInv);
    }
    if (bad) raise_status(a.status, kDevBadTree);
    __syncthreads();
    emit_tree<kEptThreads>(b, N, n_parent, n_depth, n_rank, n_token, n_count, n_score, a.tree, a.status);
}

template <int S>
cudaError_t launch_heap_t(const HeapArgs &h, int B, cudaStream_t s) {
    const size_t smem = select_smem_bytes(h.L, h.N, h.K);
    cudaError_t e = cudaFuncSetAttribute(k_plan_select<S>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_plan_select<S>, dim3((unsigned)B), dim3(kHeapThreads), smem, s, 0, h);
}

template <int KCAP, typename T>
cudaError_t launch_topk_t(const TopkArgs &a, cudaStream_t s) {
    const size_t smem = (size_t)a.C * (sizeof(float2) + sizeof(uint64_t));  // statistics, candidates
    cudaError_t e = cudaFuncSetAttribute(k_row_topk<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_row_topk<KCAP, T>, dim3((unsigned)(a.B * a.L)), dim3(kTopkThreads), smem, s, 0, a);
}

template <int KCAP, typename T>
cudaError_t launch_stats_topk_t(const TopkArgs &a, cudaStream_t s) {
    const size_t smem = (size_t)a.C * (sizeof(float2) + sizeof(uint64_t));  // statistics, candidates
    cudaError_t e =
        cudaFuncSetAttribute(k_row_stats_topk<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_row_stats_topk<KCAP, T>, dim3((unsigned)(a.B * a.L)), dim3(kRowPlanThreads), smem, s, 0, a);
}

cudaError_t launch_ept(const EptArgs &e, int B, cudaStream_t s) {
    const int G = (int)ept_layer_start(e.L + 1, e.K, e.W);
    const size_t smem = ept_smem_bytes(e.L, e.N, e.K, G);
    cudaError_t err = cudaFuncSetAttribute(k_plan_ept, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (err != cudaSuccess) return err;
    return launch_pdl(k_plan_ept, dim3((unsigned)B), dim3(kEptThreads), smem, s, 0, e);
}

// The frontier kernel with as many slots per lane as N first children need.
cudaError_t launch_heap(const HeapArgs &h, int B, cudaStream_t s) {
    // Child numbers 0..N-1 need slots: child number c is created by pop c at the earliest, so
    // number N can only come from the last pop and is never popped (its slot index N / 32 may
    // lie past the last slot, where the predicated write matches no slot).
    const int per_lane = (h.N + 31) / 32;
    if (per_lane <= 1) return launch_heap_t<1>(h, B, s);
    if (per_lane <= 2) return launch_heap_t<2>(h, B, s);
    if (per_lane <= 3) return launch_heap_t<3>(h, B, s);
    if (per_lane <= 4) return launch_heap_t<4>(h, B, s);
    if (per_lane <= 8) return launch_heap_t<8>(h, B, s);
    if (per_lane <= 16) return launch_heap_t<16>(h, B, s);
    return launch_heap_t<32>(h, B, s);  // N <= 1024
}

TopkArgs topk_args(const RowsDesc &draft, const float2 *stats, int L, int K, float invT, const PlanScratch &sc) {
    TopkArgs t;
    t.draft = draft.data;
    t.bstride = draft.batch_stride;
    t.rstride = draft.row_stride;
    t.B = draft.B;
    t.R = draft.R;
    t.V = draft.V;
    t.C = num_chunks(draft.V);
    t.L = L;
    t.K = K;
    t.stats = stats;
    t.stats_out = nullptr;
    t.status = nullptr;
    t.invT = invT;
    t.lse = sc.lse;
    t.topk_x = sc.topk_x;
    t.topk_id = sc.topk_id;
    return t;
}

HeapArgs heap_args(int L, int N, int K, const PlanScratch &sc, const TreeDesc &tree, uint32_t *status) {
    HeapArgs h;
    h.L = L;
    h.N = N;
    h.K = K;
    h.lse = sc.lse;
    h.topk_x = sc.topk_x;
    h.topk_id = sc.topk_id;
    h.tree = tree;
    h.status = status;
    return h;
}

}  // namespace

PlanScratch plan_scratch(void *ws, int B, int N, int L, int K) {
    unsigned char *p = static_cast<unsigned char *>(ws) + ws_plan_offset(B, N);
    PlanScratch s;
    s.lse = reinterpret_cast<float2 *>(p);
    s.topk_x = reinterpret_cast<float *>(p + (size_t)B * L * sizeof(float2));
    s.topk_id = reinterpret_cast<int32_t *>(p + (size_t)B * L * sizeof(float2) + (size_t)B * L * K * sizeof(float));
    return s;
}

cudaError_t launch_plan(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                        const TreeDesc &tree, void *ws, cudaStream_t s) {
    const PlanScratch sc = plan_scratch(ws, draft.B, N, L, K);
    const TopkArgs t = topk_args(draft, stats, L, K, invT, sc);
    cudaError_t e;
    if (draft.dtype == 1)
        e = K <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = K <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    return launch_heap(heap_args(L, N, K, sc, tree, static_cast<uint32_t *>(ws)), draft.B, s);
}

cudaError_t launch_plan_rows(const RowsDesc &draft, float2 *stats_out, int L, int N, int K, float invT,
                             const TreeDesc &tree, void *ws, cudaStream_t s) {
    const PlanScratch sc = plan_scratch(ws, draft.B, N, L, K);
    TopkArgs t = topk_args(draft, nullptr, L, K, invT, sc);
    t.stats_out = stats_out;
    t.status = static_cast<uint32_t *>(ws);
    cudaError_t e;
    if (draft.dtype == 1)
        e = K <= 8 ? launch_stats_topk_t<8, __nv_bfloat16>(t, s) : launch_stats_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = K <= 8 ? launch_stats_topk_t<8, float>(t, s) : launch_stats_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    return launch_heap(heap_args(L, N, K, sc, tree, static_cast<uint32_t *>(ws)), draft.B, s);
}

// The per-row top-K pass (fused with the statistics when stats_out is given), then the
// expand-then-prune planner with frontier width W.
cudaError_t launch_plan_expand(const RowsDesc &draft, const float2 *stats, float2 *stats_out, int L, int N, int K,
                               int W, float invT, const TreeDesc &tree, void *ws, cudaStream_t s) {
    const PlanScratch sc = plan_scratch(ws, draft.B, N, L, K);
    TopkArgs t = topk_args(draft, stats, L, K, invT, sc);
    cudaError_t e;
    if (stats_out) {
        t.stats_out = stats_out;
        t.status = static_cast<uint32_t *>(ws);
        if (draft.dtype == 1)
            e = K <= 8 ? launch_stats_topk_t<8, __nv_bfloat16>(t, s) : launch_stats_topk_t<32, __nv_bfloat16>(t, s);
        else
            e = K <= 8 ? launch_stats_topk_t<8, float>(t, s) : launch_stats_topk_t<32, float>(t, s);
    } else {
        if (draft.dtype == 1)
            e = K <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
        else
            e = K <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    }
    if (e != cudaSuccess) return e;
    EptArgs ea;
    ea.L = L;
    ea.N = N;
    ea.K = K;
    ea.W = W;
    ea.lse = sc.lse;
    ea.topk_x = sc.topk_x;
    ea.topk_id = sc.topk_id;
    ea.tree = tree;
    ea.status = static_cast<uint32_t *>(ws);
    return launch_ept(ea, draft.B, s);
}

// Pooled first pass: the per-row top-P pass (k_pool_select for P > 32) writes the pools (ids
// only) to pool_ids, then
// k_pool_finish turns each pool into the pooled log-normaliser and the K candidates, then the
// max-heap expansion as in launch_plan.
cudaError_t launch_plan_pooled(const RowsDesc &draft, const float2 *stats, int L, int N, int K, int P, float invT,
                               int32_t *pool_ids, const TreeDesc &tree, void *ws, cudaStream_t s) {
    const PlanScratch sc = plan_scratch(ws, draft.B, N, L, K);
    TopkArgs t = topk_args(draft, stats, L, P, invT, sc);
    t.topk_id = pool_ids;
    t.topk_x = nullptr;
    cudaError_t e;
    if (P > 32)  // pools above the top-K pass's 32: the exact selection kernel
        e = launch_pool_select(draft, stats, L, P, invT, pool_ids, s);
    else if (draft.dtype == 1)
        e = P <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = P <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    e = launch_pool_finish(draft, L, K, P, invT, pool_ids, sc.lse, sc.topk_x, sc.topk_id, static_cast<uint32_t *>(ws),
                           s);
    if (e != cudaSuccess) return e;
    return launch_heap(heap_args(L, N, K, sc, tree, static_cast<uint32_t *>(ws)), draft.B, s);
}

}  // namespace tsb

namespace tsb {

// The same two launches as launch_plan, with the per-draft-row scratch and the status word
// given explicitly instead of being carved out of a caller workspace.
cudaError_t launch_plan_scratch(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                                const TreeDesc &tree, const PlanScratch &sc, uint32_t *status, cudaStream_t s) {
    const TopkArgs t = topk_args(draft, stats, L, K, invT, sc);
    cudaError_t e;
    if (draft.dtype == 1)
        e = K <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = K <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    return launch_heap(heap_args(L, N, K, sc, tree, status), draft.B, s);
}

}  // namespace tsb
