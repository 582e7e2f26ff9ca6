// First pass (Sec. 3.1; max-heap expansion as in DDTree, Sec. 2.2 / App. B.3), two kernels.
//
// k_row_topk, one warp per draft row (every row of the batch in parallel): the row's chunk
//   statistics are staged in shared memory, merged into the log-normaliser LSE_d, and give
//   tau = the K-th largest chunk maximum, a lower bound on the K-th largest logit (K distinct
//   chunk maxima reach it). Only chunks whose maximum reaches tau are re-read; their logits
//   >= tau go through per-lane sorted lists, and a warp merge yields the top-K by
//   (x desc, id asc). Results go to the workspace.
// k_plan_heap, one CTA per tree: best-first expansion, popping N candidates. A candidate at
//   depth d holds the sum Sx of its path's logits (exact, in 64-bit fixed point) and the key
//   Sx - CL[d], CL[d] = LSE_1 + ... + LSE_d (its draft path log-probability). Pop order:
//   (key desc, depth asc, parent asc, rank asc), compared as integers. Popping (p, r) at depth d
//   pushes the next sibling (p, r+1) and, below the depth cap, the first child (i, 0).
//   Siblings are popped in rank order, so the children of u occupy
//   child_ids[child_off[u] + rank] directly.
//
// Both are latency-bound: the draft rows were streamed once by the statistics kernel and only
// the few candidate chunks per row are read again.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kTopkWarps = 4;
constexpr int kHeapThreads = 128;

struct TopkArgs {
    const void *draft;
    int64_t bstride, rstride;
    int B, R, V, C, L, K;
    const float2 *stats;
    float invT;
    float2 *lse;       // [B*L] row log-normalisers as float-float (hi, lo)
    float *topk_x;     // [B*L*K]
    int32_t *topk_id;  // [B*L*K]
};

template <int KCAP, typename T>
__global__ void __launch_bounds__(kTopkWarps * 32) k_row_topk(TopkArgs a) {
    extern __shared__ __align__(16) float2 st_all[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int row = blockIdx.x * kTopkWarps + warp;
    if (row >= a.B * a.L) return;  // warp-uniform; no block-wide barrier below
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const int C = a.C, K = a.K;
    float2 *st = st_all + (size_t)warp * C;
    const float2 *gst = a.stats + ((int64_t)b * a.R + d) * C;
    // stage the row's chunk statistics (eight independent loads in flight per lane)
    for (int c0 = lane; c0 < C; c0 += 32 * 8) {
        float2 v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int c = c0 + 32 * k;
            v[k] = c < C ? gst[c] : make_float2(-INFINITY, 0.f);
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int c = c0 + 32 * k;
            if (c < C) st[c] = v[k];
        }
    }
    __syncwarp();
    // log-normaliser (float-float; the lane partials merge in a butterfly)
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, st[c].x);
    KahanF acc;
    if (m != -INFINITY)
        for (int c = lane; c < C; c += 32) acc.add(__fmul_rn(st[c].y, expf(__fsub_rn(st[c].x, m))));
    const MaxSum tot = warp_maxsum(MaxSum{m, acc.ff()});
    if (lane == 0) {
        const FF l = maxsum_lse(tot);
        a.lse[row] = make_float2(l.hi, l.lo);
    }
    // tau = K-th largest chunk maximum (-inf with fewer than K chunks)
    float tau = -INFINITY;
    if (C >= K) {
        TopList<KCAP> cl;
        cl.clear();
        for (int c = lane; c < C; c += 32) cl.insert(pack_key(st[c].x, (uint32_t)c));
        uint64_t kth = 0;
        for (int j = 0; j < K; ++j) kth = warp_pop_max(cl);
        tau = key_value(kth);
    }
    // top-K logits among the chunks whose maximum reaches tau, four chunks per batch
    const T *rowp = static_cast<const T *>(a.draft) + (int64_t)b * a.bstride + (int64_t)d * a.rstride;
    TopList<KCAP> el;
    el.clear();
    for (int cb = 0; cb < C; cb += 32) {
        const int c = cb + lane;
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
                    if (xi >= tau) el.insert(pack_key(xi, (uint32_t)(v0 + i)));
                }
            }
        }
    }
    for (int j = 0; j < K; ++j) {
        const uint64_t best = warp_pop_max(el);
        if (lane == 0) {
            a.topk_id[(int64_t)row * K + j] = (int32_t)key_id(best);
            a.topk_x[(int64_t)row * K + j] = key_value(best);
        }
    }
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

template <int S>
struct Slots {
    unsigned long long k[S];
    unsigned w[S];
    unsigned long long bk;  // the lane's best
    unsigned bw;
    int bs;
    __device__ __forceinline__ void clear() {
#pragma unroll
        for (int s = 0; s < S; ++s) {
            k[s] = 0ull;
            w[s] = 0u;
        }
        bk = 0ull;
        bw = 0u;
        bs = 0;
    }
    __device__ __forceinline__ void put(int slot, unsigned long long kk, unsigned ww) {
#pragma unroll
        for (int s = 0; s < S; ++s)
            if (s == slot) {
                k[s] = kk;
                w[s] = ww;
            }
    }
    __device__ __forceinline__ void rescan() {
        bk = 0ull;
        bw = 0u;
        bs = 0;
#pragma unroll
        for (int s = 0; s < S; ++s)
            if (key_better(k[s], w[s], bk, bw)) {
                bk = k[s];
                bw = w[s];
                bs = s;
            }
    }
};

// Best-first expansion for one tree with one warp. Each pop: a three-stage warp maximum of
// the lanes' best keys (__reduce_max_sync on the high word, low word, tie word); the popped
// candidate's slot takes its next sibling; its first child goes to the next round-robin
// slot (children are numbered in creation order, lane = c % 32, slot = c / 32).
template <int S>
__global__ void __launch_bounds__(kHeapThreads) k_plan_heap(HeapArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int L = a.L, N = a.N, K = a.K, NN = N + 1;
    long long *CL = reinterpret_cast<long long *>(smem);           // [L+1] fixed point
    long long *n_sx = CL + (L + 1);                                // [NN] node path sums
    long long *fx = n_sx + NN;                                     // [L*K] candidate logits
    int32_t *n_parent = reinterpret_cast<int32_t *>(fx + L * K);   // [NN]
    int32_t *n_depth = n_parent + NN;
    int32_t *n_rank = n_depth + NN;
    int32_t *n_token = n_rank + NN;
    int32_t *n_count = n_token + NN;                               // [NN]
    float *n_score = reinterpret_cast<float *>(n_count + NN);      // [NN]
    int32_t *tk_id = reinterpret_cast<int32_t *>(n_score + NN);    // [L*K]

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
    if (warp == 0) {  // CL[d] = LSE_1 + ... + LSE_d in float-float, then onto the fixed grid
        FF l0 = FF{0.f, 0.f}, l1 = FF{0.f, 0.f};
        if (lane < L) {
            const float2 v = a.lse[(int64_t)b * L + lane];
            l0 = FF{v.x, v.y};
        }
        if (lane + 32 < L) {
            const float2 v = a.lse[(int64_t)b * L + lane + 32];
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
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) {
            n_parent[0] = -1;
            n_depth[0] = 0;
            n_rank[0] = -1;
            n_token[0] = -1;
        }
        Slots<S> fr;
        fr.clear();
        if (lane == 0) {  // the root's first child (depth 1, rank 0) is child number 0
            fr.put(0, okey_of(fx[0] - CL[1]), w3_of(1, 0, 0));
            fr.rescan();
        }
        int nchild = 1;
        __syncwarp();
        for (int i = 1; i <= N; ++i) {
            const unsigned hk = (unsigned)(fr.bk >> 32);
            const unsigned m1 = __reduce_max_sync(kFull, hk);
            unsigned c = __ballot_sync(kFull, hk == m1);
            if (__popc(c) > 1) {  // the high word ties: resolve with the low word, then w3
                const unsigned lk = (unsigned)fr.bk;
                const unsigned m2 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? lk : 0u);
                c &= __ballot_sync(kFull, lk == m2);
                if (__popc(c) > 1) {
                    const unsigned m3 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? fr.bw : 0u);
                    c &= __ballot_sync(kFull, fr.bw == m3);
                }
            }
            const int winner = __ffs(c) - 1;
            const unsigned long long wk = __shfl_sync(kFull, fr.bk, winner);
            const unsigned ww = __shfl_sync(kFull, fr.bw, winner);
            if (ww == 0u) {  // frontier exhausted: only with N above the tree's capacity
                if (lane == 0) raise_status(a.status, kDevBadTree);
                break;
            }
            const int depth = 255 - (int)(ww >> 24);
            const int parent = 65535 - (int)((ww >> 8) & 0xffffu);
            const int rank = 255 - (int)(ww & 0xffu);
            const bool sib = rank + 1 < K, kid = depth < L;
            // every lane computes the popped path's sum and both new keys from broadcast loads;
            // only the commits below differ per lane
            const long long sp = n_sx[parent];
            const long long sx = sp + fx[(depth - 1) * K + rank];
            const long long ks = sp + (sib ? fx[(depth - 1) * K + rank + 1] : 0) - CL[depth];
            const long long kc = sx + (kid ? fx[depth * K] : 0) - CL[kid ? depth + 1 : depth];
            if (lane == winner) {  // the next sibling takes the freed slot
                if (sib)
                    fr.put(fr.bs, okey_of(ks), w3_of(depth, parent, rank + 1));
                else
                    fr.put(fr.bs, 0ull, 0u);
                fr.rescan();
            }
            if (lane == 0) {
                n_parent[i] = parent;
                n_depth[i] = depth;
                n_rank[i] = rank;
                n_token[i] = tk_id[(depth - 1) * K + rank];
                n_score[i] = __fmul_rn(__ll2float_rn(key_of_okey(wk)), kFixInv);
                n_sx[i] = sx;
            }
            if (kid) {  // first child (i, 0), one level down, in the next round-robin slot
                if (lane == (nchild & 31)) {
                    const unsigned long long ck = okey_of(kc);
                    const unsigned cw = w3_of(depth + 1, i, 0);
                    fr.put(nchild >> 5, ck, cw);
                    if (key_better(ck, cw, fr.bk, fr.bw)) {
                        fr.bk = ck;
                        fr.bw = cw;
                        fr.bs = nchild >> 5;
                    }
                }
                ++nchild;
            }
            __syncwarp();
        }
    }
    __syncthreads();

    // child lists: count, exclusive scan (one warp), then place children by rank
    for (int i = 1 + threadIdx.x; i <= N; i += kHeapThreads) atomicAdd(&n_count[n_parent[i]], 1);
    __syncthreads();
    int32_t *off = a.tree.child_off + (int64_t)b * (NN + 1);
    if (warp == 0) {
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
    int32_t *ids = a.tree.child_ids + (int64_t)b * N;
    for (int i = 1 + threadIdx.x; i <= N; i += kHeapThreads) ids[n_count[n_parent[i]] + n_rank[i]] = i;
    int32_t *par = a.tree.parent + (int64_t)b * NN, *dep = a.tree.depth + (int64_t)b * NN;
    int32_t *rk = a.tree.rank + (int64_t)b * NN, *tok = a.tree.plan_token + (int64_t)b * NN;
    float *sc = a.tree.score + (int64_t)b * NN;
    for (int i = threadIdx.x; i < NN; i += kHeapThreads) {
        par[i] = n_parent[i];
        dep[i] = n_depth[i];
        rk[i] = n_rank[i];
        tok[i] = n_token[i];
        sc[i] = n_score[i];
    }
}

size_t heap_smem_bytes(int L, int N, int K) {
    const size_t NN = (size_t)N + 1;
    return (size_t)(L + 1) * 8 + NN * 8 + (size_t)L * K * 8 + 6 * NN * 4 + (size_t)L * K * 4;
}

template <int S>
cudaError_t launch_heap_t(const HeapArgs &h, int B, cudaStream_t s) {
    const size_t smem = heap_smem_bytes(h.L, h.N, h.K);
    cudaError_t e = cudaFuncSetAttribute(k_plan_heap<S>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_plan_heap<S><<<B, kHeapThreads, smem, s>>>(h);
    return cudaGetLastError();
}

template <int KCAP, typename T>
cudaError_t launch_topk_t(const TopkArgs &a, cudaStream_t s) {
    const size_t smem = (size_t)kTopkWarps * a.C * sizeof(float2);
    cudaError_t e = cudaFuncSetAttribute(k_row_topk<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int rows = a.B * a.L;
    k_row_topk<KCAP, T><<<(rows + kTopkWarps - 1) / kTopkWarps, kTopkWarps * 32, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

PlanScratch plan_scratch(void *ws, int B, int N, int L, int K) {
    unsigned char *p = static_cast<unsigned char *>(ws) + kWsStatusBytes + (size_t)B * (N + 1) * kWsBvRowBytes;
    PlanScratch s;
    s.lse = reinterpret_cast<float2 *>(p);
    s.topk_x = reinterpret_cast<float *>(p + (size_t)B * L * sizeof(float2));
    s.topk_id = reinterpret_cast<int32_t *>(p + (size_t)B * L * sizeof(float2) + (size_t)B * L * K * sizeof(float));
    return s;
}

cudaError_t launch_plan(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                        const TreeDesc &tree, void *ws, cudaStream_t s) {
    const PlanScratch sc = plan_scratch(ws, draft.B, N, L, K);
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
    t.invT = invT;
    t.lse = sc.lse;
    t.topk_x = sc.topk_x;
    t.topk_id = sc.topk_id;
    cudaError_t e;
    if (draft.dtype == 1)
        e = K <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = K <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    HeapArgs h;
    h.L = L;
    h.N = N;
    h.K = K;
    h.lse = sc.lse;
    h.topk_x = sc.topk_x;
    h.topk_id = sc.topk_id;
    h.tree = tree;
    h.status = static_cast<uint32_t *>(ws);
    // frontier slots per lane: at most N + 1 first children are ever created
    const int per_lane = (N + 1 + 31) / 32;
    if (per_lane <= 1) return launch_heap_t<1>(h, draft.B, s);
    if (per_lane <= 2) return launch_heap_t<2>(h, draft.B, s);
    if (per_lane <= 4) return launch_heap_t<4>(h, draft.B, s);
    if (per_lane <= 8) return launch_heap_t<8>(h, draft.B, s);
    if (per_lane <= 16) return launch_heap_t<16>(h, draft.B, s);
    return launch_heap_t<33>(h, draft.B, s);
}

}  // namespace tsb

namespace tsb {

// The same two launches as launch_plan, with the per-draft-row scratch and the status word
// given explicitly instead of being carved out of a caller workspace.
cudaError_t launch_plan_scratch(const RowsDesc &draft, const float2 *stats, int L, int N, int K, float invT,
                                const TreeDesc &tree, const PlanScratch &sc, uint32_t *status, cudaStream_t s) {
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
    t.invT = invT;
    t.lse = sc.lse;
    t.topk_x = sc.topk_x;
    t.topk_id = sc.topk_id;
    cudaError_t e;
    if (draft.dtype == 1)
        e = K <= 8 ? launch_topk_t<8, __nv_bfloat16>(t, s) : launch_topk_t<32, __nv_bfloat16>(t, s);
    else
        e = K <= 8 ? launch_topk_t<8, float>(t, s) : launch_topk_t<32, float>(t, s);
    if (e != cudaSuccess) return e;
    HeapArgs h;
    h.L = L;
    h.N = N;
    h.K = K;
    h.lse = sc.lse;
    h.topk_x = sc.topk_x;
    h.topk_id = sc.topk_id;
    h.tree = tree;
    h.status = status;
    const int per_lane = (N + 1 + 31) / 32;
    if (per_lane <= 1) return launch_heap_t<1>(h, draft.B, s);
    if (per_lane <= 2) return launch_heap_t<2>(h, draft.B, s);
    if (per_lane <= 4) return launch_heap_t<4>(h, draft.B, s);
    if (per_lane <= 8) return launch_heap_t<8>(h, draft.B, s);
    if (per_lane <= 16) return launch_heap_t<16>(h, draft.B, s);
    return launch_heap_t<33>(h, draft.B, s);
}

}  // namespace tsb
