// First pass (Sec. 3.1; max-heap expansion as in DDTree, Sec. 2.2 / App. B.3), two kernels.
//
// k_row_topk, one warp per draft row (every row of the batch in parallel): the row's chunk
//   statistics are staged in shared memory, merged into the log-normaliser LSE_d, and give
//   tau = the K-th largest chunk maximum, a lower bound on the K-th largest logit (K distinct
//   chunk maxima reach it). Only chunks whose maximum reaches tau are re-read; their logits
//   >= tau go through per-lane sorted lists, and a warp merge yields the top-K by
//   (x desc, id asc). Results go to the workspace.
// k_plan_heap, one CTA per tree: best-first expansion, popping N candidates. A candidate at
//   depth d holds the exact fp64 sum Sx of its path's logits and the key Sx - CL[d],
//   CL[d] = LSE_1 + ... + LSE_d (its draft path log-probability). Pop order: (key desc,
//   depth asc, Sx desc, parent asc, rank asc). Popping (p, r) at depth d pushes the next
//   sibling (p, r+1) and, below the depth cap, the first child (i, 0). Siblings are popped in
//   rank order, so the children of u occupy child_ids[child_off[u] + rank] directly.
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
    double *lse;       // [B*L]
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
    // log-normaliser
    float m = -INFINITY;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, st[c].x);
    m = warp_max(m);
    KahanF acc;
    for (int c = lane; c < C; c += 32) acc.add(st[c].y * expf(st[c].x - m));
    const double S = warp_sum_d(acc.value());
    if (lane == 0) a.lse[row] = (double)m + log(S);
    // tau = K-th largest chunk maximum (-inf with fewer than K chunks)
    float tau = -INFINITY;
    if (C >= K) {
        TopList<KCAP> cl;
        cl.clear();
        for (int c = lane; c < C; c += 32) cl.insert(pack_key(st[c].x, (uint32_t)c));
        uint64_t kth = 0;
        for (int j = 0; j < K; ++j) {
            const uint64_t best = warp_max_u64(cl.k[0]);
            kth = best;
            if (cl.k[0] == best) cl.pop_front();
        }
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
        const uint64_t best = warp_max_u64(el.k[0]);
        if (lane == 0) {
            a.topk_id[(int64_t)row * K + j] = (int32_t)key_id(best);
            a.topk_x[(int64_t)row * K + j] = key_value(best);
        }
        if (el.k[0] == best) el.pop_front();
    }
}

struct HeapArgs {
    int L, N, K;
    const double *lse;
    const float *topk_x;
    const int32_t *topk_id;
    TreeDesc tree;
    uint32_t *status;
};

struct Cand {
    double key, sx;
    int meta;  // parent << 16 | depth << 8 | rank
};

__device__ __forceinline__ int meta_parent(int m) { return m >> 16; }
__device__ __forceinline__ int meta_depth(int m) { return (m >> 8) & 0xff; }
__device__ __forceinline__ int meta_rank(int m) { return m & 0xff; }

// Does a pop before b?
__device__ __forceinline__ bool cand_before(const Cand &a, const Cand &b) {
    if (a.key != b.key) return a.key > b.key;
    const int da = meta_depth(a.meta), db = meta_depth(b.meta);
    if (da != db) return da < db;
    if (a.sx != b.sx) return a.sx > b.sx;
    const int pa = meta_parent(a.meta), pb = meta_parent(b.meta);
    if (pa != pb) return pa < pb;
    return meta_rank(a.meta) < meta_rank(b.meta);
}

__global__ void __launch_bounds__(kHeapThreads) k_plan_heap(HeapArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int L = a.L, N = a.N, K = a.K, NN = N + 1;
    double *CL = reinterpret_cast<double *>(smem);   // [L+1]
    double *f_key = CL + (L + 1);                    // [NN] frontier
    double *f_sx = f_key + NN;                       // [NN]
    double *n_sx = f_sx + NN;                        // [NN] node path sums
    int32_t *f_meta = reinterpret_cast<int32_t *>(n_sx + NN);  // [NN]
    int32_t *n_parent = f_meta + NN;                 // [NN]
    int32_t *n_depth = n_parent + NN;
    int32_t *n_rank = n_depth + NN;
    int32_t *n_token = n_rank + NN;
    int32_t *n_count = n_token + NN;                 // [NN]
    float *n_score = reinterpret_cast<float *>(n_count + NN);  // [NN]
    int32_t *tk_id = reinterpret_cast<int32_t *>(n_score + NN);  // [L*K]
    float *tk_x = reinterpret_cast<float *>(tk_id + L * K);      // [L*K]

    const int b = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < L * K; i += kHeapThreads) {
        tk_id[i] = a.topk_id[(int64_t)b * L * K + i];
        tk_x[i] = a.topk_x[(int64_t)b * L * K + i];
    }
    for (int i = threadIdx.x; i < NN; i += kHeapThreads) {  // defined even if the expansion stops early
        n_count[i] = 0;
        n_parent[i] = 0;
        n_depth[i] = 0;
        n_rank[i] = 0;
        n_token[i] = -1;
        n_score[i] = 0.f;
    }
    if (threadIdx.x == 0) {
        CL[0] = 0.0;
        for (int d = 1; d <= L; ++d) CL[d] = CL[d - 1] + a.lse[(int64_t)b * L + d - 1];
    }
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) {
            n_parent[0] = -1;
            n_depth[0] = 0;
            n_rank[0] = -1;
            n_token[0] = -1;
            n_score[0] = 0.f;
            n_sx[0] = 0.0;
            f_sx[0] = (double)tk_x[0];
            f_key[0] = f_sx[0] - CL[1];
            f_meta[0] = (0 << 16) | (1 << 8) | 0;
        }
        int nf = 1;
        __syncwarp();
        for (int i = 1; i <= N; ++i) {
            Cand best{-INFINITY, 0.0, 0};
            int bi = -1;
            for (int f = lane; f < nf; f += 32) {
                Cand c{f_key[f], f_sx[f], f_meta[f]};
                if (bi < 0 || cand_before(c, best)) {
                    best = c;
                    bi = f;
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                Cand other;
                other.key = __shfl_xor_sync(kFull, best.key, o);
                other.sx = __shfl_xor_sync(kFull, best.sx, o);
                other.meta = __shfl_xor_sync(kFull, best.meta, o);
                const int oi = __shfl_xor_sync(kFull, bi, o);
                if (oi >= 0 && (bi < 0 || cand_before(other, best))) {
                    best = other;
                    bi = oi;
                }
            }
            if (bi < 0) {  // frontier exhausted: only with N above the tree's capacity
                if (lane == 0) raise_status(a.status, kDevBadTree);
                break;
            }
            const int parent = meta_parent(best.meta), depth = meta_depth(best.meta), rank = meta_rank(best.meta);
            if (lane == 0) {
                n_parent[i] = parent;
                n_depth[i] = depth;
                n_rank[i] = rank;
                n_token[i] = tk_id[(depth - 1) * K + rank];
                n_score[i] = (float)best.key;
                n_sx[i] = best.sx;
                // remove the popped entry, then push its next sibling and first child
                const int last = nf - 1;
                f_key[bi] = f_key[last];
                f_sx[bi] = f_sx[last];
                f_meta[bi] = f_meta[last];
                int nn = last;
                if (rank + 1 < K) {
                    const double sx = n_sx[parent] + (double)tk_x[(depth - 1) * K + rank + 1];
                    f_sx[nn] = sx;
                    f_key[nn] = sx - CL[depth];
                    f_meta[nn] = (parent << 16) | (depth << 8) | (rank + 1);
                    ++nn;
                }
                if (depth < L) {
                    const double sx = best.sx + (double)tk_x[depth * K + 0];
                    f_sx[nn] = sx;
                    f_key[nn] = sx - CL[depth + 1];
                    f_meta[nn] = (i << 16) | ((depth + 1) << 8) | 0;
                    ++nn;
                }
                nf = nn;
            }
            nf = __shfl_sync(kFull, nf, 0);
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
    return (size_t)(L + 1) * 8 + 3 * NN * 8 + 7 * NN * 4 + 2 * (size_t)L * K * 4;
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
    s.lse = reinterpret_cast<double *>(p);
    s.topk_x = reinterpret_cast<float *>(p + (size_t)B * L * sizeof(double));
    s.topk_id = reinterpret_cast<int32_t *>(p + (size_t)B * L * sizeof(double) + (size_t)B * L * K * sizeof(float));
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
    const size_t smem = heap_smem_bytes(L, N, K);
    e = cudaFuncSetAttribute(k_plan_heap, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_plan_heap<<<draft.B, kHeapThreads, smem, s>>>(h);
    return cudaGetLastError();
}

}  // namespace tsb
