// Block verification of a sampled chain X_1..X_g (Sun et al. 2025, the chain baseline the
// paper compares against in Sec. 1, Table 2 and App. A). With Mb_i = target law after the
// prefix X^i (target row i) and Ms_i = draft law of the next token (q row of node i):
//   w_0 = 1, w_i = min(w_{i-1} Mb_{i-1}(X_i) / Ms_{i-1}(X_i), 1)
//   h_i = S_i / (S_i + 1 - w_i), S_i = sum_x max(w_i Mb_i(x) - Ms_i(x), 0)   (i < g; 1 if 0/0)
//   h_g = w_g,  tau = max{ i >= 1 : eta_i <= h_i } (0 if none)
//   final token ~ Mb_g if tau = g, else ~ max(w_tau Mb_tau - Ms_tau, 0).
//
// Every quantity that needs a full row is computed for every chain position at once, so the
// only serial work is a product of g point-value ratios:
//   k_bv_rows   one CTA per (tree, position i <= g), streaming target row i once: its chunk
//               log-masses give the row's log-normaliser and, with Gumbel keys, the chunk of
//               the draw from Mb_i; one warp re-reads that chunk (from L2) for the token. The
//               log-normaliser of q row i comes from its chunk statistics.
//   k_bv_resid  one CTA per (tree, i < g): w_i from the point values Mb_j(X_{j+1}),
//               Ms_j(X_{j+1}) (one thread per j, then a serial product), then target row i
//               and q row i streamed once for S_i and the chunk masses of the residual, whose
//               Gumbel keys pick the chunk of the draw from the residual; one warp re-reads it.
//   k_bv_final  one warp per tree: the weights again, h_i, tau, and the final token chosen
//               among the draws the first two kernels made at position tau.
// Both draws at a position are the two-level Gumbel-max of every final token (purposes final
// chunk and final, node = position), so precomputing them changes no outcome. Rows are read
// in units of U chunks per warp, all U loads issued before any arithmetic.
// Per-(tree, position) results live in the caller's workspace after the status word.
#include <cooperative_groups.h>

#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

namespace cg = cooperative_groups;

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kSplit = 4;  // CTAs (one cluster) per row of the row kernels
constexpr int kMaxChain = 64;  // g <= L <= 64

template <typename T>
struct BvUnit {  // chunks per warp iteration: 8 (bf16) or 4 (fp32) 16-byte loads per row per lane
    static constexpr int n = sizeof(T) == 2 ? 8 : 4;
};

// Per-(tree, position) results, one 32-byte workspace slot each.
struct BvSlot {
    float lt_hi, lt_lo;  // log-normaliser of target row i (float-float)
    float lq_hi, lq_lo;  // log-normaliser of q row i (i < g)
    float s_hi, s_lo;    // S_i (i < g)
    int32_t y_t;         // draw from Mb_i
    int32_t y_r;         // draw from the residual at i (i < g; -1 if it has no mass)
};
static_assert(sizeof(BvSlot) == kWsBvRowBytes, "block-verification slot size");

struct BvArgs {
    const void *target;
    int64_t t_bstride, t_rstride;
    const void *q;
    int64_t q_bstride, q_rstride;
    int q_R;
    const float2 *qstats;
    int C;
    const int32_t *qrow_of_node, *depth, *child_off, *child_ids, *token;
    int V, N, L;
    float invT;
    uint64_t seed;
    int32_t *out_tokens, *out_nodes, *out_len;
    uint32_t *status;
    BvSlot *slots;  // [B, N+1]
};

struct BlockRed {
    MaxSum ms[kWarps];
    FF ff[kWarps];
    unsigned long long k[kWarps];
    MaxSum MS;
    FF S;
    unsigned long long K;
};

// Softmax normaliser over the block (float-float); valid in every thread afterwards.
__device__ MaxSum block_maxsum(BlockRed &sh, MaxSum v) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_maxsum(v);
    if (lane == 0) sh.ms[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const MaxSum w = warp_maxsum(lane < kWarps ? sh.ms[lane] : MaxSum{-INFINITY, FF{0.f, 0.f}});
        if (lane == 0) sh.MS = w;
    }
    __syncthreads();
    const MaxSum r = sh.MS;
    __syncthreads();
    return r;
}

__device__ FF block_sum(BlockRed &sh, FF v) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum_ff(v);
    if (lane == 0) sh.ff[warp] = v;
    __syncthreads();
    if (warp == 0) {
        const FF w = warp_sum_ff(lane < kWarps ? sh.ff[lane] : FF{0.f, 0.f});
        if (lane == 0) sh.S = w;
    }
    __syncthreads();
    const FF r = sh.S;
    __syncthreads();
    return r;
}

__device__ unsigned long long block_argmax(BlockRed &sh, unsigned long long k) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned long long t = warp_max_u64(k);
    if (lane == 0) sh.k[warp] = t;
    __syncthreads();
    if (warp == 0) {
        const unsigned long long tt = warp_max_u64(lane < kWarps ? sh.k[lane] : 0ull);
        if (lane == 0) sh.K = tt;
    }
    __syncthreads();
    const unsigned long long r = sh.K;
    __syncthreads();
    return r;
}

// log of a normaliser as float-float; -inf when it has no mass
__device__ __forceinline__ FF lse_ff(MaxSum v) {
    if (!(v.s.hi > 0.f)) return FF{-INFINITY, 0.f};
    return maxsum_lse(v);
}

// exp(z * invT - (hi + lo))
__device__ __forceinline__ float prob_of(float z, float invT, float hi, float lo) {
    return expf(__fsub_rn(__fsub_rn(__fmul_rn(z, invT), hi), lo));
}

__device__ __forceinline__ int qrow_index(const BvArgs &a, int b, int node) {
    const int64_t idx = (int64_t)b * (a.N + 1) + node;
    return a.qrow_of_node ? a.qrow_of_node[idx] : a.depth[idx];
}

template <typename T>
__device__ __forceinline__ const T *trow_ptr(const BvArgs &a, int b, int i) {
    return static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)i * a.t_rstride;
}
template <typename T>
__device__ __forceinline__ const T *qrow_ptr(const BvArgs &a, int b, int r) {
    return static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;
}

// Mb_j(X_{j+1}) and Ms_j(X_{j+1}) from the point logits and the rows' log-normalisers; false
// when the token or the q row index is out of range.
template <typename T>
__device__ bool point_values(const BvArgs &a, int b, int j, float *p, float *q) {
    const int NN = a.N + 1;
    const int X = a.token[(int64_t)b * NN + j + 1];
    const int r = qrow_index(a, b, j);
    if (X < 0 || X >= a.V || r < 0 || r >= a.q_R) return false;
    const BvSlot &s = a.slots[(int64_t)b * NN + j];
    *p = prob_of(Logit<T>::load1(trow_ptr<T>(a, b, j), X), a.invT, s.lt_hi, s.lt_lo);
    *q = prob_of(Logit<T>::load1(qrow_ptr<T>(a, b, r), X), a.invT, s.lq_hi, s.lq_lo);
    return true;
}

// w_j = min(w_{j-1} p / q, 1) (a zero draft probability cannot have been sampled: ratio 1)
__device__ __forceinline__ float weight_step(float w, float p, float q) {
    const float ratio = q > 0.f ? __fdiv_rn(__fmul_rn(w, p), q) : 1.0f;
    return fminf(ratio, 1.0f);
}

// Chunk range of CTA `rank` of a row's cluster, in units of U chunks.
struct ChunkRange {
    int lo, hi, units;
};
template <int U>
__device__ __forceinline__ ChunkRange chunk_range(int C, int rank) {
    const int per = (C + kSplit - 1) / kSplit;
    const int lo = rank * per, hi = min(C, lo + per);
    return ChunkRange{lo, hi, hi > lo ? (hi - lo + U - 1) / U : 0};
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 8) k_bv_rows(BvArgs a) {
    pdl_begin();
    constexpr int U = BvUnit<T>::n;
    __shared__ BlockRed sh;
    __shared__ MaxSum s_ms;                 // this CTA's partial normaliser
    __shared__ unsigned long long s_key;    // this CTA's best chunk key
    __shared__ MaxSum s_tot;                // CTA 0: the row's normaliser
    __shared__ unsigned long long s_cb;     // CTA 0: the chosen chunk
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = a.N, NN = a.N + 1;
    const int rid = blockIdx.x / kSplit;
    const int b = rid / NN, i = rid - b * NN;
    // the topology must be the chain 0 -> 1 -> ... -> g
    if (rank == 0 && threadIdx.x == 0) {
        const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
        const int want = i < g ? 1 : 0;
        if (off[i + 1] - off[i] != want ||
            (want && (off[i] < 0 || off[i] >= a.N || a.child_ids[(int64_t)b * a.N + off[i]] != i + 1)))
            raise_status(a.status, kDevBadTree);
    }
    const T *row = trow_ptr<T>(a, b, i);
    const uint32_t ub = (uint32_t)b, un = (uint32_t)i;
    const ChunkRange cr = chunk_range<U>(a.C, rank);
    MaxSum acc{-INFINITY, FF{0.f, 0.f}};  // normaliser of the chunks this lane keeps
    unsigned long long best = 0ull;       // best chunk key for the draw from Mb_i
    bool bad = false;
    for (int un0 = warp; un0 < cr.units; un0 += kWarps) {  // uniform over the warp
        const int cu = cr.lo + un0 * U;
        RawGroup<T> raw[U];
#pragma unroll
        for (int k = 0; k < U; ++k)
            if (cu + k < cr.hi) raw[k].load(row, (cu + k) * kChunk + lane * 8, a.V);
        float mcs[U], part[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            mcs[k] = -INFINITY;
            part[k] = 0.f;
            if (cu + k >= cr.hi) continue;  // uniform over the warp
            float z[8];
            raw[k].unpack(z);  // padding past V is -inf
            float zm = z[0];
#pragma unroll
            for (int e = 1; e < 8; ++e) zm = fmaxf(zm, z[e]);
            mcs[k] = __fmul_rn(warp_max(zm), a.invT);
            const float2 offs = exp_offset(mcs[k]);
#pragma unroll
            for (int e = 0; e < 8; ++e) part[k] += chunk_term(z[e], a.invT, offs.x);
            part[k] = chunk_sum_fix(part[k], offs.y);
        }
        // the U chunk sums at once; the lane holding a chunk's sum merges and keys that chunk
        const float sm = warp_multi_sum<U>(part);
        const int ch = multi_sum_index<U>(lane), c = cu + ch;
        if (lane % (32 / U) == 0 && c < cr.hi) {
            float mc = mcs[0];
#pragma unroll
            for (int k = 1; k < U; ++k) mc = ch == k ? mcs[k] : mc;
            bad |= !(sm == sm) || isinf(mc);
            acc = maxsum_merge(acc, MaxSum{mc, FF{sm, 0.f}});
            const uint32_t w = draw_word(a.seed, kFinalChunk, ub, un, (uint32_t)c);
            const float A = __fadd_rn(mc, logf(sm));
            const unsigned long long k = pack_key(__fadd_rn(A, gumbel_of(w)), (uint32_t)c);
            best = k > best ? k : best;
        }
    }
    if (__any_sync(kFull, bad) && lane == 0) raise_status(a.status, kDevNonFinite);
    {
        const MaxSum part_ms = block_maxsum(sh, acc);
        const unsigned long long part_key = block_argmax(sh, best);
        if (threadIdx.x == 0) {
            s_ms = part_ms;
            s_key = part_key;
        }
    }
    cluster.sync();  // every CTA's partial is published
    if (rank == 0 && warp == 0) {
        MaxSum v = lane < kSplit ? *cluster.map_shared_rank(&s_ms, lane) : MaxSum{-INFINITY, FF{0.f, 0.f}};
        v = warp_maxsum(v);
        const unsigned long long k = warp_max_u64(lane < kSplit ? *cluster.map_shared_rank(&s_key, lane) : 0ull);
        if (lane == 0) {
            s_tot = v;
            s_cb = k;
        }
    }
    cluster.sync();  // CTA 0 has read the others; they may leave
    if (rank != 0) return;
    const MaxSum tot = s_tot;
    const unsigned long long cb = s_cb;
    int y_t = -1;
    if (warp == 0 && cb != 0ull) {  // the token inside the chosen chunk (re-read from L2)
        const int v0 = (int)key_id(cb) * kChunk + lane * 8;
        float x[8];
        Logit<T>::load8(row, v0, a.V, x);
        const Words4 w0 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2) + 1u);
        unsigned long long tk = 0ull;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (v0 + e < a.V) {
                const uint32_t wi = e < 4 ? w0.w[e] : w1.w[e - 4];
                const float key = __fadd_rn(__fmul_rn(x[e], a.invT), gumbel_of(wi));
                const unsigned long long k = pack_key(key, (uint32_t)(v0 + e));
                tk = k > tk ? k : tk;
            }
        }
        tk = warp_max_u64(tk);
        y_t = tk != 0ull ? (int)key_id(tk) : -1;
    }
    // log-normaliser of q row i from its chunk statistics
    FF lq = FF{0.f, 0.f};
    if (i < g) {  // uniform over the CTA
        const int r = qrow_index(a, b, i);
        float mq = -INFINITY;
        KahanF sq;
        if (r >= 0 && r < a.q_R) {
            const float2 *st = a.qstats + ((int64_t)b * a.q_R + r) * a.C;
            for (int c = threadIdx.x; c < a.C; c += kThreads) mq = fmaxf(mq, st[c].x);
            if (mq != -INFINITY)
                for (int c = threadIdx.x; c < a.C; c += kThreads)
                    sq.add(__fmul_rn(st[c].y, expf(__fsub_rn(st[c].x, mq))));
        } else if (threadIdx.x == 0) {
            raise_status(a.status, kDevBadIndex);
        }
        lq = lse_ff(block_maxsum(sh, MaxSum{mq, sq.ff()}));
    }
    if (threadIdx.x == 0) {
        BvSlot &o = a.slots[(int64_t)b * NN + i];
        const FF lt = lse_ff(tot);
        o.lt_hi = lt.hi;
        o.lt_lo = lt.lo;
        o.lq_hi = lq.hi;
        o.lq_lo = lq.lo;
        o.y_t = y_t;
        if (i == g) {  // no residual at the last position
            o.s_hi = 0.f;
            o.s_lo = 0.f;
            o.y_r = -1;
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 8) k_bv_resid(BvArgs a) {
    pdl_begin();
    constexpr int U = BvUnit<T>::n / 2;  // two rows per chunk
    __shared__ BlockRed sh;
    __shared__ float pj[kMaxChain], qj[kMaxChain];
    __shared__ float w_sh;
    __shared__ int bad_sh;
    __shared__ FF s_S;                      // this CTA's partial residual mass
    __shared__ unsigned long long s_key;    // this CTA's best chunk key
    __shared__ FF s_tot;                    // CTA 0: S_i
    __shared__ unsigned long long s_cb;     // CTA 0: the chosen chunk
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = a.N, NN = g + 1;
    const int rid = blockIdx.x / kSplit;
    const int b = rid / g, i = rid - b * g;
    if (threadIdx.x == 0) bad_sh = 0;
    __syncthreads();
    // 1. w_i: the point values of positions 0..i-1 (one thread each), then their product (every
    //    CTA of the cluster computes the same value from the same inputs)
    for (int j = threadIdx.x; j < i; j += kThreads)
        if (!point_values<T>(a, b, j, &pj[j], &qj[j])) atomicOr(&bad_sh, 1);
    const int r = qrow_index(a, b, i);
    if (threadIdx.x == 0 && (r < 0 || r >= a.q_R)) atomicOr(&bad_sh, 1);
    __syncthreads();
    const bool bad = bad_sh != 0;  // uniform over the cluster: no row is read, but every barrier is met
    if (threadIdx.x == 0) {
        if (bad && rank == 0) raise_status(a.status, kDevBadIndex);
        float w = 1.0f;
        if (!bad)
            for (int j = 0; j < i; ++j) w = weight_step(w, pj[j], qj[j]);
        w_sh = w;
    }
    __syncthreads();
    const float w = w_sh;
    const BvSlot &sl = a.slots[(int64_t)b * NN + i];
    const float th = sl.lt_hi, tl = sl.lt_lo, qh = sl.lq_hi, ql = sl.lq_lo;
    const FF L2t = ff_times_log2e(FF{th, tl}), L2q = ff_times_log2e(FF{qh, ql});  // for exp_shifted
    const T *trow = trow_ptr<T>(a, b, i);
    const T *qrow = qrow_ptr<T>(a, b, bad ? 0 : r);
    const uint32_t ub = (uint32_t)b, un = (uint32_t)i;
    // 2. S_i and the residual's chunk masses, target and q rows streamed together
    const ChunkRange cr = chunk_range<U>(a.C, rank);
    KahanF acc;
    unsigned long long best = 0ull;
    for (int un0 = warp; !bad && un0 < cr.units; un0 += kWarps) {  // uniform over the warp
        const int cu = cr.lo + un0 * U;
        RawGroup<T> rt[U], rq[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            if (cu + k < cr.hi) {
                rt[k].load(trow, (cu + k) * kChunk + lane * 8, a.V);
                rq[k].load(qrow, (cu + k) * kChunk + lane * 8, a.V);
            }
        }
        float part[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            part[k] = 0.f;
            if (cu + k >= cr.hi) continue;  // uniform over the warp
            float zt[8], zq[8];
            rt[k].unpack(zt);  // padding past V is -inf: probability 0
            rq[k].unpack(zq);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float p = exp_shifted(__fmul_rn(zt[e], a.invT), L2t);
                const float q = exp_shifted(__fmul_rn(zq[e], a.invT), L2q);
                part[k] += fmaxf(__fsub_rn(__fmul_rn(w, p), q), 0.f);
            }
        }
        // the U chunk masses at once; the lane holding a chunk's mass adds and keys it
        const float mass = warp_multi_sum<U>(part);
        const int ch = multi_sum_index<U>(lane), c = cu + ch;
        if (lane % (32 / U) == 0 && c < cr.hi) {
            acc.add(mass);
            if (mass > 0.f) {
                const uint32_t wd = draw_word(a.seed, kFinalChunk, ub, un, (uint32_t)c);
                const unsigned long long k = pack_key(__fadd_rn(logf(mass), gumbel_of(wd)), (uint32_t)c);
                best = k > best ? k : best;
            }
        }
    }
    {
        const FF part_S = block_sum(sh, acc.ff());
        const unsigned long long part_key = block_argmax(sh, best);
        if (threadIdx.x == 0) {
            s_S = part_S;
            s_key = part_key;
        }
    }
    cluster.sync();  // every CTA's partial is published
    if (rank == 0 && warp == 0) {
        const FF v = warp_sum_ff(lane < kSplit ? *cluster.map_shared_rank(&s_S, lane) : FF{0.f, 0.f});
        const unsigned long long k = warp_max_u64(lane < kSplit ? *cluster.map_shared_rank(&s_key, lane) : 0ull);
        if (lane == 0) {
            s_tot = v;
            s_cb = k;
        }
    }
    cluster.sync();  // CTA 0 has read the others; they may leave
    if (rank != 0 || warp != 0 || bad) return;
    const FF S = s_tot;
    const unsigned long long cb = s_cb;
    // 3. the token of the residual draw inside the chosen chunk (re-read from L2)
    int y = -1;
    if (cb != 0ull) {
        const int v0 = (int)key_id(cb) * kChunk + lane * 8;
        float xt[8], xq[8];
        Logit<T>::load8(trow, v0, a.V, xt);
        Logit<T>::load8(qrow, v0, a.V, xq);
        const Words4 w0 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2) + 1u);
        unsigned long long tk = 0ull;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (v0 + e >= a.V) continue;
            const float p = exp_shifted(__fmul_rn(xt[e], a.invT), L2t);
            const float q = exp_shifted(__fmul_rn(xq[e], a.invT), L2q);
            const float rv = fmaxf(__fsub_rn(__fmul_rn(w, p), q), 0.f);
            if (!(rv > 0.f)) continue;
            const uint32_t wi = e < 4 ? w0.w[e] : w1.w[e - 4];
            const unsigned long long k = pack_key(__fadd_rn(logf(rv), gumbel_of(wi)), (uint32_t)(v0 + e));
            tk = k > tk ? k : tk;
        }
        tk = warp_max_u64(tk);
        y = tk != 0ull ? (int)key_id(tk) : -1;
    }
    if (lane == 0) {
        BvSlot &o = a.slots[(int64_t)b * NN + i];
        o.s_hi = S.hi;
        o.s_lo = S.lo;
        o.y_r = y;
    }
}

// One warp per tree: weights, h_i, tau, and the outputs.
template <typename T>
__global__ void __launch_bounds__(32) k_bv_final(BvArgs a) {
    pdl_begin();
    __shared__ float pj[kMaxChain], qj[kMaxChain], eta_s[kMaxChain + 1];
    __shared__ FF S_s[kMaxChain + 1];
    const int lane = threadIdx.x;
    const int g = a.N, NN = g + 1;
    const int b = blockIdx.x;
    const BvSlot *sl = a.slots + (int64_t)b * NN;
    bool ok = true;
    for (int j = lane; j < g; j += 32) ok &= point_values<T>(a, b, j, &pj[j], &qj[j]);
    for (int i = 1 + lane; i <= g; i += 32) {  // every lane's loads and draws in parallel
        S_s[i] = FF{sl[i].s_hi, sl[i].s_lo};
        eta_s[i] = uniform_of(draw_word(a.seed, kBlockEta, (uint32_t)b, (uint32_t)i, 0u));
    }
    ok = __all_sync(kFull, ok);
    __syncwarp();
    if (lane != 0) return;
    int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
    int32_t *onode = a.out_nodes + (int64_t)b * a.L;
    for (int k = 0; k <= a.L; ++k) otok[k] = -1;
    for (int k = 0; k < a.L; ++k) onode[k] = -1;
    if (!ok) {
        raise_status(a.status, kDevBadIndex);
        a.out_len[b] = 0;
        return;
    }
    float w = 1.0f;
    int tau = 0;
    for (int i = 1; i <= g; ++i) {
        w = weight_step(w, pj[i - 1], qj[i - 1]);  // w_i
        float h;  // in fp32 (GB300's fp64 units are too slow even for this serial loop)
        if (i < g) {
            const float den = __fadd_rn(__fadd_rn(S_s[i].hi, __fsub_rn(1.0f, w)), S_s[i].lo);
            h = den > 0.f ? __fdiv_rn(__fadd_rn(S_s[i].hi, S_s[i].lo), den) : 1.0f;
        } else {
            h = w;
        }
        if (eta_s[i] <= h) tau = i;
    }
    // the final token: from Mb_g at tau = g, else from the residual at tau (from Mb_tau when
    // the residual carries no mass, which exact arithmetic rules out)
    int y;
    if (tau == g) {
        y = sl[g].y_t;
    } else {
        const bool mass = __fadd_rn(sl[tau].s_hi, sl[tau].s_lo) > 0.f && sl[tau].y_r >= 0;
        y = mass ? sl[tau].y_r : sl[tau].y_t;
    }
    for (int i = 1; i <= tau; ++i) {
        otok[i - 1] = a.token[(int64_t)b * NN + i];
        onode[i - 1] = i;
    }
    otok[tau] = y;
    a.out_len[b] = tau + 1;
}

template <typename T>
cudaError_t launch_bv_t(const BvArgs &a, int B, cudaStream_t s) {
    const int NN = a.N + 1;
    cudaError_t e = launch_pdl(k_bv_rows<T>, dim3((unsigned)(B * NN * kSplit)), dim3(kThreads), 0, s, kSplit, a);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_bv_resid<T>, dim3((unsigned)(B * a.N * kSplit)), dim3(kThreads), 0, s, kSplit, a);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_bv_final<T>, dim3((unsigned)B), dim3(32), 0, s, 0, a);
}

}  // namespace

cudaError_t launch_verify_block(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                                const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    BvArgs a;
    a.target = target.data;
    a.t_bstride = target.batch_stride;
    a.t_rstride = target.row_stride;
    a.q = q.data;
    a.q_bstride = q.batch_stride;
    a.q_rstride = q.row_stride;
    a.q_R = q.R;
    a.qstats = qstats;
    a.C = num_chunks(q.V);
    a.qrow_of_node = qrow_of_node;
    a.depth = tree.depth;
    a.child_off = tree.child_off;
    a.child_ids = tree.child_ids;
    a.token = token;
    a.V = target.V;
    a.N = N;
    a.L = L;
    a.invT = invT;
    a.seed = seed;
    a.out_tokens = out_tokens;
    a.out_nodes = out_nodes;
    a.out_len = out_len;
    a.status = status;
    a.slots = reinterpret_cast<BvSlot *>(reinterpret_cast<unsigned char *>(status) + kWsStatusBytes);
    if (target.dtype == 1) return launch_bv_t<__nv_bfloat16>(a, B, s);
    return launch_bv_t<float>(a, B, s);
}

}  // namespace tsb
