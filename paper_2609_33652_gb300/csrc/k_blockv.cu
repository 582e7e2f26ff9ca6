// Block verification of a sampled chain X_1..X_g (Sun et al. 2025, the chain baseline the
// paper compares against in Sec. 1, Table 2 and App. A). With Mb_i = target law after the
// prefix X^i (target row i) and Ms_i = draft law of the next token (q row of node i):
//   w_0 = 1, w_i = min(w_{i-1} Mb_{i-1}(X_i) / Ms_{i-1}(X_i), 1)
//   h_i = S_i / (S_i + 1 - w_i), S_i = sum_x max(w_i Mb_i(x) - Ms_i(x), 0)   (i < g; 1 if 0/0)
//   h_g = w_g,  tau = max{ i >= 1 : eta_i <= h_i } (0 if none)
//   final token ~ Mb_g if tau = g, else ~ max(w_tau Mb_tau - Ms_tau, 0).
//
// Three launches, each parallel over rows (no serial dependency between chain positions):
//   k_bv_rows   one CTA per (tree, position i <= g): log-normaliser of target row i and of
//               q row i (from its chunk statistics);
//   k_bv_resid  one CTA per (tree, i < g): w_i from point values, then S_i over the full row;
//   k_bv_final  one CTA per tree: tau, then the Gumbel-max final token over one row.
// Per-(tree, position) scalars live in the caller's workspace after the status word.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;

struct BvRow {
    double lse_t, lse_q, S, w;
};

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
    BvRow *rows;  // [B, N+1]
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

__device__ __forceinline__ double lse_of(MaxSum v) {
    if (!(v.s.hi > 0.f)) return -INFINITY;
    const FF l = maxsum_lse(v);
    return (double)l.hi + (double)l.lo;
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

__device__ __forceinline__ void split(double v, float &hi, float &lo) {
    hi = (float)v;
    lo = (float)(v - (double)hi);
}
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

template <typename T>
__global__ void __launch_bounds__(kThreads) k_bv_rows(BvArgs a) {
    pdl_begin();
    __shared__ BlockRed sh;
    const int g = a.N, NN = a.N + 1;
    const int b = blockIdx.x / NN, i = blockIdx.x - b * NN;
    // the topology must be the chain 0 -> 1 -> ... -> g
    if (threadIdx.x == 0) {
        const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
        const int want = i < g ? 1 : 0;
        if (off[i + 1] - off[i] != want ||
            (want && (off[i] < 0 || off[i] >= a.N || a.child_ids[(int64_t)b * a.N + off[i]] != i + 1)))
            raise_status(a.status, kDevBadTree);
    }
    const T *row = trow_ptr<T>(a, b, i);
    float x[8];
    float m = -INFINITY;
    const int groups = (a.V + 7) >> 3;
    for (int gg = threadIdx.x; gg < groups; gg += kThreads) {
        Logit<T>::load8(row, 8 * gg, a.V, x);
#pragma unroll
        for (int k = 0; k < 8; ++k) m = fmaxf(m, __fmul_rn(x[k], a.invT));
    }
    KahanF s;
    if (m != -INFINITY)
        for (int gg = threadIdx.x; gg < groups; gg += kThreads) {
            Logit<T>::load8(row, 8 * gg, a.V, x);
#pragma unroll
            for (int k = 0; k < 8; ++k) s.add(expf(__fsub_rn(__fmul_rn(x[k], a.invT), m)));
        }
    const MaxSum tot = block_maxsum(sh, MaxSum{m, s.ff()});
    double lse_q = 0.0;
    if (i < g) {
        const int r = qrow_index(a, b, i);
        float mq = -INFINITY;
        KahanF sq;
        if (r >= 0 && r < a.q_R) {
            const float2 *st = a.qstats + ((int64_t)b * a.q_R + r) * a.C;
            for (int c = threadIdx.x; c < a.C; c += kThreads) mq = fmaxf(mq, st[c].x);
            const float mqw = mq;
            if (mqw != -INFINITY)
                for (int c = threadIdx.x; c < a.C; c += kThreads)
                    sq.add(__fmul_rn(st[c].y, expf(__fsub_rn(st[c].x, mqw))));
        } else if (threadIdx.x == 0) {
            raise_status(a.status, kDevBadIndex);
        }
        lse_q = lse_of(block_maxsum(sh, MaxSum{mq, sq.ff()}));
    }
    if (threadIdx.x == 0) {
        BvRow &o = a.rows[(int64_t)b * NN + i];
        o.lse_t = lse_of(tot);
        o.lse_q = lse_q;
    }
}

// w_1..w_upto of tree b from point values (serial, tiny); returns w_upto.
template <typename T>
__device__ float chain_weights(const BvArgs &a, int b, int upto, float *w_all) {
    const int NN = a.N + 1;
    float w = 1.0f;
    if (w_all) w_all[0] = w;
    for (int j = 1; j <= upto; ++j) {
        const int X = a.token[(int64_t)b * NN + j];
        const BvRow &rw = a.rows[(int64_t)b * NN + j - 1];
        float th, tl, qh, ql;
        split(rw.lse_t, th, tl);
        split(rw.lse_q, qh, ql);
        const int r = qrow_index(a, b, j - 1);
        const float p = prob_of(Logit<T>::load1(trow_ptr<T>(a, b, j - 1), X), a.invT, th, tl);
        const float q = prob_of(Logit<T>::load1(qrow_ptr<T>(a, b, r), X), a.invT, qh, ql);
        const float ratio = q > 0.f ? __fdiv_rn(__fmul_rn(w, p), q) : 1.0f;
        w = fminf(ratio, 1.0f);
        if (w_all) w_all[j] = w;
    }
    return w;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) k_bv_resid(BvArgs a) {
    pdl_begin();
    __shared__ BlockRed sh;
    __shared__ float w_sh;
    __shared__ int ok_sh;
    const int g = a.N, NN = a.N + 1;
    const int b = blockIdx.x / g, i = blockIdx.x - b * g;
    if (threadIdx.x == 0) {
        int ok = 1;
        for (int j = 1; j <= i; ++j) {
            const int X = a.token[(int64_t)b * NN + j];
            const int r = qrow_index(a, b, j - 1);
            if (X < 0 || X >= a.V || r < 0 || r >= a.q_R) ok = 0;
        }
        const int r = qrow_index(a, b, i);
        if (r < 0 || r >= a.q_R) ok = 0;
        ok_sh = ok;
        w_sh = ok ? chain_weights<T>(a, b, i, nullptr) : 0.f;
        if (!ok) raise_status(a.status, kDevBadIndex);
    }
    __syncthreads();
    if (!ok_sh) return;
    const float w = w_sh;
    const BvRow &rw = a.rows[(int64_t)b * NN + i];
    float th, tl, qh, ql;
    split(rw.lse_t, th, tl);
    split(rw.lse_q, qh, ql);
    const T *trow = trow_ptr<T>(a, b, i);
    const T *qrow = qrow_ptr<T>(a, b, qrow_index(a, b, i));
    KahanF acc;
    float xt[8], xq[8];
    const int groups = (a.V + 7) >> 3;
    for (int gg = threadIdx.x; gg < groups; gg += kThreads) {
        Logit<T>::load8(trow, 8 * gg, a.V, xt);
        Logit<T>::load8(qrow, 8 * gg, a.V, xq);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (8 * gg + k >= a.V) break;
            const float p = prob_of(xt[k], a.invT, th, tl), q = prob_of(xq[k], a.invT, qh, ql);
            acc.add(fmaxf(__fsub_rn(__fmul_rn(w, p), q), 0.f));
        }
    }
    const FF Sf = block_sum(sh, acc.ff());
    const double S = (double)Sf.hi + (double)Sf.lo;
    if (threadIdx.x == 0) {
        BvRow &o = a.rows[(int64_t)b * NN + i];
        o.S = S;
        o.w = (double)w;
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) k_bv_final(BvArgs a) {
    pdl_begin();
    __shared__ BlockRed sh;
    __shared__ int tau_sh, ok_sh;
    __shared__ float wtau_sh;
    const int g = a.N, NN = a.N + 1;
    const int b = blockIdx.x;
    if (threadIdx.x == 0) {
        int ok = 1;
        for (int j = 1; j <= g; ++j) {
            const int X = a.token[(int64_t)b * NN + j];
            const int r = qrow_index(a, b, j - 1);
            if (X < 0 || X >= a.V || r < 0 || r >= a.q_R) ok = 0;
        }
        int tau = 0;
        float wt = 1.f;
        if (ok) {
            const float wg = chain_weights<T>(a, b, g, nullptr);
            for (int i = 1; i <= g; ++i) {
                float h;
                if (i < g) {
                    const BvRow &rw = a.rows[(int64_t)b * NN + i];
                    const double den = rw.S + 1.0 - rw.w;
                    h = den > 0.0 ? (float)(rw.S / den) : 1.0f;
                } else {
                    h = wg;
                }
                const float eta = uniform_of(draw_word(a.seed, kBlockEta, (uint32_t)b, (uint32_t)i, 0u));
                if (eta <= h) tau = i;
            }
            wt = tau < g ? (float)a.rows[(int64_t)b * NN + tau].w : wg;
        } else {
            raise_status(a.status, kDevBadIndex);
        }
        tau_sh = tau;
        wtau_sh = wt;
        ok_sh = ok;
    }
    __syncthreads();
    const int tau = tau_sh;
    const float wt = wtau_sh;
    // final token, two-level Gumbel-max over chunks of 256 tokens: from the residual at tau,
    // or from the target row (tau = g, or a residual without mass)
    const BvRow &rw = a.rows[(int64_t)b * NN + tau];
    const bool from_target = tau == g || !(rw.S > 0.0);
    float th, tl, qh, ql;
    split(rw.lse_t, th, tl);
    split(tau < g ? rw.lse_q : 0.0, qh, ql);
    const T *trow = trow_ptr<T>(a, b, tau);
    const T *qrow = tau < g ? qrow_ptr<T>(a, b, qrow_index(a, b, tau)) : trow;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // 8 consecutive tokens from v0: log-weights x*invT (target row) or weights r >= 0 (residual);
    // tokens past V get -inf / 0
    auto vals8 = [&](int v0, float out[8]) {
        float xt[8], xq[8];
        Logit<T>::load8(trow, v0, a.V, xt);
        if (!from_target) Logit<T>::load8(qrow, v0, a.V, xq);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (v0 + k >= a.V) {
                out[k] = from_target ? -INFINITY : 0.f;
            } else if (from_target) {
                out[k] = __fmul_rn(xt[k], a.invT);
            } else {
                const float p = prob_of(xt[k], a.invT, th, tl), q = prob_of(xq[k], a.invT, qh, ql);
                out[k] = fmaxf(__fsub_rn(__fmul_rn(wt, p), q), 0.f);
            }
        }
    };
    unsigned long long best = 0ull;
    if (ok_sh)
        for (int c = warp; c < a.C; c += kWarps) {
            float v[8];
            vals8(c * kChunk + lane * 8, v);
            float A = -INFINITY;
            if (from_target) {  // chunk log-mass = log-sum-exp of the logits
                float mx = -INFINITY;
#pragma unroll
                for (int k = 0; k < 8; ++k) mx = fmaxf(mx, v[k]);
                mx = warp_max(mx);
                float s = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) s += fast_exp2(__fmul_rn(__fsub_rn(v[k], mx), kLog2e));
                s = warp_sum(s);
                A = __fadd_rn(mx, logf(s));
            } else {  // chunk mass = sum of the residual weights
                float s = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) s += v[k];
                s = warp_sum(s);
                if (s > 0.f) A = logf(s);
            }
            if (lane == 0 && A != -INFINITY) {
                const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)tau, (uint32_t)c);
                const unsigned long long pk = pack_key(__fadd_rn(A, gumbel_of(w)), (uint32_t)c);
                best = pk > best ? pk : best;
            }
        }
    best = block_argmax(sh, best);
    unsigned long long tokk = 0ull;
    if (best != 0ull && warp == 0) {
        const int v0 = (int)key_id(best) * kChunk + lane * 8;
        float v[8];
        vals8(v0, v);
        const Words4 w0 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)tau, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)tau, (uint32_t)(v0 >> 2) + 1u);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            if (v0 + k >= a.V) break;
            float l;
            if (from_target) {
                l = v[k];
            } else {
                if (!(v[k] > 0.f)) continue;
                l = logf(v[k]);
            }
            const float key = __fadd_rn(l, gumbel_of(k < 4 ? w0.w[k] : w1.w[k - 4]));
            const unsigned long long pk = pack_key(key, (uint32_t)(v0 + k));
            tokk = pk > tokk ? pk : tokk;
        }
    }
    tokk = block_argmax(sh, tokk);
    if (threadIdx.x == 0) {
        int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
        int32_t *onode = a.out_nodes + (int64_t)b * a.L;
        const int t = ok_sh ? tau : 0;
        for (int k = 0; k <= a.L; ++k) otok[k] = -1;
        for (int k = 0; k < a.L; ++k) onode[k] = -1;
        for (int i = 1; i <= t; ++i) {
            otok[i - 1] = a.token[(int64_t)b * NN + i];
            onode[i - 1] = i;
        }
        otok[t] = (ok_sh && tokk != 0ull) ? (int32_t)key_id(tokk) : -1;
        a.out_len[b] = ok_sh ? t + 1 : 0;
    }
}

template <typename T>
cudaError_t launch_bv_t(const BvArgs &a, int B, cudaStream_t s) {
    const int NN = a.N + 1;
    cudaError_t e = launch_pdl(k_bv_rows<T>, dim3((unsigned)(B * NN)), dim3(kThreads), 0, s, 0, a);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_bv_resid<T>, dim3((unsigned)(B * a.N)), dim3(kThreads), 0, s, 0, a);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_bv_final<T>, dim3((unsigned)B), dim3(kThreads), 0, s, 0, a);
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
    a.rows = reinterpret_cast<BvRow *>(reinterpret_cast<unsigned char *>(status) + 256);
    if (target.dtype == 1) return launch_bv_t<__nv_bfloat16>(a, B, s);
    return launch_bv_t<float>(a, B, s);
}

}  // namespace tsb
