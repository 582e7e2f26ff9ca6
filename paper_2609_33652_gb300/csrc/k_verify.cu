// Tree verification by recursive rejection sampling for WoR candidates (Sec. 2.3 Eq.
// rs-overlap; App. A), lossless on the frozen topology (Prop. 1).
//
// One thread-block cluster per tree. CTA r of the cluster owns the chunk-aligned vocabulary
// slice [r*slice, (r+1)*slice) and keeps that slice of the current node in shared memory as
// fp32: P holds the target logits, later the current residual; Q holds the normalised draft
// law once it is needed. Scalars (log-normalisers, residual masses, argmax keys) are combined
// across the cluster through distributed shared memory: each CTA publishes its partial, the
// cluster barrier orders the writes, and every CTA combines all partials in rank order, so
// all CTAs hold bitwise identical values and take identical decisions.
//
// Walk at node u with children y_1..y_m (slot order), P0 = softmax(target row u),
// Q = softmax(q row of u), t_0 = 1:
//   slot i: p' = p_i(y_i), q' = Q(y_i)/t_i; accept iff U * q' < p';
//           on reject R_{i+1}(v) = max(p_i(v) - Q(v)/t_i, 0), Z_{i+1} = sum R_{i+1},
//           p_{i+1} = R_{i+1}/Z_{i+1}, t_{i+1} = t_i - Q(y_i).
//   A rejected token has p_{i+1} = 0 from then on, which is exactly the exclusion of drawn
//   tokens from the renormalised draft law. Each pass is O(1) per element: P keeps R_i and
//   p_i(v) = P[v] / Z_i; the point value p_i(y) repeats the same fp32 operations from P0(y).
// Per node: one staging pass (the target log-normaliser is accumulated while staging); the
// q row is staged by the first rejection pass only, so a node whose first child is accepted
// reads one row. Final tokens (all children rejected: from R_m; leaf: bonus from the target
// row) are drawn with the two-level Gumbel-max of the contract: chunk keys
// log(chunk mass) + G over chunks of 256 tokens, then the best token of the winning chunk.
#include <cooperative_groups.h>

#include <mutex>

#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace cg = cooperative_groups;

namespace tsb {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;

struct VerifyArgs {
    const void *target;
    int64_t t_bstride, t_rstride;
    const void *q;
    int64_t q_bstride, q_rstride;
    int q_R;
    const float2 *qstats;
    int C;
    const int32_t *qrow_of_node, *depth, *child_off, *child_ids, *token;
    int V, N, L, slice;
    float invT;
    uint64_t seed;
    int32_t *out_tokens, *out_nodes, *out_len;
    uint32_t *status;
};

// A partial of one cluster-wide reduction: two softmax normalisers (target row, q row), a
// plain sum, and an argmax key carrying a token.
struct alignas(16) Slot {
    float m1, s1h, s1l, m2, s2h, s2l, zh, zl;
    unsigned long long key;
    int tok, pad;
};

enum : int { kRedLse = 1, kRedSum = 2, kRedArg = 4 };

__device__ __forceinline__ Slot neutral_slot() {
    Slot s;
    s.m1 = s.m2 = -INFINITY;
    s.s1h = s.s1l = s.s2h = s.s2l = s.zh = s.zl = 0.f;
    s.key = 0ull;
    s.tok = -1;
    s.pad = 0;
    return s;
}

// Symmetric merge of the plain-sum and argmax fields (normalisers are reduced separately).
template <int KIND>
__device__ __forceinline__ Slot merge_slot(const Slot &a, const Slot &b) {
    Slot r = a;
    if (KIND & kRedSum) {
        const FF z = ff_add(FF{a.zh, a.zl}, FF{b.zh, b.zl});
        r.zh = z.hi;
        r.zl = z.lo;
    }
    if (KIND & kRedArg) {
        if (b.key > a.key) {
            r.key = b.key;
            r.tok = b.tok;
        }
    }
    return r;
}

// A normaliser rescaled to a larger reference maximum M (exp evaluated once).
__device__ __forceinline__ FF rescale_to(float m, FF s, float M) {
    return m == -INFINITY ? FF{0.f, 0.f} : (m == M ? s : ff_scale(s, expf(__fsub_rn(m, M))));
}

template <int KIND>
__device__ __forceinline__ Slot warp_reduce_slot(Slot v) {
    if (KIND & kRedLse) {  // maxima first, then every lane rescales once, then plain sums
        const float M1 = warp_max(v.m1), M2 = warp_max(v.m2);
        const FF a = warp_sum_ff(rescale_to(v.m1, FF{v.s1h, v.s1l}, M1));
        const FF c = warp_sum_ff(rescale_to(v.m2, FF{v.s2h, v.s2l}, M2));
        v.m1 = M1;
        v.s1h = a.hi;
        v.s1l = a.lo;
        v.m2 = M2;
        v.s2h = c.hi;
        v.s2l = c.lo;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        Slot w = v;
        if (KIND & kRedSum) {
            w.zh = __shfl_xor_sync(kFull, v.zh, o);
            w.zl = __shfl_xor_sync(kFull, v.zl, o);
        }
        if (KIND & kRedArg) {
            w.key = __shfl_xor_sync(kFull, v.key, o);
            w.tok = __shfl_xor_sync(kFull, v.tok, o);
        }
        v = merge_slot<KIND>(v, w);
    }
    return v;
}

struct Scratch {
    Slot slot[2];        // published partials, double-buffered across rounds
    Slot wpart[kWarps];  // per-warp partials of the current round
    Slot res;            // combined result
    FF L2t, L2q;         // log-normalisers of the target and q rows, times log2(e)
    unsigned long long wbest[kWarps];
    unsigned long long cbest;
    float izs[kMaxK], its[kMaxK];  // 1/Z and 1/t of every rejection so far
};

// One cluster-wide reduction: warp butterflies, the CTA's warp partials in warp 0, the
// cluster barrier, then warp 0 of every CTA reads the CS published partials (one per lane)
// and combines them with the same butterfly, so every CTA obtains identical results.
template <int KIND>
__device__ void reduce_round(Scratch &sh, int &par, const cg::cluster_group &cluster, Slot mine) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const Slot w = warp_reduce_slot<KIND>(mine);
    if (lane == 0) sh.wpart[warp] = w;
    __syncthreads();
    if (warp == 0) {
        const Slot v = warp_reduce_slot<KIND>(lane < kWarps ? sh.wpart[lane] : neutral_slot());
        if (lane == 0) sh.slot[par] = v;
    }
    cluster.sync();
    if (warp == 0) {
        const int CS = (int)cluster.num_blocks();
        const Slot v = warp_reduce_slot<KIND>(lane < CS ? *cluster.map_shared_rank(&sh.slot[par], lane)
                                                        : neutral_slot());
        if (lane == 0) {
            sh.res = v;
            if (KIND & kRedLse) {
                const FF l1 = v.s1h > 0.f ? maxsum_lse(MaxSum{v.m1, FF{v.s1h, v.s1l}}) : FF{0.f, 0.f};
                const FF l2 = v.s2h > 0.f ? maxsum_lse(MaxSum{v.m2, FF{v.s2h, v.s2l}}) : FF{0.f, 0.f};
                sh.L2t = ff_times_log2e(l1);
                sh.L2q = ff_times_log2e(l2);
            }
        }
    }
    __syncthreads();
    par ^= 1;
}

// The residual after rejecting a slot: max(p - q/t, 0) with 1/t precomputed; one fma, so the
// element passes and the point values produce the same bits.
__device__ __forceinline__ float resid(float p, float q, float it) { return fmaxf(__fmaf_rn(-q, it, p), 0.f); }

// p_i(y) from P0(y), Q(y): the same fp32 operations the element passes perform.
__device__ __forceinline__ float point_residual(float p0, float q, const float *izs, const float *its, int i) {
    float p = p0;
    for (int j = 0; j < i; ++j) p = __fmul_rn(resid(p, q, its[j]), izs[j]);
    return p;
}

// Per-thread online (max, sum of exp(x - max)) accumulation, eight logits at a time.
struct OnlineLse {
    float m = -INFINITY;
    KahanF s;
    __device__ __forceinline__ MaxSum value() const { return MaxSum{m, s.ff()}; }
    __device__ __forceinline__ void add8(const float x[8]) {
        float gm = x[0];
#pragma unroll
        for (int k = 1; k < 8; ++k) gm = fmaxf(gm, x[k]);
        if (gm == -INFINITY) return;
        if (gm > m) {
            if (m != -INFINITY) {
                const float scale = fast_exp2(__fmul_rn(__fsub_rn(m, gm), kLog2e));
                s.s = __fmul_rn(s.s, scale);
                s.c = __fmul_rn(s.c, scale);
            }
            m = gm;
        }
        float t = 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k) t += fast_exp2(__fmul_rn(__fsub_rn(x[k], m), kLog2e));
        s.add(t);
    }
};

template <typename T>
struct Walk {
    const VerifyArgs &a;
    Scratch &sh;
    const cg::cluster_group &cluster;
    float *P, *Qs;
    int &par;
    int b, lo, n, crank;

    __device__ int groups() const { return (n + 7) >> 3; }

    // Stage x = fp32(z) * invT of this CTA's target slice into P; optionally accumulate the
    // target row's log-normaliser.
    // Stage x = fp32(z) * invT of this CTA's target slice into P; optionally accumulate the
    // target row's log-normaliser. Loads are issued in batches of kBatch groups per thread
    // before any is used, so a slice costs one memory round trip per batch.
    static constexpr int kBatch = sizeof(T) == 2 ? 6 : 3;
    __device__ void stage_target(const T *row, OnlineLse *lse) {
        const int G = groups();
        for (int g0 = threadIdx.x; g0 < G; g0 += kBatch * kThreads) {
            RawGroup<T> raw[kBatch];
#pragma unroll
            for (int e = 0; e < kBatch; ++e) {
                const int g = g0 + e * kThreads;
                if (g < G) raw[e].load(row, lo + 8 * g, a.V);
            }
#pragma unroll
            for (int e = 0; e < kBatch; ++e) {
                const int g = g0 + e * kThreads;
                if (g >= G) break;
                float x[8];
                raw[e].unpack(x);
#pragma unroll
                for (int k = 0; k < 8; ++k) x[k] = __fmul_rn(x[k], a.invT);  // padding stays -inf
                reinterpret_cast<float4 *>(P)[2 * g] = make_float4(x[0], x[1], x[2], x[3]);
                reinterpret_cast<float4 *>(P)[2 * g + 1] = make_float4(x[4], x[5], x[6], x[7]);
                if (lse) lse->add8(x);
            }
        }
    }

    // Ask L2 for this CTA's slice of a row that is likely needed soon (one request per 128 B).
    __device__ void prefetch_slice(const T *row) {
        const char *base = reinterpret_cast<const char *>(row + lo);
        const int bytes = n * (int)sizeof(T);
        for (int off = threadIdx.x * 128; off < bytes; off += kThreads * 128)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(base + off));
    }

    // Two-level draw (chunk by Gumbel-max over chunk masses, then token by Gumbel-max inside
    // the chunk) in one cluster round: every CTA picks its best chunk and that chunk's best
    // token; the cluster keeps the pair with the largest chunk key. val(j, v) returns a
    // log-weight (LOGITS) or a weight >= 0 for the element at smem index j, token v.
    template <bool LOGITS, typename F>
    __device__ int draw(int node, F val) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int nch = (n + kChunk - 1) / kChunk;
        unsigned long long best = 0ull;
        for (int cl = warp; cl < nch; cl += kWarps) {
            const int i0 = cl * kChunk + lane * 8;
            float v[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) v[k] = (i0 + k < n) ? val(i0 + k, lo + i0 + k) : (LOGITS ? -INFINITY : 0.f);
            float A = -INFINITY;
            if (LOGITS) {
                float mx = -INFINITY;
#pragma unroll
                for (int k = 0; k < 8; ++k) mx = fmaxf(mx, v[k]);
                mx = warp_max(mx);
                float sm = 0.f;
                if (mx != -INFINITY) {
#pragma unroll
                    for (int k = 0; k < 8; ++k) sm += fast_exp2(__fmul_rn(__fsub_rn(v[k], mx), kLog2e));
                }
                sm = warp_sum(sm);
                if (mx != -INFINITY) A = __fadd_rn(mx, logf(sm));
            } else {
                float sm = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) sm += v[k];
                sm = warp_sum(sm);
                if (sm > 0.f) A = logf(sm);
            }
            if (lane == 0 && A != -INFINITY) {
                const int c = (lo >> 8) + cl;
                const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)node, (uint32_t)c);
                const unsigned long long pk = pack_key(__fadd_rn(A, gumbel_of(w)), (uint32_t)c);
                best = pk > best ? pk : best;
            }
        }
        if (lane == 0) sh.wbest[warp] = best;
        __syncthreads();
        if (warp == 0) {
            unsigned long long cb = warp_max_u64(lane < kWarps ? sh.wbest[lane] : 0ull);
            // the best token inside this CTA's best chunk
            unsigned long long tb = 0ull;
            if (cb != 0ull) {
                const int i0 = (int)key_id(cb) * kChunk - lo + lane * 8, v0 = lo + i0;
                const Words4 w0 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2));
                const Words4 w1 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2) + 1u);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    if (i0 + k >= n) break;
                    const float x = val(i0 + k, v0 + k);
                    float l;
                    if (LOGITS) {
                        if (x == -INFINITY) continue;
                        l = x;
                    } else {
                        if (!(x > 0.f)) continue;
                        l = logf(x);
                    }
                    const unsigned long long pk = pack_key(__fadd_rn(l, gumbel_of(k < 4 ? w0.w[k] : w1.w[k - 4])),
                                                           (uint32_t)(v0 + k));
                    tb = pk > tb ? pk : tb;
                }
                tb = warp_max_u64(tb);
            }
            if (lane == 0) {
                sh.cbest = cb;
                sh.wbest[0] = tb;
            }
        }
        __syncthreads();
        Slot mine = neutral_slot();
        if (threadIdx.x == 0 && sh.cbest != 0ull) {
            mine.key = sh.cbest;
            mine.tok = (int)key_id(sh.wbest[0]);
        }
        reduce_round<kRedArg>(sh, par, cluster, mine);
        return sh.res.key == 0ull ? -1 : sh.res.tok;
    }
};

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_verify_rrs(VerifyArgs a) {
    extern __shared__ __align__(16) float dyn[];
    float *P = dyn;
    float *Qs = dyn + a.slice;
    __shared__ Scratch sh;

    cg::cluster_group cluster = cg::this_cluster();
    const int CS = (int)cluster.num_blocks();
    const int crank = (int)cluster.block_rank();
    const int b = blockIdx.x / CS;
    const int NN = a.N + 1;
    const int lo = crank * a.slice;
    const int n = max(0, min(a.V - lo, a.slice));
    const bool writer = crank == 0 && threadIdx.x == 0;
    int par = 0;
    Walk<T> W{a, sh, cluster, P, Qs, par, b, lo, n, crank};
    const int groups = W.groups();

    const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
    const int32_t *kids = a.child_ids + (int64_t)b * a.N;
    const int32_t *tok = a.token + (int64_t)b * NN;
    int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
    int32_t *onode = a.out_nodes + (int64_t)b * a.L;

    cluster.sync();  // every CTA of the cluster runs before any distributed access

    int u = 0, nacc = 0, final_tok = -1;
    bool bad = false;
    for (int step = 0; step <= a.L; ++step) {
        const int o = off[u], m = off[u + 1] - o;
        if (m < 0 || m > kMaxK || o < 0 || o + m > a.N) {
            bad = true;
            break;
        }
        const T *trow = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
        __syncthreads();
        if (m == 0) {  // leaf: bonus token from the node's target row
            W.stage_target(trow, nullptr);
            __syncthreads();
            final_tok = W.template draw<true>(u, [&](int i, int) { return P[i]; });
            break;
        }
        const int r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : a.depth[(int64_t)b * NN + u];
        if (r < 0 || r >= a.q_R) {
            bad = true;
            break;
        }
        const T *qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;
        {  // likely next reads: this node's q row (first rejection), the first child's target row
            W.prefetch_slice(qrow);
            const int c0 = kids[o];
            if (c0 >= 1 && c0 <= a.N)
                W.prefetch_slice(static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride +
                                 (int64_t)c0 * a.t_rstride);
        }

        // staging pass with the target log-normaliser; q row log-normaliser from its chunk stats
        OnlineLse lt;
        W.stage_target(trow, &lt);
        const float2 *st = a.qstats + ((int64_t)b * a.q_R + r) * a.C;
        float m2 = -INFINITY;
        for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads) m2 = fmaxf(m2, st[c].x);
        KahanF s2;
        if (m2 != -INFINITY)
            for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads)
                s2.add(__fmul_rn(st[c].y, expf(__fsub_rn(st[c].x, m2))));
        {
            Slot mine = neutral_slot();
            const MaxSum t1 = lt.value();
            mine.m1 = t1.m;
            mine.s1h = t1.s.hi;
            mine.s1l = t1.s.lo;
            const FF q2 = s2.ff();
            mine.m2 = m2;
            mine.s2h = q2.hi;
            mine.s2l = q2.lo;
            reduce_round<kRedLse>(sh, par, cluster, mine);
        }
        const FF L2t = sh.L2t, L2q = sh.L2q;

        FF t = FF{1.f, 0.f};  // draft mass not yet drawn
        int accepted = -1;
        for (int i = 0; i < m; ++i) {
            const int c = kids[o + i];
            const int y = (c >= 1 && c <= a.N) ? tok[c] : -1;
            if (y < 0 || y >= a.V) {
                bad = true;
                break;
            }
            const float it = t.hi > 0.f ? __frcp_rn(t.hi) : 0.f;  // 1/t_i
            const float P0y = exp_shifted(__fmul_rn(Logit<T>::load1(trow, y), a.invT), L2t);
            const float Qy = exp_shifted(__fmul_rn(Logit<T>::load1(qrow, y), a.invT), L2q);
            const float pp = point_residual(P0y, Qy, sh.izs, sh.its, i);
            const float qp = __fmul_rn(Qy, it);
            const float U = uniform_of(draw_word(a.seed, kAccept, (uint32_t)b, (uint32_t)c, 0u));
            if (__fmul_rn(U, qp) < pp) {
                accepted = c;
                break;
            }
            // p_i(v) of the element at smem index j (P holds x before the first rejection,
            // R_i afterwards)
            const float izp = i > 0 ? sh.izs[i - 1] : 1.f;
            auto p_of = [&](int j) { return i == 0 ? exp_shifted(P[j], L2t) : __fmul_rn(P[j], izp); };
            if (i == m - 1) {  // every slot rejected: final token from R_m = max(p_i - Q/t_i, 0)
                if (i == 0) {  // the q slice was never staged: stage it (normalised) now
                    for (int g = threadIdx.x; g < groups; g += kThreads) {
                        float x[8];
                        Logit<T>::load8(qrow, lo + 8 * g, a.V, x);
#pragma unroll
                        for (int k = 0; k < 8; ++k) Qs[8 * g + k] = exp_shifted(__fmul_rn(x[k], a.invT), L2q);
                    }
                    __syncthreads();
                }
                final_tok = W.template draw<false>(u, [&](int j, int) { return resid(p_of(j), Qs[j], it); });
                if (final_tok < 0) {  // no residual mass (rounding only): the node's target row
                    __syncthreads();
                    W.stage_target(trow, nullptr);
                    __syncthreads();
                    final_tok = W.template draw<true>(u, [&](int j, int) { return P[j]; });
                }
                break;
            }
            // residual pass (the first one also stages the normalised q slice)
            KahanF zl;
            for (int g = threadIdx.x; g < groups; g += kThreads) {
                float q8[8], r8[8];
                if (i == 0) {
                    Logit<T>::load8(qrow, lo + 8 * g, a.V, q8);
#pragma unroll
                    for (int k = 0; k < 8; ++k) q8[k] = exp_shifted(__fmul_rn(q8[k], a.invT), L2q);
                    reinterpret_cast<float4 *>(Qs)[2 * g] = make_float4(q8[0], q8[1], q8[2], q8[3]);
                    reinterpret_cast<float4 *>(Qs)[2 * g + 1] = make_float4(q8[4], q8[5], q8[6], q8[7]);
                } else {
                    const float4 qa = reinterpret_cast<const float4 *>(Qs)[2 * g];
                    const float4 qb = reinterpret_cast<const float4 *>(Qs)[2 * g + 1];
                    q8[0] = qa.x; q8[1] = qa.y; q8[2] = qa.z; q8[3] = qa.w;
                    q8[4] = qb.x; q8[5] = qb.y; q8[6] = qb.z; q8[7] = qb.w;
                }
                float sum8 = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    r8[k] = resid(p_of(8 * g + k), q8[k], it);  // padding: p = 0 (x = -inf), q = 0
                    sum8 += r8[k];
                }
                reinterpret_cast<float4 *>(P)[2 * g] = make_float4(r8[0], r8[1], r8[2], r8[3]);
                reinterpret_cast<float4 *>(P)[2 * g + 1] = make_float4(r8[4], r8[5], r8[6], r8[7]);
                zl.add(sum8);
            }
            {
                Slot mine = neutral_slot();
                const FF z = zl.ff();
                mine.zh = z.hi;
                mine.zl = z.lo;
                reduce_round<kRedSum>(sh, par, cluster, mine);
            }
            const float Z = sh.res.zh;
            if (!(Z > 0.f)) {  // no residual mass (rounding only): the node's target row
                W.stage_target(trow, nullptr);
                __syncthreads();
                final_tok = W.template draw<true>(u, [&](int j, int) { return P[j]; });
                break;
            }
            if (threadIdx.x == 0) {
                sh.izs[i] = __frcp_rn(Z);
                sh.its[i] = it;
            }
            __syncthreads();
            t = ff_add(t, FF{-Qy, 0.f});
        }
        if (bad || accepted < 0) break;
        if (nacc >= a.L) {  // deeper than the depth cap: the tree arrays are inconsistent
            bad = true;
            break;
        }
        if (writer) {
            otok[nacc] = tok[accepted];
            onode[nacc] = accepted;
        }
        ++nacc;
        u = accepted;
    }
    if (writer) {
        if (bad) raise_status(a.status, kDevBadTree);
        otok[nacc] = final_tok;
        for (int k = nacc + 1; k <= a.L; ++k) otok[k] = -1;
        for (int k = nacc; k < a.L; ++k) onode[k] = -1;
        a.out_len[b] = bad ? 0 : nacc + 1;
    }
    cluster.sync();  // no CTA leaves while another may still read its shared memory
}

constexpr size_t kSmemLimit = 210 * 1024;

// Chunk-aligned slice of each CTA and the dynamic shared memory it needs for cluster size cs.
void slice_for(int V, int cs, int *slice_out, size_t *smem_out) {
    int slice = (V + cs - 1) / cs;
    slice = (slice + kChunk - 1) / kChunk * kChunk;
    *slice_out = slice;
    *smem_out = 2 * (size_t)slice * sizeof(float);
}

struct ClusterChoice {
    int V, B, elem, cs;
};

// The cluster size for (V, B): the largest size up to 16 (above 8 the cluster is
// non-portable) whose clusters can all be resident at once, so every tree walks in the same
// wave; when no size fits the whole batch, the size with the most concurrently resident CTAs. Decisions are
// cached per (V, B, element size); the cache is a pure function of the device.
template <typename T>
int choose_cluster(int V, int B, int *slice_out, size_t *smem_out) {
    static ClusterChoice cache[16];
    static int cache_n = 0;
    static std::mutex mu;
    {
        std::lock_guard<std::mutex> g(mu);
        for (int i = 0; i < cache_n; ++i)
            if (cache[i].V == V && cache[i].B == B && cache[i].elem == (int)sizeof(T)) {
                slice_for(V, cache[i].cs, slice_out, smem_out);
                return cache[i].cs;
            }
    }
    const int lo_cs = V >= 32768 ? 4 : V >= 8192 ? 4 : V >= 2048 ? 2 : 1;
    const int hi_cs = V >= 32768 ? 16 : lo_cs;
    int chosen = -1, best_cs = -1;
    long best_ctas = -1;
    for (int cs = hi_cs; cs >= 1; --cs) {
        int slice;
        size_t smem;
        slice_for(V, cs, &slice, &smem);
        if (smem > kSmemLimit) break;  // smaller clusters only need more shared memory
        if (cs < lo_cs && chosen < 0 && best_cs > 0) break;
        if (cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
            continue;
        if (cs > 8 && cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                          cudaSuccess)
            continue;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)(B * cs), 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = (unsigned)cs;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, k_verify_rrs<T>, &cfg) != cudaSuccess || n <= 0) continue;
        if (n >= B) {
            chosen = cs;
            break;
        }
        if ((long)n * cs > best_ctas) {
            best_ctas = (long)n * cs;
            best_cs = cs;
        }
    }
    if (chosen < 0) chosen = best_cs;
    if (chosen < 0) {  // the slices do not fit below 16 CTAs: use 16 (non-portable)
        int slice;
        size_t smem;
        slice_for(V, 16, &slice, &smem);
        chosen = smem <= kSmemLimit ? 16 : -1;
    }
    if (chosen > 0) {
        std::lock_guard<std::mutex> g(mu);
        if (cache_n < 16) cache[cache_n++] = ClusterChoice{V, B, (int)sizeof(T), chosen};
        slice_for(V, chosen, slice_out, smem_out);
    }
    return chosen;
}

template <typename T>
cudaError_t launch_rrs_t(VerifyArgs a, int B, cudaStream_t s) {
    int slice = 0;
    size_t smem = 0;
    const int cs = choose_cluster<T>(a.V, B, &slice, &smem);
    if (cs < 0) return cudaErrorInvalidValue;
    a.slice = slice;
    cudaError_t e = cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (cs > 8) {
        e = cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(B * cs), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, k_verify_rrs<T>, a);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_verify_rrs(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                              const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                              const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                              int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyArgs a;
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
    a.slice = 0;
    a.invT = invT;
    a.seed = seed;
    a.out_tokens = out_tokens;
    a.out_nodes = out_nodes;
    a.out_len = out_len;
    a.status = status;
    if (target.dtype == 1) return launch_rrs_t<__nv_bfloat16>(a, B, s);
    return launch_rrs_t<float>(a, B, s);
}

}  // namespace tsb
