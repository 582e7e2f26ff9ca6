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

struct alignas(16) Slot {
    double s1, s2, z;
    unsigned long long key;
    float m1, m2;
    float hi1, lo1, hi2, lo2;  // log-normalisers as fp32 hi + lo (filled by the combine)
};

struct Scratch {
    Slot slot[2];  // published partials, double-buffered across rounds
    Slot res;      // combined result
    double ws1[kWarps], ws2[kWarps], wz[kWarps];
    unsigned long long wkey[kWarps];
    float wm1[kWarps], wm2[kWarps];
    float zs[kMaxK], ts[kMaxK];
};

__device__ __forceinline__ float qratio(float q, float t) { return (q > 0.f && t > 0.f) ? __fdiv_rn(q, t) : 0.f; }

// exp(x - LSE) with LSE = hi + lo; x = fp32(z) * invT
__device__ __forceinline__ float prob_of(float x, float hi, float lo) { return expf(__fsub_rn(__fsub_rn(x, hi), lo)); }

// p_i(y) from P0(y), Q(y): the same fp32 operations the element passes perform.
__device__ __forceinline__ float point_residual(float p0, float q, const float *zs, const float *ts, int i) {
    float p = p0;
    for (int j = 0; j < i; ++j) {
        const float r = fmaxf(__fsub_rn(p, qratio(q, ts[j])), 0.f);
        p = __fdiv_rn(r, zs[j]);
    }
    return p;
}

// One cluster-wide reduction of (max, sum-exp) x2, a plain sum and an argmax key.
__device__ void reduce_round(Scratch &sh, int &par, const cg::cluster_group &cluster, float m1, double s1, float m2,
                             double s2, double z, unsigned long long key) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    {
        const float a1 = warp_max(m1), a2 = warp_max(m2);
        const double t1 = warp_sum_d(m1 == -INFINITY ? 0.0 : s1 * (double)expf(m1 - a1));
        const double t2 = warp_sum_d(m2 == -INFINITY ? 0.0 : s2 * (double)expf(m2 - a2));
        const double tz = warp_sum_d(z);
        const unsigned long long tk = warp_max_u64(key);
        if (lane == 0) {
            sh.wm1[warp] = a1;
            sh.ws1[warp] = t1;
            sh.wm2[warp] = a2;
            sh.ws2[warp] = t2;
            sh.wz[warp] = tz;
            sh.wkey[warp] = tk;
        }
    }
    __syncthreads();
    if (warp == 0) {
        const float b1 = lane < kWarps ? sh.wm1[lane] : -INFINITY;
        const float b2 = lane < kWarps ? sh.wm2[lane] : -INFINITY;
        const double c1 = lane < kWarps ? sh.ws1[lane] : 0.0;
        const double c2 = lane < kWarps ? sh.ws2[lane] : 0.0;
        const double cz = lane < kWarps ? sh.wz[lane] : 0.0;
        const unsigned long long ck = lane < kWarps ? sh.wkey[lane] : 0ull;
        const float a1 = warp_max(b1), a2 = warp_max(b2);
        const double t1 = warp_sum_d(b1 == -INFINITY ? 0.0 : c1 * (double)expf(b1 - a1));
        const double t2 = warp_sum_d(b2 == -INFINITY ? 0.0 : c2 * (double)expf(b2 - a2));
        const double tz = warp_sum_d(cz);
        const unsigned long long tk = warp_max_u64(ck);
        if (lane == 0) {
            Slot &s = sh.slot[par];
            s.m1 = a1;
            s.s1 = t1;
            s.m2 = a2;
            s.s2 = t2;
            s.z = tz;
            s.key = tk;
        }
    }
    cluster.sync();
    if (threadIdx.x == 0) {
        const int CS = (int)cluster.num_blocks();
        float M1 = -INFINITY, M2 = -INFINITY;
        for (int r = 0; r < CS; ++r) {
            const Slot *p = cluster.map_shared_rank(&sh.slot[par], r);
            M1 = fmaxf(M1, p->m1);
            M2 = fmaxf(M2, p->m2);
        }
        double S1 = 0.0, S2 = 0.0, Z = 0.0;
        unsigned long long Kx = 0ull;
        for (int r = 0; r < CS; ++r) {
            const Slot *p = cluster.map_shared_rank(&sh.slot[par], r);
            if (p->m1 != -INFINITY) S1 += p->s1 * (double)expf(p->m1 - M1);
            if (p->m2 != -INFINITY) S2 += p->s2 * (double)expf(p->m2 - M2);
            Z += p->z;
            Kx = p->key > Kx ? p->key : Kx;
        }
        Slot &o = sh.res;
        o.m1 = M1;
        o.m2 = M2;
        o.s1 = S1;
        o.s2 = S2;
        o.z = Z;
        o.key = Kx;
        o.hi1 = o.lo1 = o.hi2 = o.lo2 = 0.f;
        if (S1 > 0.0) {
            const double l1 = (double)M1 + log(S1);
            o.hi1 = (float)l1;
            o.lo1 = (float)(l1 - (double)o.hi1);
        }
        if (S2 > 0.0) {
            const double l2 = (double)M2 + log(S2);
            o.hi2 = (float)l2;
            o.lo2 = (float)(l2 - (double)o.hi2);
        }
    }
    __syncthreads();
    par ^= 1;
}

// Per-thread online (max, sum of exp(x - max)) accumulation.
struct OnlineLse {
    float m = -INFINITY;
    KahanF s;
    __device__ __forceinline__ void add(float x) {
        if (x > m) {
            if (m != -INFINITY) {
                const float scale = fast_exp2(__fmul_rn(__fsub_rn(m, x), kLog2e));
                s.s = __fmul_rn(s.s, scale);
                s.c = __fmul_rn(s.c, scale);
            }
            m = x;
            s.add(1.0f);
        } else {
            s.add(fast_exp2(__fmul_rn(__fsub_rn(x, m), kLog2e)));
        }
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
    __device__ void stage_target(const T *row, OnlineLse *lse) {
        for (int g = threadIdx.x; g < groups(); g += kThreads) {
            float x[8];
            Logit<T>::load8(row, lo + 8 * g, a.V, x);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const bool in = lo + 8 * g + k < a.V;
                const float xv = in ? __fmul_rn(x[k], a.invT) : -INFINITY;
                P[8 * g + k] = xv;
                if (lse && in) lse->add(xv);
            }
        }
    }

    // argmax over the winning chunk of lw + G (warp 0 of the owner CTA computes it).
    template <typename LW>
    __device__ int element_argmax(int node, int c, LW lw) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        unsigned long long best = 0ull;
        const int i0c = c * kChunk - lo;  // chunk start in this CTA's slice
        if (warp == 0 && i0c >= 0 && i0c < n) {
            const int i0 = i0c + lane * 8, v0 = lo + i0;
            const Words4 w0 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2));
            const Words4 w1 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2) + 1u);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                if (i0 + k >= n) break;
                const float l = lw(i0 + k, v0 + k);
                if (l == -INFINITY) continue;
                const float key = __fadd_rn(l, gumbel_of(k < 4 ? w0.w[k] : w1.w[k - 4]));
                const unsigned long long pk = pack_key(key, (uint32_t)(v0 + k));
                best = pk > best ? pk : best;
            }
        }
        reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, best);
        return sh.res.key == 0ull ? -1 : (int)key_id(sh.res.key);
    }

    // Two-level draw from log-weights lw(smem index, token) (-inf = no mass); chunk masses
    // are log-sum-exp of the log-weights.
    template <typename LW>
    __device__ int draw_logits(int node, LW lw) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int nch = (n + kChunk - 1) / kChunk;
        unsigned long long best = 0ull;
        for (int cl = warp; cl < nch; cl += kWarps) {
            const int i0 = cl * kChunk + lane * 8;
            float v[8];
            float mx = -INFINITY;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                v[k] = (i0 + k < n) ? lw(i0 + k, lo + i0 + k) : -INFINITY;
                mx = fmaxf(mx, v[k]);
            }
            mx = warp_max(mx);
            float s = 0.f;
            if (mx != -INFINITY) {
#pragma unroll
                for (int k = 0; k < 8; ++k) s += fast_exp2(__fmul_rn(__fsub_rn(v[k], mx), kLog2e));
            }
            s = warp_sum(s);
            if (lane == 0 && mx != -INFINITY) {
                const int c = (lo >> 8) + cl;
                const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)node, (uint32_t)c);
                const float key = __fadd_rn(__fadd_rn(mx, logf(s)), gumbel_of(w));
                const unsigned long long pk = pack_key(key, (uint32_t)c);
                best = pk > best ? pk : best;
            }
        }
        reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, best);
        if (sh.res.key == 0ull) return -1;
        return element_argmax(node, (int)key_id(sh.res.key), lw);
    }

    // Two-level draw from non-negative weights wf(smem index, token); chunk mass = sum w.
    template <typename WF>
    __device__ int draw_weights(int node, WF wf) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int nch = (n + kChunk - 1) / kChunk;
        unsigned long long best = 0ull;
        for (int cl = warp; cl < nch; cl += kWarps) {
            const int i0 = cl * kChunk + lane * 8;
            float s = 0.f;
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (i0 + k < n) s += wf(i0 + k, lo + i0 + k);
            s = warp_sum(s);
            if (lane == 0 && s > 0.f) {
                const int c = (lo >> 8) + cl;
                const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)node, (uint32_t)c);
                const float key = __fadd_rn(logf(s), gumbel_of(w));
                const unsigned long long pk = pack_key(key, (uint32_t)c);
                best = pk > best ? pk : best;
            }
        }
        reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, best);
        if (sh.res.key == 0ull) return -1;
        auto lw = [&](int i, int v) {
            const float w = wf(i, v);
            return w > 0.f ? logf(w) : -INFINITY;
        };
        return element_argmax(node, (int)key_id(sh.res.key), lw);
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
            final_tok = W.draw_logits(u, [&](int i, int) { return P[i]; });
            break;
        }
        const int r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : a.depth[(int64_t)b * NN + u];
        if (r < 0 || r >= a.q_R) {
            bad = true;
            break;
        }
        const T *qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;

        // staging pass with the target log-normaliser; q row log-normaliser from its chunk stats
        OnlineLse lt;
        W.stage_target(trow, &lt);
        const float2 *st = a.qstats + ((int64_t)b * a.q_R + r) * a.C;
        float m2 = -INFINITY;
        for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads) m2 = fmaxf(m2, st[c].x);
        KahanF s2;
        if (m2 != -INFINITY)
            for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads)
                s2.add(st[c].y * expf(st[c].x - m2));
        reduce_round(sh, par, cluster, lt.m, lt.s.value(), m2, s2.value(), 0.0, 0ull);
        const float lt_hi = sh.res.hi1, lt_lo = sh.res.lo1, lq_hi = sh.res.hi2, lq_lo = sh.res.lo2;

        double t = 1.0;
        int accepted = -1;
        for (int i = 0; i < m; ++i) {
            const int c = kids[o + i];
            const int y = (c >= 1 && c <= a.N) ? tok[c] : -1;
            if (y < 0 || y >= a.V) {
                bad = true;
                break;
            }
            const float t_i = (float)t;
            const float P0y = prob_of(__fmul_rn(Logit<T>::load1(trow, y), a.invT), lt_hi, lt_lo);
            const float Qy = prob_of(__fmul_rn(Logit<T>::load1(qrow, y), a.invT), lq_hi, lq_lo);
            const float pp = point_residual(P0y, Qy, sh.zs, sh.ts, i);
            const float qp = qratio(Qy, t_i);
            const float U = uniform_of(draw_word(a.seed, kAccept, (uint32_t)b, (uint32_t)c, 0u));
            if (__fmul_rn(U, qp) < pp) {
                accepted = c;
                break;
            }
            // p_i(v) of the element at smem index j
            const float zprev = i > 0 ? sh.zs[i - 1] : 1.f;
            auto p_of = [&](int j) { return i == 0 ? prob_of(P[j], lt_hi, lt_lo) : __fdiv_rn(P[j], zprev); };
            if (i == m - 1) {  // every slot rejected: final token from R_m = max(p_i - Q/t_i, 0)
                if (i == 0) {  // the q slice was never staged: stage it (normalised) now
                    for (int g = threadIdx.x; g < groups; g += kThreads) {
                        float x[8];
                        Logit<T>::load8(qrow, lo + 8 * g, a.V, x);
#pragma unroll
                        for (int k = 0; k < 8; ++k) Qs[8 * g + k] = prob_of(__fmul_rn(x[k], a.invT), lq_hi, lq_lo);
                    }
                    __syncthreads();
                }
                final_tok = W.draw_weights(u, [&](int j, int) {
                    return fmaxf(__fsub_rn(p_of(j), qratio(Qs[j], t_i)), 0.f);
                });
                if (final_tok < 0) {  // no residual mass (rounding only): the node's target row
                    __syncthreads();
                    W.stage_target(trow, nullptr);
                    __syncthreads();
                    final_tok = W.draw_logits(u, [&](int j, int) { return P[j]; });
                }
                break;
            }
            // residual pass (the first one also stages the normalised q slice)
            KahanF zl;
            for (int g = threadIdx.x; g < groups; g += kThreads) {
                float xq[8];
                if (i == 0) Logit<T>::load8(qrow, lo + 8 * g, a.V, xq);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int j = 8 * g + k;
                    if (lo + j >= a.V) break;
                    float qv;
                    if (i == 0) {
                        qv = prob_of(__fmul_rn(xq[k], a.invT), lq_hi, lq_lo);
                        Qs[j] = qv;
                    } else {
                        qv = Qs[j];
                    }
                    const float rr = fmaxf(__fsub_rn(p_of(j), qratio(qv, t_i)), 0.f);
                    P[j] = rr;
                    zl.add(rr);
                }
            }
            reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, zl.value(), 0ull);
            const double Z = sh.res.z;
            if (!(Z > 0.0)) {  // no residual mass (rounding only): the node's target row
                W.stage_target(trow, nullptr);
                __syncthreads();
                final_tok = W.draw_logits(u, [&](int j, int) { return P[j]; });
                break;
            }
            if (threadIdx.x == 0) {
                sh.zs[i] = (float)Z;
                sh.ts[i] = t_i;
            }
            __syncthreads();
            t -= (double)Qy;
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

// Cluster size and chunk-aligned slice for a vocabulary: enough CTAs to spread a row, and
// the two fp32 slices must fit in shared memory.
int pick_cluster(int V, int *slice_out, size_t *smem_out) {
    int cs = V >= 32768 ? 8 : V >= 8192 ? 4 : V >= 2048 ? 2 : 1;
    for (;;) {
        int slice = (V + cs - 1) / cs;
        slice = (slice + kChunk - 1) / kChunk * kChunk;
        const size_t smem = 2 * (size_t)slice * sizeof(float);
        if (smem <= kSmemLimit) {
            *slice_out = slice;
            *smem_out = smem;
            return cs;
        }
        if (cs == 16) return -1;
        cs *= 2;
    }
}

template <typename T>
cudaError_t launch_rrs_t(VerifyArgs a, int B, cudaStream_t s) {
    int slice = 0;
    size_t smem = 0;
    const int cs = pick_cluster(a.V, &slice, &smem);
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
