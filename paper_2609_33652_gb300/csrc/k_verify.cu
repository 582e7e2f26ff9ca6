// Tree verification by recursive rejection sampling for WoR candidates (Sec. 2.3 Eq.
// rs-overlap; App. A), lossless on the frozen topology (Prop. 1).
//
// One thread-block cluster per tree; CTA r of the cluster owns the vocabulary slice
// [r*slice, (r+1)*slice) and keeps that slice of the current node's target row and q row in
// shared memory, so every pass after the first reads shared memory, not L2/HBM. Scalars
// (log-normalisers, residual masses, argmax keys) are combined across the cluster through
// distributed shared memory: each CTA publishes its partial, the cluster barrier orders the
// writes, and every CTA combines all partials in rank order, so all CTAs hold bitwise
// identical values and take identical decisions.
//
// Walk at node u with children y_1..y_m (slot order), P = softmax(target row u),
// Q = softmax(q row of u), t = 1:
//   slot i: p' = P_i(y_i), q' = Q(y_i)/t_i; accept iff U * q' < p';
//           on reject R(v) = max(P_i(v) - Q(v)/t_i, 0), Z = sum R, P_{i+1} = R / Z,
//           t_{i+1} = t_i - Q(y_i). A rejected token has P_{i+1} = 0 from then on, so the
//           explicit exclusion of drawn tokens from Q is implied by the residual.
//   P_i(v) is recomputed per element from P_0(v), Q(v) and the stored (t_j, Z_j), j < i.
// All children rejected -> final token = argmax_v log R(v) + G(U_v); leaf -> bonus token =
// argmax_v x_v + G(U_v); Z = 0 (underflow only) -> argmax_v log P_i(v) + G(U_v).
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

// P_i(v) from P_0(v), Q(v) and the first i rejections.
__device__ __forceinline__ float resid_chain(float p, float q, const float *zs, const float *ts, int i) {
    for (int j = 0; j < i; ++j) {
        p = fmaxf(__fsub_rn(p, qratio(q, ts[j])), 0.f);
        p = __fdiv_rn(p, zs[j]);
    }
    return p;
}

// exp(x*invT - LSE) with LSE = hi + lo
__device__ __forceinline__ float prob_of(float z, float invT, float hi, float lo) {
    return expf(__fsub_rn(__fsub_rn(__fmul_rn(z, invT), hi), lo));
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

// Copy this CTA's slice of a row into shared memory.
template <typename T>
__device__ __forceinline__ void stage(const T *row, T *dst, int lo, int n, int V) {
    const int groups = (n + 7) >> 3;
    for (int g = threadIdx.x; g < groups; g += kThreads) {
        const int v0 = lo + 8 * g;
        if (v0 + 8 <= V) {
            if (sizeof(T) == 2) {
                reinterpret_cast<uint4 *>(dst)[g] = __ldg(reinterpret_cast<const uint4 *>(row + v0));
            } else {
                const float4 *src = reinterpret_cast<const float4 *>(row + v0);
                reinterpret_cast<float4 *>(dst)[2 * g] = __ldg(src);
                reinterpret_cast<float4 *>(dst)[2 * g + 1] = __ldg(src + 1);
            }
        } else {
            for (int i = 0; i < 8; ++i)
                if (v0 + i < V) dst[8 * g + i] = row[v0 + i];
        }
    }
}

template <typename T>
__device__ __forceinline__ float as_f32(T v);
template <>
__device__ __forceinline__ float as_f32<float>(float v) {
    return v;
}
template <>
__device__ __forceinline__ float as_f32<__nv_bfloat16>(__nv_bfloat16 v) {
    return __uint_as_float((uint32_t)__bfloat16_as_ushort(v) << 16);
}

enum PassKind { kBonus = 0, kResidualArgmax = 1, kTargetArgmax = 2 };

// Gumbel-max over this CTA's slice; returns the thread's best packed key.
// kind = kBonus: keys x_v + G; otherwise keys log w(v) + G with w = R_{i+1} (residual after
// rejecting slot i, unnormalised) or w = P_i (current target law).
template <typename T>
__device__ unsigned long long gumbel_pass(const VerifyArgs &a, const T *xt_s, const T *xq_s, int lo, int n, int b,
                                          int node, int kind, int i, float t_i, float lt_hi, float lt_lo,
                                          float lq_hi, float lq_lo, const float *zs, const float *ts) {
    unsigned long long best = 0ull;
    const int groups = (n + 7) >> 3;
    for (int g = threadIdx.x; g < groups; g += kThreads) {
        const int v0 = lo + 8 * g;
        const Words4 w0 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)(v0 >> 2) + 1u);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int v = v0 + k;
            if (v >= a.V) break;
            const float G = gumbel_of(k < 4 ? w0.w[k] : w1.w[k - 4]);
            const float zt = as_f32(xt_s[8 * g + k]);
            float key;
            if (kind == kBonus) {
                key = __fadd_rn(__fmul_rn(zt, a.invT), G);
            } else {
                const float P0 = prob_of(zt, a.invT, lt_hi, lt_lo);
                const float Q = prob_of(as_f32(xq_s[8 * g + k]), a.invT, lq_hi, lq_lo);
                float w = resid_chain(P0, Q, zs, ts, i);
                if (kind == kResidualArgmax) w = fmaxf(__fsub_rn(w, qratio(Q, t_i)), 0.f);
                if (!(w > 0.f)) continue;
                key = __fadd_rn(logf(w), G);
            }
            const unsigned long long pk = pack_key(key, (uint32_t)v);
            best = pk > best ? pk : best;
        }
    }
    return best;
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_verify_rrs(VerifyArgs a) {
    extern __shared__ __align__(16) unsigned char dyn[];
    T *xt_s = reinterpret_cast<T *>(dyn);
    T *xq_s = xt_s + a.slice;
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
        const T *qrow = nullptr;
        int r = -1;
        if (m > 0) {
            r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : a.depth[(int64_t)b * NN + u];
            if (r < 0 || r >= a.q_R) {
                bad = true;
                break;
            }
            qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;
        }
        __syncthreads();
        stage<T>(trow, xt_s, lo, n, a.V);
        if (m > 0) stage<T>(qrow, xq_s, lo, n, a.V);
        __syncthreads();

        if (m == 0) {  // leaf: bonus token from the node's target row
            const unsigned long long k =
                gumbel_pass<T>(a, xt_s, xq_s, lo, n, b, u, kBonus, 0, 0.f, 0.f, 0.f, 0.f, 0.f, sh.zs, sh.ts);
            reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, k);
            final_tok = (int)key_id(sh.res.key);
            break;
        }

        // log-normalisers: target row from the staged slice, q row from its chunk statistics
        float m1 = -INFINITY, m2 = -INFINITY;
        const int groups = (n + 7) >> 3;
        for (int g = threadIdx.x; g < groups; g += kThreads)
            for (int k = 0; k < 8 && lo + 8 * g + k < a.V; ++k)
                m1 = fmaxf(m1, __fmul_rn(as_f32(xt_s[8 * g + k]), a.invT));
        KahanF s1;
        if (m1 != -INFINITY)
            for (int g = threadIdx.x; g < groups; g += kThreads)
                for (int k = 0; k < 8 && lo + 8 * g + k < a.V; ++k)
                    s1.add(expf(__fsub_rn(__fmul_rn(as_f32(xt_s[8 * g + k]), a.invT), m1)));
        const float2 *st = a.qstats + ((int64_t)b * a.q_R + r) * a.C;
        for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads) m2 = fmaxf(m2, st[c].x);
        KahanF s2;
        if (m2 != -INFINITY)
            for (int c = crank * kThreads + threadIdx.x; c < a.C; c += CS * kThreads)
                s2.add(st[c].y * expf(st[c].x - m2));
        reduce_round(sh, par, cluster, m1, s1.value(), m2, s2.value(), 0.0, 0ull);
        const float lt_hi = sh.res.hi1, lt_lo = sh.res.lo1, lq_hi = sh.res.hi2, lq_lo = sh.res.lo2;

        double t = 1.0;
        int accepted = -1;
        for (int i = 0; i < m; ++i) {
            const int c = kids[i];
            const int y = (c >= 1 && c <= a.N) ? tok[c] : -1;
            if (y < 0 || y >= a.V) {
                bad = true;
                break;
            }
            const float t_i = (float)t;
            const float P0 = prob_of(Logit<T>::load1(trow, y), a.invT, lt_hi, lt_lo);
            const float Qy = prob_of(Logit<T>::load1(qrow, y), a.invT, lq_hi, lq_lo);
            const float pp = resid_chain(P0, Qy, sh.zs, sh.ts, i);
            const float qp = qratio(Qy, t_i);
            const float U = uniform_of(draw_word(a.seed, kAccept, (uint32_t)b, (uint32_t)c, 0u));
            if (__fmul_rn(U, qp) < pp) {
                accepted = c;
                break;
            }
            if (i == m - 1) {  // every slot rejected: final token from the last residual
                const unsigned long long k = gumbel_pass<T>(a, xt_s, xq_s, lo, n, b, u, kResidualArgmax, i, t_i,
                                                            lt_hi, lt_lo, lq_hi, lq_lo, sh.zs, sh.ts);
                reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, k);
                final_tok = (int)key_id(sh.res.key);
                break;
            }
            // residual mass after rejecting slot i
            KahanF zloc;
            for (int g = threadIdx.x; g < groups; g += kThreads)
                for (int k = 0; k < 8 && lo + 8 * g + k < a.V; ++k) {
                    const float P0v = prob_of(as_f32(xt_s[8 * g + k]), a.invT, lt_hi, lt_lo);
                    const float Qv = prob_of(as_f32(xq_s[8 * g + k]), a.invT, lq_hi, lq_lo);
                    zloc.add(fmaxf(__fsub_rn(resid_chain(P0v, Qv, sh.zs, sh.ts, i), qratio(Qv, t_i)), 0.f));
                }
            reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, zloc.value(), 0ull);
            const double Z = sh.res.z;
            if (!(Z > 0.0)) {  // underflow only: draw from the current target law
                const unsigned long long k = gumbel_pass<T>(a, xt_s, xq_s, lo, n, b, u, kTargetArgmax, i, t_i,
                                                            lt_hi, lt_lo, lq_hi, lq_lo, sh.zs, sh.ts);
                reduce_round(sh, par, cluster, -INFINITY, 0.0, -INFINITY, 0.0, 0.0, k);
                final_tok = (int)key_id(sh.res.key);
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

int pick_cluster(int V, int elem_bytes, int *slice_out, size_t *smem_out) {
    int cs = V >= 32768 ? 8 : V >= 8192 ? 4 : V >= 2048 ? 2 : 1;
    for (;;) {
        int slice = (V + cs - 1) / cs;
        slice = (slice + 7) & ~7;
        const size_t smem = 2 * (size_t)slice * elem_bytes;
        if (smem <= 200 * 1024 || cs == 16) {
            *slice_out = slice;
            *smem_out = smem;
            return smem <= 200 * 1024 ? cs : -1;
        }
        cs *= 2;
    }
}

template <typename T>
cudaError_t launch_rrs_t(VerifyArgs a, int B, cudaStream_t s) {
    int slice = 0;
    size_t smem = 0;
    const int cs = pick_cluster(a.V, (int)sizeof(T), &slice, &smem);
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
