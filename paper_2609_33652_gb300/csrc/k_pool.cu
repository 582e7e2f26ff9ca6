// Pooled draft laws (Sec. 3.1 and 3.2: a position's draft law is restricted to its P most
// probable tokens and normalised within them; Sec. 3.3: verification uses those pooled
// probabilities, while the target law and the residual stay full-vocabulary). P <= 64, so a
// pool is one warp, lane j holding pool tokens j and j + 32.
//
//   k_pool_finish     first pass: from the rows' top-P lists (the pools), the pooled
//                     log-normaliser and the K candidates the max-heap expands.
//   k_replay_pooled   one warp per parent: the m_u ordered WoR draws are the top-m_u Gumbel
//                     keys x_v + G(U[replay element, u, v]) over the pool tokens.
//   k_verify_pooled   one CTA per tree walks the tree. With q zero outside the pool, every
//                     residual equals the target law outside the pool up to one scale factor,
//                     so a visited node needs one streaming pass over its target row (chunk
//                     statistics: the log-normaliser, the chunk masses), the pool's point
//                     values, and the target mass outside the pool; the sibling tests and the
//                     residual updates then run in one warp on the P pool entries plus that
//                     scale. A final token from the residual, or a bonus token, is the
//                     two-level Gumbel-max draw over chunk masses built from the same pieces.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kMaxPool = 64;

// ---------------------------------------------------------------------------------------
struct FinishArgs {
    const void *draft;
    int64_t bstride, rstride;
    int rows, L, K, P;
    float invT;
    const int32_t *pool_ids;  // [B*L][P]
    float2 *lse;              // [B*L]
    float *topk_x;            // [B*L][K]
    int32_t *topk_id;         // [B*L][K]
    uint32_t *status;
};

template <typename T>
__global__ void __launch_bounds__(128) k_pool_finish(FinishArgs a) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int row = blockIdx.x * 4 + (threadIdx.x >> 5);
    if (row >= a.rows) return;  // uniform over the warp
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const T *rp = static_cast<const T *>(a.draft) + (int64_t)b * a.bstride + (int64_t)d * a.rstride;
    float x = -INFINITY, x1 = -INFINITY;
    int v = -1;
    if (lane < a.P) {
        v = a.pool_ids[(int64_t)row * a.P + lane];
        x = __fmul_rn(Logit<T>::load1(rp, v), a.invT);
    }
    if (lane + 32 < a.P) x1 = __fmul_rn(Logit<T>::load1(rp, a.pool_ids[(int64_t)row * a.P + lane + 32]), a.invT);
    const MaxSum ms = warp_maxsum(maxsum_merge(MaxSum{x, FF{lane < a.P ? 1.f : 0.f, 0.f}},
                                               MaxSum{x1, FF{lane + 32 < a.P ? 1.f : 0.f, 0.f}}));
    if (lane == 0) {
        const FF l = maxsum_lse(ms);
        a.lse[row] = make_float2(l.hi, l.lo);
    }
    if (lane < a.K) {  // the pool is sorted by (x desc, id asc): its first K are the candidates
        a.topk_x[(int64_t)row * a.K + lane] = x;
        a.topk_id[(int64_t)row * a.K + lane] = v;
    }
}

// ---------------------------------------------------------------------------------------
struct ReplayPoolArgs {
    const void *q;
    int64_t bstride, rstride;
    int R, V, B, N, L, P;
    float invT;
    uint64_t seed;
    const int32_t *qrow_of_node, *depth, *child_off, *child_ids, *pool_ids;
    int32_t *token;
    uint32_t *status;
};

template <typename T>
__global__ void __launch_bounds__(128) k_replay_pooled(ReplayPoolArgs a) {
    pdl_begin();
    const int lane = threadIdx.x & 31;
    const int NN = a.N + 1;
    const int64_t node = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    if (node >= (int64_t)a.B * NN) return;  // uniform over the warp
    const int b = (int)(node / NN), u = (int)(node - (int64_t)b * NN);
    if (u == 0 && lane == 0) a.token[(int64_t)b * NN] = -1;
    const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
    const int o = off[u], m = off[u + 1] - o;
    if (m <= 0) return;
    const int d = a.depth[node];
    const int r = a.qrow_of_node ? a.qrow_of_node[node] : d;
    if (m > a.P || o < 0 || o + m > a.N || d < 0 || d >= a.L || r < 0 || r >= a.R) {
        if (lane == 0) raise_status(a.status, kDevBadTree | kDevBadIndex);
        return;
    }
    const T *row = static_cast<const T *>(a.q) + (int64_t)b * a.bstride + (int64_t)r * a.rstride;
    uint64_t key[2] = {0ull, 0ull};  // pool entries lane and lane + 32
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int j = lane + 32 * h;
        if (j >= a.P) continue;
        const int v = a.pool_ids[((int64_t)b * a.L + d) * a.P + j];
        if (v >= 0 && v < a.V) {
            const float g = __fadd_rn(__fmul_rn(Logit<T>::load1(row, v), a.invT),
                                      gumbel_of(draw_word(a.seed, kReplayElem, (uint32_t)b, (uint32_t)u, (uint32_t)v)));
            key[h] = pack_key(g, (uint32_t)v);
        } else {
            raise_status(a.status, kDevBadIndex);
        }
    }
    const int32_t *kids = a.child_ids + (int64_t)b * a.N + o;
    for (int s = 0; s < m; ++s) {  // the s-th largest key fills child slot s
        const uint64_t best = warp_max_u64(key[0] > key[1] ? key[0] : key[1]);
        if (key[0] == best) key[0] = 0ull;  // keys are distinct (token ids)
        if (key[1] == best) key[1] = 0ull;
        if (lane == 0) {
            const int child = kids[s];
            if (best != 0ull && child > 0 && child < NN)
                a.token[(int64_t)b * NN + child] = (int32_t)key_id(best);
            else
                raise_status(a.status, kDevBadTree);
        }
    }
}

// ---------------------------------------------------------------------------------------
constexpr int kVpThreads = 512;
constexpr int kVpWarps = kVpThreads / 32;

template <typename T>
struct VpUnit {  // chunks per warp iteration: eight (bf16) or four (fp32) 16-byte loads per lane
    static constexpr int n = sizeof(T) == 2 ? 8 : 4;
};

struct VerifyPoolArgs {
    const void *target;
    int64_t t_bstride, t_rstride;
    const void *q;
    int64_t q_bstride, q_rstride;
    int q_R, V, C, B, N, L, P;
    float invT;
    uint64_t seed;
    const int32_t *qrow_of_node, *depth, *child_off, *child_ids, *token, *pool_ids;
    int32_t *out_tokens, *out_nodes, *out_len;
    uint32_t *status;
};

struct VpShared {
    MaxSum wms[kVpWarps];
    FF wff[kVpWarps];
    unsigned long long wk[kVpWarps];
    int pool[kMaxPool];      // the node's pool tokens
    int dirty[kMaxPool];     // distinct chunks holding a pool token
    float dmass[kMaxPool];   // their target mass outside the pool (relative to the row normaliser)
    float rj[kMaxPool];      // final residual on the pool entries
    FF L2t;                  // row log-normaliser times log2(e)
    float mout;              // target mass outside the pool
    float scale;             // final residual outside the pool = scale * p(v)
    int ndirty, next, mode;  // mode: 0 accepted, 1 residual draw, 2 target-row draw
};

__device__ __forceinline__ int find_dirty(const VpShared &sh, int c) {
    int e = -1;
    for (int k = 0; k < sh.ndirty; ++k) e = sh.dirty[k] == c ? k : e;
    return e;
}

// Two-level draw at node u: chunk keys log(mass_c) + G(U[final chunk, u, c]) over the chunks
// with mass, the best by (key desc, c asc), then log(w_v) + G(U[final, u, v]) inside it. From
// the target row (RESID false: mass_c = exp(A_c), A_c from the chunk statistics) or from the
// residual (pool entries rj, elsewhere scale * p(v)). All threads call it; returns the token.
template <bool RESID, typename T>
__device__ int pooled_draw(const VerifyPoolArgs &a, VpShared &sh, const float2 *cst, const T *trow, int b, int u) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned long long best = 0ull;
    for (int c = threadIdx.x; c < a.C; c += kVpThreads) {
        const float2 st = cst[c];
        float A;
        if (!RESID) {
            A = __fadd_rn(st.x, logf(st.y));
        } else {
            const int e = find_dirty(sh, c);
            float mass;
            if (e < 0) {
                mass = __fmul_rn(sh.scale, __fmul_rn(st.y, exp_shifted(st.x, sh.L2t)));
            } else {
                mass = __fmul_rn(sh.scale, sh.dmass[e]);
                for (int j = 0; j < a.P; ++j)
                    if (sh.pool[j] / kChunk == c) mass += sh.rj[j];
            }
            A = mass > 0.f ? logf(mass) : -INFINITY;
        }
        if (A != -INFINITY) {
            const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)u, (uint32_t)c);
            const unsigned long long k = pack_key(__fadd_rn(A, gumbel_of(w)), (uint32_t)c);
            best = k > best ? k : best;
        }
    }
    best = warp_max_u64(best);
    if (lane == 0) sh.wk[warp] = best;
    __syncthreads();
    const unsigned long long cb = warp_max_u64(lane < kVpWarps ? sh.wk[lane] : 0ull);
    __syncthreads();  // every warp has read sh.wk
    int tok = -1;
    if (warp == 0 && cb != 0ull) {
        const int v0 = (int)key_id(cb) * kChunk + lane * 8;
        float x[8];
        Logit<T>::load8(trow, v0, a.V, x);
        const Words4 w0 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)u, (uint32_t)(v0 >> 2));
        const Words4 w1 = draw_block(a.seed, kFinal, (uint32_t)b, (uint32_t)u, (uint32_t)(v0 >> 2) + 1u);
        unsigned long long tk = 0ull;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int v = v0 + e;
            if (v >= a.V) continue;
            const float xv = __fmul_rn(x[e], a.invT);
            float l = xv;
            if (RESID) {
                int j = -1;
                for (int k = 0; k < a.P; ++k) j = sh.pool[k] == v ? k : j;
                const float w = j >= 0 ? sh.rj[j] : __fmul_rn(sh.scale, exp_shifted(xv, sh.L2t));
                if (!(w > 0.f)) continue;
                l = logf(w);
            }
            const float key = __fadd_rn(l, gumbel_of(e < 4 ? w0.w[e] : w1.w[e - 4]));
            const unsigned long long k = pack_key(key, (uint32_t)v);
            tk = k > tk ? k : tk;
        }
        tk = warp_max_u64(tk);
        tok = tk != 0ull ? (int)key_id(tk) : -1;
    }
    return tok;  // valid in warp 0
}

template <typename T>
__global__ void __launch_bounds__(kVpThreads) k_verify_pooled(VerifyPoolArgs a) {
    pdl_begin();
    constexpr int U = VpUnit<T>::n;
    __shared__ VpShared sh;
    extern __shared__ __align__(16) float2 cst[];  // [C] chunk statistics of the current target row
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int b = blockIdx.x, NN = a.N + 1;
    const int32_t *off = a.child_off + (int64_t)b * (NN + 1), *ids = a.child_ids + (int64_t)b * a.N;
    int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1), *onode = a.out_nodes + (int64_t)b * a.L;
    int u = 0, nacc = 0, final_tok = -1;
    for (int step = 0; step <= a.L; ++step) {  // the depth grows by one per accepted node
        const T *trow = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
        // 1. chunk statistics of target row u (U chunks per warp iteration, loads first)
        const int units = (a.C + U - 1) / U;
        for (int un0 = warp; un0 < units; un0 += kVpWarps) {  // uniform over the warp
            const int cu = un0 * U;
            RawGroup<T> raw[U];
#pragma unroll
            for (int k = 0; k < U; ++k)
                if (cu + k < a.C) raw[k].load(trow, (cu + k) * kChunk + lane * 8, a.V);
            float mcs[U], part[U];
#pragma unroll
            for (int k = 0; k < U; ++k) {
                mcs[k] = -INFINITY;
                part[k] = 0.f;
                if (cu + k >= a.C) continue;  // uniform over the warp
                float z[8];
                raw[k].unpack(z);
                float zm = z[0];
#pragma unroll
                for (int e = 1; e < 8; ++e) zm = fmaxf(zm, z[e]);
                mcs[k] = __fmul_rn(warp_max(zm), a.invT);
                const float2 offs = exp_offset(mcs[k]);
#pragma unroll
                for (int e = 0; e < 8; ++e) part[k] += chunk_term(z[e], a.invT, offs.x);
                part[k] = chunk_sum_fix(part[k], offs.y);
            }
            const float sm = warp_multi_sum<U>(part);
            const int ch = multi_sum_index<U>(lane), c = cu + ch;
            if (lane % (32 / U) == 0 && c < a.C) {
                float mc = mcs[0];
#pragma unroll
                for (int k = 1; k < U; ++k) mc = ch == k ? mcs[k] : mc;
                if (!(sm == sm) || isinf(mc)) raise_status(a.status, kDevNonFinite);
                cst[c] = make_float2(mc, sm);
            }
        }
        __syncthreads();
        // 2. the row's log-normaliser
        {
            MaxSum acc{-INFINITY, FF{0.f, 0.f}};
            for (int c = threadIdx.x; c < a.C; c += kVpThreads)
                acc = maxsum_merge(acc, MaxSum{cst[c].x, FF{cst[c].y, 0.f}});
            acc = warp_maxsum(acc);
            if (lane == 0) sh.wms[warp] = acc;
            __syncthreads();
            if (warp == 0) {
                const MaxSum t = warp_maxsum(lane < kVpWarps ? sh.wms[lane] : MaxSum{-INFINITY, FF{0.f, 0.f}});
                if (lane == 0) sh.L2t = ff_times_log2e(maxsum_lse(t));
            }
            __syncthreads();
        }
        const int o = off[u], m = off[u + 1] - o;
        if (m <= 0 || o < 0 || o + m > a.N) {  // a leaf: the bonus token from the target row
            if (m != 0 && threadIdx.x == 0) raise_status(a.status, kDevBadTree);
            final_tok = pooled_draw<false, T>(a, sh, cst, trow, b, u);
            break;
        }
        // 3. the pool: tokens, target and q point values (warp 0), dirty chunks
        const int d = a.depth[(int64_t)b * NN + u];
        const int r = a.qrow_of_node ? a.qrow_of_node[(int64_t)b * NN + u] : d;
        const bool bad = d < 0 || d >= a.L || r < 0 || r >= a.q_R || m > a.P;  // uniform
        if (bad) {
            if (threadIdx.x == 0) raise_status(a.status, kDevBadIndex);
            final_tok = -1;
            break;
        }
        float P0[2] = {0.f, 0.f}, Q[2] = {0.f, 0.f};  // warp 0, lane j: pool entries j and j + 32
        if (warp == 0) {
            const T *qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;
            float xt[2] = {-INFINITY, -INFINITY}, xq[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int j = lane + 32 * h;
                if (j >= a.P) continue;
                int v = a.pool_ids[((int64_t)b * a.L + d) * a.P + j];
                if (v < 0 || v >= a.V) {
                    raise_status(a.status, kDevBadIndex);
                    v = 0;
                }
                xt[h] = __fmul_rn(Logit<T>::load1(trow, v), a.invT);
                xq[h] = __fmul_rn(Logit<T>::load1(qrow, v), a.invT);
                sh.pool[j] = v;
            }
            __syncwarp();  // sh.pool is read by lane 0 below
            const MaxSum mq = warp_maxsum(maxsum_merge(MaxSum{xq[0], FF{lane < a.P ? 1.f : 0.f, 0.f}},
                                                       MaxSum{xq[1], FF{lane + 32 < a.P ? 1.f : 0.f, 0.f}}));
            const FF L2q = ff_times_log2e(maxsum_lse(mq));
#pragma unroll
            for (int h = 0; h < 2; ++h)
                if (lane + 32 * h < a.P) {
                    P0[h] = exp_shifted(xt[h], sh.L2t);
                    Q[h] = exp_shifted(xq[h], L2q);
                }
            if (lane == 0) {  // distinct chunks of the pool tokens
                int n = 0;
                for (int j = 0; j < a.P; ++j) {
                    const int c = sh.pool[j] / kChunk;
                    bool seen = false;
                    for (int e = 0; e < n; ++e) seen |= sh.dirty[e] == c;
                    if (!seen) sh.dirty[n++] = c;
                }
                sh.ndirty = n;
            }
        }
        __syncthreads();
        // 4. the target mass outside the pool: whole chunks from their statistics, the chunks
        //    holding pool tokens element by element
        {
            KahanF acc;
            for (int c = threadIdx.x; c < a.C; c += kVpThreads)
                if (find_dirty(sh, c) < 0) acc.add(__fmul_rn(cst[c].y, exp_shifted(cst[c].x, sh.L2t)));
            for (int e = warp; e < sh.ndirty; e += kVpWarps) {  // uniform over the warp
                const int v0 = sh.dirty[e] * kChunk + lane * 8;
                float x[8];
                Logit<T>::load8(trow, v0, a.V, x);
                float s = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int v = v0 + k;
                    bool in_pool = false;
                    for (int j = 0; j < a.P; ++j) in_pool |= sh.pool[j] == v;
                    if (v < a.V && !in_pool) s += exp_shifted(__fmul_rn(x[k], a.invT), sh.L2t);
                }
                s = warp_sum(s);
                if (lane == 0) {
                    sh.dmass[e] = s;
                    acc.add(s);
                }
            }
            const FF part = warp_sum_ff(acc.ff());
            if (lane == 0) sh.wff[warp] = part;
            __syncthreads();
            if (warp == 0) {
                const FF t = warp_sum_ff(lane < kVpWarps ? sh.wff[lane] : FF{0.f, 0.f});
                if (lane == 0) sh.mout = __fadd_rn(t.hi, t.lo);
            }
            __syncthreads();
        }
        // 5. the sibling tests on the pool entries (warp 0): lane j holds the current law on
        //    pool entry j; outside the pool the law is the target's times out / mout
        if (warp == 0) {
            float cur[2] = {lane < a.P ? P0[0] : 0.f, lane + 32 < a.P ? P0[1] : 0.f}, out = sh.mout, t = 1.f;
            bool drawn[2] = {false, false};
            int mode = 0, next = -1;
            for (int i = 0; i < m; ++i) {
                const int c = ids[o + i];
                if (c < 1 || c > a.N) {
                    if (lane == 0) raise_status(a.status, kDevBadIndex);
                    mode = 2;
                    break;
                }
                const int y = a.token[(int64_t)b * NN + c];
                __syncwarp();
                const unsigned hit0 = __ballot_sync(kFull, lane < a.P && sh.pool[lane] == y);
                const unsigned hit1 = __ballot_sync(kFull, lane + 32 < a.P && sh.pool[lane + 32] == y);
                const int k = hit0 ? __ffs(hit0) - 1 : (hit1 ? 32 + __ffs(hit1) - 1 : -1);
                // (k is uniform over the warp: every lane takes the same branch)
                float qk = 0.f, pk = 0.f;
                if (k >= 0) {
                    const float q0 = __shfl_sync(kFull, Q[0], k & 31), q1 = __shfl_sync(kFull, Q[1], k & 31);
                    const float c0 = __shfl_sync(kFull, cur[0], k & 31), c1 = __shfl_sync(kFull, cur[1], k & 31);
                    qk = k < 32 ? q0 : q1;
                    pk = k < 32 ? c0 : c1;
                } else if (y >= 0 && y < a.V && sh.mout > 0.f) {  // outside the pool: q = 0
                    const float py = exp_shifted(__fmul_rn(Logit<T>::load1(trow, y), a.invT), sh.L2t);
                    pk = __fmul_rn(__fdiv_rn(out, sh.mout), py);
                }
                const float qp = qk > 0.f && t > 0.f ? __fdiv_rn(qk, t) : 0.f;
                const float U = uniform_of(draw_word(a.seed, kAccept, (uint32_t)b, (uint32_t)c, 0u));
                if (__fmul_rn(U, qp) < pk) {  // accept
                    next = c;
                    break;
                }
                // reject: R = max(cur - [not drawn] Q / t, 0) on the pool, unchanged outside
                float Rr[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const float qt = t > 0.f ? __fdiv_rn(Q[h], t) : 0.f;
                    Rr[h] = lane + 32 * h < a.P ? fmaxf(__fsub_rn(cur[h], drawn[h] ? 0.f : qt), 0.f) : 0.f;
                }
                const float Z = __fadd_rn(warp_sum(__fadd_rn(Rr[0], Rr[1])), out);
                if (!(Z > 0.f)) {  // no residual mass (rounding only): draw from the target row
                    mode = 2;
                    break;
                }
                if (i == m - 1) {  // every slot rejected: draw from the residual R
#pragma unroll
                    for (int h = 0; h < 2; ++h)
                        if (lane + 32 * h < a.P) sh.rj[lane + 32 * h] = Rr[h];
                    if (lane == 0) sh.scale = sh.mout > 0.f ? __fdiv_rn(out, sh.mout) : 0.f;
                    mode = 1;
                    break;
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    cur[h] = __fdiv_rn(Rr[h], Z);
                    drawn[h] |= lane + 32 * h == k;
                }
                out = __fdiv_rn(out, Z);
                t = __fsub_rn(t, qk);
            }
            if (lane == 0) {
                sh.next = next;
                sh.mode = next >= 0 ? 0 : mode;
            }
        }
        __syncthreads();
        const int mode = sh.mode, next = sh.next;
        __syncthreads();  // every thread has read the decision
        if (mode == 0 && nacc < a.L) {
            if (threadIdx.x == 0) {
                otok[nacc] = a.token[(int64_t)b * NN + next];
                onode[nacc] = next;
            }
            ++nacc;
            u = next;
            continue;
        }
        final_tok = mode == 1 ? pooled_draw<true, T>(a, sh, cst, trow, b, u)
                              : pooled_draw<false, T>(a, sh, cst, trow, b, u);
        break;
    }
    if (threadIdx.x == 0) {
        for (int k = nacc + 1; k <= a.L; ++k) otok[k] = -1;
        for (int k = nacc; k < a.L; ++k) onode[k] = -1;
        otok[nacc] = final_tok;
        a.out_len[b] = nacc + 1;
    }
}

// ---------------------------------------------------------------------------------------
// Pools of P = 33..64 tokens (the first pass's per-row top-P above the 32 the top-K pass of
// the first pass keeps): one CTA per draft row, exact (x desc, id asc) through the unique
// 64-bit keys pack_key(x, id). tau = the P-th largest chunk maximum (a bitonic sort of the
// row's chunk keys from its statistics) bounds the P-th largest logit from below, so the
// pool is among the logits >= tau of the chunks whose maximum reaches tau. Those keys are
// collected into shared memory and sorted; when more than kSelCap of them reach tau (flat
// rows, heavy ties), a most-significant-digit radix pass over the keys (8 bits at a time,
// counting only keys above the current threshold) first raises the threshold to the top of
// the digit bucket that holds the P-th key, until at most kSelCap keys remain.
constexpr int kSelThreads = 256;
constexpr int kSelCap = 4096;  // candidate keys held in shared memory

struct SelectArgs {
    const void *draft;
    int64_t bstride, rstride;
    const float2 *stats;  // [B][R][C]
    int R, L, C, V, P;
    float invT;
    int32_t *pool_ids;  // [B*L][P]
};

// Bitonic sort of keys[0, m) into descending order (m a power of two, empty slots hold 0).
__device__ void bitonic_desc(uint64_t *keys, int m) {
    for (int k = 2; k <= m; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < m; i += kSelThreads) {
                const int ixj = i ^ j;
                if (ixj > i) {
                    const uint64_t x = keys[i], y = keys[ixj];
                    if ((i & k) == 0 ? x < y : x > y) {
                        keys[i] = y;
                        keys[ixj] = x;
                    }
                }
            }
            __syncthreads();
        }
}

struct SelShared {
    int n, nch, sel;
    unsigned long long prefix, mask, above, cnt;
    int hist[256];
};

// Calls f(key) for every logit of the row whose key is >= thr (one warp per chunk whose
// maximum reaches the threshold's value). All threads call it; ends with a barrier.
template <typename T, typename F>
__device__ void for_keys_above(const SelectArgs &a, const T *row, const float2 *st, int *chunks, SelShared &sh,
                               uint64_t thr, F f) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int NW = kSelThreads / 32;
    if (threadIdx.x == 0) sh.nch = 0;
    __syncthreads();
    const uint32_t hi = (uint32_t)(thr >> 32);
    for (int c = threadIdx.x; c < a.C; c += kSelThreads)
        if (ord_f32(st[c].x) >= hi) {
            const int pos = atomicAdd(&sh.nch, 1);
            if (in_bounds(pos, a.C, nullptr)) chunks[pos] = c;
        }
    __syncthreads();
    const int nch = sh.nch;
    for (int i = warp; i < nch; i += NW) {
        const int v0 = chunks[i] * kChunk + lane * 8;
        float x[8];
        Logit<T>::load8(row, v0, a.V, x);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (v0 + e >= a.V) continue;
            const uint64_t key = pack_key(__fmul_rn(x[e], a.invT), (uint32_t)(v0 + e));
            if (key >= thr) f(key);
        }
    }
    __syncthreads();
}

template <typename T>
__global__ void __launch_bounds__(kSelThreads) k_pool_select(SelectArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) unsigned char smem[];
    uint64_t *keys = reinterpret_cast<uint64_t *>(smem);           // [kSelCap]
    float2 *st = reinterpret_cast<float2 *>(keys + kSelCap);        // [C]
    int *chunks = reinterpret_cast<int *>(st + a.C);                // [C]
    __shared__ SelShared sh;
    const int row = blockIdx.x;
    const int b = row / a.L, d = row - (row / a.L) * a.L;
    const T *rp = static_cast<const T *>(a.draft) + (int64_t)b * a.bstride + (int64_t)d * a.rstride;
    const float2 *gst = a.stats + ((int64_t)b * a.R + d) * a.C;
    for (int c = threadIdx.x; c < a.C; c += kSelThreads) st[c] = __ldg(&gst[c]);
    int mc = 1;
    while (mc < a.C) mc <<= 1;  // <= kSelCap: C <= TSB_MAX_V / 256 = 1600
    __syncthreads();
    // 1. tau from the P-th largest chunk key
    for (int i = threadIdx.x; i < mc; i += kSelThreads) keys[i] = i < a.C ? pack_key(st[i].x, (uint32_t)i) : 0ull;
    __syncthreads();
    bitonic_desc(keys, mc);
    uint64_t thr = a.C >= a.P ? (keys[a.P - 1] >> 32) << 32 : 0ull;  // every key of x >= tau
    __syncthreads();
    // 2. the keys above the threshold, raising it first if more than kSelCap reach it
    for (int round = 0; round < 2; ++round) {
        if (threadIdx.x == 0) sh.n = 0;
        __syncthreads();
        for_keys_above<T>(a, rp, st, chunks, sh, thr, [&](uint64_t k) {
            const int i = atomicAdd(&sh.n, 1);
            if (i < kSelCap) keys[i] = k;
        });
        if (sh.n <= kSelCap) break;  // uniform: read after the barrier that ends the scan
        if (threadIdx.x == 0) {
            sh.prefix = 0ull;
            sh.mask = 0ull;
            sh.above = 0ull;
            sh.cnt = ~0ull;
        }
        for (int shift = 56; shift >= 0; shift -= 8) {
            for (int i = threadIdx.x; i < 256; i += kSelThreads) sh.hist[i] = 0;
            __syncthreads();
            const uint64_t pre = sh.prefix, msk = sh.mask;
            for_keys_above<T>(a, rp, st, chunks, sh, thr, [&](uint64_t k) {
                if ((k & msk) == pre) atomicAdd(&sh.hist[(int)((k >> shift) & 255ull)], 1);
            });
            if (threadIdx.x == 0) {
                unsigned long long cum = 0ull;
                int bin = 0;
                for (int j = 255; j >= 0; --j) {
                    if (sh.above + cum + (unsigned long long)sh.hist[j] >= (unsigned long long)a.P) {
                        bin = j;
                        break;
                    }
                    cum += (unsigned long long)sh.hist[j];
                }
                sh.above += cum;
                sh.prefix |= (unsigned long long)bin << shift;
                sh.mask |= 0xFFull << shift;
                sh.cnt = sh.above + (unsigned long long)sh.hist[bin];
            }
            __syncthreads();
            if (sh.cnt <= (unsigned long long)kSelCap) break;  // uniform
        }
        thr = sh.prefix > thr ? sh.prefix : thr;
        __syncthreads();
    }
    // 3. the top P by (x desc, id asc)
    const int n = min(sh.n, kSelCap);
    int m = 1;
    while (m < n) m <<= 1;
    for (int i = n + threadIdx.x; i < m; i += kSelThreads) keys[i] = 0ull;
    __syncthreads();
    bitonic_desc(keys, m);
    for (int j = threadIdx.x; j < a.P; j += kSelThreads)
        a.pool_ids[(int64_t)row * a.P + j] = j < n ? (int32_t)key_id(keys[j]) : -1;
}

}  // namespace

cudaError_t launch_pool_finish(const RowsDesc &draft, int L, int K, int P, float invT, const int32_t *pool_ids,
                               float2 *lse, float *topk_x, int32_t *topk_id, uint32_t *status, cudaStream_t s) {
    FinishArgs a;
    a.draft = draft.data;
    a.bstride = draft.batch_stride;
    a.rstride = draft.row_stride;
    a.rows = draft.B * L;
    a.L = L;
    a.K = K;
    a.P = P;
    a.invT = invT;
    a.pool_ids = pool_ids;
    a.lse = lse;
    a.topk_x = topk_x;
    a.topk_id = topk_id;
    a.status = status;
    const dim3 grid((unsigned)((a.rows + 3) / 4));
    return draft.dtype == 1 ? launch_pdl(k_pool_finish<__nv_bfloat16>, grid, dim3(128), 0, s, 0, a)
                            : launch_pdl(k_pool_finish<float>, grid, dim3(128), 0, s, 0, a);
}

cudaError_t launch_pool_select(const RowsDesc &draft, const float2 *stats, int L, int P, float invT,
                               int32_t *pool_ids, cudaStream_t s) {
    SelectArgs a;
    a.draft = draft.data;
    a.bstride = draft.batch_stride;
    a.rstride = draft.row_stride;
    a.stats = stats;
    a.R = draft.R;
    a.L = L;
    a.C = num_chunks(draft.V);
    a.V = draft.V;
    a.P = P;
    a.invT = invT;
    a.pool_ids = pool_ids;
    if (a.C > kSelCap || P > kSelCap) return cudaErrorInvalidValue;
    const size_t smem = (size_t)kSelCap * sizeof(uint64_t) + (size_t)a.C * (sizeof(float2) + sizeof(int));
    const dim3 grid((unsigned)(draft.B * L));
    if (draft.dtype == 1) {
        cudaError_t e = cudaFuncSetAttribute(k_pool_select<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        return launch_pdl(k_pool_select<__nv_bfloat16>, grid, dim3(kSelThreads), smem, s, 0, a);
    }
    cudaError_t e = cudaFuncSetAttribute(k_pool_select<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_pool_select<float>, grid, dim3(kSelThreads), smem, s, 0, a);
}

cudaError_t launch_replay_pooled(const RowsDesc &q, const int32_t *qrow_of_node, int B, int N, int L, int P,
                                 const TreeDesc &tree, const int32_t *pool_ids, float invT, uint64_t seed,
                                 int32_t *token, uint32_t *status, cudaStream_t s) {
    ReplayPoolArgs a;
    a.q = q.data;
    a.bstride = q.batch_stride;
    a.rstride = q.row_stride;
    a.R = q.R;
    a.V = q.V;
    a.B = B;
    a.N = N;
    a.L = L;
    a.P = P;
    a.invT = invT;
    a.seed = seed;
    a.qrow_of_node = qrow_of_node;
    a.depth = tree.depth;
    a.child_off = tree.child_off;
    a.child_ids = tree.child_ids;
    a.pool_ids = pool_ids;
    a.token = token;
    a.status = status;
    const int64_t warps = (int64_t)B * (N + 1);
    if ((warps + 3) / 4 > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const dim3 grid((unsigned)((warps + 3) / 4));
    return q.dtype == 1 ? launch_pdl(k_replay_pooled<__nv_bfloat16>, grid, dim3(128), 0, s, 0, a)
                        : launch_pdl(k_replay_pooled<float>, grid, dim3(128), 0, s, 0, a);
}

cudaError_t launch_verify_pooled(const RowsDesc &target, const RowsDesc &q, const int32_t *qrow_of_node, int B,
                                 int N, int L, int P, const TreeDesc &tree, const int32_t *pool_ids,
                                 const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                 int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyPoolArgs a;
    a.target = target.data;
    a.t_bstride = target.batch_stride;
    a.t_rstride = target.row_stride;
    a.q = q.data;
    a.q_bstride = q.batch_stride;
    a.q_rstride = q.row_stride;
    a.q_R = q.R;
    a.V = target.V;
    a.C = num_chunks(target.V);
    a.B = B;
    a.N = N;
    a.L = L;
    a.P = P;
    a.invT = invT;
    a.seed = seed;
    a.qrow_of_node = qrow_of_node;
    a.depth = tree.depth;
    a.child_off = tree.child_off;
    a.child_ids = tree.child_ids;
    a.token = token;
    a.pool_ids = pool_ids;
    a.out_tokens = out_tokens;
    a.out_nodes = out_nodes;
    a.out_len = out_len;
    a.status = status;
    const size_t smem = (size_t)a.C * sizeof(float2);
    if (target.dtype == 1) {
        cudaError_t e = cudaFuncSetAttribute(k_verify_pooled<__nv_bfloat16>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        return launch_pdl(k_verify_pooled<__nv_bfloat16>, dim3((unsigned)B), dim3(kVpThreads), smem, s, 0, a);
    }
    cudaError_t e =
        cudaFuncSetAttribute(k_verify_pooled<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_verify_pooled<float>, dim3((unsigned)B), dim3(kVpThreads), smem, s, 0, a);
}

}  // namespace tsb
