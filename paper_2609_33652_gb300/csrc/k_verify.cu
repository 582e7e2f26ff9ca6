// Tree verification by recursive rejection sampling for WoR candidates (Sec. 2.3 Eq.
// rs-overlap; App. A), lossless on the frozen topology (Prop. 1).
//
// One thread-block cluster per tree. CTA r of the cluster owns the chunk-aligned vocabulary
// slice [r*slice, (r+1)*slice) and keeps that slice of the current node in shared memory as
// fp32: P holds the target logits, later their softmax P0; Q holds the normalised draft
// law once a rejection needs it. Scalars (the target log-normaliser, residual masses, argmax
// keys) are combined across the cluster through distributed shared memory: each CTA
// publishes its partial, the cluster barrier orders the writes, and every CTA combines all
// partials in rank order, so all CTAs hold bitwise identical values and take identical
// decisions.
//
// Walk at node u with children y_1..y_m (slot order), P0 = softmax(target row u),
// Q = softmax(q row of u), t_0 = 1:
//   slot i: p' = p_i(y_i), q' = Q(y_i)/t_i; accept iff U * q' < p';
//           on reject R_{i+1}(v) = max(p_i(v) - Q(v)/t_i, 0), Z_{i+1} = sum R_{i+1},
//           p_{i+1} = R_{i+1}/Z_{i+1}, t_{i+1} = t_i - Q(y_i).
//   A rejected token has p_{i+1} = 0 from then on, which is exactly the exclusion of drawn
//   tokens from the renormalised draft law. The recursion has a closed form: subtracting
//   non-negative multiples of Q and clamping at zero composes, so
//   p_i(v) = max(P0(v) - A_i Q(v), 0) / D_i with A_{i+1} = A_i + D_i / t_i and D_{i+1} the
//   mass of max(P0 - A_{i+1} Q, 0). P keeps P0 (a rejected token's entry set to zero), a pass
//   per rejection reads P0 and Q and only sums, and the point value p_i(y) uses the same fp32
//   operations as the element passes.
// Final tokens (all children rejected: from R_m; leaf: bonus from the target row) are drawn
// with the two-level Gumbel-max of the randomness contract: chunk keys log(chunk mass) + G
// over chunks of 256 tokens, then the best token of the winning chunk.
//
// Scheduling. A pre-pass (k_pre_split before the walk, or its CTAs inside the replay's grid in
// k_replay_pre) computes the target log-normalisers of the nodes a walk is most likely to
// visit, the first kPreChain internal nodes of the first-child chain from the root (slot 0 is
// accepted at most visits), as kPreSplit partials per row that the walk merges in order, and
// the q rows' log-normalisers (per depth, or per internal node for per-node rows). The walk
// kernel copies the tree's topology, the children's target and q logits and their acceptance
// uniforms to shared memory once. At
// a node with a known normaliser it needs no staging and no cluster round: every CTA takes
// the same decisions from the same inputs, and the slices are staged only if a rejection needs
// the residual. At any other node the walk runs a staging round over that node and up to two
// (bf16; one for fp32) of its first-child descendants without a value: the rows' slices are
// copied to shared memory with cp.async, all in flight together, their chunk statistics
// computed there (the node's x kept in P), and each row's log-normaliser merged from one
// partial per CTA through distributed shared memory. 12 warps per CTA: 160 registers a thread
// without spills (16 warps at 128 spilled in the walk's hot paths and ran slower). Element passes give lane l the elements 4l..4l+3 and
// 128+4l..128+4l+3 of each 256-token chunk, so every shared-memory access is a conflict-free
// 16-byte vector. Each normaliser is computed by a fixed procedure chosen by the node alone
// (pre-computed chain node, staged node), and which nodes are pre-computed depends only on the
// topology, so results do not depend on timing or on which call (tsb_verify alone or
// tsb_replay_verify) ran the pre-pass.
#include <cooperative_groups.h>

#include <mutex>

#include "tsb_device.cuh"
#include "tsb_launch.h"
#include "replay_body.cuh"

namespace cg = cooperative_groups;

namespace tsb {
namespace {

constexpr int kThreads = 384;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxSliceChunks = 128;  // slice <= 32768 tokens
constexpr int kMaxDepthRows = 64;     // per-depth q rows (depth cap L <= 64)
constexpr int kPreThreads = 512;
// Rows per staging round of the RRS walk, at most: the node being visited and up to two of its
// first-child descendants (the children a walk most often accepts next), whose target
// log-normalisers the same round computes with the copies of all rows in flight together.
constexpr int kLook = 3;
// Internal nodes of the first-child chain from the root whose target normalisers the RRS
// pre-pass computes on the whole GPU (the walk starts on that chain; nodes a walk reaches off it
// are staged by the walk's own rounds).
constexpr int kPreChain = 6;  // 8 and 6 measured the same step, 4 slower; 6 reads fewer unvisited rows
constexpr int kPreSplit = 8;           // CTAs per pre-computed target row (equal parts of its chunks)
constexpr int kPreSplitThreads = kRpThreads;  // shares a grid with the replay CTAs
static_assert((size_t)kPreChain * kPreSplit * 16 <= kWsPrePartBytes, "pre-pass partials per tree");
static_assert(kWarps % 4 == 0 && kLook <= kWarps, "groups of four warps per normaliser");

// Pre-pass results, one 32-byte workspace slot per (tree, node) (the slots block
// verification uses for its own per-position scalars): l2t = target log-normaliser of node u
// (u in the pre-computed set), l2q = log-normaliser of per-depth q row u, or of node u's own q
// row for per-node rows; both float-float, times log2(e). Pre-computed set of a tree: for
// recursive rejection sampling the first kPreChain internal nodes of the first-child chain,
// for traversal verification every internal node.
struct alignas(16) PreRow {
    float2 l2t, l2q;
    float pad[4];
};
static_assert(sizeof(PreRow) == kWsBvRowBytes, "pre-pass slot size");


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
    PreRow *pre;  // [B, N+1]
    int M;        // node ids below M with children are pre-computed (pre_chain == 0), or
                  // the first M internal nodes of the first-child chain (pre_chain == 1)
    int pre_chain;
    int copy_early;  // the pre-pass runs just before the walk: the walk copies its tree before waiting
    int Lq;       // per-depth q rows whose normaliser the pre-pass computes (0 for per-node rows)
    int qn;       // 1: the pre-pass computes each internal node's per-node q-row normaliser (slot u)
    int B;
    float4 *part;    // [B, kPreChain, kPreSplit] partial normalisers (max, float-float sum) of the chain rows
    int tokens_late; // the tokens come from the launch just before the walk: read them after the wait
};

// A partial of one cluster-wide reduction: a softmax normaliser (max, float-float sum), a
// plain float-float sum, and an argmax key carrying a token.
struct alignas(16) Slot {
    float m, sh, sl, zh, zl;
    int tok;
    unsigned long long key;
};

enum : int { kRedLse = 1, kRedSum = 2, kRedArg = 4 };

__device__ __forceinline__ Slot neutral_slot() {
    Slot s;
    s.m = -INFINITY;
    s.sh = s.sl = s.zh = s.zl = 0.f;
    s.tok = -1;
    s.key = 0ull;
    return s;
}

// A normaliser rescaled to a larger reference maximum M (exp evaluated once).
__device__ __forceinline__ FF rescale_to(float m, FF s, float M) {
    return m == -INFINITY ? FF{0.f, 0.f} : (m == M ? s : ff_scale(s, expf(__fsub_rn(m, M))));
}

template <int KIND>
__device__ __forceinline__ Slot warp_reduce_slot(Slot v) {
    __syncwarp();
    if (KIND & kRedLse) {  // maximum first, then every lane rescales once, then a plain sum
        const float M = warp_max(v.m);
        const FF a = warp_sum_ff(rescale_to(v.m, FF{v.sh, v.sl}, M));
        v.m = M;
        v.sh = a.hi;
        v.sl = a.lo;
    }
    if (KIND & kRedSum) {
        const FF z = warp_sum_ff(FF{v.zh, v.zl});
        v.zh = z.hi;
        v.zl = z.lo;
    }
    if (KIND & kRedArg) {
        int owner;
        v.key = warp_max_u64_owner(v.key, &owner);
        v.tok = __shfl_sync(kFull, v.tok, owner);
    }
    return v;
}

struct Scratch {
    Slot slot[2];        // published partials, double-buffered across rounds
    Slot wpart[kWarps];  // per-warp partials of the current round
    Slot res;            // combined result
    FF L2t, L2q;         // log-normalisers of the target and q rows, times log2(e)
    unsigned long long wbest[kWarps], wtok[kWarps];
    int cbad;
    int path[kMaxDepthRows];      // accepted node ids (written out after the walk)
    FF l2q[kMaxDepthRows];        // per-depth q log-normalisers (times log2 e)
    float2 cst[kLook][kMaxSliceChunks];  // chunk statistics of the slice's rows in a staging round
    Slot lpart[2][kLook];                // this CTA's partials of the round's normalisers, alternating
    int look[kLook];                        // nodes of the current staging round
    int nlook;
};

// One cluster-wide reduction: warp reductions, the CTA's warp partials in warp 0, the
// cluster barrier, then warp 0 of every CTA reads the CS published partials (one per lane)
// and combines them the same way, so every CTA obtains identical results.
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
                const FF l = v.sh > 0.f ? maxsum_lse(MaxSum{v.m, FF{v.sh, v.sl}}) : FF{0.f, 0.f};
                sh.L2t = ff_times_log2e(l);
            }
        }
    }
    __syncthreads();
    par ^= 1;
}

__device__ __forceinline__ float4 ld4(const float *p, int j) { return *reinterpret_cast<const float4 *>(p + j); }
__device__ __forceinline__ void st4(float *p, int j, float a, float b, float c, float d) {
    *reinterpret_cast<float4 *>(p + j) = make_float4(a, b, c, d);
}

// A row's log-normaliser from its chunk statistics (m_c, s_c) in shared memory, over a fixed
// partition: thread t < 128 of a group of four warps takes chunks t, t + 128, ... (their maximum, then a Kahan sum of
// s_c e^(m_c - m)), each of warps 0..3 merges its lanes (lse_part), and warp 0 merges the
// four warps in order (lse_final, result times log2 e). Every kernel that needs a target
// row's normaliser calls these two functions, kept out of line, so the value does not depend
// on which kernel or CTA computed it.
__device__ __noinline__ Slot lse_part(const float2 *pst, int C, int t) {
    float m = -INFINITY;
    for (int c = t; c < C; c += 128) m = fmaxf(m, pst[c].x);
    KahanF acc;
    if (m != -INFINITY)
        for (int c = t; c < C; c += 128) acc.add(__fmul_rn(pst[c].y, expf(__fsub_rn(pst[c].x, m))));
    Slot mine = neutral_slot();
    const FF sv = acc.ff();
    mine.m = m;
    mine.sh = sv.hi;
    mine.sl = sv.lo;
    return warp_reduce_slot<kRedLse>(mine);
}

__device__ __noinline__ FF lse_final(const Slot *part) {
    const int lane = threadIdx.x & 31;
    const Slot v = warp_reduce_slot<kRedLse>(lane < 4 ? part[lane] : neutral_slot());
    const FF l = v.sh > 0.f ? maxsum_lse(MaxSum{v.m, FF{v.sh, v.sl}}) : FF{0.f, 0.f};
    return ff_times_log2e(l);
}

template <typename T>
struct Walk {
    const VerifyArgs &a;
    Scratch &sh;
    const cg::cluster_group &cluster;
    float *P, *Q;
    int &par;
    int b, lo, n, nch;

    // Shared-memory index of lane `lane`'s quad h (0 or 1) in local chunk cl.
    static __device__ __forceinline__ int quad_at(int cl, int h, int lane) { return cl * kChunk + h * 128 + 4 * lane; }

    // Stage x = fp32(z) * invT of this CTA's slice of `row` into dst (warps 0..nw-1; logits
    // past the vocabulary become -inf), or store exp(x - L) instead of x (the normalised
    // law). Loads are issued in batches of kB chunks per warp before any is used, so a slice
    // costs one memory round trip per batch.
    template <bool NORMALISE, bool CHECK = false>
    __device__ void stage(const T *row, float *dst, int nw, FF L2) {
        constexpr int kB = sizeof(T) == 2 ? 9 : 5;
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        bool bad = false;  // CHECK: a NaN or +inf logit
        if (warp >= nw) return;
        const int end = lo + n;
        for (int c0 = warp; c0 < nch; c0 += nw * kB) {
            RawQuad<T> raw[kB][2];
#pragma unroll
            for (int e = 0; e < kB; ++e) {
                const int cl = c0 + e * nw;
                if (cl < nch) {
                    raw[e][0].load(row, lo + quad_at(cl, 0, lane), end);
                    raw[e][1].load(row, lo + quad_at(cl, 1, lane), end);
                }
            }
#pragma unroll
            for (int e = 0; e < kB; ++e) {
                const int cl = c0 + e * nw;
                if (cl >= nch) break;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    float x[4];
                    raw[e][h].unpack(x);
#pragma unroll
                    for (int k = 0; k < 4; ++k) x[k] = __fmul_rn(x[k], a.invT);  // padding stays -inf
                    if (CHECK) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) bad |= !(x[k] <= FLT_MAX) && x[k] != -INFINITY;
                    }
                    if (NORMALISE) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) x[k] = exp_shifted(x[k], L2);
                    }
                    st4(dst, quad_at(cl, h, lane), x[0], x[1], x[2], x[3]);
                }
            }
        }
        if (CHECK && __any_sync(kFull, bad) && lane == 0) raise_status(a.status, kDevNonFinite);
    }

    // One staging round over the target rows of nodes sh.look[0..J-1] (J <= kLookMax).
    // Every thread copies 16-byte pieces of this CTA's slice of each row into shared memory
    // with cp.async (all rows in flight at once, no registers held): row 0 into the lower half
    // of Q, row 1 into the upper half of Q (bf16) or into P (fp32), row 2 into the upper half
    // of P (bf16); the slice's tail past the vocabulary becomes -inf. Then, in the
    // chunk-statistics layout (eight lanes per 256-logit chunk, lane g holding logits 8g..8g+7
    // of each 64-logit quarter), every chunk's statistics into cst[j] (the per-chunk code of the
    // statistics kernels): rows 1..J-1 first, then row 0 with x = fp32(z) * invT into P (which
    // held the other rows' copies). Every thread takes part; ends synchronised.
    static constexpr int kLookMax = sizeof(T) == 2 ? 3 : 2;
    __device__ unsigned char *landing(int j) const {
        if (j == 0) return reinterpret_cast<unsigned char *>(Q);
        if (sizeof(T) == 4) return reinterpret_cast<unsigned char *>(P);
        return j == 1 ? reinterpret_cast<unsigned char *>(Q) + (size_t)a.slice * 2
                      : reinterpret_cast<unsigned char *>(P) + (size_t)a.slice * 2;
    }
    // This CTA's slice of `row`, raw, to shared memory at dst with cp.async (16-byte pieces);
    // the ragged tail (fewer than 16 bytes) by plain loads and the padding up to the last
    // chunk's end as -inf. The caller commits and waits.
    __device__ void copy_slice_async(const T *row, unsigned char *dst) {
        const int bytes = n * (int)sizeof(T), pieces = bytes >> 4;
        const unsigned char *src = reinterpret_cast<const unsigned char *>(row + lo);
        for (int i = threadIdx.x; i < pieces; i += kThreads) {
            const unsigned sa = (unsigned)__cvta_generic_to_shared(dst + 16 * i);
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sa), "l"(src + 16 * i) : "memory");
        }
        T *lt = reinterpret_cast<T *>(dst);
        for (int e = (pieces << 4) / (int)sizeof(T) + threadIdx.x; e < nch * kChunk; e += kThreads)
            lt[e] = e < n ? row[lo + e] : Logit<T>::neg_inf();
    }

    // The normalised law exp(fp32(z) * invT - L) of 8 raw bf16 logits at element e of zone
    // into dst[e..e+7] (the arithmetic of stage<true>).
    __device__ __forceinline__ void law8(const uint4 w, FF L2, float *dst, int e) {
        RawGroup<T> r;
        r.w = w;
        float z[8];
        r.unpack(z);
#pragma unroll
        for (int k = 0; k < 8; ++k) z[k] = exp_shifted(__fmul_rn(z[k], a.invT), L2);
        st4(dst, e, z[0], z[1], z[2], z[3]);
        st4(dst, e + 4, z[4], z[5], z[6], z[7]);
    }

    // P0 into P (from trow; skipped when trow is null) and the normalised q law into Q, for bf16
    // rows: both slices are copied raw with cp.async first (one memory round trip, no registers
    // held), the target into the lower half of Q and the q row into its upper half; then P from
    // the lower half; then Q in place: elements below slice/2 directly (their fp32 values land
    // in the consumed lower half), the others held in registers across a barrier (their fp32
    // values overwrite raw q values). Same values as stage<true>. Every thread takes part;
    // ends synchronised.
    __device__ void stage_pair(const T *trow, const T *qrow, FF L2t, FF L2q) {
        static_assert(sizeof(T) == 2, "raw bf16 slices fit the halves of Q");
        constexpr int kHold = (kMaxSliceChunks * kChunk / 2 / 8 + kThreads - 1) / kThreads;
        unsigned char *zt = reinterpret_cast<unsigned char *>(Q);
        unsigned char *zq = zt + (size_t)a.slice * 2;
        if (trow) copy_slice_async(trow, zt);
        copy_slice_async(qrow, zq);
        asm volatile("cp.async.commit_group;" ::: "memory");
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        __syncthreads();
        const int g8 = nch * kChunk / 8, half8 = a.slice / 16;  // groups of 8 elements
        if (trow) {
            for (int e8 = threadIdx.x; e8 < g8; e8 += kThreads)
                law8(*reinterpret_cast<const uint4 *>(zt + 16 * e8), L2t, P, 8 * e8);
            __syncthreads();  // the lower half is consumed
        }
        uint4 hold[kHold];
#pragma unroll
        for (int h = 0; h < kHold; ++h) {
            const int e8 = half8 + threadIdx.x + h * kThreads;
            if (e8 < g8) hold[h] = *reinterpret_cast<const uint4 *>(zq + 16 * e8);
        }
        for (int e8 = threadIdx.x; e8 < min(half8, g8); e8 += kThreads)
            law8(*reinterpret_cast<const uint4 *>(zq + 16 * e8), L2q, Q, 8 * e8);
        __syncthreads();  // every raw q value has been read
#pragma unroll
        for (int h = 0; h < kHold; ++h) {
            const int e8 = half8 + threadIdx.x + h * kThreads;
            if (e8 < g8) law8(hold[h], L2q, Q, 8 * e8);
        }
        __syncthreads();
    }

    __device__ void stage_look(int J, float *dst, float2 (*cst)[kMaxSliceChunks]) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        const int g = lane & 7, q = lane >> 3;
        for (int j = 0; j < J; ++j) {
            const T *row = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)sh.look[j] * a.t_rstride;
            copy_slice_async(row, landing(j));
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        __syncthreads();
        const int units = (nch + 3) / 4;
        for (int pass = 0; pass < 2; ++pass) {  // rows 1..J-1, then row 0 (its x overwrites P)
            const int j0 = pass == 0 ? 1 : 0, nj = pass == 0 ? J - 1 : 1;
            const int total = nj * units;
            for (int i0 = warp; i0 < total; i0 += kWarps) {  // uniform over the warp
                const int j = j0 + i0 / units, cl = (i0 - (i0 / units) * units) * 4 + q;
                const bool live = cl < nch;
                const unsigned char *zone = landing(j);
                RawGroup<T> raw[4];
                if (live)
#pragma unroll
                    for (int k = 0; k < 4; ++k) raw[k].load_shared(zone, cl * kChunk + k * 64 + g * 8);
                float mc, sc;
                chunk_stats8<T>(raw, live, a.invT, &mc, &sc);
                if (live && g == 0) cst[j][cl] = make_float2(mc, sc);
                if (live && j == 0) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        float z[8];
                        raw[k].unpack(z);
                        const int e = cl * kChunk + k * 64 + g * 8;
                        st4(dst, e, __fmul_rn(z[0], a.invT), __fmul_rn(z[1], a.invT), __fmul_rn(z[2], a.invT),
                            __fmul_rn(z[3], a.invT));
                        st4(dst, e + 4, __fmul_rn(z[4], a.invT), __fmul_rn(z[5], a.invT), __fmul_rn(z[6], a.invT),
                            __fmul_rn(z[7], a.invT));
                    }
                }
            }
            __syncthreads();
        }
    }

    // The log-normalisers of the round's J rows: each CTA merges the statistics of its own
    // chunks of row j (warp j: the maximum, then a float-float sum of s_c e^(m_c - m) over a
    // fixed lane partition), publishes that partial, and after the cluster barrier every CTA
    // merges the CS partials in rank order with the same warp reduction, so all CTAs hold
    // identical values. Ends with row j's value (times log2 e) in l2t[sh.look[j]] and the node
    // marked as known. `slot` alternates between rounds (a CTA may publish the next round's
    // partials while another still reads these).
    __device__ void gather_look(int J, const float2 (*cst)[kMaxSliceChunks], int slot, FF *l2t, int32_t *known) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        if (warp < J) {
            const float2 *c = cst[warp];
            float m = -INFINITY;
            for (int cl = lane; cl < nch; cl += 32) m = fmaxf(m, c[cl].x);
            KahanF acc;
            if (m != -INFINITY)
                for (int cl = lane; cl < nch; cl += 32) acc.add(__fmul_rn(c[cl].y, expf(__fsub_rn(c[cl].x, m))));
            Slot mine = neutral_slot();
            const FF sv = acc.ff();
            mine.m = m;
            mine.sh = sv.hi;
            mine.sl = sv.lo;
            const Slot w = warp_reduce_slot<kRedLse>(mine);
            if (lane == 0) sh.lpart[slot][warp] = w;
        }
        cluster.sync();  // every CTA's partials are published
        if (warp < J) {
            const int CS = (int)cluster.num_blocks();
            const Slot v = warp_reduce_slot<kRedLse>(lane < CS ? *cluster.map_shared_rank(&sh.lpart[slot][warp], lane)
                                                               : neutral_slot());
            if (lane == 0) {
                const FF l = v.sh > 0.f ? maxsum_lse(MaxSum{v.m, FF{v.sh, v.sl}}) : FF{0.f, 0.f};
                l2t[sh.look[warp]] = ff_times_log2e(l);
                known[sh.look[warp]] = 1;
            }
        }
        __syncthreads();
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
    // token; the cluster keeps the pair with the largest chunk key. wt(j, w) fills w[0..3]
    // with the quad at shared-memory index j: log-weights (LOGITS) or weights >= 0.
    template <bool LOGITS, typename F>
    __device__ int draw(int node, F wt) {
        const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
        // 1. chunk log-masses: eight lanes per chunk (lane g of the group takes quads g, g + 8,
        //    ..., g + 56), four chunks per warp and iteration; 2. each chunk's key by its group's
        //    first lane
        unsigned long long best = 0ull;
        {
            const int g = lane & 7, grp = lane >> 3;
            for (int c0 = warp * 4; c0 < nch; c0 += kWarps * 4) {  // uniform over the warp
                const int cl = c0 + grp;
                const bool live = cl < nch;
                float v[32];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    if (live) {
                        wt(cl * kChunk + 4 * (g + 8 * k), v + 4 * k);
                    } else {
                        v[4 * k] = v[4 * k + 1] = v[4 * k + 2] = v[4 * k + 3] = LOGITS ? -INFINITY : 0.f;
                    }
                }
                float A = -INFINITY;
                if (LOGITS) {
                    float mx = v[0];
#pragma unroll
                    for (int k = 1; k < 32; ++k) mx = fmaxf(mx, v[k]);
                    __syncwarp();  // converged before the group shuffles
                    mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 4));
                    mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 2));
                    mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 1));
                    float sm = 0.f;
                    if (mx != -INFINITY) {
#pragma unroll
                        for (int k = 0; k < 32; ++k) sm += fast_exp2(__fmul_rn(__fsub_rn(v[k], mx), kLog2e));
                    }
                    __syncwarp();
                    sm += __shfl_xor_sync(kFull, sm, 4);
                    sm += __shfl_xor_sync(kFull, sm, 2);
                    sm += __shfl_xor_sync(kFull, sm, 1);
                    if (mx != -INFINITY) A = __fadd_rn(mx, logf(sm));
                } else {
                    float sm = 0.f;
#pragma unroll
                    for (int k = 0; k < 32; ++k) sm += v[k];
                    __syncwarp();
                    sm += __shfl_xor_sync(kFull, sm, 4);
                    sm += __shfl_xor_sync(kFull, sm, 2);
                    sm += __shfl_xor_sync(kFull, sm, 1);
                    if (sm > 0.f) A = logf(sm);
                }
                if (live && g == 0 && A != -INFINITY) {  // 2. the chunk's key; the lane's best
                    const int c = (lo >> 8) + cl;
                    const uint32_t w = draw_word(a.seed, kFinalChunk, (uint32_t)b, (uint32_t)node, (uint32_t)c);
                    const unsigned long long pk = pack_key(__fadd_rn(A, gumbel_of(w)), (uint32_t)c);
                    best = pk > best ? pk : best;
                }
            }
        }
        best = warp_max_u64(best);  // the CTA's best chunk
        if (lane == 0) sh.wbest[warp] = best;
        __syncthreads();
        // 3. the best token inside this CTA's best chunk: one element per thread (threads
        //    0..255), then the CTA's maximum
        const unsigned long long cb = warp_max_u64(lane < kWarps ? sh.wbest[lane] : 0ull);
        unsigned long long tb = 0ull;
        if (cb != 0ull && threadIdx.x < kChunk) {
            const int cl = (int)key_id(cb) - (lo >> 8);
            const int e = threadIdx.x, j = cl * kChunk + (e & ~3), v = lo + cl * kChunk + e;
            float q4[4];
            wt(j, q4);
            const float x = q4[e & 3];
            const bool live = LOGITS ? x != -INFINITY : x > 0.f;
            if (live) {
                const float l = LOGITS ? x : logf(x);
                const uint32_t w = draw_word(a.seed, kFinal, (uint32_t)b, (uint32_t)node, (uint32_t)v);
                tb = pack_key(__fadd_rn(l, gumbel_of(w)), (uint32_t)v);
            }
        }
        tb = warp_max_u64(tb);
        if (lane == 0) sh.wtok[warp] = tb;
        __syncthreads();
        Slot mine = neutral_slot();  // the CTA's pair (best chunk key, its best token), from thread 0
        if (warp == 0) {
            const unsigned long long t = warp_max_u64(lane < kWarps ? sh.wtok[lane] : 0ull);
            if (lane == 0 && cb != 0ull) {
                mine.key = cb;
                mine.tok = (int)key_id(t);
            }
        }
        reduce_round<kRedArg>(sh, par, cluster, mine);
        return sh.res.key == 0ull ? -1 : sh.res.tok;
    }

    // Bonus draw from the logits of `row` (a leaf, or a residual without mass).
    template <bool CHECK = false>
    __device__ int draw_from_row(const T *row, int node) {
        __syncthreads();
        stage<false, CHECK>(row, P, kWarps, FF{0.f, 0.f});
        __syncthreads();
        return draw<true>(node, [&](int j, float *v) {
            const float4 x = ld4(P, j);
            v[0] = x.x;
            v[1] = x.y;
            v[2] = x.z;
            v[3] = x.w;
        });
    }
};

// Log-normaliser of a q row from its chunk statistics (m_c, s_c), by one warp, times
// log2(e): the maximum of the m_c, then sum s_c exp(m_c - M) (loads issued eight at a time;
// the same code on the same data in every CTA gives the same bits).
__device__ FF q_log_normaliser(const float2 *st, int C) {
    constexpr int kB = 8;
    const int lane = threadIdx.x & 31;
    float m = -INFINITY;
    for (int c0 = lane; c0 < C; c0 += 32 * kB) {
        float v[kB];
#pragma unroll
        for (int e = 0; e < kB; ++e) v[e] = c0 + 32 * e < C ? __ldg(&st[c0 + 32 * e]).x : -INFINITY;
#pragma unroll
        for (int e = 0; e < kB; ++e) m = fmaxf(m, v[e]);
    }
    m = warp_max(m);
    KahanF s;
    if (m != -INFINITY)
        for (int c0 = lane; c0 < C; c0 += 32 * kB) {
            float2 v[kB];
#pragma unroll
            for (int e = 0; e < kB; ++e)
                v[e] = c0 + 32 * e < C ? __ldg(&st[c0 + 32 * e]) : make_float2(-INFINITY, 0.f);
#pragma unroll
            for (int e = 0; e < kB; ++e)
                if (v[e].x != -INFINITY) s.add(__fmul_rn(v[e].y, expf(__fsub_rn(v[e].x, m))));
        }
    const FF S = warp_sum_ff(s.ff());
    return S.hi > 0.f ? ff_times_log2e(maxsum_lse(MaxSum{m, S})) : FF{0.f, 0.f};
}

// Node j of the first-child chain (j = 0 the root): from the root, each step moves to the
// node's first child while that child has children itself; -1 past the chain's end (or on
// inconsistent arrays). off / kid: the tree's child lists. The pre-pass and the walk select
// the chain's nodes with this one function.
__device__ __forceinline__ int chain_node(const int32_t *off, const int32_t *kid, int N, int j) {
    int v = 0;
    for (int k = 0; k < j; ++k) {
        const int o = off[v];
        if (o < 0 || o >= N) return -1;
        const int c = kid[o];
        if (c < 1 || c > N || off[c + 1] - off[c] <= 0) return -1;
        v = c;
    }
    return off[v + 1] - off[v] > 0 ? v : -1;
}

// Shared-memory bytes of the tree's copy: per node its pre-computed target log-normaliser
// (float-float) and whether it has one; topology (child_off [N+2], child_ids [N], token [N+1],
// q row of node [N+1]); per child slot its parent, target logit, q logit and uniform.
inline size_t topo_bytes(int N) {
    return (size_t)2 * (N + 1) * sizeof(float2) + (size_t)(6 * N + 6) * sizeof(int32_t) +
           (size_t)3 * N * sizeof(float);
}

// The tree's copy in shared memory, after the two row slices.
struct TreeSmem {
    FF *l2t;   // [N+1] pre-computed target normalisers (times log2 e)
    FF *l2qn;  // [N+1] pre-computed per-node q-row normalisers (when a.qn)
    int32_t *pre, *off, *kid, *tok, *row, *ps;
    float *cxt, *cxq, *cu;
};

// Copy of tree b's topology for a walk: child lists, q row per node, and each child slot's
// parent. It reads only the tree (written before the pre-pass and the replay began), so a walk
// may run it before waiting for the launch before it. Sets sh.cbad on inconsistent tree
// arrays. Every thread of the CTA calls it; it ends with the CTA synchronised.
template <typename T>
__device__ TreeSmem copy_topo(const VerifyArgs &a, Scratch &sh, float *base, int b, bool per_depth) {
    const int NN = a.N + 1;
    TreeSmem ts;
    ts.l2t = reinterpret_cast<FF *>(base);
    ts.l2qn = ts.l2t + NN;
    ts.pre = reinterpret_cast<int32_t *>(ts.l2qn + NN);
    ts.off = ts.pre + NN;
    ts.kid = ts.off + (NN + 1);
    ts.tok = ts.kid + a.N;
    ts.row = ts.tok + NN;
    ts.ps = ts.row + NN;
    ts.cxt = reinterpret_cast<float *>(ts.ps + a.N);
    ts.cxq = ts.cxt + a.N;
    ts.cu = ts.cxq + a.N;
    {
        const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
        const int32_t *kids = a.child_ids + (int64_t)b * a.N;
        const int32_t *row = per_depth ? a.depth + (int64_t)b * NN : a.qrow_of_node + (int64_t)b * NN;
        for (int i = threadIdx.x; i <= NN; i += kThreads) ts.off[i] = __ldg(off + i);
        for (int i = threadIdx.x; i < a.N; i += kThreads) {
            ts.kid[i] = __ldg(kids + i);
            ts.ps[i] = -1;
        }
        for (int i = threadIdx.x; i < NN; i += kThreads) ts.row[i] = __ldg(row + i);
        if (threadIdx.x == 0) sh.cbad = 0;
    }
    __syncthreads();
    {  // every valid internal node claims its child slots
        bool bad_here = false;
        for (int u = threadIdx.x; u < NN; u += kThreads) {
            const int o = ts.off[u], m = ts.off[u + 1] - o;
            if (m == 0) continue;
            const int r = ts.row[u];
            if (m < 0 || m > kMaxK || o < 0 || o + m > a.N || r < 0 || r >= a.q_R || (per_depth && r >= a.Lq)) {
                bad_here = true;
                continue;
            }
            for (int i = 0; i < m; ++i) ts.ps[o + i] = u;
        }
        if (bad_here) sh.cbad = 1;
    }
    // the pre-computed set by node id (the chain's nodes are marked by load_pre)
    for (int u = threadIdx.x; u < NN; u += kThreads)
        ts.pre[u] = !a.pre_chain && u < a.M && ts.off[u + 1] - ts.off[u] > 0 ? 1 : 0;
    __syncthreads();
    return ts;
}

// The tokens of tree b (plain loads: they may come from the launch just before the walk); a
// barrier must follow before they are read.
__device__ __forceinline__ void copy_tokens(const VerifyArgs &a, const TreeSmem &ts, int b) {
    const int NN = a.N + 1;
    const int32_t *tok = a.token + (int64_t)b * NN;
    for (int i = threadIdx.x; i < NN; i += kThreads) ts.tok[i] = tok[i];
}

// Per child slot, after copy_topo and copy_tokens and a barrier: its token's target and q
// logits (from the parent's rows) and acceptance uniform. Every thread of the CTA calls it; it
// ends with the CTA synchronised.
template <typename T>
__device__ void slot_values(const VerifyArgs &a, Scratch &sh, const TreeSmem &ts, int b) {
    {  // every child slot: its token's target and q logits (from the parent's rows) and uniform
        bool bad_here = false;
        for (int j = threadIdx.x; j < a.N; j += kThreads) {
            const int u = ts.ps[j];
            if (u < 0) continue;  // not a child slot of a valid node (never read by the walk)
            const int c = ts.kid[j];
            const int y = (c >= 1 && c <= a.N) ? ts.tok[c] : -1;
            if (y < 0 || y >= a.V) {
                bad_here = true;
                continue;
            }
            const T *trow = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
            const T *qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)ts.row[u] * a.q_rstride;
            ts.cxt[j] = __fmul_rn(Logit<T>::load1(trow, y), a.invT);
            ts.cxq[j] = __fmul_rn(Logit<T>::load1(qrow, y), a.invT);
            ts.cu[j] = uniform_of(draw_word(a.seed, kAccept, (uint32_t)b, (uint32_t)c, 0u));
        }
        if (bad_here) sh.cbad = 1;
    }
    __syncthreads();
}

// The whole copy, for walks whose tokens were written before the launch before them.
template <typename T>
__device__ TreeSmem copy_tree(const VerifyArgs &a, Scratch &sh, float *base, int b, bool per_depth) {
    const TreeSmem ts = copy_topo<T>(a, sh, base, b, per_depth);
    copy_tokens(a, ts, b);
    __syncthreads();
    slot_values<T>(a, sh, ts, b);
    return ts;
}

// The pre-pass results for tree b (after the walk waited for the pre-pass), after copy_topo:
// the target normalisers of the pre-computed set (for the chain, merged from the partials and
// the chain's nodes marked), and the q-row normalisers (per depth with pre_q, per node with
// a.qn). All its loads form one round. Every thread of the CTA calls it; ends synchronised.
__device__ void load_pre(const VerifyArgs &a, Scratch &sh, const TreeSmem &ts, int b, bool pre_q) {
    const int NN = a.N + 1;
    if (pre_q)
        for (int i = threadIdx.x; i < a.Lq; i += kThreads) {
            const float2 v = a.pre[(int64_t)b * NN + i].l2q;
            sh.l2q[i] = FF{v.x, v.y};
        }
    if (a.M > 0 || a.qn)  // every node's slot in one round of loads (only the set's are used)
        for (int i = threadIdx.x; i < NN; i += kThreads) {
            const float4 pr = *reinterpret_cast<const float4 *>(&a.pre[(int64_t)b * NN + i]);
            if (!a.pre_chain) ts.l2t[i] = FF{pr.x, pr.y};
            ts.l2qn[i] = FF{pr.z, pr.w};
        }
    if (a.pre_chain) {  // chain node j's normaliser from the pre-pass's kPreSplit partials, in order
        if (threadIdx.x < a.M) {
            const int v = chain_node(ts.off, ts.kid, a.N, threadIdx.x);
            if (v >= 0) {
                const float4 *pp = a.part + ((int64_t)b * kPreChain + threadIdx.x) * kPreSplit;
                MaxSum acc{-INFINITY, FF{0.f, 0.f}};
#pragma unroll
                for (int k = 0; k < kPreSplit; ++k) {
                    const float4 p = pp[k];
                    acc = maxsum_merge(acc, MaxSum{p.x, FF{p.y, p.z}});
                }
                ts.l2t[v] = acc.s.hi > 0.f ? ff_times_log2e(maxsum_lse(acc)) : FF{0.f, 0.f};
                ts.pre[v] = 1;
            }
        }
    }
    __syncthreads();
}

// Pre-pass of traversal verification, in clusters of two CTAs. Clusters [0, B*M): cluster (b, j)
// streams target row j of tree b (if node j has children), each CTA half of its four-chunk
// units: the chunk statistics
// of every 256-logit chunk (eight lanes per chunk, two units in flight per warp, the same
// per-chunk code as the row statistics kernel) into shared memory; rank 0 gathers rank 1's
// half through distributed shared memory and computes the row's log-normaliser over a fixed
// 128-thread partition of all chunks, merged in a fixed order. Later CTAs: one warp per
// per-depth q row (tree b, depth d < Lq), from its chunk statistics (no cluster barrier).
template <typename T>
__global__ void __launch_bounds__(kPreThreads, 2) k_verify_pre(VerifyArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) float2 pst[];  // [C] the row's chunk statistics
    __shared__ Slot part[4];
    constexpr int nwarps = kPreThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int ntarget = 2 * a.B * a.M;  // even: a cluster is all target or all q-row CTAs
    if ((int)blockIdx.x >= ntarget) {  // q-row log-normalisers, one warp each
        const int task = ((int)blockIdx.x - ntarget) * nwarps + warp;
        const int per = a.qn ? NN : a.Lq;  // per-node rows of internal nodes, or per-depth rows
        if (task >= a.B * per) return;  // warp-uniform; no barrier in this branch
        const int b = task / per, d = task - (task / per) * per;
        int r = d;
        if (a.qn) {
            const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
            if (__ldg(off + d + 1) - __ldg(off + d) <= 0) return;  // a leaf needs no draft law
            r = __ldg(a.qrow_of_node + (int64_t)b * NN + d);
            if (r < 0 || r >= a.q_R) return;  // the walk flags the tree
        }
        const FF L2q = q_log_normaliser(a.qstats + ((int64_t)b * a.q_R + r) * a.C, a.C);
        if (lane == 0) a.pre[(int64_t)b * NN + d].l2q = make_float2(L2q.hi, L2q.lo);
        return;
    }
    cg::cluster_group cluster = cg::this_cluster();
    const int half = (int)cluster.block_rank();
    const int pair = (int)blockIdx.x >> 1;
    const int b = pair / a.M;
    int j = pair - (pair / a.M) * a.M;
    const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
    if (__ldg(off + j + 1) - __ldg(off + j) <= 0) return;  // leaves need no normaliser (both CTAs return)
    const T *row = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)j * a.t_rstride;
    const int g = lane & 7, q = lane >> 3;
    const int C = a.C, units = (C + 3) / 4;
    const int ulo = half == 0 ? 0 : (units + 1) / 2, uhi = half == 0 ? (units + 1) / 2 : units;
    constexpr int kU = sizeof(T) == 2 ? 2 : 1;  // units in flight per warp (register budget)
    for (int u0 = ulo + warp; u0 < uhi; u0 += kU * nwarps) {  // uniform over the warp
        RawGroup<T> raw[kU][4];
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * nwarps) * 4 + q;
            if (u0 + e * nwarps < uhi && c < C)
#pragma unroll
                for (int k = 0; k < 4; ++k) raw[e][k].load(row, c * kChunk + k * 64 + g * 8, a.V);
        }
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * nwarps) * 4 + q;
            const bool live = u0 + e * nwarps < uhi && c < C;
            float mc, sc;
            chunk_stats8<T>(raw[e], live, a.invT, &mc, &sc);
            if (live && g == 0) pst[c] = make_float2(mc, sc);
        }
    }
    cluster.sync();  // both halves written
    if (half == 1) {
        cluster.sync();  // rank 0 has copied this half
        return;
    }
    {
        const float2 *other = cluster.map_shared_rank(pst, 1);
        for (int c = (units + 1) / 2 * 4 + threadIdx.x; c < C; c += kPreThreads) pst[c] = other[c];
    }
    cluster.sync();  // rank 1 may leave; rank 0's copy is complete (the barrier also orders the CTA)
    if (warp < 4) {  // the log-normaliser over threads 0..127, then warps 0..3 in order
        const Slot w = lse_part(pst, C, threadIdx.x);
        if (lane == 0) part[warp] = w;
    }
    __syncthreads();
    if (warp == 0) {
        const FF L2 = lse_final(part);
        if (lane == 0) a.pre[(int64_t)b * NN + j].l2t = make_float2(L2.hi, L2.lo);
    }
}

// Chunks of one part of the split pre-pass (parts are equal runs of four-chunk units).
__host__ __device__ inline int pre_part_chunks(int C) { return ((C + 3) / 4 + kPreSplit - 1) / kPreSplit * 4; }
inline size_t pre_split_smem(int C, int N) {
    return (size_t)pre_part_chunks(C) * sizeof(float2) + (size_t)(2 * N + 2) * sizeof(int32_t);
}

// Pre-pass of recursive rejection sampling, CTA blk of kPreSplitThreads threads (dynamic shared
// memory: pre_split_smem). CTAs [0, B*kPreChain*kPreSplit): CTA (b, j, k) streams the k-th of
// kPreSplit equal parts (four-chunk units) of the target row of node j of tree b's first-child
// chain: chunk statistics (eight lanes per chunk, two units in flight per warp, the per-chunk
// code of the statistics kernels) into shared memory, then warp 0 merges them into one partial
// normaliser (maximum, float-float sum) at a.part[b][j][k]; the walk merges the kPreSplit
// partials in order. It reads only the tree and the target rows, so it may run beside the
// replay. Later CTAs: one warp per q-row normaliser (per-depth rows, or each internal node's
// per-node row). Every thread calls it; it may return early.
template <typename T>
__device__ __forceinline__ void pre_split_cta(const VerifyArgs &a, int blk, float2 *pst) {
    constexpr int nwarps = kPreSplitThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int ntarget = a.B * kPreChain * kPreSplit;
    if (blk >= ntarget) {  // q-row log-normalisers, one warp each
        const int task = (blk - ntarget) * nwarps + warp;
        const int per = a.qn ? NN : a.Lq;
        if (task >= a.B * per) return;  // warp-uniform; no barrier in this branch
        const int b = task / per, d = task - (task / per) * per;
        int r = d;
        if (a.qn) {
            const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
            if (__ldg(off + d + 1) - __ldg(off + d) <= 0) return;  // a leaf needs no draft law
            r = __ldg(a.qrow_of_node + (int64_t)b * NN + d);
            if (r < 0 || r >= a.q_R) return;  // the walk flags the tree
        }
        const FF L2q = q_log_normaliser(a.qstats + ((int64_t)b * a.q_R + r) * a.C, a.C);
        if (lane == 0) a.pre[(int64_t)b * NN + d].l2q = make_float2(L2q.hi, L2q.lo);
        return;
    }
    const int k = blk % kPreSplit, bj = blk / kPreSplit;
    const int b = bj / kPreChain, j = bj - (bj / kPreChain) * kPreChain;
    const int C = a.C, units = (C + 3) / 4, pc = pre_part_chunks(C);
    int32_t *s_off = reinterpret_cast<int32_t *>(pst + pc);
    int32_t *s_kid = s_off + NN + 1;
    {
        const int32_t *off = a.child_off + (int64_t)b * (NN + 1);
        const int32_t *kids = a.child_ids + (int64_t)b * a.N;
        for (int i = threadIdx.x; i <= NN; i += kPreSplitThreads) s_off[i] = __ldg(off + i);
        for (int i = threadIdx.x; i < a.N; i += kPreSplitThreads) s_kid[i] = __ldg(kids + i);
    }
    __syncthreads();
    const int v = chain_node(s_off, s_kid, a.N, j);  // the walk finds the same node
    if (v < 0) return;                               // uniform over the CTA
    const T *row = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)v * a.t_rstride;
    const int g = lane & 7, q = lane >> 3;
    const int ulo = k * (pc / 4), uhi = min(units, ulo + pc / 4), clo = 4 * ulo;
    constexpr int kU = sizeof(T) == 2 ? 2 : 1;  // units in flight per warp (register budget)
    for (int u0 = ulo + warp; u0 < uhi; u0 += kU * nwarps) {  // uniform over the warp
        RawGroup<T> raw[kU][4];
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * nwarps) * 4 + q;
            if (u0 + e * nwarps < uhi && c < C)
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) raw[e][kk].load(row, c * kChunk + kk * 64 + g * 8, a.V);
        }
#pragma unroll
        for (int e = 0; e < kU; ++e) {
            const int c = (u0 + e * nwarps) * 4 + q;
            const bool live = u0 + e * nwarps < uhi && c < C;
            float mc, sc;
            chunk_stats8<T>(raw[e], live, a.invT, &mc, &sc);
            if (live && g == 0) pst[c - clo] = make_float2(mc, sc);
        }
    }
    __syncthreads();
    if (warp == 0) {
        const int n = max(0, min(4 * uhi, C) - clo);
        float m = -INFINITY;
        for (int c = lane; c < n; c += 32) m = fmaxf(m, pst[c].x);
        m = warp_max(m);
        KahanF acc;
        if (m != -INFINITY)
            for (int c = lane; c < n; c += 32) acc.add(__fmul_rn(pst[c].y, expf(__fsub_rn(pst[c].x, m))));
        const FF sv = warp_sum_ff(acc.ff());
        if (lane == 0) a.part[(int64_t)bj * kPreSplit + k] = make_float4(m, sv.hi, sv.lo, 0.f);
    }
}

template <typename T>
__global__ void __launch_bounds__(kPreSplitThreads, 8) k_pre_split(VerifyArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) float2 pst[];
    pre_split_cta<T>(a, (int)blockIdx.x, pst);
}

// The replay CTAs and the split pre-pass CTAs in one grid: blocks [0, nrep) draw the tokens,
// the rest run the pre-pass (which reads neither the tokens nor anything else the replay
// writes).
template <int KCAP, typename T>
__global__ void __launch_bounds__(kRpThreads, KCAP <= 8 ? kRpMinBlocks : 2)
    k_replay_pre(ReplayArgs ra, VerifyArgs va, int nrep) {
    pdl_begin();
    if ((int)blockIdx.x < nrep) {
        replay_node<KCAP, T>(ra, (int)blockIdx.x);
        return;
    }
    extern __shared__ __align__(16) float2 pst[];
    pre_split_cta<T>(va, (int)blockIdx.x - nrep, pst);
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_verify_rrs(VerifyArgs a) {
    if (!a.copy_early) pdl_begin();
    extern __shared__ __align__(16) float dyn[];
    float *P = dyn;
    float *Q = dyn + a.slice;
    __shared__ Scratch sh;

    cg::cluster_group cluster = cg::this_cluster();
    const int CS = (int)cluster.num_blocks();
    const int crank = (int)cluster.block_rank();
    const int b = blockIdx.x / CS;
    const int NN = a.N + 1;
    const int lo = crank * a.slice;
    const int n = max(0, min(a.V - lo, a.slice));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool writer = crank == 0 && threadIdx.x == 0;
    const bool per_depth = a.qrow_of_node == nullptr;
    int par = 0;
    Walk<T> W{a, sh, cluster, P, Q, par, b, lo, n, (n + kChunk - 1) / kChunk};

    // the tree's copy in shared memory; with the pre-pass launched just before this kernel it
    // overlaps the pre-pass's tail (it reads nothing the pre-pass writes), then the wait for
    // the pre-pass and its results; tokens written by that launch (replay beside the
    // pre-pass) are read after the wait
    const TreeSmem ts = copy_topo<T>(a, sh, dyn + 2 * a.slice, b, per_depth);
    if (!a.tokens_late) {
        copy_tokens(a, ts, b);
        __syncthreads();
        slot_values<T>(a, sh, ts, b);
    }
    if (a.copy_early) pdl_begin();
    if (a.tokens_late) copy_tokens(a, ts, b);  // in the round of load_pre's loads
    load_pre(a, sh, ts, b, true);
    if (a.tokens_late) slot_values<T>(a, sh, ts, b);
    const FF *s_l2t = ts.l2t;
    const int32_t *s_known = ts.pre, *s_off = ts.off, *s_kid = ts.kid, *s_tok = ts.tok, *s_row = ts.row;
    const float *s_cxt = ts.cxt, *s_cxq = ts.cxq, *s_cu = ts.cu;
    int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
    int32_t *onode = a.out_nodes + (int64_t)b * a.L;

    cluster.sync();  // the copy is complete; every CTA of the cluster runs before any distributed access

    int u = 0, nacc = 0, final_tok = -1, ncst = 0;
    bool bad = sh.cbad != 0;  // every CTA checked the same arrays
    for (int step = 0; step <= a.L && !bad; ++step) {
        const int o = s_off[u], m = s_off[u + 1] - o;
        const T *trow = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
        if (m == 0) {  // leaf: bonus token from the node's target row
            final_tok = W.draw_from_row(trow, u);
            break;
        }
        const int r = s_row[u];
        const T *qrow = static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)r * a.q_rstride;
        bool staged = s_known[u] == 0;  // P holds this node's x after its staging round
        if (staged) {
            W.prefetch_slice(qrow);  // likely next read: this node's q row (a first rejection)
            __syncthreads();         // earlier readers of P, Q and the round's node list are done
            if (threadIdx.x == 0) {  // u, then first children while they have children and no value
                int J = 0, v = u;
                for (;;) {
                    sh.look[J++] = v;
                    if (J == Walk<T>::kLookMax) break;
                    const int c = s_kid[s_off[v]];
                    if (s_off[c + 1] - s_off[c] <= 0 || s_known[c] != 0) break;
                    v = c;
                }
                sh.nlook = J;
            }
            __syncthreads();
            const int J = sh.nlook;
            float2(*cst)[kMaxSliceChunks] = sh.cst;
            // x of u into P with the chunk statistics of all J rows, then their log-normalisers
            // from all chunks of the cluster (gathered into Q, free until u's first rejection)
            W.stage_look(J, P, cst);
            W.gather_look(J, cst, ncst, ts.l2t, ts.pre);
            ncst ^= 1;
        }
        const FF L2t = s_l2t[u];
        const FF L2q = per_depth ? sh.l2q[r] : ts.l2qn[u];
        // After i rejections p_i(v) = max(P0(v) - A_i Q(v), 0) / D_i with A_0 = 0, D_0 = 1,
        // A_{i+1} = A_i + D_i / t_i and D_{i+1} = sum_v max(P0(v) - A_{i+1} Q(v), 0): the
        // recursive residual max(p_i - Q/t_i, 0), renormalised, in closed form. A pass over the
        // slice reads P0 and Q and writes nothing; a rejected token's P0 is set to zero.
        FF t = FF{1.f, 0.f};  // draft mass not yet drawn
        int accepted = -1;
        bool q_staged = false;
        bool p_is_x = staged;  // P holds x (staged node) until its first pass stores P0
        float A = 0.f, D = 1.f, iD = 1.f;
        for (int i = 0; i < m; ++i) {
            const float it = t.hi > 0.f ? __frcp_rn(t.hi) : 0.f;  // 1/t_i
            const float P0y = exp_shifted(s_cxt[o + i], L2t);
            const float Qy = exp_shifted(s_cxq[o + i], L2q);
            const float pp = __fmul_rn(fmaxf(__fmaf_rn(-A, Qy, P0y), 0.f), iD);
            const float qp = __fmul_rn(Qy, it);
            if (__fmul_rn(s_cu[o + i], qp) < pp) {
                accepted = s_kid[o + i];
                break;
            }
            __syncthreads();  // earlier readers of P and Q are done
            if (!staged || !q_staged) {  // the slices a rejection needs, once per node
                if constexpr (sizeof(T) == 2) {
                    W.stage_pair(staged ? nullptr : trow, qrow, L2t, L2q);  // P0 directly when not staged
                } else {
                    if (!staged) W.template stage<true>(trow, P, kWarps, L2t);
                    W.template stage<true>(qrow, Q, kWarps, L2q);
                }
                staged = q_staged = true;
                __syncthreads();
            }
            {  // the rejected token leaves the residual for good
                const int y = s_tok[s_kid[o + i]];
                if (threadIdx.x == 0 && y >= lo && y < lo + n) P[y - lo] = p_is_x ? -INFINITY : 0.f;
            }
            __syncthreads();
            const float A1 = __fmaf_rn(D, it, A);
            // max(P0 - A1 Q, 0) of the quad at shared-memory index j
            auto w_quad = [&](int j, float *v) {
                float4 x = ld4(P, j);
                if (p_is_x) {
                    x.x = exp_shifted(x.x, L2t);
                    x.y = exp_shifted(x.y, L2t);
                    x.z = exp_shifted(x.z, L2t);
                    x.w = exp_shifted(x.w, L2t);
                }
                const float4 q = ld4(Q, j);
                v[0] = fmaxf(__fmaf_rn(-A1, q.x, x.x), 0.f);
                v[1] = fmaxf(__fmaf_rn(-A1, q.y, x.y), 0.f);
                v[2] = fmaxf(__fmaf_rn(-A1, q.z, x.z), 0.f);
                v[3] = fmaxf(__fmaf_rn(-A1, q.w, x.w), 0.f);
            };
            if (i == m - 1) {  // every slot rejected: final token from R_m = max(P0 - A_m Q, 0)
                final_tok = W.template draw<false>(u, w_quad);
                if (final_tok < 0) final_tok = W.draw_from_row(trow, u);  // no residual mass (rounding)
                break;
            }
            // residual pass: the mass of R_{i+1} (storing P0 the first time P holds x)
            KahanF zl[2];  // one per half chunk: two independent chains
            for (int cl = warp; cl < W.nch; cl += kWarps) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = Walk<T>::quad_at(cl, h, lane);
                    float4 x = ld4(P, j);  // padding: P0 = 0 (x = -inf), Q = 0
                    if (p_is_x) {
                        x.x = exp_shifted(x.x, L2t);
                        x.y = exp_shifted(x.y, L2t);
                        x.z = exp_shifted(x.z, L2t);
                        x.w = exp_shifted(x.w, L2t);
                        st4(P, j, x.x, x.y, x.z, x.w);
                    }
                    const float4 q = ld4(Q, j);
                    const float r0 = fmaxf(__fmaf_rn(-A1, q.x, x.x), 0.f), r1 = fmaxf(__fmaf_rn(-A1, q.y, x.y), 0.f);
                    const float r2 = fmaxf(__fmaf_rn(-A1, q.z, x.z), 0.f), r3 = fmaxf(__fmaf_rn(-A1, q.w, x.w), 0.f);
                    zl[h].add(__fadd_rn(__fadd_rn(r0, r1), __fadd_rn(r2, r3)));
                }
            }
            {
                Slot mine = neutral_slot();
                const FF z = ff_add(zl[0].ff(), zl[1].ff());
                mine.zh = z.hi;
                mine.zl = z.lo;
                reduce_round<kRedSum>(sh, par, cluster, mine);
            }
            const float Z = sh.res.zh;
            if (!(Z > 0.f)) {  // no residual mass (rounding only): the node's target row
                final_tok = W.draw_from_row(trow, u);
                break;
            }
            p_is_x = false;
            A = A1;
            D = Z;
            iD = __frcp_rn(Z);
            t = ff_add(t, FF{-Qy, 0.f});
        }
        if (accepted < 0) break;
        if (nacc >= a.L) {  // deeper than the depth cap: the tree arrays are inconsistent
            bad = true;
            break;
        }
        if (writer) sh.path[nacc] = accepted;  // no global store while cluster barriers follow
        ++nacc;
        u = accepted;
    }
    if (writer) {
        if (bad) raise_status(a.status, kDevBadTree);
        for (int k = 0; k < nacc; ++k) {
            otok[k] = s_tok[sh.path[k]];
            onode[k] = sh.path[k];
        }
        otok[nacc] = final_tok;
        for (int k = nacc + 1; k <= a.L; ++k) otok[k] = -1;
        for (int k = nacc; k < a.L; ++k) onode[k] = -1;
        a.out_len[b] = bad ? 0 : nacc + 1;
    }
    cluster.sync();  // no CTA leaves while another may still read its shared memory
}

// Traversal verification (Weng et al. 2025 as cited in Sec. 2.3, Table 2 and App. A:
// recursive rejection sampling lifted to sequences for WoR candidates). One cluster per tree,
// the slice layout and cluster reductions of the RRS walk. The tree is traversed depth first,
// children in slot order; a node is tried only after every child subtree below it has been
// rejected, and is then accepted iff U[accept, node] < p_a(node) (the root always). Entering
// child c (token y) of u gives p_a(c) = min(p_a(u) Mb_u(y) / Ms_u(y), 1). After k rejected
// child subtrees, u's target-side law is Mb_k = max(P0 - A_k Q, 0) / D_k (A_0 = 0, D_0 = 1),
// Ms_k = Q / t_k over the tokens not yet rejected, and the update after the next rejection is
//     A_{k+1} = A_k + D_k / (p_a t_k),  D_{k+1} = sum_v max(P0(v) - A_{k+1} Q(v), 0),
//     S = p_a D_{k+1} / D_k,  p_a <- S / (S + 1 - p_a),  t_{k+1} = t_k - Q(y):
// the residual max(p_a Mb_k - Ms_k, 0) = (p_a / D_k) max(P0 - A_{k+1} Q, 0) (subtracting
// non-negative multiples of Q and clamping compose, and a rejected token already has zero
// residual). Each update is one pass over u's slices of P0 and Q that only sums; the slices
// are staged again when the walk returns to u after staging another node. A child whose
// weight is 0 is rejected without entering it (every node below it has weight 0). An accepted
// node that had children draws its final token from max(P0 - A Q, 0), a leaf its bonus from
// its target row. Every internal node's target log-normaliser (and per-node q-row normaliser)
// comes from the pre-pass; per-depth q normalisers too.
constexpr int kMaxStack = kMaxDepthRows + 2;

struct TravStack {
    int node[kMaxStack], next[kMaxStack], deg[kMaxStack];
    float pa[kMaxStack], A[kMaxStack], D[kMaxStack], th[kMaxStack], tl[kMaxStack];
};

template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_verify_trav(VerifyArgs a) {
    pdl_begin();
    extern __shared__ __align__(16) float dyn[];
    float *P = dyn;
    float *Q = dyn + a.slice;
    __shared__ Scratch sh;
    __shared__ TravStack st;

    cg::cluster_group cluster = cg::this_cluster();
    const int CS = (int)cluster.num_blocks();
    const int crank = (int)cluster.block_rank();
    const int b = blockIdx.x / CS;
    const int lo = crank * a.slice;
    const int n = max(0, min(a.V - lo, a.slice));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool writer = threadIdx.x == 0;  // one writer per CTA: every CTA keeps the same stack
    const bool per_depth = a.qrow_of_node == nullptr;
    int par = 0;
    Walk<T> W{a, sh, cluster, P, Q, par, b, lo, n, (n + kChunk - 1) / kChunk};
    const TreeSmem ts = copy_tree<T>(a, sh, dyn + 2 * a.slice, b, per_depth);
    load_pre(a, sh, ts, b, true);

    auto trow_of = [&](int u) {
        return static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
    };
    auto qrow_of = [&](int u) {
        return static_cast<const T *>(a.q) + (int64_t)b * a.q_bstride + (int64_t)ts.row[u] * a.q_rstride;
    };
    auto l2q_of = [&](int u) { return per_depth ? sh.l2q[ts.row[u]] : ts.l2qn[u]; };

    if (writer) {
        st.node[0] = 0;
        st.next[0] = 0;
        st.deg[0] = 0;
        st.pa[0] = 1.f;
        st.A[0] = 0.f;
        st.D[0] = 1.f;
        st.th[0] = 1.f;
        st.tl[0] = 0.f;
    }
    cluster.sync();  // the copy is complete; every CTA of the cluster runs before any distributed access

    bool bad = sh.cbad != 0;  // every CTA checked the same arrays
    int lev = 0, accepted = -1, final_tok = -1;
    int staged = -1, staged_rej = 0;  // node whose P0 / Q slices are in P / Q; its rejected tokens zeroed

    // u (stack level lv) after the subtree of its child slot ci was rejected
    auto update = [&](int lv, int ci) {
        const int u = st.node[lv], o = ts.off[u];
        const float pa = st.pa[lv];
        const FF L2t = ts.l2t[u], L2q = l2q_of(u);
        const float Qy = exp_shifted(ts.cxq[o + ci], L2q);
        float npa = pa, nA = st.A[lv], nD = st.D[lv];
        int ndeg = 0;
        if (pa > 0.f) {
            const float A1 = __fmaf_rn(st.D[lv], __frcp_rn(__fmul_rn(pa, st.th[lv])), st.A[lv]);
            __syncthreads();  // earlier readers of P and Q are done
            if (staged != u) {
                W.template stage<true>(trow_of(u), P, kWarps, L2t);
                W.template stage<true>(qrow_of(u), Q, kWarps, L2q);
                staged = u;
                staged_rej = 0;
                __syncthreads();
            }
            for (int j = staged_rej + threadIdx.x; j <= ci; j += kThreads) {  // rejected tokens leave P0
                const int y = ts.tok[ts.kid[o + j]];
                if (y >= lo && y < lo + n) P[y - lo] = 0.f;
            }
            staged_rej = ci + 1;
            __syncthreads();
            KahanF zl[2];  // one per half chunk: two independent chains
            for (int cl = warp; cl < W.nch; cl += kWarps) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = Walk<T>::quad_at(cl, h, lane);
                    const float4 x = ld4(P, j), q = ld4(Q, j);
                    const float r0 = fmaxf(__fmaf_rn(-A1, q.x, x.x), 0.f), r1 = fmaxf(__fmaf_rn(-A1, q.y, x.y), 0.f);
                    const float r2 = fmaxf(__fmaf_rn(-A1, q.z, x.z), 0.f), r3 = fmaxf(__fmaf_rn(-A1, q.w, x.w), 0.f);
                    zl[h].add(__fadd_rn(__fadd_rn(r0, r1), __fadd_rn(r2, r3)));
                }
            }
            Slot mine = neutral_slot();
            const FF z = ff_add(zl[0].ff(), zl[1].ff());
            mine.zh = z.hi;
            mine.zl = z.lo;
            reduce_round<kRedSum>(sh, par, cluster, mine);
            const float D1 = sh.res.zh;
            if (D1 > 0.f) {
                const float S = __fmul_rn(__fmul_rn(pa, D1), __frcp_rn(st.D[lv]));
                npa = __fdiv_rn(S, __fadd_rn(S, __fsub_rn(1.f, pa)));
                nA = A1;
                nD = D1;
            } else if (pa < 1.f) {
                npa = 0.f;
            } else {
                ndeg = 1;  // no residual mass with p_a = 1 (rounding only)
            }
        }
        const FF t = ff_add(FF{st.th[lv], st.tl[lv]}, FF{-Qy, 0.f});
        __syncthreads();  // every thread has read the level's state
        if (writer) {
            st.pa[lv] = npa;
            st.A[lv] = nA;
            st.D[lv] = nD;
            st.deg[lv] = ndeg;
            st.th[lv] = t.hi;
            st.tl[lv] = t.lo;
        }
        __syncthreads();
    };

    for (int iter = 0; !bad; ++iter) {
        if (iter > 2 * (a.N + 1) + 2) {  // each node is entered and left once: cannot happen
            bad = true;
            break;
        }
        const int u = st.node[lev];
        const int o = ts.off[u], m = ts.off[u + 1] - o;
        const int i = st.next[lev];
        if (st.deg[lev] == 0 && i < m) {  // the next child subtree
            const int c = ts.kid[o + i];
            const int y = ts.tok[c];
            const float pa = st.pa[lev];
            float w = 0.f;
            bool drawn = false;  // a token repeated among rejected siblings: no residual mass left
            for (int j = 0; j < i; ++j) drawn |= ts.tok[ts.kid[o + j]] == y;
            if (pa > 0.f && !drawn) {
                const float P0y = exp_shifted(ts.cxt[o + i], ts.l2t[u]);
                const float Qy = exp_shifted(ts.cxq[o + i], l2q_of(u));
                const float num = __fmul_rn(pa, __fmul_rn(fmaxf(__fmaf_rn(-st.A[lev], Qy, P0y), 0.f),
                                                          __frcp_rn(st.D[lev])));
                const float qp = __fmul_rn(Qy, __frcp_rn(st.th[lev]));
                w = qp > 0.f ? fminf(__fdiv_rn(num, qp), 1.f) : (num > 0.f ? 1.f : 0.f);
            }
            if (w > 0.f && lev + 1 >= min(a.L + 1, kMaxStack)) {  // deeper than the depth cap
                bad = true;
                break;
            }
            __syncthreads();  // every thread has read the level's state
            if (writer) {
                st.next[lev] = i + 1;
                if (w > 0.f) {
                    st.node[lev + 1] = c;
                    st.next[lev + 1] = 0;
                    st.deg[lev + 1] = 0;
                    st.pa[lev + 1] = w;
                    st.A[lev + 1] = 0.f;
                    st.D[lev + 1] = 1.f;
                    st.th[lev + 1] = 1.f;
                    st.tl[lev + 1] = 0.f;
                }
            }
            __syncthreads();
            if (w > 0.f)
                ++lev;
            else
                update(lev, i);  // a weight-0 subtree is rejected without entering it
            continue;
        }
        // u is a leaf of the remaining tree
        bool acc = true;
        if (lev > 0 && st.deg[lev] == 0) {
            const int pu = st.node[lev - 1];
            acc = ts.cu[ts.off[pu] + st.next[lev - 1] - 1] < st.pa[lev];
        }
        if (acc) {
            accepted = lev;
            if (m == 0 || st.deg[lev] != 0) {  // bonus from the node's target row
                final_tok = W.draw_from_row(trow_of(u), u);
            } else {  // every child rejected: from max(P0 - A Q, 0)
                if (staged != u) {  // cannot happen: the last update staged u (p_a > 0)
                    bad = true;
                    break;
                }
                const float A = st.A[lev];
                final_tok = W.template draw<false>(u, [&](int j, float *v) {
                    const float4 x = ld4(P, j), q = ld4(Q, j);
                    v[0] = fmaxf(__fmaf_rn(-A, q.x, x.x), 0.f);
                    v[1] = fmaxf(__fmaf_rn(-A, q.y, x.y), 0.f);
                    v[2] = fmaxf(__fmaf_rn(-A, q.z, x.z), 0.f);
                    v[3] = fmaxf(__fmaf_rn(-A, q.w, x.w), 0.f);
                });
                if (final_tok < 0) final_tok = W.draw_from_row(trow_of(u), u);  // no mass (rounding)
            }
            break;
        }
        --lev;  // u's subtree is rejected: update its parent
        update(lev, st.next[lev] - 1);
    }
    if (writer && crank == 0) {
        int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
        int32_t *onode = a.out_nodes + (int64_t)b * a.L;
        const int nacc = bad ? 0 : accepted;
        if (bad) raise_status(a.status, kDevBadTree);
        for (int k = 0; k < nacc; ++k) {
            otok[k] = ts.tok[st.node[k + 1]];
            onode[k] = st.node[k + 1];
        }
        otok[nacc] = bad ? -1 : final_tok;
        for (int k = nacc + 1; k <= a.L; ++k) otok[k] = -1;
        for (int k = nacc; k < a.L; ++k) onode[k] = -1;
        a.out_len[b] = bad ? 0 : nacc + 1;
    }
    cluster.sync();  // no CTA leaves while another may still read its shared memory
}

// Target-sample matching's pre-pass: the draw of each of the first kNaiveChain nodes of every
// tree's first-child chain (the nodes a walk most likely visits; the chain's first leaf
// included), all rows at once over the GPU, one cluster of kNaiveSplit CTAs per (tree, chain
// position): CTA r takes the r-th quarter of the row's chunks, chunk log-masses with one warp per
// chunk (lane l holds logits 8l..8l+7) and U chunks per warp iteration (all loads issued first,
// the U sums reduced together), the chunk keys; the CTAs' best keys meet in CTA 0 through
// distributed shared memory and one of its warps draws the token inside the best chunk. The
// token goes to the node's workspace slot.
constexpr int kNaiveChain = 10;
constexpr int kNaiveSplit = 4;
constexpr int kNaiveWarps = 4;

// Node j of the first-child chain from the root, leaves included (the chain ends at its first
// leaf); -1 past the end or on inconsistent arrays.
__device__ __forceinline__ int chain_node_to_leaf(const int32_t *off, const int32_t *kid, int N, int j) {
    int v = 0;
    for (int k = 0; k < j; ++k) {
        const int o = off[v];
        if (off[v + 1] - o <= 0 || o < 0 || o >= N) return -1;
        const int c = kid[o];
        if (c < 1 || c > N) return -1;
        v = c;
    }
    return v;
}

template <typename T>
__global__ void __launch_bounds__(kNaiveWarps * 32, 8) k_naive_pre(VerifyArgs a) {
    pdl_begin();
    constexpr int U = sizeof(T) == 2 ? 8 : 4;  // chunks per warp iteration (16-byte loads in flight per lane)
    __shared__ uint64_t s_best[kNaiveWarps];
    __shared__ uint64_t s_part;  // this CTA's best chunk key
    __shared__ int s_node;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int NN = a.N + 1;
    const int rid = blockIdx.x / kNaiveSplit;
    const int b = rid / a.M, j = rid - (rid / a.M) * a.M;
    if (threadIdx.x == 0) {  // the chain's j-th node (every CTA of the cluster finds the same)
        const int32_t *off = a.child_off + (int64_t)b * (NN + 1), *kids = a.child_ids + (int64_t)b * a.N;
        int v = 0;
        for (int k = 0; k < j && v >= 0; ++k) {
            const int o = __ldg(off + v);
            if (__ldg(off + v + 1) - o <= 0 || o < 0 || o >= a.N) {
                v = -1;
                break;
            }
            const int c = __ldg(kids + o);
            v = c >= 1 && c <= a.N ? c : -1;
        }
        s_node = v;
    }
    __syncthreads();
    const int u = s_node;
    if (u < 0) return;  // past the chain's end (the whole cluster returns)
    const T *row = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
    const uint32_t ub = (uint32_t)b, un = (uint32_t)u;
    const int per = (a.C + kNaiveSplit - 1) / kNaiveSplit;
    const int c_lo = rank * per, c_hi = min(a.C, c_lo + per);
    const int units = c_hi > c_lo ? (c_hi - c_lo + U - 1) / U : 0;
    uint64_t best = 0ull;
    bool bad = false;
    for (int un0 = warp; un0 < units; un0 += kNaiveWarps) {  // uniform over the warp
        const int cu = c_lo + un0 * U;
        RawGroup<T> raw[U];
#pragma unroll
        for (int k = 0; k < U; ++k)
            if (cu + k < c_hi) raw[k].load(row, (cu + k) * kChunk + lane * 8, a.V);
        float mcs[U], part[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            mcs[k] = -INFINITY;
            part[k] = 0.f;
            if (cu + k >= c_hi) continue;  // uniform over the warp
            float z[8];
            raw[k].unpack(z);  // padding past V is -inf
            float zm = z[0];
#pragma unroll
            for (int i = 1; i < 8; ++i) zm = fmaxf(zm, z[i]);
            mcs[k] = __fmul_rn(warp_max(zm), a.invT);
            const float2 offs = exp_offset(mcs[k]);
#pragma unroll
            for (int i = 0; i < 8; ++i) part[k] += chunk_term(z[i], a.invT, offs.x);
            part[k] = chunk_sum_fix(part[k], offs.y);
        }
        // the U chunk sums at once; the lane holding a chunk's sum keys that chunk
        const float tot = warp_multi_sum<U>(part);
        const int ch = multi_sum_index<U>(lane), c = cu + ch;
        if (lane % (32 / U) == 0 && c < c_hi) {
            float mc = mcs[0];
#pragma unroll
            for (int k = 1; k < U; ++k) mc = ch == k ? mcs[k] : mc;
            bad |= !(tot == tot) || isinf(mc);
            const uint32_t w = draw_word(a.seed, kFinalChunk, ub, un, (uint32_t)c);
            const uint64_t k = pack_key(__fadd_rn(__fadd_rn(mc, logf(tot)), gumbel_of(w)), (uint32_t)c);
            best = k > best ? k : best;
        }
    }
    if (__any_sync(kFull, bad) && lane == 0) raise_status(a.status, kDevNonFinite);
    best = warp_max_u64(best);
    if (lane == 0) s_best[warp] = best;
    __syncthreads();
    if (warp == 0) {
        const uint64_t v = warp_max_u64(lane < kNaiveWarps ? s_best[lane] : 0ull);
        if (lane == 0) s_part = v;
    }
    cluster.sync();  // every CTA's best chunk key is published
    uint64_t cb = 0ull;
    if (rank == 0 && warp == 0) cb = warp_max_u64(lane < kNaiveSplit ? *cluster.map_shared_rank(&s_part, lane) : 0ull);
    cluster.sync();  // CTA 0 has read the others; they may leave
    if (rank != 0 || warp != 0) return;
    int32_t *slot = reinterpret_cast<int32_t *>(&a.pre[(int64_t)b * NN + u].pad[0]);
    if (cb == 0ull) {  // no finite logit (status already raised)
        if (lane == 0) *slot = -1;
        return;
    }
    const int c = (int)key_id(cb);
    const int v0 = c * kChunk + lane * 8;
    float x[8];
    Logit<T>::load8(row, v0, a.V, x);
    const Words4 w0 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2));
    const Words4 w1 = draw_block(a.seed, kFinal, ub, un, (uint32_t)(v0 >> 2) + 1u);
    uint64_t tk = 0ull;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        if (v0 + i < a.V) {
            const uint32_t wi = i < 4 ? w0.w[i] : w1.w[i - 4];
            const uint64_t k = pack_key(__fadd_rn(__fmul_rn(x[i], a.invT), gumbel_of(wi)), (uint32_t)(v0 + i));
            tk = k > tk ? k : tk;
        }
    }
    tk = warp_max_u64(tk);
    if (lane == 0) *slot = tk == 0ull ? -1 : (int32_t)key_id(tk);
}

// Target-sample matching ("Naive" in Table 2; Sec. 2.3) by walking: at the current node u a
// token y is drawn from the target law p_u with the two-level Gumbel-max of the bonus token
// (chunk keys log(chunk mass) + G(U[final chunk, u, c]), then x_v + G(U[final, u, v]) inside
// the best chunk); the first child of u carrying y is accepted and the walk continues there,
// otherwise y is the final token (at a leaf: the bonus token). One cluster per tree with the
// RRS walk's slices; the first kNaiveChain nodes of the first-child chain come drawn from the
// pre-pass, any other visit stages the node's target row (its x into P) and draws, so only the
// chain's rows and the visited ones are read. A row holding a NaN or +inf logit sets the
// non-finite status bit. Which kernel draws a node depends only on the topology.
template <typename T>
__global__ void __launch_bounds__(kThreads, 1) k_verify_naive(VerifyArgs a) {
    extern __shared__ __align__(16) float dyn[];
    float *P = dyn;
    float *Q = dyn + a.slice;
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
    Walk<T> W{a, sh, cluster, P, Q, par, b, lo, n, (n + kChunk - 1) / kChunk};

    int32_t *s_off = reinterpret_cast<int32_t *>(dyn + 2 * a.slice);  // [N+2]
    int32_t *s_kid = s_off + (NN + 1);                                // [N]
    int32_t *s_tok = s_kid + a.N;                                     // [N+1]
    int32_t *s_pre = s_tok + NN;                                      // [N+1] pre-drawn token, -2 none
    // the tree and tokens (complete before the pre-pass passed its own wait, and not written by
    // it) before waiting for the pre-pass, then the pre-drawn tokens of the chain's nodes
    for (int i = threadIdx.x; i <= NN; i += kThreads) s_off[i] = __ldg(a.child_off + (int64_t)b * (NN + 1) + i);
    for (int i = threadIdx.x; i < a.N; i += kThreads) s_kid[i] = __ldg(a.child_ids + (int64_t)b * a.N + i);
    for (int i = threadIdx.x; i < NN; i += kThreads) {
        s_tok[i] = __ldg(a.token + (int64_t)b * NN + i);
        s_pre[i] = -2;
    }
    pdl_begin();
    __syncthreads();
    if (threadIdx.x < a.M) {
        const int v = chain_node_to_leaf(s_off, s_kid, a.N, threadIdx.x);
        if (v >= 0) s_pre[v] = *reinterpret_cast<const int32_t *>(&a.pre[(int64_t)b * NN + v].pad[0]);
    }
    __syncthreads();
    cluster.sync();  // every CTA of the cluster runs before any distributed access

    int u = 0, nacc = 0, final_tok = -1;
    bool bad = false;
    for (int step = 0; step <= a.L; ++step) {
        const T *trow = static_cast<const T *>(a.target) + (int64_t)b * a.t_bstride + (int64_t)u * a.t_rstride;
        // every CTA holds the same y: pre-drawn, or drawn here from the node's staged row
        const int y = s_pre[u] != -2 ? s_pre[u] : W.template draw_from_row<true>(trow, u);
        const int o = s_off[u], m = s_off[u + 1] - o;
        if (o < 0 || m < 0 || m > kMaxK || o + m > a.N) {
            bad = true;
            break;
        }
        int next = -1;
        for (int i = 0; i < m && y >= 0; ++i) {
            const int c = s_kid[o + i];
            if (c < 1 || c > a.N) {
                bad = true;
                break;
            }
            if (s_tok[c] == y) {
                next = c;
                break;
            }
        }
        if (bad || next < 0) {
            final_tok = y;
            break;
        }
        if (nacc >= a.L) {  // deeper than the depth cap: the tree arrays are inconsistent
            bad = true;
            break;
        }
        if (writer) sh.path[nacc] = next;  // no global store while cluster barriers follow
        ++nacc;
        u = next;
    }
    if (writer) {
        int32_t *otok = a.out_tokens + (int64_t)b * (a.L + 1);
        int32_t *onode = a.out_nodes + (int64_t)b * a.L;
        if (bad) raise_status(a.status, kDevBadTree);
        if (!bad && final_tok < 0) raise_status(a.status, kDevNonFinite);  // no finite logit to draw
        const int k_acc = bad ? 0 : nacc;
        for (int k = 0; k < k_acc; ++k) {
            otok[k] = s_tok[sh.path[k]];
            onode[k] = sh.path[k];
        }
        otok[k_acc] = bad ? -1 : final_tok;
        for (int k = k_acc + 1; k <= a.L; ++k) otok[k] = -1;
        for (int k = k_acc; k < a.L; ++k) onode[k] = -1;
        a.out_len[b] = bad ? 0 : k_acc + 1;
    }
    cluster.sync();  // no CTA leaves while another may still read its shared memory
}

constexpr size_t kSmemLimit = 210 * 1024;

// Chunk-aligned slice of each CTA and the dynamic shared memory it needs for cluster size cs
// (SIZE_MAX when the slice exceeds the per-CTA chunk table).
void slice_for(int V, int N, int cs, int *slice_out, size_t *smem_out) {
    int slice = (V + cs - 1) / cs;
    slice = (slice + kChunk - 1) / kChunk * kChunk;
    *slice_out = slice;
    *smem_out = slice > kMaxSliceChunks * kChunk ? (size_t)-1 : 2 * (size_t)slice * sizeof(float) + topo_bytes(N);
}

struct ClusterChoice {
    int V, N, B, elem, cs;
};

// The cluster size for (V, N, B): the largest size up to 16 (above 8 the cluster is
// non-portable) whose clusters can all be resident at once, so every tree walks in the same
// wave; when no size fits the whole batch, the size with the most concurrently resident
// CTAs. Decisions are cached per (V, N, B, element size); the cache is a pure function of
// the device.
template <typename T>
int choose_cluster(int V, int N, int B, int *slice_out, size_t *smem_out) {
    static ClusterChoice cache[16];
    static int cache_n = 0;
    static std::mutex mu;
    {
        std::lock_guard<std::mutex> g(mu);
        for (int i = 0; i < cache_n; ++i)
            if (cache[i].V == V && cache[i].N == N && cache[i].B == B && cache[i].elem == (int)sizeof(T)) {
                slice_for(V, N, cache[i].cs, slice_out, smem_out);
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
        slice_for(V, N, cs, &slice, &smem);
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
        slice_for(V, N, 16, &slice, &smem);
        chosen = smem <= kSmemLimit ? 16 : -1;
    }
    if (chosen > 0) {
        std::lock_guard<std::mutex> g(mu);
        if (cache_n < 16) cache[cache_n++] = ClusterChoice{V, N, B, (int)sizeof(T), chosen};
        slice_for(V, N, chosen, slice_out, smem_out);
    }
    return chosen;
}

// The pre-pass kernel for a's pre-computed set (target rows of M nodes per tree, q-row
// normalisers), launched ahead of a walk.
int64_t pre_blocks_of(const VerifyArgs &a, int B) {
    const int per = a.qn ? a.N + 1 : a.Lq;
    int64_t pre_blocks = 2 * (int64_t)B * a.M + ((int64_t)B * per + kPreThreads / 32 - 1) / (kPreThreads / 32);
    return pre_blocks + (pre_blocks & 1);  // whole clusters of two (a spare q-row CTA finds no task)
}
bool pre_launched(const VerifyArgs &a, int B) { return pre_blocks_of(a, B) > 0; }

template <typename T>
cudaError_t launch_pre_t(const VerifyArgs &a, int B, cudaStream_t s) {
    const int64_t pre_blocks = pre_blocks_of(a, B);
    if (pre_blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    if (pre_blocks == 0) return cudaSuccess;
    const size_t psmem = (size_t)a.C * sizeof(float2) + (a.pre_chain ? (size_t)(2 * a.N + 2) * sizeof(int32_t) : 0);
    cudaError_t e = cudaFuncSetAttribute(k_verify_pre<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)psmem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_verify_pre<T>, dim3((unsigned)pre_blocks), dim3(kPreThreads), psmem, s, 2, a);
}

// The split pre-pass's grid: kPreSplit CTAs per chain row, then the q-row normaliser warps.
int64_t pre_split_blocks(const VerifyArgs &a, int B) {
    const int per = a.qn ? a.N + 1 : a.Lq;
    return (int64_t)B * kPreChain * kPreSplit + ((int64_t)B * per + kPreSplitThreads / 32 - 1) / (kPreSplitThreads / 32);
}

// The RRS walk's cluster shape and shared memory, set on the kernel before any launch.
template <typename T>
cudaError_t prepare_rrs_walk(VerifyArgs &a, int B, int *cs_out, size_t *smem_out) {
    int slice = 0;
    size_t smem = 0;
    const int cs = choose_cluster<T>(a.V, a.N, B, &slice, &smem);
    if (cs < 0) return cudaErrorInvalidValue;
    a.slice = slice;
    cudaError_t e = cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (cs > 8) {
        e = cudaFuncSetAttribute(k_verify_rrs<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    *cs_out = cs;
    *smem_out = smem;
    return cudaSuccess;
}

template <typename T>
cudaError_t launch_rrs_t(VerifyArgs a, int B, cudaStream_t s) {
    int cs = 0;
    size_t smem = 0;
    cudaError_t e = prepare_rrs_walk<T>(a, B, &cs, &smem);
    if (e != cudaSuccess) return e;
    const int64_t blocks = pre_split_blocks(a, B);
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const size_t psmem = pre_split_smem(a.C, a.N);
    e = cudaFuncSetAttribute(k_pre_split<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)psmem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_pre_split<T>, dim3((unsigned)blocks), dim3(kPreSplitThreads), psmem, s, 0, a);
    if (e != cudaSuccess) return e;
    a.copy_early = 1;  // the walk copies its tree and tokens while the pre-pass runs
    return launch_pdl(k_verify_rrs<T>, dim3((unsigned)(B * cs)), dim3(kThreads), smem, s, cs, a);
}

template <int KCAP, typename T>
cudaError_t launch_replay_verify_t(const ReplayArgs &ra, VerifyArgs a, int B, cudaStream_t s) {
    int cs = 0;
    size_t smem = 0;
    cudaError_t e = prepare_rrs_walk<T>(a, B, &cs, &smem);
    if (e != cudaSuccess) return e;
    const int64_t nrep = (int64_t)B * (a.N + 1), npre = pre_split_blocks(a, B);
    if (nrep + npre > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const size_t rsmem = (size_t)key_buf_len(a.C) * sizeof(uint64_t), psmem = pre_split_smem(a.C, a.N);
    const size_t smem1 = rsmem > psmem ? rsmem : psmem;
    e = cudaFuncSetAttribute(k_replay_pre<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return e;
    e = launch_pdl(k_replay_pre<KCAP, T>, dim3((unsigned)(nrep + npre)), dim3(kRpThreads), smem1, s, 0, ra, a,
                   (int)nrep);
    if (e != cudaSuccess) return e;
    a.copy_early = 1;  // the topology before the wait,
    a.tokens_late = 1; // the tokens after it
    return launch_pdl(k_verify_rrs<T>, dim3((unsigned)(B * cs)), dim3(kThreads), smem, s, cs, a);
}

template <typename T>
cudaError_t launch_trav_t(VerifyArgs a, int B, cudaStream_t s) {
    int slice = 0;
    size_t smem = 0;
    const int cs = choose_cluster<T>(a.V, a.N, B, &slice, &smem);  // same slices and shared memory
    if (cs < 0) return cudaErrorInvalidValue;
    a.slice = slice;
    cudaError_t e = cudaFuncSetAttribute(k_verify_trav<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (cs > 8) {
        e = cudaFuncSetAttribute(k_verify_trav<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    e = launch_pre_t<T>(a, B, s);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_verify_trav<T>, dim3((unsigned)(B * cs)), dim3(kThreads), smem, s, cs, a);
}

template <typename T>
cudaError_t launch_naive_walk_t(VerifyArgs a, int B, cudaStream_t s) {
    int slice = 0;
    size_t smem = 0;
    const int cs = choose_cluster<T>(a.V, a.N, B, &slice, &smem);  // the RRS walk's slices
    if (cs < 0) return cudaErrorInvalidValue;
    a.slice = slice;
    cudaError_t e = cudaFuncSetAttribute(k_verify_naive<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (cs > 8) {
        e = cudaFuncSetAttribute(k_verify_naive<T>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    e = launch_pdl(k_naive_pre<T>, dim3((unsigned)(B * a.M * kNaiveSplit)), dim3(kNaiveWarps * 32), 0, s,
                   kNaiveSplit, a);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_verify_naive<T>, dim3((unsigned)(B * cs)), dim3(kThreads), smem, s, cs, a);
}

VerifyArgs verify_args(const RowsDesc &target, const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node,
                       int B, int N, int L, const TreeDesc &tree, const int32_t *token, float invT, uint64_t seed,
                       int32_t *out_tokens, int32_t *out_nodes, int32_t *out_len, uint32_t *status) {
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
    // the pre-pass results use the workspace's per-(tree, node) slots (status word is ws[0])
    a.pre = reinterpret_cast<PreRow *>(reinterpret_cast<char *>(status) + kWsStatusBytes);
    a.M = 0;
    a.pre_chain = 0;
    a.copy_early = 0;
    a.Lq = qrow_of_node ? 0 : (L < N + 1 ? L : N + 1);
    a.qn = 0;
    a.B = B;
    a.part = reinterpret_cast<float4 *>(reinterpret_cast<char *>(status) + ws_pre_part_offset(B, N));
    a.tokens_late = 0;
    return a;
}

}  // namespace

cudaError_t launch_verify_traversal(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                    const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                                    const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                    int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyArgs a = verify_args(target, q, qstats, qrow_of_node, B, N, L, tree, token, invT, seed, out_tokens,
                               out_nodes, out_len, status);
    a.M = N + 1;                       // every internal node's target normaliser
    a.qn = qrow_of_node ? 1 : 0;       // and, for per-node q rows, each internal node's q normaliser
    if (target.dtype == 1) return launch_trav_t<__nv_bfloat16>(a, B, s);
    return launch_trav_t<float>(a, B, s);
}

cudaError_t launch_verify_rrs(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                              const int32_t *qrow_of_node, int B, int N, int L, const TreeDesc &tree,
                              const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                              int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyArgs a = verify_args(target, q, qstats, qrow_of_node, B, N, L, tree, token, invT, seed, out_tokens,
                               out_nodes, out_len, status);
    a.M = kPreChain;  // the first-child chain's first internal nodes from the pre-pass
    a.pre_chain = 1;
    a.qn = qrow_of_node ? 1 : 0;  // per-node q rows: every internal node's normaliser
    if (target.dtype == 1) return launch_rrs_t<__nv_bfloat16>(a, B, s);
    return launch_rrs_t<float>(a, B, s);
}

cudaError_t launch_replay_verify(const RowsDesc &target, const RowsDesc &q, const float2 *qstats,
                                 const int32_t *qrow_of_node, int B, int N, int L, int K, const TreeDesc &tree,
                                 int32_t *token, float invT, uint64_t seed, int32_t *out_tokens, int32_t *out_nodes,
                                 int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyArgs a = verify_args(target, q, qstats, qrow_of_node, B, N, L, tree, token, invT, seed, out_tokens,
                               out_nodes, out_len, status);
    a.M = kPreChain;
    a.pre_chain = 1;
    a.qn = qrow_of_node ? 1 : 0;
    const ReplayArgs ra = replay_args(q, qstats, qrow_of_node, B, N, tree, invT, seed, token, status);
    // sibling groups have at most K members: a list of 8 covers K <= 8 (as in launch_replay)
    if (target.dtype == 1)
        return K <= 8 ? launch_replay_verify_t<8, __nv_bfloat16>(ra, a, B, s)
                      : launch_replay_verify_t<32, __nv_bfloat16>(ra, a, B, s);
    return K <= 8 ? launch_replay_verify_t<8, float>(ra, a, B, s) : launch_replay_verify_t<32, float>(ra, a, B, s);
}

cudaError_t launch_verify_naive(const RowsDesc &target, int B, int N, int L, const TreeDesc &tree,
                                const int32_t *token, float invT, uint64_t seed, int32_t *out_tokens,
                                int32_t *out_nodes, int32_t *out_len, uint32_t *status, cudaStream_t s) {
    VerifyArgs a = verify_args(target, target, nullptr, nullptr, B, N, L, tree, token, invT, seed, out_tokens,
                               out_nodes, out_len, status);
    a.q = nullptr;
    a.q_R = 0;
    a.Lq = 0;
    a.M = N + 1 < kNaiveChain ? N + 1 : kNaiveChain;  // chain positions drawn by the pre-pass
    if (target.dtype == 1) return launch_naive_walk_t<__nv_bfloat16>(a, B, s);
    return launch_naive_walk_t<float>(a, B, s);
}

}  // namespace tsb
