// Device primitives of libtsb: counter-based uniforms, Gumbel keys, order-preserving key
// packing, warp reductions and per-lane sorted candidate lists.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tsb {

constexpr int kChunk = 256;   // logits per chunk (chunk statistics, replay sampler)
constexpr int kMaxK = 32;
constexpr unsigned kFull = 0xffffffffu;

enum Purpose : uint32_t { kReplayChunk = 0, kReplayElem = 1, kAccept = 2, kFinal = 3, kBlockEta = 4, kFinalChunk = 5 };

constexpr uint32_t kDevNonFinite = 1u, kDevBadIndex = 2u, kDevBadTree = 4u, kDevCheck = 8u;

__device__ __forceinline__ void raise_status(uint32_t *status, uint32_t bits) { atomicOr(status, bits); }

// Bounds check of a data-dependent index (a shared-memory fill position from an atomic counter,
// a node, token or row index read from the caller's arrays). In the checked build (TSB_CHECKED)
// an index outside [0, n) sets kDevCheck in the status word (when there is one) and the caller
// skips the access; otherwise it returns true and compiles to nothing.
__device__ __forceinline__ bool in_bounds(long long i, long long n, uint32_t *status) {
#ifdef TSB_CHECKED
    if (i >= 0 && i < n) return true;
    if (status) raise_status(status, kDevCheck);
    return false;
#else
    (void)i;
    (void)n;
    (void)status;
    return true;
#endif
}

// ---------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror & Shaw, SC 2011): ten rounds of two 32x32->64
// multiplies with xor-mixing; the key advances by the golden-ratio Weyl constants.
struct Words4 {
    uint32_t w[4];
};

__device__ __forceinline__ Words4 philox10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                           uint32_t k1) {
#pragma unroll
    for (int round = 0; round < 10; ++round) {
        const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
        const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
        const uint32_t n0 = hi1 ^ c1 ^ k0;
        const uint32_t n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    Words4 r;
    r.w[0] = c0;
    r.w[1] = c1;
    r.w[2] = c2;
    r.w[3] = c3;
    return r;
}

// The four words of the block holding draws 4j..4j+3 of (purpose, batch, node).
__device__ __forceinline__ Words4 draw_block(uint64_t seed, uint32_t purpose, uint32_t batch, uint32_t node,
                                             uint32_t j) {
    return philox10(j, node, batch, purpose, (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ uint32_t draw_word(uint64_t seed, uint32_t purpose, uint32_t batch, uint32_t node,
                                              uint32_t draw) {
    Words4 b = draw_block(seed, purpose, batch, node, draw >> 2);
    const uint32_t i = draw & 3u;
    return i == 0 ? b.w[0] : i == 1 ? b.w[1] : i == 2 ? b.w[2] : b.w[3];
}

// U = (k + 1/2) 2^-24 with k = w >> 8, rounded to fp32 (exact below 1/2).
__device__ __forceinline__ float uniform_of(uint32_t w) {
    return __fmaf_rn((float)(w >> 8), 5.9604644775390625e-08f, 2.98023223876953125e-08f);
}

// -log U computed from exact operands: for U < 1/2 the uniform itself is exact in fp32;
// for U >= 1/2 its complement 1 - U = (2(2^24-1-k)+1) 2^-25 is, and log1p keeps accuracy.
__device__ __forceinline__ float neg_log_uniform(uint32_t w) {
    const uint32_t k = w >> 8;
    if (k < (1u << 23)) {
        const float u = (float)(2u * k + 1u) * 2.98023223876953125e-08f;
        return -logf(u);
    }
    const float c = (float)(2u * ((1u << 24) - 1u - k) + 1u) * 2.98023223876953125e-08f;
    return -log1pf(-c);
}

// Standard Gumbel G = -log(-log U) of a draw word.
__device__ __forceinline__ float gumbel_of(uint32_t w) { return -logf(neg_log_uniform(w)); }

// Gumbel key g of the top-down construction shifted to the law conditional on its chunk's
// maximum Z being T (Kool, van Hoof & Welling 2019, App. B; the stable softplus form):
// T - softplus(T - g + log1p(-exp(g - Z))).
__device__ __forceinline__ float shifted_gumbel_key(float T, float Z, float g) {
    const float u = T - g + log1pf(-expf(g - Z));
    const float sp = fmaxf(u, 0.f) + log1pf(expf(-fabsf(u)));
    return T - sp;
}

// ---------------------------------------------------------------------------------------
// Keys. A (value desc, id asc) order is packed into one u64 so that "larger u64 first" is
// the order: high word = order-preserving image of the fp32 value, low word = ~id.
__device__ __forceinline__ uint32_t ord_f32(float f) {
    const uint32_t u = __float_as_uint(__fadd_rn(f, 0.0f));  // -0 -> +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float f32_of_ord(uint32_t o) {
    return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
__device__ __forceinline__ uint64_t pack_key(float value, uint32_t id) {
    return ((uint64_t)ord_f32(value) << 32) | (uint64_t)(~id);
}
__device__ __forceinline__ uint32_t key_id(uint64_t k) { return ~(uint32_t)k; }
__device__ __forceinline__ float key_value(uint64_t k) { return f32_of_ord((uint32_t)(k >> 32)); }

// ---------------------------------------------------------------------------------------
// Warp reductions (butterfly: every lane ends with the result). Each starts with __syncwarp():
// a warp that reaches a full-mask shuffle still split from earlier divergent code (a lane-0
// store, a loop with lane-dependent trip counts; a CTA barrier does not merge it) pays a
// synchronisation at every shuffle, measured at ~500 cycles each on GB300 against ~16 once
// the warp is converged.
// Warp maximum of a float in one instruction (redux.sync.max.f32, sm_100a family); like
// fmaxf, NaN inputs are ignored unless every input is NaN.
__device__ __forceinline__ float warp_max(float v) {
    __syncwarp();
    float r;
    asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
    return r;
}
__device__ __forceinline__ float warp_sum(float v) {
    __syncwarp();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
    __syncwarp();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
    __syncwarp();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t w = __shfl_xor_sync(kFull, v, o);
        v = w > v ? w : v;
    }
    return v;
}

// Warp sums of U per-lane partials at once (U = 2, 4 or 8), for U chunks read side by side:
// each halving step exchanges half of the remaining partials with the lane 16, 8, ... apart,
// then the last partial is summed over the remaining lanes. On return every lane holds the
// total of partial multi_sum_index<U>(lane); the lanes with lane % (32 / U) == 0 hold the U
// totals once each. 2U - 1 + log2(32 / U) shuffles in place of 5U.
template <int U>
__device__ __forceinline__ int multi_sum_index(int lane) {
    static_assert(U == 2 || U == 4 || U == 8, "U");
    return U == 8 ? ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1)
                  : (U == 4 ? ((lane >> 4) & 1) * 2 + ((lane >> 3) & 1) : (lane >> 4) & 1);
}
template <int U>
__device__ __forceinline__ float warp_multi_sum(const float (&v)[U]) {
    __syncwarp();
    const int lane = threadIdx.x & 31;
    float c8[8];
#pragma unroll
    for (int j = 0; j < U; ++j) c8[j] = v[j];
    if (U == 8) {  // offset 16: keep four
        const bool up = (lane & 16) != 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float send = up ? c8[j] : c8[j + 4], keep = up ? c8[j + 4] : c8[j];
            c8[j] = keep + __shfl_xor_sync(kFull, send, 16);
        }
    }
    if (U >= 4) {  // keep two
        const int off = U == 8 ? 8 : 16;
        const bool up = (lane & off) != 0;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const float send = up ? c8[j] : c8[j + 2], keep = up ? c8[j + 2] : c8[j];
            c8[j] = keep + __shfl_xor_sync(kFull, send, off);
        }
    }
    const int off = U == 8 ? 4 : (U == 4 ? 8 : 16);  // keep one
    {
        const bool up = (lane & off) != 0;
        const float send = up ? c8[0] : c8[1], keep = up ? c8[1] : c8[0];
        c8[0] = keep + __shfl_xor_sync(kFull, send, off);
    }
    float y = c8[0];
#pragma unroll
    for (int o = off >> 1; o > 0; o >>= 1) y += __shfl_xor_sync(kFull, y, o);
    return y;
}

// ---------------------------------------------------------------------------------------
// Float-float arithmetic (an unevaluated sum hi + lo of two fp32 values) for reductions that
// need more than fp32 accuracy without touching the slow fp64 units.

struct FF {
    float hi, lo;
};

// Knuth's TwoSum: a + b = s + e exactly; symmetric in a and b bit for bit.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ FF ff_add(FF a, FF b) {
    float s, e;
    two_sum(a.hi, b.hi, s, e);
    e = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
    const float hi = __fadd_rn(s, e);
    return FF{hi, __fsub_rn(e, __fsub_rn(hi, s))};
}

// a * f for f >= 0 (the product's rounding error is kept through an fma)
__device__ __forceinline__ FF ff_scale(FF a, float f) {
    const float p = __fmul_rn(a.hi, f);
    const float err = __fmaf_rn(a.hi, f, -p);
    const float lo = __fmaf_rn(a.lo, f, err);
    const float hi = __fadd_rn(p, lo);
    return FF{hi, __fsub_rn(lo, __fsub_rn(hi, p))};
}

__device__ __forceinline__ FF ff_shfl_xor(FF v, int o) {
    return FF{__shfl_xor_sync(kFull, v.hi, o), __shfl_xor_sync(kFull, v.lo, o)};
}

__device__ __forceinline__ FF warp_sum_ff(FF v) {
    __syncwarp();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = ff_add(v, ff_shfl_xor(v, o));
    return v;
}

// A partial softmax normaliser: S = sum exp(x - m) over some set of logits.
struct MaxSum {
    float m;
    FF s;
};

// Merge of two partial normalisers (symmetric bit for bit, so butterflies agree in all lanes).
__device__ __forceinline__ MaxSum maxsum_merge(MaxSum a, MaxSum b) {
    const float M = fmaxf(a.m, b.m);
    if (M == -INFINITY) return MaxSum{M, FF{0.f, 0.f}};
    const FF ta = a.m == -INFINITY ? FF{0.f, 0.f} : ff_scale(a.s, expf(__fsub_rn(a.m, M)));
    const FF tb = b.m == -INFINITY ? FF{0.f, 0.f} : ff_scale(b.s, expf(__fsub_rn(b.m, M)));
    return MaxSum{M, ff_add(ta, tb)};
}

__device__ __forceinline__ MaxSum warp_maxsum(MaxSum v) {
    __syncwarp();
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MaxSum w{__shfl_xor_sync(kFull, v.m, o), ff_shfl_xor(v.s, o)};
        v = maxsum_merge(v, w);
    }
    return v;
}

// log(S.hi + S.lo) for S > 0 as float-float, absolute error about 1e-7 at any magnitude:
// S = f 2^k with f in [1, 2); log S = k ln2 + log f + S.lo/S.hi. ln 2 is split Cody-Waite
// style into a head with 12 trailing zero bits (so k * head is exact) and a tail; logf is
// only evaluated on [1, 2), where its result is below 0.7.
__device__ __forceinline__ FF ff_log(FF S) {
    constexpr float kLn2Head = 0.693145751953125f;        // 0x3F317200
    constexpr float kLn2Tail = 1.4286068203094173e-06f;   // ln 2 - head
    int e;
    const float f = __fmul_rn(frexpf(S.hi, &e), 2.0f);
    const float k = (float)(e - 1);
    const float head = __fmul_rn(k, kLn2Head);
    const float tail = __fadd_rn(__fmaf_rn(k, kLn2Tail, logf(f)), __fdiv_rn(S.lo, S.hi));
    float s, err;
    two_sum(head, tail, s, err);
    return FF{s, err};
}

// log2(e) as a head (fp32 rounding) and a tail, so x * log2(e) is carried to ~2^-46.
constexpr float kLog2eHi = 1.44269502162933349609375f;
constexpr float kLog2eLo = 1.925963033500011e-08f;

// (L.hi + L.lo) * log2(e) as float-float.
__device__ __forceinline__ FF ff_times_log2e(FF L) {
    const float hi = __fmul_rn(L.hi, kLog2eHi);
    const float err = __fmaf_rn(L.hi, kLog2eHi, -hi);
    const float lo = __fadd_rn(err, __fmaf_rn(L.hi, kLog2eLo, __fmul_rn(L.lo, kLog2eHi)));
    const float h2 = __fadd_rn(hi, lo);
    return FF{h2, __fsub_rn(lo, __fsub_rn(h2, hi))};
}

// e^(x - L) with L2 = L * log2(e) in float-float: the exponent x log2(e) - L2 is formed with
// two fmas (exact products, one rounding each), then ex2. Relative error about
// |x - L| 2^-24 + the ex2 approximation's few ulp; used identically wherever the same
// probability must come out bit for bit (element passes and point values).
__device__ __forceinline__ float exp_shifted(float x, FF L2) {
    const float a = __fmaf_rn(x, kLog2eHi, -L2.hi);
    const float b = __fmaf_rn(x, kLog2eLo, -L2.lo);
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(__fadd_rn(a, b)));
    return y;
}

// m + log(S) of a normaliser as float-float (the row log-sum-exp).
__device__ __forceinline__ FF maxsum_lse(MaxSum v) {
    const FF l = ff_log(v.s);
    return ff_add(FF{v.m, 0.f}, l);
}

// Compensated (Neumaier) accumulation in fp32.
struct KahanF {
    float s = 0.f, c = 0.f;
    __device__ __forceinline__ void add(float x) {
        const float t = __fadd_rn(s, x);
        if (fabsf(s) >= fabsf(x))
            c = __fadd_rn(c, __fadd_rn(__fsub_rn(s, t), x));
        else
            c = __fadd_rn(c, __fadd_rn(__fsub_rn(x, t), s));
        s = t;
    }
    __device__ __forceinline__ double value() const { return (double)s + (double)c; }
    __device__ __forceinline__ FF ff() const {
        const float hi = __fadd_rn(s, c);
        return FF{hi, __fsub_rn(c, __fsub_rn(hi, s))};
    }
};

// Order-preserving image of an fp64 value as u64 ("larger u64" = larger value; -0 == +0).
__device__ __forceinline__ unsigned long long ord_f64(double d) {
    const unsigned long long u = (unsigned long long)__double_as_longlong(d + 0.0);
    return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}

// ---------------------------------------------------------------------------------------
// Per-lane list of the CAP largest packed keys, kept sorted descending in registers.
// Insertion is a compare-exchange chain (no dynamic indexing, no local memory).
template <int CAP>
struct TopList {
    uint64_t k[CAP];
    __device__ __forceinline__ void clear() {
#pragma unroll
        for (int i = 0; i < CAP; ++i) k[i] = 0ull;
    }
    __device__ __forceinline__ void insert(uint64_t key) {
        if (key <= k[CAP - 1]) return;
#pragma unroll
        for (int i = 0; i < CAP; ++i) {
            const uint64_t hi = key > k[i] ? key : k[i];
            const uint64_t lo = key > k[i] ? k[i] : key;
            k[i] = hi;
            key = lo;
        }
    }
    __device__ __forceinline__ void pop_front() {
#pragma unroll
        for (int i = 0; i < CAP - 1; ++i) k[i] = k[i + 1];
        k[CAP - 1] = 0ull;
    }
    // pop_front where p holds, as selects (no branch: every lane runs the same instructions)
    __device__ __forceinline__ void pop_front_if(bool p) {
#pragma unroll
        for (int i = 0; i < CAP - 1; ++i) k[i] = p ? k[i + 1] : k[i];
        k[CAP - 1] = p ? 0ull : k[CAP - 1];
    }
};

// Number of keys in keys[0..n) larger than v (the keys are distinct); every thread of a warp
// reading the same key is a shared-memory broadcast.
__device__ __forceinline__ int rank_among(const uint64_t *keys, int n, uint64_t v) {
    int r = 0;
    for (int j = 0; j < n; ++j) r += keys[j] > v ? 1 : 0;
    return r;
}

// The largest of the lanes' 64-bit values (distinct unless zero): a hardware max over the
// high words, then over the low words only among the lanes that tie. Returns the value to
// every lane and the lane that holds it in *owner.
__device__ __forceinline__ uint64_t warp_max_u64_owner(uint64_t v, int *owner) {
    __syncwarp();
    const int lane = threadIdx.x & 31;
    const unsigned hi = (unsigned)(v >> 32);
    const unsigned m1 = __reduce_max_sync(kFull, hi);
    unsigned c = __ballot_sync(kFull, hi == m1);
    if (__popc(c) > 1) {
        const unsigned lo = (unsigned)v;
        const unsigned m2 = __reduce_max_sync(kFull, ((c >> lane) & 1u) ? lo : 0u);
        c &= __ballot_sync(kFull, lo == m2);
    }
    *owner = __ffs(c) - 1;
    return __shfl_sync(kFull, v, *owner);
}

// Take the warp's largest key out of the lanes' lists (0 when all lists are empty).
template <int CAP>
__device__ __forceinline__ uint64_t warp_pop_max(TopList<CAP> &list) {
    int owner;
    const uint64_t best = warp_max_u64_owner(list.k[0], &owner);
    list.pop_front_if((threadIdx.x & 31) == owner && best != 0ull);
    return best;
}

// ---------------------------------------------------------------------------------------
// Loads of 8 consecutive logits as fp32. Rows start on 16-byte boundaries; a group that
// would run past V is read element by element and padded with -inf.
template <typename T>
struct Logit;

template <>
struct Logit<float> {
    __device__ __forceinline__ static void load8(const float *row, int v0, int V, float x[8]) {
        if (v0 + 8 <= V) {
            const float4 a = __ldg(reinterpret_cast<const float4 *>(row + v0));
            const float4 b = __ldg(reinterpret_cast<const float4 *>(row + v0 + 4));
            x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
            x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
        } else {
#pragma unroll
            for (int i = 0; i < 8; ++i) x[i] = (v0 + i < V) ? __ldg(row + v0 + i) : -INFINITY;
        }
    }
    __device__ __forceinline__ static float load1(const float *row, int v) { return __ldg(row + v); }
    __device__ __forceinline__ static float neg_inf() { return -INFINITY; }
};

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t bits16) { return __uint_as_float(bits16 << 16); }

template <>
struct Logit<__nv_bfloat16> {
    __device__ __forceinline__ static void load8(const __nv_bfloat16 *row, int v0, int V, float x[8]) {
        if (v0 + 8 <= V) {
            const uint4 a = __ldg(reinterpret_cast<const uint4 *>(row + v0));
            const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                x[2 * i] = __uint_as_float(w[i] << 16);
                x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
            }
        } else {
            const unsigned short *r = reinterpret_cast<const unsigned short *>(row);
#pragma unroll
            for (int i = 0; i < 8; ++i) x[i] = (v0 + i < V) ? bf16_bits_to_f32(__ldg(r + v0 + i)) : -INFINITY;
        }
    }
    __device__ __forceinline__ static float load1(const __nv_bfloat16 *row, int v) {
        return bf16_bits_to_f32(__ldg(reinterpret_cast<const unsigned short *>(row) + v));
    }
    __device__ __forceinline__ static __nv_bfloat16 neg_inf() { return __ushort_as_bfloat16((unsigned short)0xff80u); }
};

template <typename T>
struct RawGroup;  // 8 consecutive logits as raw 16-byte words (loaded now, unpacked later)
template <>
struct RawGroup<__nv_bfloat16> {
    uint4 w;
    __device__ __forceinline__ void load(const __nv_bfloat16 *row, int v0, int V) {
        if (v0 + 8 <= V) {
            w = __ldg(reinterpret_cast<const uint4 *>(row + v0));
        } else {  // ragged tail: missing logits become -inf (0xff80)
            const unsigned short *r = reinterpret_cast<const unsigned short *>(row);
            unsigned short h[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) h[i] = (v0 + i < V) ? __ldg(r + v0 + i) : (unsigned short)0xff80u;
            w.x = h[0] | ((uint32_t)h[1] << 16);
            w.y = h[2] | ((uint32_t)h[3] << 16);
            w.z = h[4] | ((uint32_t)h[5] << 16);
            w.w = h[6] | ((uint32_t)h[7] << 16);
        }
    }
    // logits v0..v0+7 of a copy in shared memory (v0 a multiple of 8)
    __device__ __forceinline__ void load_shared(const unsigned char *zone, int v0) {
        w = *reinterpret_cast<const uint4 *>(zone + 2 * v0);
    }
    __device__ __forceinline__ void unpack(float z[8]) const {
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            z[2 * i] = __uint_as_float(u[i] << 16);
            z[2 * i + 1] = __uint_as_float(u[i] & 0xffff0000u);
        }
    }
};
template <>
struct RawGroup<float> {
    float4 a, b;
    __device__ __forceinline__ void load(const float *row, int v0, int V) {
        if (v0 + 8 <= V) {
            a = __ldg(reinterpret_cast<const float4 *>(row + v0));
            b = __ldg(reinterpret_cast<const float4 *>(row + v0 + 4));
        } else {
            float z[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) z[i] = (v0 + i < V) ? __ldg(row + v0 + i) : -INFINITY;
            a = make_float4(z[0], z[1], z[2], z[3]);
            b = make_float4(z[4], z[5], z[6], z[7]);
        }
    }
    __device__ __forceinline__ void load_shared(const unsigned char *zone, int v0) {
        a = *reinterpret_cast<const float4 *>(zone + 4 * v0);
        b = *reinterpret_cast<const float4 *>(zone + 4 * v0 + 16);
    }
    __device__ __forceinline__ void unpack(float z[8]) const {
        z[0] = a.x; z[1] = a.y; z[2] = a.z; z[3] = a.w;
        z[4] = b.x; z[5] = b.y; z[6] = b.z; z[7] = b.w;
    }
};

template <typename T>
struct RawQuad;  // 4 consecutive logits as raw words (8 bytes of bf16 or 16 of fp32)
template <>
struct RawQuad<__nv_bfloat16> {
    uint2 w;
    // logits v0..v0+3 (v0 a multiple of 4); those at or beyond `end` become -inf (0xff80)
    __device__ __forceinline__ void load(const __nv_bfloat16 *row, int v0, int end) {
        if (v0 + 4 <= end) {
            w = __ldg(reinterpret_cast<const uint2 *>(row + v0));
        } else {
            const unsigned short *r = reinterpret_cast<const unsigned short *>(row);
            unsigned short h[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) h[i] = (v0 + i < end) ? __ldg(r + v0 + i) : (unsigned short)0xff80u;
            w.x = h[0] | ((uint32_t)h[1] << 16);
            w.y = h[2] | ((uint32_t)h[3] << 16);
        }
    }
    __device__ __forceinline__ void unpack(float z[4]) const {
        z[0] = __uint_as_float(w.x << 16);
        z[1] = __uint_as_float(w.x & 0xffff0000u);
        z[2] = __uint_as_float(w.y << 16);
        z[3] = __uint_as_float(w.y & 0xffff0000u);
    }
};
template <>
struct RawQuad<float> {
    float4 w;
    __device__ __forceinline__ void load(const float *row, int v0, int end) {
        if (v0 + 4 <= end) {
            w = __ldg(reinterpret_cast<const float4 *>(row + v0));
        } else {
            float z[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) z[i] = (v0 + i < end) ? __ldg(row + v0 + i) : -INFINITY;
            w = make_float4(z[0], z[1], z[2], z[3]);
        }
    }
    __device__ __forceinline__ void unpack(float z[4]) const {
        z[0] = w.x;
        z[1] = w.y;
        z[2] = w.z;
        z[3] = w.w;
    }
};

// Programmatic dependent launch. Every kernel of the library starts with pdl_begin(): it
// waits until the kernel launched before it on the stream has completed and its memory is
// visible (griddepcontrol.wait; immediate when there is no programmatic dependency), then
// lets the next kernel on the stream be launched (griddepcontrol.launch_dependents). Before
// the wait a kernel touches no global memory, with one exception: the RRS walk, launched right
// after its own pre-pass, first copies its tree, tokens and logits, which were complete before
// the pre-pass passed its own wait (and so before the walk could launch), and none of which the
// pre-pass writes. Launches with the programmatic-serialisation attribute otherwise only
// overlap a kernel's launch and CTA scheduling with its predecessor's tail.
__device__ __forceinline__ void pdl_begin() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

constexpr float kLog2e = 1.4426950408889634f;

// Terms of a chunk sum s_c = sum_v e^(x_v - m_c), x_v = fp32(z_v * invT) (the contract's x,
// one rounding). m_c log2 e is split into the head hi = fp32(m_c log2 e), which every term
// subtracts inside one fma (x log2 e - hi, rounded once: an error relative to that small
// exponent), and the exact remainder lo = m_c log2 e - hi, which would otherwise be an error
// shared by every term of the chunk (up to 2^-24 |m_c log2 e|); it is applied to the sum once,
// s * 2^-lo = s - s lo ln 2 (|lo| < 4e-6, so the omitted second-order term is below 1e-11).
constexpr float kLn2 = 0.6931471805599453f;
__device__ __forceinline__ float2 exp_offset(float mc) {
    const float hi = __fmul_rn(mc, kLog2e);
    const float lo = isfinite(hi) ? __fmaf_rn(mc, kLog2e, -hi) : 0.f;
    return make_float2(hi, lo);
}
__device__ __forceinline__ float chunk_term(float z, float invT, float off_hi) {
    return fast_exp2(__fmaf_rn(__fmul_rn(z, invT), kLog2e, -off_hi));
}
__device__ __forceinline__ float chunk_sum_fix(float s, float off_lo) {
    return __fmaf_rn(s, __fmul_rn(-off_lo, kLn2), s);
}

// Statistics of one 256-logit chunk held by an 8-lane group (lane g holds logits 8g..8g+7 of
// each 64-logit quarter, raw[k] = quarter k): the maximum m_c = fp32(max z * invT) and
// s_c = sum e^(x - m_c) by the chunk_term form above, in a fixed order, then xor 4, 2, 1
// inside the group. Every lane of the warp must call it (the shuffles are warp-wide); a group
// with live == false contributes -inf / 0. Shared by the statistics kernels so that they
// produce the same bits.
// Maximum of a lane's 32 raw logits (exact: the maximum of bf16 values is a bf16 value).
__device__ __forceinline__ float group_max32(const RawGroup<float> (&raw)[4]) {
    float zm = -INFINITY;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        float z[8];
        raw[k].unpack(z);
#pragma unroll
        for (int i = 0; i < 8; ++i) zm = fmaxf(zm, z[i]);
    }
    return zm;
}
__device__ __forceinline__ float group_max32(const RawGroup<__nv_bfloat16> (&raw)[4]) {
    // packed bf16x2 maxima: 16 instructions for 32 logits
    __nv_bfloat162 h[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint4 w = raw[k].w;
        const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&w.x);
        const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&w.y);
        const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162 *>(&w.z);
        const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162 *>(&w.w);
        h[k] = __hmax2(__hmax2(a, b), __hmax2(c, d));
    }
    const __nv_bfloat162 m2 = __hmax2(__hmax2(h[0], h[1]), __hmax2(h[2], h[3]));
    return fmaxf(__low2float(m2), __high2float(m2));
}

template <typename T>
__device__ __forceinline__ void chunk_stats8(const RawGroup<T> (&raw)[4], bool live, float invT, float *mc_out,
                                             float *s_out) {
    __syncwarp();
    float zm = live ? group_max32(raw) : -INFINITY;
    zm = fmaxf(zm, __shfl_xor_sync(kFull, zm, 4));
    zm = fmaxf(zm, __shfl_xor_sync(kFull, zm, 2));
    zm = fmaxf(zm, __shfl_xor_sync(kFull, zm, 1));
    const float mc = __fmul_rn(zm, invT);
    const float2 off = exp_offset(mc);
    float s = 0.f;
    if (live) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            float z[8];
            raw[k].unpack(z);  // unpacked again rather than kept: fewer registers
#pragma unroll
            for (int i = 0; i < 8; ++i) s += chunk_term(z[i], invT, off.x);
        }
        s = chunk_sum_fix(s, off.y);
    }
    __syncwarp();
    s += __shfl_xor_sync(kFull, s, 4);
    s += __shfl_xor_sync(kFull, s, 2);
    s += __shfl_xor_sync(kFull, s, 1);
    *mc_out = mc;
    *s_out = s;
}

}  // namespace tsb
