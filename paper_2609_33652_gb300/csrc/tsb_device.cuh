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

constexpr uint32_t kDevNonFinite = 1u, kDevBadIndex = 2u, kDevBadTree = 4u;

__device__ __forceinline__ void raise_status(uint32_t *status, uint32_t bits) { atomicOr(status, bits); }

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
// Warp reductions (butterfly: every lane ends with the result).
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFull, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t w = __shfl_xor_sync(kFull, v, o);
        v = w > v ? w : v;
    }
    return v;
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
};

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
};

// Merge the lanes' lists: out[j] (j < n) = j-th largest key over the warp (0 if fewer keys).
// Every lane receives every key; n <= CAP. Keys must be distinct (they carry their id).
template <int CAP>
__device__ __forceinline__ void warp_merge_top(TopList<CAP> &list, int n, uint64_t *out) {
    for (int j = 0; j < n; ++j) {
        const uint64_t best = warp_max_u64(list.k[0]);
        out[j] = best;
        if (best != 0ull && list.k[0] == best) list.pop_front();
    }
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
};

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

constexpr float kLog2e = 1.4426950408889634f;

}  // namespace tsb
