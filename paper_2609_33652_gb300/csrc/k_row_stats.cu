// Streaming pass over logit rows: per chunk of 256 logits, the maximum m_c and the sum
// s_c = sum exp(x - m_c) of x = fp32(z) * fp32(1/T). The row's log-normaliser, its top-K
// candidate pool (first pass, Sec. 3.1) and the chunk log-masses A_c = m_c + log s_c of
// the replay sampler (Sec. 3.2) all follow from these without touching the row again.
//
// HBM-bound: every logit is read once with 16-byte loads; 8 bytes are written per chunk.
// A warp owns groups of 8 consecutive chunks of a row (lane l holds logits 8l..8l+7 of each
// chunk) and issues all 8 loads before any arithmetic; the grid is persistent (grid-stride
// over groups) so there is no partial last wave. Per logit: one conversion, one max, one
// fma, one ex2 and one add. Rounding to nearest is monotone, so the chunk maximum is taken on
// the raw logits and scaled once: max_v fp32(z_v * invT) = fp32(max_v z_v * invT).
// Non-finite logits are detected per chunk (an infinite maximum or a NaN sum).
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kWarps = 8;
constexpr int kPerWarp = 8;  // chunks per warp group

template <typename T>
__global__ void __launch_bounds__(kWarps * 32) k_row_stats(const T *__restrict__ data, int R, int V,
                                                           int64_t bstride, int64_t rstride, int C,
                                                           int64_t groups_total, float invT,
                                                           float2 *__restrict__ stats, uint32_t *status) {
    const int lane = threadIdx.x & 31;
    const int groups = (C + kPerWarp - 1) / kPerWarp;
    const float c2 = __fmul_rn(invT, kLog2e);  // exp(x - m) = 2^(z invT log2e - m log2e)
    bool bad = false;
    for (int64_t gw = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5); gw < groups_total;
         gw += (int64_t)gridDim.x * kWarps) {
        const int64_t row = gw / groups;
        const int g = (int)(gw - row * groups);
        const int b = (int)(row / R);
        const int r = (int)(row - (int64_t)b * R);
        const T *rp = data + (int64_t)b * bstride + (int64_t)r * rstride;
        const int c0 = g * kPerWarp;
        const int nc = min(kPerWarp, C - c0);
        RawGroup<T> raw[kPerWarp];
#pragma unroll
        for (int k = 0; k < kPerWarp; ++k)
            if (k < nc) raw[k].load(rp, (c0 + k) * kChunk + lane * 8, V);
#pragma unroll
        for (int k = 0; k < kPerWarp; ++k) {
            if (k >= nc) break;  // warp-uniform
            float z[8];
            raw[k].unpack(z);
            float zm = z[0];
#pragma unroll
            for (int i = 1; i < 8; ++i) zm = fmaxf(zm, z[i]);
            zm = warp_max(zm);
            const float mc = __fmul_rn(zm, invT);
            const float off = __fmul_rn(mc, kLog2e);
            float s = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) s += fast_exp2(__fmaf_rn(z[i], c2, -off));
            s = warp_sum(s);
            if (lane == 0) {
                stats[row * C + c0 + k] = make_float2(mc, s);
                bad |= !(s == s) || isinf(mc);
            }
        }
    }
    if (bad) raise_status(status, kDevNonFinite);
}

template <typename T>
int blocks_per_sm() {
    static int cached = 0;
    if (cached == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_row_stats<T>, kWarps * 32, 0) != cudaSuccess || n < 1)
            n = 1;
        cached = n;
    }
    return cached;
}

int sm_count() {
    static int cached = 0;
    if (cached == 0) {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
                                                     cudaSuccess || n < 1)
            n = 1;
        cached = n;
    }
    return cached;
}

template <typename T>
cudaError_t launch_t(const RowsDesc &rows, float invT, float2 *stats, uint32_t *status, cudaStream_t s) {
    const int C = num_chunks(rows.V);
    const int64_t groups_total = (int64_t)rows.B * rows.R * ((C + kPerWarp - 1) / kPerWarp);
    const int64_t needed = (groups_total + kWarps - 1) / kWarps;
    const int64_t resident = (int64_t)sm_count() * blocks_per_sm<T>();
    const int64_t blocks = needed < resident ? needed : resident;
    k_row_stats<T><<<(unsigned)blocks, kWarps * 32, 0, s>>>(static_cast<const T *>(rows.data), rows.R, rows.V,
                                                             rows.batch_stride, rows.row_stride, C, groups_total,
                                                             invT, stats, status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_row_stats(const RowsDesc &rows, float invT, float2 *stats, uint32_t *status, cudaStream_t s) {
    if (rows.dtype == 1) return launch_t<__nv_bfloat16>(rows, invT, stats, status, s);
    return launch_t<float>(rows, invT, stats, status, s);
}

}  // namespace tsb
