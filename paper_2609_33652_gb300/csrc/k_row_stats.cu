// Streaming pass over logit rows: per chunk of 256 logits, the maximum m_c and the sum
// s_c = sum exp(x - m_c) of x = fp32(z) * fp32(1/T). The row's log-normaliser, its top-K
// candidate pool (first pass, Sec. 3.1) and the chunk log-masses A_c = m_c + log s_c of
// the replay sampler (Sec. 3.2) all follow from these without touching the row again.
//
// HBM-bound: every logit is read once with 16-byte loads; 8 bytes are written per chunk.
// One warp owns 4 consecutive chunks of a row (lane l holds logits 8l..8l+7 of each chunk),
// issuing all of its loads before any arithmetic.
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kWarps = 8;
constexpr int kPerWarp = 4;  // chunks per warp

template <typename T>
__global__ void __launch_bounds__(kWarps * 32) k_row_stats(const T *__restrict__ data, int R, int V,
                                                           int64_t bstride, int64_t rstride, int C,
                                                           int64_t groups_total, float invT,
                                                           float2 *__restrict__ stats, uint32_t *status) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (gw >= groups_total) return;
    const int groups = (C + kPerWarp - 1) / kPerWarp;
    const int64_t row = gw / groups;
    const int g = (int)(gw - row * groups);
    const int b = (int)(row / R);
    const int r = (int)(row - (int64_t)b * R);
    const T *rp = data + (int64_t)b * bstride + (int64_t)r * rstride;
    const int c0 = g * kPerWarp;
    const int nc = min(kPerWarp, C - c0);

    float x[kPerWarp][8];
#pragma unroll
    for (int k = 0; k < kPerWarp; ++k)
        if (k < nc) Logit<T>::load8(rp, (c0 + k) * kChunk + lane * 8, V, x[k]);

    bool bad = false;
#pragma unroll
    for (int k = 0; k < kPerWarp; ++k) {
        if (k >= nc) break;  // warp-uniform
        const int v0 = (c0 + k) * kChunk + lane * 8;
        float m = -INFINITY;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float xi = -INFINITY;
            if (v0 + i < V) {
                xi = __fmul_rn(x[k][i], invT);
                bad |= !isfinite(xi);
            }
            x[k][i] = xi;
            m = fmaxf(m, xi);
        }
        m = warp_max(m);
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) s += fast_exp2(__fmul_rn(__fsub_rn(x[k][i], m), kLog2e));
        s = warp_sum(s);
        if (lane == 0) stats[row * C + c0 + k] = make_float2(m, s);
    }
    if (__any_sync(kFull, bad) && lane == 0) raise_status(status, kDevNonFinite);
}

}  // namespace

cudaError_t launch_row_stats(const RowsDesc &rows, float invT, float2 *stats, uint32_t *status, cudaStream_t s) {
    const int C = num_chunks(rows.V);
    const int64_t groups_total = (int64_t)rows.B * rows.R * ((C + kPerWarp - 1) / kPerWarp);
    const int64_t blocks = (groups_total + kWarps - 1) / kWarps;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    if (rows.dtype == 1)
        k_row_stats<__nv_bfloat16><<<(unsigned)blocks, kWarps * 32, 0, s>>>(
            static_cast<const __nv_bfloat16 *>(rows.data), rows.R, rows.V, rows.batch_stride, rows.row_stride, C,
            groups_total, invT, stats, status);
    else
        k_row_stats<float><<<(unsigned)blocks, kWarps * 32, 0, s>>>(static_cast<const float *>(rows.data), rows.R,
                                                                     rows.V, rows.batch_stride, rows.row_stride, C,
                                                                     groups_total, invT, stats, status);
    return cudaGetLastError();
}

}  // namespace tsb
