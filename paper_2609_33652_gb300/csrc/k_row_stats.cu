// Streaming pass over logit rows: per chunk of 256 logits, the maximum m_c and the sum
// s_c = sum exp(x - m_c) of x = fp32(z) * fp32(1/T). The row's log-normaliser, its top-K
// candidate pool (first pass, Sec. 3.1) and the chunk log-masses A_c = m_c + log s_c of
// the replay sampler (Sec. 3.2) all follow from these without touching the row again.
//
// HBM-bound: every logit is read once with 16-byte loads; 8 bytes are written per chunk.
// Eight lanes own one chunk (lane g of the group reads logits 8g..8g+7 of each 64-logit
// quarter, so a group's load instruction covers 128 contiguous bytes), a warp owns four
// chunks at a time and issues two such units' loads before any arithmetic. The grid is
// persistent (grid-stride over units), so there is no partial last wave. Per logit: one
// conversion, one max, one fma, one ex2 and one add; per chunk only three shuffle levels.
// Rounding to nearest is monotone, so the chunk maximum is taken on the raw logits and
// scaled once: max_v fp32(z_v * invT) = fp32(max_v z_v * invT). Non-finite logits are
// detected per chunk (an infinite maximum or a NaN sum).
#include "tsb_device.cuh"
#include "tsb_launch.h"

namespace tsb {
namespace {

constexpr int kWarps = 8;
constexpr int kUnitChunks = 4;  // chunks per warp unit (8 lanes each)
constexpr int kUnits = 2;       // units per warp iteration (loads in flight together)

template <typename T>
__global__ void __launch_bounds__(kWarps * 32) k_row_stats(const T *__restrict__ data, int R, int V,
                                                           int64_t bstride, int64_t rstride, int C,
                                                           int64_t units_total, float invT,
                                                           float2 *__restrict__ stats, uint32_t *status) {
    pdl_begin();
    const int lane = threadIdx.x & 31, g = lane & 7, q = lane >> 3;
    const int upr = (C + kUnitChunks - 1) / kUnitChunks;  // units per row
    bool bad = false;
    const int64_t stride = (int64_t)gridDim.x * kWarps;
    for (int64_t u0 = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5); u0 < units_total; u0 += stride * kUnits) {
        RawGroup<T> raw[kUnits][4];
        int64_t row_of[kUnits];
        int c_of[kUnits];
#pragma unroll
        for (int e = 0; e < kUnits; ++e) {
            const int64_t un = u0 + e * stride;
            c_of[e] = -1;
            row_of[e] = 0;
            if (un >= units_total) continue;
            const int64_t row = un / upr;
            const int c = (int)(un - row * upr) * kUnitChunks + q;
            row_of[e] = row;
            if (c >= C) continue;
            c_of[e] = c;
            const int b = (int)(row / R);
            const int r = (int)(row - (int64_t)b * R);
            const T *rp = data + (int64_t)b * bstride + (int64_t)r * rstride;
#pragma unroll
            for (int k = 0; k < 4; ++k) raw[e][k].load(rp, c * kChunk + k * 64 + g * 8, V);
        }
#pragma unroll
        for (int e = 0; e < kUnits; ++e) {
            const int c = c_of[e];
            float mc, s;
            chunk_stats8<T>(raw[e], c >= 0, invT, &mc, &s);
            if (c >= 0 && g == 0) {
                stats[row_of[e] * C + c] = make_float2(mc, s);
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
    const int64_t units_total = (int64_t)rows.B * rows.R * ((C + kUnitChunks - 1) / kUnitChunks);
    const int64_t needed = (units_total + kWarps - 1) / kWarps;
    const int64_t resident = (int64_t)sm_count() * blocks_per_sm<T>();
    const int64_t blocks = needed < resident ? needed : resident;
    return launch_pdl(k_row_stats<T>, dim3((unsigned)blocks), dim3(kWarps * 32), 0, s, 0,
                      static_cast<const T *>(rows.data), rows.R, rows.V, rows.batch_stride, rows.row_stride, C,
                      units_total, invT, stats, status);
}

}  // namespace

cudaError_t launch_row_stats(const RowsDesc &rows, float invT, float2 *stats, uint32_t *status, cudaStream_t s) {
    if (rows.dtype == 1) return launch_t<__nv_bfloat16>(rows, invT, stats, status, s);
    return launch_t<float>(rows, invT, stats, status, s);
}

}  // namespace tsb
