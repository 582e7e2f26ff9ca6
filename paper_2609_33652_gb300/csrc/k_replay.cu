// Second pass (Sec. 3.2, Eq. replay-distribution; sampling without replacement, App. A).
//
// For every parent u with m_u children, the m_u ordered draws without replacement from
// q_u = softmax(x_row(u)) are the top-m_u Gumbel keys x_v + G_v (Gumbel-top-k). The keys are
// built top-down (Maddison et al. 2014; Kool et al. 2019, App. B):
//   1. chunk keys K_c = A_c + G(U[chunk c]) with A_c = m_c + log s_c from the chunk
//      statistics; keep the top-m_u chunks by (K_c desc, c asc);
//   2. inside each kept chunk, element keys g_v = x_v + G(U[token v]) are shifted to the law
//      conditional on their maximum Z_c being K_c:
//        k_v = K_c - softplus(K_c - g_v + log1p(-exp(g_v - Z_c))),  k_argmax = K_c;
//   3. the top-m_u keys by (k desc, v asc) over the kept chunks are the draws; draw j fills
//      child slot j.
// Every token outside the kept chunks is below m_u distinct chunk maxima, so it can never
// be among the top m_u: the joint law is exactly that of flat Gumbel-top-k over V tokens,
// at ceil(V/256) + m_u*256 draws per parent instead of V.
//
// One CTA of 4 warps per (tree, node); nodes without children return at once. Chunk keys are
// spread over the CTA (four chunks per thread share one Philox block) and kept in shared
// memory; the top-m_u are ranked among those that reach a lower bound (the m_u-th largest of
// the warps' few largest). Each warp then takes one kept chunk at a time; only elements whose
// key can reach the m_u-th chunk key get a shifted key, and those are ranked in shared memory
// (per-lane lists and merges when more of them than the buffer holds).
// A parent with one child takes the Gumbel-max token directly (running maxima, no shift).
#include "tsb_device.cuh"
#include "tsb_launch.h"
#include "replay_body.cuh"

namespace tsb {
namespace {

template <int KCAP, typename T>
__global__ void __launch_bounds__(kRpThreads, KCAP <= 8 ? kRpMinBlocks : 2) k_replay(ReplayArgs a) {
    pdl_begin();
    replay_node<KCAP, T>(a, (int)blockIdx.x);
}

template <int KCAP, typename T>
cudaError_t launch_replay_t(const ReplayArgs &a, cudaStream_t s) {
    const int64_t blocks = (int64_t)a.B * (a.N + 1);
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const size_t smem = (size_t)key_buf_len(a.C) * sizeof(uint64_t);
    cudaError_t e = cudaFuncSetAttribute(k_replay<KCAP, T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_replay<KCAP, T>, dim3((unsigned)blocks), dim3(kRpThreads), smem, s, 0, a);
}

}  // namespace

cudaError_t launch_replay(const RowsDesc &q, const float2 *qstats, const int32_t *qrow_of_node, int B, int N,
                          int K, const TreeDesc &tree, float invT, uint64_t seed, int32_t *token, uint32_t *status,
                          cudaStream_t s) {
    const ReplayArgs a = replay_args(q, qstats, qrow_of_node, B, N, tree, invT, seed, token, status);
    // sibling groups have at most K members: a list of 8 covers K <= 8
    if (q.dtype == 1)
        return K <= 8 ? launch_replay_t<8, __nv_bfloat16>(a, s) : launch_replay_t<32, __nv_bfloat16>(a, s);
    return K <= 8 ? launch_replay_t<8, float>(a, s) : launch_replay_t<32, float>(a, s);
}

}  // namespace tsb
