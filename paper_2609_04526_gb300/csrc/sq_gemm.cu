// Dense launches of the contraction kernels: one weight, all M tokens.
#include "sq_gemm_kernels.cuh"

namespace sqi {

// Adds the token splits' partial planes of a dense scale gradient in split order
// and applies the STE mask: g[i] = (sum_s partial[s][i]) * mask[i]. count = N * G
// is a multiple of 4 (N % 8 == 0) and every pointer is 16-byte aligned.
__global__ void sq_split_reduce_kernel(const float *__restrict__ partial, int splits, int64_t count,
                                       const uint8_t *__restrict__ mask, float *__restrict__ g) {
  const int64_t n4 = count / 4;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float4 acc = __ldg(reinterpret_cast<const float4 *>(partial) + i);
    for (int sp = 1; sp < splits; ++sp) {
      const float4 v = __ldg(reinterpret_cast<const float4 *>(partial + sp * count) + i);
      acc.x += v.x;
      acc.y += v.y;
      acc.z += v.z;
      acc.w += v.w;
    }
    if (mask) {
      const uchar4 m = __ldg(reinterpret_cast<const uchar4 *>(mask) + i);
      acc.x *= static_cast<float>(m.x);
      acc.y *= static_cast<float>(m.y);
      acc.z *= static_cast<float>(m.z);
      acc.w *= static_cast<float>(m.w);
    }
    reinterpret_cast<float4 *>(g)[i] = acc;
  }
}

cudaError_t launch_gemm(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB, const CUtensorMap *tmOut,
                        int sm_count, cudaStream_t stream) {
  if (a.mode != MODE_SGRAD && !tmOut) return cudaErrorInvalidValue;
  KParams p{a.codes, a.scales, a.ws2, a.M, a.N, a.K, a.out, a.mask, a.err, 0, 0, 0, nullptr, 1};
  if (a.mode == MODE_SGRAD) {
    p.tiles_m = static_cast<int>((a.N + kSgradTile - 1) / kSgradTile);
    p.tiles_n = static_cast<int>((a.K + kSgradTile - 1) / kSgradTile);
  } else {
    const int64_t Ng = a.mode == MODE_FWD ? a.N : a.K;
    p.tiles_m = static_cast<int>((a.M + kPairMTile - 1) / kPairMTile);
    p.tiles_n = static_cast<int>((Ng + kPairNTile - 1) / kPairNTile);
  }
  p.total = p.tiles_m * p.tiles_n;
  if (a.mode != MODE_SGRAD) {
    if (a.fmt == 0 && a.mode == MODE_FWD) return launch_pair<MODE_FWD, 0, false>(p, tmA, tmB, *tmOut, sm_count, stream);
    if (a.fmt == 0) return launch_pair<MODE_DX, 0, false>(p, tmA, tmB, *tmOut, sm_count, stream);
    if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, 1, false>(p, tmA, tmB, *tmOut, sm_count, stream);
    return launch_pair<MODE_DX, 1, false>(p, tmA, tmB, *tmOut, sm_count, stream);
  }
  if (a.splits > 1) {
    if (!a.partial || a.splits > kMaxSgradSplits) return cudaErrorInvalidValue;
    p.splits = a.splits;
    p.partial = a.partial;
    p.total *= a.splits;
  }
  cudaError_t e = a.fmt == 0 ? launch_sgrad<0, false>(p, tmA, tmB, sm_count, stream)
                             : launch_sgrad<1, false>(p, tmA, tmB, sm_count, stream);
  if (e != cudaSuccess || a.splits <= 1) return e;
  const int64_t count = a.N * (a.K / (a.fmt == 0 ? 16 : 32));
  const int64_t blocks = (count / 4 + 255) / 256;
  const int grid = static_cast<int>(blocks < 4 * sm_count ? blocks : 4 * sm_count);
  sq_split_reduce_kernel<<<grid, 256, 0, stream>>>(a.partial, a.splits, count, a.mask, static_cast<float *>(a.out));
  return cudaGetLastError();
}

// The failure-path self-test: the same bounded spin the contraction kernels use,
// on a barrier whose phase never completes.
__global__ void sq_wait_probe_kernel(int *err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  abort_flag = 0;
  fence_barrier_init();
  (void)mbar_spin(&bar, 0u, &abort_flag, err);  // runs out after kWaitLimitNs and records it
}

cudaError_t launch_wait_probe(int *err, cudaStream_t stream) {
  sq_wait_probe_kernel<<<1, 32, 0, stream>>>(err);
  return cudaGetLastError();
}

}  // namespace sqi
