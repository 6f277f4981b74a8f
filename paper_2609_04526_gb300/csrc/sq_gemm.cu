// Dense launches of the contraction kernels: one weight, all M tokens.
#include "sq_gemm_kernels.cuh"

namespace sqi {

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
  if (a.fmt == 0) {
    if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, 0, false>(p, tmA, tmB, *tmOut, sm_count, stream);
    if (a.mode == MODE_DX) return launch_pair<MODE_DX, 0, false>(p, tmA, tmB, *tmOut, sm_count, stream);
    return launch_sgrad<0, false>(p, tmA, tmB, sm_count, stream);
  }
  if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, 1, false>(p, tmA, tmB, *tmOut, sm_count, stream);
  if (a.mode == MODE_DX) return launch_pair<MODE_DX, 1, false>(p, tmA, tmB, *tmOut, sm_count, stream);
  return launch_sgrad<1, false>(p, tmA, tmB, sm_count, stream);
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
