// Launches of the contraction kernels for the full-precision multiplicative control
// of the ablation appendix: unquantized bf16 weights W with one coefficient per
// (row, block of 16), W' = W (1 + dS). The pair kernels load the bf16 weight tile
// into the decoded-weight slot and scale it in place; the scale-gradient kernel
// multiplies dW by W instead of a decoded code.
#include "sq_gemm_kernels.cuh"

namespace sqi {

cudaError_t launch_control(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB,
                           const CUtensorMap *tmOut, int sm_count, cudaStream_t stream) {
  if (a.mode != MODE_SGRAD && !tmOut) return cudaErrorInvalidValue;
  KParams p{a.codes, a.scales, 1.0f, a.M, a.N, a.K, a.out, a.mask, a.err, 0, 0, 0, nullptr, 1};
  if (a.mode == MODE_SGRAD) {
    p.tiles_m = static_cast<int>((a.N + kSgradTile - 1) / kSgradTile);
    p.tiles_n = static_cast<int>((a.K + kSgradTile - 1) / kSgradTile);
  } else {
    const int64_t Ng = a.mode == MODE_FWD ? a.N : a.K;
    p.tiles_m = static_cast<int>((a.M + kPairMTile - 1) / kPairMTile);
    p.tiles_n = static_cast<int>((Ng + kPairNTile - 1) / kPairNTile);
  }
  p.total = p.tiles_m * p.tiles_n;
  if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, kFmtBf16Mul, false>(p, tmA, tmB, *tmOut, sm_count, stream);
  if (a.mode == MODE_DX) return launch_pair<MODE_DX, kFmtBf16Mul, false>(p, tmA, tmB, *tmOut, sm_count, stream);
  return launch_sgrad<kFmtBf16Mul, false>(p, tmA, tmB, sm_count, stream);
}

}  // namespace sqi
