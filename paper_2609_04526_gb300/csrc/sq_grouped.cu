// Grouped launches of the contraction kernels: the experts of a mixture-of-experts
// layer, each with its own token rows, in one persistent launch per contraction.
#include "sq_gemm_kernels.cuh"

namespace sqi {

cudaError_t launch_grouped(const GroupedArgs &a, const CUtensorMap &tmCodes, int sm_count, cudaStream_t stream) {
  // The kernels read every per-expert descriptor from the table; the dense
  // descriptor parameters they do not use are passed as the code descriptor.
  KParams p{a.codes, a.scales, 1.0f, 0, a.N, a.K, a.out, a.mask, a.err, 0, 0, a.total_tiles, a.table, a.E};
  if (a.mode == MODE_SGRAD) {
    p.tiles_m = static_cast<int>((a.N + kSgradTile - 1) / kSgradTile);
    p.tiles_n = static_cast<int>((a.K + kSgradTile - 1) / kSgradTile);
  } else {
    p.tiles_n = static_cast<int>(((a.mode == MODE_FWD ? a.N : a.K) + kPairNTile - 1) / kPairNTile);
  }
  if (a.fmt == 0) {
    if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, 0, true>(p, tmCodes, tmCodes, tmCodes, sm_count, stream);
    if (a.mode == MODE_DX) return launch_pair<MODE_DX, 0, true>(p, tmCodes, tmCodes, tmCodes, sm_count, stream);
    return launch_sgrad<0, true>(p, tmCodes, tmCodes, sm_count, stream);
  }
  if (a.mode == MODE_FWD) return launch_pair<MODE_FWD, 1, true>(p, tmCodes, tmCodes, tmCodes, sm_count, stream);
  if (a.mode == MODE_DX) return launch_pair<MODE_DX, 1, true>(p, tmCodes, tmCodes, tmCodes, sm_count, stream);
  return launch_sgrad<1, true>(p, tmCodes, tmCodes, sm_count, stream);
}

}  // namespace sqi
