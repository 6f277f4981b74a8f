// Internal declarations shared by the host layer (sq_api.cu) and the kernel
// translation units of libscaleqlora. Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace sqi {

enum GemmMode : int {
  MODE_FWD = 0,    // Y  = X  . W^T   (GEMM M=tokens, N=out, contraction=in)
  MODE_DX = 1,     // dX = dY . W     (GEMM M=tokens, N=in,  contraction=out)
  MODE_SGRAD = 2   // g  = blockreduce(code * dY^T X)  (GEMM M=out, N=in, contraction=tokens)
};

// Rows of one activation TMA box of the pair kernels (the rows a CTA holds of a tile half).
constexpr int kBM = 128;
// Tokens per shared-memory stage of the scale-gradient kernel (also the height of its TMA boxes).
constexpr int kSgradBK = 128;

struct GemmArgs {
  int mode;
  int fmt;               // 0 NVFP4, 1 MXFP4
  int64_t M, N, K;       // tokens, out features, in features
  const uint8_t *codes;  // [N, K/2]
  const uint8_t *scales; // [N, K/B]
  float ws2;
  void *out;             // Y [M,N] bf16 | dX [M,K] bf16 | g [N,K/B] f32
  const uint8_t *mask;   // [N, K/B] or null (MODE_SGRAD only)
  int *err;              // device error word
  int splits = 1;            // MODE_SGRAD: token splits (sgrad_splits)
  float *partial = nullptr;  // MODE_SGRAD with splits > 1: [splits, N, K/B] fp32 partial sums
};

// Expert table of a grouped launch, built by the host for each call and copied
// to the device ahead of the kernel (64-byte aligned):
//   GroupMaps[E]         two TMA descriptors per expert, each addressing only that
//                        expert's token rows: FWD / DX the streamed activations and
//                        the output; SGRAD dY and X
//   int32 tile_start[E+1] first tile of each expert in the launch's tile list
//   int32 rows[E]        the expert's token count M_e
//   float ws2[E]         the expert's tensor scale (1.0 for MXFP4)
//   int32 id[E]          the expert of each entry: the scale gradient lists the experts
//                        longest first (its units last M_e tokens; dealt round-robin to
//                        the clusters, equal-length units then share a round), the
//                        forward and input gradient in order (their tiles are all K long)
struct GroupMaps {
  CUtensorMap m[2];
};
static_assert(sizeof(GroupMaps) == 256, "two 128-byte tensor maps per expert");
__host__ __device__ constexpr size_t group_off_tiles(int E) { return static_cast<size_t>(E) * sizeof(GroupMaps); }
__host__ __device__ constexpr size_t group_off_rows(int E) { return group_off_tiles(E) + static_cast<size_t>(E + 1) * 4; }
__host__ __device__ constexpr size_t group_off_ws2(int E) { return group_off_rows(E) + static_cast<size_t>(E) * 4; }
__host__ __device__ constexpr size_t group_off_ids(int E) { return group_off_ws2(E) + static_cast<size_t>(E) * 4; }
__host__ __device__ constexpr size_t group_table_bytes(int E) { return group_off_ids(E) + static_cast<size_t>(E) * 4; }

// Output rows of one FWD / DX tile and tokens of one scale-gradient stage: the
// host sizes the grouped tile list with these.
constexpr int kPairMTile = 512;
constexpr int kPairNTile = 256;
constexpr int kSgradTile = 256;

// Token splits of a dense scale-gradient launch. Each 256 x 256 tile contracts over
// all M tokens, so a launch with few tiles (q/k/v/o of the layer: 256 or 64) leaves
// much of its last wave idle, and a launch with many tiles streams every dY and X
// panel past the L2 once per wave of tiles that reads it. The tokens are then cut
// into up to kMaxSgradSplits parts of at least kMinSplitTokens each, one unit per
// (part, tile), walked part by part; every part writes a partial gradient plane and
// a second kernel adds the parts in order. A shorter part keeps the panels its
// waves share resident in L2 (measured on the 8B layer's shapes at M = 32768: 8
// parts read 1.3-2.0x the algorithmic bytes from DRAM against 2.2-3.5x for 5 parts
// or none), and each extra part adds ~0.2 % to the launch (the part sum's reads).
// Rule: with w(s) = ceil(tiles * s / clusters) / s, the launch's length in
// full-M tiles per cluster, take the largest s whose w(s) is within 1 % of the
// smallest w and no longer than the unsplit launch.
constexpr int kMaxSgradSplits = 8;
constexpr int64_t kMinSplitTokens = 2048;
inline int sgrad_splits(int64_t tiles, int clusters, int64_t M) {
  if (tiles <= 0 || clusters <= 0) return 1;
  auto waves = [&](int s) { return static_cast<double>((tiles * s + clusters - 1) / clusters) / s; };
  int top = 1;
  while (top < kMaxSgradSplits && M >= (top + 1) * kMinSplitTokens) ++top;
  double best = waves(1);
  for (int s = 2; s <= top; ++s) best = waves(s) < best ? waves(s) : best;
  const double limit = best * 1.01 < waves(1) ? best * 1.01 : waves(1);
  for (int s = top; s > 1; --s)
    if (waves(s) <= limit + 1e-9) return s;
  return 1;
}

struct GroupedArgs {
  int mode;
  int fmt;
  int E;                 // experts
  int64_t N, K;          // per expert: out features, in features
  const uint8_t *codes;  // [E, N, K/2]
  const uint8_t *scales; // [E, N, K/B]
  void *out;             // MODE_SGRAD: g [E, N, K/B] f32 (FWD / DX write through the table's maps)
  const uint8_t *mask;   // [E, N, K/B] or null (MODE_SGRAD only)
  int *err;
  const uint8_t *table;  // device copy of the expert table
  int total_tiles;       // tile_start[E]
};

// Launch one grouped contraction. tmCodes is the descriptor of all experts'
// packed codes as one [E * N, K/2] tensor (MODE_FWD / MODE_DX; unused for MODE_SGRAD).
cudaError_t launch_grouped(const GroupedArgs &a, const CUtensorMap &tmCodes, int sm_count, cudaStream_t stream);

// The contractions of the full-precision multiplicative control (a.fmt ignored):
// a.codes is the bf16 weight W [N, K], a.scales the fp32 coefficients dS [N, K/16];
// tmB the descriptor of W in 64 x 128 boxes with the 128-byte swizzle (FWD / DX),
// or of X (SGRAD, as launch_gemm).
cudaError_t launch_control(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB,
                           const CUtensorMap *tmOut, int sm_count, cudaStream_t stream);
// out = alpha_over_r * B A (B [N, r], A [r, G] bf16), through `workspace`
// (lowrank_product_workspace bytes): the control's low-rank coefficient plane.
size_t lowrank_product_workspace(int64_t N, int64_t G, int r, int sm_count);
cudaError_t launch_lowrank_product(int64_t N, int64_t G, int r, float alpha_over_r, const uint16_t *B,
                                   const uint16_t *A, float *out, float *workspace, int sm_count, cudaStream_t stream);

// Launch one contraction. tmA is the TMA descriptor of the streamed bf16
// activations; tmB that of the packed codes (MODE_FWD / MODE_DX) or of the second
// bf16 operand (MODE_SGRAD); tmOut that of the bf16 output (MODE_FWD / MODE_DX:
// 32-row x 32-column boxes, 64-byte swizzle; null for MODE_SGRAD).
cudaError_t launch_gemm(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB, const CUtensorMap *tmOut,
                        int sm_count, cudaStream_t stream);
// One thread waiting on a barrier nothing arrives on, bounded like every kernel wait:
// records kErrWaitTimeout in *err and returns (the failure-path self-test).
cudaError_t launch_wait_probe(int *err, cudaStream_t stream);

// Projection / merge of `count` latents. With ws2_per (device, one float per
// expert; NVFP4 only) the latents are the planes of several experts, `plane` (a
// multiple of 16) elements each, and element i uses ws2_per[i / plane] instead of ws2.
cudaError_t launch_project(int fmt, int64_t count, float ws2, const float *latent, uint8_t *bytes_out,
                           uint8_t *mask_out, int32_t *nonfinite, int sm_count, cudaStream_t stream,
                           const float *ws2_per = nullptr, int64_t plane = 0);

cudaError_t launch_merge(int fmt, int64_t count, float ws2, const float *latent, uint8_t *scales_inout,
                         float *ongrid_delta, int64_t *changed, int sm_count, cudaStream_t stream,
                         const float *ws2_per = nullptr, int64_t plane = 0);

// Projection / merge of several scale planes of different shapes in one launch
// (the planes of all linears of a layer). The table travels by value in the
// kernel's parameters; each plane's N * G is a multiple of 16. Counters are summed
// per CTA into `acc` (kMaxPlanes int64 plus a uint32 ticket, zero between calls:
// the last CTA writes each plane's count to its counter and clears them).
constexpr int kMaxPlanes = 16;
struct PlaneArgs {
  int64_t count;     // scale blocks (N * G)
  float ws2;         // NVFP4 tensor scale (1 for MXFP4)
  const float *latent;
  uint8_t *bytes;    // projection: bytes out; merge: the scale plane, in place
  uint8_t *mask;     // projection: mask out or null
  float *delta;      // merge: on-grid delta or null
  void *counter;     // projection: int32 NaN count; merge: int64 changed bytes; or null
};
struct PlaneTable {
  int n;
  PlaneArgs p[kMaxPlanes];
};
constexpr size_t kPlaneAccBytes = kMaxPlanes * sizeof(int64_t) + 16;
cudaError_t launch_project_planes(int fmt, const PlaneTable &t, int64_t *acc, cudaStream_t stream);
cudaError_t launch_merge_planes(int fmt, const PlaneTable &t, int64_t *acc, cudaStream_t stream);

// Rollback of a merge by its on-grid delta (in place, counting changed bytes), and
// copy a -> b (write) or only count the bytes in which a and b differ.
cudaError_t launch_rollback(int fmt, int64_t count, float ws2, const float *delta, uint8_t *scales_inout,
                            int64_t *changed, int sm_count, cudaStream_t stream);
cudaError_t launch_swap_or_diff(int64_t count, const uint8_t *a, uint8_t *b, bool write, int64_t *differing,
                                int sm_count, cudaStream_t stream);

// Low-rank scale adapter (Sec. 3 "Scale-QLoRA forward"): latent eff + (alpha/r) B A
// projected onto the grid; and the gradients of B and A from the masked scale
// gradient, through `workspace` (lowrank_grad_workspace bytes). With experts > 1
// the planes and factors of that many experts follow each other in memory (one
// launch for all); ws2_per (device, NVFP4) gives each expert's tensor scale.
cudaError_t launch_project_lowrank(int fmt, int64_t N, int64_t G, int r, float ws2, float alpha_over_r,
                                   const uint8_t *base, const uint16_t *B, const uint16_t *A, uint8_t *bytes_out,
                                   uint8_t *mask_out, int32_t *nonfinite, float *latent_out, cudaStream_t stream,
                                   int experts = 1, const float *ws2_per = nullptr);
// Ranks up to 128 run on the tensor cores (sq_adapter_tc.cu), larger ones on CUDA
// cores; `err` is the device error word (bounded waits of the tensor-core path).
size_t lowrank_grad_workspace(int64_t N, int64_t G, int r, int sm_count, int experts = 1);
cudaError_t launch_lowrank_grad(int64_t N, int64_t G, int r, float alpha_over_r, const float *g, const uint16_t *B,
                                const uint16_t *A, float *dB, float *dA, float *workspace, int sm_count,
                                cudaStream_t stream, int *err, int experts = 1);
bool lowrank_grad_tc_supported(int r);
size_t lowrank_grad_tc_workspace(int64_t N, int64_t G, int r, int experts, int sm_count);
cudaError_t launch_lowrank_grad_tc(int64_t N, int64_t G, int r, float alpha_over_r, const float *g,
                                   const uint16_t *B, const uint16_t *A, float *dB, float *dA, float *workspace,
                                   int *err, int sm_count, cudaStream_t stream, int experts);
constexpr int kMaxLowRank = 256;  // r limit of the adapter kernels

// Scale-family variants (ablation appendix): the least-squares code-preserving fit
// of a weight update per block; the group gradient and the group-delta projection
// of the granularity ladder (gd groups of G / gd blocks per row).
cudaError_t launch_fit(int fmt, int64_t N, int64_t K, float ws2, const uint8_t *codes, const uint8_t *scales,
                       const uint16_t *dW, float *delta, float *captured, float *total, float *latent, int sm_count,
                       cudaStream_t stream);
cudaError_t launch_group_reduce(int64_t N, int64_t G, int64_t gd, const float *g, float *out, int sm_count,
                                cudaStream_t stream);
cudaError_t launch_project_group_delta(int fmt, int64_t N, int64_t G, int64_t gd, float ws2, const uint8_t *base,
                                       const float *delta, uint8_t *bytes_out, uint8_t *mask_out, int32_t *nonfinite,
                                       float *latent_out, int sm_count, cudaStream_t stream);

// Device-side error codes written to the error word.
constexpr int kErrWaitTimeout = 1;

}  // namespace sqi
