// Grid projection and merge kernels (sm_103a): Sec. 3 QAST round_grid with the
// E4M3 ceiling clamp of the stability recipe, and the merge that rewrites scale
// bytes only (Sec. 3 "QAST makes merge exact by construction").
//
// Both are HBM-bandwidth kernels: each thread owns 16 consecutive latents per
// step (four 16-byte loads), writes 16 bytes of each output with one 16-byte
// store, and the grid is a whole number of waves over the SMs (grid-stride).
// Counters (NaN latents, changed bytes) are reduced within each warp and added
// with one atomic per warp.
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "sq_internal.h"

namespace sqi {
namespace {

constexpr int kThreads = 256;
constexpr int kCtasPerSm = 4;

// fp32 pair -> two E4M3 bytes, round to nearest even, out-of-range magnitudes
// saturate to 448 (the callers clamp first, so this only matters at 448 + ulp).
__device__ __forceinline__ uint32_t e4m3x2_rn(float lo, float hi) {
  unsigned short r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// NVFP4 projection of one latent (absolute units) to (byte, mask, is_nan).
__device__ __forceinline__ void project_nv(float L, float ws2, float cap, uint32_t &byte, uint32_t &mask,
                                           uint32_t &nan) {
  nan = (L != L) ? 1u : 0u;
  mask = (L >= -cap && L <= cap) ? 1u : 0u;
  const float Lc = fminf(fmaxf(L, -cap), cap);
  const float q = __fdiv_rn(Lc, ws2);
  byte = e4m3x2_rn(q, 0.f) & 0xFFu;
  if (nan) byte = 0x7Fu;
}

// MXFP4 projection: byte = round(log2 L) + 127, rounding up iff the significand
// exceeds sqrt(2) (fp32 mantissa field > 0x3504F3, since
// 1 + 0x3504F3 / 2^23 < sqrt(2) < 1 + 0x3504F4 / 2^23).
__device__ __forceinline__ void project_mx(float L, uint32_t &byte, uint32_t &mask, uint32_t &nan) {
  const uint32_t u = __float_as_uint(L);
  nan = (L != L) ? 1u : 0u;
  if (nan) {
    byte = 0xFFu;
    mask = 0u;
    return;
  }
  if (!(L > 0.f)) {
    byte = 0u;
    mask = 0u;
    return;
  }
  const uint32_t ex = (u >> 23) & 0xFFu;
  if (ex == 0xFFu) {  // +inf
    byte = 254u;
    mask = 0u;
    return;
  }
  uint32_t man = u & 0x7FFFFFu;
  int e;
  if (ex == 0) {  // subnormal: L = man * 2^-149, normalise the significand
    const int msb = 31 - __clz(static_cast<int>(man));
    e = msb - 149;
    man = (man << (23 - msb)) & 0x7FFFFFu;
  } else {
    e = static_cast<int>(ex) - 127;
  }
  e += (man > 0x3504F3u) ? 1 : 0;
  int b = e + 127;
  mask = 1u;
  if (b < 0) {
    b = 0;
    mask = 0u;
  }
  if (b > 254) {
    b = 254;
    mask = 0u;
  }
  byte = static_cast<uint32_t>(b);
}

template <int FMT>
__device__ __forceinline__ void project_one(float L, float ws2, float cap, uint32_t &byte, uint32_t &mask,
                                            uint32_t &nan) {
  if (FMT == 0)
    project_nv(L, ws2, cap, byte, mask, nan);
  else
    project_mx(L, byte, mask, nan);
}

// Decoded on-grid scale in fp32: fl32(E4M3(byte) * ws2) or 2^(byte - 127).
template <int FMT>
__device__ __forceinline__ float scale_value(uint32_t byte, float ws2) {
  if (FMT == 0) {
    const __half_raw hr = __nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(byte), __NV_E4M3);
    return __fmul_rn(__half2float(__half(hr)), ws2);
  }
  if (byte == 255u) return __uint_as_float(0x7FC00000u);
  if (byte == 0u) return __uint_as_float(0x00400000u);  // 2^-127, an fp32 subnormal
  return __uint_as_float(byte << 23);
}

__device__ __forceinline__ void warp_add_i32(int32_t *counter, uint32_t v) {
  v = __reduce_add_sync(0xFFFFFFFFu, v);
  if ((threadIdx.x & 31) == 0 && v) atomicAdd(counter, static_cast<int32_t>(v));
}

__device__ __forceinline__ void warp_add_i64(int64_t *counter, uint32_t v) {
  v = __reduce_add_sync(0xFFFFFFFFu, v);
  if ((threadIdx.x & 31) == 0 && v)
    atomicAdd(reinterpret_cast<unsigned long long *>(counter), static_cast<unsigned long long>(v));
}

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_project_kernel(int64_t count, float ws2, float cap,
                                                              const float *__restrict__ latent,
                                                              uint8_t *__restrict__ bytes_out,
                                                              uint8_t *__restrict__ mask_out,
                                                              int32_t *__restrict__ nonfinite) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t nan_count = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const float4 *src = reinterpret_cast<const float4 *>(latent) + 4 * v;
    float L[16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldcs(src + q);
      L[4 * q] = f.x;
      L[4 * q + 1] = f.y;
      L[4 * q + 2] = f.z;
      L[4 * q + 3] = f.w;
    }
    uint32_t ob[4] = {0, 0, 0, 0}, om[4] = {0, 0, 0, 0};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      uint32_t b, m, n;
      project_one<FMT>(L[i], ws2, cap, b, m, n);
      ob[i >> 2] |= b << (8 * (i & 3));
      om[i >> 2] |= m << (8 * (i & 3));
      nan_count += n;
    }
    __stcs(reinterpret_cast<uint4 *>(bytes_out) + v, make_uint4(ob[0], ob[1], ob[2], ob[3]));
    if (mask_out) __stcs(reinterpret_cast<uint4 *>(mask_out) + v, make_uint4(om[0], om[1], om[2], om[3]));
  }
  // ragged tail (< 16 values) by the first threads of block 0
  if (blockIdx.x == 0 && threadIdx.x < count - nvec * 16) {
    const int64_t i = nvec * 16 + threadIdx.x;
    uint32_t b, m, n;
    project_one<FMT>(latent[i], ws2, cap, b, m, n);
    bytes_out[i] = static_cast<uint8_t>(b);
    if (mask_out) mask_out[i] = static_cast<uint8_t>(m);
    nan_count += n;
  }
  if (nonfinite) warp_add_i32(nonfinite, nan_count);
}

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_merge_kernel(int64_t count, float ws2, float cap,
                                                            const float *__restrict__ latent,
                                                            uint8_t *__restrict__ scales,
                                                            float *__restrict__ delta,
                                                            int64_t *__restrict__ changed) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t n_changed = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const float4 *src = reinterpret_cast<const float4 *>(latent) + 4 * v;
    float L[16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldcs(src + q);
      L[4 * q] = f.x;
      L[4 * q + 1] = f.y;
      L[4 * q + 2] = f.z;
      L[4 * q + 3] = f.w;
    }
    const uint4 old4 = *(reinterpret_cast<const uint4 *>(scales) + v);
    const uint32_t old[4] = {old4.x, old4.y, old4.z, old4.w};
    uint32_t ob[4] = {0, 0, 0, 0};
    float d[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      uint32_t b, m, n;
      project_one<FMT>(L[i], ws2, cap, b, m, n);
      const uint32_t o = (old[i >> 2] >> (8 * (i & 3))) & 0xFFu;
      ob[i >> 2] |= b << (8 * (i & 3));
      n_changed += (b != o) ? 1u : 0u;
      d[i] = __fsub_rn(scale_value<FMT>(b, ws2), scale_value<FMT>(o, ws2));
    }
    *(reinterpret_cast<uint4 *>(scales) + v) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
    if (delta) {
      float4 *dst = reinterpret_cast<float4 *>(delta) + 4 * v;
#pragma unroll
      for (int q = 0; q < 4; ++q) __stcs(dst + q, make_float4(d[4 * q], d[4 * q + 1], d[4 * q + 2], d[4 * q + 3]));
    }
  }
  if (blockIdx.x == 0 && threadIdx.x < count - nvec * 16) {
    const int64_t i = nvec * 16 + threadIdx.x;
    uint32_t b, m, n;
    project_one<FMT>(latent[i], ws2, cap, b, m, n);
    const uint32_t o = scales[i];
    scales[i] = static_cast<uint8_t>(b);
    n_changed += (b != o) ? 1u : 0u;
    if (delta) delta[i] = __fsub_rn(scale_value<FMT>(b, ws2), scale_value<FMT>(o, ws2));
  }
  if (changed) warp_add_i64(changed, n_changed);
}

// ---------------------------------------------------------------- low-rank scale adapter
//
// Sec. 3 "Scale-QLoRA forward": the latent block scale eff' = eff + (alpha/r) (B A),
// B [N, r] and A [r, G] bf16, formed in fp32 in a fixed order -- eff = fl32(decoded
// base byte * ws2) (scale_value), acc = fused multiply-adds over j = 0 .. r-1 from 0,
// eff' = fma(alpha/r, acc, eff) -- and projected exactly as sq_project_kernel. A CTA
// owns a 32 x 64 block of the plane with its 32 B rows and 64 A columns staged in
// shared memory; each thread accumulates 4 rows x 2 columns (the B values are warp
// broadcasts, the A values consecutive).
constexpr int kLrRows = 32;
constexpr int kLrCols = 64;

__device__ __forceinline__ float bf16_bits(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_project_lowrank_kernel(
    int64_t N, int64_t G, int r, float ws2, float cap, float aor, const uint8_t *__restrict__ base,
    const uint16_t *__restrict__ B, const uint16_t *__restrict__ A, uint8_t *__restrict__ bytes_out,
    uint8_t *__restrict__ mask_out, int32_t *__restrict__ nonfinite, float *__restrict__ latent_out) {
  extern __shared__ uint16_t lr_smem[];
  uint16_t *sB = lr_smem;                // [kLrRows][r]
  uint16_t *sA = lr_smem + kLrRows * r;  // [r][kLrCols]
  const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kLrRows;
  const int64_t b0 = static_cast<int64_t>(blockIdx.y) * kLrCols;
  for (int i = threadIdx.x; i < kLrRows * r; i += kThreads) {
    const int64_t n = n0 + i / r;
    sB[i] = n < N ? B[n * r + i % r] : static_cast<uint16_t>(0);
  }
  for (int i = threadIdx.x; i < r * kLrCols; i += kThreads) {
    const int64_t b = b0 + i % kLrCols;
    sA[i] = b < G ? A[static_cast<int64_t>(i / kLrCols) * G + b] : static_cast<uint16_t>(0);
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float acc[4][2];
#pragma unroll
  for (int q = 0; q < 4; ++q) acc[q][0] = acc[q][1] = 0.f;
  for (int j = 0; j < r; ++j) {
    const float a0 = bf16_bits(sA[j * kLrCols + lane]);
    const float a1 = bf16_bits(sA[j * kLrCols + 32 + lane]);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float bq = bf16_bits(sB[(warp * 4 + q) * r + j]);
      acc[q][0] = fmaf(bq, a0, acc[q][0]);
      acc[q][1] = fmaf(bq, a1, acc[q][1]);
    }
  }
  uint32_t nan_count = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const int64_t n = n0 + warp * 4 + q, b = b0 + lane + 32 * c;
      if (n < N && b < G) {
        const int64_t i = n * G + b;
        const float L = fmaf(aor, acc[q][c], scale_value<FMT>(base[i], ws2));
        uint32_t by, mk, na;
        project_one<FMT>(L, ws2, cap, by, mk, na);
        bytes_out[i] = static_cast<uint8_t>(by);
        if (mask_out) mask_out[i] = static_cast<uint8_t>(mk);
        if (latent_out) latent_out[i] = L;
        nan_count += na;
      }
    }
  }
  if (nonfinite) warp_add_i32(nonfinite, nan_count);
}

// Adapter gradients from the masked scale gradient g [N, G]: dB[n,j] = (alpha/r) sum_b
// g[n,b] A[j,b] and dA[j,b] = (alpha/r) sum_n B[n,j] g[n,b], fp32 accumulation in a fixed
// order (the same result on every run).
//
// dB: one warp per row n, 32 j at a time; each lane sums over the columns b = lane
// (mod 32) of 256-column chunks of A staged in shared memory, then a butterfly sums
// the lanes.
constexpr int kDbChunk = 256;
constexpr int kWarps = kThreads / 32;

__global__ void __launch_bounds__(kThreads) sq_lowrank_db_kernel(int64_t N, int64_t G, int r, float aor,
                                                                 const float *__restrict__ g,
                                                                 const uint16_t *__restrict__ A,
                                                                 float *__restrict__ dB) {
  extern __shared__ uint16_t db_smem[];  // [r][kDbChunk] chunk of A
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
  for (int jc = 0; jc < r; jc += 32) {
    const int nj = min(32, r - jc);
    float acc[32];
#pragma unroll
    for (int t = 0; t < 32; ++t) acc[t] = 0.f;
    for (int64_t bc = 0; bc < G; bc += kDbChunk) {
      const int w = G - bc < kDbChunk ? static_cast<int>(G - bc) : kDbChunk;
      __syncthreads();
      for (int i = threadIdx.x; i < nj * kDbChunk; i += kThreads) {
        const int t = i / kDbChunk, c = i % kDbChunk;
        db_smem[i] = c < w ? A[static_cast<int64_t>(jc + t) * G + bc + c] : static_cast<uint16_t>(0);
      }
      __syncthreads();
      if (n < N) {
        for (int c = lane; c < w; c += 32) {
          const float gv = g[n * G + bc + c];
#pragma unroll
          for (int t = 0; t < 32; ++t)
            if (t < nj) acc[t] = fmaf(gv, bf16_bits(db_smem[t * kDbChunk + c]), acc[t]);
        }
      }
    }
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      float v = acc[t];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
      if (n < N && lane == t && t < nj) dB[n * r + jc + t] = aor * v;
    }
  }
}

// dA, pass 1: a CTA takes kDaRows rows n and 32 columns b; lane = column, warp w takes
// j = w, w + 8, ...; the rows are summed in order into partial[chunk][j][b].
constexpr int kDaRows = 128;
constexpr int kDaJ = 32;  // accumulators per thread: r <= 8 * kDaJ = 256

__global__ void __launch_bounds__(kThreads) sq_lowrank_da_partial_kernel(int64_t N, int64_t G, int r,
                                                                         const float *__restrict__ g,
                                                                         const uint16_t *__restrict__ B,
                                                                         float *__restrict__ partial) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t chunk = blockIdx.x;
  const int64_t b = static_cast<int64_t>(blockIdx.y) * 32 + lane;
  const int64_t n0 = chunk * kDaRows, n1 = N < n0 + kDaRows ? N : n0 + kDaRows;
  float acc[kDaJ];
#pragma unroll
  for (int t = 0; t < kDaJ; ++t) acc[t] = 0.f;
  for (int64_t n = n0; n < n1; ++n) {
    const float gv = b < G ? g[n * G + b] : 0.f;
#pragma unroll
    for (int t = 0; t < kDaJ; ++t) {
      const int j = warp + kWarps * t;
      if (j < r) acc[t] = fmaf(bf16_bits(B[n * r + j]), gv, acc[t]);
    }
  }
  if (b < G) {
#pragma unroll
    for (int t = 0; t < kDaJ; ++t) {
      const int j = warp + kWarps * t;
      if (j < r) partial[(chunk * r + j) * G + b] = acc[t];
    }
  }
}

// dA, pass 2: dA[j,b] = (alpha/r) * sum over chunks, in chunk order.
__global__ void __launch_bounds__(kThreads) sq_lowrank_da_reduce_kernel(int64_t G, int r, int64_t chunks, float aor,
                                                                        const float *__restrict__ partial,
                                                                        float *__restrict__ dA) {
  const int64_t count = static_cast<int64_t>(r) * G;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < count;
       i += static_cast<int64_t>(gridDim.x) * kThreads) {
    float s = 0.f;
    for (int64_t c = 0; c < chunks; ++c) s += partial[c * count + i];
    dA[i] = aor * s;
  }
}

unsigned grid_for(int64_t count, int sm_count) {
  const int64_t nvec = count / 16;
  const int64_t want = (nvec + kThreads - 1) / kThreads;
  const int64_t cap = static_cast<int64_t>(sm_count) * kCtasPerSm;
  int64_t g = want < cap ? want : cap;
  if (g < 1) g = 1;
  return static_cast<unsigned>(g);
}

}  // namespace

cudaError_t launch_project(int fmt, int64_t count, float ws2, const float *latent, uint8_t *bytes_out,
                           uint8_t *mask_out, int32_t *nonfinite, int sm_count, cudaStream_t stream) {
  if (nonfinite) {
    cudaError_t e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (fmt == 0)
    sq_project_kernel<0><<<grid, kThreads, 0, stream>>>(count, ws2, cap, latent, bytes_out, mask_out, nonfinite);
  else
    sq_project_kernel<1><<<grid, kThreads, 0, stream>>>(count, ws2, cap, latent, bytes_out, mask_out, nonfinite);
  return cudaGetLastError();
}

cudaError_t launch_merge(int fmt, int64_t count, float ws2, const float *latent, uint8_t *scales_inout,
                         float *ongrid_delta, int64_t *changed, int sm_count, cudaStream_t stream) {
  if (changed) {
    cudaError_t e = cudaMemsetAsync(changed, 0, sizeof(int64_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (fmt == 0)
    sq_merge_kernel<0><<<grid, kThreads, 0, stream>>>(count, ws2, cap, latent, scales_inout, ongrid_delta, changed);
  else
    sq_merge_kernel<1><<<grid, kThreads, 0, stream>>>(count, ws2, cap, latent, scales_inout, ongrid_delta, changed);
  return cudaGetLastError();
}

cudaError_t launch_project_lowrank(int fmt, int64_t N, int64_t G, int r, float ws2, float alpha_over_r,
                                   const uint8_t *base, const uint16_t *B, const uint16_t *A, uint8_t *bytes_out,
                                   uint8_t *mask_out, int32_t *nonfinite, float *latent_out, cudaStream_t stream) {
  if (nonfinite) {
    cudaError_t e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const dim3 grid(static_cast<unsigned>((N + kLrRows - 1) / kLrRows), static_cast<unsigned>((G + kLrCols - 1) / kLrCols));
  const size_t smem = static_cast<size_t>(kLrRows + kLrCols) * r * sizeof(uint16_t);
  if (fmt == 0)
    sq_project_lowrank_kernel<0><<<grid, kThreads, smem, stream>>>(N, G, r, ws2, cap, alpha_over_r, base, B, A,
                                                                   bytes_out, mask_out, nonfinite, latent_out);
  else
    sq_project_lowrank_kernel<1><<<grid, kThreads, smem, stream>>>(N, G, r, ws2, cap, alpha_over_r, base, B, A,
                                                                   bytes_out, mask_out, nonfinite, latent_out);
  return cudaGetLastError();
}

size_t lowrank_grad_workspace(int64_t N, int64_t G, int r) {
  const int64_t chunks = (N + kDaRows - 1) / kDaRows;
  return static_cast<size_t>(chunks) * r * G * sizeof(float);
}

cudaError_t launch_lowrank_grad(int64_t N, int64_t G, int r, float alpha_over_r, const float *g, const uint16_t *B,
                                const uint16_t *A, float *dB, float *dA, float *workspace, int sm_count,
                                cudaStream_t stream) {
  if (dB) {
    const unsigned grid = static_cast<unsigned>((N + kWarps - 1) / kWarps);
    const size_t smem = static_cast<size_t>(min(r, 32)) * kDbChunk * sizeof(uint16_t);
    sq_lowrank_db_kernel<<<grid, kThreads, smem, stream>>>(N, G, r, alpha_over_r, g, A, dB);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (dA) {
    const int64_t chunks = (N + kDaRows - 1) / kDaRows;
    const dim3 grid1(static_cast<unsigned>(chunks), static_cast<unsigned>((G + 31) / 32));
    sq_lowrank_da_partial_kernel<<<grid1, kThreads, 0, stream>>>(N, G, r, g, B, workspace);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t count = static_cast<int64_t>(r) * G;
    int64_t blocks = (count + kThreads - 1) / kThreads;
    if (blocks > static_cast<int64_t>(sm_count) * kCtasPerSm) blocks = static_cast<int64_t>(sm_count) * kCtasPerSm;
    sq_lowrank_da_reduce_kernel<<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(G, r, chunks, alpha_over_r,
                                                                                      workspace, dA);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace sqi
