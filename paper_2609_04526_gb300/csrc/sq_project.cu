// Grid projection and merge kernels (sm_103a): Sec. 3 QAST round_grid with the
// E4M3 ceiling clamp of the stability recipe, and the merge that rewrites scale
// bytes only (Sec. 3 "QAST makes merge exact by construction").
//
// Both are HBM-bandwidth kernels: each thread owns 16 consecutive latents per
// step (four 16-byte loads), writes 16 bytes of each output with one 16-byte
// store, and the grid is a whole number of waves over the SMs (grid-stride).
// Counters (NaN latents, changed bytes) are reduced within each warp and added
// with one atomic per warp.
#include <algorithm>

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

// Planes of several experts in one launch (PER instantiations): element i belongs
// to expert i / plane and takes that expert's tensor scale; plane is a multiple
// of 16, so one 16-element vector never straddles two experts.
__device__ __forceinline__ void expert_scale(const float *ws2_per, int64_t plane, int64_t i, float &ws2, float &cap) {
  ws2 = __ldg(ws2_per + i / plane);
  cap = 448.0f * ws2;  // the same IEEE fp32 product as the host's single-plane cap
}

template <int FMT, bool PER>
__global__ void __launch_bounds__(kThreads) sq_project_kernel(int64_t count, float ws2_all, float cap_all,
                                                              const float *__restrict__ ws2_per, int64_t plane,
                                                              const float *__restrict__ latent,
                                                              uint8_t *__restrict__ bytes_out,
                                                              uint8_t *__restrict__ mask_out,
                                                              int32_t *__restrict__ nonfinite) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t nan_count = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    float ws2 = ws2_all, cap = cap_all;
    if (PER) expert_scale(ws2_per, plane, 16 * v, ws2, cap);
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
    float ws2 = ws2_all, cap = cap_all;
    if (PER) expert_scale(ws2_per, plane, i, ws2, cap);
    uint32_t b, m, n;
    project_one<FMT>(latent[i], ws2, cap, b, m, n);
    bytes_out[i] = static_cast<uint8_t>(b);
    if (mask_out) mask_out[i] = static_cast<uint8_t>(m);
    nan_count += n;
  }
  if (nonfinite) warp_add_i32(nonfinite, nan_count);
}

template <int FMT, bool PER>
__global__ void __launch_bounds__(kThreads) sq_merge_kernel(int64_t count, float ws2_all, float cap_all,
                                                            const float *__restrict__ ws2_per, int64_t plane,
                                                            const float *__restrict__ latent,
                                                            uint8_t *__restrict__ scales,
                                                            float *__restrict__ delta,
                                                            int64_t *__restrict__ changed) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t n_changed = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    float ws2 = ws2_all, cap = cap_all;
    if (PER) expert_scale(ws2_per, plane, 16 * v, ws2, cap);
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
    float ws2 = ws2_all, cap = cap_all;
    if (PER) expert_scale(ws2_per, plane, i, ws2, cap);
    uint32_t b, m, n;
    project_one<FMT>(latent[i], ws2, cap, b, m, n);
    const uint32_t o = scales[i];
    scales[i] = static_cast<uint8_t>(b);
    n_changed += (b != o) ? 1u : 0u;
    if (delta) delta[i] = __fsub_rn(scale_value<FMT>(b, ws2), scale_value<FMT>(o, ws2));
  }
  if (changed) warp_add_i64(changed, n_changed);
}

// ---------------------------------------------------------------- several planes per launch
//
// The planes of all linears of a layer (Sec. 5 Payoff 3: the merge touches every
// target linear) in one launch each for projection and merge. Every CTA works on
// kPlaneVecs 16-element vectors of one plane (the CTAs of plane j follow those of
// plane j - 1), so it reduces its counter within the block and adds it with one
// atomic; the last CTA to finish (a ticket) writes every plane's count and clears
// the accumulators for the next call.
constexpr int kPlaneVecsPerThread = 2;
constexpr int kPlaneVecs = kThreads * kPlaneVecsPerThread;

__device__ __forceinline__ int plane_of_block(const PlaneTable &t, int64_t b, int64_t &first_block) {
  int64_t start = 0;
  for (int j = 0; j < t.n; ++j) {
    const int64_t nb = (t.p[j].count / 16 + kPlaneVecs - 1) / kPlaneVecs;
    if (b < start + nb) {
      first_block = start;
      return j;
    }
    start += nb;
  }
  first_block = start;
  return t.n;  // not reached: the grid covers the planes exactly
}

// Block sum of v; the result is valid in thread 0.
__device__ __forceinline__ uint32_t block_sum(uint32_t v, uint32_t *red) {
  v = __reduce_add_sync(0xFFFFFFFFu, v);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  uint32_t s = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kThreads / 32; ++w) s += red[w];
  return s;
}

// Adds this CTA's count of plane j to acc[j]; the last CTA writes the totals to the
// planes' counters (int32 for the projection, int64 for the merge) and clears acc.
template <bool I64>
__device__ __forceinline__ void plane_counters(const PlaneTable &t, int j, uint32_t mine, int64_t *acc,
                                               uint32_t *red) {
  const uint32_t s = block_sum(mine, red);
  if (threadIdx.x != 0) return;
  if (s) atomicAdd(reinterpret_cast<unsigned long long *>(acc + j), static_cast<unsigned long long>(s));
  __threadfence();
  unsigned int *ticket = reinterpret_cast<unsigned int *>(acc + kMaxPlanes);
  if (atomicAdd(ticket, 1u) != gridDim.x - 1) return;
  __threadfence();
  for (int q = 0; q < t.n; ++q) {
    const unsigned long long v = atomicExch(reinterpret_cast<unsigned long long *>(acc + q), 0ull);
    if (t.p[q].counter) {
      if (I64)
        *static_cast<int64_t *>(t.p[q].counter) = static_cast<int64_t>(v);
      else
        *static_cast<int32_t *>(t.p[q].counter) = static_cast<int32_t>(v);
    }
  }
  *ticket = 0u;
}

// Four consecutive blocks of a plane (one float4 of latents) -> their bytes, mask bytes
// and NaN count, each block exactly as project_one. NVFP4 converts two blocks per
// instruction; a NaN latent's byte is patched afterwards (rare).
template <int FMT>
__device__ __forceinline__ void project4(float4 L4, float ws2, float cap, uint32_t &bytes, uint32_t &mask,
                                         uint32_t &nan) {
  const float l[4] = {L4.x, L4.y, L4.z, L4.w};
  bytes = mask = nan = 0;
  if (FMT == 0) {
    float q[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      nan += (l[c] != l[c]) ? 1u : 0u;
      mask |= (fabsf(l[c]) <= cap ? 1u : 0u) << (8 * c);  // false for NaN, as -cap <= L <= cap
      q[c] = __fdiv_rn(fminf(fmaxf(l[c], -cap), cap), ws2);
    }
    bytes = e4m3x2_rn(q[0], q[1]) | (e4m3x2_rn(q[2], q[3]) << 16);
    if (nan) {
#pragma unroll
      for (int c = 0; c < 4; ++c)
        if (l[c] != l[c]) bytes = (bytes & ~(0xFFu << (8 * c))) | (0x7Fu << (8 * c));
    }
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint32_t b, m, n;
      project_one<FMT>(l[c], ws2, cap, b, m, n);
      bytes |= b << (8 * c);
      mask |= m << (8 * c);
      nan += n;
    }
  }
}

// A CTA's chunk is kPlaneVecs x 16 blocks: lane t of the CTA takes float4 t + kThreads * i
// of it (i < 4 kPlaneVecsPerThread), so each warp-wide load reads 512 contiguous bytes and
// each store of bytes writes 128. A thread loads all its latents (and, merging, the old
// bytes) before it computes and stores any: the byte stores could alias the latent
// loads as far as the compiler knows, so interleaving them would serialise every
// float4 on the memory latency.
constexpr int kPlaneF4 = 4 * kPlaneVecsPerThread;  // float4s per thread per chunk

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_project_planes_kernel(const __grid_constant__ PlaneTable t,
                                                                        int64_t *acc) {
  __shared__ uint32_t red[kThreads / 32];
  int64_t first_block;
  const int j = plane_of_block(t, blockIdx.x, first_block);
  const PlaneArgs &pl = t.p[j];
  const float ws2 = pl.ws2, cap = 448.0f * pl.ws2;  // the same IEEE fp32 product as the single-plane cap
  const int64_t nf4 = pl.count / 4;
  const int64_t f0 = (static_cast<int64_t>(blockIdx.x) - first_block) * (4 * kPlaneVecs) + threadIdx.x;
  const float4 *src = reinterpret_cast<const float4 *>(pl.latent);
  float4 L[kPlaneF4];
#pragma unroll
  for (int i = 0; i < kPlaneF4; ++i) {
    const int64_t f = f0 + static_cast<int64_t>(i) * kThreads;
    if (f < nf4) L[i] = __ldcs(src + f);
  }
  uint32_t nan_count = 0;
#pragma unroll
  for (int i = 0; i < kPlaneF4; ++i) {
    const int64_t f = f0 + static_cast<int64_t>(i) * kThreads;
    if (f >= nf4) break;
    uint32_t by, mk, na;
    project4<FMT>(L[i], ws2, cap, by, mk, na);
    __stcs(reinterpret_cast<unsigned int *>(pl.bytes) + f, by);
    if (pl.mask) __stcs(reinterpret_cast<unsigned int *>(pl.mask) + f, mk);
    nan_count += na;
  }
  plane_counters<false>(t, j, nan_count, acc, red);
}

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_merge_planes_kernel(const __grid_constant__ PlaneTable t,
                                                                      int64_t *acc) {
  __shared__ uint32_t red[kThreads / 32];
  int64_t first_block;
  const int j = plane_of_block(t, blockIdx.x, first_block);
  const PlaneArgs &pl = t.p[j];
  const float ws2 = pl.ws2, cap = 448.0f * pl.ws2;
  const int64_t nf4 = pl.count / 4;
  const int64_t f0 = (static_cast<int64_t>(blockIdx.x) - first_block) * (4 * kPlaneVecs) + threadIdx.x;
  const float4 *src = reinterpret_cast<const float4 *>(pl.latent);
  uint32_t *art = reinterpret_cast<uint32_t *>(pl.bytes);
  float4 L[kPlaneF4];
  uint32_t old[kPlaneF4];
#pragma unroll
  for (int i = 0; i < kPlaneF4; ++i) {
    const int64_t f = f0 + static_cast<int64_t>(i) * kThreads;
    if (f < nf4) {
      L[i] = __ldcs(src + f);
      old[i] = art[f];
    }
  }
  uint32_t n_changed = 0;
#pragma unroll
  for (int i = 0; i < kPlaneF4; ++i) {
    const int64_t f = f0 + static_cast<int64_t>(i) * kThreads;
    if (f >= nf4) break;
    uint32_t by, mk, na;
    project4<FMT>(L[i], ws2, cap, by, mk, na);
    art[f] = by;
    n_changed += static_cast<uint32_t>(__popc(__vcmpne4(by, old[i]))) >> 3;  // 0xFF per differing byte
    if (pl.delta) {
      float d[4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
        d[c] = __fsub_rn(scale_value<FMT>((by >> (8 * c)) & 0xFFu, ws2), scale_value<FMT>((old[i] >> (8 * c)) & 0xFFu, ws2));
      __stcs(reinterpret_cast<float4 *>(pl.delta) + f, make_float4(d[0], d[1], d[2], d[3]));
    }
  }
  plane_counters<true>(t, j, n_changed, acc, red);
}

// ---------------------------------------------------------------- rollback, swap, audit
//
// Sec. 5 Payoff 3: a merge is undone by subtracting the on-grid delta it applied;
// each byte becomes the projection (the merge's grid and clamp path) of
// fl32(s(byte) - delta). Sec. 5 "Hot-swap": the served task changes by overwriting
// the scale plane with another adapter's bytes. Both count the bytes they change;
// the audit counts the bytes in which two buffers differ (e.g. a code plane before
// and after a merge). Same layout as the merge: 16 bytes per thread per step.

__device__ __forceinline__ uint32_t bytes_differing(uint32_t a, uint32_t b) {
  return static_cast<uint32_t>(__popc(__vcmpne4(a, b))) >> 3;  // 0xFF per differing byte
}

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_rollback_kernel(int64_t count, float ws2, float cap,
                                                               const float *__restrict__ delta,
                                                               uint8_t *__restrict__ scales,
                                                               int64_t *__restrict__ changed) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  uint32_t n_changed = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const float4 *src = reinterpret_cast<const float4 *>(delta) + 4 * v;
    float d[16];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 f = __ldcs(src + q);
      d[4 * q] = f.x;
      d[4 * q + 1] = f.y;
      d[4 * q + 2] = f.z;
      d[4 * q + 3] = f.w;
    }
    const uint4 old4 = *(reinterpret_cast<const uint4 *>(scales) + v);
    const uint32_t old[4] = {old4.x, old4.y, old4.z, old4.w};
    uint32_t ob[4] = {0, 0, 0, 0};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t o = (old[i >> 2] >> (8 * (i & 3))) & 0xFFu;
      uint32_t b, m, n;
      project_one<FMT>(__fsub_rn(scale_value<FMT>(o, ws2), d[i]), ws2, cap, b, m, n);
      ob[i >> 2] |= b << (8 * (i & 3));
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) n_changed += bytes_differing(ob[q], old[q]);
    *(reinterpret_cast<uint4 *>(scales) + v) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
  }
  if (blockIdx.x == 0 && threadIdx.x < count - nvec * 16) {
    const int64_t i = nvec * 16 + threadIdx.x;
    const uint32_t o = scales[i];
    uint32_t b, m, n;
    project_one<FMT>(__fsub_rn(scale_value<FMT>(o, ws2), delta[i]), ws2, cap, b, m, n);
    scales[i] = static_cast<uint8_t>(b);
    n_changed += (b != o) ? 1u : 0u;
  }
  if (changed) warp_add_i64(changed, n_changed);
}

// b <- a (when `write`) and count the bytes in which a and b differ. A thread loads
// four 16-byte vectors of each buffer before it stores any: a store to the address
// just loaded waits for that load, so one vector per step would serialise every
// thread on the memory latency.
constexpr int kSwapUnroll = 4;

__global__ void __launch_bounds__(kThreads) sq_swap_or_diff_kernel(int64_t count, const uint8_t *__restrict__ a,
                                                                   uint8_t *__restrict__ b, bool write,
                                                                   int64_t *__restrict__ differing) {
  const int64_t nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const uint4 *va = reinterpret_cast<const uint4 *>(a);
  uint4 *vb = reinterpret_cast<uint4 *>(b);
  uint32_t n = 0;
  for (int64_t v0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; v0 < nvec;
       v0 += stride * kSwapUnroll) {
    uint4 x[kSwapUnroll], y[kSwapUnroll];
#pragma unroll
    for (int u = 0; u < kSwapUnroll; ++u) {
      const int64_t v = v0 + stride * u;
      if (v < nvec) {
        x[u] = __ldcs(va + v);
        y[u] = vb[v];
      }
    }
#pragma unroll
    for (int u = 0; u < kSwapUnroll; ++u) {
      const int64_t v = v0 + stride * u;
      if (v < nvec) {
        n += bytes_differing(x[u].x, y[u].x) + bytes_differing(x[u].y, y[u].y) + bytes_differing(x[u].z, y[u].z) +
             bytes_differing(x[u].w, y[u].w);
        if (write) __stcs(vb + v, x[u]);
      }
    }
  }
  if (blockIdx.x == 0 && threadIdx.x < count - nvec * 16) {
    const int64_t i = nvec * 16 + threadIdx.x;
    n += (a[i] != b[i]) ? 1u : 0u;
    if (write) b[i] = a[i];
  }
  if (differing) warp_add_i64(differing, n);
}

// ---------------------------------------------------------------- low-rank scale adapter
//
// Sec. 3 "Scale-QLoRA forward": the latent block scale eff' = eff + (alpha/r) (B A),
// B [N, r] and A [r, G] bf16, formed in fp32 in a fixed order -- eff = fl32(decoded
// base byte * ws2) (scale_value), acc = fused multiply-adds over j = 0 .. r-1 from 0,
// eff' = fma(alpha/r, acc, eff) -- and projected exactly as sq_project_kernel.
// The adapters of the E experts of an MoE linear (Sec. 3 "MoE: a batched
// grouped-expert kernel") run in the same launches: expert e's planes and factors
// follow expert e - 1's, and grid z (with the contraction chunk for the products)
// selects the expert; a dense call is the case E = 1.
// The three adapter kernels are register-tiled fp32 CUDA-core products: a CTA of 256
// threads owns a 64 x 64 output tile, its operands staged in shared memory as fp32
// (contraction index outermost), and each thread accumulates a 4 x 4 sub-tile (rows
// ty*4 .. +3, columns tx*4 .. +3), so two 16-byte shared-memory loads feed 16 fused
// multiply-adds. Every output is summed sequentially over the contraction index, so
// results do not change between runs.
constexpr int kT = 64;   // output tile edge
constexpr int kTP = 68;  // padded row of a staged operand (16-byte multiple; spreads the transposed stores)

__device__ __forceinline__ float bf16_bits(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_project_lowrank_kernel(
    int64_t N, int64_t G, int r, float ws2, float cap, const float *__restrict__ ws2_per, float aor,
    const uint8_t *__restrict__ base, const uint16_t *__restrict__ B, const uint16_t *__restrict__ A,
    uint8_t *__restrict__ bytes_out, uint8_t *__restrict__ mask_out, int32_t *__restrict__ nonfinite,
    float *__restrict__ latent_out) {
  extern __shared__ float lr_smem[];
  float *sB = lr_smem;             // [r][kTP]: B[n0 + row][j] at j * kTP + row
  float *sA = lr_smem + kTP * r;   // [r][kT columns]
  const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kT;
  const int64_t b0 = static_cast<int64_t>(blockIdx.y) * kT;
  // expert blockIdx.z: its planes, factors and (NVFP4 experts) tensor scale
  const int64_t e = blockIdx.z, plane = N * G;
  base += e * plane;
  B += e * N * r;
  A += e * r * G;
  bytes_out += e * plane;
  if (mask_out) mask_out += e * plane;
  if (latent_out) latent_out += e * plane;
  if (ws2_per) {
    ws2 = __ldg(ws2_per + e);
    cap = 448.0f * ws2;  // the same IEEE fp32 product as the host's single-plane cap
  }
  {  // B's rows n0 .. n0 + 63 are kT * r contiguous elements; (row, j) of element i advance
     // by (kThreads / r, kThreads % r) per step, so no step divides by r
    int row = static_cast<int>(threadIdx.x) / r, j = static_cast<int>(threadIdx.x) % r;
    const int drow = kThreads / r, dj = kThreads % r;
    for (int i = threadIdx.x; i < kT * r; i += kThreads) {
      const int64_t n = n0 + row;
      sB[j * kTP + row] = n < N ? bf16_bits(B[n0 * r + i]) : 0.f;
      row += drow;
      j += dj;
      if (j >= r) {
        j -= r;
        ++row;
      }
    }
  }
  for (int i = threadIdx.x; i < r * kT; i += kThreads) {
    const int64_t b = b0 + i % kT;
    sA[i] = b < G ? bf16_bits(A[static_cast<int64_t>(i / kT) * G + b]) : 0.f;
  }
  __syncthreads();
  const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
  float acc[4][4];
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[q][c] = 0.f;
  for (int j = 0; j < r; ++j) {
    const float4 b4 = *reinterpret_cast<const float4 *>(sB + j * kTP + ty * 4);
    const float4 a4 = *reinterpret_cast<const float4 *>(sA + j * kT + tx * 4);
    const float bv[4] = {b4.x, b4.y, b4.z, b4.w}, av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[q][c] = fmaf(bv[q], av[c], acc[q][c]);
  }
  uint32_t nan_count = 0;
  // four consecutive blocks of a row per thread: one 4-byte load of the base bytes and
  // one 4-byte (16-byte for the latent) store per output where the row allows it
  const bool vec = (G & 3) == 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int64_t n = n0 + ty * 4 + q, bq = b0 + tx * 4;
    if (n >= N) continue;
    const int64_t i0 = n * G + bq;
    if (vec && bq + 3 < G) {
      const uint32_t base4 = __ldg(reinterpret_cast<const uint32_t *>(base + i0));
      float Lv[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) Lv[c] = fmaf(aor, acc[q][c], scale_value<FMT>((base4 >> (8 * c)) & 0xFFu, ws2));
      uint32_t by4, mk4, na;
      project4<FMT>(make_float4(Lv[0], Lv[1], Lv[2], Lv[3]), ws2, cap, by4, mk4, na);
      nan_count += na;
      *reinterpret_cast<uint32_t *>(bytes_out + i0) = by4;
      if (mask_out) *reinterpret_cast<uint32_t *>(mask_out + i0) = mk4;
      if (latent_out) *reinterpret_cast<float4 *>(latent_out + i0) = make_float4(Lv[0], Lv[1], Lv[2], Lv[3]);
      continue;
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int64_t b = bq + c;
      if (b < G) {
        const int64_t i = i0 + c;
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

// Adapter gradients from the masked scale gradient g [N, G], as two products with
// the contraction split into chunks (one CTA per 64 x 64 output tile and chunk,
// partial results summed by a second kernel in chunk order):
//   dB[n,j] = (alpha/r) sum_b g[n,b] A[j,b]      (P = g, Q^T = A; contraction over b)
//   dA[j,b] = (alpha/r) sum_n B[n,j] g[n,b]      (P = B^T, Q = g; contraction over n)
// A CTA stages kKStep contraction indices of both operands per step in shared
// memory (fp32), loading the next step into registers while it computes this one.
constexpr int kKStep = 16;  // contraction indices per staged step

// Operand element (row i of the output, contraction index k) for the two products.
// `estride` is the distance between two experts' operands; expert(e) is expert e's.
struct DbLeft {  // g[n = i][b = k]
  const float *g;
  int64_t G, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return g[i * G + k]; }
  __device__ DbLeft expert(int64_t e) const { return DbLeft{g + e * estride, G, estride}; }
};
struct DbRight {  // A[j = i][b = k]
  const uint16_t *A;
  int64_t G, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return bf16_bits(A[i * G + k]); }
  __device__ DbRight expert(int64_t e) const { return DbRight{A + e * estride, G, estride}; }
};
struct DaLeft {  // B[n = k][j = i]
  const uint16_t *B;
  int64_t r, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return bf16_bits(B[k * r + i]); }
  __device__ DaLeft expert(int64_t e) const { return DaLeft{B + e * estride, r, estride}; }
};
struct DaRight {  // g[n = k][b = i]
  const float *g;
  int64_t G, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return g[k * G + i]; }
  __device__ DaRight expert(int64_t e) const { return DaRight{g + e * estride, G, estride}; }
};

struct DsLeft {  // B[n = i][j = k] (the control's coefficient plane dS = (alpha/r) B A)
  const uint16_t *B;
  int64_t r, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return bf16_bits(B[i * r + k]); }
  __device__ DsLeft expert(int64_t e) const { return DsLeft{B + e * estride, r, estride}; }
};
struct DsRight {  // A[j = k][b = i]
  const uint16_t *A;
  int64_t G, estride;
  __device__ float operator()(int64_t i, int64_t k) const { return bf16_bits(A[k * G + i]); }
  __device__ DsRight expert(int64_t e) const { return DsRight{A + e * estride, G, estride}; }
};

// partial[e][c][i][j] = sum_{k in chunk c} L_e(i, k) R_e(j, k), i < rows, j < cols,
// for expert e = blockIdx.z / chunks and chunk c = blockIdx.z % chunks.
template <class LeftT, class RightT, bool LEFT_K_FAST, bool RIGHT_K_FAST>
__global__ void __launch_bounds__(kThreads) sq_adapter_product_kernel(int64_t rows, int64_t cols, int64_t kdim,
                                                                      int64_t kchunk, int64_t chunks, LeftT left_all,
                                                                      RightT right_all, float *__restrict__ partial) {
  __shared__ __align__(16) float sl[2][kKStep][kTP];  // [buffer][k][i]
  __shared__ __align__(16) float sr[2][kKStep][kTP];  // [buffer][k][j]
  const int64_t expert = blockIdx.z / chunks, chunk = blockIdx.z % chunks;
  const LeftT left = left_all.expert(expert);
  const RightT right = right_all.expert(expert);
  const int64_t i0 = static_cast<int64_t>(blockIdx.x) * kT;
  const int64_t j0 = static_cast<int64_t>(blockIdx.y) * kT;
  const int64_t kb = chunk * kchunk;
  const int64_t ke = kdim < kb + kchunk ? kdim : kb + kchunk;
  const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
  // staging map: 4 elements of each operand per thread and step; consecutive threads
  // walk the operand's contiguous index (k when it is the fast one, else the row)
  float pl[4], pr[4];
  auto load = [&](int64_t k0) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = threadIdx.x + kThreads * e;  // 0 .. 1023 = kKStep * kT
      const int kk_l = LEFT_K_FAST ? idx % kKStep : idx / kT, ii = LEFT_K_FAST ? idx / kKStep : idx % kT;
      const int64_t k = k0 + kk_l, i = i0 + ii;
      pl[e] = (k < ke && i < rows) ? left(i, k) : 0.f;
      const int kk_r = RIGHT_K_FAST ? idx % kKStep : idx / kT, jj = RIGHT_K_FAST ? idx / kKStep : idx % kT;
      const int64_t k2 = k0 + kk_r, j = j0 + jj;
      pr[e] = (k2 < ke && j < cols) ? right(j, k2) : 0.f;
    }
  };
  auto store = [&](int buf) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = threadIdx.x + kThreads * e;
      const int kk_l = LEFT_K_FAST ? idx % kKStep : idx / kT, ii = LEFT_K_FAST ? idx / kKStep : idx % kT;
      sl[buf][kk_l][ii] = pl[e];
      const int kk_r = RIGHT_K_FAST ? idx % kKStep : idx / kT, jj = RIGHT_K_FAST ? idx / kKStep : idx % kT;
      sr[buf][kk_r][jj] = pr[e];
    }
  };
  float acc[4][4];
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[q][c] = 0.f;
  int buf = 0;
  load(kb);
  store(0);
  __syncthreads();
  for (int64_t k0 = kb; k0 < ke; k0 += kKStep) {
    const bool more = k0 + kKStep < ke;
    if (more) load(k0 + kKStep);  // in flight while this step computes
#pragma unroll
    for (int kk = 0; kk < kKStep; ++kk) {
      const float4 l4 = *reinterpret_cast<const float4 *>(&sl[buf][kk][ty * 4]);
      const float4 r4 = *reinterpret_cast<const float4 *>(&sr[buf][kk][tx * 4]);
      const float lv[4] = {l4.x, l4.y, l4.z, l4.w}, rv[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
      for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[q][c] = fmaf(lv[q], rv[c], acc[q][c]);
    }
    if (more) {
      store(buf ^ 1);
      __syncthreads();
      buf ^= 1;
    }
  }
  float *out = partial + static_cast<int64_t>(blockIdx.z) * rows * cols;
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int64_t i = i0 + ty * 4 + q, j = j0 + tx * 4 + c;
      if (i < rows && j < cols) out[i * cols + j] = acc[q][c];
    }
}

// out[e][i] = scale * sum over chunks c (in order) of partial[e][c][i], for the
// `experts` outputs of `count` elements each.
__global__ void __launch_bounds__(kThreads) sq_adapter_reduce_kernel(int64_t count, int64_t experts, int64_t chunks,
                                                                     float scale, const float *__restrict__ partial,
                                                                     float *__restrict__ out) {
  const int64_t total = count * experts;
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * kThreads) {
    const int64_t e = t / count, i = t - e * count;
    const float *src = partial + e * chunks * count + i;
    float s = 0.f;
    for (int64_t c = 0; c < chunks; ++c) s += src[c * count];
    out[t] = scale * s;
  }
}

// ---------------------------------------------------------------- scale-family variants
//
// Least-squares code-preserving fit (ablation appendix, the Spider paragraph): the
// updates a block can represent are multiples t * c of its code values c, so the
// best scale delta for a weight update dW is <c, dW> / <c, c> (0 for a block of
// zero codes), in absolute scale units. One thread per block; the block's codes
// and bf16 update are contiguous (B / 2 and 2 B bytes), so a warp reads whole
// segments. fp32 sums in element order: c * dW, c * c and dW * dW are exact (E2M1
// values have two significant bits, bf16 eight), the sums round.

// E2M1 nibble -> fp32 from the format's fields: sign bit 3, exponent bits 1-2
// (bias 1), mantissa bit 0; exponent 0 is the subnormal 0 or 0.5.
__device__ __forceinline__ float e2m1_value(uint32_t nib) {
  const uint32_t e = (nib >> 1) & 3u, m = nib & 1u;
  const uint32_t mag = e == 0 ? (m ? 0x3F000000u : 0u) : (((126u + e) << 23) | (m << 22));
  return __uint_as_float(mag | ((nib & 8u) << 28));
}

template <int FMT>
__device__ __forceinline__ void fit_one(int64_t i, float ws2, const uint32_t (&cw32)[(FMT == 0 ? 16 : 32) / 8],
                                        const uint4 (&w4)[(FMT == 0 ? 16 : 32) / 8],
                                        const uint8_t *__restrict__ scales, float *__restrict__ delta,
                                        float *__restrict__ captured, float *__restrict__ total,
                                        float *__restrict__ latent) {
  constexpr int B = FMT == 0 ? 16 : 32;
  float cwsum = 0.f, ccsum = 0.f, wwsum = 0.f;
#pragma unroll
  for (int q = 0; q < B / 8; ++q) {
    const uint32_t wv[4] = {w4[q].x, w4[q].y, w4[q].z, w4[q].w};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float c = e2m1_value((cw32[q] >> (4 * j)) & 0xFu);
      const float w = __uint_as_float(j & 1 ? wv[j >> 1] & 0xFFFF0000u : wv[j >> 1] << 16);
      // the products are exact in fp32 (at most 2 + 8 or 8 + 8 significant bits), so a
      // fused multiply-add rounds exactly as the product followed by the sum
      cwsum = __fmaf_rn(c, w, cwsum);
      ccsum = __fmaf_rn(c, c, ccsum);
      wwsum = __fmaf_rn(w, w, wwsum);
    }
  }
  const float d = ccsum > 0.f ? __fdiv_rn(cwsum, ccsum) : 0.f;
  delta[i] = d;
  if (captured) captured[i] = ccsum > 0.f ? __fdiv_rn(__fmul_rn(cwsum, cwsum), ccsum) : 0.f;
  if (total) total[i] = wwsum;
  if (latent) latent[i] = __fadd_rn(scale_value<FMT>(scales[i], ws2), d);
}

// Each thread fits blocks i and i + stride per iteration, so the loads of both are in
// flight before either is reduced.
template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_fit_kernel(int64_t blocks, float ws2, const uint8_t *__restrict__ codes,
                                                          const uint8_t *__restrict__ scales,
                                                          const uint16_t *__restrict__ dW, float *__restrict__ delta,
                                                          float *__restrict__ captured, float *__restrict__ total,
                                                          float *__restrict__ latent) {
  constexpr int B = FMT == 0 ? 16 : 32;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; i < blocks; i += 2 * stride) {
    const int64_t i2 = i + stride;
    const bool two = i2 < blocks;
    uint32_t ca[B / 8], cb[B / 8];
    uint4 wa[B / 8], wb[B / 8];
#pragma unroll
    for (int q = 0; q < B / 8; ++q) {
      ca[q] = __ldg(reinterpret_cast<const uint32_t *>(codes + i * (B / 2)) + q);
      wa[q] = __ldcs(reinterpret_cast<const uint4 *>(dW + i * B) + q);
      if (two) {
        cb[q] = __ldg(reinterpret_cast<const uint32_t *>(codes + i2 * (B / 2)) + q);
        wb[q] = __ldcs(reinterpret_cast<const uint4 *>(dW + i2 * B) + q);
      }
    }
    fit_one<FMT>(i, ws2, ca, wa, scales, delta, captured, total, latent);
    if (two) fit_one<FMT>(i2, ws2, cb, wb, scales, delta, captured, total, latent);
  }
}

// Granularity ladder (ablation appendix): one additive scale delta per group of
// W = G / gd consecutive blocks of a row. Its gradient is the sum of the group's
// block gradients. One warp per group: lane l sums blocks l, l + 32, ... in order
// (coalesced loads), then a fixed butterfly of shuffles adds the 32 partial sums,
// so the result is the same on every run.
__global__ void __launch_bounds__(kThreads) sq_group_reduce_kernel(int64_t groups, int64_t W,
                                                                   const float *__restrict__ g,
                                                                   float *__restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5); t < groups; t += warps) {
    const float *src = g + t * W;
    float s = 0.f;
    for (int64_t b = lane; b < W; b += 32) s = __fadd_rn(s, __ldg(src + b));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s = __fadd_rn(s, __shfl_xor_sync(0xFFFFFFFFu, s, o));
    if (lane == 0) out[t] = s;
  }
}

// The group-delta latent fl32(s(base byte) + delta[n, b / W]) projected onto the grid
// (the a5 device code), with mask, NaN count and the latent itself for the merge.
// 16 consecutive blocks per thread (16-byte loads and stores, as the projection);
// the row and group of each block are stepped along, since a vector may cross rows.
template <int FMT>
__device__ __forceinline__ void project_group_one(int64_t n, int64_t b, int64_t gd, int64_t W, float ws2, float cap,
                                                  uint32_t base_byte, const float *__restrict__ delta, uint32_t &by,
                                                  uint32_t &mk, uint32_t &na, float &L) {
  L = __fadd_rn(scale_value<FMT>(base_byte, ws2), __ldg(delta + n * gd + b / W));
  project_one<FMT>(L, ws2, cap, by, mk, na);
}

template <int FMT>
__global__ void __launch_bounds__(kThreads) sq_project_group_delta_kernel(
    int64_t N, int64_t G, int64_t W, float ws2, float cap, const uint8_t *__restrict__ base,
    const float *__restrict__ delta, uint8_t *__restrict__ bytes_out, uint8_t *__restrict__ mask_out,
    int32_t *__restrict__ nonfinite, float *__restrict__ latent_out) {
  const int64_t count = N * G, gd = G / W, nvec = count / 16;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
  uint32_t nan_count = 0;
  for (int64_t v = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; v < nvec; v += stride) {
    const uint4 b4 = __ldcs(reinterpret_cast<const uint4 *>(base) + v);
    const uint32_t bw[4] = {b4.x, b4.y, b4.z, b4.w};
    int64_t n = (16 * v) / G, b = 16 * v - n * G;
    uint32_t ob[4] = {0, 0, 0, 0}, om[4] = {0, 0, 0, 0};
    float L[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      uint32_t by, mk, na;
      project_group_one<FMT>(n, b, gd, W, ws2, cap, (bw[i >> 2] >> (8 * (i & 3))) & 0xFFu, delta, by, mk, na, L[i]);
      ob[i >> 2] |= by << (8 * (i & 3));
      om[i >> 2] |= mk << (8 * (i & 3));
      nan_count += na;
      if (++b == G) {
        b = 0;
        ++n;
      }
    }
    __stcs(reinterpret_cast<uint4 *>(bytes_out) + v, make_uint4(ob[0], ob[1], ob[2], ob[3]));
    if (mask_out) __stcs(reinterpret_cast<uint4 *>(mask_out) + v, make_uint4(om[0], om[1], om[2], om[3]));
    if (latent_out) {
      float4 *dst = reinterpret_cast<float4 *>(latent_out) + 4 * v;
#pragma unroll
      for (int q = 0; q < 4; ++q) __stcs(dst + q, make_float4(L[4 * q], L[4 * q + 1], L[4 * q + 2], L[4 * q + 3]));
    }
  }
  // ragged tail (< 16 blocks) by the first threads of block 0
  if (blockIdx.x == 0 && threadIdx.x < count - nvec * 16) {
    const int64_t i = nvec * 16 + threadIdx.x, n = i / G, b = i - n * G;
    uint32_t by, mk, na;
    float L;
    project_group_one<FMT>(n, b, gd, W, ws2, cap, base[i], delta, by, mk, na, L);
    bytes_out[i] = static_cast<uint8_t>(by);
    if (mask_out) mask_out[i] = static_cast<uint8_t>(mk);
    if (latent_out) latent_out[i] = L;
    nan_count += na;
  }
  if (nonfinite) warp_add_i32(nonfinite, nan_count);
}

// Contraction chunks for an output of `tiles` 64 x 64 tiles: enough CTAs for about
// two per SM, chunks of at least 4 steps.
int64_t adapter_chunks(int64_t kdim, int64_t tiles, int sm_count) {
  int64_t want = (2 * static_cast<int64_t>(sm_count) + tiles - 1) / tiles;
  const int64_t most = (kdim + 4 * kKStep - 1) / (4 * kKStep);
  if (want > most) want = most;
  return want < 1 ? 1 : want;
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
                           uint8_t *mask_out, int32_t *nonfinite, int sm_count, cudaStream_t stream,
                           const float *ws2_per, int64_t plane) {
  if (nonfinite) {
    cudaError_t e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (ws2_per)  // several NVFP4 experts, each with its own tensor scale
    sq_project_kernel<0, true><<<grid, kThreads, 0, stream>>>(count, ws2, cap, ws2_per, plane, latent, bytes_out,
                                                              mask_out, nonfinite);
  else if (fmt == 0)
    sq_project_kernel<0, false><<<grid, kThreads, 0, stream>>>(count, ws2, cap, nullptr, 0, latent, bytes_out,
                                                               mask_out, nonfinite);
  else
    sq_project_kernel<1, false><<<grid, kThreads, 0, stream>>>(count, ws2, cap, nullptr, 0, latent, bytes_out,
                                                               mask_out, nonfinite);
  return cudaGetLastError();
}

cudaError_t launch_merge(int fmt, int64_t count, float ws2, const float *latent, uint8_t *scales_inout,
                         float *ongrid_delta, int64_t *changed, int sm_count, cudaStream_t stream,
                         const float *ws2_per, int64_t plane) {
  if (changed) {
    cudaError_t e = cudaMemsetAsync(changed, 0, sizeof(int64_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (ws2_per)  // several NVFP4 experts, each with its own tensor scale
    sq_merge_kernel<0, true><<<grid, kThreads, 0, stream>>>(count, ws2, cap, ws2_per, plane, latent, scales_inout,
                                                            ongrid_delta, changed);
  else if (fmt == 0)
    sq_merge_kernel<0, false><<<grid, kThreads, 0, stream>>>(count, ws2, cap, nullptr, 0, latent, scales_inout,
                                                             ongrid_delta, changed);
  else
    sq_merge_kernel<1, false><<<grid, kThreads, 0, stream>>>(count, ws2, cap, nullptr, 0, latent, scales_inout,
                                                             ongrid_delta, changed);
  return cudaGetLastError();
}

static unsigned planes_grid(const PlaneTable &t) {
  int64_t g = 0;
  for (int j = 0; j < t.n; ++j) g += (t.p[j].count / 16 + kPlaneVecs - 1) / kPlaneVecs;
  return static_cast<unsigned>(g);
}

cudaError_t launch_project_planes(int fmt, const PlaneTable &t, int64_t *acc, cudaStream_t stream) {
  const unsigned grid = planes_grid(t);
  if (grid == 0) {  // no blocks at all: the counters still receive 0
    for (int j = 0; j < t.n; ++j)
      if (t.p[j].counter) {
        cudaError_t e = cudaMemsetAsync(t.p[j].counter, 0, sizeof(int32_t), stream);
        if (e != cudaSuccess) return e;
      }
    return cudaSuccess;
  }
  if (fmt == 0)
    sq_project_planes_kernel<0><<<grid, kThreads, 0, stream>>>(t, acc);
  else
    sq_project_planes_kernel<1><<<grid, kThreads, 0, stream>>>(t, acc);
  return cudaGetLastError();
}

cudaError_t launch_merge_planes(int fmt, const PlaneTable &t, int64_t *acc, cudaStream_t stream) {
  const unsigned grid = planes_grid(t);
  if (grid == 0) {
    for (int j = 0; j < t.n; ++j)
      if (t.p[j].counter) {
        cudaError_t e = cudaMemsetAsync(t.p[j].counter, 0, sizeof(int64_t), stream);
        if (e != cudaSuccess) return e;
      }
    return cudaSuccess;
  }
  if (fmt == 0)
    sq_merge_planes_kernel<0><<<grid, kThreads, 0, stream>>>(t, acc);
  else
    sq_merge_planes_kernel<1><<<grid, kThreads, 0, stream>>>(t, acc);
  return cudaGetLastError();
}

cudaError_t launch_project_lowrank(int fmt, int64_t N, int64_t G, int r, float ws2, float alpha_over_r,
                                   const uint8_t *base, const uint16_t *B, const uint16_t *A, uint8_t *bytes_out,
                                   uint8_t *mask_out, int32_t *nonfinite, float *latent_out, cudaStream_t stream,
                                   int experts, const float *ws2_per) {
  if (nonfinite) {
    cudaError_t e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const dim3 grid(static_cast<unsigned>((N + kT - 1) / kT), static_cast<unsigned>((G + kT - 1) / kT),
                  static_cast<unsigned>(experts));
  const size_t smem = static_cast<size_t>(kTP + kT) * r * sizeof(float);  // <= 132 KiB for r <= 256
  cudaError_t e;
  if (fmt == 0) {
    if ((e = cudaFuncSetAttribute(sq_project_lowrank_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess)
      return e;
    sq_project_lowrank_kernel<0><<<grid, kThreads, smem, stream>>>(N, G, r, ws2, cap, ws2_per, alpha_over_r, base,
                                                                   B, A, bytes_out, mask_out, nonfinite, latent_out);
  } else {
    if ((e = cudaFuncSetAttribute(sq_project_lowrank_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess)
      return e;
    sq_project_lowrank_kernel<1><<<grid, kThreads, smem, stream>>>(N, G, r, ws2, cap, nullptr, alpha_over_r, base,
                                                                   B, A, bytes_out, mask_out, nonfinite, latent_out);
  }
  return cudaGetLastError();
}

// Workspace of the adapter gradients: the partial products of dB and of dA (all experts).
size_t lowrank_grad_workspace(int64_t N, int64_t G, int r, int sm_count, int experts) {
  if (lowrank_grad_tc_supported(r)) return lowrank_grad_tc_workspace(N, G, r, experts, sm_count);
  const int64_t tb = ((N + kT - 1) / kT) * ((r + kT - 1) / kT) * experts;
  const int64_t ta = ((r + kT - 1) / kT) * ((G + kT - 1) / kT) * experts;
  const int64_t cb = adapter_chunks(G, tb, sm_count), ca = adapter_chunks(N, ta, sm_count);
  return static_cast<size_t>(experts) * static_cast<size_t>(cb * N * r + ca * r * G) * sizeof(float);
}

cudaError_t launch_lowrank_grad(int64_t N, int64_t G, int r, float alpha_over_r, const float *g, const uint16_t *B,
                                const uint16_t *A, float *dB, float *dA, float *workspace, int sm_count,
                                cudaStream_t stream, int *err, int experts) {
  if (lowrank_grad_tc_supported(r))
    return launch_lowrank_grad_tc(N, G, r, alpha_over_r, g, B, A, dB, dA, workspace, err, sm_count, stream, experts);
  const int64_t tb = ((N + kT - 1) / kT) * ((r + kT - 1) / kT) * experts;
  const int64_t ta = ((r + kT - 1) / kT) * ((G + kT - 1) / kT) * experts;
  const int64_t cb = adapter_chunks(G, tb, sm_count), ca = adapter_chunks(N, ta, sm_count);
  float *pb = workspace, *pa = workspace + static_cast<int64_t>(experts) * cb * N * r;
  const unsigned reduce_cap = static_cast<unsigned>(sm_count) * kCtasPerSm;
  cudaError_t e;
  if (dB) {  // rows n, columns j, contraction b: g is b-contiguous, A is b-contiguous
    const int64_t kc = ((G + cb - 1) / cb + kKStep - 1) / kKStep * kKStep;
    const int64_t chunks = (G + kc - 1) / kc;
    const dim3 grid(static_cast<unsigned>((N + kT - 1) / kT), static_cast<unsigned>((r + kT - 1) / kT),
                    static_cast<unsigned>(chunks * experts));
    sq_adapter_product_kernel<DbLeft, DbRight, true, true><<<grid, kThreads, 0, stream>>>(
        N, r, G, kc, chunks, DbLeft{g, G, N * G}, DbRight{A, G, static_cast<int64_t>(r) * G}, pb);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int64_t count = N * r;
    const unsigned blocks =
        static_cast<unsigned>(std::min<int64_t>((count * experts + kThreads - 1) / kThreads, reduce_cap));
    sq_adapter_reduce_kernel<<<blocks, kThreads, 0, stream>>>(count, experts, chunks, alpha_over_r, pb, dB);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (dA) {  // rows j, columns b, contraction n: B is j-contiguous (row index fast), g is b-contiguous
    const int64_t kc = ((N + ca - 1) / ca + kKStep - 1) / kKStep * kKStep;
    const int64_t chunks = (N + kc - 1) / kc;
    const dim3 grid(static_cast<unsigned>((r + kT - 1) / kT), static_cast<unsigned>((G + kT - 1) / kT),
                    static_cast<unsigned>(chunks * experts));
    sq_adapter_product_kernel<DaLeft, DaRight, false, false><<<grid, kThreads, 0, stream>>>(
        r, G, N, kc, chunks, DaLeft{B, r, N * r}, DaRight{g, G, N * G}, pa);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int64_t count = static_cast<int64_t>(r) * G;
    const unsigned blocks =
        static_cast<unsigned>(std::min<int64_t>((count * experts + kThreads - 1) / kThreads, reduce_cap));
    sq_adapter_reduce_kernel<<<blocks, kThreads, 0, stream>>>(count, experts, chunks, alpha_over_r, pa, dA);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_fit(int fmt, int64_t N, int64_t K, float ws2, const uint8_t *codes, const uint8_t *scales,
                       const uint16_t *dW, float *delta, float *captured, float *total, float *latent, int sm_count,
                       cudaStream_t stream) {
  const int64_t blocks = N * (K / (fmt == 0 ? 16 : 32));
  if (blocks == 0) return cudaSuccess;
  // two blocks per thread and iteration; up to eight CTAs per SM keep enough loads in flight
  const int64_t want = (blocks + 2 * kThreads - 1) / (2 * kThreads), cap = static_cast<int64_t>(sm_count) * 8;
  const unsigned grid = static_cast<unsigned>(want < cap ? want : cap);
  if (fmt == 0)
    sq_fit_kernel<0><<<grid, kThreads, 0, stream>>>(blocks, ws2, codes, scales, dW, delta, captured, total, latent);
  else
    sq_fit_kernel<1><<<grid, kThreads, 0, stream>>>(blocks, ws2, codes, scales, dW, delta, captured, total, latent);
  return cudaGetLastError();
}

cudaError_t launch_group_reduce(int64_t N, int64_t G, int64_t gd, const float *g, float *out, int sm_count,
                                cudaStream_t stream) {
  const int64_t groups = N * gd;
  if (groups == 0) return cudaSuccess;
  const int64_t per = kThreads / 32;  // one warp per group
  const int64_t want = (groups + per - 1) / per, cap = static_cast<int64_t>(sm_count) * 8;
  sq_group_reduce_kernel<<<static_cast<unsigned>(want < cap ? want : cap), kThreads, 0, stream>>>(groups, G / gd, g,
                                                                                                   out);
  return cudaGetLastError();
}

cudaError_t launch_project_group_delta(int fmt, int64_t N, int64_t G, int64_t gd, float ws2, const uint8_t *base,
                                       const float *delta, uint8_t *bytes_out, uint8_t *mask_out, int32_t *nonfinite,
                                       float *latent_out, int sm_count, cudaStream_t stream) {
  if (nonfinite) {
    cudaError_t e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  const int64_t count = N * G;
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (fmt == 0)
    sq_project_group_delta_kernel<0><<<grid, kThreads, 0, stream>>>(N, G, G / gd, ws2, cap, base, delta, bytes_out,
                                                                    mask_out, nonfinite, latent_out);
  else
    sq_project_group_delta_kernel<1><<<grid, kThreads, 0, stream>>>(N, G, G / gd, ws2, cap, base, delta, bytes_out,
                                                                    mask_out, nonfinite, latent_out);
  return cudaGetLastError();
}

size_t lowrank_product_workspace(int64_t N, int64_t G, int r, int sm_count) {
  const int64_t tiles = ((N + kT - 1) / kT) * ((G + kT - 1) / kT);
  return static_cast<size_t>(adapter_chunks(r, tiles, sm_count) * N * G) * sizeof(float);
}

cudaError_t launch_lowrank_product(int64_t N, int64_t G, int r, float alpha_over_r, const uint16_t *B,
                                   const uint16_t *A, float *out, float *workspace, int sm_count,
                                   cudaStream_t stream) {
  const int64_t tiles = ((N + kT - 1) / kT) * ((G + kT - 1) / kT);
  const int64_t c = adapter_chunks(r, tiles, sm_count);
  const int64_t kc = ((r + c - 1) / c + kKStep - 1) / kKStep * kKStep;
  const int64_t chunks = (r + kc - 1) / kc;
  const dim3 grid(static_cast<unsigned>((N + kT - 1) / kT), static_cast<unsigned>((G + kT - 1) / kT),
                  static_cast<unsigned>(chunks));
  // rows n, columns b, contraction j: B is j-contiguous, A is b-contiguous
  sq_adapter_product_kernel<DsLeft, DsRight, true, false><<<grid, kThreads, 0, stream>>>(
      N, G, r, kc, chunks, DsLeft{B, r, 0}, DsRight{A, G, 0}, workspace);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t count = N * G;
  const unsigned cap = static_cast<unsigned>(sm_count) * kCtasPerSm;
  const unsigned blocks = static_cast<unsigned>(std::min<int64_t>((count + kThreads - 1) / kThreads, cap));
  sq_adapter_reduce_kernel<<<blocks, kThreads, 0, stream>>>(count, 1, chunks, alpha_over_r, workspace, out);
  return cudaGetLastError();
}

cudaError_t launch_rollback(int fmt, int64_t count, float ws2, const float *delta, uint8_t *scales_inout,
                            int64_t *changed, int sm_count, cudaStream_t stream) {
  if (changed) {
    cudaError_t e = cudaMemsetAsync(changed, 0, sizeof(int64_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  const float cap = 448.0f * ws2;  // one IEEE fp32 multiply
  const unsigned grid = grid_for(count, sm_count);
  if (fmt == 0)
    sq_rollback_kernel<0><<<grid, kThreads, 0, stream>>>(count, ws2, cap, delta, scales_inout, changed);
  else
    sq_rollback_kernel<1><<<grid, kThreads, 0, stream>>>(count, ws2, cap, delta, scales_inout, changed);
  return cudaGetLastError();
}

cudaError_t launch_swap_or_diff(int64_t count, const uint8_t *a, uint8_t *b, bool write, int64_t *differing,
                                int sm_count, cudaStream_t stream) {
  if (differing) {
    cudaError_t e = cudaMemsetAsync(differing, 0, sizeof(int64_t), stream);
    if (e != cudaSuccess) return e;
  }
  if (count == 0) return cudaSuccess;
  sq_swap_or_diff_kernel<<<grid_for(count, sm_count), kThreads, 0, stream>>>(count, a, b, write, differing);
  return cudaGetLastError();
}

}  // namespace sqi
