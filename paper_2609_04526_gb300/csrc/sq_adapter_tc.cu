// Adapter gradients of the low-rank scale adapter on the tensor cores (sm_103a).
//
// Sec. 3 "Scale-QLoRA forward": the latent is eff + (alpha/r) B A with B [N, r] and
// A [r, G] in bf16, so with gm = g * mask (the masked scale gradient, fp32 [N, G])
//   dB[n, j] = (alpha/r) sum_b gm[n, b] A[j, b]
//   dA[j, b] = (alpha/r) sum_n B[n, j] gm[n, b]
// One CTA owns 128 rows n of one expert's plane and a range of its blocks b, in
// steps of 64 blocks. Both products are tcgen05.mma kind::f16 (bf16 operands, fp32
// accumulation, M = 128). B and A are bf16 already; gm is split into three bf16
// parts hi + mid + lo (each the bf16 rounding of what the parts before it left), so
// the three products carry gm to about 2^-24 relative error. One shared-memory tile
// of a part, [128 n][64 b] with the 128-byte swizzle, is both dB's K-major A operand
// (rows n, contraction b) and dA's MN-major B operand (contraction n, columns b);
// B's rows [128 n][r j] are dA's MN-major A operand and A's step [r j][64 b] dB's
// K-major B operand, each in its natural layout. dB rows are written whole when one
// CTA covers all blocks, else per part and added in part order; the partial dA of a
// row chunk is added over the chunks in chunk order. Fixed order throughout, so
// reruns give identical bits.
#include "sq_gemm_kernels.cuh"

namespace sqi {
namespace {

constexpr int kAtThreads = 256;   // eight warps; warp w drains TMEM lanes 32 (w % 4) .. + 31, column half w / 4
constexpr int kAtRows = 128;      // rows n of gm per CTA: dB's M and dA's contraction per step
constexpr int kAtStep = 64;       // blocks b per step: one 128-byte row of bf16
constexpr int kAtMaxRank = 128;   // r limit of this path (dA's M)

// Shared memory, 1024-byte aligned, every tile with the 128-byte swizzle:
//   G[3]  [128 n][64 b] bf16  gm's step, parts hi, mid, lo            3 x 16 KiB
//   A     [128 j][64 b] bf16  A's step (rows j >= r zero)                 16 KiB
//   B     [128 n][128 j] bf16 B's rows, two 64-wide j atoms (j >= r zero) 32 KiB
struct AtSmem {
  static constexpr int kTile = kAtRows * 128;  // 16 KiB
  static constexpr int kOffG = 0, kOffA = 3 * kTile, kOffB = 4 * kTile, kOffBar = 6 * kTile;
  static constexpr int kBytes = kOffBar + 64 + 1024;  // barriers, TMEM slot, abort flag; alignment
};

// Byte offset of the 16-byte chunk `chunk` (8 bf16) of row `row` in a tile of
// 128-byte rows with the 128-byte swizzle (8-row, 1 KiB atoms).
__device__ __forceinline__ uint32_t sw128_chunk(int row, int chunk) {
  return static_cast<uint32_t>((row >> 3) * 1024 + (row & 7) * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ void sts32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.b32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t bf16_rn(float x) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(x)));
}

// x = hi + mid + lo, each a bf16 (round to nearest even), the remainders exact in fp32.
__device__ __forceinline__ void split3(float x, uint32_t &hi, uint32_t &mid, uint32_t &lo) {
  hi = bf16_rn(x);
  const float r1 = __fsub_rn(x, __uint_as_float(hi << 16));
  mid = bf16_rn(r1);
  const float r2 = __fsub_rn(r1, __uint_as_float(mid << 16));
  lo = bf16_rn(r2);
}

// grid (ceil(N / 128), parts * experts): CTA (c, p, e) covers rows 128 c .. + 127 and
// steps [p * steps_per, (p + 1) * steps_per) of 64 blocks. With one part its dB rows
// go to dB scaled by alpha_over_r; with several, each part's unscaled rows go to
// dB_part[e][p]. The partial dA of rows 128 c .. + 127 goes to dA_part[e][c].
__global__ void __launch_bounds__(kAtThreads, 2)
    sq_adapter_grad_tc_kernel(int64_t N, int64_t G, int r, float alpha_over_r, int parts, int steps_per,
                              const float *__restrict__ g_all, const uint16_t *__restrict__ B_all,
                              const uint16_t *__restrict__ A_all, float *__restrict__ dB_all,
                              float *__restrict__ dB_part, float *__restrict__ dA_part, int *err) {
  using S = AtSmem;
  extern __shared__ uint8_t at_smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(at_smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *bar = reinterpret_cast<uint64_t *>(smem + S::kOffBar);  // [0] MMAs done, [3] teardown
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bar + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t e = blockIdx.y / parts;
  const int part = static_cast<int>(blockIdx.y % parts);
  const int64_t chunks = gridDim.x;
  const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kAtRows;
  const float *g = g_all + e * N * G;
  const uint16_t *Bm = B_all + e * N * r;
  const uint16_t *Am = A_all + e * static_cast<int64_t>(r) * G;
  const int rp16 = (r + 15) & ~15;  // dB's N
  const uint32_t base = smem_u32(smem);
  const int all_steps = static_cast<int>((G + kAtStep - 1) / kAtStep);
  const int s_first = part * steps_per;
  const int steps = all_steps - s_first < steps_per ? all_steps - s_first : steps_per;

  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    mbar_init(bar + 3, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 0) tmem_alloc(tmem_slot, 256);  // dB: columns 0-127; dA steps: 128-191, 192-255

  // One step's gm in registers: thread t covers chunk (t & 7) of rows (t >> 3) + 32 i
  // (8 blocks each), loaded one step ahead of its use.
  const bool vec = (G & 3) == 0;  // rows 16-byte aligned (the plane is)
  const bool vecA = (G & 7) == 0 && (reinterpret_cast<uintptr_t>(Am) & 15u) == 0;  // A's bf16 rows likewise
  constexpr int kRowsPerThread = kAtRows * 8 / kAtThreads;
  float gv[kRowsPerThread][8];
  auto load = [&](int s) {
    const int64_t b0 = static_cast<int64_t>(s_first + s) * kAtStep + (threadIdx.x & 7) * 8;
#pragma unroll
    for (int i = 0; i < kRowsPerThread; ++i) {
      const int64_t n = n0 + (threadIdx.x >> 3) + (kAtThreads / 8) * i;
      const float *src = g + n * G + b0;
      if (n < N && vec && b0 + 8 <= G) {
        const float4 a = __ldg(reinterpret_cast<const float4 *>(src));
        const float4 c = __ldg(reinterpret_cast<const float4 *>(src) + 1);
        gv[i][0] = a.x; gv[i][1] = a.y; gv[i][2] = a.z; gv[i][3] = a.w;
        gv[i][4] = c.x; gv[i][5] = c.y; gv[i][6] = c.z; gv[i][7] = c.w;
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) gv[i][q] = (n < N && b0 + q < G) ? __ldg(src + q) : 0.f;
      }
    }
  };
  if (steps > 0) load(0);  // in flight while B is staged

  // B's rows of this chunk: row n (contraction), 128 j in two 64-wide atoms 16 KiB apart.
  // Each thread issues all its loads before any store (the shared stores are volatile:
  // interleaved, each load would wait for the store before it).
  if ((r & 1) == 0) {
    // the chunk's rows are contiguous in B: 4-byte pairs (j, j + 1), coalesced loads,
    // 32 in flight per thread before the stores; rows past N and j >= r stay zero below
    const int pairs = r / 2, words = kAtRows * pairs;
    const int64_t rows_here = N - n0 < kAtRows ? N - n0 : kAtRows;
    const uint32_t *src = reinterpret_cast<const uint32_t *>(Bm + n0 * r);  // 4-byte aligned: r even
    // zero fill of the pairs' 16-byte chunks that hold no data (j >= r rounded to 8, rows past N)
    for (int u = threadIdx.x; u < kAtRows * 16; u += kAtThreads) {
      const int nn = u >> 4, ch = u & 15;
      if (ch * 8 >= ((r + 7) & ~7) || nn >= rows_here)
        st_shared_v4(base + S::kOffB + (ch >> 3) * S::kTile + sw128_chunk(nn, ch & 7), 0u, 0u, 0u, 0u);
    }
    if ((r & 7) != 0) {  // the partial last chunk of each row: its words past r are zero
      for (int nn = threadIdx.x; nn < kAtRows; nn += kAtThreads) {
        const int ch = r >> 3;
        st_shared_v4(base + S::kOffB + (ch >> 3) * S::kTile + sw128_chunk(nn, ch & 7), 0u, 0u, 0u, 0u);
      }
    }
    __syncthreads();  // zeros before the data words that share their chunks
    for (int w0 = 0; w0 < words; w0 += 16 * kAtThreads) {
      uint32_t v[16];
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int w = w0 + q * kAtThreads + threadIdx.x;
        v[q] = (w < words && w / pairs < rows_here) ? __ldg(src + w) : 0u;
      }
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int w = w0 + q * kAtThreads + threadIdx.x;
        if (w < words && w / pairs < rows_here) {
          const int nn = w / pairs, j = 2 * (w - nn * pairs);
          const int ch = j >> 3;
          sts32(base + S::kOffB + (ch >> 3) * S::kTile + sw128_chunk(nn, ch & 7) + (j & 7) * 2, v[q]);
        }
      }
    }
  } else {
    const int nch = r <= 64 ? 8 : 16;  // 16-byte chunks of j per row holding data
    if (r <= 64) {  // the second atom (j >= 64) is all zeros
      for (int u = threadIdx.x; u < kAtRows * 8; u += kAtThreads)
        st_shared_v4(base + S::kOffB + S::kTile + sw128_chunk(u >> 3, u & 7), 0u, 0u, 0u, 0u);
    }
    uint32_t wb[kAtRows * 16 / kAtThreads][4];
#pragma unroll
    for (int i = 0; i < kAtRows * 16 / kAtThreads; ++i) {
      const int u = threadIdx.x + kAtThreads * i;  // 0 .. 2047 = 128 rows x 16 chunks
      const int nn = u >> 4, ch = u & 15;
      const int64_t n = n0 + nn;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int j = ch * 8 + 2 * q;
        const uint32_t lo = (ch < nch && n < N && j < r) ? static_cast<uint32_t>(__ldg(Bm + n * r + j)) : 0u;
        const uint32_t hi = (ch < nch && n < N && j + 1 < r) ? static_cast<uint32_t>(__ldg(Bm + n * r + j + 1)) : 0u;
        wb[i][q] = lo | (hi << 16);
      }
    }
#pragma unroll
    for (int i = 0; i < kAtRows * 16 / kAtThreads; ++i) {
      const int u = threadIdx.x + kAtThreads * i;
      const int nn = u >> 4, ch = u & 15;
      if (ch < nch)
        st_shared_v4(base + S::kOffB + (ch >> 3) * S::kTile + sw128_chunk(nn, ch & 7), wb[i][0], wb[i][1], wb[i][2],
                     wb[i][3]);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_lane = static_cast<uint32_t>((warp & 3) * 32) << 16;
  const int col_half = warp >> 2;  // which 32-column groups this warp drains
  const uint32_t idesc_db = idesc_bf16(128, rp16, 0, 0);         // A = gm part (K-major), B = A step (K-major)
  constexpr uint32_t idesc_da = idesc_bf16(128, kAtStep, 1, 1);  // A = B rows (MN-major), B = gm part (MN-major)
  bool ok = true;
  for (int s = 0; s < steps; ++s) {
    const int64_t b0 = static_cast<int64_t>(s_first + s) * kAtStep;
    // stage gm's three parts and A's step
#pragma unroll
    for (int i = 0; i < kRowsPerThread; ++i) {
      const int nn = (threadIdx.x >> 3) + (kAtThreads / 8) * i;
      uint32_t hi[4], mid[4], lo[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint32_t h0, m0, l0, h1, m1, l1;
        split3(gv[i][2 * q], h0, m0, l0);
        split3(gv[i][2 * q + 1], h1, m1, l1);
        hi[q] = h0 | (h1 << 16);
        mid[q] = m0 | (m1 << 16);
        lo[q] = l0 | (l1 << 16);
      }
      const uint32_t off = sw128_chunk(nn, threadIdx.x & 7);
      st_shared_v4(base + S::kOffG + off, hi[0], hi[1], hi[2], hi[3]);
      st_shared_v4(base + S::kOffG + S::kTile + off, mid[0], mid[1], mid[2], mid[3]);
      st_shared_v4(base + S::kOffG + 2 * S::kTile + off, lo[0], lo[1], lo[2], lo[3]);
    }
    {  // A's step: rows j < rp16, 8 chunks of 8 blocks; loads first, then the stores. A chunk
       // is 16 contiguous bytes of row j: one vector load where rows are 16-byte aligned.
      uint32_t wa[kAtMaxRank * 8 / kAtThreads][4];
#pragma unroll
      for (int i = 0; i < kAtMaxRank * 8 / kAtThreads; ++i) {
        const int u = threadIdx.x + kAtThreads * i;  // 0 .. 1023 = 128 rows x 8 chunks
        const int j = u >> 3, ch = u & 7;
        const int64_t bc = b0 + ch * 8;
        if (vecA && j < r && bc + 8 <= G) {
          const uint4 a = __ldg(reinterpret_cast<const uint4 *>(Am + j * G + bc));
          wa[i][0] = a.x;
          wa[i][1] = a.y;
          wa[i][2] = a.z;
          wa[i][3] = a.w;
          continue;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int64_t b = bc + 2 * q;
          const uint32_t lo = (j < r && b < G) ? static_cast<uint32_t>(__ldg(Am + j * G + b)) : 0u;
          const uint32_t hi = (j < r && b + 1 < G) ? static_cast<uint32_t>(__ldg(Am + j * G + b + 1)) : 0u;
          wa[i][q] = lo | (hi << 16);
        }
      }
#pragma unroll
      for (int i = 0; i < kAtMaxRank * 8 / kAtThreads; ++i) {
        const int u = threadIdx.x + kAtThreads * i;
        const int j = u >> 3, ch = u & 7;
        if (j < rp16) st_shared_v4(base + S::kOffA + sw128_chunk(j, ch), wa[i][0], wa[i][1], wa[i][2], wa[i][3]);
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) {
      tc_fence_after();
      // dB[n, j] += sum_b part[n, b] A[j, b]: 4 K-steps of 16 blocks, three parts each
#pragma unroll
      for (int kk = 0; kk < kAtStep / 16; ++kk) {
        const uint64_t bdesc = smem_desc_sw128(base + S::kOffA + kk * 32, 16, 1024);
#pragma unroll
        for (int pt = 0; pt < 3; ++pt)
          umma_bf16(tmem, smem_desc_sw128(base + S::kOffG + pt * S::kTile + kk * 32, 16, 1024), bdesc, idesc_db,
                    (s > 0 || kk > 0 || pt > 0) ? 1u : 0u);
      }
      // dA step [j, b] = sum_n B[n, j] part[n, b]: 8 K-steps of 16 rows n (2 KiB), three parts
      const uint32_t d_da = tmem + 128 + (s & 1) * kAtStep;
#pragma unroll
      for (int kk = 0; kk < kAtRows / 16; ++kk) {
        const uint64_t adesc = smem_desc_sw128(base + S::kOffB + kk * 2048, S::kTile, 1024);
#pragma unroll
        for (int pt = 0; pt < 3; ++pt)
          umma_bf16(d_da, adesc, smem_desc_sw128(base + S::kOffG + pt * S::kTile + kk * 2048, S::kTile, 1024),
                    idesc_da, (kk > 0 || pt > 0) ? 1u : 0u);
      }
      umma_commit(bar);
    }
    if (s + 1 < steps) load(s + 1);  // in flight during the MMAs
    if (!(ok = mbar_wait(bar, static_cast<uint32_t>(s) & 1u, abort_flag, err))) break;
    tc_fence_after();
    // drain this step's dA: lanes j = 32 (warp % 4) + lane, columns b 32 (warp / 4) .. + 31
    const int j = (warp & 3) * 32 + lane;
    {
      const int c0 = 32 * col_half;
      uint32_t v[32];
      tmem_ld32(tmem + t_lane + 128 + (s & 1) * kAtStep + c0, v);
      tmem_ld_wait();
      if (j < r) {
        float *dst = dA_part + ((e * chunks + blockIdx.x) * r + j) * G + b0 + c0;
        if (vec && b0 + c0 + 32 <= G) {
#pragma unroll
          for (int c = 0; c < 32; c += 4)
            *reinterpret_cast<float4 *>(dst + c) = make_float4(__uint_as_float(v[c]), __uint_as_float(v[c + 1]),
                                                               __uint_as_float(v[c + 2]), __uint_as_float(v[c + 3]));
        } else {
          for (int c = 0; c < 32 && b0 + c0 + c < G; ++c) dst[c] = __uint_as_float(v[c]);
        }
      }
    }
    tc_fence_before();
    __syncthreads();  // shared memory and this dA buffer are free for the next step
  }
  if (ok && dB_all && steps > 0) {
    tc_fence_after();
    // dB rows n0 .. n0 + 127 are one contiguous [rows x r] span of the output: staged
    // row-major in the (now free) gm / A tiles, then copied out with coalesced stores
    const float scale = parts > 1 ? 1.0f : alpha_over_r;
    float *dst = (parts > 1 ? dB_part + (e * parts + part) * N * r : dB_all + e * N * r) + n0 * r;
    const int nn = (warp & 3) * 32 + lane;
#pragma unroll 1
    for (int c0 = 32 * col_half; c0 < rp16; c0 += 64) {
      uint32_t v[32];
      tmem_ld32(tmem + t_lane + c0, v);
      tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < 32; ++c)
        if (c0 + c < r) sts32(base + S::kOffG + (nn * r + c0 + c) * 4, __float_as_uint(scale * __uint_as_float(v[c])));
    }
    __syncthreads();
    const int64_t rows_here = N - n0 < kAtRows ? N - n0 : kAtRows;
    const int64_t count = rows_here * r;
    const float *tile = reinterpret_cast<const float *>(smem + S::kOffG);
    if ((reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
      for (int64_t i = threadIdx.x; i < count / 4; i += kAtThreads)
        reinterpret_cast<float4 *>(dst)[i] = reinterpret_cast<const float4 *>(tile)[i];
      for (int64_t i = count / 4 * 4 + threadIdx.x; i < count; i += kAtThreads) dst[i] = tile[i];
    } else {
      for (int64_t i = threadIdx.x; i < count; i += kAtThreads) dst[i] = tile[i];
    }
  }
  if (!ok && threadIdx.x == 0) {  // a wait ran out: let this CTA's MMAs finish before TMEM is freed
    umma_commit(bar + 3);
    mbar_drain(bar + 3, 0);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// out[e][i] = scale * the sum of part[e][c][i] over c. A CTA covers 32 consecutive
// outputs; its warp w sums the parts c = w, w + W, ... (W warps, four loads in flight
// per lane), and warp 0 adds the W sums in warp order. The order depends only on the
// part count, so the result does not depend on the launch.
__global__ void __launch_bounds__(256) sq_adapter_tc_reduce_kernel(int64_t count, int64_t experts, int64_t nparts,
                                                                   float scale, const float *__restrict__ part,
                                                                   float *__restrict__ out) {
  __shared__ float red[8][32];
  const int W = blockDim.x >> 5, w = threadIdx.x >> 5, l = threadIdx.x & 31;
  const int64_t t = static_cast<int64_t>(blockIdx.x) * 32 + l;
  float acc = 0.f;
  if (t < count * experts) {
    const int64_t e = t / count, i = t - e * count;
    const float *src = part + e * nparts * count + i;
    float s[4] = {0.f, 0.f, 0.f, 0.f};
    int64_t c = w;
    for (; c + 3 * W < nparts; c += 4 * W) {
      float v[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) v[q] = __ldg(src + (c + q * W) * count);
#pragma unroll
      for (int q = 0; q < 4; ++q) s[q] += v[q];
    }
    for (int q = 0; c < nparts; c += W, ++q) s[q] += __ldg(src + c * count);
    acc = (s[0] + s[1]) + (s[2] + s[3]);
  }
  red[w][l] = acc;
  __syncthreads();
  if (w == 0 && t < count * experts) {
    float sum = red[0][l];
    for (int q = 1; q < W; ++q) sum += red[q][l];
    out[t] = scale * sum;
  }
}

// Few parts: each thread adds four consecutive outputs' parts in part order with
// 16-byte loads (count % 4 == 0 and 16-byte aligned planes), grid-stride.
__global__ void __launch_bounds__(256) sq_adapter_tc_reduce4_kernel(int64_t count, int64_t experts, int64_t nparts,
                                                                    float scale, const float *__restrict__ part,
                                                                    float *__restrict__ out) {
  const int64_t quads = count / 4 * experts;
  for (int64_t q = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x; q < quads;
       q += static_cast<int64_t>(gridDim.x) * 256) {
    const int64_t e = q / (count / 4), i = q - e * (count / 4);
    const float4 *src = reinterpret_cast<const float4 *>(part + e * nparts * count) + i;
    float4 s = __ldg(src);
    for (int64_t c = 1; c < nparts; ++c) {
      const float4 v = __ldg(src + c * (count / 4));
      s.x += v.x;
      s.y += v.y;
      s.z += v.z;
      s.w += v.w;
    }
    reinterpret_cast<float4 *>(out + e * count)[i] = make_float4(scale * s.x, scale * s.y, scale * s.z, scale * s.w);
  }
}

// Launch shape of the reductions: up to 16 parts (and 4 | count) the grid-stride
// vector kernel, else 32 outputs per CTA with one warp per part up to 8. Both add
// the parts of an output in a fixed order.
static cudaError_t launch_tc_reduce(int64_t count, int64_t experts, int64_t nparts, float scale, const float *part,
                                    float *out, int sm_count, cudaStream_t stream) {
  if (nparts <= 16 && count % 4 == 0 && ((reinterpret_cast<uintptr_t>(out) | reinterpret_cast<uintptr_t>(part)) & 15u) == 0) {
    const int64_t want = (count / 4 * experts + 255) / 256, cap = static_cast<int64_t>(sm_count) * 8;
    sq_adapter_tc_reduce4_kernel<<<static_cast<unsigned>(want < cap ? want : cap), 256, 0, stream>>>(
        count, experts, nparts, scale, part, out);
    return cudaGetLastError();
  }
  const int64_t blocks = (count * experts + 31) / 32;
  const int warps = nparts < 8 ? static_cast<int>(nparts) : 8;
  sq_adapter_tc_reduce_kernel<<<static_cast<unsigned>(blocks), 32 * warps, 0, stream>>>(count, experts, nparts, scale,
                                                                                        part, out);
  return cudaGetLastError();
}

// Parts of the block range per row chunk: about one wave of CTAs (two fit per SM);
// every part costs its own staging of B's rows and, dB, a partial plane.
int tc_parts(int64_t N, int64_t G, int experts, int sm_count) {
  const int64_t chunks = (N + kAtRows - 1) / kAtRows, steps = (G + kAtStep - 1) / kAtStep;
  const int64_t ctas = chunks * experts;
  int64_t p = 2 * static_cast<int64_t>(sm_count) / ctas;
  if (p > steps) p = steps;
  if (p > 65535 / experts) p = 65535 / experts;
  if (p < 1) p = 1;
  const int64_t per = (steps + p - 1) / p;
  return static_cast<int>((steps + per - 1) / per);  // every part has steps
}

}  // namespace

bool lowrank_grad_tc_supported(int r) { return r >= 1 && r <= kAtMaxRank; }

size_t lowrank_grad_tc_workspace(int64_t N, int64_t G, int r, int experts, int sm_count) {
  const int64_t chunks = (N + kAtRows - 1) / kAtRows;
  const int parts = tc_parts(N, G, experts, sm_count);
  const int64_t dbp = parts > 1 ? static_cast<int64_t>(parts) * N * r : 0;
  return static_cast<size_t>(experts) * static_cast<size_t>(chunks * r * G + dbp) * sizeof(float);
}

cudaError_t launch_lowrank_grad_tc(int64_t N, int64_t G, int r, float alpha_over_r, const float *g,
                                   const uint16_t *B, const uint16_t *A, float *dB, float *dA, float *workspace,
                                   int *err, int sm_count, cudaStream_t stream, int experts) {
  static int done_mask = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (!(done_mask & (1 << (dev & 31)))) {
    cudaError_t e = cudaFuncSetAttribute(sq_adapter_grad_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         AtSmem::kBytes);
    if (e != cudaSuccess) return e;
    done_mask |= 1 << (dev & 31);
  }
  const int64_t chunks = (N + kAtRows - 1) / kAtRows, steps = (G + kAtStep - 1) / kAtStep;
  const int parts = tc_parts(N, G, experts, sm_count);
  const int steps_per = static_cast<int>((steps + parts - 1) / parts);
  float *dA_part = workspace, *dB_part = workspace + experts * chunks * r * G;
  const dim3 grid(static_cast<unsigned>(chunks), static_cast<unsigned>(parts * experts));
  sq_adapter_grad_tc_kernel<<<grid, kAtThreads, AtSmem::kBytes, stream>>>(
      N, G, r, alpha_over_r, parts, steps_per, g, B, A, dB, dB_part, dA_part, err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (dB && parts > 1 &&
      (e = launch_tc_reduce(N * r, experts, parts, alpha_over_r, dB_part, dB, sm_count, stream)) != cudaSuccess)
    return e;
  if (!dA) return cudaSuccess;
  return launch_tc_reduce(static_cast<int64_t>(r) * G, experts, chunks, alpha_over_r, dA_part, dA, sm_count, stream);
}

}  // namespace sqi
