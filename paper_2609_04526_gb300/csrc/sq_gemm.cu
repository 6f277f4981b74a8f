// tcgen05 contraction kernels of the scale-only training step (sm_103a).
//
//   MODE_FWD   Y[m,n]  = sum_k X[m,k] W[n,k]        Sec. 3 "Scale-QLoRA forward"
//   MODE_DX    dX[m,k] = sum_n dY[m,n] W[n,k]       its input gradient
//   MODE_SGRAD g[n,b]  = sum_{k in b} code[n,k] sum_m dY[m,n] X[m,k]   its scale gradient
//
// with W[n,k] = code[n,k] * s[n, k/B] (Sec. 2). One CTA owns one 128 x 256 fp32
// accumulator tile in tensor memory (TMEM) and runs warp-specialised roles:
//   warps 0-3  decode (FWD/DX): packed E2M1 nibbles x scale byte -> bf16 operand
//              tile written straight into the 128B-swizzled smem layout the
//              tensor core reads; then the epilogue (TMEM -> registers -> HBM).
//   warp 4     TMA producer: streams the bf16 activation tiles into a 4-stage ring.
//   warp 5     TMEM allocator and the single MMA-issuing thread (tcgen05.mma,
//              kind::f16 with bf16 operands, fp32 accumulation).
// For MODE_SGRAD both operands are MN-major TMA tiles (dY^T and X, contraction
// over tokens); the epilogue multiplies each dW element by its code and sums
// every block of B columns in registers, so dW never reaches HBM.
//
// Every mbarrier wait is bounded (kWaitLimitNs): on expiry the CTA records
// kErrWaitTimeout in the device error word, stops issuing, drains what it has
// in flight and frees its TMEM.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "sq_internal.h"

namespace sqi {
namespace {

constexpr int kThreads = 192;
constexpr int kDecodeWarps = 4;
constexpr uint32_t kTmemCols = 256;
constexpr int kAStageBytes = kBM * kBK * 2;  // 16 KiB
constexpr int kBStageBytes = kBN * kBK * 2;  // 32 KiB
constexpr int kSmemBytes = kStages * (kAStageBytes + kBStageBytes) + 1024 /*align*/ + 256 /*barriers*/;
constexpr unsigned long long kWaitLimitNs = 1000000000ull;  // 1 s

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on a phase parity. Returns false if the CTA has aborted or the
// wait ran out (then the abort flag and the device error word are set).
__device__ __noinline__ bool mbar_wait_slow(uint64_t *bar, uint32_t parity, volatile int *abort_flag, int *err) {
  const unsigned long long t0 = globaltimer();
  while (true) {
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) {
      *abort_flag = 1;
      atomicOr(err, kErrWaitTimeout);
      return false;
    }
  }
}

__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag, int *err) {
  if (mbar_try_wait(bar, parity)) return true;
  return mbar_wait_slow(bar, parity, abort_flag, err);
}

// Bounded wait used only while tearing down after an abort: waits for work this
// CTA already put in flight (TMA copies, MMAs), ignoring the abort flag.
__device__ __noinline__ void mbar_drain(uint64_t *bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer() - t0 > kWaitLimitNs) return;
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, uint64_t *bar, int32_t x,
                                            int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 in, fp32 accumulate).
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread completes.
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 consecutive fp32 columns: thread i of the warp gets lane (base lane + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
        "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
        "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr)
      : "memory");
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor, 128-byte swizzle (sm_100 family format):
// start address >> 4 in bits 0-13, leading byte offset >> 4 in 16-29, stride
// byte offset >> 4 in 32-45, descriptor version 1 in bits 46-47, swizzle mode
// 2 (128B) in bits 61-63. K-major tiles: SBO = 1024 (8 rows x 128 B), LBO
// unused. MN-major tiles: LBO = distance between 64-element MN atoms, SBO =
// 1024 (8 contraction rows).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A and B bf16
// (bits 7-9 = 1, 10-12 = 1), A / B MN-major flags (bits 15 / 16), N >> 3 in
// bits 17-22, M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, int a_mn, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(a_mn) << 15) |
         (static_cast<uint32_t>(b_mn) << 16) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
               : "memory");
}

// ------------------------------------------------------------- code decode

// prmt with the sign-replicate mode (selector nibble bit 3 set).
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

__device__ __forceinline__ uint32_t bf16x2_mul(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Eight E2M1 nibbles (element j in bits 4j..4j+3) -> four bf16x2 words, element
// 2i in the low half of word i. Magnitude bytes come from two 8-entry byte
// tables indexed with prmt (bf16 of 0, .5, 1, 1.5, 2, 3, 4, 6 is
// 0000 3F00 3F80 3FC0 4000 4040 4080 40C0); the sign bit of each nibble is
// replicated with prmt's sign mode and OR-ed into the high byte.
__device__ __forceinline__ void e2m1x8_to_bf16(uint32_t w, uint32_t (&o)[4]) {
  constexpr uint32_t kLoA = 0xC0800000u, kLoB = 0xC0804000u;  // low bytes, magnitudes 0-3 / 4-7
  constexpr uint32_t kHiA = 0x3F3F3F00u, kHiB = 0x40404040u;  // high bytes
  const uint32_t m_lo = w & 0x7777u;
  const uint32_t m_hi = (w >> 16) & 0x7777u;
  const uint32_t e = w << 4;  // msb of byte i of e = sign of element 2i
  const uint32_t s0 = prmt(e, w, 0xD9C8u);  // sign-replicated bytes of elements 0..3
  const uint32_t s1 = prmt(e, w, 0xFBEAu);  // elements 4..7
  const uint32_t l0 = prmt(kLoA, kLoB, m_lo);
  const uint32_t h0 = prmt(kHiA, kHiB, m_lo) | (s0 & 0x80808080u);
  const uint32_t l1 = prmt(kLoA, kLoB, m_hi);
  const uint32_t h1 = prmt(kHiA, kHiB, m_hi) | (s1 & 0x80808080u);
  o[0] = prmt(l0, h0, 0x5140u);
  o[1] = prmt(l0, h0, 0x7362u);
  o[2] = prmt(l1, h1, 0x5140u);
  o[3] = prmt(l1, h1, 0x7362u);
}

// Scale byte -> bf16 value replicated in both halves (exact: E4M3 has 4
// significant bits, E8M0 is a power of two).
template <int FMT>
__device__ __forceinline__ uint32_t scale_bf16x2(uint32_t byte) {
  uint32_t u;
  if (FMT == 0) {
    const __half_raw hr = __nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(byte), __NV_E4M3);
    const float f = __half2float(__half(hr));
    u = __bfloat16_as_ushort(__float2bfloat16_rn(f));
  } else {
    u = byte == 0 ? 0x0040u : (byte == 255 ? 0x7FC0u : (byte << 7));
  }
  return u | (u << 16);
}

// ------------------------------------------------------------- the kernel

struct KParams {
  const uint8_t *codes;
  const uint8_t *scales;
  float ws2;
  int64_t M, N, K;
  void *out;
  const uint8_t *mask;
  int *err;
};

template <int MODE, int FMT>
__global__ void __launch_bounds__(kThreads, 1)
    sq_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const KParams p) {
  constexpr int B = FMT == 0 ? 16 : 32;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *sA = smem;
  uint8_t *sB = smem + kStages * kAStageBytes;
  uint64_t *bars = reinterpret_cast<uint64_t *>(sB + kStages * kBStageBytes);
  uint64_t *afull = bars;                  // TMA tiles landed        (1 arrival + tx)
  uint64_t *bfull = bars + kStages;        // decoded B tile written  (kDecodeWarps arrivals)
  uint64_t *empty = bars + 2 * kStages;    // MMAs reading the stage completed (tcgen05.commit)
  uint64_t *tfull = bars + 3 * kStages;    // accumulator complete
  uint64_t *drain = bars + 3 * kStages + 1;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 3 * kStages + 2);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // GEMM view: rows (TMEM lanes) x cols (TMEM columns), contraction Kg.
  const int64_t row0 = static_cast<int64_t>(blockIdx.x) * kBM;
  const int64_t col0 = static_cast<int64_t>(blockIdx.y) * kBN;
  const int64_t Mg = MODE == MODE_SGRAD ? p.N : p.M;
  const int64_t Ng = MODE == MODE_FWD ? p.N : p.K;
  const int64_t Kg = MODE == MODE_FWD ? p.K : (MODE == MODE_DX ? p.N : p.M);
  const int num_k = static_cast<int>((Kg + kBK - 1) / kBK);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&afull[s], 1);
      mbar_init(&bfull[s], kDecodeWarps);
      mbar_init(&empty[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, kTmemCols);
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&tmA);
    if (MODE == MODE_SGRAD) tma_prefetch_desc(&tmB);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 4) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      int issued = 0;
      for (int it = 0; it < num_k; ++it) {
        const int s = it % kStages;
        const uint32_t use = static_cast<uint32_t>(it / kStages);
        if (it >= kStages && !mbar_wait(&empty[s], (use & 1u) ^ 1u, abort_flag, p.err)) break;
        const int32_t kc = it * kBK;  // contraction offset
        const uint32_t a_dst = smem_u32(sA + s * kAStageBytes);
        if (MODE == MODE_SGRAD) {
          mbar_arrive_expect_tx(&afull[s], kAStageBytes + kBStageBytes);
          const uint32_t b_dst = smem_u32(sB + s * kBStageBytes);
          // dY^T tile: two 64(n) x 64(m) boxes; X tile: four 64(k) x 64(m) boxes.
          for (int j = 0; j < kBM / 64; ++j)
            tma_load_2d(a_dst + j * (kBK * 128), &tmA, &afull[s], static_cast<int32_t>(row0) + 64 * j, kc);
          for (int j = 0; j < kBN / 64; ++j)
            tma_load_2d(b_dst + j * (kBK * 128), &tmB, &afull[s], static_cast<int32_t>(col0) + 64 * j, kc);
        } else {
          mbar_arrive_expect_tx(&afull[s], kAStageBytes);
          tma_load_2d(a_dst, &tmA, &afull[s], kc, static_cast<int32_t>(row0));
        }
        issued = it + 1;
      }
      if (*abort_flag) {
        // Let every issued copy land before the CTA's shared memory goes away.
        for (int it = (issued > kStages ? issued - kStages : 0); it < issued; ++it)
          mbar_drain(&afull[it % kStages], static_cast<uint32_t>(it / kStages) & 1u);
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(kBM, kBN, MODE == MODE_SGRAD ? 1 : 0, MODE == MODE_FWD ? 0 : 1);
      bool ok = true;
      for (int it = 0; it < num_k && ok; ++it) {
        const int s = it % kStages;
        const uint32_t ph = static_cast<uint32_t>(it / kStages) & 1u;
        ok = mbar_wait(&afull[s], ph, abort_flag, p.err);
        if (ok && MODE != MODE_SGRAD) ok = mbar_wait(&bfull[s], ph, abort_flag, p.err);
        if (!ok) break;
        tc_fence_after();
        const uint32_t a_base = smem_u32(sA + s * kAStageBytes);
        const uint32_t b_base = smem_u32(sB + s * kBStageBytes);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          uint64_t ad, bd;
          if (MODE == MODE_SGRAD) {
            ad = smem_desc_sw128(a_base + kk * 2048, kBK * 128, 1024);
          } else {
            ad = smem_desc_sw128(a_base + kk * 32, 16, 1024);
          }
          if (MODE == MODE_FWD) {
            bd = smem_desc_sw128(b_base + kk * 32, 16, 1024);
          } else {
            bd = smem_desc_sw128(b_base + kk * 2048, kBK * 128, 1024);
          }
          umma_bf16(tmem_base, ad, bd, idesc, (it > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&empty[s]);
      }
      if (ok) {
        umma_commit(tfull);
      } else {
        umma_commit(drain);  // completes once every MMA issued so far has finished
        mbar_drain(drain, 0);
      }
    }
  } else {
    // ------------------------------------------------------ decode (warps 0-3)
    if (MODE != MODE_SGRAD) {
      const int t = threadIdx.x;  // 0..127
      const int64_t K2 = p.K / 2;
      const int64_t G = p.K / B;
      // 512 units of 32 consecutive weight elements per stage, 4 per thread.
      uint4 cw[4], cn[4];
      uint32_t sw[4], sn[4];
      auto load_units = [&](int it, uint4 (&c)[4], uint32_t (&sc)[4]) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int u = t + 128 * i;
          int64_t n, k;
          if (MODE == MODE_FWD) {  // tile rows = out features n, cols = k (K-major)
            n = col0 + (u >> 1);
            k = static_cast<int64_t>(it) * kBK + 32 * (u & 1);
          } else {  // tile rows = contraction n (MN-major), cols = 256 k-values
            const int j = (u & 7) + 8 * (u >> 6);
            const int part = (u >> 3) & 7;
            n = static_cast<int64_t>(it) * kBK + j;
            k = col0 + 32 * part;
          }
          if (n < p.N && k < p.K) {
            c[i] = __ldg(reinterpret_cast<const uint4 *>(p.codes + n * K2 + k / 2));
            if (FMT == 0)
              sc[i] = __ldg(reinterpret_cast<const unsigned short *>(p.scales + n * G + k / 16));
            else
              sc[i] = __ldg(p.scales + n * G + k / 32);
          } else {
            c[i] = make_uint4(0u, 0u, 0u, 0u);
            sc[i] = FMT == 0 ? 0x3838u : 127u;  // any finite scale; the codes are zero
          }
        }
      };
      if (num_k > 0) load_units(0, cw, sw);
      for (int it = 0; it < num_k; ++it) {
        const int s = it % kStages;
        const uint32_t use = static_cast<uint32_t>(it / kStages);
        if (it + 1 < num_k) load_units(it + 1, cn, sn);
        if (it >= kStages && !mbar_wait(&empty[s], (use & 1u) ^ 1u, abort_flag, p.err)) break;
        const uint32_t b_base = smem_u32(sB + s * kBStageBytes);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int u = t + 128 * i;
          uint32_t sc_lo, sc_hi;
          if (FMT == 0) {
            sc_lo = scale_bf16x2<0>(sw[i] & 0xFFu);
            sc_hi = scale_bf16x2<0>(sw[i] >> 8);
          } else {
            sc_lo = sc_hi = scale_bf16x2<1>(sw[i]);
          }
          const uint32_t words[4] = {cw[i].x, cw[i].y, cw[i].z, cw[i].w};
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            uint32_t o[4];
            e2m1x8_to_bf16(words[c], o);
            const uint32_t sc = c < 2 ? sc_lo : sc_hi;
#pragma unroll
            for (int q = 0; q < 4; ++q) o[q] = bf16x2_mul(o[q], sc);
            uint32_t addr;
            if (MODE == MODE_FWD) {
              const int r = u >> 1;
              const int chunk = 4 * (u & 1) + c;
              addr = b_base + (r >> 3) * 1024 + (r & 7) * 128 + ((chunk ^ (r & 7)) << 4);
            } else {
              const int j = (u & 7) + 8 * (u >> 6);
              const int part = (u >> 3) & 7;
              const int atom = part >> 1;
              const int chunk = 4 * (part & 1) + c;
              addr = b_base + atom * (kBK * 128) + j * 128 + ((chunk ^ (j & 7)) << 4);
            }
            st_shared_v4(addr, o[0], o[1], o[2], o[3]);
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bfull[s]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          cw[i] = cn[i];
          sw[i] = sn[i];
        }
      }
    }

    // ------------------------------------------------------ epilogue (warps 0-3)
    const bool ok = num_k > 0 && mbar_wait(tfull, 0, abort_flag, p.err);
    tc_fence_after();
    const int r = warp * 32 + lane;
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(warp * 32) << 16);
    if (MODE != MODE_SGRAD) {
      const int64_t grow = row0 + r;
      const float scale = FMT == 0 ? p.ws2 : 1.0f;
      __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
      for (int c0 = 0; c0 < kBN; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(t_row + c0, v);
        tmem_ld_wait();
        if (!ok || grow >= Mg) continue;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int64_t gc = col0 + c0 + 8 * q;
          if (gc >= Ng) continue;
          uint32_t packed[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float a = __uint_as_float(v[8 * q + 2 * e]) * scale;
            const float b = __uint_as_float(v[8 * q + 2 * e + 1]) * scale;
            const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
            packed[e] = *reinterpret_cast<const uint32_t *>(&h);
          }
          *reinterpret_cast<uint4 *>(out + grow * Ng + gc) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
        }
      }
    } else {
      const int64_t n = row0 + r;
      const int64_t G = p.K / B;
      float *g = static_cast<float *>(p.out);
      for (int c0 = 0; c0 < kBN; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(t_row + c0, v);
        tmem_ld_wait();
        const int64_t k = col0 + c0;
        if (!ok || n >= p.N || k >= p.K) continue;
        const uint4 cw = __ldg(reinterpret_cast<const uint4 *>(p.codes + n * (p.K / 2) + k / 2));
        const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
        float part[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t o[4];
          e2m1x8_to_bf16(words[c], o);
          float acc = 0.f;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            acc = fmaf(__uint_as_float(o[e] << 16), __uint_as_float(v[8 * c + 2 * e]), acc);
            acc = fmaf(__uint_as_float(o[e] & 0xFFFF0000u), __uint_as_float(v[8 * c + 2 * e + 1]), acc);
          }
          part[c] = acc;
        }
        if (FMT == 0) {
          const int64_t b = k / 16;
          float g0 = part[0] + part[1];
          float g1 = part[2] + part[3];
          if (p.mask) {
            g0 *= static_cast<float>(p.mask[n * G + b]);
            g1 *= static_cast<float>(p.mask[n * G + b + 1]);
          }
          *reinterpret_cast<float2 *>(g + n * G + b) = make_float2(g0, g1);
        } else {
          const int64_t b = k / 32;
          float g0 = (part[0] + part[1]) + (part[2] + part[3]);
          if (p.mask) g0 *= static_cast<float>(p.mask[n * G + b]);
          g[n * G + b] = g0;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

template <int MODE, int FMT>
cudaError_t launch_one(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB, cudaStream_t stream) {
  static bool attr_done = false;  // per process; the attribute is per function
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(sq_gemm_kernel<MODE, FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int64_t Mg = MODE == MODE_SGRAD ? a.N : a.M;
  const int64_t Ng = MODE == MODE_FWD ? a.N : a.K;
  dim3 grid(static_cast<unsigned>((Mg + kBM - 1) / kBM), static_cast<unsigned>((Ng + kBN - 1) / kBN));
  KParams p{a.codes, a.scales, a.ws2, a.M, a.N, a.K, a.out, a.mask, a.err};
  sq_gemm_kernel<MODE, FMT><<<grid, kThreads, kSmemBytes, stream>>>(tmA, tmB, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm(const GemmArgs &a, const CUtensorMap &tmA, const CUtensorMap &tmB, int sm_count,
                        cudaStream_t stream) {
  (void)sm_count;
  if (a.fmt == 0) {
    if (a.mode == MODE_FWD) return launch_one<MODE_FWD, 0>(a, tmA, tmB, stream);
    if (a.mode == MODE_DX) return launch_one<MODE_DX, 0>(a, tmA, tmB, stream);
    return launch_one<MODE_SGRAD, 0>(a, tmA, tmB, stream);
  }
  if (a.mode == MODE_FWD) return launch_one<MODE_FWD, 1>(a, tmA, tmB, stream);
  if (a.mode == MODE_DX) return launch_one<MODE_DX, 1>(a, tmA, tmB, stream);
  return launch_one<MODE_SGRAD, 1>(a, tmA, tmB, stream);
}

}  // namespace sqi
