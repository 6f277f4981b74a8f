// tcgen05 contraction kernels of the scale-only training step (sm_103a),
// shared by the dense launches (sq_gemm.cu) and the grouped expert launches
// (sq_grouped.cu); each translation unit instantiates only what it launches.
//
//   MODE_FWD   Y[m,n]  = sum_k X[m,k] W[n,k]        Sec. 3 "Scale-QLoRA forward"
//   MODE_DX    dX[m,k] = sum_n dY[m,n] W[n,k]       its input gradient
//   MODE_SGRAD g[n,b]  = sum_{k in b} code[n,k] sum_m dY[m,n] X[m,k]   its scale gradient
//
// with W[n,k] = code[n,k] * s[n, k/B] (Sec. 2). All kernels are persistent
// (one CTA per SM, tiles walked in an L2-friendly grouped order) and keep two
// 256-column fp32 accumulators in tensor memory (TMEM), so the epilogue of one
// tile overlaps the mainloop of the next.
//
// FWD / DX (sq_gemm_pair_kernel): a cluster of two CTAs computes a 512 x 256
// tile with tcgen05.mma.cta_group::2, as two 256-row halves that share every
// decoded weight stage. Each CTA streams 128 activation rows of each half and
// its half of the packed-code tile by TMA, and 16 decode warps turn nibbles and
// scale bytes into the bf16 weight operand directly in the 128B-swizzled
// shared-memory layout the tensor core reads (K-major for FWD, MN-major for DX).
//
// SGRAD (sq_sgrad_pair_kernel): a cluster of two CTAs per 256 x 256 tile of
// dW = dY^T X with both operands as MN-major TMA tiles; each CTA's epilogue
// reduces code x dW per block for its 128 rows. A dense launch with few tiles
// may cut the tokens into parts (KParams::splits): each (part, tile) unit writes
// a partial plane, which sq_split_reduce_kernel (sq_gemm.cu) adds in order.
//
// Every mbarrier wait is bounded (kWaitLimitNs): on expiry the CTA records
// kErrWaitTimeout in the device error word, stops issuing, drains what it has
// in flight and frees its TMEM.
//
// Grouped launches (template flag GR) run one contraction per expert of a
// mixture-of-experts layer in a single persistent launch: the tiles of all
// experts form one list, and a device table built by the host per call gives
// each expert its TMA descriptors (addressing only that expert's token rows, so
// rows of other experts read as zero and are never written), its token count
// and its tensor scale.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "sq_internal.h"

namespace sqi {
namespace {

constexpr uint32_t kTmemCols = 256;          // one accumulator buffer (two are allocated)
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

// Non-suspending variants for the threads on the critical path of the pair
// kernel (MMA issue, gate): mbarrier.try_wait may suspend the thread, and a
// suspended thread resumes a few hundred cycles after the phase completes;
// test_wait returns at once, so these spin (with the same time limit).
__device__ __forceinline__ bool mbar_test_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_test_wait_cluster(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

template <bool CLUSTER>
__device__ __noinline__ bool mbar_spin_slow(uint64_t *bar, uint32_t parity, volatile int *abort_flag, int *err) {
  const unsigned long long t0 = globaltimer();
  while (true) {
    for (int i = 0; i < 256; ++i)
      if (CLUSTER ? mbar_test_wait_cluster(bar, parity) : mbar_test_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) {
      *abort_flag = 1;
      atomicOr(err, kErrWaitTimeout);
      return false;
    }
  }
}

__device__ __forceinline__ bool mbar_spin(uint64_t *bar, uint32_t parity, volatile int *abort_flag, int *err) {
  return mbar_test_wait(bar, parity) || mbar_spin_slow<false>(bar, parity, abort_flag, err);
}

__device__ __forceinline__ bool mbar_spin_cluster(uint64_t *bar, uint32_t parity, volatile int *abort_flag,
                                                  int *err) {
  return mbar_test_wait_cluster(bar, parity) || mbar_spin_slow<true>(bar, parity, abort_flag, err);
}

// Bounded wait used only while tearing down after an abort: waits for work this
// CTA already put in flight (TMA copies, MMAs), ignoring the abort flag.
__device__ __noinline__ void mbar_drain(uint64_t *bar, uint32_t parity) {
  const unsigned long long t0 = globaltimer();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer() - t0 > kWaitLimitNs) return;
}

// The same bounded wait with cluster-scope acquire, for barriers that threads of
// the peer CTA arrive on with cluster-scope release.
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __noinline__ bool mbar_wait_cluster(uint64_t *bar, uint32_t parity, volatile int *abort_flag, int *err) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  while (true) {
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait_cluster(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer() - t0 > kWaitLimitNs) {
      *abort_flag = 1;
      atomicOr(err, kErrWaitTimeout);
      return false;
    }
  }
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
// significant bits, E8M0 is a power of two). E4M3: the 7 magnitude bits placed
// at fp32 bit 20 read as E4M3(byte) * 2^-120 for normal and subnormal bytes
// alike, so one multiply by 2^120 gives the value; byte 0x7F / 0xFF is NaN.
template <int FMT>
__device__ __forceinline__ uint32_t scale_bf16x2(uint32_t byte) {
  uint32_t u;
  if (FMT == 0) {
    const uint32_t mag = byte & 0x7Fu;
    const float f = __uint_as_float(mag << 20) * 0x1p120f;
    u = (__float_as_uint(f) >> 16) | ((byte & 0x80u) << 8);
    if (mag == 0x7Fu) u = 0x7FC0u;
  } else {
    u = byte == 0 ? 0x0040u : (byte == 255 ? 0x7FC0u : (byte << 7));
  }
  return u | (u << 16);
}

// ------------------------------------------------------------- shared pieces

// Weight formats of the contraction kernels: NVFP4 (0) and MXFP4 (1) codes with
// block scales, and the full-precision multiplicative control of the ablation
// appendix (2): bf16 weights W times fl32(1 + dS) per (row, block of 16).
constexpr int kFmtBf16Mul = 2;

struct KParams {
  const uint8_t *codes;
  const uint8_t *scales;
  float ws2;
  int64_t M, N, K;
  void *out;
  const uint8_t *mask;
  int *err;
  int tiles_m, tiles_n;  // dense: the tile grid; grouped: tiles_n is the column tiles of every expert
  int total;             // tiles of the launch
  const uint8_t *gtab;   // grouped: the device expert table (GroupMaps[E], tile_start, rows, ws2); else null
  int groups;            // experts of a grouped launch, 1 for a dense one
  int splits = 1;            // dense scale gradient: token splits (total = tiles x splits units)
  float *partial = nullptr;  // ... with splits > 1: [splits, N, G] partial planes (no mask)
};

// Tuning constants of the decode warps (compile-time; the defaults are the measured best).
#ifndef SQ_EPI_HOLD_GR
#define SQ_EPI_HOLD_GR 2  // 32-column groups a grouped epilogue stores after releasing the accumulator
#endif
#ifndef SQ_SCALE_DEPTH
#define SQ_SCALE_DEPTH 4      // scale bytes are loaded this many of a group's k-steps ahead
#endif

// Persistent tile order: tiles are walked in groups of GROUP row-tiles, the
// column index varying slowest inside a group, so the CTAs resident at any
// moment share a few row panels and column panels in L2. For the 512 x 256 pair
// tiles, 2: a wave of 76 tiles then holds ~5 streamed activation panels with all
// their column tiles, each panel leaves DRAM once, and the decoded weight's column
// panels are what recurs from wave to wave (measured on the 8B layer's shapes at
// M = 32768: 0.98-1.62x the algorithmic DRAM bytes against 1.16-2.40x for 8, and
// 1 % faster per layer step). For the scale-gradient tiles, 16.
constexpr int kGroup = 2;
constexpr int kSgradGroup = 16;

template <int GROUP = kGroup>
__device__ __forceinline__ void tile_coords(int id, int tiles_m, int tiles_n, int &tm, int &tn) {
  const int per_group = GROUP * tiles_n;
  const int g = id / per_group;
  const int first = g * GROUP;
  const int gm = min(GROUP, tiles_m - first);
  const int local = id - g * per_group;
  tm = first + local % gm;
  tn = local / gm;
}

// A TMA descriptor that lives in global memory (the expert table) is read by the
// tensor-map proxy; this orders the table's earlier generic-proxy writes before
// the descriptor fetch of the copies this thread issues with it.
__device__ __forceinline__ void tensormap_acquire(const CUtensorMap *map) {
  asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(reinterpret_cast<uint64_t>(map))
               : "memory");
}

__device__ __forceinline__ const GroupMaps *group_maps(const KParams &p, int e) {
  return reinterpret_cast<const GroupMaps *>(p.gtab) + e;
}
__device__ __forceinline__ int group_rows(const KParams &p, int e) {
  return __ldg(reinterpret_cast<const int *>(p.gtab + group_off_rows(p.groups)) + e);
}
__device__ __forceinline__ int group_id(const KParams &p, int e) {
  return __ldg(reinterpret_cast<const int *>(p.gtab + group_off_ids(p.groups)) + e);
}
__device__ __forceinline__ float group_ws2(const KParams &p, int e) {
  return __ldg(reinterpret_cast<const float *>(p.gtab + group_off_ws2(p.groups)) + e);
}

// Tile `tile` of a launch -> expert e, row tile tm, column tile tn. A dense launch
// is one expert. A grouped launch lists the tiles expert by expert (tile_start[e]
// up to tile_start[e + 1]: rows tiles of the expert x tiles_n), each expert's in
// the grouped order of tile_coords. Every role walks its tiles in increasing
// order, so the caller keeps e between calls and it only moves forward; experts
// without tiles are stepped over.
template <bool GR, int GROUP = kGroup>
__device__ __forceinline__ void resolve_tile(const KParams &p, int tile, int &e, int &tm, int &tn) {
  if (!GR) {
    e = 0;
    tile_coords<GROUP>(tile, p.tiles_m, p.tiles_n, tm, tn);
    return;
  }
  const int *ts = reinterpret_cast<const int *>(p.gtab + group_off_tiles(p.groups));
  while (e + 1 < p.groups && __ldg(ts + e + 1) <= tile) ++e;
  const int first = __ldg(ts + e);
  tile_coords<GROUP>(tile - first, (__ldg(ts + e + 1) - first) / p.tiles_n, p.tiles_n, tm, tn);
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

// Scale byte(s) covering the 32 weights of one decode unit of the weight whose
// scale plane starts at `scales`: two E4M3 bytes (blocks of 16) or one E8M0 byte.
// Units outside the weight read scale 0, so their decoded weights are zero
// whatever codes the tile holds there (TMA zero fill past the last row, or the
// next expert's rows in a grouped launch).
template <int FMT>
__device__ __forceinline__ uint32_t load_unit_scale(const KParams &p, const uint8_t *scales, int64_t n, int64_t k) {
  if (n >= p.N || k >= p.K) return 0u;
  const int64_t G = p.K / (FMT == 0 ? 16 : 32);
  if (FMT == 0) return __ldg(reinterpret_cast<const unsigned short *>(scales + n * G + k / 16));
  return __ldg(scales + n * G + k / 32);
}

// ------------------------------------------------------------- scale-gradient kernel
//
// D[n, k] = sum_m dY[m, n] X[m, k], contraction over the tokens: both operands
// are MN-major TMA tiles (64 features x kSgradBK tokens per box). The epilogue
// multiplies each dW element by its E2M1 code and sums every block of B columns,
// applies the STE mask and writes g[n, b]; the dW tile never leaves the SM.

// ------------------------------------------------------------- CTA-pair kernels
//
// Two CTAs of a cluster share one output tile through tcgen05.mma.cta_group::2
// (M = 256, N = 256): each CTA holds 128 rows of the A operand and half (128
// columns) of the B operand; the leader CTA (cluster rank 0) issues the MMAs and
// multicasts each commit to the barriers of both CTAs. Each CTA keeps the
// accumulator of its 128 rows in its own TMEM and runs its own epilogue.

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Shared-memory address of the same variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

// Asynchronous 4-byte store into another CTA's shared memory that completes 4
// bytes of transaction on that CTA's mbarrier; the complete-tx has release
// semantics at cluster scope and the issuing thread does not wait for it.
__device__ __forceinline__ void st_async_signal(uint32_t cluster_dst, uint32_t cluster_bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.u32 [%0], %1, [%2];" ::"r"(cluster_dst), "r"(1u),
               "r"(cluster_bar)
               : "memory");
}



// TMEM allocation for a CTA pair: one warp of each CTA executes these collectively.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t *slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on `bar` in both CTAs of the pair when the pair's MMAs issued so far complete.
__device__ __forceinline__ void umma_commit_pair_mc(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          smem_u32(bar)),
      "h"(static_cast<unsigned short>(3))
      : "memory");
}

__device__ __forceinline__ void umma_commit_pair(uint64_t *bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// TMA store of one box from this CTA's shared memory, tracked by the thread's bulk groups.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, uint32_t src, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}

__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

// Wait until at most N of this thread's bulk groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

// Wait until all of this thread's bulk groups have completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// TMA load into this CTA's shared memory whose complete-tx lands on an mbarrier
// of either CTA of the pair (`bar_cluster` is a shared::cluster address): the
// activation tiles of both CTAs are counted on the leader's barrier.
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster, int32_t x,
                                                 int32_t y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
      : "memory");
}

// Shared-memory rings of the pair kernel, each advancing on its own:
//   activations     kAStages slots of 128 rows x one 128-deep stage (32 KiB): a
//                   k-step loads two of them, one per 256-row half of the tile;
//   decoded weights kStages slots of this CTA's 128 weight rows x one stage (32 KiB);
//   packed codes    kCStages slots (8 KiB), released by the decode warps once read;
//   output staging  one 2 KiB box (32 rows x 32 columns) per epilogue warp for the
//                   TMA stores of the result.
// A pair computes a 512 x 256 output tile: every decoded weight stage feeds the
// MMAs of both 256-row halves, into two TMEM accumulators (all 512 columns), so
// the decode-and-signal chain of a stage is covered by twice the tensor work. The
// next tile's MMAs wait for the epilogue to drain both accumulators; eight
// epilogue warps (two per TMEM lane quadrant, one per column half) shorten that
// wait.
struct PairCfg {
  // Roles are numbered 0-27 as below; role_of() places them on the physical warps.
  static constexpr int kEpiWarps = 8;    // roles 0-7: warp w drains lane quadrant w % 4, column half w / 4
  static constexpr int kDecWarps = 16;   // roles 8-23: one 32-weight unit per thread per stage
  static constexpr int kTmaWarp = kEpiWarps + kDecWarps;  // activation tiles
  static constexpr int kCodeWarp = kTmaWarp + 1;          // packed-code tiles
  static constexpr int kMmaWarp = kCodeWarp + 1;
  static constexpr int kGateWarp = kMmaWarp + 1;  // leader: hands each k-step to the MMA thread
  static constexpr int kThreads = 32 * (kGateWarp + 1);
  static constexpr int kBK = 128;        // contraction depth of a stage: 8 MMAs of K = 16 per tile half
  static constexpr int kAStages = 4;     // activation slots (two per k-step)
  static constexpr int kStages = 2;      // decoded-weight slots (a k-step feeds 16 MMAs)
  static constexpr int kCStages = 2;     // code slots (a k-step lasts >= 2048 tensor cycles)
  static constexpr int kA = 128 * kBK * 2;  // 32 KiB: this CTA's 128 rows of one tile half, two 64-wide K chunks
  static constexpr int kB = 128 * kBK * 2;  // 32 KiB: this CTA's half of the decoded weight tile
  static constexpr int kC = 128 * kBK / 2;  // 8 KiB: packed codes of that half (64-byte rows, 64-byte swizzle)
  static constexpr int kOffB = kAStages * kA;
  static constexpr int kOffC = kOffB + kStages * kB;
  static constexpr int kOffS = kOffC + kCStages * kC;   // output staging: [kEpiWarps][32 x 32 bf16]
  static constexpr int kBoxBytes = 32 * 32 * 2;
  static constexpr int kOffBar = kOffS + kEpiWarps * kBoxBytes;
  static constexpr int kSmemBytes = kOffBar + 1024 + 1024;
  static constexpr uint32_t kATx = 2 * kA;                      // both CTAs' activation tiles, on the leader
  static constexpr uint32_t kSignalBytes = 4 * kDecWarps * 2;   // st.async bytes per stage: all decode warps, 2 CTAs
  static constexpr int kTile = kPairNTile;   // output columns of a pair tile (and rows of one half)
  static constexpr int kMTile = kPairMTile;  // output rows of a pair tile: two halves of kTile
};
static_assert(PairCfg::kSmemBytes <= 232448, "pair kernel exceeds the opt-in shared memory of one CTA");
static_assert(PairCfg::kMTile == 2 * PairCfg::kTile, "a pair tile is two halves");
static_assert(PairCfg::kAStages == 2 * PairCfg::kStages, "half 1's activation slots are released with the decoded slots");
static_assert(PairCfg::kEpiWarps == 8, "the epilogue maps warp w to lane quadrant w % 4 and column half w / 4");

// Role of physical warp pw. Warp pw issues from scheduler pw % 4, and a
// tcgen05.mma holds the MMA thread until the tensor core takes it, so every cycle
// that thread waits for an issue slot can idle the tensor core. The MMA warp
// (physical 26) therefore shares its scheduler with the two TMA warps (physical 18
// and 22, mostly asleep on barriers), two epilogue warps and only two decode warps;
// the decode roles fill physical 8-17, 19-21 and 23-25 and the gate stays on 27.
// Measured against the plain numbering (the MMA warp beside four decode warps):
// the MMA thread's 8 MMAs of a tile half issued in ~750 instead of ~1,030 cycles.
// The epilogue roles keep their warps: TMEM lane quadrant access is by warp % 4.
__device__ __forceinline__ int pair_role_of(int pw) {
  switch (pw) {
    case 18: return PairCfg::kCodeWarp;
    case 22: return PairCfg::kTmaWarp;
    case 19: return 18;
    case 20: return 19;
    case 21: return 20;
    case 23: return 21;
    case 24: return 22;
    case 25: return 23;
    default: return pw;
  }
}
static_assert(PairCfg::kTmaWarp == 24 && PairCfg::kCodeWarp == 25 && PairCfg::kMmaWarp == 26 &&
                  PairCfg::kGateWarp == 27,
              "pair_role_of places these roles");

// Decode unit u (0..511) of this CTA's half at stage kb covers 32 consecutive
// weights: row (u & 7) + 8 * (u >> 5) of the half, quarter (u >> 3) & 3 of its
// 128 columns (k for FWD, k-columns of the MN-major tile for DX), so the 8
// lanes that share a shared-memory wavefront always touch 8 different rows.
template <int MODE>
__device__ __forceinline__ void pair_unit_coords(int u, int64_t half0, int kb, int64_t &n, int64_t &k) {
  const int row = (u & 7) + 8 * (u >> 5), quarter = (u >> 3) & 3;
  if (MODE == MODE_FWD) {  // 128 out-feature rows x 128 k
    n = half0 + row;
    k = static_cast<int64_t>(kb) * PairCfg::kBK + 32 * quarter;
  } else {  // 128 contraction rows x 128 k-columns
    n = static_cast<int64_t>(kb) * PairCfg::kBK + row;
    k = half0 + 32 * quarter;
  }
}

template <int MODE, int FMT, bool GR>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairCfg::kThreads, 1)
    sq_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmC,
                        const __grid_constant__ CUtensorMap tmO, const KParams p) {
  using C = PairCfg;
  constexpr int SA = C::kAStages;
  constexpr int S = C::kStages;
  constexpr int SC = C::kCStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + C::kOffBar);
  uint64_t *afull = bars;             // [SA] leader: both CTAs' activation tiles landed (1 arrival + 2 x kA tx)
  uint64_t *aempty = afull + SA;      // [SA] pair MMAs reading half 0's slot a done     (multicast commit)
  uint64_t *empty = aempty + SA;      // [S] pair MMAs of k-step s done: decoded slot s and
                                      //     half 1's activation slot free      (multicast commit)
  uint64_t *pready = empty + S;       // [S] leader: both weight halves decoded          (1 arrival + st.async tx)
  uint64_t *gready = pready + S;      // [S] leader: pready and half 0's afull seen by the gate (1 arrival)
  uint64_t *cfull = gready + S;       // [SC] this CTA's code tile landed                 (1 arrival + tx)
  uint64_t *cempty = cfull + SC;      // [SC] this CTA's decode warps read the codes      (kDecWarps arrivals)
  uint64_t *tfull = cempty + SC;      // [2] accumulator h of the tile complete          (multicast commit)
  uint64_t *tempty = tfull + 2;       // [2] leader: both epilogues drained accumulator h
                                      //     (kEpiWarps arrivals + the peer warps' st.async tx)
  uint64_t *drain = tempty + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  uint32_t *sink = reinterpret_cast<uint32_t *>(drain + 2);  // leader: st.async targets, [2][kDecWarps] + [kEpiWarps]

  const int warp = pair_role_of(threadIdx.x >> 5);  // this warp's role
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int cluster = blockIdx.x >> 1;
  const int nclusters = gridDim.x >> 1;
  const int total = p.total;
  const int64_t Kg = MODE == MODE_FWD ? p.K : p.N;
  const int num_k = static_cast<int>((Kg + C::kBK - 1) / C::kBK);
  const int my_tiles = cluster < total ? (total - cluster + nclusters - 1) / nclusters : 0;

  auto ring_a = [&](int a) { return smem + a * C::kA; };
  auto ring_b = [&](int s) { return smem + C::kOffB + s * C::kB; };
  auto ring_c = [&](int c) { return smem + C::kOffC + c * C::kC; };

  if (threadIdx.x == 0) {
    for (int a = 0; a < SA; ++a) {
      mbar_init(&afull[a], 1);
      mbar_init(&aempty[a], 1);
    }
    for (int s = 0; s < S; ++s) {
      mbar_init(&empty[s], 1);
      mbar_init(&pready[s], 1);
      mbar_init(&gready[s], 1);
    }
    for (int c = 0; c < SC; ++c) {
      mbar_init(&cfull[c], 1);
      mbar_init(&cempty[c], C::kDecWarps);
    }
    for (int h = 0; h < 2; ++h) {
      mbar_init(&tfull[h], 1);
      mbar_init(&tempty[h], C::kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == C::kMmaWarp) tmem_alloc_pair(tmem_slot, 2 * kTmemCols);
  if (warp == C::kTmaWarp && lane == 0) {
    if (!GR) tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmC);
    if (!GR) tma_prefetch_desc(&tmO);
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == C::kTmaWarp) {
    // ------------------------------------------------------ activation TMA (both CTAs)
    // Per k-step, one slot per tile half: each CTA loads its own 128 rows of the
    // half; both loads complete on the leader's afull, which the leader arms with
    // the bytes of the two.
    if (lane == 0) {
      int ja = 0;  // activation slots filled
      bool ok = true;
      int e = 0, e_seen = -1;
      const CUtensorMap *mA = &tmA;
      for (int tile = cluster; tile < total && ok; tile += nclusters) {
        int tm, tn;
        resolve_tile<GR>(p, tile, e, tm, tn);
        if (GR && e != e_seen) {  // the expert's own activation rows
          mA = &group_maps(p, e)->m[0];
          tensormap_acquire(mA);
          e_seen = e;
        }
        const int32_t row0 = tm * C::kMTile + 128 * static_cast<int32_t>(rank);
        for (int kb = 0; kb < num_k && ok; ++kb) {
          for (int h = 0; h < 2; ++h, ++ja) {
            const int a = ja % SA;
            const uint32_t use = static_cast<uint32_t>(ja / SA);
            // half 0's slot is freed by the commit after its 8 MMAs; half 1's together
            // with the decoded slot, by the commit that ends k-step ja / 2 - S
            if (ja >= SA && !(ok = h == 0 ? mbar_wait(&aempty[a], (use & 1u) ^ 1u, abort_flag, p.err)
                                          : mbar_wait(&empty[(ja / 2) % S],
                                                      (static_cast<uint32_t>(ja / 2 / S) & 1u) ^ 1u, abort_flag, p.err)))
              break;
            if (rank == 0) mbar_arrive_expect_tx(&afull[a], C::kATx);
            const uint32_t bar = mapa_shared(smem_u32(&afull[a]), 0);
            // two 128 x 64 boxes (one per 64-wide K chunk, 16 KiB apart)
            for (int j = 0; j < C::kBK / 64; ++j)
              tma_load_2d_pair(smem_u32(ring_a(a)) + j * 16384, mA, bar, kb * C::kBK + 64 * j, row0 + C::kTile * h);
          }
        }
      }
      if (*abort_flag && rank == 0) {
        for (int i = (ja > SA ? ja - SA : 0); i < ja; ++i)
          mbar_drain(&afull[i % SA], static_cast<uint32_t>(i / SA) & 1u);
      }
    }
  } else if (FMT == kFmtBf16Mul && warp == C::kCodeWarp) {
    // ------------------------------------------------------ bf16 weight TMA (both CTAs)
    // The multiplicative control: this CTA's half of the bf16 weight tile goes
    // straight into the decoded-weight slot (two 64-wide boxes, 128-byte swizzle:
    // the layout the MMAs read), once the MMAs of the slot's previous use are done;
    // the decode warps then scale it in place. cfull[s] counts its bytes.
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      int e = 0;
      for (int tile = cluster; tile < total && ok; tile += nclusters) {
        int tm, tn;
        resolve_tile<GR>(p, tile, e, tm, tn);
        const int32_t half0 = tn * C::kTile + 128 * static_cast<int32_t>(rank);
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int s = it % S;
          const uint32_t use = static_cast<uint32_t>(it / S);
          if (it >= S && !(ok = mbar_wait(&empty[s], (use & 1u) ^ 1u, abort_flag, p.err))) break;
          mbar_arrive_expect_tx(&cfull[s], C::kB);
          for (int j = 0; j < 2; ++j) {
            if (MODE == MODE_FWD)  // 128 weight rows (out features) x 64 k
              tma_load_2d(smem_u32(ring_b(s)) + j * 16384, &tmC, &cfull[s], kb * C::kBK + 64 * j, half0);
            else                   // 128 contraction rows x 64 k-columns
              tma_load_2d(smem_u32(ring_b(s)) + j * 16384, &tmC, &cfull[s], half0 + 64 * j, kb * C::kBK);
          }
        }
      }
      if (*abort_flag) {
        for (int i = (it > S ? it - S : 0); i < it; ++i) mbar_drain(&cfull[i % S], static_cast<uint32_t>(i / S) & 1u);
      }
    }
  } else if (warp == C::kCodeWarp) {
    // ------------------------------------------------------ code TMA (both CTAs)
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      int e = 0;
      for (int tile = cluster; tile < total && ok; tile += nclusters) {
        int tm, tn;
        resolve_tile<GR>(p, tile, e, tm, tn);
        const int32_t half0 = tn * C::kTile + 128 * static_cast<int32_t>(rank);
        const int32_t erow = GR ? e * static_cast<int32_t>(p.N) : 0;  // the expert's first row of the code tensor
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int c = it % SC;
          const uint32_t use = static_cast<uint32_t>(it / SC);
          if (it >= SC && !(ok = mbar_wait(&cempty[c], (use & 1u) ^ 1u, abort_flag, p.err))) break;
          mbar_arrive_expect_tx(&cfull[c], C::kC);
          if (MODE == MODE_FWD)  // 128 rows x 64 bytes at (byte k/2, row n)
            tma_load_2d(smem_u32(ring_c(c)), &tmC, &cfull[c], kb * (C::kBK / 2), erow + half0);
          else                   // 128 contraction rows x 64 bytes
            tma_load_2d(smem_u32(ring_c(c)), &tmC, &cfull[c], half0 / 2, erow + kb * C::kBK);
        }
      }
      if (*abort_flag) {
        for (int i = (it > SC ? it - SC : 0); i < it; ++i)
          mbar_drain(&cfull[i % SC], static_cast<uint32_t>(i / SC) & 1u);
      }
    }
  } else if (warp == C::kMmaWarp) {
    // ------------------------------------------------------ MMA issuer (leader CTA)
    // A k-step needs both decoded weight halves and the activation tiles of both
    // halves. The gate warp folds the decoded halves and half 0's activations into
    // one barrier (gready); half 1's activations, whose slot is refilled last, are
    // checked here just before half 1's MMAs, which gives their loads half a k-step
    // more time. Every barrier wait and every commit of this thread costs issue time
    // the tensor core cannot hide, so it waits spinning (test_wait), polls nothing
    // between MMAs and commits twice: half 0's activation slot after its 8 MMAs (the
    // TMA warp refills it a half step early) and, after all 16, the decoded slot
    // together with half 1's activation slot.
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16(2 * 128, C::kTile, 0, MODE == MODE_FWD ? 0 : 1);
      // slot s of a ring starts s slot sizes after slot 0 (the start address field is >> 4).
      // K-major tiles: K step kk lives in 64-wide chunk kk / 4 (16 KiB apart) at byte 32 * (kk % 4) of
      // each 128-byte row; the MN-major DX tile: 16 contraction rows (2 KiB) per step, MN atoms 16 KiB apart.
      const uint64_t ad_base = smem_desc_sw128(smem_u32(ring_a(0)), 16, 1024);
      const uint64_t bd_base = MODE == MODE_FWD ? smem_desc_sw128(smem_u32(ring_b(0)), 16, 1024)
                                                : smem_desc_sw128(smem_u32(ring_b(0)), 16384, 1024);
      int s = 0, a = 0;             // decoded slot of the current k-step, activation slot of its first half
      uint32_t ph = 0;              // phase parity of the decoded slot
      int tc = 0, it = 0;           // tiles and k-steps of this cluster so far
      int e_mma = 0;
      bool ok = true;
      for (int tile = cluster; tile < total && ok; tile += nclusters, ++tc) {
        // A grouped tile whose half 1 lies wholly past its expert's last row skips that
        // half's MMAs; every wait and commit stays, so the rings keep their phases and
        // the epilogue (which does not store those rows) still sees accumulator 1 commit.
        bool skip1 = false;
        if (GR) {
          int tm, tn;
          resolve_tile<GR>(p, tile, e_mma, tm, tn);
          skip1 = tm * C::kMTile + C::kTile >= group_rows(p, e_mma);
        }
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          if (!(ok = mbar_spin(&gready[s], ph, abort_flag, p.err))) break;
          const uint64_t b0 = bd_base + static_cast<uint64_t>(s * (C::kB >> 4));
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            // half 1's activation tiles landed
            if (h == 1 && !(ok = mbar_spin(&afull[a], static_cast<uint32_t>((2 * it + 1) / SA) & 1u, abort_flag, p.err)))
              break;
            // the previous tile's epilogue has drained accumulator h
            if (kb == 0 && tc >= 1 &&
                !(ok = mbar_spin_cluster(&tempty[h], static_cast<uint32_t>(tc - 1) & 1u, abort_flag, p.err)))
              break;
            if (kb == 0) tc_fence_after();
            const uint32_t d_tmem = tmem_base + h * kTmemCols;
            const uint64_t a0 = ad_base + static_cast<uint64_t>(a * (C::kA >> 4));
            if (!(h == 1 && skip1)) {
#pragma unroll
              for (int kk = 0; kk < C::kBK / 16; ++kk) {
                const uint32_t ka = ((kk >> 2) * 16384 + (kk & 3) * 32) >> 4;
                const uint32_t kb_ = MODE == MODE_FWD ? ka : (kk * 2048) >> 4;
                umma_bf16_pair(d_tmem, a0 + ka, b0 + kb_, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
              }
            }
            if (h == 0) umma_commit_pair_mc(&aempty[a]);
            if (kb == num_k - 1) umma_commit_pair_mc(&tfull[h]);  // the epilogue may start on accumulator h
            if (++a == SA) a = 0;
          }
          if (!ok) break;
          umma_commit_pair_mc(&empty[s]);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      umma_commit_pair(drain);
      mbar_drain(drain, 0);
    }
  } else if (warp == C::kGateWarp) {
    // ------------------------------------------------------ gate (leader CTA)
    // Waits, for each k-step, for half 0's activation tiles (afull; they usually
    // land first) and then for both decoded halves (pready, a cluster-scope acquire
    // that costs a few hundred cycles even on a completed barrier), and hands the
    // step to the MMA thread through one CTA-local barrier. It also arms pready with
    // the signal bytes of each use (decode warps may signal before it is armed: the
    // missing arrival keeps the phase open).
    if (lane == 0 && rank == 0) {
      const int iters = my_tiles * num_k;
      for (int s = 0; s < S && s < iters; ++s) mbar_arrive_expect_tx(&pready[s], C::kSignalBytes);
      for (int it = 0; it < iters; ++it) {
        const int s = it % S;
        if (!mbar_spin(&afull[(2 * it) % SA], static_cast<uint32_t>((2 * it) / SA) & 1u, abort_flag, p.err)) break;
        if (!mbar_spin_cluster(&pready[s], static_cast<uint32_t>(it / S) & 1u, abort_flag, p.err)) break;
        mbar_arrive(&gready[s]);
        if (it + S < iters) mbar_arrive_expect_tx(&pready[s], C::kSignalBytes);
      }
    }
  } else if (FMT == kFmtBf16Mul && warp >= C::kEpiWarps) {
    // ------------------------------------------------------ in-place scaling (both CTAs)
    // Each thread scales its 32-weight unit of the landed bf16 tile: W' =
    // bf16(fl32(W * f)) with f = fl32(1 + dS[n, k / 16]) per block of 16, rounded
    // to nearest even, written back in place; factors are loaded one stage ahead.
    const int dw = warp - C::kEpiWarps;
    const int u = dw * 32 + lane;
    const int row = (u & 7) + 8 * (u >> 5), quarter = (u >> 3) & 3;
    uint32_t b_off[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int chunk = 4 * (quarter & 1) + c;
      b_off[c] = MODE == MODE_FWD
                     ? (quarter >> 1) * 16384 + (row >> 3) * 1024 + (row & 7) * 128 + ((chunk ^ (row & 7)) << 4)
                     : (quarter >> 1) * 16384 + row * 128 + ((chunk ^ (row & 7)) << 4);
    }
    const float *dS = reinterpret_cast<const float *>(p.scales);
    const int64_t G = p.K / 16;
    auto factors = [&](int tile, int kb, int tn, float &f0, float &f1) {
      f0 = f1 = 0.f;
      if (tile >= total) return;
      int64_t n, k;
      pair_unit_coords<MODE>(u, static_cast<int64_t>(tn) * C::kTile + 128 * rank, kb, n, k);
      if (n >= p.N || k >= p.K) return;  // outside the weight: the tile holds zeros there
      f0 = __fadd_rn(1.0f, __ldg(dS + n * G + k / 16));
      f1 = __fadd_rn(1.0f, __ldg(dS + n * G + k / 16 + 1));
    };
    const uint32_t sink_addr = mapa_shared(smem_u32(&sink[rank * C::kDecWarps + dw]), 0);
    int it = 0, s = 0, e = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int tile = cluster; tile < total && ok; tile += nclusters) {
      int tm, tn;
      resolve_tile<GR>(p, tile, e, tm, tn);
      float f0, f1;
      factors(tile, 0, tn, f0, f1);
      for (int kb = 0; kb < num_k && ok; ++kb, ++it) {
        float g0, g1;
        factors(tile, kb + 1 < num_k ? kb + 1 : num_k, tn, g0, g1);  // next stage's factors
        if (lane == 0) ok = mbar_wait(&cfull[s], ph, abort_flag, p.err);
        ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
        __syncwarp();
        if (!ok) break;
        const uint32_t b_base = smem_u32(ring_b(s));
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const uint4 v = lds128(b_base + b_off[c]);
          const float f = c < 2 ? f0 : f1;
          const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
          uint32_t o[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(__fmul_rn(__uint_as_float(wv[q] << 16), f),
                                                            __fmul_rn(__uint_as_float(wv[q] & 0xFFFF0000u), f));
            o[q] = *reinterpret_cast<const uint32_t *>(&h2);
          }
          st_shared_v4(b_base + b_off[c], o[0], o[1], o[2], o[3]);
        }
        fence_proxy_async_smem();  // this thread's shared-memory writes -> async proxy
        __syncwarp();
        if (lane == 0) st_async_signal(sink_addr, mapa_shared(smem_u32(&pready[s]), 0));
        f0 = g0;
        f1 = g1;
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
      }
    }
  } else if (warp >= C::kEpiWarps) {
    // ------------------------------------------------------ decode (both CTAs)
    // Every decode thread turns one 32-weight unit of every stage into bf16:
    // codes from the code ring, into the decoded slot the MMAs of k-step it - S freed.
    // (grouped launches keep per-expert tile state in the decode warps: a shallower scale
    // prefetch keeps them within the 72 registers without spilling)
    constexpr int kD = GR ? 2 : SQ_SCALE_DEPTH;
    const int dw = warp - C::kEpiWarps;
    const int u = dw * 32 + lane;  // this thread's unit, 0..511
    struct Pos {
      int tile, kb, e, tm, tn;
    };
    auto step = [&](Pos &q) {
      if (++q.kb == num_k) {
        q.kb = 0;
        q.tile += nclusters;
        if (q.tile < total) resolve_tile<GR>(p, q.tile, q.e, q.tm, q.tn);
      }
    };
    Pos cur{cluster, 0, 0, 0, 0};
    if (cur.tile < total) resolve_tile<GR>(p, cur.tile, cur.e, cur.tm, cur.tn);
    Pos ahead = cur;
    const int64_t plane = p.N * (p.K / (FMT == 0 ? 16 : 32));  // scale bytes of one expert
    auto scale_at = [&](const Pos &q) -> uint32_t {
      if (q.tile >= total) return 0u;
      int64_t n, k;
      pair_unit_coords<MODE>(u, static_cast<int64_t>(q.tn) * C::kTile + 128 * rank, q.kb, n, k);
      return load_unit_scale<FMT>(p, GR ? p.scales + q.e * plane : p.scales, n, k);
    };
    uint32_t sc[kD];
#pragma unroll
    for (int d = 0; d < kD; ++d) {
      sc[d] = scale_at(ahead);
      step(ahead);
    }
    // unit geometry inside the stage (fixed for the thread): code bytes in the
    // 64-byte-swizzled code tile, 16-byte chunks of the 128-byte-swizzled bf16 tile
    const int row = (u & 7) + 8 * (u >> 5), quarter = (u >> 3) & 3;
    const uint32_t c_off = row * 64 + ((quarter ^ ((row >> 1) & 3)) << 4);
    uint32_t b_off[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int chunk = 4 * (quarter & 1) + c;
      b_off[c] = MODE == MODE_FWD
                     ? (quarter >> 1) * 16384 + (row >> 3) * 1024 + (row & 7) * 128 + ((chunk ^ (row & 7)) << 4)
                     : (quarter >> 1) * 16384 + row * 128 + ((chunk ^ (row & 7)) << 4);
    }
    const uint32_t sink_addr = mapa_shared(smem_u32(&sink[rank * C::kDecWarps + dw]), 0);
    int it = 0, s = 0, cs = 0;
    uint32_t ph = 0, cph = 0;  // phase parities of the decoded slot and the code slot
    bool ok = true;
    while (cur.tile < total && ok) {
#pragma unroll
      for (int d = 0; d < kD; ++d) {
        if (cur.tile >= total || !ok) break;
        // The stage is decoded into registers as soon as its codes land; only the
        // stores wait for the decoded slot (freed by the MMAs of k-step it - S), and
        // that wait spins, so the slot is refilled within a few hundred cycles of
        // its release (the slot's round trip bounds the k-step rate).
        if (lane == 0) ok = mbar_wait(&cfull[cs], cph, abort_flag, p.err);
        ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
        __syncwarp();
        if (!ok) break;
        uint32_t sc_lo, sc_hi;
        if (FMT == 0) {
          sc_lo = scale_bf16x2<0>(sc[d] & 0xFFu);
          sc_hi = scale_bf16x2<0>(sc[d] >> 8);
        } else {
          sc_lo = sc_hi = scale_bf16x2<1>(sc[d]);
        }
        const uint4 cw = lds128(smem_u32(ring_c(cs)) + c_off);
        const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
        uint32_t o[4][4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          e2m1x8_to_bf16(words[c], o[c]);
          const uint32_t scv = c < 2 ? sc_lo : sc_hi;
#pragma unroll
          for (int q = 0; q < 4; ++q) o[c][q] = bf16x2_mul(o[c][q], scv);
        }
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&cempty[cs]);  // the warp's code reads are done
          if (it >= S) ok = mbar_spin(&empty[s], ph ^ 1u, abort_flag, p.err);
        }
        ok = __shfl_sync(0xFFFFFFFFu, ok ? 1 : 0, 0) != 0;
        __syncwarp();
        if (!ok) break;
        const uint32_t b_base = smem_u32(ring_b(s));
#pragma unroll
        for (int c = 0; c < 4; ++c) st_shared_v4(b_base + b_off[c], o[c][0], o[c][1], o[c][2], o[c][3]);
        fence_proxy_async_smem();  // this thread's shared-memory writes -> async proxy
        __syncwarp();
        if (lane == 0) {
          // tell the leader without waiting: an async store whose complete-tx on the
          // leader's stage barrier is a cluster-scope release (both CTAs, all decode warps)
          st_async_signal(sink_addr, mapa_shared(smem_u32(&pready[s]), 0));
        }
        sc[d] = scale_at(ahead);
        step(ahead);
        step(cur);
        ++it;
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
        if (++cs == SC) {
          cs = 0;
          cph ^= 1u;
        }
      }
    }
  } else {
    // ------------------------------------------------------ epilogue (warps 0-7, both CTAs)
    // Drains accumulator 0 (rows 0-255 of the tile), releases it so the next
    // tile's first MMAs can start, then accumulator 1. Warp w reads TMEM lanes
    // 32 (w % 4) .. +31 and columns 128 (w / 4) .. +127, 32 columns at a time:
    // it scales and rounds them to bf16 into a 32 x 32 box in shared memory
    // (64-byte swizzle) and stores the box with TMA, which writes whole row
    // segments and clips the ragged edges of the output. The dense input gradient
    // keeps a warp's last group in registers and releases the accumulator before
    // staging it, the grouped kernels their last two groups (measured: it helps
    // those, not the dense forward; two groups cost the dense input gradient).
    const int quad = warp & 3;
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quad * 32) << 16);
    const int cbase = (warp >> 2) * (C::kTile / 2);
    const int64_t Ng = MODE == MODE_FWD ? p.N : p.K;
    float scale = FMT == 0 ? p.ws2 : 1.0f;
    int64_t rows = p.M;
    const CUtensorMap *mO = &tmO;
    const uint32_t box = smem_u32(smem + C::kOffS + warp * C::kBoxBytes);
    const uint32_t row_base = box + lane * 64;  // this lane's 64-byte box row
    int tc = 0;
    int e = 0, e_seen = -1;
    for (int tile = cluster; tile < total; tile += nclusters, ++tc) {
      int tm, tn;
      resolve_tile<GR>(p, tile, e, tm, tn);
      if (GR && e != e_seen) {  // the expert's output rows, token count and tensor scale
        mO = &group_maps(p, e)->m[1];
        rows = group_rows(p, e);
        if (FMT == 0) scale = group_ws2(p, e);
        if (lane == 0) tensormap_acquire(mO);
        e_seen = e;
      }
      const int32_t col0 = tn * C::kTile;
      bool ok = true;
      for (int h = 0; h < 2 && ok; ++h) {
        if (!(ok = mbar_wait(&tfull[h], static_cast<uint32_t>(tc) & 1u, abort_flag, p.err))) break;
        tc_fence_after();
        const int32_t row = tm * C::kMTile + C::kTile * h + 128 * static_cast<int32_t>(rank) + 32 * quad;
        // a grouped tile's rows past its expert's last row are not stored, so a warp whose
        // 32 rows all lie there only releases the accumulator (those rows of it may not
        // even have been computed: see skip1 in the MMA issuer)
        if (GR && row >= rows) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (rank == 0) {
              if (warp == 0)
                mbar_arrive_expect_tx(&tempty[h], 4 * C::kEpiWarps);
              else
                mbar_arrive(&tempty[h]);
            } else {
              st_async_signal(mapa_shared(smem_u32(&sink[2 * C::kDecWarps + warp]), 0),
                              mapa_shared(smem_u32(&tempty[h]), 0));
            }
          }
          continue;
        }
        if constexpr (GR) {
          const uint32_t t_buf = t_row + h * kTmemCols;
          // the last SQ_EPI_HOLD_GR 32-column groups are read into registers and stored
          // after the accumulator is released (the loop is unrolled to keep them there)
          constexpr int kGroups = C::kTile / 2 / 32;
          constexpr int kHeld = SQ_EPI_HOLD_GR;
          uint32_t held[kHeld][16];
          auto store_box = [&](const uint32_t (&w)[16], int c) {
            if (lane == 0) bulk_wait_read<0>();  // the previous box's store has read the buffer
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 4; ++q)
              st_shared_v4(row_base + ((q ^ ((lane >> 1) & 3)) << 4), w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
            fence_proxy_async_smem();  // the box -> async proxy (the TMA store)
            __syncwarp();
            if (lane == 0) {
              if (row < rows && col0 + c < Ng) tma_store_2d(mO, box, col0 + c, row);
              bulk_commit_group();
            }
          };
#pragma unroll
          for (int gi = 0; gi < kGroups; ++gi) {
            const int c = cbase + 32 * gi;
            uint32_t v[32];
            tmem_ld32(t_buf + c, v);
            tmem_ld_wait();
            uint32_t packed[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const __nv_bfloat162 h2 =
                  __floats2bfloat162_rn(__uint_as_float(v[2 * q]) * scale, __uint_as_float(v[2 * q + 1]) * scale);
              packed[q] = *reinterpret_cast<const uint32_t *>(&h2);
            }
            if (gi >= kGroups - kHeld) {
#pragma unroll
              for (int q = 0; q < 16; ++q) held[gi - (kGroups - kHeld)][q] = packed[q];
            } else {
              store_box(packed, c);
            }
          }
          tc_fence_before();
          __syncwarp();
          // accumulator h drained: the leader's warps arrive (warp 0 arming the peer's
          // bytes), the peer's warps signal with a non-blocking async store
          if (lane == 0) {
            if (rank == 0) {
              if (warp == 0)
                mbar_arrive_expect_tx(&tempty[h], 4 * C::kEpiWarps);
              else
                mbar_arrive(&tempty[h]);
            } else {
              st_async_signal(mapa_shared(smem_u32(&sink[2 * C::kDecWarps + warp]), 0),
                              mapa_shared(smem_u32(&tempty[h]), 0));
            }
          }
#pragma unroll
          for (int hi = 0; hi < kHeld; ++hi) store_box(held[hi], cbase + 32 * (kGroups - kHeld + hi));
        } else {
          const uint32_t t_buf = t_row + h * kTmemCols;
          // the input gradient: the last 32-column group is read into registers and
          // stored after the accumulator is released
          constexpr bool kHold = MODE == MODE_DX;
          uint32_t held[16];
#pragma unroll 1
          for (int j = 0; j < C::kTile / 2; j += 32) {
            const int c = cbase + j;
            uint32_t v[32];
            tmem_ld32(t_buf + c, v);
            tmem_ld_wait();
            uint32_t packed[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const __nv_bfloat162 h2 =
                  __floats2bfloat162_rn(__uint_as_float(v[2 * q]) * scale, __uint_as_float(v[2 * q + 1]) * scale);
              packed[q] = *reinterpret_cast<const uint32_t *>(&h2);
            }
            if (kHold && j == C::kTile / 2 - 32) {
#pragma unroll
              for (int q = 0; q < 16; ++q) held[q] = packed[q];
              break;
            }
            if (lane == 0) bulk_wait_read<0>();  // the previous box's store has read the buffer
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 4; ++q)
              st_shared_v4(row_base + ((q ^ ((lane >> 1) & 3)) << 4), packed[4 * q], packed[4 * q + 1],
                           packed[4 * q + 2], packed[4 * q + 3]);
            fence_proxy_async_smem();  // the box -> async proxy (the TMA store)
            __syncwarp();
            if (lane == 0) {
              if (row < rows && col0 + c < Ng) tma_store_2d(mO, box, col0 + c, row);
              bulk_commit_group();
            }
          }
          tc_fence_before();
          __syncwarp();
          // accumulator h drained: the leader's warps arrive (warp 0 arming the peer's
          // bytes), the peer's warps signal with a non-blocking async store
          if (lane == 0) {
            if (rank == 0) {
              if (warp == 0)
                mbar_arrive_expect_tx(&tempty[h], 4 * C::kEpiWarps);
              else
                mbar_arrive(&tempty[h]);
            } else {
              st_async_signal(mapa_shared(smem_u32(&sink[2 * C::kDecWarps + warp]), 0),
                              mapa_shared(smem_u32(&tempty[h]), 0));
            }
          }
          if (kHold) {  // the held group: staged and stored now
            const int c = cbase + C::kTile / 2 - 32;
            if (lane == 0) bulk_wait_read<0>();
            __syncwarp();
#pragma unroll
            for (int q = 0; q < 4; ++q)
              st_shared_v4(row_base + ((q ^ ((lane >> 1) & 3)) << 4), held[4 * q], held[4 * q + 1], held[4 * q + 2],
                           held[4 * q + 3]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              if (row < rows && col0 + c < Ng) tma_store_2d(mO, box, col0 + c, row);
              bulk_commit_group();
            }
          }
        }
      }
      if (!ok) break;
    }
    if (lane == 0) bulk_wait_all();
  }

  __syncwarp();
  tc_fence_before();
  cluster_sync_all();
  if (warp == C::kMmaWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, 2 * kTmemCols);
  }
}

// ------------------------------------------------------------- CTA-pair scale-gradient kernel
//
// A cluster of two CTAs owns a 256 (n) x 256 (k) tile of dW = dY^T X and issues
// tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 16 tokens). Each CTA loads 128
// n-rows of dY^T (A) and 128 k-columns of X (B) per stage, both MN-major, so per
// MMA each SM reads 8 KiB of operands from its shared memory instead of the
// 12 KiB of a single-CTA 128 x 256 MMA, and the TMA traffic per SM drops by a
// third. Each CTA keeps the accumulator of its 128 n-rows (all 256 columns) in
// its TMEM and reduces it by blocks in its own epilogue.
struct SgradPairCfg {
  static constexpr int kEpiWarps = 4;  // warps 0-3: TMEM lanes 0-127
  static constexpr int kTmaWarp = 4;
  static constexpr int kMmaWarp = 5;
  static constexpr int kThreads = 192;
  static constexpr int kBK = kSgradBK;         // tokens per stage: 8 MMAs of K = 16
  static constexpr int kStages = 3;
  static constexpr int kA = 128 * kBK * 2;     // 16 KiB: this CTA's 128 n-rows of dY^T, two MN atoms of 64 n
  static constexpr int kB = 128 * kBK * 2;     // 16 KiB: this CTA's 128 k-columns of X, two MN atoms of 64 k
  static constexpr int kAtom = kBK * 128;      // bytes of one 64-wide MN atom (kBK rows of 128 B)
  static constexpr int kStageBytes = kA + kB;
  static constexpr uint32_t kTx = 2 * kStageBytes;  // both CTAs' tiles, counted on the leader's barrier
  static constexpr int kTile = kSgradTile;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 1024;
};
static_assert(SgradPairCfg::kSmemBytes <= 232448, "scale-gradient kernel exceeds the opt-in shared memory");

template <int FMT, bool GR>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(SgradPairCfg::kThreads, 1)
    sq_sgrad_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const KParams p) {
  using C = SgradPairCfg;
  constexpr int S = C::kStages;
  constexpr int B = FMT == 1 ? 32 : 16;  // the multiplicative control has one factor per 16 weights
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + S * C::kStageBytes);
  uint64_t *full = bars;              // [S] leader: both CTAs' tiles of the stage landed (1 arrival + tx)
  uint64_t *empty = full + S;         // [S] pair MMAs reading the stage completed     (multicast commit)
  uint64_t *tfull = empty + S;        // [2] accumulator buffer complete                (multicast commit)
  uint64_t *tempty = tfull + 2;       // [2] leader: both epilogues drained the buffer
                                      //     (kEpiWarps arrivals + the peer warps' st.async tx)
  uint64_t *drain = tempty + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  uint32_t *sink = reinterpret_cast<uint32_t *>(drain + 2);  // [kEpiWarps] leader: st.async targets

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int cluster = blockIdx.x >> 1;
  const int nclusters = gridDim.x >> 1;
  const int total = p.total;
  // Unit u of the launch: tile (tm, tn) (of expert e in a grouped launch) over the
  // token stages [m0, m0 + kBK * num_k): all M tokens, the expert's own M_e, or in
  // a dense launch cut into token splits, part sp of them (an expert or part
  // without tokens gets zero gradient blocks). Returns num_k.
  const int tiles_per_split = p.tiles_m * p.tiles_n;
  const int64_t split_tokens =
      ((p.M + p.splits - 1) / p.splits + C::kBK - 1) / C::kBK * C::kBK;  // a multiple of kBK
  auto unit_of = [&](int u, int &e, int &tm, int &tn, int &sp, int32_t &m0) -> int {
    if (GR) {
      resolve_tile<GR, kSgradGroup>(p, u, e, tm, tn);
      sp = 0;
      m0 = 0;
      return static_cast<int>((static_cast<int64_t>(group_rows(p, e)) + C::kBK - 1) / C::kBK);
    }
    sp = p.splits > 1 ? u / tiles_per_split : 0;
    resolve_tile<GR, kSgradGroup>(p, u - sp * tiles_per_split, e, tm, tn);
    const int64_t first = static_cast<int64_t>(sp) * split_tokens;
    const int64_t len = p.M - first < split_tokens ? p.M - first : split_tokens;
    m0 = static_cast<int32_t>(first);
    return len > 0 ? static_cast<int>((len + C::kBK - 1) / C::kBK) : 0;
  };

  auto stage_a = [&](int s) { return smem + s * C::kStageBytes; };
  auto stage_b = [&](int s) { return smem + s * C::kStageBytes + C::kA; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], C::kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == C::kMmaWarp) tmem_alloc_pair(tmem_slot, 2 * kTmemCols);
  if (!GR && warp == C::kTmaWarp && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == C::kTmaWarp) {
    // ------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      int e = 0, e_seen = -1;
      const CUtensorMap *mA = &tmA, *mB = &tmB;
      for (int tile = cluster; tile < total && ok; tile += nclusters) {
        int tm, tn, sp;
        int32_t m0;
        const int num_k = unit_of(tile, e, tm, tn, sp, m0);
        if (GR && e != e_seen && num_k > 0) {  // the expert's own token rows of dY and X (an expert
          mA = &group_maps(p, e)->m[0];        // without tokens has no descriptors and loads nothing)
          mB = &group_maps(p, e)->m[1];
          tensormap_acquire(mA);
          tensormap_acquire(mB);
          e_seen = e;
        }
        const int32_t row0 = tm * C::kTile + 128 * static_cast<int32_t>(rank);  // n
        const int32_t col0 = tn * C::kTile + 128 * static_cast<int32_t>(rank);  // k
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int s = it % S;
          const uint32_t use = static_cast<uint32_t>(it / S);
          if (it >= S && !(ok = mbar_wait(&empty[s], (use & 1u) ^ 1u, abort_flag, p.err))) break;
          if (rank == 0) mbar_arrive_expect_tx(&full[s], C::kTx);
          const uint32_t bar = mapa_shared(smem_u32(&full[s]), 0);
          const int32_t kc = m0 + kb * C::kBK;
          for (int j = 0; j < 2; ++j) tma_load_2d_pair(smem_u32(stage_a(s)) + j * C::kAtom, mA, bar, row0 + 64 * j, kc);
          for (int j = 0; j < 2; ++j) tma_load_2d_pair(smem_u32(stage_b(s)) + j * C::kAtom, mB, bar, col0 + 64 * j, kc);
        }
      }
      if (*abort_flag && rank == 0) {
        for (int i = (it > S ? it - S : 0); i < it; ++i) mbar_drain(&full[i % S], static_cast<uint32_t>(i / S) & 1u);
      }
    }
  } else if (warp == C::kMmaWarp) {
    // ------------------------------------------------------ MMA issuer (leader CTA)
    // One barrier wait per stage, spinning (test_wait); nothing polled between MMAs.
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16(2 * 128, C::kTile, 1, 1);
      const uint64_t ad_base = smem_desc_sw128(smem_u32(stage_a(0)), C::kAtom, 1024);
      const uint64_t bd_base = smem_desc_sw128(smem_u32(stage_b(0)), C::kAtom, 1024);
      int s = 0;
      uint32_t ph = 0;
      int tc = 0;
      bool ok = true;
      int e = 0;
      for (int tile = cluster; tile < total && ok; tile += nclusters, ++tc) {
        int tm, tn, sp;
        int32_t m0;
        const int num_k = unit_of(tile, e, tm, tn, sp, m0);
        const int ab = tc & 1;
        const uint32_t au = static_cast<uint32_t>(tc >> 1);
        if (tc >= 2 && !(ok = mbar_spin_cluster(&tempty[ab], (au & 1u) ^ 1u, abort_flag, p.err))) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + ab * kTmemCols;
        for (int kb = 0; kb < num_k; ++kb) {
          if (!(ok = mbar_spin(&full[s], ph, abort_flag, p.err))) break;
          const uint64_t so = static_cast<uint64_t>(s * (C::kStageBytes >> 4));
          const uint64_t a0 = ad_base + so, b0 = bd_base + so;
#pragma unroll
          for (int kk = 0; kk < C::kBK / 16; ++kk) {
            // MN-major operands: 16 token rows (2 KiB) per K step
            umma_bf16_pair(d_tmem, a0 + static_cast<uint64_t>(kk * 2048 >> 4),
                           b0 + static_cast<uint64_t>(kk * 2048 >> 4), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit_pair_mc(&empty[s]);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (ok) umma_commit_pair_mc(&tfull[ab]);
      }
      umma_commit_pair(drain);
      mbar_drain(drain, 0);
    }
  } else if (warp < C::kEpiWarps) {
    // ------------------------------------------------------ epilogue (warps 0-3, both CTAs)
    const int r = warp * 32 + lane;
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(warp * 32) << 16);
    const int64_t G = p.K / B;
    int tc = 0;
    int e = 0;
    for (int tile = cluster; tile < total; tile += nclusters, ++tc) {
      int tm, tn, sp;
      int32_t m0;
      const int num_k = unit_of(tile, e, tm, tn, sp, m0);
      // the expert's code plane (the multiplicative control: its bf16 weights), gradient plane and
      // mask; a token split writes its own partial plane, masked when the parts are added
      const int64_t eid = GR ? group_id(p, e) : 0;  // the expert of table entry e
      const uint8_t *codes = GR ? p.codes + eid * p.N * (p.K / 2) : p.codes;
      float *g = p.splits > 1 ? p.partial + sp * p.N * G : static_cast<float *>(p.out) + (GR ? eid * p.N * G : 0);
      const uint8_t *mask = p.mask && p.splits == 1 ? p.mask + (GR ? eid * p.N * G : 0) : nullptr;
      const bool empty_sum = num_k == 0;  // no tokens: the accumulator was never written
      const int64_t n = static_cast<int64_t>(tm) * C::kTile + 128 * rank + r;
      const int64_t col0 = static_cast<int64_t>(tn) * C::kTile;
      const int ab = tc & 1;
      const uint32_t au = static_cast<uint32_t>(tc >> 1);
      if (!mbar_wait(&tfull[ab], au & 1u, abort_flag, p.err)) break;
      tc_fence_after();
      const uint32_t t_buf = t_row + ab * kTmemCols;
      for (int c0 = 0; c0 < C::kTile; c0 += 32) {
        uint32_t v[32];
        tmem_ld32(t_buf + c0, v);
        tmem_ld_wait();
        if (empty_sum) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0u;
        }
        const int64_t k = col0 + c0;
        if (n >= p.N || k >= p.K) continue;
        uint4 cw = make_uint4(0, 0, 0, 0);
        if (FMT != kFmtBf16Mul) cw = __ldg(reinterpret_cast<const uint4 *>(codes + n * (p.K / 2) + k / 2));
        const uint32_t words[4] = {cw.x, cw.y, cw.z, cw.w};
        float part[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t o[4];  // 8 weights of the row as bf16 pairs: decoded codes, or the control's bf16 W
          if (FMT == kFmtBf16Mul) {
            const uint4 wq = __ldg(reinterpret_cast<const uint4 *>(codes + (n * p.K + k + 8 * c) * 2));
            o[0] = wq.x;
            o[1] = wq.y;
            o[2] = wq.z;
            o[3] = wq.w;
          } else {
            e2m1x8_to_bf16(words[c], o);
          }
          float acc = 0.f;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            acc = fmaf(__uint_as_float(o[e] << 16), __uint_as_float(v[8 * c + 2 * e]), acc);
            acc = fmaf(__uint_as_float(o[e] & 0xFFFF0000u), __uint_as_float(v[8 * c + 2 * e + 1]), acc);
          }
          part[c] = acc;
        }
        if (FMT != 1) {
          const int64_t b = k / 16;
          float g0 = part[0] + part[1];
          float g1 = part[2] + part[3];
          if (mask) {
            g0 *= static_cast<float>(mask[n * G + b]);
            g1 *= static_cast<float>(mask[n * G + b + 1]);
          }
          *reinterpret_cast<float2 *>(g + n * G + b) = make_float2(g0, g1);
        } else {
          const int64_t b = k / 32;
          float g0 = (part[0] + part[1]) + (part[2] + part[3]);
          if (mask) g0 *= static_cast<float>(mask[n * G + b]);
          g[n * G + b] = g0;
        }
      }
      tc_fence_before();
      __syncwarp();
      // buffer drained: the leader's warps arrive (warp 0 arming the peer's bytes),
      // the peer's warps signal with a non-blocking async store
      if (lane == 0) {
        if (rank == 0) {
          if (warp == 0)
            mbar_arrive_expect_tx(&tempty[ab], 4 * C::kEpiWarps);
          else
            mbar_arrive(&tempty[ab]);
        } else {
          st_async_signal(mapa_shared(smem_u32(&sink[warp]), 0), mapa_shared(smem_u32(&tempty[ab]), 0));
        }
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  cluster_sync_all();
  if (warp == C::kMmaWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, 2 * kTmemCols);
  }
}


// Persistent launch of one cluster kernel: as many two-CTA clusters as fit on the
// GPU at once (queried once per device), capped by the tiles of the launch.
template <typename Kernel, typename... Args>
cudaError_t launch_persistent(Kernel kernel, int threads, int smem_bytes, int64_t tiles, int sm_count,
                              cudaStream_t stream, int *max_clusters, int *done_mask, Args... args) {
  int dev = 0;
  cudaGetDevice(&dev);
  if (!(*done_mask & (1 << (dev & 31)))) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (sm_count / 2), 1, 1);
    cfg.blockDim = dim3(threads, 1, 1);
    cfg.dynamicSmemBytes = smem_bytes;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
      cudaGetLastError();
      n = sm_count / 2;
    }
    max_clusters[dev & 31] = n;
    *done_mask |= 1 << (dev & 31);
  }
  const int64_t nc = tiles < max_clusters[dev & 31] ? tiles : max_clusters[dev & 31];
  if (nc <= 0) return cudaSuccess;
  kernel<<<static_cast<unsigned>(2 * nc), threads, smem_bytes, stream>>>(args...);
  return cudaGetLastError();
}

template <int MODE, int FMT, bool GR>
cudaError_t launch_pair(const KParams &p, const CUtensorMap &tmA, const CUtensorMap &tmC, const CUtensorMap &tmO,
                        int sm_count, cudaStream_t stream) {
  static int done_mask = 0;  // per device ordinal (first 31)
  static int max_clusters[32] = {0};
  return launch_persistent(sq_gemm_pair_kernel<MODE, FMT, GR>, PairCfg::kThreads, PairCfg::kSmemBytes, p.total,
                           sm_count, stream, max_clusters, &done_mask, tmA, tmC, tmO, p);
}

template <int FMT, bool GR>
cudaError_t launch_sgrad(const KParams &p, const CUtensorMap &tmA, const CUtensorMap &tmB, int sm_count,
                         cudaStream_t stream) {
  static int done_mask = 0;
  static int max_clusters[32] = {0};
  return launch_persistent(sq_sgrad_pair_kernel<FMT, GR>, SgradPairCfg::kThreads, SgradPairCfg::kSmemBytes, p.total,
                           sm_count, stream, max_clusters, &done_mask, tmA, tmB, p);
}

}  // namespace
}  // namespace sqi
