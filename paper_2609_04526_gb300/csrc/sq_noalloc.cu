// Allocation-free variant of the scale-gradient entry point.
//
// The regular entry points keep their scratch memory -- the device word that a
// kernel sets when one of its bounded waits runs out -- in the sq_handle, which
// allocates it with cudaMalloc on the first call on each device. Some callers
// cannot call cudaMalloc: code whose device memory belongs to an outside pool or
// allocator that must account for every byte, and hot loops that cannot accept
// the device-wide synchronisation that cudaMalloc / cudaFree may cause. For them
// sq_scale_grad_noalloc runs the same scale-gradient kernel with its scratch in a
// file-scope static __device__ array instead, and allocates nothing.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "scaleqlora.h"
#include "sq_internal.h"

namespace {

// Scratch of the allocation-free entry point. It is part of the loaded module:
// every GPU that loads the library holds these 256 bytes until the process exits,
// and every call of sq_scale_grad_noalloc on that GPU shares them. Word 0 is the
// kernel's error word; the rest is headroom.
constexpr size_t kScratchBytes = 256;
static __device__ __align__(256) int g_noalloc_scratch[kScratchBytes / sizeof(int)];

constexpr size_t kScratchNeeded = sizeof(int);  // one error word, whatever M, N and K are
constexpr int kMaxDevices = 64;

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

struct NoAllocDevice {
  bool ready;
  int sm_count;
};

std::mutex g_mu;
NoAllocDevice g_dev[kMaxDevices];
EncodeTiledFn g_encode = nullptr;

// With the caller's device current: check it once (compute capability 10.3, SM
// count, the driver's tensor-map encoder), then on every call look up the device
// address of the static scratch array. In host code the array's name is only a
// host-side stand-in, so the kernel must be given this address; looking it up
// each time (it allocates nothing) keeps it right after a device reset.
sq_status setup_current_device(NoAllocDevice **out, int **scratch) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return SQ_ERR_DEVICE;
  if (dev >= kMaxDevices) return SQ_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  NoAllocDevice &d = g_dev[dev];
  if (!d.ready) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return SQ_ERR_CUDA;
    if (major != 10 || minor != 3) return SQ_ERR_UNSUPPORTED;
    if (!g_encode) {
      void *fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || !fn)
        return SQ_ERR_DEVICE;
      g_encode = reinterpret_cast<EncodeTiledFn>(fn);
    }
    d.sm_count = sms;
    d.ready = true;
  }
  int *ptr = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void **>(&ptr), g_noalloc_scratch) != cudaSuccess || !ptr)
    return SQ_ERR_CUDA;
  *scratch = ptr;
  *out = &d;
  return SQ_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// bf16 [outer, inner] tensor in 64 x kSgradBK boxes with the 128-byte swizzle (MN-major operand tiles).
bool encode_act(CUtensorMap *map, const void *ptr, int64_t inner, int64_t outer) {
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(sqi::kSgradBK)};
  const cuuint32_t estr[2] = {1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

extern "C" sq_status sq_scale_grad_noalloc(const sq_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                                           const uint8_t *mask, float *g, int32_t *device_status, void *stream) {
  // Same argument rules as sq_scale_grad.
  if (!w || (w->fmt != SQ_NVFP4 && w->fmt != SQ_MXFP4)) return SQ_ERR_INVALID_ARG;
  if (w->fmt == SQ_NVFP4 ? !(std::isfinite(w->ws2) && w->ws2 > 0.0f) : w->ws2 != 1.0f) return SQ_ERR_INVALID_ARG;
  if (w->N <= 0 || w->N % 8 != 0 || w->N > (1 << 24) || w->K <= 0 || w->K % 32 != 0 || w->K > (1 << 24))
    return SQ_ERR_INVALID_ARG;
  if (!w->codes || !aligned16(w->codes) || !g || !aligned16(g)) return SQ_ERR_INVALID_ARG;
  if (M < 0 || M > (int64_t(1) << 31) - 1) return SQ_ERR_INVALID_ARG;
  if (M > 0 && (!X || !aligned16(X) || !dY || !aligned16(dY))) return SQ_ERR_INVALID_ARG;
  if (device_status && (reinterpret_cast<uintptr_t>(device_status) & 3u)) return SQ_ERR_INVALID_ARG;
  // Scratch need against the static array (the need does not grow with M, N or K).
  if (kScratchNeeded > kScratchBytes) return SQ_ERR_INVALID_ARG;

  NoAllocDevice *dev = nullptr;
  int *scratch = nullptr;
  sq_status st = setup_current_device(&dev, &scratch);
  if (st != SQ_OK) return st;
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int B = w->fmt == SQ_NVFP4 ? 16 : 32;

  // The shared array keeps the last call's contents: clear the error word first.
  if (cudaMemsetAsync(scratch, 0, kScratchNeeded, s) != cudaSuccess) return SQ_ERR_CUDA;
  if (M == 0) {
    if (cudaMemsetAsync(g, 0, static_cast<size_t>(w->N) * (w->K / B) * sizeof(float), s) != cudaSuccess)
      return SQ_ERR_CUDA;
  } else {
    CUtensorMap tmA, tmB;
    if (!encode_act(&tmA, dY, w->N, M) || !encode_act(&tmB, X, w->K, M)) return SQ_ERR_CUDA;
    sqi::GemmArgs a;
    a.mode = sqi::MODE_SGRAD;
    a.fmt = w->fmt;
    a.M = M;
    a.N = w->N;
    a.K = w->K;
    a.codes = w->codes;
    a.scales = w->scales;
    a.ws2 = w->ws2;
    a.out = g;
    a.mask = mask;
    a.err = scratch;
    if (sqi::launch_gemm(a, tmA, tmB, nullptr, dev->sm_count, s) != cudaSuccess) return SQ_ERR_CUDA;
  }
  if (device_status &&
      cudaMemcpyAsync(device_status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return SQ_ERR_CUDA;
  return SQ_OK;
}
