// Host layer of libscaleqlora: argument validation, device checks, TMA
// descriptor encoding and kernel launches behind the C ABI of scaleqlora.h.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "scaleqlora.h"
#include "sq_internal.h"

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// One expert table of a grouped launch: built in pinned host memory, copied to
// the device on the call's stream. `done` is recorded after the launch that reads
// it, so the slot is rewritten only once that launch (and its copy) completed.
struct TableSlot {
  uint8_t *host = nullptr;
  uint8_t *dev = nullptr;
  size_t bytes = 0;
  cudaEvent_t done = nullptr;
  bool pending = false;
};
constexpr int kTableSlots = 4;

// Device scratch that grows on demand. Once a graph capture has recorded the buffer
// it is never freed while the handle lives: growing it then retires the old buffer
// (freed by sq_destroy), so graphs captured earlier keep valid pointers.
struct Scratch {
  void *ptr = nullptr;
  size_t bytes = 0;
  bool captured = false;        // a capture has recorded ptr
  std::vector<void *> retired;  // earlier buffers recorded by captures
};

struct DeviceState {
  int device;
  int sm_count;
  int *err_word;         // device int, written by kernels whose bounded waits ran out
  Scratch workspace;     // scratch of the adapter-gradient kernels
  TableSlot tables[kTableSlots];
  int next_table;
  Scratch partial;       // token-split partial planes of the dense scale gradient
  int64_t *plane_acc;    // counter accumulators of the multi-plane calls (zero between calls)
};

constexpr int64_t kMaxDim = int64_t(1) << 24;       // N, K limit
constexpr int64_t kMaxTokens = (int64_t(1) << 31) - 1;  // TMA coordinates are int32

}  // namespace

struct sq_handle_s {
  std::string last_error;
  std::vector<DeviceState> devices;
  EncodeTiledFn encode = nullptr;
};

namespace {

sq_status fail(sq_handle h, sq_status s, const char *fmt, ...) {
  if (h) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    h->last_error = buf;
  }
  return s;
}

sq_status cuda_fail(sq_handle h, cudaError_t e, const char *what) {
  return fail(h, SQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Current device: checked for compute capability 10.3, error word allocated once.
sq_status ensure_device(sq_handle h, DeviceState **out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(h, SQ_ERR_DEVICE, "no CUDA device: %s", cudaGetErrorString(e));
  for (auto &d : h->devices)
    if (d.device == dev) {
      *out = &d;
      return SQ_OK;
    }
  int major = 0, minor = 0, sms = 0;
  if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
      (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return cuda_fail(h, e, "device query");
  if (major != 10 || minor != 3)
    return fail(h, SQ_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a only", dev, major,
                minor);
  if (!h->encode) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
      return fail(h, SQ_ERR_DEVICE, "driver entry point cuTensorMapEncodeTiled unavailable");
    h->encode = reinterpret_cast<EncodeTiledFn>(fn);
  }
  int *err_word = nullptr;
  if ((e = cudaMalloc(&err_word, sizeof(int))) != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(error word)");
  if ((e = cudaMemset(err_word, 0, sizeof(int))) != cudaSuccess) return cuda_fail(h, e, "cudaMemset(error word)");
  int64_t *plane_acc = nullptr;
  if ((e = cudaMalloc(&plane_acc, sqi::kPlaneAccBytes)) != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(plane counters)");
  if ((e = cudaMemset(plane_acc, 0, sqi::kPlaneAccBytes)) != cudaSuccess) return cuda_fail(h, e, "cudaMemset(plane counters)");
  DeviceState d{};
  d.device = dev;
  d.sm_count = sms;
  d.err_word = err_word;
  d.plane_acc = plane_acc;
  d.next_table = 0;
  h->devices.push_back(std::move(d));
  *out = &h->devices.back();
  return SQ_OK;
}

// 2-D tensor [outer, inner] (row-major, inner contiguous) moved in
// box_inner x box_outer tiles; out-of-range elements read as zero and are
// not written.
sq_status make_map(sq_handle h, CUtensorMap *map, const void *ptr, CUtensorMapDataType dtype, int elem_bytes,
                   int64_t inner, int64_t outer, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz) {
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * elem_bytes};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = h->encode(map, dtype, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(h, SQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return SQ_OK;
}

// bf16 activation tensor with the 128-byte swizzle the MMA descriptors expect.
sq_status make_act_map(sq_handle h, CUtensorMap *map, const void *ptr, int64_t inner, int64_t outer,
                       uint32_t box_inner, uint32_t box_outer) {
  return make_map(h, map, ptr, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, inner, outer, box_inner, box_outer,
                  CU_TENSOR_MAP_SWIZZLE_128B);
}

// bf16 output [outer, inner] of the pair kernels, written by the epilogue warps as
// 32-row x 32-column TMA store boxes (64-byte rows, 64-byte swizzle).
sq_status make_out_map(sq_handle h, CUtensorMap *map, void *ptr, int64_t inner, int64_t outer) {
  return make_map(h, map, ptr, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, inner, outer, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
}

int block_of(int fmt) { return fmt == SQ_NVFP4 ? 16 : 32; }

sq_status check_ws2(sq_handle h, int fmt, float ws2) {
  if (fmt == SQ_NVFP4) {
    if (!(std::isfinite(ws2) && ws2 > 0.0f)) return fail(h, SQ_ERR_INVALID_ARG, "NVFP4 ws2 must be finite and > 0");
  } else if (fmt == SQ_MXFP4) {
    if (ws2 != 1.0f) return fail(h, SQ_ERR_INVALID_ARG, "MXFP4 ws2 must be 1.0");
  } else {
    return fail(h, SQ_ERR_INVALID_ARG, "unknown format %d", fmt);
  }
  return SQ_OK;
}

sq_status check_weight(sq_handle h, const sq_weight *w, bool need_scales) {
  if (!w) return fail(h, SQ_ERR_INVALID_ARG, "weight is NULL");
  sq_status s = check_ws2(h, w->fmt, w->ws2);
  if (s != SQ_OK) return s;
  if (w->N <= 0 || w->N % 8 != 0 || w->N > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "N=%d must be positive, a multiple of 8 and <= 2^24", w->N);
  if (w->K <= 0 || w->K % 32 != 0 || w->K > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "K=%d must be positive, a multiple of 32 and <= 2^24", w->K);
  if (!w->codes || !aligned16(w->codes)) return fail(h, SQ_ERR_INVALID_ARG, "codes must be non-NULL and 16-byte aligned");
  if (need_scales && (!w->scales || !aligned16(w->scales)))
    return fail(h, SQ_ERR_INVALID_ARG, "scales must be non-NULL and 16-byte aligned");
  return SQ_OK;
}

sq_status check_tokens(sq_handle h, int64_t M) {
  if (M < 0 || M > kMaxTokens) return fail(h, SQ_ERR_INVALID_ARG, "M=%lld out of range [0, 2^31)", (long long)M);
  return SQ_OK;
}

sq_status check_buf(sq_handle h, const void *p, const char *name) {
  if (!p || !aligned16(p)) return fail(h, SQ_ERR_INVALID_ARG, "%s must be non-NULL and 16-byte aligned", name);
  return SQ_OK;
}

#define SQ_TRY(expr)                    \
  do {                                  \
    sq_status _s = (expr);              \
    if (_s != SQ_OK) return _s;         \
  } while (0)

#define SQ_GUARD_BEGIN try {
#define SQ_GUARD_END                                                             \
  }                                                                              \
  catch (...) {                                                                  \
    return fail(h, SQ_ERR_CUDA, "internal error (host exception)");              \
  }

// Token splits of a dense scale gradient of M tokens on this device (sgrad_splits).
int sgrad_splits_of(const DeviceState *dev, const sq_weight *w, int64_t M) {
  const int64_t tiles = ((w->N + sqi::kSgradTile - 1) / sqi::kSgradTile) * ((w->K + sqi::kSgradTile - 1) / sqi::kSgradTile);
  return sqi::sgrad_splits(tiles, dev->sm_count / 2, M);
}

// Scratch `s` on the current device, at least `bytes`. Growing it is refused while
// `stream` is being captured into a graph (no allocation there); a buffer that was
// used during a capture is retired instead of freed when it grows. `need` names the
// scratch in the error text.
sq_status ensure_scratch(sq_handle h, Scratch &s, size_t bytes, cudaStream_t stream, const char *need) {
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(stream, &cap);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaStreamIsCapturing");
  const bool capturing = cap != cudaStreamCaptureStatusNone;
  if (bytes <= s.bytes) {
    if (capturing) s.captured = true;
    return SQ_OK;
  }
  if (capturing)
    return fail(h, SQ_ERR_UNSUPPORTED, "%s needs %zu bytes of scratch: make one call outside graph capture first", need,
                bytes);
  if (s.ptr) {
    if (s.captured)
      s.retired.push_back(s.ptr);
    else if ((e = cudaFree(s.ptr)) != cudaSuccess)  // waits for the work that may still use it
      return cuda_fail(h, e, "cudaFree(scratch)");
  }
  s.ptr = nullptr;
  s.bytes = 0;
  s.captured = false;
  if ((e = cudaMalloc(&s.ptr, bytes)) != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(scratch)");
  s.bytes = bytes;
  return SQ_OK;
}

void free_scratch(Scratch &s) {
  if (s.ptr) cudaFree(s.ptr);
  for (void *p : s.retired) cudaFree(p);
  s.ptr = nullptr;
  s.bytes = 0;
  s.retired.clear();
}

sq_status run_gemm(sq_handle h, int mode, const sq_weight *w, const void *a_ptr, const void *b_ptr, int64_t M,
                   void *out, const uint8_t *mask, cudaStream_t stream) {
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  CUtensorMap tmA, tmB, tmOut;
  const int64_t K2 = w->K / 2;  // code bytes per row
  if (mode == sqi::MODE_FWD) {
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->K, M, 64, sqi::kBM));  // X, 128 x 64 K-major boxes
    // codes: 128 rows x 64 bytes (128 weights) per stage and CTA of the pair, 64-byte swizzle
    SQ_TRY(make_map(h, &tmB, w->codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, K2, w->N, 64, 128,
                    CU_TENSOR_MAP_SWIZZLE_64B));
    // Y [M, N]: 32-row x 32-column store boxes (the epilogue's staging tiles), 64-byte swizzle
    SQ_TRY(make_out_map(h, &tmOut, out, w->N, M));
  } else if (mode == sqi::MODE_DX) {
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->N, M, 64, sqi::kBM));  // dY, 128 x 64 K-major boxes
    // codes: 128 contraction rows x 64 bytes (128 weights) per stage and CTA, 64-byte swizzle
    SQ_TRY(make_map(h, &tmB, w->codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, K2, w->N, 64, 128,
                    CU_TENSOR_MAP_SWIZZLE_64B));
    // dX [M, K]: the same store boxes
    SQ_TRY(make_out_map(h, &tmOut, out, w->K, M));
  } else {
    // dY and X as MN-major boxes of 64 features x kSgradBK tokens
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->N, M, 64, sqi::kSgradBK));
    SQ_TRY(make_act_map(h, &tmB, b_ptr, w->K, M, 64, sqi::kSgradBK));
  }
  sqi::GemmArgs a;
  a.mode = mode;
  a.fmt = w->fmt;
  a.M = M;
  a.N = w->N;
  a.K = w->K;
  a.codes = w->codes;
  a.scales = w->scales;
  a.ws2 = w->ws2;
  a.out = out;
  a.mask = mask;
  a.err = dev->err_word;
  if (mode == sqi::MODE_SGRAD) {
    a.splits = sgrad_splits_of(dev, w, M);
    if (a.splits > 1) {
      const size_t bytes = static_cast<size_t>(a.splits) * w->N * (w->K / block_of(w->fmt)) * sizeof(float);
      SQ_TRY(ensure_scratch(h, dev->partial, bytes, stream,
                            "the split scale gradient (sq_scale_grad_workspace reports the size)"));
      a.partial = static_cast<float *>(dev->partial.ptr);
    }
  }
  cudaError_t e = sqi::launch_gemm(a, tmA, tmB, mode == sqi::MODE_SGRAD ? nullptr : &tmOut, dev->sm_count, stream);
  if (e != cudaSuccess) return cuda_fail(h, e, "kernel launch");
  return SQ_OK;
}

// ------------------------------------------------------------------ multiplicative control

sq_status check_control(sq_handle h, const sq_control_weight *w, bool need_dS) {
  if (!w) return fail(h, SQ_ERR_INVALID_ARG, "control weight is NULL");
  if (w->N <= 0 || w->N % 8 != 0 || w->N > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "N=%d must be positive, a multiple of 8 and <= 2^24", w->N);
  if (w->K <= 0 || w->K % 32 != 0 || w->K > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "K=%d must be positive, a multiple of 32 and <= 2^24", w->K);
  if (!w->W || !aligned16(w->W)) return fail(h, SQ_ERR_INVALID_ARG, "W must be non-NULL and 16-byte aligned");
  if (need_dS && (!w->dS || !aligned16(w->dS)))
    return fail(h, SQ_ERR_INVALID_ARG, "dS must be non-NULL and 16-byte aligned");
  return SQ_OK;
}

// One control contraction: FWD a = X, out = Y; DX a = dY, out = dX; SGRAD a = dY, b = X, out = g.
sq_status run_control(sq_handle h, int mode, const sq_control_weight *w, const void *a_ptr, const void *b_ptr,
                      int64_t M, void *out, cudaStream_t stream) {
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  CUtensorMap tmA, tmB, tmOut;
  if (mode == sqi::MODE_FWD) {
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->K, M, 64, sqi::kBM));
    SQ_TRY(make_act_map(h, &tmB, w->W, w->K, w->N, 64, 128));  // W [N, K] in 64 x 128 boxes
    SQ_TRY(make_out_map(h, &tmOut, out, w->N, M));
  } else if (mode == sqi::MODE_DX) {
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->N, M, 64, sqi::kBM));
    SQ_TRY(make_act_map(h, &tmB, w->W, w->K, w->N, 64, 128));
    SQ_TRY(make_out_map(h, &tmOut, out, w->K, M));
  } else {
    SQ_TRY(make_act_map(h, &tmA, a_ptr, w->N, M, 64, sqi::kSgradBK));
    SQ_TRY(make_act_map(h, &tmB, b_ptr, w->K, M, 64, sqi::kSgradBK));
  }
  sqi::GemmArgs a;
  a.mode = mode;
  a.fmt = 2;
  a.M = M;
  a.N = w->N;
  a.K = w->K;
  a.codes = reinterpret_cast<const uint8_t *>(w->W);
  a.scales = reinterpret_cast<const uint8_t *>(w->dS);
  a.ws2 = 1.0f;
  a.out = out;
  a.mask = nullptr;
  a.err = dev->err_word;
  cudaError_t e = sqi::launch_control(a, tmA, tmB, mode == sqi::MODE_SGRAD ? nullptr : &tmOut, dev->sm_count, stream);
  if (e != cudaSuccess) return cuda_fail(h, e, "control kernel launch");
  return SQ_OK;
}

// ------------------------------------------------------------------ grouped (experts)

constexpr int kMaxExperts = 1 << 16;
constexpr int kMaxGridZ = 65535;  // experts of the adapter launches (grid z)

// Shape and tensor-scale checks of a grouped weight (codes and scales pointers
// only where the call reads them).
sq_status check_grouped_weight(sq_handle h, const sq_grouped_weight *w, bool need_codes, bool need_scales) {
  if (!w) return fail(h, SQ_ERR_INVALID_ARG, "grouped weight is NULL");
  if (w->E < 1 || w->E > kMaxExperts) return fail(h, SQ_ERR_INVALID_ARG, "E=%d must be in [1, 65536]", w->E);
  if (w->fmt != SQ_NVFP4 && w->fmt != SQ_MXFP4) return fail(h, SQ_ERR_INVALID_ARG, "unknown format %d", w->fmt);
  for (int e = 0; e < w->E; ++e) {
    const float ws2 = w->ws2 ? w->ws2[e] : 1.0f;
    if (w->fmt == SQ_NVFP4 && !w->ws2) return fail(h, SQ_ERR_INVALID_ARG, "NVFP4 experts need ws2[E]");
    if (w->fmt == SQ_NVFP4 && !(std::isfinite(ws2) && ws2 > 0.0f))
      return fail(h, SQ_ERR_INVALID_ARG, "ws2[%d] must be finite and > 0", e);
    if (w->fmt == SQ_MXFP4 && ws2 != 1.0f) return fail(h, SQ_ERR_INVALID_ARG, "MXFP4 ws2[%d] must be 1.0", e);
  }
  if (w->N <= 0 || w->N % 8 != 0 || w->N > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "N=%d must be positive, a multiple of 8 and <= 2^24", w->N);
  if (w->K <= 0 || w->K % 32 != 0 || w->K > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "K=%d must be positive, a multiple of 32 and <= 2^24", w->K);
  // code rows of all experts are addressed with int32 TMA coordinates (plus one tile of overhang)
  if (static_cast<int64_t>(w->E) * w->N + 1024 > kMaxTokens)
    return fail(h, SQ_ERR_INVALID_ARG, "E * N = %lld code rows exceed 2^31 - 1024", (long long)w->E * w->N);
  if (need_codes && (!w->codes || !aligned16(w->codes)))
    return fail(h, SQ_ERR_INVALID_ARG, "codes must be non-NULL and 16-byte aligned");
  if (need_scales && (!w->scales || !aligned16(w->scales)))
    return fail(h, SQ_ERR_INVALID_ARG, "scales must be non-NULL and 16-byte aligned");
  return SQ_OK;
}

// Weight and token-layout checks of a grouped contraction; on success `rows`
// holds each expert's token count and M the total.
sq_status check_grouped(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, bool need_scales,
                        std::vector<int64_t> &rows, int64_t &M) {
  SQ_TRY(check_grouped_weight(h, w, true, need_scales));
  if (!offsets) return fail(h, SQ_ERR_INVALID_ARG, "offsets is NULL");
  if (offsets[0] != 0) return fail(h, SQ_ERR_INVALID_ARG, "offsets[0] must be 0");
  rows.assign(w->E, 0);
  for (int e = 0; e < w->E; ++e) {
    if (offsets[e + 1] < offsets[e])
      return fail(h, SQ_ERR_INVALID_ARG, "offsets must be non-decreasing (offsets[%d] < offsets[%d])", e + 1, e);
    rows[e] = offsets[e + 1] - offsets[e];
  }
  M = offsets[w->E];
  return check_tokens(h, M);
}

// The next expert-table slot of the device, at least `bytes` large. Waits on the
// host for the launch that last read the slot (kTableSlots grouped calls back).
sq_status acquire_table(sq_handle h, DeviceState *dev, size_t bytes, TableSlot **out) {
  TableSlot &t = dev->tables[dev->next_table];
  dev->next_table = (dev->next_table + 1) % kTableSlots;
  cudaError_t e;
  if (!t.done && (e = cudaEventCreateWithFlags(&t.done, cudaEventDisableTiming)) != cudaSuccess)
    return cuda_fail(h, e, "cudaEventCreate(table)");
  if (t.pending) {
    if ((e = cudaEventSynchronize(t.done)) != cudaSuccess) return cuda_fail(h, e, "waiting for an expert table");
    t.pending = false;
  }
  if (bytes > t.bytes) {
    if (t.dev) cudaFree(t.dev);
    if (t.host) cudaFreeHost(t.host);
    t.dev = t.host = nullptr;
    t.bytes = 0;
    const size_t cap = (bytes + 65535) & ~size_t(65535);
    if ((e = cudaMalloc(&t.dev, cap)) != cudaSuccess) return cuda_fail(h, e, "cudaMalloc(expert table)");
    if ((e = cudaMallocHost(&t.host, cap)) != cudaSuccess) return cuda_fail(h, e, "cudaMallocHost(expert table)");
    t.bytes = cap;
  }
  *out = &t;
  return SQ_OK;
}

// One grouped contraction. FWD: a = X [M, K], out = Y [M, N]. DX: a = dY [M, N],
// out = dX [M, K]. SGRAD: a = dY, b = X, out = g [E, N, G].
// Grouped calls copy a host-built table on the stream: not while it is captured.
sq_status check_not_capturing(sq_handle h, cudaStream_t stream) {
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(stream, &cap);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaStreamIsCapturing");
  if (cap != cudaStreamCaptureStatusNone)
    return fail(h, SQ_ERR_UNSUPPORTED, "grouped calls copy a host-built expert table and cannot be graph-captured");
  return SQ_OK;
}

sq_status run_grouped(sq_handle h, int mode, const sq_grouped_weight *w, const std::vector<int64_t> &rows,
                      const int64_t *offsets, const uint16_t *a_ptr, const uint16_t *b_ptr, void *out,
                      const uint8_t *mask, cudaStream_t stream) {
  SQ_TRY(check_not_capturing(h, stream));
  cudaError_t e;
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const int E = w->E;
  const int64_t N = w->N, K = w->K;
  // the tile list: FWD / DX ceil(M_e / 512) row tiles of each expert x its column
  // tiles; SGRAD every expert's full (N / 256) x (K / 256) grid, empty experts included
  // table entry x holds expert order[x]: the scale gradient's units of one expert last
  // M_e tokens, so its entries go longest first; the other modes keep the experts' order
  std::vector<int> order(E);
  for (int x = 0; x < E; ++x) order[x] = x;
  if (mode == sqi::MODE_SGRAD)
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rows[a] > rows[b]; });
  std::vector<int32_t> tile_start(E + 1, 0);
  int64_t total = 0;
  if (mode == sqi::MODE_SGRAD) {
    const int64_t per = ((N + sqi::kSgradTile - 1) / sqi::kSgradTile) * ((K + sqi::kSgradTile - 1) / sqi::kSgradTile);
    for (int x = 0; x < E; ++x) {
      tile_start[x] = static_cast<int32_t>(total);
      total += per;
      if (total > kMaxTokens) return fail(h, SQ_ERR_INVALID_ARG, "too many tiles");
    }
  } else {
    const int64_t tn = ((mode == sqi::MODE_FWD ? N : K) + sqi::kPairNTile - 1) / sqi::kPairNTile;
    for (int x = 0; x < E; ++x) {
      tile_start[x] = static_cast<int32_t>(total);
      total += (rows[order[x]] + sqi::kPairMTile - 1) / sqi::kPairMTile * tn;
      if (total > kMaxTokens) return fail(h, SQ_ERR_INVALID_ARG, "too many tiles");
    }
  }
  tile_start[E] = static_cast<int32_t>(total);
  if (total == 0) return SQ_OK;

  TableSlot *t = nullptr;
  const size_t bytes = sqi::group_table_bytes(E);
  SQ_TRY(acquire_table(h, dev, bytes, &t));
  std::memset(t->host, 0, bytes);
  auto *maps = reinterpret_cast<sqi::GroupMaps *>(t->host);
  for (int x = 0; x < E; ++x) {
    const int ex = order[x];
    if (rows[ex] == 0) continue;  // no tiles read this expert's descriptors
    const int64_t m = rows[ex], r0 = offsets[ex];
    if (mode == sqi::MODE_FWD) {
      SQ_TRY(make_act_map(h, &maps[x].m[0], a_ptr + r0 * K, K, m, 64, sqi::kBM));
      SQ_TRY(make_out_map(h, &maps[x].m[1], static_cast<uint16_t *>(out) + r0 * N, N, m));
    } else if (mode == sqi::MODE_DX) {
      SQ_TRY(make_act_map(h, &maps[x].m[0], a_ptr + r0 * N, N, m, 64, sqi::kBM));
      SQ_TRY(make_out_map(h, &maps[x].m[1], static_cast<uint16_t *>(out) + r0 * K, K, m));
    } else {
      SQ_TRY(make_act_map(h, &maps[x].m[0], a_ptr + r0 * N, N, m, 64, sqi::kSgradBK));
      SQ_TRY(make_act_map(h, &maps[x].m[1], b_ptr + r0 * K, K, m, 64, sqi::kSgradBK));
    }
  }
  auto *ts = reinterpret_cast<int32_t *>(t->host + sqi::group_off_tiles(E));
  auto *rw = reinterpret_cast<int32_t *>(t->host + sqi::group_off_rows(E));
  auto *ws = reinterpret_cast<float *>(t->host + sqi::group_off_ws2(E));
  auto *id = reinterpret_cast<int32_t *>(t->host + sqi::group_off_ids(E));
  for (int x = 0; x <= E; ++x) ts[x] = tile_start[x];
  for (int x = 0; x < E; ++x) {
    rw[x] = static_cast<int32_t>(rows[order[x]]);
    ws[x] = w->ws2 ? w->ws2[order[x]] : 1.0f;
    id[x] = order[x];
  }
  // all experts' codes as one [E * N, K/2] tensor, the dense kernels' code boxes
  CUtensorMap tmCodes;
  SQ_TRY(make_map(h, &tmCodes, w->codes, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, K / 2, static_cast<int64_t>(E) * N, 64,
                  128, CU_TENSOR_MAP_SWIZZLE_64B));
  if ((e = cudaMemcpyAsync(t->dev, t->host, bytes, cudaMemcpyHostToDevice, stream)) != cudaSuccess)
    return cuda_fail(h, e, "copying the expert table");
  sqi::GroupedArgs ga;
  ga.mode = mode;
  ga.fmt = w->fmt;
  ga.E = E;
  ga.N = N;
  ga.K = K;
  ga.codes = w->codes;
  ga.scales = w->scales;
  ga.out = out;
  ga.mask = mask;
  ga.err = dev->err_word;
  ga.table = t->dev;
  ga.total_tiles = static_cast<int>(total);
  e = sqi::launch_grouped(ga, tmCodes, dev->sm_count, stream);
  // the slot is busy until the copy and the kernel complete (recorded even after a
  // failed launch, so the slot's next user waits only for the copy)
  cudaError_t e2 = cudaEventRecord(t->done, stream);
  if (e2 == cudaSuccess) t->pending = true;
  if (e != cudaSuccess) return cuda_fail(h, e, "grouped kernel launch");
  if (e2 != cudaSuccess) return cuda_fail(h, e2, "cudaEventRecord(table)");
  return SQ_OK;
}

// Projection (merge = false) or merge of the E experts' latent planes in one
// launch. MXFP4 experts share ws2 = 1; NVFP4 experts' tensor scales go to the
// device in an expert-table slot (one float per expert).
sq_status run_grouped_plane(sq_handle h, const sq_grouped_weight *w, bool merge, const float *latent, uint8_t *bytes,
                            uint8_t *mask_out, int32_t *nonfinite, float *delta, int64_t *changed,
                            cudaStream_t stream) {
  SQ_TRY(check_not_capturing(h, stream));
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const int64_t plane = static_cast<int64_t>(w->N) * (w->K / block_of(w->fmt));
  const int64_t count = plane * w->E;
  cudaError_t e;
  if (w->fmt == SQ_MXFP4) {
    e = merge ? sqi::launch_merge(w->fmt, count, 1.0f, latent, bytes, delta, changed, dev->sm_count, stream)
              : sqi::launch_project(w->fmt, count, 1.0f, latent, bytes, mask_out, nonfinite, dev->sm_count, stream);
    if (e != cudaSuccess) return cuda_fail(h, e, merge ? "grouped merge launch" : "grouped projection launch");
    return SQ_OK;
  }
  TableSlot *t = nullptr;
  const size_t tbytes = static_cast<size_t>(w->E) * sizeof(float);
  SQ_TRY(acquire_table(h, dev, tbytes, &t));
  std::memcpy(t->host, w->ws2, tbytes);
  if ((e = cudaMemcpyAsync(t->dev, t->host, tbytes, cudaMemcpyHostToDevice, stream)) != cudaSuccess)
    return cuda_fail(h, e, "copying the expert tensor scales");
  const float *ws2_dev = reinterpret_cast<const float *>(t->dev);
  e = merge ? sqi::launch_merge(w->fmt, count, 1.0f, latent, bytes, delta, changed, dev->sm_count, stream, ws2_dev,
                                plane)
            : sqi::launch_project(w->fmt, count, 1.0f, latent, bytes, mask_out, nonfinite, dev->sm_count, stream,
                                  ws2_dev, plane);
  cudaError_t e2 = cudaEventRecord(t->done, stream);
  if (e2 == cudaSuccess) t->pending = true;
  if (e != cudaSuccess) return cuda_fail(h, e, merge ? "grouped merge launch" : "grouped projection launch");
  if (e2 != cudaSuccess) return cuda_fail(h, e2, "cudaEventRecord(table)");
  return SQ_OK;
}

}  // namespace

extern "C" {

sq_status sq_create(sq_handle *out) {
  if (!out) return SQ_ERR_INVALID_ARG;
  try {
    *out = new sq_handle_s();
  } catch (...) {
    *out = nullptr;
    return SQ_ERR_CUDA;
  }
  return SQ_OK;
}

sq_status sq_destroy(sq_handle h) {
  if (!h) return SQ_ERR_INVALID_ARG;
  int cur = -1;
  cudaGetDevice(&cur);
  for (auto &d : h->devices) {
    if (cudaSetDevice(d.device) == cudaSuccess) {
      cudaFree(d.err_word);
      if (d.plane_acc) cudaFree(d.plane_acc);
      free_scratch(d.workspace);
      free_scratch(d.partial);
      for (auto &t : d.tables) {
        if (t.done) {
          cudaEventSynchronize(t.done);
          cudaEventDestroy(t.done);
        }
        if (t.dev) cudaFree(t.dev);
        if (t.host) cudaFreeHost(t.host);
      }
    }
  }
  if (cur >= 0) cudaSetDevice(cur);
  delete h;
  return SQ_OK;
}

const char *sq_status_string(sq_status s) {
  switch (s) {
    case SQ_OK: return "SQ_OK";
    case SQ_ERR_INVALID_ARG: return "SQ_ERR_INVALID_ARG";
    case SQ_ERR_UNSUPPORTED: return "SQ_ERR_UNSUPPORTED";
    case SQ_ERR_DEVICE: return "SQ_ERR_DEVICE";
    case SQ_ERR_CUDA: return "SQ_ERR_CUDA";
    case SQ_ERR_DEVICE_TIMEOUT: return "SQ_ERR_DEVICE_TIMEOUT";
  }
  return "SQ_ERR_UNKNOWN";
}

const char *sq_last_error(sq_handle h) { return h ? h->last_error.c_str() : "NULL handle"; }

sq_status sq_sync(sq_handle h, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaStreamSynchronize");
  int dev = -1;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return cuda_fail(h, e, "cudaGetDevice");
  for (auto &d : h->devices) {
    if (d.device != dev) continue;
    int word = 0;
    if ((e = cudaMemcpy(&word, d.err_word, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
      return cuda_fail(h, e, "reading the device error word");
    if (word != 0) {
      cudaMemset(d.err_word, 0, sizeof(int));
      return fail(h, SQ_ERR_DEVICE_TIMEOUT, "a bounded device wait ran out (error word 0x%x)", word);
    }
  }
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_selftest_wait_timeout(sq_handle h, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const cudaError_t e = sqi::launch_wait_probe(dev->err_word, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "launching the wait self-test");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_fwd(sq_handle h, const sq_weight *w, const uint16_t *X, int64_t M, uint16_t *Y, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_weight(h, w, true));
  SQ_TRY(check_tokens(h, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, Y, "Y"));
  return run_gemm(h, sqi::MODE_FWD, w, X, nullptr, M, Y, nullptr, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_bwd_dx(sq_handle h, const sq_weight *w, const uint16_t *dY, int64_t M, uint16_t *dX, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_weight(h, w, true));
  SQ_TRY(check_tokens(h, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, dY, "dY"));
  SQ_TRY(check_buf(h, dX, "dX"));
  return run_gemm(h, sqi::MODE_DX, w, dY, nullptr, M, dX, nullptr, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_scale_grad_workspace(sq_handle h, const sq_weight *w, int64_t M, int32_t *splits, int64_t *bytes) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_weight(h, w, false));
  SQ_TRY(check_tokens(h, M));
  if (!splits && !bytes) return fail(h, SQ_ERR_INVALID_ARG, "splits and bytes are both NULL");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const int s = M == 0 ? 1 : sgrad_splits_of(dev, w, M);
  if (splits) *splits = s;
  if (bytes) *bytes = s > 1 ? static_cast<int64_t>(s) * w->N * (w->K / block_of(w->fmt)) * 4 : 0;
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_scale_grad(sq_handle h, const sq_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                        const uint8_t *mask, float *g, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_weight(h, w, false));
  SQ_TRY(check_tokens(h, M));
  SQ_TRY(check_buf(h, g, "g"));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (M == 0) {
    DeviceState *dev = nullptr;
    SQ_TRY(ensure_device(h, &dev));
    const size_t bytes = static_cast<size_t>(w->N) * (w->K / block_of(w->fmt)) * sizeof(float);
    cudaError_t e = cudaMemsetAsync(g, 0, bytes, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(g)");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, dY, "dY"));
  return run_gemm(h, sqi::MODE_SGRAD, w, dY, X, M, g, mask, st);
  SQ_GUARD_END
}

static sq_status ensure_workspace(sq_handle h, DeviceState *dev, size_t bytes, cudaStream_t stream) {
  return ensure_scratch(h, dev->workspace, bytes, stream, "the adapter kernels");
}

static sq_status check_plane(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2) {
  SQ_TRY(check_ws2(h, fmt, ws2));
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  return SQ_OK;
}

sq_status sq_project_scales(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *latent,
                            uint8_t *bytes_out, uint8_t *mask_out, int32_t *nonfinite, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_plane(h, fmt, N, G, ws2));
  SQ_TRY(check_buf(h, latent, "latent"));
  SQ_TRY(check_buf(h, bytes_out, "bytes_out"));
  if (mask_out && !aligned16(mask_out)) return fail(h, SQ_ERR_INVALID_ARG, "mask_out must be 16-byte aligned");
  if (nonfinite && (reinterpret_cast<uintptr_t>(nonfinite) & 3u))
    return fail(h, SQ_ERR_INVALID_ARG, "nonfinite must be 4-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_project(fmt, N * G, ws2, latent, bytes_out, mask_out, nonfinite, dev->sm_count,
                                      static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "projection launch");
  return SQ_OK;
  SQ_GUARD_END
}

// Checks the plane table of a multi-plane call and fills the kernel's copy.
static sq_status planes_table(sq_handle h, int32_t fmt, int32_t nplanes, const sq_plane *planes, bool merge,
                              sqi::PlaneTable *t) {
  if (nplanes < 0 || nplanes > sqi::kMaxPlanes)
    return fail(h, SQ_ERR_INVALID_ARG, "nplanes=%d out of range [0, %d]", nplanes, sqi::kMaxPlanes);
  if (nplanes > 0 && !planes) return fail(h, SQ_ERR_INVALID_ARG, "planes is NULL");
  t->n = nplanes;
  for (int j = 0; j < nplanes; ++j) {
    const sq_plane &p = planes[j];
    SQ_TRY(check_plane(h, fmt, p.N, p.G, p.ws2));
    if ((p.N * p.G) % 16 != 0)
      return fail(h, SQ_ERR_INVALID_ARG, "plane %d: N * G = %lld is not a multiple of 16", j, (long long)(p.N * p.G));
    SQ_TRY(check_buf(h, p.latent, "plane latent"));
    SQ_TRY(check_buf(h, p.bytes, merge ? "plane scales" : "plane bytes"));
    if (!merge && p.mask && !aligned16(p.mask)) return fail(h, SQ_ERR_INVALID_ARG, "plane %d: mask must be 16-byte aligned", j);
    if (merge && p.ongrid_delta && !aligned16(p.ongrid_delta))
      return fail(h, SQ_ERR_INVALID_ARG, "plane %d: ongrid_delta must be 16-byte aligned", j);
    if (!merge && p.nonfinite && (reinterpret_cast<uintptr_t>(p.nonfinite) & 3u))
      return fail(h, SQ_ERR_INVALID_ARG, "plane %d: nonfinite must be 4-byte aligned", j);
    if (merge && p.changed_bytes && (reinterpret_cast<uintptr_t>(p.changed_bytes) & 7u))
      return fail(h, SQ_ERR_INVALID_ARG, "plane %d: changed_bytes must be 8-byte aligned", j);
    sqi::PlaneArgs &a = t->p[j];
    a.count = p.N * p.G;
    a.ws2 = p.ws2;
    a.latent = p.latent;
    a.bytes = p.bytes;
    a.mask = merge ? nullptr : p.mask;
    a.delta = merge ? p.ongrid_delta : nullptr;
    a.counter = merge ? static_cast<void *>(p.changed_bytes) : static_cast<void *>(p.nonfinite);
  }
  return SQ_OK;
}

sq_status sq_project_planes(sq_handle h, int32_t fmt, int32_t nplanes, const sq_plane *planes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  sqi::PlaneTable t{};
  SQ_TRY(planes_table(h, fmt, nplanes, planes, false, &t));
  if (nplanes == 0) return SQ_OK;
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_project_planes(fmt, t, dev->plane_acc, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "multi-plane projection launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_merge_planes(sq_handle h, int32_t fmt, int32_t nplanes, const sq_plane *planes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  sqi::PlaneTable t{};
  SQ_TRY(planes_table(h, fmt, nplanes, planes, true, &t));
  if (nplanes == 0) return SQ_OK;
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_merge_planes(fmt, t, dev->plane_acc, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "multi-plane merge launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_merge(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *latent,
                   uint8_t *scales_inout, float *ongrid_delta, int64_t *changed_bytes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_plane(h, fmt, N, G, ws2));
  SQ_TRY(check_buf(h, latent, "latent"));
  SQ_TRY(check_buf(h, scales_inout, "scales_inout"));
  if (ongrid_delta && !aligned16(ongrid_delta)) return fail(h, SQ_ERR_INVALID_ARG, "ongrid_delta must be 16-byte aligned");
  if (changed_bytes && (reinterpret_cast<uintptr_t>(changed_bytes) & 7u))
    return fail(h, SQ_ERR_INVALID_ARG, "changed_bytes must be 8-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_merge(fmt, N * G, ws2, latent, scales_inout, ongrid_delta, changed_bytes, dev->sm_count,
                                    static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "merge launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_rollback(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *ongrid_delta,
                      uint8_t *scales_inout, int64_t *changed_bytes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_plane(h, fmt, N, G, ws2));
  if (N * G > 0) {
    SQ_TRY(check_buf(h, ongrid_delta, "ongrid_delta"));
    SQ_TRY(check_buf(h, scales_inout, "scales_inout"));
  }
  if (changed_bytes && (reinterpret_cast<uintptr_t>(changed_bytes) & 7u))
    return fail(h, SQ_ERR_INVALID_ARG, "changed_bytes must be 8-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_rollback(fmt, N * G, ws2, ongrid_delta, scales_inout, changed_bytes, dev->sm_count,
                                       static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "rollback launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_swap_scales(sq_handle h, int64_t N, int64_t G, const uint8_t *src, uint8_t *scales_inout,
                         int64_t *changed_bytes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  if (N * G > 0) {
    SQ_TRY(check_buf(h, src, "src"));
    SQ_TRY(check_buf(h, scales_inout, "scales_inout"));
  }
  if (changed_bytes && (reinterpret_cast<uintptr_t>(changed_bytes) & 7u))
    return fail(h, SQ_ERR_INVALID_ARG, "changed_bytes must be 8-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_swap_or_diff(N * G, src, scales_inout, true, changed_bytes, dev->sm_count,
                                           static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "swap launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_count_diff(sq_handle h, const uint8_t *a, const uint8_t *b, int64_t nbytes, int64_t *count,
                        void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (nbytes < 0 || nbytes > (int64_t(1) << 40)) return fail(h, SQ_ERR_INVALID_ARG, "nbytes out of range");
  if (nbytes > 0) {
    SQ_TRY(check_buf(h, a, "a"));
    SQ_TRY(check_buf(h, b, "b"));
  }
  if (!count || (reinterpret_cast<uintptr_t>(count) & 7u))
    return fail(h, SQ_ERR_INVALID_ARG, "count must be non-NULL and 8-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  cudaError_t e = sqi::launch_swap_or_diff(nbytes, a, const_cast<uint8_t *>(b), false, count, dev->sm_count,
                                           static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "audit launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_project_lowrank(sq_handle h, int32_t fmt, int64_t N, int64_t G, int32_t r, float ws2, float alpha_over_r,
                             const uint8_t *base_scales, const uint16_t *B, const uint16_t *A, uint8_t *bytes_out,
                             uint8_t *mask_out, int32_t *nonfinite, float *latent_out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_plane(h, fmt, N, G, ws2));
  if (r < 1 || r > sqi::kMaxLowRank) return fail(h, SQ_ERR_INVALID_ARG, "rank r=%d must be in [1, 256]", r);
  if (!std::isfinite(alpha_over_r)) return fail(h, SQ_ERR_INVALID_ARG, "alpha_over_r must be finite");
  if (nonfinite && (reinterpret_cast<uintptr_t>(nonfinite) & 3u))
    return fail(h, SQ_ERR_INVALID_ARG, "nonfinite must be 4-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (N == 0 || G == 0) {  // empty plane: the arrays may be NULL
    if (nonfinite && (e = cudaMemsetAsync(nonfinite, 0, sizeof(int32_t), st)) != cudaSuccess)
      return cuda_fail(h, e, "cudaMemsetAsync");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, base_scales, "base_scales"));
  SQ_TRY(check_buf(h, B, "B"));
  SQ_TRY(check_buf(h, A, "A"));
  SQ_TRY(check_buf(h, bytes_out, "bytes_out"));
  if (mask_out && !aligned16(mask_out)) return fail(h, SQ_ERR_INVALID_ARG, "mask_out must be 16-byte aligned");
  if (latent_out && !aligned16(latent_out)) return fail(h, SQ_ERR_INVALID_ARG, "latent_out must be 16-byte aligned");
  e = sqi::launch_project_lowrank(fmt, N, G, r, ws2, alpha_over_r, base_scales, B, A, bytes_out, mask_out, nonfinite,
                                  latent_out, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "adapter projection launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_lowrank_grad(sq_handle h, int64_t N, int64_t G, int32_t r, float alpha_over_r, const float *g,
                          const uint16_t *B, const uint16_t *A, float *dB, float *dA, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  if (r < 1 || r > sqi::kMaxLowRank) return fail(h, SQ_ERR_INVALID_ARG, "rank r=%d must be in [1, 256]", r);
  if (!std::isfinite(alpha_over_r)) return fail(h, SQ_ERR_INVALID_ARG, "alpha_over_r must be finite");
  if (!dB && !dA) return fail(h, SQ_ERR_INVALID_ARG, "dB and dA are both NULL");
  // dB [N, r] is non-empty iff N > 0 and dA [r, G] iff G > 0; g, B, A are read only when N, G > 0
  if (dB && N > 0 && !aligned16(dB)) return fail(h, SQ_ERR_INVALID_ARG, "dB must be non-NULL and 16-byte aligned");
  if (dA && G > 0 && !aligned16(dA)) return fail(h, SQ_ERR_INVALID_ARG, "dA must be non-NULL and 16-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (N == 0 || G == 0) {  // empty sums: the gradients are zero
    if (dB && N > 0 && (e = cudaMemsetAsync(dB, 0, static_cast<size_t>(N) * r * sizeof(float), st)) != cudaSuccess)
      return cuda_fail(h, e, "cudaMemsetAsync");
    if (dA && G > 0 && (e = cudaMemsetAsync(dA, 0, static_cast<size_t>(G) * r * sizeof(float), st)) != cudaSuccess)
      return cuda_fail(h, e, "cudaMemsetAsync");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, g, "g"));
  SQ_TRY(check_buf(h, B, "B"));
  SQ_TRY(check_buf(h, A, "A"));
  SQ_TRY(ensure_workspace(h, dev, sqi::lowrank_grad_workspace(N, G, r, dev->sm_count), st));
  e = sqi::launch_lowrank_grad(N, G, r, alpha_over_r, g, B, A, dB, dA, static_cast<float *>(dev->workspace.ptr),
                               dev->sm_count, st, dev->err_word);
  if (e != cudaSuccess) return cuda_fail(h, e, "adapter gradient launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_fit_scale_delta(sq_handle h, int32_t fmt, int64_t N, int64_t K, float ws2, const uint8_t *codes,
                             const uint8_t *scales, const uint16_t *dW, float *delta_out, float *captured_out,
                             float *total_out, float *latent_out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_ws2(h, fmt, ws2));
  if (N < 0 || N > kMaxDim || K < 0 || K % 32 != 0 || K > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "shape [%lld, %lld]: N in [0, 2^24], K a multiple of 32 in [0, 2^24]",
                (long long)N, (long long)K);
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  if (N == 0 || K == 0) return SQ_OK;
  SQ_TRY(check_buf(h, codes, "codes"));
  SQ_TRY(check_buf(h, dW, "dW"));
  SQ_TRY(check_buf(h, delta_out, "delta_out"));
  if (captured_out && !aligned16(captured_out)) return fail(h, SQ_ERR_INVALID_ARG, "captured_out must be 16-byte aligned");
  if (total_out && !aligned16(total_out)) return fail(h, SQ_ERR_INVALID_ARG, "total_out must be 16-byte aligned");
  if (latent_out) {
    if (!aligned16(latent_out)) return fail(h, SQ_ERR_INVALID_ARG, "latent_out must be 16-byte aligned");
    SQ_TRY(check_buf(h, scales, "scales (needed for latent_out)"));
  }
  cudaError_t e = sqi::launch_fit(fmt, N, K, ws2, codes, scales, dW, delta_out, captured_out, total_out, latent_out,
                                  dev->sm_count, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "fit launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_group_reduce(sq_handle h, int64_t N, int64_t G, int64_t gd, const float *g, float *out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  if (gd < 1 || (G > 0 && (gd > G || G % gd != 0)))
    return fail(h, SQ_ERR_INVALID_ARG, "gd=%lld must be >= 1 and divide G=%lld", (long long)gd, (long long)G);
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  if (N == 0 || G == 0) return SQ_OK;
  SQ_TRY(check_buf(h, g, "g"));
  SQ_TRY(check_buf(h, out, "out"));
  cudaError_t e = sqi::launch_group_reduce(N, G, gd, g, out, dev->sm_count, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "group reduction launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_project_group_delta(sq_handle h, int32_t fmt, int64_t N, int64_t G, int64_t gd, float ws2,
                                 const uint8_t *base_scales, const float *delta, uint8_t *bytes_out, uint8_t *mask_out,
                                 int32_t *nonfinite, float *latent_out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_plane(h, fmt, N, G, ws2));
  if (gd < 1 || (G > 0 && (gd > G || G % gd != 0)))
    return fail(h, SQ_ERR_INVALID_ARG, "gd=%lld must be >= 1 and divide G=%lld", (long long)gd, (long long)G);
  if (nonfinite && (reinterpret_cast<uintptr_t>(nonfinite) & 3u))
    return fail(h, SQ_ERR_INVALID_ARG, "nonfinite must be 4-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (N > 0 && G > 0) {
    SQ_TRY(check_buf(h, base_scales, "base_scales"));
    SQ_TRY(check_buf(h, delta, "delta"));
    SQ_TRY(check_buf(h, bytes_out, "bytes_out"));
    if (mask_out && !aligned16(mask_out)) return fail(h, SQ_ERR_INVALID_ARG, "mask_out must be 16-byte aligned");
    if (latent_out && !aligned16(latent_out)) return fail(h, SQ_ERR_INVALID_ARG, "latent_out must be 16-byte aligned");
  }
  cudaError_t e = sqi::launch_project_group_delta(fmt, N, G, gd, ws2, base_scales, delta, bytes_out, mask_out,
                                                  nonfinite, latent_out, dev->sm_count, st);
  if (e != cudaSuccess) return cuda_fail(h, e, "group-delta projection launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_control_fwd(sq_handle h, const sq_control_weight *w, const uint16_t *X, int64_t M, uint16_t *Y,
                         void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_control(h, w, true));
  SQ_TRY(check_tokens(h, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, Y, "Y"));
  return run_control(h, sqi::MODE_FWD, w, X, nullptr, M, Y, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_control_bwd_dx(sq_handle h, const sq_control_weight *w, const uint16_t *dY, int64_t M, uint16_t *dX,
                            void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_control(h, w, true));
  SQ_TRY(check_tokens(h, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, dY, "dY"));
  SQ_TRY(check_buf(h, dX, "dX"));
  return run_control(h, sqi::MODE_DX, w, dY, nullptr, M, dX, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_control_grad(sq_handle h, const sq_control_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                          float *g, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_control(h, w, false));
  SQ_TRY(check_tokens(h, M));
  SQ_TRY(check_buf(h, g, "g"));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (M == 0) {
    DeviceState *dev = nullptr;
    SQ_TRY(ensure_device(h, &dev));
    cudaError_t e = cudaMemsetAsync(g, 0, static_cast<size_t>(w->N) * (w->K / 16) * sizeof(float), st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(g)");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, dY, "dY"));
  return run_control(h, sqi::MODE_SGRAD, w, dY, X, M, g, st);
  SQ_GUARD_END
}

sq_status sq_lowrank_product(sq_handle h, int64_t N, int64_t G, int32_t r, float alpha_over_r, const uint16_t *B,
                             const uint16_t *A, float *out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  if (r < 1 || r > sqi::kMaxLowRank) return fail(h, SQ_ERR_INVALID_ARG, "rank r=%d must be in [1, 256]", r);
  if (!std::isfinite(alpha_over_r)) return fail(h, SQ_ERR_INVALID_ARG, "alpha_over_r must be finite");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  if (N == 0 || G == 0) return SQ_OK;
  SQ_TRY(check_buf(h, B, "B"));
  SQ_TRY(check_buf(h, A, "A"));
  SQ_TRY(check_buf(h, out, "out"));
  SQ_TRY(ensure_workspace(h, dev, sqi::lowrank_product_workspace(N, G, r, dev->sm_count),
                          static_cast<cudaStream_t>(stream)));
  cudaError_t e = sqi::launch_lowrank_product(N, G, r, alpha_over_r, B, A, out, static_cast<float *>(dev->workspace.ptr),
                                              dev->sm_count, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(h, e, "low-rank product launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_grouped_fwd(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *X,
                         uint16_t *Y, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  std::vector<int64_t> rows;
  int64_t M = 0;
  SQ_TRY(check_grouped(h, w, offsets, true, rows, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, Y, "Y"));
  return run_grouped(h, sqi::MODE_FWD, w, rows, offsets, X, nullptr, Y, nullptr, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_grouped_bwd_dx(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *dY,
                            uint16_t *dX, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  std::vector<int64_t> rows;
  int64_t M = 0;
  SQ_TRY(check_grouped(h, w, offsets, true, rows, M));
  if (M == 0) return SQ_OK;
  SQ_TRY(check_buf(h, dY, "dY"));
  SQ_TRY(check_buf(h, dX, "dX"));
  return run_grouped(h, sqi::MODE_DX, w, rows, offsets, dY, nullptr, dX, nullptr, static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_grouped_project_scales(sq_handle h, const sq_grouped_weight *w, const float *latent, uint8_t *bytes_out,
                                    uint8_t *mask_out, int32_t *nonfinite, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_grouped_weight(h, w, false, false));
  SQ_TRY(check_buf(h, latent, "latent"));
  SQ_TRY(check_buf(h, bytes_out, "bytes_out"));
  if (mask_out && !aligned16(mask_out)) return fail(h, SQ_ERR_INVALID_ARG, "mask_out must be 16-byte aligned");
  if (nonfinite && (reinterpret_cast<uintptr_t>(nonfinite) & 3u))
    return fail(h, SQ_ERR_INVALID_ARG, "nonfinite must be 4-byte aligned");
  return run_grouped_plane(h, w, false, latent, bytes_out, mask_out, nonfinite, nullptr, nullptr,
                           static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_grouped_merge(sq_handle h, const sq_grouped_weight *w, const float *latent, uint8_t *scales_inout,
                           float *ongrid_delta, int64_t *changed_bytes, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_grouped_weight(h, w, false, false));
  SQ_TRY(check_buf(h, latent, "latent"));
  SQ_TRY(check_buf(h, scales_inout, "scales_inout"));
  if (ongrid_delta && !aligned16(ongrid_delta)) return fail(h, SQ_ERR_INVALID_ARG, "ongrid_delta must be 16-byte aligned");
  if (changed_bytes && (reinterpret_cast<uintptr_t>(changed_bytes) & 7u))
    return fail(h, SQ_ERR_INVALID_ARG, "changed_bytes must be 8-byte aligned");
  return run_grouped_plane(h, w, true, latent, scales_inout, nullptr, nullptr, ongrid_delta, changed_bytes,
                           static_cast<cudaStream_t>(stream));
  SQ_GUARD_END
}

sq_status sq_grouped_project_lowrank(sq_handle h, const sq_grouped_weight *w, int32_t r, float alpha_over_r,
                                     const uint16_t *B, const uint16_t *A, uint8_t *bytes_out, uint8_t *mask_out,
                                     int32_t *nonfinite, float *latent_out, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  SQ_TRY(check_grouped_weight(h, w, false, true));
  if (w->E > kMaxGridZ) return fail(h, SQ_ERR_INVALID_ARG, "E=%d exceeds 65535 for the adapter launches", w->E);
  if (r < 1 || r > sqi::kMaxLowRank) return fail(h, SQ_ERR_INVALID_ARG, "rank r=%d must be in [1, 256]", r);
  if (!std::isfinite(alpha_over_r)) return fail(h, SQ_ERR_INVALID_ARG, "alpha_over_r must be finite");
  SQ_TRY(check_buf(h, B, "B"));
  SQ_TRY(check_buf(h, A, "A"));
  SQ_TRY(check_buf(h, bytes_out, "bytes_out"));
  if (mask_out && !aligned16(mask_out)) return fail(h, SQ_ERR_INVALID_ARG, "mask_out must be 16-byte aligned");
  if (latent_out && !aligned16(latent_out)) return fail(h, SQ_ERR_INVALID_ARG, "latent_out must be 16-byte aligned");
  if (nonfinite && (reinterpret_cast<uintptr_t>(nonfinite) & 3u))
    return fail(h, SQ_ERR_INVALID_ARG, "nonfinite must be 4-byte aligned");
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  SQ_TRY(check_not_capturing(h, st));
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const int64_t N = w->N, G = w->K / block_of(w->fmt);
  cudaError_t e;
  if (w->fmt == SQ_MXFP4) {
    e = sqi::launch_project_lowrank(w->fmt, N, G, r, 1.0f, alpha_over_r, w->scales, B, A, bytes_out, mask_out,
                                    nonfinite, latent_out, st, w->E, nullptr);
    if (e != cudaSuccess) return cuda_fail(h, e, "grouped adapter projection launch");
    return SQ_OK;
  }
  TableSlot *t = nullptr;
  const size_t tbytes = static_cast<size_t>(w->E) * sizeof(float);
  SQ_TRY(acquire_table(h, dev, tbytes, &t));
  std::memcpy(t->host, w->ws2, tbytes);
  if ((e = cudaMemcpyAsync(t->dev, t->host, tbytes, cudaMemcpyHostToDevice, st)) != cudaSuccess)
    return cuda_fail(h, e, "copying the expert tensor scales");
  e = sqi::launch_project_lowrank(w->fmt, N, G, r, 1.0f, alpha_over_r, w->scales, B, A, bytes_out, mask_out,
                                  nonfinite, latent_out, st, w->E, reinterpret_cast<const float *>(t->dev));
  cudaError_t e2 = cudaEventRecord(t->done, st);
  if (e2 == cudaSuccess) t->pending = true;
  if (e != cudaSuccess) return cuda_fail(h, e, "grouped adapter projection launch");
  if (e2 != cudaSuccess) return cuda_fail(h, e2, "cudaEventRecord(table)");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_grouped_lowrank_grad(sq_handle h, int32_t E, int64_t N, int64_t G, int32_t r, float alpha_over_r,
                                  const float *g, const uint16_t *B, const uint16_t *A, float *dB, float *dA,
                                  void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  if (E < 1 || E > kMaxGridZ) return fail(h, SQ_ERR_INVALID_ARG, "E=%d must be in [1, 65535]", E);
  if (N < 0 || G < 0 || N > kMaxDim || G > kMaxDim)
    return fail(h, SQ_ERR_INVALID_ARG, "plane shape [%lld, %lld] out of range", (long long)N, (long long)G);
  if (r < 1 || r > sqi::kMaxLowRank) return fail(h, SQ_ERR_INVALID_ARG, "rank r=%d must be in [1, 256]", r);
  if (!std::isfinite(alpha_over_r)) return fail(h, SQ_ERR_INVALID_ARG, "alpha_over_r must be finite");
  if (!dB && !dA) return fail(h, SQ_ERR_INVALID_ARG, "dB and dA are both NULL");
  if (dB && N > 0 && !aligned16(dB)) return fail(h, SQ_ERR_INVALID_ARG, "dB must be non-NULL and 16-byte aligned");
  if (dA && G > 0 && !aligned16(dA)) return fail(h, SQ_ERR_INVALID_ARG, "dA must be non-NULL and 16-byte aligned");
  DeviceState *dev = nullptr;
  SQ_TRY(ensure_device(h, &dev));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (N == 0 || G == 0) {  // empty sums: the gradients are zero
    if (dB && N > 0 &&
        (e = cudaMemsetAsync(dB, 0, static_cast<size_t>(E) * N * r * sizeof(float), st)) != cudaSuccess)
      return cuda_fail(h, e, "cudaMemsetAsync");
    if (dA && G > 0 &&
        (e = cudaMemsetAsync(dA, 0, static_cast<size_t>(E) * G * r * sizeof(float), st)) != cudaSuccess)
      return cuda_fail(h, e, "cudaMemsetAsync");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, g, "g"));
  SQ_TRY(check_buf(h, B, "B"));
  SQ_TRY(check_buf(h, A, "A"));
  SQ_TRY(ensure_workspace(h, dev, sqi::lowrank_grad_workspace(N, G, r, dev->sm_count, E), st));
  e = sqi::launch_lowrank_grad(N, G, r, alpha_over_r, g, B, A, dB, dA, static_cast<float *>(dev->workspace.ptr),
                               dev->sm_count, st, dev->err_word, E);
  if (e != cudaSuccess) return cuda_fail(h, e, "grouped adapter gradient launch");
  return SQ_OK;
  SQ_GUARD_END
}

sq_status sq_grouped_scale_grad(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *X,
                                const uint16_t *dY, const uint8_t *mask, float *g, void *stream) {
  if (!h) return SQ_ERR_INVALID_ARG;
  SQ_GUARD_BEGIN
  std::vector<int64_t> rows;
  int64_t M = 0;
  SQ_TRY(check_grouped(h, w, offsets, false, rows, M));
  SQ_TRY(check_buf(h, g, "g"));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (M == 0) {  // every sum is empty
    DeviceState *dev = nullptr;
    SQ_TRY(ensure_device(h, &dev));
    const size_t bytes = static_cast<size_t>(w->E) * w->N * (w->K / block_of(w->fmt)) * sizeof(float);
    cudaError_t e = cudaMemsetAsync(g, 0, bytes, st);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaMemsetAsync(g)");
    return SQ_OK;
  }
  SQ_TRY(check_buf(h, X, "X"));
  SQ_TRY(check_buf(h, dY, "dY"));
  return run_grouped(h, sqi::MODE_SGRAD, w, rows, offsets, dY, X, g, mask, st);
  SQ_GUARD_END
}

}  // extern "C"
