/*
 * scaleqlora.h -- C ABI of the GB300 (sm_103a) hot path of Scale-QLoRA's
 * scale-only training step (arXiv 2609.04526).
 *
 * The E2M1 code plane of a native FP4 checkpoint is frozen; only the per-block
 * scales train. Per linear layer with weight W[N=out, K=in]:
 *   sq_fwd             Y  = X . W^T                        (Sec. 3 "Scale-QLoRA forward")
 *   sq_bwd_dx          dX = dY . W                         (backward of that forward)
 *   sq_scale_grad      g[n,b] = sum_{k in b} code[n,k] (dY^T X)[n,k]   (optionally x mask)
 *   sq_project_scales  latent scale -> on-grid E4M3 / E8M0 byte + STE mask (Sec. 3 QAST, clamp)
 *   sq_merge           write on-grid bytes into the scale plane; never a code (Sec. 3, Sec. 5)
 *   sq_project_lowrank the low-rank adapter's latent eff + (alpha/r) B A, projected (Sec. 3)
 *   sq_lowrank_grad    gradients of the adapter factors B and A from the masked scale gradient
 *   sq_rollback        undo a merge with its on-grid delta (Sec. 5 Payoff 3)
 *   sq_swap_scales     scale-only hot-swap of the served adapter (Sec. 5)
 *   sq_count_diff      byte-level audit of two buffers (Sec. 5)
 *   sq_grouped_*       the contractions, projection, merge and adapters over the experts of
 *                      an MoE linear, one launch each (Sec. 3)
 *   sq_fit_scale_delta, sq_group_reduce, sq_project_group_delta, sq_control_*,
 *   sq_lowrank_product scale-family variants of the ablation appendix
 * with W[n,k] = code[n,k] * s[n, k / B] decoded on the fly, where (Sec. 2)
 *   NVFP4: B = 16, s = E4M3(scale byte) * ws2 (fp32 tensor scale)
 *   MXFP4: B = 32, s = E8M0(scale byte) = 2^(byte - 127), ws2 must be 1.0
 *
 * Conventions for every entry point
 *  - Pointers named as device buffers are device pointers owned by the caller;
 *    the library never frees or keeps them. Calls are asynchronous on `stream`
 *    (a cudaStream_t passed as void*, NULL = the legacy default stream) and
 *    return once the work is enqueued.
 *  - Layouts are dense row-major. bf16 tensors are passed as uint16_t bit patterns.
 *  - codes [N, K/2] u8: element k of row n is nibble (k & 1) of byte k/2, the even
 *    k in the low nibble. scales [N, K/B] u8.
 *  - Shape rules: N > 0 with N % 8 == 0; K > 0 with K % 32 == 0; M >= 0 (M == 0
 *    is an empty batch). Every device pointer must be 16-byte aligned.
 *  - Argument errors return SQ_ERR_INVALID_ARG before anything is launched; the
 *    text is in sq_last_error(h). No exception or abort crosses the ABI.
 *  - A handle is not thread-safe; use one handle per host thread. The scratch a
 *    handle owns (a split scale gradient's partial planes; the adapter kernels'
 *    partial sums) is one buffer per kind and device: calls of one handle that
 *    use it must run on one stream or be ordered by the caller. It is allocated,
 *    or grown, by the first call that needs it; a call that would grow it while
 *    its stream is being captured into a CUDA graph returns SQ_ERR_UNSUPPORTED,
 *    so make one call outside the capture first. A buffer that a capture has
 *    used is never freed while the handle lives: when a later call grows it,
 *    the old buffer is kept (and freed by sq_destroy), so graphs captured
 *    earlier replay correctly until the handle is destroyed. Grouped calls that
 *    take an sq_grouped_weight copy a host-built expert table and cannot be
 *    captured.
 *  - Device waits are bounded: a wait that runs out sets a device error word
 *    instead of hanging; sq_sync reports it as SQ_ERR_DEVICE_TIMEOUT.
 *  - Decoded weights are formed exactly in bf16 (the code x scale-byte product
 *    has at most 6 significant bits); for MXFP4 this holds for scale bytes 2..252
 *    (decoded magnitudes within bf16's normal range).
 */
#ifndef SCALEQLORA_H
#define SCALEQLORA_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SQ_NVFP4 = 0, /* block 16, E4M3 scale byte times an fp32 tensor scale ws2 */
  SQ_MXFP4 = 1  /* block 32, E8M0 power-of-two scale byte */
} sq_format;

typedef enum {
  SQ_OK = 0,
  SQ_ERR_INVALID_ARG = -1,    /* bad pointer, alignment, shape or scalar          */
  SQ_ERR_UNSUPPORTED = -2,    /* current device is not compute capability 10.3    */
  SQ_ERR_DEVICE = -3,         /* no usable CUDA device / driver entry point        */
  SQ_ERR_CUDA = -4,           /* a CUDA runtime call or launch failed             */
  SQ_ERR_DEVICE_TIMEOUT = -5  /* a bounded device-side wait ran out (see sq_sync)  */
} sq_status;

/* Opaque per-thread context: last error text, device properties, the device
 * error word. */
typedef struct sq_handle_s *sq_handle;

/* One quantized linear, weight [N = out features, K = in features]. */
typedef struct {
  int32_t fmt;           /* sq_format                                           */
  int32_t N;             /* out features, N % 8 == 0                            */
  int32_t K;             /* in features,  K % 32 == 0                           */
  const uint8_t *codes;  /* device [N, K/2]: packed E2M1 codes                  */
  const uint8_t *scales; /* device [N, K/B]: E4M3 (NVFP4) or E8M0 (MXFP4) bytes */
  float ws2;             /* NVFP4: finite and > 0; MXFP4: exactly 1.0           */
} sq_weight;

/* Create / destroy a handle. sq_create makes no CUDA call; the device is
 * queried on the first compute call. */
sq_status sq_create(sq_handle *out);
sq_status sq_destroy(sq_handle h);

/* Static text for a status code; never NULL. */
const char *sq_status_string(sq_status s);
/* Text of the last error on this handle ("" if none). Valid until the next call. */
const char *sq_last_error(sq_handle h);

/* Synchronise `stream` and report device-side wait timeouts raised since the
 * previous sq_sync on this handle's device (then clear them).
 * Returns SQ_OK, SQ_ERR_DEVICE_TIMEOUT or SQ_ERR_CUDA. */
sq_status sq_sync(sq_handle h, void *stream);

/* Self-test of the failure path: launches one thread that waits on a shared-
 * memory barrier nothing arrives on, with the bounded wait every contraction
 * kernel uses (1 s); when it runs out the thread records the timeout in the
 * device error word and returns, so the context stays usable. The next sq_sync
 * on `stream` returns SQ_ERR_DEVICE_TIMEOUT (and clears the word). Returns
 * SQ_OK once enqueued, SQ_ERR_UNSUPPORTED / SQ_ERR_CUDA as the compute calls. */
sq_status sq_selftest_wait_timeout(sq_handle h, void *stream);

/* Forward, Sec. 3 "Scale-QLoRA forward": Y[m,n] = sum_k X[m,k] W[n,k].
 * X  device bf16 [M, K] (input), Y device bf16 [M, N] (output, overwritten).
 * Accumulation in fp32; ws2 is applied to the fp32 accumulator; Y is rounded
 * to nearest-even bf16. */
sq_status sq_fwd(sq_handle h, const sq_weight *w, const uint16_t *X, int64_t M, uint16_t *Y, void *stream);

/* Input gradient of the forward: dX[m,k] = sum_n dY[m,n] W[n,k].
 * dY device bf16 [M, N] (input), dX device bf16 [M, K] (output). fp32 accumulation. */
sq_status sq_bwd_dx(sq_handle h, const sq_weight *w, const uint16_t *dY, int64_t M, uint16_t *dX, void *stream);

/* Scale gradient with respect to the effective scale s[n,b] (absolute units):
 *   g[n,b] = mask[n,b] * sum_{k in block b} code[n,k] * sum_m dY[m,n] X[m,k]
 * The derivative of sum(Y * dY) by s[n,b] under the forward above (Sec. 3), with
 * the QAST straight-through estimator passing it unchanged through the grid
 * rounding and the clamp zeroing it where the latent is outside the clamp
 * (mask from sq_project_scales; NULL means all ones). The gradient of the
 * latent in E4M3 units is g * ws2 (not computed here).
 * X device bf16 [M, K], dY device bf16 [M, N], mask device u8 [N, K/B] or NULL,
 * g device fp32 [N, K/B] (output, overwritten; all zero when M == 0). The
 * weight's scale bytes are not read (w->scales may be NULL).
 * The dW = dY^T X tile is reduced per block on chip and never written.
 * A weight with few 256 x 256 tiles (fewer than a handful of waves over the
 * GPU's SMs) has its M tokens cut into up to 8 parts: each part's unmasked
 * partial gradient goes to scratch the handle owns, and a second kernel adds
 * the parts in order and applies the mask (deterministic; the fp32 sums round
 * differently from an unsplit launch). The scratch is allocated, or grown, on
 * the first call that needs it (cudaMalloc, which may synchronise the device);
 * sq_scale_grad_workspace reports the split and the scratch size. A call that
 * would have to grow the scratch while `stream` is being captured into a CUDA
 * graph returns SQ_ERR_UNSUPPORTED instead: size it with one call outside the
 * capture, after which captured calls allocate nothing. */
sq_status sq_scale_grad(sq_handle h, const sq_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                        const uint8_t *mask, float *g, void *stream);

/* The token split sq_scale_grad uses for this weight shape and M on the current
 * device: *splits (host, nullable) = the number of parts (1 = a single launch, no
 * scratch), *bytes (host, nullable) = the handle scratch it needs, splits * N * (K/B)
 * * 4 (0 when unsplit). Host-only; returns SQ_ERR_INVALID_ARG for a bad shape. */
sq_status sq_scale_grad_workspace(sq_handle h, const sq_weight *w, int64_t M, int32_t *splits, int64_t *bytes);

/* Grid projection, Sec. 3 QAST round_grid with the ceiling clamp of the
 * stability recipe (ii)/(iii), for count = N*G latent scales (absolute units):
 *  NVFP4: cap = fl32(448*ws2); q = fl32(clamp(L, -cap, cap) / ws2);
 *         byte = E4M3 nearest to q, ties to even (sign kept, -0 -> 0x80);
 *         mask = 1 iff -cap <= L <= cap; NaN -> 0x7F with mask 0.
 *  MXFP4: byte = round(log2 L) + 127 with the rounding at sqrt(2) * 2^E, clamped
 *         to [0, 254] (mask 0 when clamped); L <= 0 -> 0 with mask 0;
 *         +inf -> 254 with mask 0; NaN -> 0xFF with mask 0.
 * latent device fp32 [N, G]; bytes_out device u8 [N, G]; mask_out device u8
 * [N, G] or NULL; nonfinite device int32 or NULL: set to the number of NaN
 * latents (written on `stream`). */
sq_status sq_project_scales(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *latent,
                            uint8_t *bytes_out, uint8_t *mask_out, int32_t *nonfinite, void *stream);

/* Merge, Sec. 3 "QAST makes merge exact by construction": rewrite the artifact's
 * scale plane in place with the projection above (the same clamp and grid
 * path) of `latent`. No code pointer is taken, so no code byte can change.
 * scales_inout device u8 [N, G]; ongrid_delta device fp32 [N, G] or NULL:
 *   fl32(s(new) - s(old)) with s(byte) = fl32(E4M3(byte) * ws2) or E8M0(byte),
 *   the delta whose subtraction restores the base (Sec. 5, Payoff 3);
 * changed_bytes device int64 or NULL: set to the number of bytes that changed. */
sq_status sq_merge(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *latent,
                   uint8_t *scales_inout, float *ongrid_delta, int64_t *changed_bytes, void *stream);

/* One scale plane of a multi-plane call: the N x G blocks of one linear (layouts
 * as above). N * G must be a multiple of 16 (it is for every linear: N % 8 == 0
 * and G % 16 == 0). sq_project_planes uses latent, bytes (bytes_out), mask
 * (nullable) and nonfinite (nullable, device int32); sq_merge_planes uses latent,
 * bytes (the artifact's scale plane, in place), ongrid_delta (nullable) and
 * changed_bytes (nullable, device int64). Fields a call does not use are ignored. */
typedef struct {
  int64_t N, G;
  float ws2;                 /* NVFP4 tensor scale of this plane; 1.0f for MXFP4 */
  const float *latent;       /* device fp32 [N, G] */
  uint8_t *bytes;            /* device u8 [N, G] */
  uint8_t *mask;             /* device u8 [N, G] or NULL */
  float *ongrid_delta;       /* device fp32 [N, G] or NULL */
  int32_t *nonfinite;        /* device int32 or NULL */
  int64_t *changed_bytes;    /* device int64 or NULL */
} sq_plane;
#define SQ_MAX_PLANES 16

/* The projection of sq_project_scales applied to up to SQ_MAX_PLANES planes of
 * different shapes in ONE kernel launch (the scale planes of every linear of a
 * layer, Sec. 3 QAST round_grid; bytes identical to one sq_project_scales call
 * per plane). The plane table is copied into the launch's parameters (`planes` is
 * a host array and may be reused as soon as the call returns); the call makes no
 * allocation and no copy, so it can be captured into a CUDA graph. Each plane's
 * counter receives its own NaN count. Uses a small counter accumulator of the
 * handle (allocated with the handle's device state): calls of one handle must be
 * ordered on the GPU. nplanes == 0 is a no-op. Returns SQ_ERR_INVALID_ARG for a bad
 * plane (shape, alignment, ws2) before anything is launched. */
sq_status sq_project_planes(sq_handle h, int32_t fmt, int32_t nplanes, const sq_plane *planes, void *stream);

/* The merge of sq_merge (Sec. 3 "QAST makes merge exact by construction"; Sec. 5
 * Payoff 3: one merge touches every target linear) over up to SQ_MAX_PLANES planes
 * in ONE kernel launch, with the same table, counter and ordering rules as
 * sq_project_planes; bytes, deltas and changed counts identical to one sq_merge
 * call per plane. No code pointer is taken. */
sq_status sq_merge_planes(sq_handle h, int32_t fmt, int32_t nplanes, const sq_plane *planes, void *stream);

/* Rollback, Sec. 5 Payoff 3 ("invertible merges and rollback"): subtracting the
 * on-grid scale delta a merge applied restores the base plane byte for byte. In
 * place, every byte b of scales_inout becomes the projection (the merge's grid and
 * clamp path) of fl32(s(b) - ongrid_delta), s(b) = fl32(E4M3(b) * ws2) or
 * E8M0(b). The restoration is exact whenever each merged scale is within a factor
 * 2 of its base (the subtraction is then exact in fp32); the raw training delta
 * does not restore it. ongrid_delta device fp32 [N, G] (sq_merge's output);
 * scales_inout device u8 [N, G]; changed_bytes device int64 or NULL (set). */
sq_status sq_rollback(sq_handle h, int32_t fmt, int64_t N, int64_t G, float ws2, const float *ongrid_delta,
                      uint8_t *scales_inout, int64_t *changed_bytes, void *stream);

/* Scale-only hot-swap, Sec. 5 "Hot-swap": the served task changes by overwriting
 * the artifact's scale plane with another adapter's on-grid bytes; no code
 * pointer is taken. src device u8 [N, G] (read); scales_inout device u8 [N, G]
 * (overwritten); changed_bytes device int64 or NULL: set to the number of bytes
 * that changed. */
sq_status sq_swap_scales(sq_handle h, int64_t N, int64_t G, const uint8_t *src, uint8_t *scales_inout,
                         int64_t *changed_bytes, void *stream);

/* Byte-level audit (Sec. 5): *count (device int64, required) is set to the number
 * of positions where the device buffers a and b (nbytes each, 16-byte aligned)
 * differ, e.g. a code plane before and after a merge (expected 0). */
sq_status sq_count_diff(sq_handle h, const uint8_t *a, const uint8_t *b, int64_t nbytes, int64_t *count,
                        void *stream);

/* Low-rank scale adapter, Sec. 3 "Scale-QLoRA forward": Delta S = (B A)(alpha/r)
 * with B [N, r] and A [r, G] (bf16 trainable factors), eff' = eff + Delta S per
 * block, then the grid projection of sq_project_scales (same clamp, bytes, mask
 * and NaN count). The latent is formed in fp32 in a fixed order, the same on
 * every run:
 *   eff = fl32(E4M3(base byte) * ws2) (NVFP4) or 2^(base byte - 127) (MXFP4);
 *   acc = fp32 fused multiply-adds over j = 0 .. r-1 from 0 of B[n,j] * A[j,b];
 *   eff' = fma(alpha_over_r, acc, eff).
 * base_scales device u8 [N, G] (the frozen base plane, read only); B device bf16
 * [N, r]; A device bf16 [r, G]; bytes_out device u8 [N, G]; mask_out device u8
 * [N, G] or NULL; nonfinite device int32 or NULL (set to the NaN count);
 * latent_out device fp32 [N, G] or NULL (receives eff', e.g. for sq_merge).
 * Requires 1 <= r <= 256, finite alpha_over_r and the ws2 rule of the format;
 * N, G in [0, 2^24]; when N or G is 0 only nonfinite is written and the arrays
 * may be NULL. */
sq_status sq_project_lowrank(sq_handle h, int32_t fmt, int64_t N, int64_t G, int32_t r, float ws2, float alpha_over_r,
                             const uint8_t *base_scales, const uint16_t *B, const uint16_t *A, uint8_t *bytes_out,
                             uint8_t *mask_out, int32_t *nonfinite, float *latent_out, void *stream);

/* Gradients of the adapter factors (Sec. 3: the gradient reaches eff' through the
 * straight-through estimator, masked by the ceiling clamp, and eff' is linear in
 * B and in A). With g the masked scale gradient [N, G] (sq_scale_grad with the
 * mask of sq_project_lowrank):
 *   dB[n,j] = alpha_over_r * sum_b g[n,b] A[j,b]    device fp32 [N, r], or NULL
 *   dA[j,b] = alpha_over_r * sum_n B[n,j] g[n,b]    device fp32 [r, G], or NULL
 * (not both NULL). fp32 accumulation in a fixed order (the same result on every
 * run). g device fp32 [N, G]; B device bf16 [N, r]; A device bf16 [r, G].
 * dA uses scratch in the handle (allocated on first use, grown when needed).
 * Requires 1 <= r <= 256 and finite alpha_over_r; N, G in [0, 2^24]. An empty
 * sum gives zeros: with N == 0, dA is zeroed; with G == 0, dB is zeroed; the
 * arrays of an empty side may be NULL. */
sq_status sq_lowrank_grad(sq_handle h, int64_t N, int64_t G, int32_t r, float alpha_over_r, const float *g,
                          const uint16_t *B, const uint16_t *A, float *dB, float *dA, void *stream);

/* Allocation-free variant of sq_scale_grad. The paper has no counterpart: this
 * entry point exists for callers of this library that cannot call cudaMalloc --
 * code whose device memory is owned by an outside pool or allocator that must
 * account for every byte, and hot loops that cannot accept the device-wide
 * synchronisation cudaMalloc / cudaFree may cause. It takes no handle and
 * allocates nothing: the kernel's scratch (the device error word its bounded
 * waits set) lives in a file-scope static __device__ array of 256 bytes that
 * every GPU loading the library holds until the process exits.
 *  - Arguments, layouts and results are those of sq_scale_grad, always in one
 *    pass over the tokens: where sq_scale_grad cuts them into parts (its
 *    partial planes need scratch), the two results agree up to fp32 rounding.
 *  - Scratch limit: 256 bytes; this kernel needs one 4-byte word for any M, N, K,
 *    and a call whose need exceeded the array would return SQ_ERR_INVALID_ARG.
 *  - The first call on each device sets up (checks the device, resolves the
 *    driver's tensor-map encoder); make that first call before any stream
 *    capture. Every call, with the device current, looks up the array's device
 *    address with cudaGetSymbolAddress (no allocation), so the address stays
 *    right if the device's primary context is reset and the module reloaded.
 *  - Every call on a device shares the array: the error word is cleared at the
 *    start of each call, and calls that overlap on the GPU race on it.
 *  - device_status: device int32 or NULL; if given, it receives the error word
 *    after the kernel (0, or nonzero when a bounded device wait ran out).
 * Returns SQ_OK, SQ_ERR_INVALID_ARG, SQ_ERR_UNSUPPORTED, SQ_ERR_DEVICE or
 * SQ_ERR_CUDA; there is no handle, so no error text. */
sq_status sq_scale_grad_noalloc(const sq_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                                const uint8_t *mask, float *g, int32_t *device_status, void *stream);

/* ---------------------------------------------------------------- scale-family variants
 * (ablation appendix; the same frozen codes, other reduction sets) */

/* Least-squares code-preserving fit of a weight-space update dW (the Spider
 * paragraph: the best per-block scale delta for a given update): block b of row n
 * can only move by t * c (c its E2M1 code values), so
 *   delta[n,b]    = <c, dW_b> / <c, c>      (0 for a block of zero codes)
 *   captured[n,b] = <c, dW_b>^2 / <c, c>    (energy of the projection onto the block's codes)
 *   total[n,b]    = ||dW_b||^2
 *   latent[n,b]   = fl32(scale(byte) + delta)  (the fitted scale; project it with sq_project_scales)
 * fp32 sums in element order. codes device [N, K/2]; dW device bf16 [N, K]; delta_out
 * device fp32 [N, K/B]; captured_out, total_out, latent_out device fp32 [N, K/B] or NULL;
 * scales device u8 [N, K/B], needed only with latent_out. K % 32 == 0. */
sq_status sq_fit_scale_delta(sq_handle h, int32_t fmt, int64_t N, int64_t K, float ws2, const uint8_t *codes,
                             const uint8_t *scales, const uint16_t *dW, float *delta_out, float *captured_out,
                             float *total_out, float *latent_out, void *stream);

/* Granularity ladder (ablation appendix, "Granularity alone over-perturbs"): a direct
 * additive scale delta at granularity gd, one value per group of G / gd consecutive
 * blocks of a row (gd = 1: per row, PEQA; gd = G: per block). The gradient of the
 * group deltas is the sum of the group's (masked) block scale gradients:
 *   out[n, j] = sum_{b in group j} g[n, b]     (fp32, block order)
 * g device fp32 [N, G]; out device fp32 [N, gd]; gd >= 1 divides G. */
sq_status sq_group_reduce(sq_handle h, int64_t N, int64_t G, int64_t gd, const float *g, float *out, void *stream);

/* The group-delta latent fl32(scale(base byte) + delta[n, b / (G / gd)]) projected as
 * sq_project_scales does (bytes, mask, NaN count), the latent optionally kept for
 * sq_merge. base_scales device u8 [N, G]; delta device fp32 [N, gd]; bytes_out device
 * u8 [N, G]; mask_out, latent_out or NULL; nonfinite device int32 or NULL. */
sq_status sq_project_group_delta(sq_handle h, int32_t fmt, int64_t N, int64_t G, int64_t gd, float ws2,
                                 const uint8_t *base_scales, const float *delta, uint8_t *bytes_out, uint8_t *mask_out,
                                 int32_t *nonfinite, float *latent_out, void *stream);

/* Full-precision multiplicative control (ablation appendix: on unquantized bf16
 * weights the within-block pattern is frozen and one coefficient per (row, block of
 * 16) is learned, W' = W (1 + dS[o, i / 16]); no codes, no grid, no STE). Arithmetic:
 * f = fl32(1 + dS), W' = bf16(fl32(W * f)) rounded to nearest even, then the
 * contractions of sq_fwd / sq_bwd_dx with W' (bf16 operands, fp32 accumulation). */
typedef struct {
  int32_t N;            /* out features, N % 8 == 0                          */
  int32_t K;            /* in features, K % 32 == 0                          */
  const uint16_t *W;    /* device bf16 [N, K], frozen                        */
  const float *dS;      /* device fp32 [N, K/16] coefficients (FWD, DX)      */
} sq_control_weight;

/* Y = X W'^T. X device bf16 [M, K]; Y device bf16 [M, N]. */
sq_status sq_control_fwd(sq_handle h, const sq_control_weight *w, const uint16_t *X, int64_t M, uint16_t *Y,
                         void *stream);

/* dX = dY W'. dY device bf16 [M, N]; dX device bf16 [M, K]. */
sq_status sq_control_bwd_dx(sq_handle h, const sq_control_weight *w, const uint16_t *dY, int64_t M, uint16_t *dX,
                            void *stream);

/* Coefficient gradient through W' = W (1 + dS) (its bf16 rounding passed straight
 * through): g[o, b] = sum_{i in block b} W[o, i] (dY^T X)[o, i], the dW tile reduced
 * on chip as in sq_scale_grad. g device fp32 [N, K/16]; dS is not read; M == 0
 * gives zeros. */
sq_status sq_control_grad(sq_handle h, const sq_control_weight *w, const uint16_t *X, const uint16_t *dY, int64_t M,
                          float *g, void *stream);

/* The control's low-rank coefficient plane: out = alpha_over_r * B A, B [N, r] and
 * A [r, G] bf16, out device fp32 [N, G], fp32 sums in a fixed order (the same on
 * every run); its gradients are sq_lowrank_grad of the coefficient gradient. Uses
 * the handle's scratch. 1 <= r <= 256. */
sq_status sq_lowrank_product(sq_handle h, int64_t N, int64_t G, int32_t r, float alpha_over_r, const uint16_t *B,
                             const uint16_t *A, float *out, void *stream);

/* ---------------------------------------------------------------- experts
 * Mixture-of-experts layers (Sec. 3 "MoE: a batched grouped-expert kernel": the
 * quantized linears are the experts, and every expert's contraction runs in one
 * batched launch instead of a per-expert loop). One call covers the E experts of
 * one linear; each expert e computes exactly what the dense entry point computes
 * for its own weight and its own tokens.
 *
 * Token layout: the M = offsets[E] rows of X, dY, Y and dX are sorted by expert;
 * rows offsets[e] .. offsets[e+1]-1 belong to expert e (a token routed to k
 * experts appears k times). offsets is a HOST int64 array of E + 1 values with
 * offsets[0] == 0, non-decreasing, offsets[E] < 2^31; an expert may have no rows.
 *
 * Each call builds a table of per-expert TMA descriptors in pinned host memory
 * and copies it to the device on `stream` ahead of the kernel. The handle keeps
 * four such tables per device and reuses them in turn: a call waits on the host
 * until the grouped launch four calls back (on any stream) has completed. The
 * host arrays (offsets, ws2) are read before the call returns. Grouped calls
 * cannot be captured into a CUDA graph (SQ_ERR_UNSUPPORTED while the stream is
 * capturing). */
typedef struct {
  int32_t fmt;           /* sq_format, shared by all experts                            */
  int32_t E;             /* experts, 1 <= E <= 65536, with E * N <= 2^31 - 1025         */
  int32_t N;             /* out features of each expert, N % 8 == 0                     */
  int32_t K;             /* in features of each expert,  K % 32 == 0                    */
  const uint8_t *codes;  /* device [E, N, K/2]: expert e's codes at e * N * K/2 bytes   */
  const uint8_t *scales; /* device [E, N, K/B]: expert e's scale plane                  */
  const float *ws2;      /* HOST [E]: NVFP4 tensor scale of each expert (finite, > 0);
                            MXFP4: NULL, or every entry exactly 1.0                     */
} sq_grouped_weight;

/* Y[offsets[e] + m, :] = X[offsets[e] + m, :] . W_e^T for every expert e.
 * X device bf16 [M, K]; Y device bf16 [M, N]. M == 0 writes nothing. */
sq_status sq_grouped_fwd(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *X,
                         uint16_t *Y, void *stream);

/* dX[offsets[e] + m, :] = dY[offsets[e] + m, :] . W_e for every expert e.
 * dY device bf16 [M, N]; dX device bf16 [M, K]. */
sq_status sq_grouped_bwd_dx(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *dY,
                            uint16_t *dX, void *stream);

/* g[e, n, b] = sum_{k in b} code_e[n, k] sum over expert e's rows m of dY[m, n] X[m, k]
 * (optionally x mask[e, n, b]); an expert with no rows gets g[e] = 0.
 * X device bf16 [M, K]; dY device bf16 [M, N]; mask device u8 [E, N, K/B] or NULL;
 * g device fp32 [E, N, K/B]. The scale bytes are not read (scales may be NULL). */
sq_status sq_grouped_scale_grad(sq_handle h, const sq_grouped_weight *w, const int64_t *offsets, const uint16_t *X,
                                const uint16_t *dY, const uint8_t *mask, float *g, void *stream);

/* The low-rank adapters of all E experts in one launch (Sec. 3 "MoE: a batched
 * grouped-expert kernel": one batched product forms every expert's Delta S):
 * expert e's latent eff' = eff + (alpha/r) B[e] A[e], formed and projected
 * exactly as sq_project_lowrank with ws2[e]. w->scales are the frozen base planes
 * [E, N, K/B] (read only; codes are not read); B device bf16 [E, N, r]; A device
 * bf16 [E, r, K/B]; bytes_out, mask_out (or NULL), latent_out (fp32, or NULL)
 * device [E, N, K/B]; nonfinite device int32 or NULL (count over all experts).
 * Requires E <= 65535, 1 <= r <= 256 and finite alpha_over_r. */
sq_status sq_grouped_project_lowrank(sq_handle h, const sq_grouped_weight *w, int32_t r, float alpha_over_r,
                                     const uint16_t *B, const uint16_t *A, uint8_t *bytes_out, uint8_t *mask_out,
                                     int32_t *nonfinite, float *latent_out, void *stream);

/* sq_lowrank_grad for E experts in one set of launches: g device fp32 [E, N, G];
 * B [E, N, r], A [E, r, G] bf16; dB device fp32 [E, N, r] or NULL; dA device fp32
 * [E, r, G] or NULL (not both NULL). Same arithmetic, order and empty-sum rules
 * per expert; 1 <= E <= 65535. Uses the handle's scratch, like sq_lowrank_grad. */
sq_status sq_grouped_lowrank_grad(sq_handle h, int32_t E, int64_t N, int64_t G, int32_t r, float alpha_over_r,
                                  const float *g, const uint16_t *B, const uint16_t *A, float *dB, float *dA,
                                  void *stream);

/* Grid projection (sq_project_scales) of all E experts' latent planes in one
 * launch: latent device fp32 [E, N, K/B], plane e projected with ws2[e];
 * bytes_out device u8 [E, N, K/B]; mask_out device u8 [E, N, K/B] or NULL;
 * nonfinite device int32 or NULL (the NaN count over all planes). codes and
 * scales of w are not read (may be NULL). */
sq_status sq_grouped_project_scales(sq_handle h, const sq_grouped_weight *w, const float *latent, uint8_t *bytes_out,
                                    uint8_t *mask_out, int32_t *nonfinite, void *stream);

/* Merge (sq_merge) of all E experts' latent planes in one launch into the scale
 * planes scales_inout device u8 [E, N, K/B] (plane e with ws2[e]); ongrid_delta
 * device fp32 [E, N, K/B] or NULL; changed_bytes device int64 or NULL (the count
 * over all planes). No code byte is read or written. */
sq_status sq_grouped_merge(sq_handle h, const sq_grouped_weight *w, const float *latent, uint8_t *scales_inout,
                           float *ongrid_delta, int64_t *changed_bytes, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* SCALEQLORA_H */
