"""ctypes binding of libscaleqlora (include/scaleqlora.h).

Argument marshalling only: torch tensors supply device pointers and the current
CUDA stream; every step of the path runs in the library's kernels. There is no
fallback: if the shared library is missing, loading raises.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libscaleqlora.so")

NVFP4 = 0
MXFP4 = 1
BLOCK = {NVFP4: 16, MXFP4: 32}

SQ_OK = 0
STATUS = {0: "SQ_OK", -1: "SQ_ERR_INVALID_ARG", -2: "SQ_ERR_UNSUPPORTED", -3: "SQ_ERR_DEVICE", -4: "SQ_ERR_CUDA",
          -5: "SQ_ERR_DEVICE_TIMEOUT"}

# Every entry point the header declares (checked against include/scaleqlora.h by the tests).
EXPORTS = ("sq_create", "sq_destroy", "sq_status_string", "sq_last_error", "sq_sync", "sq_fwd", "sq_bwd_dx",
           "sq_scale_grad", "sq_project_scales", "sq_merge", "sq_project_lowrank", "sq_lowrank_grad",
           "sq_rollback", "sq_swap_scales", "sq_count_diff", "sq_scale_grad_noalloc", "sq_grouped_fwd",
           "sq_grouped_bwd_dx", "sq_grouped_scale_grad", "sq_grouped_project_scales", "sq_grouped_merge",
           "sq_grouped_project_lowrank", "sq_grouped_lowrank_grad", "sq_fit_scale_delta", "sq_group_reduce",
           "sq_project_group_delta", "sq_control_fwd", "sq_control_bwd_dx", "sq_control_grad", "sq_lowrank_product",
           "sq_selftest_wait_timeout", "sq_scale_grad_workspace", "sq_project_planes", "sq_merge_planes")


class SQError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


class _SqWeight(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int32), ("N", ctypes.c_int32), ("K", ctypes.c_int32),
                ("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p), ("ws2", ctypes.c_float)]


class _SqGroupedWeight(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int32), ("E", ctypes.c_int32), ("N", ctypes.c_int32), ("K", ctypes.c_int32),
                ("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p), ("ws2", ctypes.POINTER(ctypes.c_float))]


class _SqControlWeight(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int32), ("K", ctypes.c_int32), ("W", ctypes.c_void_p), ("dS", ctypes.c_void_p)]


_lib = None


def load() -> ctypes.CDLL:
    """Load libscaleqlora.so from the package directory (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with `python -m paper_2609_04526_gb300.build` "
                          "(or __graft_entry__.build()); there is no fallback path")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
    W = ctypes.POINTER(_SqWeight)
    L.sq_create.argtypes = [ctypes.POINTER(vp)]
    L.sq_destroy.argtypes = [vp]
    L.sq_status_string.argtypes = [ctypes.c_int]
    L.sq_status_string.restype = ctypes.c_char_p
    L.sq_last_error.argtypes = [vp]
    L.sq_last_error.restype = ctypes.c_char_p
    L.sq_sync.argtypes = [vp, vp]
    L.sq_selftest_wait_timeout.argtypes = [vp, vp]
    L.sq_scale_grad_workspace.argtypes = [vp, W, i64, vp, vp]
    L.sq_fwd.argtypes = [vp, W, vp, i64, vp, vp]
    L.sq_bwd_dx.argtypes = [vp, W, vp, i64, vp, vp]
    L.sq_scale_grad.argtypes = [vp, W, vp, vp, i64, vp, vp, vp]
    L.sq_project_scales.argtypes = [vp, i32, i64, i64, f32, vp, vp, vp, vp, vp]
    L.sq_merge.argtypes = [vp, i32, i64, i64, f32, vp, vp, vp, vp, vp]
    L.sq_project_planes.argtypes = [vp, i32, i32, ctypes.POINTER(_SqPlane), vp]
    L.sq_merge_planes.argtypes = [vp, i32, i32, ctypes.POINTER(_SqPlane), vp]
    L.sq_project_lowrank.argtypes = [vp, i32, i64, i64, i32, f32, f32, vp, vp, vp, vp, vp, vp, vp, vp]
    L.sq_lowrank_grad.argtypes = [vp, i64, i64, i32, f32, vp, vp, vp, vp, vp, vp]
    L.sq_rollback.argtypes = [vp, i32, i64, i64, f32, vp, vp, vp, vp]
    L.sq_swap_scales.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    L.sq_count_diff.argtypes = [vp, vp, vp, i64, vp, vp]
    L.sq_scale_grad_noalloc.argtypes = [W, vp, vp, i64, vp, vp, vp, vp]
    GW, OFF = ctypes.POINTER(_SqGroupedWeight), ctypes.POINTER(ctypes.c_int64)
    L.sq_grouped_fwd.argtypes = [vp, GW, OFF, vp, vp, vp]
    L.sq_grouped_bwd_dx.argtypes = [vp, GW, OFF, vp, vp, vp]
    L.sq_grouped_scale_grad.argtypes = [vp, GW, OFF, vp, vp, vp, vp, vp]
    L.sq_grouped_project_scales.argtypes = [vp, GW, vp, vp, vp, vp, vp]
    L.sq_grouped_merge.argtypes = [vp, GW, vp, vp, vp, vp, vp]
    L.sq_grouped_project_lowrank.argtypes = [vp, GW, i32, f32, vp, vp, vp, vp, vp, vp, vp]
    L.sq_grouped_lowrank_grad.argtypes = [vp, i32, i64, i64, i32, f32, vp, vp, vp, vp, vp, vp]
    L.sq_fit_scale_delta.argtypes = [vp, i32, i64, i64, f32, vp, vp, vp, vp, vp, vp, vp, vp]
    L.sq_group_reduce.argtypes = [vp, i64, i64, i64, vp, vp, vp]
    L.sq_project_group_delta.argtypes = [vp, i32, i64, i64, i64, f32, vp, vp, vp, vp, vp, vp, vp]
    CW = ctypes.POINTER(_SqControlWeight)
    L.sq_control_fwd.argtypes = [vp, CW, vp, i64, vp, vp]
    L.sq_control_bwd_dx.argtypes = [vp, CW, vp, i64, vp, vp]
    L.sq_control_grad.argtypes = [vp, CW, vp, vp, i64, vp, vp]
    L.sq_lowrank_product.argtypes = [vp, i64, i64, i32, f32, vp, vp, vp, vp]
    for name in EXPORTS:
        if name not in ("sq_status_string", "sq_last_error"):
            getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


class _SqPlane(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int64), ("G", ctypes.c_int64), ("ws2", ctypes.c_float), ("latent", ctypes.c_void_p),
                ("bytes", ctypes.c_void_p), ("mask", ctypes.c_void_p), ("ongrid_delta", ctypes.c_void_p),
                ("nonfinite", ctypes.c_void_p), ("changed_bytes", ctypes.c_void_p)]


@dataclasses.dataclass
class QuantWeight:
    """One native-FP4 linear, weight [N, K]: packed codes [N, K/2] u8, scales [N, K/B] u8, ws2."""
    fmt: int
    N: int
    K: int
    codes: torch.Tensor
    scales: Optional[torch.Tensor]
    ws2: float

    def _c(self) -> _SqWeight:
        return _SqWeight(self.fmt, self.N, self.K, _ptr(self.codes), _ptr(self.scales), self.ws2)


@dataclasses.dataclass
class GroupedWeight:
    """The E experts of one MoE linear, each [N, K]: codes [E, N, K/2] u8, scales
    [E, N, K/B] u8 (device), ws2 one tensor scale per expert (host floats)."""
    fmt: int
    E: int
    N: int
    K: int
    codes: torch.Tensor
    scales: Optional[torch.Tensor]
    ws2: list

    def _c(self):
        ws = (ctypes.c_float * self.E)(*[float(x) for x in self.ws2])
        c = _SqGroupedWeight(self.fmt, self.E, self.N, self.K, _ptr(self.codes), _ptr(self.scales),
                             ctypes.cast(ws, ctypes.POINTER(ctypes.c_float)))
        return c, ws  # keep the array alive for the call

    def expert(self, e: int) -> QuantWeight:
        """Expert e as a dense weight (views into the grouped planes)."""
        return QuantWeight(self.fmt, self.N, self.K, self.codes[e],
                           None if self.scales is None else self.scales[e], float(self.ws2[e]))


def _offsets(offsets, E: int):
    vals = [int(x) for x in offsets]
    if len(vals) != E + 1:  # the library reads exactly E + 1 values
        raise ValueError(f"offsets has {len(vals)} values; a grouped call over {E} experts needs {E + 1}")
    return (ctypes.c_int64 * len(vals))(*vals), vals


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


class Handle:
    """Owns one sq_handle (not thread-safe: one per host thread)."""

    def __init__(self):
        self._L = load()
        h = ctypes.c_void_p()
        st = self._L.sq_create(ctypes.byref(h))
        if st != SQ_OK:
            raise SQError(st, "sq_create failed")
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            self._L.sq_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, st: int):
        if st != SQ_OK:
            raise SQError(st, self._L.sq_last_error(self._h).decode())

    # raw status variants (no exception) -------------------------------------
    def status_of(self, name: str, *args) -> int:
        return getattr(self._L, name)(self._h, *args)

    def last_error(self) -> str:
        return self._L.sq_last_error(self._h).decode()

    # entry points ------------------------------------------------------------
    def sq_sync(self, stream=None):
        self._check(self._L.sq_sync(self._h, _stream(stream)))

    def sq_selftest_wait_timeout(self, stream=None):
        """Enqueue a bounded wait that runs out (about 1 s); the next sq_sync raises
        SQError with status SQ_ERR_DEVICE_TIMEOUT."""
        self._check(self._L.sq_selftest_wait_timeout(self._h, _stream(stream)))

    def sq_fwd(self, w: QuantWeight, X: torch.Tensor, Y: Optional[torch.Tensor] = None, stream=None):
        M = X.shape[0]
        if Y is None:
            Y = torch.empty(M, w.N, dtype=torch.bfloat16, device=X.device)
        wc = w._c()
        self._check(self._L.sq_fwd(self._h, ctypes.byref(wc), _ptr(X), M, _ptr(Y), _stream(stream)))
        return Y

    def sq_bwd_dx(self, w: QuantWeight, dY: torch.Tensor, dX: Optional[torch.Tensor] = None, stream=None):
        M = dY.shape[0]
        if dX is None:
            dX = torch.empty(M, w.K, dtype=torch.bfloat16, device=dY.device)
        wc = w._c()
        self._check(self._L.sq_bwd_dx(self._h, ctypes.byref(wc), _ptr(dY), M, _ptr(dX), _stream(stream)))
        return dX

    def sq_scale_grad_workspace(self, w: QuantWeight, M: int):
        """(splits, scratch bytes) of sq_scale_grad for this weight shape and M tokens."""
        sp = ctypes.c_int32(0)
        nb = ctypes.c_int64(0)
        wc = w._c()
        self._check(self._L.sq_scale_grad_workspace(self._h, ctypes.byref(wc), int(M), ctypes.byref(sp),
                                                    ctypes.byref(nb)))
        return sp.value, nb.value

    def sq_scale_grad(self, w: QuantWeight, X: torch.Tensor, dY: torch.Tensor, mask: Optional[torch.Tensor] = None,
                      g: Optional[torch.Tensor] = None, stream=None):
        M = X.shape[0]
        if g is None:
            g = torch.empty(w.N, w.K // BLOCK[w.fmt], dtype=torch.float32, device=X.device)
        wc = w._c()
        self._check(self._L.sq_scale_grad(self._h, ctypes.byref(wc), _ptr(X), _ptr(dY), M, _ptr(mask), _ptr(g),
                                          _stream(stream)))
        return g

    def sq_project_scales(self, fmt: int, latent: torch.Tensor, ws2: float, bytes_out: Optional[torch.Tensor] = None,
                          mask_out: Optional[torch.Tensor] = None, nonfinite: Optional[torch.Tensor] = None,
                          want_mask: bool = True, stream=None):
        N, G = latent.shape
        if bytes_out is None:
            bytes_out = torch.empty(N, G, dtype=torch.uint8, device=latent.device)
        if mask_out is None and want_mask:
            mask_out = torch.empty(N, G, dtype=torch.uint8, device=latent.device)
        self._check(self._L.sq_project_scales(self._h, fmt, N, G, ws2, _ptr(latent), _ptr(bytes_out), _ptr(mask_out),
                                              _ptr(nonfinite), _stream(stream)))
        return bytes_out, mask_out

    def sq_project_lowrank(self, fmt: int, base_scales: torch.Tensor, B: torch.Tensor, A: torch.Tensor, ws2: float,
                           alpha_over_r: float, bytes_out: Optional[torch.Tensor] = None,
                           mask_out: Optional[torch.Tensor] = None, nonfinite: Optional[torch.Tensor] = None,
                           latent_out: Optional[torch.Tensor] = None, stream=None):
        """Latent eff + (alpha/r) B A of the low-rank adapter, projected onto the grid.
        base_scales [N, G] u8; B [N, r] and A [r, G] bf16. Returns (bytes, mask, latent)."""
        N, G = base_scales.shape
        r = B.shape[1]
        if bytes_out is None:
            bytes_out = torch.empty(N, G, dtype=torch.uint8, device=base_scales.device)
        self._check(self._L.sq_project_lowrank(self._h, fmt, N, G, r, ws2, alpha_over_r, _ptr(base_scales), _ptr(B),
                                               _ptr(A), _ptr(bytes_out), _ptr(mask_out), _ptr(nonfinite),
                                               _ptr(latent_out), _stream(stream)))
        return bytes_out, mask_out, latent_out

    def sq_lowrank_grad(self, g: torch.Tensor, B: torch.Tensor, A: torch.Tensor, alpha_over_r: float,
                        dB: Optional[torch.Tensor] = None, dA: Optional[torch.Tensor] = None, want_dB: bool = True,
                        want_dA: bool = True, stream=None):
        """dB = (alpha/r) g A^T [N, r] and dA = (alpha/r) B^T g [r, G] (fp32) from the masked
        scale gradient g [N, G]."""
        N, G = g.shape
        r = B.shape[1]
        if dB is None and want_dB:
            dB = torch.empty(N, r, dtype=torch.float32, device=g.device)
        if dA is None and want_dA:
            dA = torch.empty(r, G, dtype=torch.float32, device=g.device)
        self._check(self._L.sq_lowrank_grad(self._h, N, G, r, alpha_over_r, _ptr(g), _ptr(B), _ptr(A), _ptr(dB),
                                            _ptr(dA), _stream(stream)))
        return dB, dA

    def sq_rollback(self, fmt: int, ongrid_delta: torch.Tensor, ws2: float, scales_inout: torch.Tensor,
                    changed: Optional[torch.Tensor] = None, stream=None):
        """Undo a merge in place with the on-grid delta it applied."""
        N, G = scales_inout.shape
        self._check(self._L.sq_rollback(self._h, fmt, N, G, ws2, _ptr(ongrid_delta), _ptr(scales_inout),
                                        _ptr(changed), _stream(stream)))
        return scales_inout

    def sq_swap_scales(self, src: torch.Tensor, scales_inout: torch.Tensor, changed: Optional[torch.Tensor] = None,
                       stream=None):
        """Overwrite the scale plane with src (scale-only hot-swap), counting changed bytes."""
        N, G = scales_inout.shape
        self._check(self._L.sq_swap_scales(self._h, N, G, _ptr(src), _ptr(scales_inout), _ptr(changed),
                                           _stream(stream)))
        return scales_inout

    def sq_count_diff(self, a: torch.Tensor, b: torch.Tensor, count: Optional[torch.Tensor] = None, stream=None):
        """Device int64 tensor holding the number of differing bytes of a and b."""
        if count is None:
            count = torch.empty(1, dtype=torch.int64, device=a.device)
        nbytes = a.numel() * a.element_size()
        assert b.numel() * b.element_size() == nbytes
        self._check(self._L.sq_count_diff(self._h, _ptr(a), _ptr(b), nbytes, _ptr(count), _stream(stream)))
        return count

    def sq_merge(self, fmt: int, latent: torch.Tensor, ws2: float, scales_inout: torch.Tensor,
                 ongrid_delta: Optional[torch.Tensor] = None, changed: Optional[torch.Tensor] = None, stream=None):
        N, G = latent.shape
        self._check(self._L.sq_merge(self._h, fmt, N, G, ws2, _ptr(latent), _ptr(scales_inout), _ptr(ongrid_delta),
                                     _ptr(changed), _stream(stream)))
        return scales_inout

    def _planes(self, planes):
        arr = (_SqPlane * max(1, len(planes)))()
        for i, p in enumerate(planes):
            N, G = p["latent"].shape
            arr[i] = _SqPlane(N, G, float(p.get("ws2", 1.0)), _ptr(p["latent"]), _ptr(p["bytes"]), _ptr(p.get("mask")),
                              _ptr(p.get("ongrid_delta")), _ptr(p.get("nonfinite")), _ptr(p.get("changed")))
        return arr

    def sq_project_planes(self, fmt: int, planes, stream=None):
        """One launch for several planes: planes is a list of dicts with latent [N, G]
        fp32, bytes [N, G] u8 (out), and optional ws2, mask (out), nonfinite (int32 [1])."""
        arr = self._planes(planes)
        self._check(self._L.sq_project_planes(self._h, fmt, len(planes), arr, _stream(stream)))

    def sq_merge_planes(self, fmt: int, planes, stream=None):
        """One launch for several planes: planes is a list of dicts with latent [N, G]
        fp32, bytes [N, G] u8 (the scale plane, in place), and optional ws2,
        ongrid_delta [N, G] fp32, changed (int64 [1])."""
        arr = self._planes(planes)
        self._check(self._L.sq_merge_planes(self._h, fmt, len(planes), arr, _stream(stream)))

    # experts of an MoE linear ------------------------------------------------
    def sq_grouped_fwd(self, w: GroupedWeight, offsets, X: torch.Tensor, Y: Optional[torch.Tensor] = None,
                       stream=None):
        """Y rows offsets[e]..offsets[e+1]-1 = X rows of expert e times W_e^T (offsets: E + 1 host ints)."""
        off, vals = _offsets(offsets, w.E)
        if Y is None:
            Y = torch.empty(vals[-1], w.N, dtype=torch.bfloat16, device=X.device)
        wc, keep = w._c()
        self._check(self._L.sq_grouped_fwd(self._h, ctypes.byref(wc), off, _ptr(X), _ptr(Y), _stream(stream)))
        return Y

    def sq_grouped_bwd_dx(self, w: GroupedWeight, offsets, dY: torch.Tensor, dX: Optional[torch.Tensor] = None,
                          stream=None):
        off, vals = _offsets(offsets, w.E)
        if dX is None:
            dX = torch.empty(vals[-1], w.K, dtype=torch.bfloat16, device=dY.device)
        wc, keep = w._c()
        self._check(self._L.sq_grouped_bwd_dx(self._h, ctypes.byref(wc), off, _ptr(dY), _ptr(dX), _stream(stream)))
        return dX

    def sq_grouped_scale_grad(self, w: GroupedWeight, offsets, X: torch.Tensor, dY: torch.Tensor,
                              mask: Optional[torch.Tensor] = None, g: Optional[torch.Tensor] = None, stream=None):
        """g [E, N, K/B] fp32: every expert's block-reduced scale gradient over its own rows."""
        off, _ = _offsets(offsets, w.E)
        if g is None:
            g = torch.empty(w.E, w.N, w.K // BLOCK[w.fmt], dtype=torch.float32, device=X.device)
        wc, keep = w._c()
        self._check(self._L.sq_grouped_scale_grad(self._h, ctypes.byref(wc), off, _ptr(X), _ptr(dY), _ptr(mask),
                                                  _ptr(g), _stream(stream)))
        return g

    def sq_grouped_project_scales(self, w: GroupedWeight, latent: torch.Tensor, bytes_out: Optional[torch.Tensor] = None,
                                  mask_out: Optional[torch.Tensor] = None, nonfinite: Optional[torch.Tensor] = None,
                                  want_mask: bool = True, stream=None):
        """Project every expert's latent plane [E, N, G] with its own ws2. Returns (bytes, mask)."""
        if bytes_out is None:
            bytes_out = torch.empty(latent.shape, dtype=torch.uint8, device=latent.device)
        if mask_out is None and want_mask:
            mask_out = torch.empty(latent.shape, dtype=torch.uint8, device=latent.device)
        wc, keep = w._c()
        self._check(self._L.sq_grouped_project_scales(self._h, ctypes.byref(wc), _ptr(latent), _ptr(bytes_out),
                                                      _ptr(mask_out), _ptr(nonfinite), _stream(stream)))
        return bytes_out, mask_out

    def sq_grouped_merge(self, w: GroupedWeight, latent: torch.Tensor, scales_inout: torch.Tensor,
                         ongrid_delta: Optional[torch.Tensor] = None, changed: Optional[torch.Tensor] = None,
                         stream=None):
        """Merge every expert's latent plane into scales_inout [E, N, G] with its own ws2."""
        wc, keep = w._c()
        self._check(self._L.sq_grouped_merge(self._h, ctypes.byref(wc), _ptr(latent), _ptr(scales_inout),
                                             _ptr(ongrid_delta), _ptr(changed), _stream(stream)))
        return scales_inout

    def sq_grouped_project_lowrank(self, w: GroupedWeight, B: torch.Tensor, A: torch.Tensor, alpha_over_r: float,
                                   bytes_out: Optional[torch.Tensor] = None, mask_out: Optional[torch.Tensor] = None,
                                   nonfinite: Optional[torch.Tensor] = None, latent_out: Optional[torch.Tensor] = None,
                                   stream=None):
        """Every expert's adapter latent eff + (alpha/r) B[e] A[e] over its base plane w.scales[e],
        projected with its ws2. B [E, N, r], A [E, r, G] bf16. Returns (bytes, mask, latent)."""
        r = B.shape[2]
        if bytes_out is None:
            bytes_out = torch.empty(w.scales.shape, dtype=torch.uint8, device=w.scales.device)
        wc, keep = w._c()
        self._check(self._L.sq_grouped_project_lowrank(self._h, ctypes.byref(wc), r, alpha_over_r, _ptr(B), _ptr(A),
                                                       _ptr(bytes_out), _ptr(mask_out), _ptr(nonfinite),
                                                       _ptr(latent_out), _stream(stream)))
        return bytes_out, mask_out, latent_out

    def sq_grouped_lowrank_grad(self, g: torch.Tensor, B: torch.Tensor, A: torch.Tensor, alpha_over_r: float,
                                dB: Optional[torch.Tensor] = None, dA: Optional[torch.Tensor] = None,
                                want_dB: bool = True, want_dA: bool = True, stream=None):
        """Adapter gradients of every expert: g [E, N, G] fp32 -> dB [E, N, r], dA [E, r, G]."""
        E, N, G = g.shape
        r = B.shape[2]
        if dB is None and want_dB:
            dB = torch.empty(E, N, r, dtype=torch.float32, device=g.device)
        if dA is None and want_dA:
            dA = torch.empty(E, r, G, dtype=torch.float32, device=g.device)
        self._check(self._L.sq_grouped_lowrank_grad(self._h, E, N, G, r, alpha_over_r, _ptr(g), _ptr(B), _ptr(A),
                                                    _ptr(dB), _ptr(dA), _stream(stream)))
        return dB, dA


    # scale-family variants -----------------------------------------------------
    def sq_fit_scale_delta(self, fmt: int, codes: torch.Tensor, dW: torch.Tensor, ws2: float = 1.0,
                           scales: Optional[torch.Tensor] = None, want_energy: bool = False, stream=None):
        """Least-squares per-block scale delta of a bf16 weight update dW [N, K] against the
        codes [N, K/2]. Returns (delta, captured, total, latent); the last three are None
        unless asked for (energies with want_energy, the latent when scales are given)."""
        N, K = dW.shape
        G = K // BLOCK[fmt]
        delta = torch.empty(N, G, dtype=torch.float32, device=dW.device)
        cap = torch.empty_like(delta) if want_energy else None
        tot = torch.empty_like(delta) if want_energy else None
        lat = torch.empty_like(delta) if scales is not None else None
        self._check(self._L.sq_fit_scale_delta(self._h, fmt, N, K, ws2, _ptr(codes), _ptr(scales), _ptr(dW),
                                               _ptr(delta), _ptr(cap), _ptr(tot), _ptr(lat), _stream(stream)))
        return delta, cap, tot, lat

    def sq_group_reduce(self, g: torch.Tensor, gd: int, out: Optional[torch.Tensor] = None, stream=None):
        """Gradient of per-group scale deltas: sums of each group's G / gd block gradients, [N, gd]."""
        N, G = g.shape
        if out is None:
            out = torch.empty(N, gd, dtype=torch.float32, device=g.device)
        self._check(self._L.sq_group_reduce(self._h, N, G, gd, _ptr(g), _ptr(out), _stream(stream)))
        return out

    def sq_project_group_delta(self, fmt: int, base_scales: torch.Tensor, delta: torch.Tensor, ws2: float,
                               bytes_out: Optional[torch.Tensor] = None, mask_out: Optional[torch.Tensor] = None,
                               nonfinite: Optional[torch.Tensor] = None, latent_out: Optional[torch.Tensor] = None,
                               stream=None):
        """Projection of s(base byte) + delta[n, b // (G / gd)]; delta [N, gd]. Returns (bytes, mask, latent)."""
        N, G = base_scales.shape
        gd = delta.shape[1]
        if bytes_out is None:
            bytes_out = torch.empty(N, G, dtype=torch.uint8, device=base_scales.device)
        self._check(self._L.sq_project_group_delta(self._h, fmt, N, G, gd, ws2, _ptr(base_scales), _ptr(delta),
                                                   _ptr(bytes_out), _ptr(mask_out), _ptr(nonfinite), _ptr(latent_out),
                                                   _stream(stream)))
        return bytes_out, mask_out, latent_out

    # full-precision multiplicative control -------------------------------------
    def sq_control_fwd(self, W: torch.Tensor, dS: torch.Tensor, X: torch.Tensor, Y: Optional[torch.Tensor] = None,
                       stream=None):
        """Y = X W'^T with W' = bf16(W (1 + dS)) per row and block of 16; W [N, K] bf16, dS [N, K/16]."""
        N, K = W.shape
        M = X.shape[0]
        if Y is None:
            Y = torch.empty(M, N, dtype=torch.bfloat16, device=X.device)
        cw = _SqControlWeight(N, K, _ptr(W), _ptr(dS))
        self._check(self._L.sq_control_fwd(self._h, ctypes.byref(cw), _ptr(X), M, _ptr(Y), _stream(stream)))
        return Y

    def sq_control_bwd_dx(self, W: torch.Tensor, dS: torch.Tensor, dY: torch.Tensor,
                          dX: Optional[torch.Tensor] = None, stream=None):
        N, K = W.shape
        M = dY.shape[0]
        if dX is None:
            dX = torch.empty(M, K, dtype=torch.bfloat16, device=dY.device)
        cw = _SqControlWeight(N, K, _ptr(W), _ptr(dS))
        self._check(self._L.sq_control_bwd_dx(self._h, ctypes.byref(cw), _ptr(dY), M, _ptr(dX), _stream(stream)))
        return dX

    def sq_control_grad(self, W: torch.Tensor, X: torch.Tensor, dY: torch.Tensor, g: Optional[torch.Tensor] = None,
                        stream=None):
        """Coefficient gradient g[o, b] = sum over the block of W[o, i] (dY^T X)[o, i], [N, K/16]."""
        N, K = W.shape
        M = X.shape[0]
        if g is None:
            g = torch.empty(N, K // 16, dtype=torch.float32, device=X.device)
        cw = _SqControlWeight(N, K, _ptr(W), None)
        self._check(self._L.sq_control_grad(self._h, ctypes.byref(cw), _ptr(X), _ptr(dY), M, _ptr(g), _stream(stream)))
        return g

    def sq_lowrank_product(self, B: torch.Tensor, A: torch.Tensor, alpha_over_r: float,
                           out: Optional[torch.Tensor] = None, stream=None):
        """(alpha/r) B A, B [N, r] and A [r, G] bf16 -> fp32 [N, G]."""
        N, r = B.shape
        G = A.shape[1]
        if out is None:
            out = torch.empty(N, G, dtype=torch.float32, device=B.device)
        self._check(self._L.sq_lowrank_product(self._h, N, G, r, alpha_over_r, _ptr(B), _ptr(A), _ptr(out),
                                               _stream(stream)))
        return out
