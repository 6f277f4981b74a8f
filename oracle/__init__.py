"""Float64 CPU oracle for the Scale-QLoRA scale-only training step (numpy front end).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` legs may import this module;
the product path (``paper_2609_04526_gb300``) never does. The arithmetic lives in
``sq_oracle.c`` (plain loops, float64 accumulation), which shares no code with the
CUDA sources. Each wrapper names the paper passage its C function follows.
"""
import ctypes
import os

import numpy as np

from . import build as _build

NVFP4 = 0
MXFP4 = 1
BLOCK = {NVFP4: 16, MXFP4: 32}

_lib = None

_i64 = ctypes.c_int64
_p = ctypes.c_void_p


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        L.or_e2m1.restype = ctypes.c_double
        L.or_e2m1.argtypes = [ctypes.c_int]
        L.or_e4m3.restype = ctypes.c_double
        L.or_e4m3.argtypes = [ctypes.c_int]
        L.or_e8m0.restype = ctypes.c_double
        L.or_e8m0.argtypes = [ctypes.c_int]
        L.or_e4m3_rne.restype = ctypes.c_int
        L.or_e4m3_rne.argtypes = [ctypes.c_float]
        L.or_round_log2.restype = ctypes.c_int
        L.or_round_log2.argtypes = [ctypes.c_float]
        L.or_decode_weight.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _p]
        L.or_fwd_f64.argtypes = [_i64, _i64, _i64, _p, _p, _p]
        L.or_dx_f64.argtypes = [_i64, _i64, _i64, _p, _p, _p]
        L.or_scale_grad_f64.argtypes = [_i64, _i64, _i64, ctypes.c_int, _p, _p, _p, _p, _i64, _p, _p]
        L.or_fwd.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _i64, _p, _p]
        L.or_dx.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _i64, _p, _p]
        L.or_scale_grad.argtypes = [ctypes.c_int, _i64, _i64, _p, _i64, _p, _p, _p, _i64, _p, _p]
        L.or_fwd_at.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _i64, _p, _i64, _p, _p, _p]
        L.or_dx_at.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _i64, _p, _i64, _p, _p, _p]
        L.or_project.argtypes = [ctypes.c_int, _i64, ctypes.c_float, _p, _p, _p, _p]
        L.or_merge.argtypes = [ctypes.c_int, _i64, ctypes.c_float, _p, _p, _p, _p]
        L.or_rollback.argtypes = [ctypes.c_int, _i64, ctypes.c_float, _p, _p, _p]
        L.or_swap.argtypes = [_i64, _p, _p, _p]
        L.or_count_diff.restype = _i64
        L.or_count_diff.argtypes = [_i64, _p, _p]
        L.or_lowrank_latent.restype = ctypes.c_float
        L.or_lowrank_latent.argtypes = [ctypes.c_int, ctypes.c_float, ctypes.c_float, ctypes.c_int, ctypes.c_uint8,
                                         _p, _p, _i64, _i64]
        L.or_project_lowrank.argtypes = [ctypes.c_int, _i64, _i64, ctypes.c_int, ctypes.c_float, ctypes.c_float,
                                         _p, _p, _p, _p, _p, _p, _p]
        L.or_lowrank_grad.argtypes = [_i64, _i64, ctypes.c_int, ctypes.c_double, _p, _p, _p, _p, _p]
        L.or_fit_scale_delta.argtypes = [ctypes.c_int, _i64, _i64, _p, _p, ctypes.c_float, _p, _p, _p, _p, _p]
        L.or_group_reduce.argtypes = [_i64, _i64, _i64, _p, _p]
        L.or_project_group_delta.argtypes = [ctypes.c_int, _i64, _i64, _i64, ctypes.c_float, _p, _p, _p, _p, _p, _p]
        L.or_control_weight.argtypes = [_i64, _i64, _p, _p, _p]
        L.or_control_grad.argtypes = [_i64, _i64, _i64, _p, _p, _p, _p]
        L.or_lowrank_product.argtypes = [_i64, _i64, ctypes.c_int, ctypes.c_double, _p, _p, _p]
        L.or_num_threads.restype = ctypes.c_int
        _lib = L
    return _lib


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(lib().or_num_threads())


# --- format decode (Sec. 2) -------------------------------------------------

def e2m1(nibble: int) -> float:
    return lib().or_e2m1(int(nibble))


def e4m3(byte: int) -> float:
    return lib().or_e4m3(int(byte))


def e8m0(byte: int) -> float:
    return lib().or_e8m0(int(byte))


def e4m3_rne(q: float) -> int:
    return lib().or_e4m3_rne(float(q))


def round_log2(L: float) -> int:
    return lib().or_round_log2(float(L))


def decode_weight(fmt, codes, scales, ws2, N, K):
    """W[n,k] = code[n,k] * eff_scale[n, k // block] in float64 (Sec. 2)."""
    codes = _c(codes, np.uint8)
    scales = _c(scales, np.uint8)
    W = np.empty((N, K), dtype=np.float64)
    lib().or_decode_weight(fmt, N, K, _ptr(codes), _ptr(scales), float(ws2), _ptr(W))
    return W


# --- contractions on float64 operands ---------------------------------------

def fwd_f64(X, W):
    """Y = X W^T (Sec. 3 forward)."""
    X = _c(X, np.float64)
    W = _c(W, np.float64)
    M, K = X.shape
    N = W.shape[0]
    Y = np.empty((M, N), dtype=np.float64)
    lib().or_fwd_f64(M, N, K, _ptr(X), _ptr(W), _ptr(Y))
    return Y


def dx_f64(dY, W):
    """dX = dY W (input gradient of Y = X W^T)."""
    dY = _c(dY, np.float64)
    W = _c(W, np.float64)
    M, N = dY.shape
    K = W.shape[1]
    dX = np.empty((M, K), dtype=np.float64)
    lib().or_dx_f64(M, N, K, _ptr(dY), _ptr(W), _ptr(dX))
    return dX


def scale_grad_f64(fmt, codes, X, dY, mask=None, rows=None):
    """g[n,b] = sum_{k in b} code[n,k] (dY^T X)[n,k], optionally times mask[n,b]."""
    X = _c(X, np.float64)
    dY = _c(dY, np.float64)
    codes = _c(codes, np.uint8)
    M, K = X.shape
    N = dY.shape[1]
    B = BLOCK[fmt]
    G = K // B
    mask_a = _c(mask, np.uint8) if mask is not None else None
    if rows is None:
        g = np.empty((N, G), dtype=np.float64)
        lib().or_scale_grad_f64(M, N, K, B, _ptr(codes), _ptr(X), _ptr(dY), _ptr(mask_a), 0, None, _ptr(g))
    else:
        rows = _c(rows, np.int64)
        g = np.empty((len(rows), G), dtype=np.float64)
        lib().or_scale_grad_f64(M, N, K, B, _ptr(codes), _ptr(X), _ptr(dY), _ptr(mask_a), len(rows),
                                _ptr(rows), _ptr(g))
    return g


# --- entry points on packed formats (bf16 activations as uint16 bit patterns) --

def fwd(fmt, codes, scales, ws2, X_bits):
    X_bits = _c(X_bits, np.uint16)
    codes = _c(codes, np.uint8)
    scales = _c(scales, np.uint8)
    M, K = X_bits.shape
    N = codes.shape[0]
    Y = np.empty((M, N), dtype=np.float64)
    lib().or_fwd(fmt, N, K, _ptr(codes), _ptr(scales), float(ws2), M, _ptr(X_bits), _ptr(Y))
    return Y


def dx(fmt, codes, scales, ws2, dY_bits):
    dY_bits = _c(dY_bits, np.uint16)
    codes = _c(codes, np.uint8)
    scales = _c(scales, np.uint8)
    M, N = dY_bits.shape
    K = codes.shape[1] * 2
    dX = np.empty((M, K), dtype=np.float64)
    lib().or_dx(fmt, N, K, _ptr(codes), _ptr(scales), float(ws2), M, _ptr(dY_bits), _ptr(dX))
    return dX


def scale_grad(fmt, codes, X_bits, dY_bits, mask=None, rows=None):
    X_bits = _c(X_bits, np.uint16)
    dY_bits = _c(dY_bits, np.uint16)
    codes = _c(codes, np.uint8)
    M, K = X_bits.shape
    N = dY_bits.shape[1]
    G = K // BLOCK[fmt]
    mask_a = _c(mask, np.uint8) if mask is not None else None
    if rows is None:
        g = np.empty((N, G), dtype=np.float64)
        lib().or_scale_grad(fmt, N, K, _ptr(codes), M, _ptr(X_bits), _ptr(dY_bits), _ptr(mask_a), 0, None,
                            _ptr(g))
    else:
        rows = _c(rows, np.int64)
        g = np.empty((len(rows), G), dtype=np.float64)
        lib().or_scale_grad(fmt, N, K, _ptr(codes), M, _ptr(X_bits), _ptr(dY_bits), _ptr(mask_a), len(rows),
                            _ptr(rows), _ptr(g))
    return g


def fwd_at(fmt, codes, scales, ws2, X_bits, ms, ns):
    X_bits = _c(X_bits, np.uint16)
    codes = _c(codes, np.uint8)
    scales = _c(scales, np.uint8)
    ms = _c(ms, np.int64)
    ns = _c(ns, np.int64)
    M, K = X_bits.shape
    N = codes.shape[0]
    out = np.empty(len(ms), dtype=np.float64)
    lib().or_fwd_at(fmt, N, K, _ptr(codes), _ptr(scales), float(ws2), M, _ptr(X_bits), len(ms), _ptr(ms),
                    _ptr(ns), _ptr(out))
    return out


def dx_at(fmt, codes, scales, ws2, dY_bits, ms, ks):
    dY_bits = _c(dY_bits, np.uint16)
    codes = _c(codes, np.uint8)
    scales = _c(scales, np.uint8)
    ms = _c(ms, np.int64)
    ks = _c(ks, np.int64)
    M, N = dY_bits.shape
    K = codes.shape[1] * 2
    out = np.empty(len(ms), dtype=np.float64)
    lib().or_dx_at(fmt, N, K, _ptr(codes), _ptr(scales), float(ws2), M, _ptr(dY_bits), len(ms), _ptr(ms),
                   _ptr(ks), _ptr(out))
    return out


# --- projection and merge (Sec. 3 QAST round_grid, clamp; Sec. 5 rollback) ---

def project(fmt, latent, ws2):
    """Returns (bytes, mask, nonfinite) for a latent scale plane (any shape)."""
    L = _c(latent, np.float32)
    out = np.empty(L.shape, dtype=np.uint8)
    mask = np.empty(L.shape, dtype=np.uint8)
    nf = ctypes.c_int64(0)
    lib().or_project(fmt, L.size, float(ws2), _ptr(L), _ptr(out), _ptr(mask), ctypes.byref(nf))
    return out, mask, int(nf.value)


def merge(fmt, latent, scales, ws2, want_delta=True):
    """Returns (new_scales, delta or None, changed). `scales` is not modified."""
    L = _c(latent, np.float32)
    s = np.array(scales, dtype=np.uint8, copy=True, order="C")
    delta = np.empty(L.shape, dtype=np.float32) if want_delta else None
    ch = ctypes.c_int64(0)
    lib().or_merge(fmt, L.size, float(ws2), _ptr(L), _ptr(s), _ptr(delta), ctypes.byref(ch))
    return s, delta, int(ch.value)


# --- rollback, hot-swap, audit (Sec. 5 Payoff 3, "Hot-swap") ----------------

def rollback(fmt, scales, delta, ws2):
    """Returns (restored bytes, changed): every byte replaced by the projection of
    fl32(s(byte) - delta). `scales` is not modified."""
    s = np.array(scales, dtype=np.uint8, copy=True, order="C")
    d = _c(delta, np.float32)
    assert d.shape == s.shape
    ch = ctypes.c_int64(0)
    lib().or_rollback(fmt, s.size, float(ws2), _ptr(d), _ptr(s), ctypes.byref(ch))
    return s, int(ch.value)


def swap(src, dst):
    """Returns (new plane, changed): dst overwritten by src. `dst` is not modified."""
    a = _c(src, np.uint8)
    d = np.array(dst, dtype=np.uint8, copy=True, order="C")
    assert a.shape == d.shape
    ch = ctypes.c_int64(0)
    lib().or_swap(a.size, _ptr(a), _ptr(d), ctypes.byref(ch))
    return d, int(ch.value)


def count_diff(a, b):
    x = _c(a, np.uint8).reshape(-1)
    y = _c(b, np.uint8).reshape(-1)
    assert x.size == y.size
    return int(lib().or_count_diff(x.size, _ptr(x), _ptr(y)))


# --- low-rank scale adapter (Sec. 3 "Scale-QLoRA forward") -------------------

def project_lowrank(fmt, base_scales, B_bits, A_bits, ws2, alpha_over_r):
    """The adapter's latent eff' = eff + (alpha/r) (B A) per block, in fp32 with the
    order fixed in sq_oracle.c, projected onto the grid (QAST round_grid + clamp).
    base_scales [N, G] u8; B_bits [N, r] and A_bits [r, G] are bf16 bit patterns.
    Returns (bytes, mask, nonfinite, latent)."""
    base = _c(base_scales, np.uint8)
    B = _c(B_bits, np.uint16)
    A = _c(A_bits, np.uint16)
    N, G = base.shape
    r = B.shape[1]
    assert B.shape == (N, r) and A.shape == (r, G)
    out = np.empty((N, G), dtype=np.uint8)
    mask = np.empty((N, G), dtype=np.uint8)
    latent = np.empty((N, G), dtype=np.float32)
    nf = ctypes.c_int(0)
    lib().or_project_lowrank(fmt, N, G, r, float(ws2), float(alpha_over_r), _ptr(base), _ptr(B), _ptr(A), _ptr(out),
                             _ptr(mask), ctypes.byref(nf), _ptr(latent))
    return out, mask, int(nf.value), latent


def lowrank_grad(gm, B_bits, A_bits, alpha_over_r):
    """Adapter gradients from the masked scale gradient gm [N, G] (fp32 values):
    dB = (alpha/r) gm A^T [N, r] and dA = (alpha/r) B^T gm [r, G], in float64."""
    g = _c(gm, np.float32)
    B = _c(B_bits, np.uint16)
    A = _c(A_bits, np.uint16)
    N, G = g.shape
    r = B.shape[1]
    assert B.shape == (N, r) and A.shape == (r, G)
    dB = np.empty((N, r), dtype=np.float64)
    dA = np.empty((r, G), dtype=np.float64)
    lib().or_lowrank_grad(N, G, r, float(alpha_over_r), _ptr(g), _ptr(B), _ptr(A), _ptr(dB), _ptr(dA))
    return dB, dA


# --- experts of an MoE linear (Sec. 3 "MoE: a batched grouped-expert kernel") -
# The quantized linears of an MoE layer are its experts: expert e owns the token
# rows offsets[e] .. offsets[e+1]-1 (sorted by expert) and computes, on those rows
# alone, exactly the dense step above with its own codes, scales and ws2.

def _expert_rows(offsets, e):
    return int(offsets[e]), int(offsets[e + 1])


def grouped_fwd(fmt, codes, scales, ws2, offsets, X_bits):
    """Y [M, N]: the forward of expert e on its rows, for every e.
    codes [E, N, K/2], scales [E, N, G] u8; ws2 one value per expert."""
    E, N = codes.shape[0], codes.shape[1]
    Y = np.zeros((int(offsets[E]), N), dtype=np.float64)
    for e in range(E):
        a, b = _expert_rows(offsets, e)
        if b > a:
            Y[a:b] = fwd(fmt, codes[e], scales[e], ws2[e], X_bits[a:b])
    return Y


def grouped_dx(fmt, codes, scales, ws2, offsets, dY_bits):
    """dX [M, K]: the input gradient of expert e on its rows, for every e."""
    E, K = codes.shape[0], codes.shape[2] * 2
    dX = np.zeros((int(offsets[E]), K), dtype=np.float64)
    for e in range(E):
        a, b = _expert_rows(offsets, e)
        if b > a:
            dX[a:b] = dx(fmt, codes[e], scales[e], ws2[e], dY_bits[a:b])
    return dX


def grouped_scale_grad(fmt, codes, offsets, X_bits, dY_bits, mask=None, experts=None):
    """g [E, N, G]: expert e's block-reduced scale gradient over its own rows (zero
    for an expert without rows), optionally times mask [E, N, G]. `experts` limits
    the work to those experts (the others are left zero)."""
    E, N, K = codes.shape[0], codes.shape[1], codes.shape[2] * 2
    G = K // BLOCK[fmt]
    g = np.zeros((E, N, G), dtype=np.float64)
    for e in (range(E) if experts is None else experts):
        a, b = _expert_rows(offsets, e)
        if b > a:
            g[e] = scale_grad(fmt, codes[e], X_bits[a:b], dY_bits[a:b], None if mask is None else mask[e])
    return g


def grouped_project(fmt, latent, ws2):
    """(bytes, mask, nonfinite) of every expert's latent plane [E, N, G], plane e
    projected with its own tensor scale ws2[e]."""
    L = _c(latent, np.float32)
    out = np.empty(L.shape, dtype=np.uint8)
    mask = np.empty(L.shape, dtype=np.uint8)
    nf = 0
    for e in range(L.shape[0]):
        out[e], mask[e], n = project(fmt, L[e], ws2[e])
        nf += n
    return out, mask, nf


def grouped_merge(fmt, latent, scales, ws2):
    """(new planes, on-grid deltas, changed bytes) of the merge of every expert's plane."""
    L = _c(latent, np.float32)
    new = np.empty(L.shape, dtype=np.uint8)
    delta = np.empty(L.shape, dtype=np.float32)
    ch = 0
    for e in range(L.shape[0]):
        new[e], delta[e], c = merge(fmt, L[e], scales[e], ws2[e])
        ch += c
    return new, delta, ch


def grouped_project_lowrank(fmt, base_scales, B_bits, A_bits, ws2, alpha_over_r):
    """Every expert's adapter latent and projection (project_lowrank per expert):
    base [E, N, G] u8, B [E, N, r] and A [E, r, G] bf16 bits, ws2 one value per expert.
    Returns (bytes, mask, nonfinite, latent) over all experts."""
    base = _c(base_scales, np.uint8)
    E = base.shape[0]
    out = np.empty(base.shape, dtype=np.uint8)
    mask = np.empty(base.shape, dtype=np.uint8)
    latent = np.empty(base.shape, dtype=np.float32)
    nf = 0
    for e in range(E):
        out[e], mask[e], n, latent[e] = project_lowrank(fmt, base[e], B_bits[e], A_bits[e], ws2[e], alpha_over_r)
        nf += n
    return out, mask, nf, latent


def grouped_lowrank_grad(gm, B_bits, A_bits, alpha_over_r):
    """Every expert's adapter gradients (lowrank_grad per expert): gm [E, N, G]."""
    E = gm.shape[0]
    dB = np.empty((E,) + B_bits.shape[1:], dtype=np.float64)
    dA = np.empty((E,) + A_bits.shape[1:], dtype=np.float64)
    for e in range(E):
        dB[e], dA[e] = lowrank_grad(gm[e], B_bits[e], A_bits[e], alpha_over_r)
    return dB, dA


# --- scale-family variants (ablation appendix) --------------------------------

def fit_scale_delta(fmt, codes, scales, ws2, dW_bits):
    """Least-squares code-preserving fit of a weight update dW [N, K] (bf16 bits):
    per block delta = <c, dW> / <c, c> (0 for an all-zero code block). Returns
    (delta, captured, total, latent): float64 [N, G] x 3 and the fp32 latent
    fl32(s(byte) + fl32(delta)) (None when scales is None)."""
    dW = _c(dW_bits, np.uint16)
    codes = _c(codes, np.uint8)
    N, K = dW.shape
    G = K // BLOCK[fmt]
    delta = np.empty((N, G), dtype=np.float64)
    cap = np.empty((N, G), dtype=np.float64)
    tot = np.empty((N, G), dtype=np.float64)
    latent = None
    sc = None
    if scales is not None:
        sc = _c(scales, np.uint8)
        latent = np.empty((N, G), dtype=np.float32)
    lib().or_fit_scale_delta(fmt, N, K, _ptr(codes), _ptr(sc), float(ws2), _ptr(dW), _ptr(delta), _ptr(cap),
                             _ptr(tot), _ptr(latent))
    return delta, cap, tot, latent


def group_reduce(g, gd):
    """Gradient of a per-group additive scale delta: the sum of each group's G / gd
    consecutive block gradients, float64 [N, gd]."""
    g = _c(g, np.float32)
    N, G = g.shape
    assert G % gd == 0
    out = np.empty((N, gd), dtype=np.float64)
    lib().or_group_reduce(N, G, int(gd), _ptr(g), _ptr(out))
    return out


def project_group_delta(fmt, base_scales, delta, ws2):
    """Projection of fl32(s(base byte) + delta[n, b // (G / gd)]). Returns
    (bytes, mask, nonfinite, latent)."""
    base = _c(base_scales, np.uint8)
    d = _c(delta, np.float32)
    N, G = base.shape
    gd = d.shape[1]
    assert d.shape[0] == N and G % gd == 0
    out = np.empty((N, G), dtype=np.uint8)
    mask = np.empty((N, G), dtype=np.uint8)
    latent = np.empty((N, G), dtype=np.float32)
    nf = ctypes.c_int64(0)
    lib().or_project_group_delta(fmt, N, G, int(gd), float(ws2), _ptr(base), _ptr(d), _ptr(out), _ptr(mask),
                                 ctypes.byref(nf), _ptr(latent))
    return out, mask, int(nf.value), latent


def control_weight(W_bits, dS):
    """W' = bf16(fl32(W * fl32(1 + dS[n, k // 16]))) of the multiplicative control, float64 [N, K]."""
    W = _c(W_bits, np.uint16)
    d = _c(dS, np.float32)
    N, K = W.shape
    assert d.shape == (N, K // 16)
    out = np.empty((N, K), dtype=np.float64)
    lib().or_control_weight(N, K, _ptr(W), _ptr(d), _ptr(out))
    return out


def control_grad_f64(W_bits, X, dY):
    """g[n, b] = sum over the block's columns of W[n, k] (dY^T X)[n, k], float64 [N, K/16]."""
    W = _c(W_bits, np.uint16)
    X = _c(X, np.float64)
    dY = _c(dY, np.float64)
    M, K = X.shape
    N = dY.shape[1]
    g = np.empty((N, K // 16), dtype=np.float64)
    lib().or_control_grad(M, N, K, _ptr(W), _ptr(X), _ptr(dY), _ptr(g))
    return g


def lowrank_product(B_bits, A_bits, alpha_over_r):
    """(alpha/r) B A in float64 from bf16 bits B [N, r], A [r, G]."""
    B = _c(B_bits, np.uint16)
    A = _c(A_bits, np.uint16)
    N, r = B.shape
    G = A.shape[1]
    out = np.empty((N, G), dtype=np.float64)
    lib().or_lowrank_product(N, G, r, float(alpha_over_r), _ptr(B), _ptr(A), _ptr(out))
    return out
