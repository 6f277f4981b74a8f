"""The C-ABI library loads without a GPU, exports every entry point the header
declares, and rejects bad arguments before touching CUDA."""
import ctypes
import os
import re

import pytest

from conftest import ROOT

pkg = pytest.importorskip("paper_2609_04526_gb300")


@pytest.fixture(scope="module")
def built():
    from paper_2609_04526_gb300 import build
    build.build()
    return pkg.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "scaleqlora.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sq_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_symbol(built):
    declared = _declared()
    assert set(declared) == set(pkg._lib.EXPORTS)
    for name in declared:
        assert hasattr(built, name), name


def test_status_strings(built):
    for code, name in pkg._lib.STATUS.items():
        assert built.sq_status_string(code).decode() == name
    assert built.sq_status_string(7).decode() == "SQ_ERR_UNKNOWN"


def test_null_handle_and_create(built):
    assert built.sq_fwd(None, None, None, 0, None, None) == -1
    assert built.sq_create(None) == -1
    h = pkg.Handle()
    h.close()


A16 = 0x10000  # a 16-byte aligned address that is never dereferenced (validation fails first)


def _w(fmt=0, N=256, K=512, codes=A16, scales=A16, ws2=0.01):
    return pkg._lib._SqWeight(fmt, N, K, codes, scales, ws2)


@pytest.mark.parametrize("w, why", [
    (None, "weight is NULL"),
    (_w(fmt=2), "unknown format"),
    (_w(N=0), "N=0"),
    (_w(N=12), "N=12"),
    (_w(K=48), "K=48"),
    (_w(K=-32), "K=-32"),
    (_w(codes=0), "codes"),
    (_w(codes=A16 + 8), "codes"),
    (_w(scales=0), "scales"),
    (_w(ws2=0.0), "ws2"),
    (_w(ws2=float("nan")), "ws2"),
    (_w(fmt=1, ws2=0.5), "MXFP4 ws2"),
])
def test_weight_validation(built, w, why):
    h = pkg.Handle()
    wp = ctypes.byref(w) if w is not None else None
    assert h.status_of("sq_fwd", wp, ctypes.c_void_p(A16), 4, ctypes.c_void_p(A16), None) == -1
    assert why.split("=")[0].split()[0] in h.last_error()


def test_buffer_and_token_validation(built):
    h = pkg.Handle()
    w = _w()
    vp = ctypes.c_void_p
    assert h.status_of("sq_fwd", ctypes.byref(w), vp(A16), -1, vp(A16), None) == -1
    assert h.status_of("sq_fwd", ctypes.byref(w), vp(A16), 1 << 31, vp(A16), None) == -1
    assert h.status_of("sq_fwd", ctypes.byref(w), vp(A16 + 2), 4, vp(A16), None) == -1
    assert h.status_of("sq_bwd_dx", ctypes.byref(w), vp(A16), 4, None, None) == -1
    assert h.status_of("sq_scale_grad", ctypes.byref(w), vp(A16), vp(A16), 4, None, None, None) == -1
    assert h.status_of("sq_project_scales", 0, 4, 16, 0.0, vp(A16), vp(A16), None, None, None) == -1
    assert h.status_of("sq_project_scales", 0, 4, 16, 1.0, vp(A16), vp(A16 + 1), None, None, None) == -1
    assert h.status_of("sq_project_scales", 1, 4, 16, 2.0, vp(A16), vp(A16), None, None, None) == -1
    assert h.status_of("sq_merge", 0, -1, 16, 1.0, vp(A16), vp(A16), None, None, None) == -1
    assert h.status_of("sq_merge", 0, 4, 16, 1.0, vp(A16), vp(A16), vp(A16 + 4), None, None) == -1


def test_scale_grad_workspace_validation(built):
    """The split query validates the weight, the token count and its outputs before
    it looks at a device."""
    h = pkg.Handle()
    vp = ctypes.c_void_p
    sp, nb = ctypes.c_int32(0), ctypes.c_int64(0)
    assert h.status_of("sq_scale_grad_workspace", ctypes.byref(_w(N=12)), 4096, ctypes.byref(sp), ctypes.byref(nb)) == -1
    assert h.status_of("sq_scale_grad_workspace", ctypes.byref(_w()), -1, ctypes.byref(sp), ctypes.byref(nb)) == -1
    assert h.status_of("sq_scale_grad_workspace", ctypes.byref(_w()), 4096, None, None) == -1
    assert h.status_of("sq_scale_grad_workspace", None, 4096, ctypes.byref(sp), None) == -1


def test_empty_batch_is_a_noop_without_device(built):
    """M == 0 for the forward / input gradient enqueues nothing."""
    h = pkg.Handle()
    w = _w()
    assert h.status_of("sq_fwd", ctypes.byref(w), None, 0, None, None) == 0
    assert h.status_of("sq_bwd_dx", ctypes.byref(w), None, 0, None, None) == 0


def test_binding_refuses_to_fall_back(tmp_path, monkeypatch):
    """Without the shared library the binding raises instead of computing elsewhere."""
    import paper_2609_04526_gb300._lib as L
    monkeypatch.setattr(L, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(L, "_lib", None)
    with pytest.raises(ImportError):
        L.load()


def _gw(fmt=0, E=3, N=64, K=128, codes=A16, scales=A16, ws2=(0.01, 0.02, 0.03)):
    L = pkg._lib
    arr = None if ws2 is None else (ctypes.c_float * len(ws2))(*ws2)
    w = L._SqGroupedWeight(fmt, E, N, K, codes, scales,
                           None if arr is None else ctypes.cast(arr, ctypes.POINTER(ctypes.c_float)))
    return w, arr


def _off(vals):
    return (ctypes.c_int64 * len(vals))(*vals)


def test_grouped_validation(built):
    """Grouped calls reject bad experts, tensor scales and token layouts before any
    device work; an empty batch is a no-op."""
    h = pkg.Handle()
    vp = ctypes.c_void_p
    good_off = _off([0, 4, 4, 9])
    cases = [
        (_gw(E=0, ws2=()), good_off, "E=0"),
        (_gw(ws2=None), good_off, "ws2"),                                   # NVFP4 needs ws2[E]
        (_gw(ws2=(0.01, float("inf"), 0.03)), good_off, "ws2[1]"),
        (_gw(fmt=1, ws2=(1.0, 0.5, 1.0)), good_off, "MXFP4"),
        (_gw(N=12), good_off, "N=12"),
        (_gw(K=48), good_off, "K=48"),
        (_gw(codes=A16 + 4), good_off, "codes"),
        (_gw(), _off([1, 4, 4, 9]), "offsets[0]"),
        (_gw(), _off([0, 4, 3, 9]), "non-decreasing"),
        (_gw(E=40000, N=65536, ws2=[1.0] * 40000), _off([0] * 40000 + [8]), "code rows"),
    ]
    for (w, keep), off, why in cases:
        assert h.status_of("sq_grouped_fwd", ctypes.byref(w), off, vp(A16), vp(A16), None) == -1, why
        assert why.split("[")[0].split("=")[0] in h.last_error(), (why, h.last_error())
    w, keep = _gw()
    assert h.status_of("sq_grouped_fwd", ctypes.byref(w), None, vp(A16), vp(A16), None) == -1
    assert h.status_of("sq_grouped_fwd", ctypes.byref(w), _off([0, 0, 0, 0]), None, None, None) == 0
    assert h.status_of("sq_grouped_bwd_dx", ctypes.byref(w), good_off, vp(A16 + 2), vp(A16), None) == -1
    assert h.status_of("sq_grouped_scale_grad", ctypes.byref(w), good_off, vp(A16), vp(A16), None, None,
                       None) == -1                                           # g is NULL
    assert h.status_of("sq_grouped_project_lowrank", ctypes.byref(w), 0, 1.0, vp(A16), vp(A16), vp(A16), None,
                       None, None, None) == -1                               # r = 0
    assert h.status_of("sq_grouped_lowrank_grad", 0, 8, 8, 4, 1.0, vp(A16), vp(A16), vp(A16), vp(A16), vp(A16),
                       None) == -1                                           # E = 0


def test_variant_validation(built):
    """The scale-family variants reject bad shapes, scales and groupings before any
    device work; the control's empty batch is a no-op."""
    h = pkg.Handle()
    vp = ctypes.c_void_p
    L = pkg._lib
    assert h.status_of("sq_fit_scale_delta", 0, 8, 48, 1.0, vp(A16), None, vp(A16), vp(A16), None, None, None,
                       None) == -1                                           # K % 32
    assert h.status_of("sq_fit_scale_delta", 0, 8, 64, float("nan"), vp(A16), None, vp(A16), vp(A16), None, None,
                       None, None) == -1                                     # ws2
    assert h.status_of("sq_group_reduce", 8, 6, 4, vp(A16), vp(A16), None) == -1        # 4 does not divide 6
    assert h.status_of("sq_group_reduce", 8, 6, 0, vp(A16), vp(A16), None) == -1
    assert h.status_of("sq_project_group_delta", 1, 8, 6, 2, 0.5, vp(A16), vp(A16), vp(A16), None, None, None,
                       None) == -1                                           # MXFP4 ws2
    bad_n = L._SqControlWeight(12, 64, A16, A16)
    assert h.status_of("sq_control_fwd", ctypes.byref(bad_n), vp(A16), 4, vp(A16), None) == -1
    bad_w = L._SqControlWeight(8, 64, A16 + 2, A16)
    assert h.status_of("sq_control_bwd_dx", ctypes.byref(bad_w), vp(A16), 4, vp(A16), None) == -1
    ok = L._SqControlWeight(8, 64, A16, A16)
    assert h.status_of("sq_control_fwd", ctypes.byref(ok), None, 0, None, None) == 0
    assert h.status_of("sq_lowrank_product", 8, 8, 300, 1.0, vp(A16), vp(A16), vp(A16), None) == -1   # r > 256


def test_plane_table_validation(built):
    """The multi-plane projection and merge check every plane (count, shape,
    alignment, ws2) before anything is launched; zero planes is a no-op."""
    h = pkg.Handle()
    P = pkg._lib._SqPlane

    def call(name, planes, n=None, fmt=0):
        arr = (P * max(1, len(planes)))(*planes)
        return h.status_of(name, fmt, len(planes) if n is None else n, arr, None)

    ok = P(8, 16, 0.5, A16, A16, A16, A16, A16, A16)
    for name in ("sq_project_planes", "sq_merge_planes"):
        assert call(name, []) == 0
        assert call(name, [ok], n=17) == -1 and "nplanes" in h.last_error()
        assert call(name, [ok], n=-1) == -1
        assert h.status_of(name, 0, 2, None, None) == -1
        assert call(name, [ok, P(8, 16, 0.0, A16, A16, None, None, None, None)]) == -1 and "ws2" in h.last_error()
        assert call(name, [P(8, 16, 2.0, A16, A16, None, None, None, None)], fmt=1) == -1
        assert call(name, [P(-8, 16, 1.0, A16, A16, None, None, None, None)]) == -1
        assert call(name, [P(1, 8, 1.0, A16, A16, None, None, None, None)]) == -1 and "multiple of 16" in h.last_error()
        assert call(name, [P(8, 16, 1.0, 0, A16, None, None, None, None)]) == -1 and "latent" in h.last_error()
        assert call(name, [P(8, 16, 1.0, A16, A16 + 4, None, None, None, None)]) == -1
    assert call("sq_project_planes", [P(8, 16, 1.0, A16, A16, A16 + 8, None, None, None)]) == -1
    assert call("sq_project_planes", [P(8, 16, 1.0, A16, A16, None, None, A16 + 2, None)]) == -1
    assert call("sq_merge_planes", [P(8, 16, 1.0, A16, A16, None, A16 + 8, None, None)]) == -1
    assert call("sq_merge_planes", [P(8, 16, 1.0, A16, A16, None, None, None, A16 + 4)]) == -1
