"""Pins of the oracle's rollback, scale-only swap and byte audit (Sec. 5 Payoff 3
"invertible merges and rollback", the hot-swap paragraph, the byte-level audit):
against the paper's invariants (merge followed by rollback with the on-grid delta
is the identity, the raw delta is not) and numpy's element-wise definitions."""
import numpy as np
import torch

NV, MX = 0, 1


def _scale(fmt, bytes_, ws2):
    if fmt == NV:
        g = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float32).numpy()
        return (g[bytes_] * np.float32(ws2)).astype(np.float32)
    return np.ldexp(np.float32(1.0), bytes_.astype(np.int32) - 127).astype(np.float32)


def test_merge_then_rollback_restores_the_base_bytes(oracle_mod):
    """A merge followed by a rollback with the on-grid delta it produced gives back
    the base plane byte for byte, whenever each merged scale is within a factor 2 of
    its base (then s_new - s_old is exact in fp32, Sterbenz), which covers realistic
    adapters; subtracting the raw training delta instead leaves bytes off."""
    rng = np.random.default_rng(8)
    for fmt, ws2 in ((NV, 0.0021), (NV, 1.0 / (6 * 448)), (NV, 1.0), (MX, 1.0)):
        if fmt == NV:
            old = rng.integers(0x10, 0x76, size=(256, 96), dtype=np.uint8)
        else:
            old = rng.integers(60, 190, size=(256, 96), dtype=np.uint8)
        s_old = _scale(fmt, old, ws2)
        L = (s_old * np.exp(rng.uniform(-0.6, 0.6, size=old.shape))).astype(np.float32)   # within a factor 2
        new, delta, ch = oracle_mod.merge(fmt, L, old, ws2)
        assert ch > 0.05 * old.size
        s_new = _scale(fmt, new, ws2)
        assert (s_new <= 2 * s_old).all() and (s_new >= s_old / 2).all()
        back, ch2 = oracle_mod.rollback(fmt, new, delta, ws2)
        assert np.array_equal(back, old) and ch2 == ch
        raw = (L - s_old).astype(np.float32)                                 # the training delta
        off, _ = oracle_mod.rollback(fmt, new, raw, ws2)
        assert oracle_mod.count_diff(off, old) > 0


def test_rollback_of_an_unchanged_plane_is_the_identity(oracle_mod):
    """Zero delta: every finite byte maps to itself (the merge round trip; -0 - 0
    stays -0, so even the negative-zero byte is kept)."""
    for fmt, ws2, rng_b in ((NV, 3.7e-5, np.r_[0:0x7F, 0x80:0xFF]), (NV, 1.0, np.r_[0:0x7F]), (MX, 1.0, np.r_[0:255])):
        b = np.tile(rng_b.astype(np.uint8), (2, 1))
        back, ch = oracle_mod.rollback(fmt, b, np.zeros(b.shape, dtype=np.float32), ws2)
        assert np.array_equal(back, b) and ch == 0


def test_swap_and_count_diff_match_numpy(oracle_mod):
    rng = np.random.default_rng(9)
    a = rng.integers(0, 256, size=(300, 77), dtype=np.uint8)
    b = a.copy()
    flip = rng.random(a.shape) < 0.047
    b[flip] = (b[flip] + rng.integers(1, 256, size=int(flip.sum()))).astype(np.uint8)
    assert oracle_mod.count_diff(a, b) == int((a != b).sum()) == int(flip.sum())
    new, ch = oracle_mod.swap(b, a)
    assert np.array_equal(new, b) and ch == int(flip.sum())
    assert oracle_mod.count_diff(a, a) == 0
