"""Pins of the oracle's grid projection and merge (Sec. 3 QAST round_grid, the
E4M3 ceiling clamp; Sec. 5 rollback) against torch's float8 cast, exact integer
arithmetic, and the paper's invariants (round trip, zero-delta identity,
byte-exact rollback, cross-grid non-identity)."""
import numpy as np
import torch

NV, MX = 0, 1


def _torch_e4m3(q):
    return torch.from_numpy(np.asarray(q, dtype=np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def _e4m3_grid():
    return torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float32).numpy()


def test_nvfp4_projection_matches_torch_cast_in_range(oracle_mod):
    """Inside the clamp the projection is the round-to-nearest-even E4M3 cast of
    fl32(L / ws2) (the non-saturating torch cast that overflows to NaN without the
    clamp, Sec. 3 stability recipe (iii))."""
    rng = np.random.default_rng(11)
    grid = _e4m3_grid()
    pos = grid[1:0x7F].astype(np.float64)
    mids = (pos[:-1] + pos[1:]) / 2.0                               # exact ties
    sub = np.array([2.0 ** -10, 1.5 * 2 ** -10, 3 * 2 ** -11, 2.0 ** -12], dtype=np.float64)
    dense = np.linspace(-448, 448, 200001)
    logu = np.exp(rng.uniform(np.log(1e-6), np.log(448), size=200000)) * rng.choice([-1, 1], size=200000)
    for ws2 in (1.0, 2.0 ** -9, 3.7e-5, 0.0123):
        q = np.concatenate([pos, mids, -mids, sub, -sub, dense, logu, [0.0, -0.0]]).astype(np.float32)
        L = (q.astype(np.float64) * ws2).astype(np.float32)
        cap = np.float32(448.0) * np.float32(ws2)
        inside = np.abs(L) <= cap
        b, m, nf = oracle_mod.project(NV, L, ws2)
        qq = (L / np.float32(ws2)).astype(np.float32)
        ref = _torch_e4m3(qq)
        assert nf == 0
        assert (m[inside] == 1).all() and (m[~inside] == 0).all()
        assert np.array_equal(b[inside], ref[inside])


def test_nvfp4_clamp_and_nan(oracle_mod):
    ws2 = 0.011
    cap = np.float32(448.0) * np.float32(ws2)
    L = np.array([cap, np.nextafter(cap, np.float32(np.inf)), cap * 3, np.inf,
                  -cap, -cap * 2, -np.inf, np.nan, 0.0, -0.0], dtype=np.float32)
    b, m, nf = oracle_mod.project(NV, L, ws2)
    assert list(b) == [0x7E, 0x7E, 0x7E, 0x7E, 0xFE, 0xFE, 0xFE, 0x7F, 0x00, 0x80]
    assert list(m) == [1, 0, 0, 0, 1, 0, 0, 0, 1, 1]
    assert nf == 1


def test_mxfp4_exact_round_log2_over_binade(oracle_mod):
    """All 2^23 fp32 values of [1, 2) (and of a subnormal binade) against an exact
    integer test: round up iff (2^23 + j)^2 > 2 * 2^46."""
    j = np.arange(1 << 23, dtype=np.int64)
    L = (1.0 + j / float(1 << 23)).astype(np.float32)
    b, m, nf = oracle_mod.project(MX, L, 1.0)
    up = (((1 << 23) + j) ** 2) > 2 * (1 << 46)
    assert np.array_equal(b.astype(np.int64), 127 + up.astype(np.int64))
    assert (m == 1).all() and nf == 0
    # scale the binade: L * 2^e lands on byte 127 + e + up
    for e in (-100, -5, 3, 90):
        b2, _, _ = oracle_mod.project(MX, (L * np.float32(2.0 ** e)).astype(np.float32), 1.0)
        assert np.array_equal(b2.astype(np.int64), 127 + e + up.astype(np.int64))
    # subnormal fp32 binade [2^-140, 2^-139): m = 1 + j'/2^9 with 9 mantissa bits
    jj = np.arange(1 << 9, dtype=np.int64)
    Ls = (np.ldexp(1.0 + jj / 512.0, -140)).astype(np.float32)
    bs, ms, _ = oracle_mod.project(MX, Ls, 1.0)
    ups = (((1 << 9) + jj) ** 2) > 2 * (1 << 18)
    e = -140 + ups.astype(np.int64)
    assert (bs == 0).all() and (ms == 0).all() and (e + 127 < 0).all()


def test_mxfp4_edges(oracle_mod):
    L = np.array([0.0, -0.0, -1.0, np.inf, -np.inf, np.nan, 2.0 ** -127, 2.0 ** 127,
                  1.5 * 2.0 ** 127, 2.0 ** -127 * 1.41], dtype=np.float32)
    b, m, nf = oracle_mod.project(MX, L, 1.0)
    assert list(b) == [0, 0, 0, 254, 0, 255, 0, 254, 254, 0]
    assert list(m) == [0, 0, 0, 0, 0, 0, 1, 1, 0, 1]
    assert nf == 1


def test_round_trip_every_byte(oracle_mod):
    """Merge is a round trip on the scale plane (Sec. 3): projecting the decoded
    on-grid scale of any finite byte returns that byte."""
    rng = np.random.default_rng(2)
    grid = _e4m3_grid()
    for ws2 in [1.0, 2.0 ** -9, 0.004413, 7.1e-6] + list(rng.uniform(1e-6, 1.0, size=4)):
        ws2 = float(np.float32(ws2))
        bytes_ = np.array([b for b in range(256) if b not in (0x7F, 0xFF)], dtype=np.uint8)
        L = (grid[bytes_] * np.float32(ws2)).astype(np.float32)
        b, m, _ = oracle_mod.project(NV, L, ws2)
        assert np.array_equal(b, bytes_)
        assert (m == 1).all()
    bytes_ = np.arange(255, dtype=np.uint8)
    L = np.ldexp(np.float32(1.0), bytes_.astype(np.int32) - 127).astype(np.float32)
    b, m, _ = oracle_mod.project(MX, L, 1.0)
    assert np.array_equal(b, bytes_)


def test_merge_zero_delta_is_identity(oracle_mod):
    """A zero-delta re-projection moves zero bytes (Appendix census control)."""
    rng = np.random.default_rng(3)
    old = rng.integers(0, 0x7F, size=(64, 32), dtype=np.uint8)
    ws2 = 0.003
    L = (_e4m3_grid()[old] * np.float32(ws2)).astype(np.float32)
    new, delta, ch = oracle_mod.merge(NV, L, old, ws2)
    assert ch == 0 and np.array_equal(new, old) and (delta == 0).all()


def test_merge_changed_count_and_rollback(oracle_mod):
    """Subtracting the on-grid delta restores the base bytes exactly (Sec. 5,
    Payoff 3); the raw latent delta would not."""
    rng = np.random.default_rng(4)
    for fmt, ws2 in ((NV, 0.0021), (MX, 1.0)):
        if fmt == NV:
            old = rng.integers(0x08, 0x7E, size=(128, 64), dtype=np.uint8)
            s_old = (_e4m3_grid()[old] * np.float32(ws2)).astype(np.float32)
        else:
            old = rng.integers(100, 140, size=(128, 64), dtype=np.uint8)
            s_old = np.ldexp(np.float32(1.0), old.astype(np.int32) - 127).astype(np.float32)
        L = (s_old * (1.0 + 0.2 * rng.standard_normal(old.shape))).astype(np.float32)
        L = np.abs(L)
        new, delta, ch = oracle_mod.merge(fmt, L, old, ws2)
        assert ch == int((new != old).sum()) and ch > 0
        proj, _, _ = oracle_mod.project(fmt, L, ws2)
        assert np.array_equal(new, proj)
        if fmt == NV:
            s_new = (_e4m3_grid()[new] * np.float32(ws2)).astype(np.float32)
        else:
            s_new = np.ldexp(np.float32(1.0), new.astype(np.int32) - 127).astype(np.float32)
        back = (s_new - delta).astype(np.float32)
        rb, _, _ = oracle_mod.project(fmt, back, ws2)
        assert np.array_equal(rb, old)
        raw = (s_new - (L - s_old)).astype(np.float32)
        rraw, _, _ = oracle_mod.project(fmt, np.abs(raw), ws2)
        assert not np.array_equal(rraw, old)


def test_cross_grid_merge_is_not_identity(oracle_mod):
    """An E4M3-trained on-grid scale merged onto the E8M0 grid re-rounds (Appendix
    grid ablation): most non-power-of-two E4M3 scales move."""
    ws2 = 1.0
    grid = _e4m3_grid()
    bytes_ = np.arange(0x08, 0x7F, dtype=np.uint8)
    s = (grid[bytes_] * np.float32(ws2)).astype(np.float32)
    b, _, _ = oracle_mod.project(MX, s, 1.0)
    back = np.ldexp(1.0, b.astype(np.int32) - 127)
    moved = back != s
    non_pow2 = (bytes_ & 7) != 0
    assert moved[non_pow2].all() and not moved[~non_pow2].any()
