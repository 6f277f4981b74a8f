"""Pins of the oracle's low-rank scale adapter (Sec. 3 "Scale-QLoRA forward":
Delta S = (B A)(alpha/r), eff' = eff + Delta S per block, projected by the QAST
round_grid with the ceiling clamp; the adapter gradients are the derivatives of
that bilinear form). Each check compares against something the oracle does not
compute itself: numpy fp32/fp64 arithmetic, torch's float8 cast, or central
finite differences of the bilinear form."""
import numpy as np
import torch

NV, MX = 0, 1


def _bf16(x):
    """float array -> (bf16 bit patterns, the exact float64 values of those bf16s)."""
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


def _e4m3_f64(bytes_):
    return torch.from_numpy(np.asarray(bytes_, dtype=np.uint8)).view(torch.float8_e4m3fn).to(torch.float64).numpy()


def test_zero_adapter_is_the_base_plane(oracle_mod):
    """B = 0: eff' is the base effective scale (one fp32 multiply E4M3(byte)*ws2, or
    2^(byte-127)), and projecting it returns every finite base byte unchanged (the
    merge round trip, Sec. 3) -- except the negative-zero byte 0x80: eff + Delta S is
    -0 + (+0) = +0 in IEEE arithmetic, which projects to 0x00 (the same zero scale)."""
    rng = np.random.default_rng(5)
    r = 7
    for ws2 in (1.0, 2.0 ** -9, 3.7e-5):
        base = np.concatenate([np.arange(0, 0x7F), np.arange(0x80, 0xFF)]).astype(np.uint8)  # every finite byte
        base = np.tile(base, (3, 1))
        N, G = base.shape
        Bb, _ = _bf16(np.zeros((N, r)))
        Ab, _ = _bf16(rng.normal(0, 1, (r, G)))
        b, m, nf, L = oracle_mod.project_lowrank(NV, base, Bb, Ab, ws2, 2.0)
        eff32 = (_e4m3_f64(base).astype(np.float32) * np.float32(ws2)).astype(np.float32)
        nz = base != 0x80
        assert np.array_equal(L[nz].view(np.uint32), eff32[nz].view(np.uint32))
        assert (L[~nz].view(np.uint32) == 0).all()                        # +0, not -0
        expect = np.where(nz, base, np.uint8(0))
        assert np.array_equal(b, expect) and nf == 0 and (m == 1).all()
    base = np.tile(np.arange(0, 255, dtype=np.uint8), (2, 1))
    Bb, _ = _bf16(np.zeros((2, r)))
    Ab, _ = _bf16(rng.normal(0, 1, (r, base.shape[1])))
    b, m, nf, L = oracle_mod.project_lowrank(MX, base, Bb, Ab, 1.0, 0.5)
    assert np.array_equal(b, base) and nf == 0
    assert np.array_equal(L.astype(np.float64), np.ldexp(1.0, base.astype(np.int64) - 127))


def test_latent_matches_float64_within_the_fp32_error_bound(oracle_mod):
    """eff' against numpy's float64 eff + (alpha/r) B @ A: the fp32 evaluation (one
    product for eff, r fused multiply-adds, one fused multiply-add) stays within
    2^-23 (|eff| + (alpha/r)(r+2) sum_j |B_j A_j| + |eff'|). A dropped term, a wrong
    sign or a transposed factor misses this by orders of magnitude."""
    rng = np.random.default_rng(17)
    for N, G, r, aor, ws2 in ((64, 48, 58, 2.0, 1.0 / (6 * 448)), (33, 80, 13, 0.25, 3.1e-4), (16, 16, 1, 1.0, 1.0)):
        base = rng.integers(0x20, 0x70, size=(N, G), dtype=np.uint8)
        eff64 = _e4m3_f64(base) * ws2
        scale = float(np.median(eff64))
        Bb, B64 = _bf16(rng.normal(0, 1, (N, r)) * np.sqrt(scale))
        Ab, A64 = _bf16(rng.normal(0, 1, (r, G)) * np.sqrt(scale) * 0.1)
        _, _, _, L = oracle_mod.project_lowrank(NV, base, Bb, Ab, ws2, aor)
        L64 = eff64 + aor * (B64 @ A64)
        absprod = np.abs(B64) @ np.abs(A64)
        bound = 2.0 ** -23 * (np.abs(eff64) + aor * (r + 2) * absprod + np.abs(L64))
        assert (np.abs(L.astype(np.float64) - L64) <= bound).all()
        # and the correction is really there: it moves the latent by far more than the bound
        assert np.abs(L64 - eff64).max() > 100 * bound.max()


def test_exact_case_bytes_match_the_torch_cast(oracle_mod):
    """With power-of-two ws2 and small dyadic B, A every fp32 step is exact, so eff'
    equals the float64 value and the projected byte is torch's RNE float8_e4m3fn
    cast of eff'/ws2 (inside the clamp)."""
    rng = np.random.default_rng(23)
    N, G, r, aor, ws2 = 40, 64, 3, 0.5, 2.0 ** -6
    base = rng.integers(0x30, 0x60, size=(N, G), dtype=np.uint8)
    Bb, B64 = _bf16(rng.choice([0.0, 0.5, -0.5, 1.0, -1.0, 2.0], size=(N, r)) * ws2)
    Ab, A64 = _bf16(rng.choice([0.0, 0.25, -0.25, 1.0, -1.0], size=(r, G)))
    b, m, nf, L = oracle_mod.project_lowrank(NV, base, Bb, Ab, ws2, aor)
    L64 = _e4m3_f64(base) * ws2 + aor * (B64 @ A64)
    assert np.array_equal(L.astype(np.float64), L64)
    q = (L / np.float32(ws2)).astype(np.float32)
    ref = torch.from_numpy(q).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert (np.abs(L64) <= 448 * ws2).all() and np.array_equal(b, ref) and (m == 1).all() and nf == 0


def test_adapter_above_the_ceiling_is_clamped_and_masked(oracle_mod):
    """Latents the adapter pushes above 448*ws2 project to the E4M3 maximum (0x7E)
    with mask 0, so no gradient leaks above the ceiling (Sec. 3 stability recipe
    (ii)); the rest keep mask 1."""
    ws2 = 2.0 ** -4
    base = np.full((4, 16), 0x7D, dtype=np.uint8)                       # 416 * ws2, just under the ceiling
    Bb, _ = _bf16(np.array([[64.0 * ws2], [0.0], [-64.0 * ws2], [1.0 * ws2]]))
    Ab, _ = _bf16(np.ones((1, 16)))
    b, m, nf, L = oracle_mod.project_lowrank(NV, base, Bb, Ab, ws2, 1.0)
    assert (b[0] == 0x7E).all() and (m[0] == 0).all()                  # 480 * ws2 > cap
    assert (b[1] == 0x7D).all() and (m[1] == 1).all()
    assert (m[2] == 1).all() and (m[3] == 1).all() and nf == 0


def test_adapter_gradients_match_central_differences(oracle_mod):
    """F(B, A) = sum gm * (alpha/r) (B A) is linear in B and in A, so central
    differences of F (numpy, float64) equal dF/dB and dF/dA up to round-off, for
    every entry."""
    rng = np.random.default_rng(31)
    N, G, r, aor = 24, 32, 5, 0.75
    gm = rng.normal(0, 1, (N, G)).astype(np.float32)
    gm[rng.random((N, G)) < 0.2] = 0.0                                  # masked blocks
    Bb, B64 = _bf16(rng.normal(0, 0.05, (N, r)))
    Ab, A64 = _bf16(rng.normal(0, 0.05, (r, G)))
    dB, dA = oracle_mod.lowrank_grad(gm, Bb, Ab, aor)
    g64 = gm.astype(np.float64)

    def F(Bx, Ax):
        return float(np.sum(g64 * (aor * (Bx @ Ax))))

    h = 0.5
    for n in range(N):
        for j in range(r):
            E = np.zeros_like(B64)
            E[n, j] = h
            fd = (F(B64 + E, A64) - F(B64 - E, A64)) / (2 * h)
            assert abs(fd - dB[n, j]) <= 1e-12 * (1 + np.abs(g64).sum())
    for j in range(r):
        for b in range(G):
            E = np.zeros_like(A64)
            E[j, b] = h
            fd = (F(B64, A64 + E) - F(B64, A64 - E)) / (2 * h)
            assert abs(fd - dA[j, b]) <= 1e-12 * (1 + np.abs(g64).sum())


def test_rank_one_all_ones_reduces_to_row_and_weighted_column_sums(oracle_mod):
    """r = 1, A = 1: dB is (alpha/r) times the row sums of gm and dA the B-weighted
    column sums (numpy reductions)."""
    rng = np.random.default_rng(41)
    N, G, aor = 50, 40, 3.0
    gm = rng.normal(0, 1, (N, G)).astype(np.float32)
    Bb, B64 = _bf16(rng.normal(0, 1, (N, 1)))
    Ab, _ = _bf16(np.ones((1, G)))
    dB, dA = oracle_mod.lowrank_grad(gm, Bb, Ab, aor)
    assert np.allclose(dB[:, 0], aor * gm.astype(np.float64).sum(axis=1), rtol=1e-13, atol=1e-12)
    assert np.allclose(dA[0], aor * (B64[:, 0:1] * gm.astype(np.float64)).sum(axis=0), rtol=1e-13, atol=1e-12)
