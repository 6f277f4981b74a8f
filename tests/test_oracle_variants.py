"""Pins of the oracle's scale-family variants (ablation appendix).

Least-squares code-preserving fit (the Spider paragraph: "solve per block for the
least-squares best code-preserving scale delta"):
- an update that already is a per-block multiple of the codes is recovered exactly;
- the residual dW - delta * c is orthogonal to c (numpy), and the fit equals numpy's
  lstsq on every block of a small plane;
- for an update with no relation to the codes the captured energy
  sum ||P(dW)||^2 / sum ||dW||^2 is 1 / block (the appendix's chance value, 6.25% for
  NVFP4) to within its sampling error, and 1/32 for MXFP4;
- an all-zero code block has no representable direction (delta 0).

Granularity ladder (a per-group additive scale delta, gd groups per row):
- the group gradient is the sum of its blocks' gradients, checked against numpy's
  block sums of code x dW from the brute-force dW = dY^T X; gd = G is the identity and
  gd = 1 the row sums;
- the group-delta latent is numpy's fp32 s + delta; zero delta returns every finite
  base byte; in range the byte is torch's E4M3 cast of latent / ws2.

Full-precision multiplicative control (W' = W (1 + dS) per row and block of 16):
- W' equals numpy's fp32 factor and product followed by torch's bf16 cast, and W for
  dS = 0;
- the coefficient gradient equals central differences of the (unrounded) bilinear
  form sum(dY * X W'^T); the low-rank coefficient plane equals numpy's (alpha/r) B A.
"""
import numpy as np
import torch

from conftest import read_golden

NV, MX = 0, 1
BLOCK = {NV: 16, MX: 32}


def _alphabet():
    printed = read_golden("e2m1_alphabet.txt")["_rows"][0]
    return np.array(printed + [-v for v in printed])


def _codes(rng, N, K):
    nib = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    return nib, (nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8)


def _bf16_bits(x):
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16), t.to(torch.float64).numpy()


def _e4m3(bytes_):
    return torch.from_numpy(np.asarray(bytes_, dtype=np.uint8)).view(torch.float8_e4m3fn).to(torch.float64).numpy()


def test_fit_recovers_a_scale_change_exactly(oracle_mod):
    """dW = c * t_b with dyadic t and codes whose <c, c> makes the division exact."""
    rng = np.random.default_rng(70)
    alpha = _alphabet()
    for fmt in (NV, MX):
        B = BLOCK[fmt]
        N, K = 6, 4 * B
        nib, codes = _codes(rng, N, K)
        t = rng.choice([0.25, -0.5, 1.0, 0.125, -2.0], size=(N, K // B))
        dW = alpha[nib] * np.repeat(t, B, axis=1)
        bits, dW64 = _bf16_bits(dW)
        assert np.array_equal(dW64, dW)                                 # exact in bf16
        delta, cap, tot, _ = oracle_mod.fit_scale_delta(fmt, codes, None, 1.0, bits)
        cc = (alpha[nib] ** 2).reshape(N, K // B, B).sum(axis=2)
        nz = cc > 0
        assert np.allclose(delta[nz], t[nz], rtol=1e-15, atol=0)
        assert np.allclose(cap[nz], tot[nz], rtol=1e-12)               # all energy captured
        assert (delta[~nz] == 0).all()


def test_fit_is_the_least_squares_solution(oracle_mod):
    rng = np.random.default_rng(71)
    alpha = _alphabet()
    B = 16
    N, K = 5, 6 * B
    nib, codes = _codes(rng, N, K)
    nib[0, :B] = 0                                                      # an all-zero code block
    codes = (nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8)
    bits, dW = _bf16_bits(rng.normal(0, 0.01, (N, K)))
    delta, cap, tot, _ = oracle_mod.fit_scale_delta(NV, codes, None, 1.0, bits)
    assert delta[0, 0] == 0.0 and cap[0, 0] == 0.0
    c = alpha[nib]
    for n in range(N):
        for b in range(K // B):
            cb, wb = c[n, b * B:(b + 1) * B], dW[n, b * B:(b + 1) * B]
            if not cb.any():
                continue
            ref = np.linalg.lstsq(cb[:, None], wb, rcond=None)[0][0]
            assert abs(delta[n, b] - ref) <= 1e-12 * (abs(ref) + 1e-12)
            assert abs(np.dot(wb - delta[n, b] * cb, cb)) <= 1e-12 * np.abs(wb).sum() * np.abs(cb).sum()
            assert abs(tot[n, b] - np.dot(wb, wb)) <= 1e-15 + 1e-12 * tot[n, b]


def test_projection_energy_is_one_over_block(oracle_mod):
    """sum ||P(dW)||^2 / sum ||dW||^2 for a Gaussian dW drawn without regard to the
    codes: 1/16 (NVFP4) and 1/32 (MXFP4). With n blocks the captured energy is a sum
    of n chi-square(1)-like terms, so its relative error is about sqrt(2/n); 40k
    blocks put 1/B within 2% at 6 sigma."""
    rng = np.random.default_rng(72)
    for fmt in (NV, MX):
        B = BLOCK[fmt]
        N, K = 400, 100 * B
        _, codes = _codes(rng, N, K)
        bits, _ = _bf16_bits(rng.normal(0, 0.02, (N, K)))
        _, cap, tot, _ = oracle_mod.fit_scale_delta(fmt, codes, None, 1.0, bits)
        ratio = cap.sum() / tot.sum()
        assert abs(ratio * B - 1.0) < 0.04, (fmt, ratio)


def test_fit_latent_is_scale_plus_delta(oracle_mod):
    rng = np.random.default_rng(73)
    N, K, ws2 = 8, 64, 2.0 ** -6
    _, codes = _codes(rng, N, K)
    scales = rng.integers(0x30, 0x60, size=(N, K // 16), dtype=np.uint8)
    bits, _ = _bf16_bits(rng.normal(0, 1e-3, (N, K)))
    delta, _, _, latent = oracle_mod.fit_scale_delta(NV, codes, scales, ws2, bits)
    ref = (_e4m3(scales).astype(np.float32) * np.float32(ws2)).astype(np.float32) + delta.astype(np.float32)
    assert np.array_equal(latent.view(np.uint32), ref.astype(np.float32).view(np.uint32))


def test_group_gradient_is_the_sum_of_its_blocks(oracle_mod):
    """g per block from the oracle's scale gradient; the group gradient equals numpy's
    sums of code x dW over each group's columns (brute-force dW = dY^T X)."""
    rng = np.random.default_rng(74)
    alpha = _alphabet()
    M, N, K, B = 7, 6, 256, 16
    nib, codes = _codes(rng, N, K)
    X = rng.normal(0, 1, (M, K))
    dY = rng.normal(0, 1, (M, N))
    g = oracle_mod.scale_grad_f64(NV, codes, X, dY).astype(np.float32)
    dW = dY.T @ X
    G = K // B
    for gd in (1, 2, 4, G):
        out = oracle_mod.group_reduce(g, gd)
        W = K // gd
        ref = (alpha[nib] * dW).reshape(N, gd, W).sum(axis=2)
        assert np.allclose(out, ref, rtol=1e-5, atol=1e-5 * np.abs(ref).max())
    assert np.array_equal(oracle_mod.group_reduce(g, G), g.astype(np.float64))
    assert np.allclose(oracle_mod.group_reduce(g, 1)[:, 0], g.astype(np.float64).sum(axis=1), rtol=1e-12)


def test_group_delta_projection(oracle_mod):
    rng = np.random.default_rng(75)
    N, G, gd, ws2 = 12, 32, 4, 2.0 ** -5
    base = np.concatenate([rng.integers(0x28, 0x70, size=(N, G - 1)), np.full((N, 1), 0x30)], axis=1).astype(np.uint8)
    b, m, nf, L = oracle_mod.project_group_delta(NV, base, np.zeros((N, gd), np.float32), ws2)
    assert np.array_equal(b, base) and (m == 1).all() and nf == 0
    delta = (rng.normal(0, 1, (N, gd)) * 0.3 * ws2 * 8).astype(np.float32)
    b, m, nf, L = oracle_mod.project_group_delta(NV, base, delta, ws2)
    s = (_e4m3(base).astype(np.float32) * np.float32(ws2)).astype(np.float32)
    ref = s + np.repeat(delta, G // gd, axis=1)
    assert np.array_equal(L.view(np.uint32), ref.astype(np.float32).view(np.uint32))
    inrange = (ref > 0) & (ref <= 448 * ws2)
    q = (ref / np.float32(ws2)).astype(np.float32)
    cast = torch.from_numpy(np.where(inrange, q, 1.0).astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8)
    assert np.array_equal(b[inrange], cast.numpy()[inrange])
    assert (b != base).mean() > 0.3


def test_control_weight_rounding(oracle_mod):
    """W' against numpy: fp32 factor 1 + dS, fp32 product, torch's bf16 (RNE) cast.
    dS = 0 returns W exactly; a product just above a bf16 midpoint rounds up."""
    rng = np.random.default_rng(80)
    N, K = 6, 64
    Wb, W64 = _bf16_bits(rng.normal(0, 0.05, (N, K)))
    dS = (rng.normal(0, 0.1, (N, K // 16))).astype(np.float32)
    Wp = oracle_mod.control_weight(Wb, dS)
    f = (np.float32(1.0) + dS).astype(np.float32)
    prod = (W64.astype(np.float32) * np.repeat(f, 16, axis=1)).astype(np.float32)
    ref = torch.from_numpy(prod).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(Wp, ref)
    assert np.array_equal(oracle_mod.control_weight(Wb, np.zeros_like(dS)), W64)
    # w = 1 + 2^-7 (bf16), f = 1 + 2^-8: 1 + 1.5 * 2^-7 + 2^-15 lies just above a midpoint -> 1 + 2^-6
    Wt, _ = _bf16_bits(np.full((1, 16), 1 + 2 ** -7))
    out = oracle_mod.control_weight(Wt, np.full((1, 1), 2 ** -8, np.float32))
    assert (out == 1 + 2 ** -6).all()


def test_control_gradient_is_the_derivative_of_the_bilinear_form(oracle_mod):
    """L(dS) = sum(dY * X (W (1 + dS))^T) is linear in dS (unrounded W'), so its central
    differences (numpy) equal g for every block."""
    rng = np.random.default_rng(81)
    M, N, K = 5, 4, 48
    Wb, W64 = _bf16_bits(rng.normal(0, 0.05, (N, K)))
    X = rng.normal(0, 1, (M, K))
    dY = rng.normal(0, 1, (M, N))
    g = oracle_mod.control_grad_f64(Wb, X, dY)

    def L(dS):
        Wp = W64 * (1 + np.repeat(dS, 16, axis=1))
        return float(np.sum(dY * (X @ Wp.T)))

    for n in range(N):
        for b in range(K // 16):
            E = np.zeros((N, K // 16))
            E[n, b] = 0.5
            fd = (L(E) - L(-E)) / 1.0
            assert abs(fd - g[n, b]) <= 1e-12 * (1 + np.abs(g).max())


def test_lowrank_product_matches_numpy(oracle_mod):
    rng = np.random.default_rng(82)
    Bb, B64 = _bf16_bits(rng.normal(0, 1, (9, 5)))
    Ab, A64 = _bf16_bits(rng.normal(0, 1, (5, 7)))
    assert np.allclose(oracle_mod.lowrank_product(Bb, Ab, 0.75), 0.75 * (B64 @ A64), rtol=1e-14, atol=1e-14)
