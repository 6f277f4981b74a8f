"""Pins of the oracle's contractions (Sec. 3 forward y = x W'^T and its backward).

- L = sum(Y * dY) is linear in every effective scale s[n,b] and every X[m,k], so
  central differences equal g and dX up to float64 round-off, for any step.
- One block of g equals the dot product of its codes with the matching dW = dY^T X
  row segment, dW formed by numpy's matmul (brute force).
- With all scale bytes at 1.0 the decoded weight is the code matrix, so Y, dX and
  g reduce to numpy matmuls on the printed E2M1 alphabet.
"""
import numpy as np
import torch

from conftest import bf16_bits, read_golden

NV, MX = 0, 1


def _alphabet():
    printed = read_golden("e2m1_alphabet.txt")["_rows"][0]
    return np.array(printed + [-v for v in printed])


def _rand_codes(rng, N, K):
    nib = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    return nib, (nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8)


def _w_from_scales(nib, s_eff, B):
    return _alphabet()[nib] * np.repeat(s_eff, B, axis=1)


def test_scale_gradient_finite_differences_every_block(oracle_mod):
    rng = np.random.default_rng(21)
    for fmt, B in ((NV, 16), (MX, 32)):
        M, N, K = 5, 6, 64
        G = K // B
        nib, codes = _rand_codes(rng, N, K)
        s = rng.uniform(0.1, 2.0, size=(N, G))
        X = rng.standard_normal((M, K))
        dY = rng.standard_normal((M, N))
        g = oracle_mod.scale_grad_f64(fmt, codes, X, dY)
        for n in range(N):
            for b in range(G):
                h = 0.37
                sp, sm = s.copy(), s.copy()
                sp[n, b] += h
                sm[n, b] -= h
                Lp = (oracle_mod.fwd_f64(X, _w_from_scales(nib, sp, B)) * dY).sum()
                Lm = (oracle_mod.fwd_f64(X, _w_from_scales(nib, sm, B)) * dY).sum()
                fd = (Lp - Lm) / (2 * h)
                assert abs(fd - g[n, b]) <= 1e-9 * (1 + abs(g[n, b]))


def test_scale_gradient_directional_derivatives_c1_shape(oracle_mod):
    """At the 64x256x512 NVFP4 shape: <g, V> equals the central difference of L
    along random directions V over all 8192 scales."""
    rng = np.random.default_rng(22)
    M, N, K, B = 64, 256, 512, 16
    nib, codes = _rand_codes(rng, N, K)
    s = rng.uniform(0.01, 0.05, size=(N, K // B))
    X = rng.standard_normal((M, K))
    dY = rng.standard_normal((M, N)) * 1e-3
    g = oracle_mod.scale_grad_f64(NV, codes, X, dY)
    for _ in range(4):
        V = rng.standard_normal(s.shape)
        h = 1e-2
        Lp = (oracle_mod.fwd_f64(X, _w_from_scales(nib, s + h * V, B)) * dY).sum()
        Lm = (oracle_mod.fwd_f64(X, _w_from_scales(nib, s - h * V, B)) * dY).sum()
        fd = (Lp - Lm) / (2 * h)
        assert abs(fd - (g * V).sum()) <= 1e-9 * np.abs(g * V).sum()


def test_input_gradient_finite_differences(oracle_mod):
    rng = np.random.default_rng(23)
    M, N, K = 4, 5, 32
    W = rng.standard_normal((N, K))
    X = rng.standard_normal((M, K))
    dY = rng.standard_normal((M, N))
    dX = oracle_mod.dx_f64(dY, W)
    for m in range(M):
        for k in range(K):
            h = 0.5
            Xp, Xm = X.copy(), X.copy()
            Xp[m, k] += h
            Xm[m, k] -= h
            fd = ((oracle_mod.fwd_f64(Xp, W) - oracle_mod.fwd_f64(Xm, W)) * dY).sum() / (2 * h)
            assert abs(fd - dX[m, k]) <= 1e-10 * (1 + abs(dX[m, k]))


def test_scale_gradient_single_block_brute_force(oracle_mod):
    rng = np.random.default_rng(24)
    for fmt, B in ((NV, 16), (MX, 32)):
        M, N, K = 37, 9, 128
        nib, codes = _rand_codes(rng, N, K)
        X = rng.standard_normal((M, K))
        dY = rng.standard_normal((M, N))
        g = oracle_mod.scale_grad_f64(fmt, codes, X, dY)
        dW = dY.T @ X
        for (n, b) in ((0, 0), (3, 1), (N - 1, K // B - 1)):
            seg = slice(b * B, (b + 1) * B)
            want = float(np.dot(_alphabet()[nib[n, seg]], dW[n, seg]))
            assert abs(g[n, b] - want) <= 1e-12 * (1 + np.abs(dW[n, seg]).sum() * 6)


def test_unit_scales_reduce_to_matmul_on_codes(oracle_mod):
    """Scale byte = 1.0 (E4M3 0x38 with ws2 = 1, E8M0 127): the packed-format
    entry points equal numpy matmuls on the printed code alphabet."""
    rng = np.random.default_rng(25)
    for fmt, B, one in ((NV, 16, 0x38), (MX, 32, 127)):
        M, N, K = 19, 24, 96
        nib, codes = _rand_codes(rng, N, K)
        scales = np.full((N, K // B), one, dtype=np.uint8)
        x = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32)).to(torch.bfloat16)
        dy = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).to(torch.bfloat16)
        Xd = x.double().numpy()
        dYd = dy.double().numpy()
        C = _alphabet()[nib]
        Y = oracle_mod.fwd(fmt, codes, scales, 1.0, bf16_bits(x))
        dX = oracle_mod.dx(fmt, codes, scales, 1.0, bf16_bits(dy))
        g = oracle_mod.scale_grad(fmt, codes, bf16_bits(x), bf16_bits(dy))
        assert np.allclose(Y, Xd @ C.T, rtol=1e-13, atol=1e-12)
        assert np.allclose(dX, dYd @ C, rtol=1e-13, atol=1e-12)
        gref = (C * (dYd.T @ Xd)).reshape(N, K // B, B).sum(axis=2)
        assert np.allclose(g, gref, rtol=1e-12, atol=1e-12)


def test_per_block_scales_against_library_decode(oracle_mod):
    """Varying scale bytes: Y equals numpy X @ W^T with W built from the printed
    alphabet and torch's float8 decode of each byte (times ws2)."""
    rng = np.random.default_rng(26)
    M, N, K, B = 11, 16, 64, 16
    nib, codes = _rand_codes(rng, N, K)
    scales = rng.integers(0x10, 0x70, size=(N, K // B), dtype=np.uint8)
    ws2 = float(np.float32(0.0173))
    s = torch.from_numpy(scales).view(torch.float8_e4m3fn).double().numpy() * ws2
    W = _w_from_scales(nib, s, B)
    x = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32)).to(torch.bfloat16)
    dy = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).to(torch.bfloat16)
    Y = oracle_mod.fwd(NV, codes, scales, ws2, bf16_bits(x))
    dX = oracle_mod.dx(NV, codes, scales, ws2, bf16_bits(dy))
    assert np.allclose(Y, x.double().numpy() @ W.T, rtol=1e-13, atol=1e-13)
    assert np.allclose(dX, dy.double().numpy() @ W, rtol=1e-13, atol=1e-13)


def test_sampled_and_row_subsets_agree_with_full(oracle_mod):
    rng = np.random.default_rng(27)
    M, N, K = 33, 40, 96
    nib, codes = _rand_codes(rng, N, K)
    scales = rng.integers(0x20, 0x60, size=(N, K // 16), dtype=np.uint8)
    x = torch.from_numpy(rng.standard_normal((M, K)).astype(np.float32)).to(torch.bfloat16)
    dy = torch.from_numpy(rng.standard_normal((M, N)).astype(np.float32)).to(torch.bfloat16)
    Y = oracle_mod.fwd(NV, codes, scales, 0.5, bf16_bits(x))
    dX = oracle_mod.dx(NV, codes, scales, 0.5, bf16_bits(dy))
    ms = rng.integers(0, M, 50)
    ns = rng.integers(0, N, 50)
    ks = rng.integers(0, K, 50)
    assert np.allclose(oracle_mod.fwd_at(NV, codes, scales, 0.5, bf16_bits(x), ms, ns), Y[ms, ns], rtol=1e-13)
    assert np.allclose(oracle_mod.dx_at(NV, codes, scales, 0.5, bf16_bits(dy), ms, ks), dX[ms, ks], rtol=1e-13)
    mask = rng.integers(0, 2, size=(N, K // 16), dtype=np.uint8)
    g = oracle_mod.scale_grad(NV, codes, bf16_bits(x), bf16_bits(dy))
    gm = oracle_mod.scale_grad(NV, codes, bf16_bits(x), bf16_bits(dy), mask=mask)
    rows = np.array([3, 0, 39, 17])
    gr = oracle_mod.scale_grad(NV, codes, bf16_bits(x), bf16_bits(dy), mask=mask, rows=rows)
    assert np.array_equal(gm, g * mask)
    assert np.array_equal(gr, gm[rows])
