"""Pins of the oracle's grouped-expert contractions (Sec. 3 "MoE: a batched
grouped-expert kernel": the quantized linears of an MoE layer are its experts, and
each expert computes the dense step on the tokens routed to it).

- Brute force on tiny inputs: pure-Python loops that assign every token row to
  its expert by scanning the offsets, decode the weights from the printed E2M1
  alphabet, torch's float8_e4m3fn cast and 2^(byte - 127), and sum in float64.
- The scale gradient against the forward it differentiates: Y is linear in every
  expert's effective scales, so sum g[e] * V[e] equals the change of
  L = sum(Y * dY) along V, formed with numpy matmuls on each expert's rows.
- Relabelling the experts (weights, ws2 and token blocks together) relabels the
  outputs; an expert without tokens contributes no rows and a zero gradient.
"""
import numpy as np
import torch

from conftest import bf16_bits, read_golden

NV, MX = 0, 1
BLOCK = {NV: 16, MX: 32}


def _alphabet():
    printed = read_golden("e2m1_alphabet.txt")["_rows"][0]
    return np.array(printed + [-v for v in printed])


def _experts(rng, fmt, E, N, K):
    """Codes [E, N, K/2], scale bytes [E, N, G], ws2 [E] and the nibbles."""
    nib = rng.integers(0, 16, size=(E, N, K), dtype=np.uint8)
    codes = (nib[:, :, 0::2] | (nib[:, :, 1::2] << 4)).astype(np.uint8)
    G = K // BLOCK[fmt]
    if fmt == NV:
        scales = rng.integers(0x28, 0x60, size=(E, N, G), dtype=np.uint8)
        ws2 = [float(2.0 ** rng.integers(-8, -2) * (1 + e / 8)) for e in range(E)]   # distinct per expert
    else:
        scales = rng.integers(118, 132, size=(E, N, G), dtype=np.uint8)
        ws2 = [1.0] * E
    return nib, codes, scales, ws2


def _bf16(rng, shape, scale=1.0):
    t = torch.from_numpy(rng.standard_normal(shape) * scale).to(torch.bfloat16)
    return bf16_bits(t), t.to(torch.float64).numpy()


def _eff(fmt, byte, ws2):
    if fmt == NV:
        return float(torch.tensor([int(byte)], dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float64)) * ws2
    return 2.0 ** (int(byte) - 127)


def _offsets(counts):
    return np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)


def test_brute_force_tiny_both_formats(oracle_mod):
    rng = np.random.default_rng(61)
    alpha = _alphabet()
    for fmt in (NV, MX):
        E, N, K = 3, 8, 64
        B = BLOCK[fmt]
        counts = [3, 0, 2]
        off = _offsets(counts)
        M = int(off[-1])
        nib, codes, scales, ws2 = _experts(rng, fmt, E, N, K)
        Xb, X = _bf16(rng, (M, K))
        dYb, dY = _bf16(rng, (M, N))
        Y = oracle_mod.grouped_fwd(fmt, codes, scales, ws2, off, Xb)
        dX = oracle_mod.grouped_dx(fmt, codes, scales, ws2, off, dYb)
        g = oracle_mod.grouped_scale_grad(fmt, codes, off, Xb, dYb)

        def expert_of(m):
            for e in range(E):
                if off[e] <= m < off[e + 1]:
                    return e
            raise AssertionError(m)

        def w(e, n, k):
            return alpha[nib[e, n, k]] * _eff(fmt, scales[e, n, k // B], ws2[e])

        for m in range(M):
            e = expert_of(m)
            for n in range(N):
                ref = sum(X[m, k] * w(e, n, k) for k in range(K))
                assert abs(Y[m, n] - ref) <= 1e-12 * (1 + abs(ref))
            for k in range(K):
                ref = sum(dY[m, n] * w(e, n, k) for n in range(N))
                assert abs(dX[m, k] - ref) <= 1e-12 * (1 + abs(ref))
        for e in range(E):
            for n in range(N):
                for b in range(K // B):
                    ref = 0.0
                    for k in range(b * B, (b + 1) * B):
                        ref += alpha[nib[e, n, k]] * sum(dY[m, n] * X[m, k] for m in range(off[e], off[e + 1]))
                    assert abs(g[e, n, b] - ref) <= 1e-12 * (1 + abs(ref))
        assert not g[1].any()                                            # expert 1 has no tokens


def test_scale_gradient_is_the_derivative_of_each_experts_forward(oracle_mod):
    """<g, V> = L(s + V) - L(s) exactly in exact arithmetic (L is linear in s), with
    L = sum over experts of sum(dY_e * X_e W_e(s)^T) formed by numpy matmuls."""
    rng = np.random.default_rng(62)
    alpha = _alphabet()
    for fmt in (NV, MX):
        E, N, K = 4, 16, 128
        B = BLOCK[fmt]
        counts = [7, 1, 0, 12]
        off = _offsets(counts)
        nib, codes, _, _ = _experts(rng, fmt, E, N, K)
        Xb, X = _bf16(rng, (int(off[-1]), K))
        dYb, dY = _bf16(rng, (int(off[-1]), N))
        g = oracle_mod.grouped_scale_grad(fmt, codes, off, Xb, dYb)
        for _ in range(3):
            V = rng.standard_normal((E, N, K // B))
            dL = 0.0
            for e in range(E):
                a, b = off[e], off[e + 1]
                Wv = alpha[nib[e]] * np.repeat(V[e], B, axis=1)
                dL += float(np.sum(dY[a:b] * (X[a:b] @ Wv.T)))
            assert abs(float(np.sum(g * V)) - dL) <= 1e-10 * (1 + np.abs(g).sum())


def test_relabelling_experts_relabels_outputs(oracle_mod):
    rng = np.random.default_rng(63)
    E, N, K = 5, 16, 64
    counts = [4, 0, 9, 1, 6]
    off = _offsets(counts)
    nib, codes, scales, ws2 = _experts(rng, NV, E, N, K)
    M = int(off[-1])
    Xb, _ = _bf16(rng, (M, K))
    dYb, _ = _bf16(rng, (M, N))
    mask = rng.integers(0, 2, size=(E, N, K // 16), dtype=np.uint8)
    Y = oracle_mod.grouped_fwd(NV, codes, scales, ws2, off, Xb)
    dX = oracle_mod.grouped_dx(NV, codes, scales, ws2, off, dYb)
    g = oracle_mod.grouped_scale_grad(NV, codes, off, Xb, dYb, mask=mask)
    perm = [3, 0, 4, 2, 1]                               # new expert i is old expert perm[i]
    rows = np.concatenate([np.arange(off[p], off[p + 1]) for p in perm]).astype(np.int64)
    off2 = _offsets([counts[p] for p in perm])
    Y2 = oracle_mod.grouped_fwd(NV, codes[perm], scales[perm], [ws2[p] for p in perm], off2, Xb[rows])
    dX2 = oracle_mod.grouped_dx(NV, codes[perm], scales[perm], [ws2[p] for p in perm], off2, dYb[rows])
    g2 = oracle_mod.grouped_scale_grad(NV, codes[perm], off2, Xb[rows], dYb[rows], mask=mask[perm])
    assert np.array_equal(Y2, Y[rows]) and np.array_equal(dX2, dX[rows]) and np.array_equal(g2, g[perm])
    # the expert's own ws2 scales its rows: doubling ws2[2] doubles exactly those rows
    ws2b = list(ws2)
    ws2b[2] *= 2
    Yb = oracle_mod.grouped_fwd(NV, codes, scales, ws2b, off, Xb)
    a, b = off[2], off[3]
    assert np.array_equal(Yb[a:b], 2 * Y[a:b])
    assert np.array_equal(np.delete(Yb, np.arange(a, b), 0), np.delete(Y, np.arange(a, b), 0))


def test_no_tokens_at_all(oracle_mod):
    rng = np.random.default_rng(64)
    nib, codes, scales, ws2 = _experts(rng, MX, 3, 8, 64)
    off = _offsets([0, 0, 0])
    Xb = np.zeros((0, 64), dtype=np.uint16)
    dYb = np.zeros((0, 8), dtype=np.uint16)
    assert oracle_mod.grouped_fwd(MX, codes, scales, ws2, off, Xb).shape == (0, 8)
    g = oracle_mod.grouped_scale_grad(MX, codes, off, Xb, dYb)
    assert g.shape == (3, 8, 2) and not g.any()


def test_grouped_projection_uses_each_experts_tensor_scale(oracle_mod):
    """Inside the E4M3 range the projected byte of plane e is torch's RNE float8
    cast of fl32(L / ws2[e]); latents placed on the grid of one expert's ws2 land
    on different bytes under another's, so a plane projected with the wrong
    expert's scale fails. The merge then rewrites exactly the bytes that differ."""
    rng = np.random.default_rng(65)
    E, N, G = 3, 16, 8
    ws2 = [2.0 ** -7, 3.0 * 2.0 ** -9, 2.0 ** -5]
    L = np.empty((E, N, G), dtype=np.float32)
    for e in range(E):
        L[e] = (rng.uniform(0.02, 400.0, size=(N, G)) * ws2[e]).astype(np.float32)
    b, m, nf = oracle_mod.grouped_project(NV, L, ws2)
    for e in range(E):
        q = (L[e] / np.float32(ws2[e])).astype(np.float32)
        ref = torch.from_numpy(q).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
        assert np.array_equal(b[e], ref) and (m[e] == 1).all()
    assert nf == 0
    assert not np.array_equal(oracle_mod.grouped_project(NV, L, ws2[::-1])[0], b)
    old = rng.integers(0x30, 0x70, size=(E, N, G), dtype=np.uint8)
    new, delta, ch = oracle_mod.grouped_merge(NV, L, old, ws2)
    assert np.array_equal(new, b) and ch == int((old != b).sum())


def test_grouped_adapter_uses_each_experts_factors_and_scale(oracle_mod):
    """An expert with B = 0 keeps its base plane byte for byte while the others move;
    relabelling the experts (base plane, factors, ws2 together) relabels every
    output; the gradients of expert e depend only on expert e's g, B and A."""
    rng = np.random.default_rng(66)
    E, N, G, r, aor = 4, 16, 24, 5, 0.5
    base = rng.integers(0x30, 0x68, size=(E, N, G), dtype=np.uint8)
    ws2 = [2.0 ** -7, 2.0 ** -6, 3.0 * 2.0 ** -9, 2.0 ** -8]
    Bf = rng.normal(0, 1, (E, N, r)) * 0.05 * np.array(ws2)[:, None, None] * 40
    Bf[2] = 0.0
    Bb = torch.from_numpy(Bf.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    Ab = torch.from_numpy(rng.normal(0, 1, (E, r, G)).astype(np.float32)).to(torch.bfloat16).view(
        torch.int16).numpy().view(np.uint16)
    b, m, nf, L = oracle_mod.grouped_project_lowrank(NV, base, Bb, Ab, ws2, aor)
    assert np.array_equal(b[2], base[2]) and nf == 0
    for e in (0, 1, 3):
        assert (b[e] != base[e]).mean() > 0.05
    perm = [3, 1, 0, 2]
    b2, m2, _, L2 = oracle_mod.grouped_project_lowrank(NV, base[perm], Bb[perm], Ab[perm], [ws2[p] for p in perm], aor)
    assert np.array_equal(b2, b[perm]) and np.array_equal(m2, m[perm])
    assert np.array_equal(L2.view(np.uint32), L[perm].view(np.uint32))
    gm = rng.normal(0, 1, (E, N, G)).astype(np.float32)
    dB, dA = oracle_mod.grouped_lowrank_grad(gm, Bb, Ab, aor)
    gm2 = gm.copy()
    gm2[1] *= 2.0                                                       # exact in fp32
    dB2, dA2 = oracle_mod.grouped_lowrank_grad(gm2, Bb, Ab, aor)
    assert np.array_equal(np.delete(dB2, 1, 0), np.delete(dB, 1, 0)) and np.array_equal(dB2[1], 2 * dB[1])
    assert np.array_equal(np.delete(dA2, 1, 0), np.delete(dA, 1, 0)) and np.array_equal(dA2[1], 2 * dA[1])
