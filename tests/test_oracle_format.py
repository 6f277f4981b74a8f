"""Pins of the oracle's format decode against the paper's printed values and
torch's float8 library casts (Sec. 2, Appendix worked example)."""
import itertools
import math

import numpy as np
import torch

from conftest import read_golden


def test_e2m1_alphabet_matches_printed_set(oracle_mod):
    printed = read_golden("e2m1_alphabet.txt")["_rows"][0]
    vals = [oracle_mod.e2m1(v) for v in range(16)]
    # nibbles 0..7 are the non-negative codes in increasing order, 8..15 their negatives
    assert vals[:8] == printed
    assert [-v for v in vals[8:]] == printed
    assert math.copysign(1.0, vals[8]) == -1.0          # nibble 0x8 is -0


def test_e4m3_decode_matches_torch_cast(oracle_mod):
    ref = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    mine = np.array([oracle_mod.e4m3(b) for b in range(256)])
    nan = np.isnan(ref)
    assert (np.isnan(mine) == nan).all()
    assert (mine[~nan] == ref[~nan]).all()
    assert nan.sum() == 2 and nan[0x7F] and nan[0xFF]


def test_e4m3_facts(oracle_mod):
    facts = read_golden("format_facts.txt")
    vals = np.array([oracle_mod.e4m3(b) for b in range(256)])
    finite = vals[~np.isnan(vals)]
    assert finite.max() == facts["e4m3_max"][0]
    assert ((finite > 0)).sum() == int(facts["e4m3_positive_finite_count"][0])


def test_e8m0_decode_matches_torch_cast(oracle_mod):
    ref = torch.arange(256, dtype=torch.uint8).view(torch.float8_e8m0fnu).to(torch.float64).numpy()
    mine = np.array([oracle_mod.e8m0(b) for b in range(256)])
    assert np.isnan(mine[255]) and np.isnan(ref[255])
    assert (mine[:255] == ref[:255]).all()
    # no mantissa: every finite value is a power of two
    assert all(math.frexp(v)[0] == 0.5 for v in mine[:255])


def test_two_element_counterexample(oracle_mod):
    """Appendix worked example: decode of codes (6, 1.5) at scale 0.5 is (3, 0.75),
    the SSE values print to 5 decimals, and an exhaustive search over power-of-two
    scales (all E8M0 bytes) and all E2M1 code pairs finds Q' as the optimum other
    than the base itself."""
    gold = read_golden("two_element_example.txt")
    W = np.array(gold["W"])
    T = W + np.array(gold["delta"])
    assert round(float(((T - W) ** 2).sum()), 5) == gold["sse_base"][0]
    code_val = {oracle_mod.e2m1(v): v for v in range(8)}
    c6, c15 = code_val[gold["competitor_codes"][0]], code_val[gold["competitor_codes"][1]]
    half_e8m0 = 126
    half_e4m3 = 0x30
    assert oracle_mod.e8m0(half_e8m0) == gold["competitor_scale"][0]
    assert oracle_mod.e4m3(half_e4m3) == gold["competitor_scale"][0]
    for s in (oracle_mod.e8m0(half_e8m0), oracle_mod.e4m3(half_e4m3)):
        Q = np.array([oracle_mod.e2m1(c6) * s, oracle_mod.e2m1(c15) * s])
        assert list(Q) == gold["competitor_values"]
        assert round(float(((T - Q) ** 2).sum()), 5) == gold["sse_competitor"][0]
    best = None
    for byte in range(255):
        s = oracle_mod.e8m0(byte)
        for a, b in itertools.product(range(16), range(16)):
            Q = np.array([oracle_mod.e2m1(a) * s, oracle_mod.e2m1(b) * s])
            if (Q == W).all():
                continue
            sse = float(((T - Q) ** 2).sum())
            if best is None or sse < best[0]:
                best = (sse, tuple(Q))
    assert best[1] == tuple(gold["competitor_values"])
    assert round(best[0], 5) == gold["sse_competitor"][0]


def test_nibble_layout_and_block_mapping(oracle_mod):
    """decode_weight = printed alphabet[nibble] * scale[n, k // B], nibble of k
    taken from byte k/2, low nibble for even k; scale bytes decoded by torch."""
    printed = read_golden("e2m1_alphabet.txt")["_rows"][0]
    table = np.array(printed + [-v for v in printed])
    rng = np.random.default_rng(5)
    for fmt, B in ((0, 16), (1, 32)):
        N, K = 7, 96
        nib = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
        codes = (nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8)
        if fmt == 0:
            scales = rng.integers(0, 0x7F, size=(N, K // B), dtype=np.uint8)
            ws2 = 0.37
            s = torch.from_numpy(scales).view(torch.float8_e4m3fn).to(torch.float64).numpy() * np.float64(np.float32(ws2))
        else:
            scales = rng.integers(100, 150, size=(N, K // B), dtype=np.uint8)
            ws2 = 1.0
            s = torch.from_numpy(scales).view(torch.float8_e8m0fnu).to(torch.float64).numpy()
        expect = table[nib] * np.repeat(s, B, axis=1)
        got = oracle_mod.decode_weight(fmt, codes, scales, ws2, N, K)
        assert np.array_equal(got, expect)


def test_bf16_decode_matches_torch(oracle_mod):
    x = torch.randn(1000, generator=torch.Generator().manual_seed(3)).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    lib = oracle_mod.lib()
    lib.or_bf16.restype = __import__("ctypes").c_double
    lib.or_bf16.argtypes = [__import__("ctypes").c_uint16]
    got = np.array([lib.or_bf16(int(b)) for b in bits])
    assert np.array_equal(got, x.to(torch.float64).numpy())
