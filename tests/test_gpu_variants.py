"""GPU parity of the scale-family variants (ablation appendix) against the oracle,
through the C ABI: the least-squares code-preserving fit, the granularity-ladder
group gradient and group-delta projection, and one linear's ladder step."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_close, f64, hbits, host, setup_linear

pytestmark = pytest.mark.gpu

NV, MX = 0, 1
BLOCK = {NV: 16, MX: 32}


@pytest.fixture(scope="module")
def h():
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    return pkg.Handle()


def _weight(key, fmt, N, K, seed):
    from paper_2609_04526_gb300 import synth
    wl = synth.custom(key, fmt, 8, N, K, seed=seed)
    return synth.gen_weight(wl, wl.linears[0], device="cuda")


@pytest.mark.parametrize("fmt,N,K", [(NV, 40, 608), (MX, 33 * 8, 320), (NV, 1, 32)])
def test_fit_matches_oracle(h, fmt, N, K):
    w = _weight(f"fit{fmt}", fmt, N, K, seed=N + K)
    codes = w.codes.clone()
    codes[0, :BLOCK[fmt] // 2] = 0                                         # a block of zero codes
    gen = torch.Generator(device="cuda").manual_seed(N)
    dW = (torch.randn(N, K, device="cuda", generator=gen) * 1e-3).to(torch.bfloat16)
    delta, cap, tot, lat = h.sq_fit_scale_delta(fmt, codes, dW, w.ws2, scales=w.scales, want_energy=True)
    h.sq_sync()
    rd, rc, rt, rl = oracle.fit_scale_delta(fmt, host(codes), host(w.scales), w.ws2, hbits(dW))
    assert host(delta)[0, 0] == 0.0 and host(cap)[0, 0] == 0.0
    assert_close(host(delta), rd, what="delta")
    assert_close(host(cap), rc, what="captured")
    assert_close(host(tot), rt, what="total")
    assert_close(host(lat), rl, what="latent")


def test_fit_recovers_a_scale_change_bit_exactly(h):
    """dW = c * t per block with dyadic t: every fp32 step is exact, delta == t."""
    from paper_2609_04526_gb300 import synth
    N, K = 64, 512
    w = _weight("fit_exact", NV, N, K, seed=3)
    nib = torch.stack((w.codes & 0xF, w.codes >> 4), dim=-1).reshape(N, K).long()
    table = torch.tensor(synth._E2M1_MAG, dtype=torch.float32, device="cuda")
    c = table[nib & 7] * torch.where(nib >= 8, -1.0, 1.0)
    gen = torch.Generator(device="cuda").manual_seed(4)
    t = torch.tensor([0.25, -0.5, 1.0, 2.0, -0.125], device="cuda")[torch.randint(0, 5, (N, K // 16), device="cuda",
                                                                                   generator=gen)]
    dW = (c * t.repeat_interleave(16, dim=1)).to(torch.bfloat16)
    delta, _, _, _ = h.sq_fit_scale_delta(NV, w.codes, dW)
    h.sq_sync()
    cc = (c * c).reshape(N, K // 16, 16).sum(-1)
    nz = cc > 0
    assert torch.equal(delta[nz], t[nz]) and (delta[~nz] == 0).all()


def test_fit_energy_is_one_over_block_full_size(h):
    """The Llama-3-8B gate_proj plane (14336 x 4096) and a Gaussian update: the GPU's
    captured / total energy is 1/16 within its sampling error, and every block matches
    the oracle."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c3"]
    w = synth.gen_weight(wl, wl.linears[0], device="cuda")
    gen = torch.Generator(device="cuda").manual_seed(11)
    dW = (torch.randn(w.N, w.K, device="cuda", generator=gen) * 2e-4).to(torch.bfloat16)
    delta, cap, tot, _ = h.sq_fit_scale_delta(NV, w.codes, dW, want_energy=True)
    h.sq_sync()
    ratio = float(cap.double().sum() / tot.double().sum())
    assert abs(ratio * 16 - 1) < 0.01, ratio                              # 3.7M blocks: sigma ~ 0.07%
    rows = slice(0, 512)
    rd, rc, rt, _ = oracle.fit_scale_delta(NV, host(w.codes)[rows], None, 1.0, hbits(dW)[rows])
    assert_close(host(delta)[rows], rd, what="delta")
    assert_close(host(cap)[rows], rc, what="captured")


@pytest.mark.parametrize("N,G,gd", [(40, 48, 1), (40, 48, 4), (40, 48, 48), (300, 256, 16), (1, 2, 2)])
def test_group_reduce_matches_oracle(h, N, G, gd):
    gen = torch.Generator(device="cuda").manual_seed(N * G + gd)
    g = torch.randn(N, G, device="cuda", generator=gen)
    out = h.sq_group_reduce(g, gd)
    h.sq_sync()
    assert_close(host(out), oracle.group_reduce(host(g), gd), what="group gradient")
    if gd == G:
        assert torch.equal(out, g)


@pytest.mark.parametrize("fmt,N,G,gd,ws2", [(NV, 64, 96, 4, 2.0 ** -6), (NV, 37, 32, 1, 1.0 / (6 * 448)),
                                            (MX, 50, 40, 8, 1.0)])
def test_group_delta_projection_bit_exact(h, fmt, N, G, gd, ws2):
    rng = np.random.default_rng(N + G)
    base = (rng.integers(0x28, 0x70, size=(N, G)) if fmt == NV else rng.integers(110, 140, size=(N, G))).astype(np.uint8)
    scale = ws2 * 64 if fmt == NV else 2.0 ** -2
    delta = (rng.normal(0, 1, (N, gd)) * scale).astype(np.float32)
    delta[0, 0] = np.nan
    bd, dd = torch.from_numpy(base).cuda(), torch.from_numpy(delta).cuda()
    mask = torch.empty(N, G, dtype=torch.uint8, device="cuda")
    lat = torch.empty(N, G, dtype=torch.float32, device="cuda")
    nf = torch.zeros(1, dtype=torch.int32, device="cuda")
    b, _, _ = h.sq_project_group_delta(fmt, bd, dd, ws2, mask_out=mask, nonfinite=nf, latent_out=lat)
    h.sq_sync()
    rb, rm, rnf, rl = oracle.project_group_delta(fmt, base, delta, ws2)
    assert np.array_equal(host(b), rb) and np.array_equal(host(mask), rm) and int(nf.item()) == rnf > 0
    gl = host(lat)
    nan = np.isnan(rl)
    assert np.array_equal(np.isnan(gl), nan) and np.array_equal(gl[~nan].view(np.uint32), rl[~nan].view(np.uint32))


def test_granularity_ladder_step_one_linear(h):
    """gd = 4 groups per row: group delta -> projection (bytes + mask) -> forward with the
    projected bytes -> masked scale gradient -> group gradient, against the oracle chain."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("ladder", NV, 300, 264, 512, seed=21)
    lin = wl.linears[0]
    qw0, X, dY = setup_linear(wl, lin)
    N, G, gd = lin.N, lin.K // 16, 4
    gen = torch.Generator(device="cuda").manual_seed(22)
    delta = torch.randn(N, gd, device="cuda", generator=gen) * qw0.ws2 * 16
    mask = torch.empty(N, G, dtype=torch.uint8, device="cuda")
    qb, _, _ = h.sq_project_group_delta(NV, qw0.scales, delta, qw0.ws2, mask_out=mask)
    qw = pkg.QuantWeight(NV, N, lin.K, qw0.codes, qb, qw0.ws2)
    Y = h.sq_fwd(qw, X)
    g = h.sq_scale_grad(qw, X, dY, mask=mask)
    gg = h.sq_group_reduce(g, gd)
    h.sq_sync()
    rb, rm, _, _ = oracle.project_group_delta(NV, host(qw0.scales), host(delta), qw0.ws2)
    assert np.array_equal(host(qb), rb) and np.array_equal(host(mask), rm)
    assert (rb != host(qw0.scales)).mean() > 0.1
    W = oracle.decode_weight(NV, host(qw.codes), rb, qw0.ws2, N, lin.K)
    assert_close(f64(Y), oracle.fwd_f64(f64(X), W), what="Y")
    rg = oracle.scale_grad_f64(NV, host(qw.codes), f64(X), f64(dY), mask=rm)
    assert_close(host(gg), oracle.group_reduce(rg.astype(np.float32), gd), what="group gradient")


def test_variants_invalid_args(h):
    import paper_2609_04526_gb300 as pkg
    dev = "cuda"
    codes = torch.zeros(8, 16, dtype=torch.uint8, device=dev)
    dW = torch.zeros(8, 32, dtype=torch.bfloat16, device=dev)
    dWbig = torch.zeros(8 * 32 + 8, dtype=torch.bfloat16, device=dev)
    g = torch.zeros(8, 6, device=dev)
    base = torch.zeros(8, 6, dtype=torch.uint8, device=dev)
    bad = [
        lambda: h.sq_fit_scale_delta(NV, codes, torch.zeros(8, 40, dtype=torch.bfloat16, device=dev)),  # K % 32
        lambda: h.sq_fit_scale_delta(NV, codes, dW, float("nan")),                                     # ws2
        lambda: h.sq_fit_scale_delta(NV, codes, dWbig[1:1 + 8 * 32].view(8, 32)),                     # misaligned dW
        lambda: h.sq_group_reduce(g, 4),                                                                # 4 does not divide 6
        lambda: h.sq_group_reduce(g, 0),
        lambda: h.sq_project_group_delta(NV, base, torch.zeros(8, 4, device=dev), 1.0),                  # gd = 4
        lambda: h.sq_project_group_delta(MX, base, torch.zeros(8, 2, device=dev), 0.5),                  # MXFP4 ws2
    ]
    for i, call in enumerate(bad):
        with pytest.raises(pkg.SQError) as ei:
            call()
        assert ei.value.status == -1, i


def _control_inputs(M, N, K, seed, ds_scale=0.05):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    W = (torch.randn(N, K, device="cuda", generator=gen) * 0.02).to(torch.bfloat16)
    dS = torch.randn(N, K // 16, device="cuda", generator=gen) * ds_scale
    X = torch.randn(M, K, device="cuda", generator=gen).to(torch.bfloat16)
    dY = (torch.randn(M, N, device="cuda", generator=gen) * 1e-3).to(torch.bfloat16)
    return W, dS, X, dY


@pytest.mark.parametrize("M,N,K", [(300, 392, 608), (64, 256, 512), (1, 8, 32), (1030, 264, 2080)])
def test_control_parity_small(h, M, N, K):
    """The multiplicative control's forward, input gradient and coefficient gradient
    against the oracle (W' rounded as the oracle rounds it, contractions in float64)."""
    W, dS, X, dY = _control_inputs(M, N, K, seed=M + N + K)
    Y = h.sq_control_fwd(W, dS, X)
    dX = h.sq_control_bwd_dx(W, dS, dY)
    g = h.sq_control_grad(W, X, dY)
    h.sq_sync()
    Wp = oracle.control_weight(hbits(W), host(dS))
    assert_close(f64(Y), oracle.fwd_f64(f64(X), Wp), what="Y")
    assert_close(f64(dX), oracle.dx_f64(f64(dY), Wp), what="dX")
    assert_close(host(g), oracle.control_grad_f64(hbits(W), f64(X), f64(dY)), what="g")


def test_control_full_size_sampled(h):
    """8192 x 14336 x 4096 (the c3 shape): sampled Y and dX elements and whole rows of
    g against the oracle."""
    M, N, K = 8192, 14336, 4096
    W, dS, X, dY = _control_inputs(M, N, K, seed=9)
    Y = h.sq_control_fwd(W, dS, X)
    dX = h.sq_control_bwd_dx(W, dS, dY)
    g = h.sq_control_grad(W, X, dY)
    h.sq_sync()
    rng = np.random.default_rng(9)
    ns = np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, 24)]))
    ks = np.unique(np.concatenate([[0, K - 1], rng.integers(0, K, 24)]))
    ms = np.unique(np.concatenate([[0, M - 1], rng.integers(0, M, 48)]))
    Wp_rows = oracle.control_weight(hbits(W)[ns], host(dS)[ns])
    Xm = f64(X[torch.from_numpy(ms).cuda()])
    assert_close(f64(Y)[np.ix_(ms, ns)], Xm @ Wp_rows.T, what="Y samples")
    Wp_all = oracle.control_weight(hbits(W), host(dS))
    dYm = f64(dY[torch.from_numpy(ms).cuda()])
    assert_close(f64(dX)[np.ix_(ms, ks)], dYm @ Wp_all[:, ks], what="dX samples")
    rg = oracle.control_grad_f64(hbits(W)[ns], f64(X), f64(dY)[:, ns])
    assert_close(host(g)[ns], rg, what="g rows")


def test_control_adapter_chain(h):
    """The control's low-rank coefficients dS = (alpha/r) B A -> forward -> coefficient
    gradient -> adapter gradients, against the oracle chain; the product repeats."""
    M, N, K, r = 300, 264, 512, 16
    gen = torch.Generator(device="cuda").manual_seed(31)
    W, _, X, dY = _control_inputs(M, N, K, seed=31)
    B = (torch.randn(N, r, device="cuda", generator=gen) * 0.05).to(torch.bfloat16)
    A = (torch.randn(r, K // 16, device="cuda", generator=gen) * 0.05).to(torch.bfloat16)
    aor = 2.0
    dS = h.sq_lowrank_product(B, A, aor)
    dS2 = h.sq_lowrank_product(B, A, aor)
    Y = h.sq_control_fwd(W, dS, X)
    g = h.sq_control_grad(W, X, dY)
    dB, dA = h.sq_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    assert torch.equal(dS, dS2)
    assert_close(host(dS), oracle.lowrank_product(hbits(B), hbits(A), aor), what="dS")
    Wp = oracle.control_weight(hbits(W), host(dS))
    assert_close(f64(Y), oracle.fwd_f64(f64(X), Wp), what="Y")
    rg = oracle.control_grad_f64(hbits(W), f64(X), f64(dY))
    assert_close(host(g), rg, what="g")
    rdB, rdA = oracle.lowrank_grad(rg.astype(np.float32), hbits(B), hbits(A), aor)
    assert_close(host(dB), rdB, what="dB")
    assert_close(host(dA), rdA, what="dA")


def test_control_invalid_args(h):
    import paper_2609_04526_gb300 as pkg
    W = torch.zeros(8, 32, dtype=torch.bfloat16, device="cuda")
    dS = torch.zeros(8, 2, device="cuda")
    X = torch.zeros(4, 32, dtype=torch.bfloat16, device="cuda")
    bad = [
        lambda: h.sq_control_fwd(torch.zeros(12, 32, dtype=torch.bfloat16, device="cuda"), dS, X),     # N % 8
        lambda: h.sq_control_fwd(torch.zeros(8, 48, dtype=torch.bfloat16, device="cuda"), dS, X),      # K % 32
        lambda: h.sq_lowrank_product(torch.zeros(8, 300, dtype=torch.bfloat16, device="cuda"),
                                     torch.zeros(300, 2, dtype=torch.bfloat16, device="cuda"), 1.0),  # r > 256
    ]
    for call in bad:
        with pytest.raises(pkg.SQError) as ei:
            call()
        assert ei.value.status == -1
    Y = h.sq_control_fwd(W, dS, torch.zeros(0, 32, dtype=torch.bfloat16, device="cuda"))
    g = h.sq_control_grad(W, torch.zeros(0, 32, dtype=torch.bfloat16, device="cuda"),
                          torch.zeros(0, 8, dtype=torch.bfloat16, device="cuda"), g=torch.full((8, 2), 3.0, device="cuda"))
    h.sq_sync()
    assert Y.shape == (0, 8) and (g == 0).all()
