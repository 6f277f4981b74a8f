"""GPU parity of the low-rank scale adapter (Sec. 3 "Scale-QLoRA forward") against
the oracle, through the C ABI: the fused latent + projection is bit-exact (the
latent is formed in the same fp32 order on both sides), the adapter gradients are
within the floating-point bar, and one linear's whole training step (adapter ->
projection -> forward -> masked scale gradient -> adapter gradients) matches the
oracle's chain."""
import zlib

import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_close, f64, hbits, host, setup_linear

pytestmark = pytest.mark.gpu

NV, MX = 0, 1


@pytest.fixture(scope="module")
def h():
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    return pkg.Handle()


def _plane(key, fmt, N, G, r, seed):
    """A weight's scale plane [N, G] plus adapter factors for it (device tensors)."""
    from paper_2609_04526_gb300 import synth
    block = 16 if fmt == NV else 32
    wl = synth.custom(key, fmt, 8, N, G * block, seed=seed, kind="gauss")
    lin = wl.linears[0]
    w = synth.gen_weight(wl, lin, device="cuda")
    B, A, aor = synth.gen_adapter(wl, lin, w, r=r, device="cuda")
    return w, B, A, aor


def _check_projection(h, fmt, base, B, A, ws2, aor):
    N, G = base.shape
    mask = torch.empty(N, G, dtype=torch.uint8, device="cuda")
    latent = torch.empty(N, G, dtype=torch.float32, device="cuda")
    nf = torch.zeros(1, dtype=torch.int32, device="cuda")
    b, _, _ = h.sq_project_lowrank(fmt, base, B, A, ws2, aor, mask_out=mask, nonfinite=nf, latent_out=latent)
    h.sq_sync()
    rb, rm, rnf, rL = oracle.project_lowrank(fmt, host(base), hbits(B), hbits(A), ws2, aor)
    gL = host(latent)
    nan = np.isnan(rL)
    assert np.array_equal(np.isnan(gL), nan)
    assert np.array_equal(gL[~nan].view(np.uint32), rL[~nan].view(np.uint32)), "latent differs from the oracle"
    assert np.array_equal(host(b), rb), "projected bytes differ"
    assert np.array_equal(host(mask), rm), "mask differs"
    assert int(nf.item()) == rnf
    return rb, rm, rL


CASES = [
    # key, fmt, N, G, r
    ("lr_min", NV, 1, 16, 1),
    ("lr_nv", NV, 40, 48, 13),
    ("lr_nv58", NV, 136, 80, 58),
    ("lr_mx", MX, 300, 96, 64),
    ("lr_rmax", NV, 37, 16, 256),
    ("lr_mx_ragged", MX, 65, 144, 33),
    ("lr_nv_g6", NV, 24, 6, 5),        # G % 4 != 0: the per-block store path
    ("lr_mx_g71", MX, 72, 71, 9),
]


@pytest.mark.parametrize("key,fmt,N,G,r", CASES, ids=[c[0] for c in CASES])
def test_adapter_projection_bit_exact(h, key, fmt, N, G, r):
    w, B, A, aor = _plane(key, fmt, N, G, r, seed=zlib.crc32(key.encode()) % 1000)
    if fmt == NV and N >= 4:
        B[1] = torch.abs(B[1]) * 0 + 448.0 * w.ws2 / max(aor, 1e-3)   # pushes row 1 above the ceiling
        B[2, 0] = float("nan")                                          # a NaN latent row
    _check_projection(h, fmt, w.scales, B, A, w.ws2, aor)


@pytest.mark.parametrize("N,G,r", [(1, 16, 1), (40, 48, 13), (300, 96, 58), (1000, 32, 256), (129, 1040, 7),
                                   (256, 64, 128), (64, 32, 129)])
def test_adapter_gradients_match_oracle_and_repeat(h, N, G, r):
    gen = torch.Generator(device="cuda").manual_seed(N * 131 + G * 7 + r)
    g = torch.randn(N, G, device="cuda", generator=gen)
    g[torch.rand(N, G, device="cuda", generator=gen) < 0.3] = 0.0     # masked blocks
    B = (torch.randn(N, r, device="cuda", generator=gen) * 0.05).to(torch.bfloat16)
    A = (torch.randn(r, G, device="cuda", generator=gen) * 0.05).to(torch.bfloat16)
    aor = 16.0 / r
    dB, dA = h.sq_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    rdB, rdA = oracle.lowrank_grad(host(g), hbits(B), hbits(A), aor)
    assert_close(host(dB), rdB, what="dB")
    assert_close(host(dA), rdA, what="dA")
    dB2, dA2 = h.sq_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    assert torch.equal(dB, dB2) and torch.equal(dA, dA2), "adapter gradients are not reproducible"
    only_dA = h.sq_lowrank_grad(g, B, A, aor, want_dB=False)[1]
    h.sq_sync()
    assert torch.equal(only_dA, dA)


def test_adapter_training_step_one_linear(h):
    """Adapter latent -> projection (bytes + mask) -> forward with the projected
    bytes -> masked scale gradient -> adapter gradients, against the oracle chain."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("lr_step", NV, 300, 392, 608, seed=77, kind="gauss")
    lin = wl.linears[0]
    qw0, X, dY = setup_linear(wl, lin)
    B, A, aor = synth.gen_adapter(wl, lin, synth.gen_weight(wl, lin, device="cuda"), r=58, device="cuda")
    N, G = lin.N, lin.K // 16
    mask = torch.empty(N, G, dtype=torch.uint8, device="cuda")
    qb, _, _ = h.sq_project_lowrank(NV, qw0.scales, B, A, qw0.ws2, aor, mask_out=mask)
    qw = pkg.QuantWeight(NV, N, lin.K, qw0.codes, qb, qw0.ws2)
    Y = h.sq_fwd(qw, X)
    g = h.sq_scale_grad(qw, X, dY, mask=mask)
    dB, dA = h.sq_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    rb, rm, _, _ = oracle.project_lowrank(NV, host(qw0.scales), hbits(B), hbits(A), qw0.ws2, aor)
    assert np.array_equal(host(qb), rb) and np.array_equal(host(mask), rm)
    assert (rb != host(qw0.scales)).mean() > 0.01                      # the adapter moved bytes
    W = oracle.decode_weight(NV, host(qw.codes), rb, qw0.ws2, N, lin.K)
    assert_close(f64(Y), oracle.fwd_f64(f64(X), W), what="Y")
    rg = oracle.scale_grad_f64(NV, host(qw.codes), f64(X), f64(dY), mask=rm)
    assert_close(host(g), rg, what="g")
    rdB, rdA = oracle.lowrank_grad(rg.astype(np.float32), hbits(B), hbits(A), aor)
    assert_close(host(dB), rdB, what="dB")
    assert_close(host(dA), rdA, what="dA")


def test_adapter_full_size_gate_proj(h):
    """The Llama-3-8B gate_proj plane (14336 x 256 blocks, r = 58): every latent,
    byte and mask bit-exact; the adapter gradients of a full-size g within the bar."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c5"]
    lin = [l for l in wl.linears if l.name == "gate_proj"][0]
    w = synth.gen_weight(wl, lin, device="cuda")
    B, A, aor = synth.gen_adapter(wl, lin, w, device="cuda")
    _, rm, _ = _check_projection(h, wl.fmt, w.scales, B, A, w.ws2, aor)
    gen = torch.Generator(device="cuda").manual_seed(5)
    g = torch.randn(lin.N, lin.K // 16, device="cuda", generator=gen) * torch.from_numpy(rm).cuda().float()
    dB, dA = h.sq_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    rdB, rdA = oracle.lowrank_grad(host(g), hbits(B), hbits(A), aor)
    assert_close(host(dB), rdB, what="dB")
    assert_close(host(dA), rdA, what="dA")


def test_adapter_empty_and_invalid_args(h):
    import paper_2609_04526_gb300 as pkg
    dev = "cuda"
    base = torch.zeros(0, 16, dtype=torch.uint8, device=dev)
    B = torch.zeros(0, 4, dtype=torch.bfloat16, device=dev)
    A = torch.zeros(4, 16, dtype=torch.bfloat16, device=dev)
    nf = torch.full((1,), 7, dtype=torch.int32, device=dev)
    h.sq_project_lowrank(NV, base, B, A, 1.0, 0.5, nonfinite=nf)
    g = torch.zeros(0, 16, device=dev)
    dA = torch.full((4, 16), 3.0, device=dev)
    h.sq_lowrank_grad(g, B, A, 0.5, dA=dA, want_dB=False)
    h.sq_sync()
    assert int(nf.item()) == 0 and (dA == 0).all()                     # empty sum over n
    base = torch.zeros(8, 16, dtype=torch.uint8, device=dev)
    B = torch.zeros(8, 4, dtype=torch.bfloat16, device=dev)
    g = torch.zeros(8, 16, device=dev)
    bad = [
        lambda: h.sq_project_lowrank(NV, base, B[:, :0].contiguous(), A[:0].contiguous(), 1.0, 0.5),   # r = 0
        lambda: h.sq_project_lowrank(NV, base, torch.zeros(8, 257, dtype=torch.bfloat16, device=dev),
                                     torch.zeros(257, 16, dtype=torch.bfloat16, device=dev), 1.0, 0.5),  # r > 256
        lambda: h.sq_project_lowrank(NV, base, B, A, float("inf"), 0.5),                   # ws2
        lambda: h.sq_project_lowrank(NV, base, B, A, 1.0, float("nan")),                   # alpha/r
        lambda: h.sq_project_lowrank(MX, base, B, A, 2.0, 0.5),                            # MXFP4 ws2 != 1
        lambda: h.sq_lowrank_grad(g, B, A, 0.5, want_dB=False, want_dA=False),              # no output
        lambda: h.sq_lowrank_grad(g.view(-1)[1:113].view(7, 16), B[:7], A, 0.5),          # misaligned g
    ]
    for call in bad:
        with pytest.raises(pkg.SQError) as ei:
            call()
        assert ei.value.status == -1
