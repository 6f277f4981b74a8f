"""GPU parity of the grouped expert contractions (Sec. 3 "MoE: a batched
grouped-expert kernel") against the oracle, through the C ABI.

Small ragged cases (empty experts, experts of 1 row, experts whose rows straddle
the 512-row tiles, ragged N and K) are compared element by element with the
oracle's grouped definitions; every expert's slice is also bit-identical to the
dense entry point called on that expert alone (the same kernels, the same
arithmetic order). The full-size Qwen3-30B-A3B- and gpt-oss-120B-shaped expert
linears are checked on oracle samples of several experts and bit for bit against
the per-expert dense calls over every output."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_close, f64, hbits, host

pytestmark = pytest.mark.gpu

NV, MX = 0, 1


@pytest.fixture(scope="module")
def h():
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    return pkg.Handle()


def _setup(wl, lin):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    ex = synth.gen_experts(wl, lin, device="cuda")
    off = synth.offsets_of(synth.gen_routing(wl))
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, ex.codes, ex.scales, ex.ws2)
    X = synth.gen_act(wl, lin.x, M=off[-1], device="cuda").contiguous()
    dY = synth.gen_dy(wl, lin, M=off[-1], device="cuda").contiguous()
    return gw, off, X, dY


def _dense_per_expert(h, gw, off, X, dY, mask=None):
    """Y, dX, g from the dense entry points, one call per expert with tokens. An
    expert with enough tokens (>= 4096 here) has its dense scale gradient cut into
    token parts, whose fp32 sums round differently from the grouped launch's
    single pass: _split_experts lists them."""
    Y = torch.zeros(off[-1], gw.N, dtype=torch.bfloat16, device="cuda")
    dX = torch.zeros(off[-1], gw.K, dtype=torch.bfloat16, device="cuda")
    g = torch.zeros(gw.E, gw.N, gw.K // (16 if gw.fmt == NV else 32), dtype=torch.float32, device="cuda")
    for e in range(gw.E):
        a, b = off[e], off[e + 1]
        if b == a:
            continue
        w = gw.expert(e)
        w.scales = w.scales.clone()   # the dense entry points take 16-byte aligned planes
        h.sq_fwd(w, X[a:b], Y=Y[a:b])
        h.sq_bwd_dx(w, dY[a:b], dX=dX[a:b])
        h.sq_scale_grad(w, X[a:b], dY[a:b], mask=None if mask is None else mask[e], g=g[e])
    return Y, dX, g


def _split_experts(h, gw, off):
    return [e for e in range(gw.E) if off[e + 1] > off[e] and h.sq_scale_grad_workspace(gw.expert(e), off[e + 1] - off[e])[0] > 1]


SMALL = [
    # key, fmt, per-expert token counts, N, K
    ("g_nv", NV, [300, 0, 517, 64], 136, 608),
    ("g_mx", MX, [1, 700, 33], 264, 320),
    ("g_nv_one", NV, [1029], 392, 256),
    ("g_mx_many", MX, [0, 0, 0, 5, 130, 0, 512, 513, 1, 0], 40, 96),
    ("g_nv_tail_empty", NV, [77, 0, 0], 8, 32),
    ("g_nv_long_k", NV, [3, 260], 264, 2080),
    # 256-row tile halves: exactly one half, one row past it, one short of it, a half past a tile
    ("g_nv_half_edges", NV, [256, 257, 255, 768, 769], 264, 512),
]


@pytest.mark.parametrize("key,fmt,counts,N,K", SMALL, ids=[s[0] for s in SMALL])
def test_grouped_parity_small(h, key, fmt, counts, N, K):
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe(key, fmt, counts, N, K, seed=sum(counts) + N + K, kind="outlier" if fmt else "gauss")
    gw, off, X, dY = _setup(wl, wl.linears[0])
    G = K // (16 if fmt == NV else 32)
    rng = np.random.default_rng(N * 3 + K)
    mask = torch.from_numpy(rng.integers(0, 2, size=(gw.E, N, G), dtype=np.uint8)).cuda()
    g0 = torch.full((gw.E, N, G), 7.0, device="cuda")                 # stale values must be overwritten
    Y = h.sq_grouped_fwd(gw, off, X)
    dX = h.sq_grouped_bwd_dx(gw, off, dY)
    g = h.sq_grouped_scale_grad(gw, off, X, dY, g=g0)
    gm = h.sq_grouped_scale_grad(gw, off, X, dY, mask=mask)
    h.sq_sync()
    codes, scales = host(gw.codes), host(gw.scales)
    Y_ref = oracle.grouped_fwd(fmt, codes, scales, gw.ws2, off, hbits(X))
    dX_ref = oracle.grouped_dx(fmt, codes, scales, gw.ws2, off, hbits(dY))
    g_ref = oracle.grouped_scale_grad(fmt, codes, off, hbits(X), hbits(dY))
    assert_close(f64(Y), Y_ref, what="Y")
    assert_close(f64(dX), dX_ref, what="dX")
    assert_close(f64(g), g_ref, what="g")
    assert_close(f64(gm), g_ref * host(mask), rms=float(np.sqrt(np.mean(g_ref ** 2))), what="g*mask")
    for e in range(gw.E):
        if off[e + 1] == off[e]:
            assert not host(g[e]).any(), f"expert {e} has no tokens but a nonzero gradient"
    Yd, dXd, gd = _dense_per_expert(h, gw, off, X, dY)
    _, _, gmd = _dense_per_expert(h, gw, off, X, dY, mask=mask)
    h.sq_sync()
    assert torch.equal(Y, Yd) and torch.equal(dX, dXd), "grouped and per-expert dense outputs differ"
    assert not _split_experts(h, gw, off)              # every dense call is a single pass over its tokens
    assert torch.equal(g, gd) and torch.equal(gm, gmd), "grouped and per-expert dense gradients differ"


def _sampled(h, wl, lin, n_experts=4, n_samples=2048, n_rows=16):
    gw, off, X, dY = _setup(wl, lin)
    codes0 = gw.codes.clone()
    Y = h.sq_grouped_fwd(gw, off, X)
    dX = h.sq_grouped_bwd_dx(gw, off, dY)
    g = h.sq_grouped_scale_grad(gw, off, X, dY)
    h.sq_sync()
    counts = np.diff(np.asarray(off))
    rng = np.random.default_rng(wl.seed)
    nz = np.flatnonzero(counts)
    chosen = {int(nz[np.argmax(counts[nz])]), int(nz[np.argmin(counts[nz])]), int(nz[-1])}
    chosen |= set(int(e) for e in rng.choice(nz, n_experts, replace=False))
    Xb, dYb = hbits(X), hbits(dY)
    for e in sorted(chosen):
        a, b = off[e], off[e + 1]
        w = gw.expert(e)
        c, s = host(w.codes), host(w.scales)
        ms = rng.integers(0, b - a, n_samples)
        ns = rng.integers(0, gw.N, n_samples)
        ks = rng.integers(0, gw.K, n_samples)
        ms[:4] = [0, b - a - 1, 0, b - a - 1]
        ns[:4] = [0, 0, gw.N - 1, gw.N - 1]
        ks[:4] = [0, 0, gw.K - 1, gw.K - 1]
        Y_ref = oracle.fwd_at(gw.fmt, c, s, w.ws2, Xb[a:b], ms, ns)
        dX_ref = oracle.dx_at(gw.fmt, c, s, w.ws2, dYb[a:b], ms, ks)
        assert_close(f64(Y[a:b])[ms, ns], Y_ref, what=f"{wl.key}/{lin.name} expert {e} Y samples")
        assert_close(f64(dX[a:b])[ms, ks], dX_ref, what=f"{wl.key}/{lin.name} expert {e} dX samples")
        rows = np.unique(np.concatenate([[0, gw.N - 1], rng.integers(0, gw.N, n_rows)]))
        g_ref = oracle.scale_grad(gw.fmt, c, Xb[a:b], dYb[a:b], rows=rows)
        assert_close(host(g[e])[rows], g_ref, what=f"{wl.key}/{lin.name} expert {e} g rows")
    Yd, dXd, gd = _dense_per_expert(h, gw, off, X, dY)
    h.sq_sync()
    assert torch.equal(Y, Yd) and torch.equal(dX, dXd)
    split = _split_experts(h, gw, off)
    same = [e for e in range(gw.E) if e not in split]
    assert torch.equal(g[same], gd[same])               # one pass over the tokens on both sides: same bits
    if split:                                           # token parts: the same sums up to fp32 rounding
        assert_close(f64(gd[split]), f64(g[split]), what=f"{wl.key}/{lin.name} split experts' g")
    assert torch.equal(gw.codes, codes0)


@pytest.mark.parametrize("key,name", [("moe_qwen", "gate_proj"), ("moe_qwen", "down_proj"), ("moe_gptoss", "up_proj")])
def test_grouped_full_size_sampled(h, key, name):
    from paper_2609_04526_gb300 import synth
    wl = synth.MOE_WORKLOADS[key]
    _sampled(h, wl, next(l for l in wl.linears if l.name == name))
    torch.cuda.empty_cache()


def test_table_ring_reuse_with_calls_in_flight(h):
    """More grouped calls than the handle has expert tables, each with its own
    routing and output, enqueued without a sync: every result matches its own
    per-expert dense calls."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe("ring", NV, [1] * 6, 264, 512, seed=5)
    lin = wl.linears[0]
    ex = synth.gen_experts(wl, lin, device="cuda")
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, ex.codes, ex.scales, ex.ws2)
    rng = np.random.default_rng(9)
    X = synth.gen_act(wl, "x", M=6000, device="cuda")
    outs = []
    for i in range(9):
        counts = rng.integers(0, 1000, size=6)
        counts[i % 6] = 0
        off = synth.offsets_of(counts)
        outs.append((off, h.sq_grouped_fwd(gw, off, X[:off[-1]])))
    h.sq_sync()
    for off, Y in outs:
        Yd, _, _ = _dense_per_expert(h, gw, off, X[:off[-1]], torch.zeros(off[-1], gw.N, dtype=torch.bfloat16,
                                                                           device="cuda"))
        h.sq_sync()
        assert torch.equal(Y, Yd)


def test_grouped_empty_batches(h):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe("empty", MX, [0, 0], 16, 64, seed=3)
    ex = synth.gen_experts(wl, wl.linears[0], device="cuda")
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, ex.codes, ex.scales, ex.ws2)
    X = torch.zeros(0, 64, dtype=torch.bfloat16, device="cuda")
    dY = torch.zeros(0, 16, dtype=torch.bfloat16, device="cuda")
    Y = h.sq_grouped_fwd(gw, [0, 0, 0], X)
    g = h.sq_grouped_scale_grad(gw, [0, 0, 0], X, dY, g=torch.full((2, 16, 2), 5.0, device="cuda"))
    h.sq_sync()
    assert Y.shape == (0, 16) and (g == 0).all()


def test_grouped_invalid_args_and_capture(h):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe("bad", NV, [4, 4], 16, 64, seed=4)
    ex = synth.gen_experts(wl, wl.linears[0], device="cuda")
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, ex.codes, ex.scales, ex.ws2)
    X = synth.gen_act(wl, "x", M=8, device="cuda")
    Xbig = torch.zeros(9, 64, dtype=torch.bfloat16, device="cuda")

    def with_(**kw):
        d = dict(fmt=gw.fmt, E=gw.E, N=gw.N, K=gw.K, codes=gw.codes, scales=gw.scales, ws2=gw.ws2)
        d.update(kw)
        return pkg.GroupedWeight(**d)

    bad = [
        lambda: h.sq_grouped_fwd(gw, [1, 4, 8], X),                            # offsets[0] != 0
        lambda: h.sq_grouped_fwd(gw, [0, 5, 4], X),                            # decreasing
        lambda: h.sq_grouped_fwd(with_(ws2=[1.0, float("nan")]), [0, 4, 8], X),
        lambda: h.sq_grouped_fwd(with_(fmt=MX, ws2=[1.0, 0.5]), [0, 4, 8], X),  # MXFP4 ws2 != 1
        lambda: h.sq_grouped_fwd(with_(N=12), [0, 4, 8], X),                    # N % 8
        lambda: h.sq_grouped_fwd(with_(E=40000, ws2=[1.0] * 40000, N=65536),
                                 [0] * 40000 + [8], X),                         # E * N >= 2^31
        lambda: h.sq_grouped_fwd(gw, [0, 4, 8], Xbig.view(-1)[1:1 + 8 * 64].view(8, 64)),  # misaligned X
    ]
    for call in bad:
        with pytest.raises(pkg.SQError) as ei:
            call()
        assert ei.value.status == -1, ei.value
    with pytest.raises(ValueError):
        h.sq_grouped_fwd(gw, [0, 8], X)                                        # E + 1 offsets needed
    Y = h.sq_grouped_fwd(gw, [0, 4, 8], X)                                     # the handle still works
    s = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with pytest.raises(pkg.SQError) as ei:
        with torch.cuda.graph(graph, stream=s):
            h.sq_grouped_fwd(gw, [0, 4, 8], X, Y=Y, stream=s)
    assert ei.value.status == -2
    h.sq_sync()


@pytest.mark.parametrize("key,fmt,E,N,K", [("p_nv", NV, 5, 40, 96 * 2), ("p_mx", MX, 3, 24, 96),
                                           ("p_nv_qwen_gate", NV, 128, 768, 2048)])
def test_grouped_projection_and_merge_bit_exact(h, key, fmt, E, N, K):
    """Every expert's plane projected / merged with its own ws2 in one launch: bytes,
    masks, deltas and counters bit-exact against the oracle (NaN and above-ceiling
    latents included)."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe(key, fmt, [1] * E, N, K, seed=E + N)
    lin = wl.linears[0]
    ex = synth.gen_experts(wl, lin, device="cuda")
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, None, None, ex.ws2)
    L = synth.gen_expert_latents(wl, lin, ex, device="cuda")
    L[0, 0, 0] = float("nan")
    L[E - 1, N - 1, 1] = float("inf")
    nf = torch.zeros(1, dtype=torch.int32, device="cuda")
    b, m = h.sq_grouped_project_scales(gw, L, nonfinite=nf)
    art = ex.scales.clone()
    delta = torch.empty_like(L)
    ch = torch.zeros(1, dtype=torch.int64, device="cuda")
    h.sq_grouped_merge(gw, L, art, ongrid_delta=delta, changed=ch)
    h.sq_sync()
    Lh = host(L)
    rb, rm, rnf = oracle.grouped_project(fmt, Lh, ex.ws2)
    assert np.array_equal(host(b), rb) and np.array_equal(host(m), rm) and int(nf.item()) == rnf
    rnew, rdelta, rch = oracle.grouped_merge(fmt, Lh, host(ex.scales), ex.ws2)
    assert np.array_equal(host(art), rnew) and int(ch.item()) == rch
    dh = host(delta)
    assert np.array_equal(np.isnan(dh), np.isnan(rdelta))
    ok = ~np.isnan(rdelta)
    assert np.array_equal(dh[ok].view(np.uint32), rdelta[ok].view(np.uint32))
    assert (rb != host(ex.scales)).mean() > 0.005                      # the latents moved bytes


@pytest.mark.parametrize("key,fmt,E,N,K,r", [("a_nv", NV, 5, 40, 192, 13), ("a_mx", MX, 3, 24, 96 * 4, 7),
                                             ("a_qwen_gate", NV, 128, 768, 2048, 54)])
def test_grouped_adapter_projection_bit_exact_and_gradients(h, key, fmt, E, N, K, r):
    """Every expert's adapter latent, byte, mask and NaN count bit-exact against the
    oracle in one launch; the adapter gradients of all experts within the bar and
    the same on a second run."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom_moe(key, fmt, [1] * E, N, K, seed=E * 7 + r)
    lin = wl.linears[0]
    ex = synth.gen_experts(wl, lin, device="cuda")
    gw = pkg.GroupedWeight(ex.fmt, ex.E, ex.N, ex.K, None, ex.scales, ex.ws2)
    B, A, aor = synth.gen_expert_adapters(wl, lin, ex, r=r, device="cuda")
    B_clean = B.clone()
    if fmt == NV:
        B[1, 0, 0] = float("nan")                                      # one NaN latent row in expert 1
    G = K // (16 if fmt == NV else 32)
    mask = torch.empty(E, N, G, dtype=torch.uint8, device="cuda")
    latent = torch.empty(E, N, G, dtype=torch.float32, device="cuda")
    nf = torch.zeros(1, dtype=torch.int32, device="cuda")
    b, _, _ = h.sq_grouped_project_lowrank(gw, B, A, aor, mask_out=mask, nonfinite=nf, latent_out=latent)
    gen = torch.Generator(device="cuda").manual_seed(E + N)
    g = torch.randn(E, N, G, device="cuda", generator=gen) * mask.float()
    B = B_clean                                                         # finite factors for the gradients
    dB, dA = h.sq_grouped_lowrank_grad(g, B, A, aor)
    dB2, dA2 = h.sq_grouped_lowrank_grad(g, B, A, aor)
    h.sq_sync()
    Bn = B_clean.clone()
    if fmt == NV:
        Bn[1, 0, 0] = float("nan")
    rb, rm, rnf, rL = oracle.grouped_project_lowrank(fmt, host(ex.scales), hbits(Bn), hbits(A), ex.ws2, aor)
    gL = host(latent)
    nan = np.isnan(rL)
    assert np.array_equal(np.isnan(gL), nan)
    assert np.array_equal(gL[~nan].view(np.uint32), rL[~nan].view(np.uint32)), "latent differs from the oracle"
    assert np.array_equal(host(b), rb) and np.array_equal(host(mask), rm) and int(nf.item()) == rnf
    if fmt == NV:  # a 2% relative move crosses E4M3 grid midpoints, never the E8M0 ones (factor sqrt 2)
        assert (rb != host(ex.scales)).mean() > 0.005
    gh = host(g)
    rdB, rdA = oracle.grouped_lowrank_grad(gh, hbits(B), hbits(A), aor)
    assert_close(host(dB), rdB, what="dB")
    assert_close(host(dA), rdA, what="dA")
    assert torch.equal(dB, dB2) and torch.equal(dA, dA2), "adapter gradients are not reproducible"
