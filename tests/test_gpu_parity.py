"""GPU parity of the five C-ABI entry points against the float64 oracle.

Small shapes (several tiles each, with ragged tails in every dimension) are
compared element by element over the whole output; the full-size workloads
are compared on seeded samples the oracle computes one by one, and their
projected / merged planes bit for bit over every byte."""
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


SMALL = [
    # key, fmt, M, N, K      (pair tiles: 512 x 256 with 128-deep k-steps; scale-gradient tiles: 256 x 256)
    ("c1", NV, 64, 256, 512),
    ("nv_ragged", NV, 300, 392, 608),
    ("mx_ragged", MX, 257, 264, 544),
    ("nv_min", NV, 1, 8, 32),
    ("mx_min", MX, 3, 8, 32),
    ("mx_tall", MX, 1000, 520, 96),
    ("nv_long_k", NV, 70, 136, 2080),
    ("nv_long_m", NV, 1500, 40, 256),
    ("nv_last_tile_short", NV, 600, 264, 320),    # last 512-row tile: 88 rows
    ("mx_last_tile_one_half", MX, 1280, 136, 256),  # last 512-row tile: exactly 256 rows
]


def _wl(key, fmt, M, N, K):
    from paper_2609_04526_gb300 import synth
    if key in synth.WORKLOADS:
        return synth.WORKLOADS[key]
    return synth.custom(key, fmt, M, N, K, seed=abs(hash((fmt, M, N, K))) % 10000, kind="outlier" if fmt else "gauss")


@pytest.mark.parametrize("key,fmt,M,N,K", SMALL, ids=[s[0] for s in SMALL])
def test_full_parity_small(h, key, fmt, M, N, K):
    wl = _wl(key, fmt, M, N, K)
    lin = wl.linears[0]
    w, X, dY = setup_linear(wl, lin)
    assert (w.N, w.K, X.shape[0]) == (N, K, M)
    rng = np.random.default_rng(M * 7 + N)
    G = K // (16 if fmt == NV else 32)
    mask = torch.from_numpy(rng.integers(0, 2, size=(N, G), dtype=np.uint8)).cuda()
    Y = h.sq_fwd(w, X)
    dX = h.sq_bwd_dx(w, dY)
    g = h.sq_scale_grad(w, X, dY)
    gm = h.sq_scale_grad(w, X, dY, mask=mask)
    h.sq_sync()
    codes, scales = host(w.codes), host(w.scales)
    Y_ref = oracle.fwd(fmt, codes, scales, w.ws2, hbits(X))
    dX_ref = oracle.dx(fmt, codes, scales, w.ws2, hbits(dY))
    g_ref = oracle.scale_grad(fmt, codes, hbits(X), hbits(dY))
    assert_close(f64(Y), Y_ref, what="Y")
    assert_close(f64(dX), dX_ref, what="dX")
    assert_close(f64(g), g_ref, what="g")
    assert_close(f64(gm), g_ref * host(mask), rms=float(np.sqrt(np.mean(g_ref ** 2))), what="g*mask")


def _at(T, i, j):
    """T[i[s], j[s]] for index arrays i, j, read back as float64."""
    return f64(T[torch.from_numpy(np.asarray(i, dtype=np.int64)).to(T.device),
                 torch.from_numpy(np.asarray(j, dtype=np.int64)).to(T.device)])


def _step_checks(h, wl, lin, n_samples=4096, n_rows=32):
    """One linear run the way the benchmark's step runs it: the latent projected onto
    the grid (bytes + STE mask), the forward and input gradient on the projected bytes,
    the masked scale gradient (cut into token parts where the weight has few tiles),
    and the merge into the artifact plane. The oracle projects the same latent itself
    and feeds its own bytes and mask to its contractions; the GPU's bytes, mask, NaN
    count and merged plane must equal them bit for bit, Y and dX on seeded samples
    (corners of the last tiles included) and g on full rows (rows with masked blocks
    included) within the tolerance, and the code plane must be untouched."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    w = synth.gen_weight(wl, lin, device="cuda")
    codes0 = w.codes.clone()
    L = synth.gen_latent(wl, lin, w, device="cuda")
    X = synth.gen_act(wl, lin.x, device="cuda")
    dY = synth.gen_dy(wl, lin, device="cuda")
    nf = torch.zeros(1, dtype=torch.int32, device="cuda")
    q, mask = h.sq_project_scales(wl.fmt, L, w.ws2, nonfinite=nf)
    qw = pkg.QuantWeight(wl.fmt, lin.N, lin.K, w.codes, q, w.ws2)
    Y = h.sq_fwd(qw, X)
    dX = h.sq_bwd_dx(qw, dY)
    g = h.sq_scale_grad(qw, X, dY, mask=mask)
    art = w.scales.clone()
    ch = torch.zeros(1, dtype=torch.int64, device="cuda")
    h.sq_merge(wl.fmt, L, w.ws2, art, changed=ch)
    h.sq_sync()
    M, N, K = X.shape[0], lin.N, lin.K
    codes, Lh = host(w.codes), host(L)
    rb, rm, rnf = oracle.project(wl.fmt, Lh, w.ws2)
    assert np.array_equal(host(q), rb) and np.array_equal(host(mask), rm) and int(nf.item()) == rnf
    rs, _, rch = oracle.merge(wl.fmt, Lh, host(w.scales), w.ws2, want_delta=False)
    assert np.array_equal(host(art), rs) and int(ch.item()) == rch
    rng = np.random.default_rng(wl.seed * 31 + N + K)
    ms = rng.integers(0, M, n_samples)
    ns = rng.integers(0, N, n_samples)
    ks = rng.integers(0, K, n_samples)
    # the first and last row of every 512-row tile, the first and last column of every
    # 256-column tile, and the corners of the whole output
    tm = np.arange(0, M, 512)
    ms[:2 * len(tm)] = np.concatenate([tm, np.minimum(tm + 511, M - 1)])[: min(2 * len(tm), n_samples)]
    tn = np.arange(0, N, 256)
    ns[-2 * len(tn):] = np.concatenate([tn, np.minimum(tn + 255, N - 1)])
    tk = np.arange(0, K, 256)
    ks[-2 * len(tk):] = np.concatenate([tk, np.minimum(tk + 255, K - 1)])
    ms[:4], ns[:4], ks[:4] = [0, M - 1, 0, M - 1], [0, 0, N - 1, N - 1], [0, 0, K - 1, K - 1]
    Xb, dYb = hbits(X), hbits(dY)
    Y_ref = oracle.fwd_at(wl.fmt, codes, rb, w.ws2, Xb, ms, ns)
    dX_ref = oracle.dx_at(wl.fmt, codes, rb, w.ws2, dYb, ms, ks)
    assert_close(_at(Y, ms, ns), Y_ref, what=f"{wl.key}/{lin.name} Y samples")
    assert_close(_at(dX, ms, ks), dX_ref, what=f"{wl.key}/{lin.name} dX samples")
    masked_rows = np.nonzero((rm == 0).any(axis=1))[0]
    rows = np.unique(np.concatenate([[0, N - 1], np.arange(255, N - 1, 256)[:4], np.arange(256, N, 256)[:4],
                                     rng.integers(0, N, n_rows), masked_rows[:4]]))
    g_ref = oracle.scale_grad(wl.fmt, codes, Xb, dYb, mask=rm, rows=rows)
    rms = float(np.sqrt(np.mean(oracle.scale_grad(wl.fmt, codes, Xb, dYb, rows=rows[:8]) ** 2)))
    assert_close(f64(g)[rows], g_ref, rms=rms, what=f"{wl.key}/{lin.name} masked g rows")
    if len(masked_rows):
        assert (f64(g)[rows][rm[rows] == 0] == 0).all()
    assert torch.equal(w.codes, codes0)


@pytest.mark.parametrize("key", ["c3", "c4"])
def test_sampled_parity_full_size(h, key):
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS[key]
    _step_checks(h, wl, wl.linears[0], n_samples=8192, n_rows=48)
    torch.cuda.empty_cache()


def test_full_parity_c2(h):
    """The 4096 x 4096 x 4096 MXFP4 linear with 1% outlier channels, compared in full:
    every element of Y, dX, g and masked g against the oracle, and the projected
    E8M0 plane and mask bit for bit."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c2"]
    lin = wl.linears[0]
    w = synth.gen_weight(wl, lin, device="cuda")
    L = synth.gen_latent(wl, lin, w, device="cuda")
    L[::3] *= 2                                         # a binade step on every third row: E8M0 bytes move
    X = synth.gen_act(wl, lin.x, device="cuda")
    dY = synth.gen_dy(wl, lin, device="cuda")
    q, mask = h.sq_project_scales(wl.fmt, L, 1.0)
    mask[::7, ::5] = 0                                  # blocks the projection would pass, masked too
    qw = pkg.QuantWeight(wl.fmt, lin.N, lin.K, w.codes, q, 1.0)
    Y = h.sq_fwd(qw, X)
    dX = h.sq_bwd_dx(qw, dY)
    g = h.sq_scale_grad(qw, X, dY)
    gm = h.sq_scale_grad(qw, X, dY, mask=mask)
    h.sq_sync()
    codes = host(w.codes)
    rb, rm, _ = oracle.project(wl.fmt, host(L), 1.0)
    rm[::7, ::5] = 0
    assert np.array_equal(host(q), rb)
    Xb, dYb = hbits(X), hbits(dY)
    assert_close(f64(Y), oracle.fwd(wl.fmt, codes, rb, 1.0, Xb), what="c2 Y")
    assert_close(f64(dX), oracle.dx(wl.fmt, codes, rb, 1.0, dYb), what="c2 dX")
    g_ref = oracle.scale_grad(wl.fmt, codes, Xb, dYb)
    assert_close(f64(g), g_ref, what="c2 g")
    assert_close(f64(gm), g_ref * rm, rms=float(np.sqrt(np.mean(g_ref ** 2))), what="c2 g*mask")
    del Y, dX, X, dY
    torch.cuda.empty_cache()


C5_LINEARS = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


@pytest.mark.parametrize("name", C5_LINEARS)
def test_layer_step_c5(h, name):
    """Every linear of the 16 x 2048-token decoder layer at its launched size (the
    q/o and gate/up/down scale gradients in 5 token parts, k/v in 7) through the
    benchmark's step, checked against the oracle (see _step_checks)."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c5"]
    lin = {l.name: l for l in wl.linears}[name]
    _step_checks(h, wl, lin, n_samples=4096, n_rows=32)
    torch.cuda.empty_cache()


def test_layer_merge_c5(h):
    """Projection and merge of all 7 scale planes of the layer bit-exact against the
    oracle (bytes, mask, NaN count, merged plane, on-grid delta, changed count), with
    every code plane byte-identical."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c5"]
    total_changed = 0
    for lin in wl.linears:
        w = synth.gen_weight(wl, lin, device="cuda")
        codes_before = w.codes.clone()
        L = synth.gen_latent(wl, lin, w, device="cuda")
        nf = torch.zeros(1, dtype=torch.int32, device="cuda")
        b, m = h.sq_project_scales(wl.fmt, L, w.ws2, nonfinite=nf)
        scales = w.scales.clone()
        delta = torch.empty_like(L)
        ch = torch.zeros(1, dtype=torch.int64, device="cuda")
        h.sq_merge(wl.fmt, L, w.ws2, scales, ongrid_delta=delta, changed=ch)
        h.sq_sync()
        Lh = host(L)
        rb, rm, rnf = oracle.project(wl.fmt, Lh, w.ws2)
        rs, rd, rch = oracle.merge(wl.fmt, Lh, host(w.scales), w.ws2)
        assert np.array_equal(host(b), rb) and np.array_equal(host(m), rm) and int(nf.item()) == rnf
        assert np.array_equal(host(scales), rs) and int(ch.item()) == rch
        dh = host(delta)
        assert np.array_equal(np.isnan(dh), np.isnan(rd))
        assert np.array_equal(dh.view(np.uint32)[~np.isnan(dh)], rd.view(np.uint32)[~np.isnan(rd)])
        assert torch.equal(w.codes, codes_before)
        total_changed += rch
    frac = total_changed / sum(l.N * l.K // wl.block for l in wl.linears)
    assert 0.005 < frac < 0.2, frac


def test_layer_planes_in_one_launch_c5(h):
    """The 7 scale planes of the layer projected in one launch and merged in one
    launch (sq_project_planes / sq_merge_planes): bytes, masks, NaN counts, merged
    planes, on-grid deltas and changed counts bit-exact against the oracle, twice in
    a row (the counters' accumulators reset between calls)."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c5"]
    st = []
    for lin in wl.linears:
        w = synth.gen_weight(wl, lin, device="cuda")
        L = synth.gen_latent(wl, lin, w, device="cuda")
        L[5, :3] = float("nan")
        st.append(dict(w=w, L=L, b=torch.empty_like(w.scales), m=torch.empty_like(w.scales),
                       nf=torch.full((1,), -3, dtype=torch.int32, device="cuda"), art=w.scales.clone(),
                       d=torch.empty_like(L), ch=torch.full((1,), -3, dtype=torch.int64, device="cuda")))
    for rep in range(2):
        h.sq_project_planes(wl.fmt, [dict(latent=x["L"], bytes=x["b"], mask=x["m"], nonfinite=x["nf"], ws2=x["w"].ws2)
                                     for x in st])
        olds = [x["art"].clone() for x in st]
        h.sq_merge_planes(wl.fmt, [dict(latent=x["L"], bytes=x["art"], ongrid_delta=x["d"], changed=x["ch"],
                                        ws2=x["w"].ws2) for x in st])
        h.sq_sync()
        for x, old in zip(st, olds):
            Lh = host(x["L"])
            rb, rm, rnf = oracle.project(wl.fmt, Lh, x["w"].ws2)
            assert np.array_equal(host(x["b"]), rb) and np.array_equal(host(x["m"]), rm)
            assert int(x["nf"].item()) == rnf == 3
            rs, rd, rch = oracle.merge(wl.fmt, Lh, host(old), x["w"].ws2)
            assert np.array_equal(host(x["art"]), rs) and int(x["ch"].item()) == rch
            assert rch > 0 if rep == 0 else rch == 0
            dh = host(x["d"])
            assert np.array_equal(np.isnan(dh), np.isnan(rd))
            assert np.array_equal(dh.view(np.uint32)[~np.isnan(dh)], rd.view(np.uint32)[~np.isnan(rd)])


@pytest.mark.parametrize("fmt", [NV, MX])
def test_planes_of_mixed_shapes(h, fmt):
    """16 planes of different shapes (one block row up to a few thousand rows, the
    CTA boundaries of the one-launch kernel falling inside and between planes), edge
    latents and NaNs, per-plane ws2: equal to the oracle and to one single-plane
    call per plane, counters per plane."""
    rng = np.random.default_rng(41 + fmt)
    shapes = [(8, 16), (1, 16), (24, 32), (640, 48), (3, 256), (1000, 16), (16, 16), (2048, 64), (5, 32), (8, 896),
              (100, 160), (1, 32), (64, 16), (4096, 16), (7, 48), (33, 16)]
    planes, singles = [], []
    for j, (N, G) in enumerate(shapes):
        ws2 = float(np.float32(2.0 ** rng.integers(-12, 2) * rng.uniform(1, 2))) if fmt == NV else 1.0
        base = 448.0 * ws2 if fmt == NV else 1.0
        L = (rng.standard_normal((N, G)) * base * (0.3 if fmt == NV else 4.0)).astype(np.float32)
        if fmt == MX:
            L = np.exp2(L).astype(np.float32)
        L.flat[rng.integers(0, L.size, 1 + j % 3)] = np.nan
        L.flat[0] = base * 3
        Ld = torch.from_numpy(L).cuda()
        art = torch.from_numpy(rng.integers(0, 0x7F if fmt == NV else 255, size=(N, G), dtype=np.uint8)).cuda()
        planes.append(dict(latent=Ld, bytes=torch.empty(N, G, dtype=torch.uint8, device="cuda"),
                           mask=torch.empty(N, G, dtype=torch.uint8, device="cuda"),
                           nonfinite=torch.full((1,), 9, dtype=torch.int32, device="cuda"), ws2=ws2,
                           art=art, art0=art.clone(), ongrid_delta=torch.empty_like(Ld),
                           changed=torch.full((1,), 9, dtype=torch.int64, device="cuda")))
    h.sq_project_planes(fmt, planes)
    h.sq_merge_planes(fmt, [dict(latent=p["latent"], bytes=p["art"], ongrid_delta=p["ongrid_delta"],
                                 changed=p["changed"], ws2=p["ws2"]) for p in planes])
    h.sq_sync()
    for p in planes:
        Lh = host(p["latent"])
        rb, rm, rnf = oracle.project(fmt, Lh, p["ws2"])
        assert np.array_equal(host(p["bytes"]), rb) and np.array_equal(host(p["mask"]), rm)
        assert int(p["nonfinite"].item()) == rnf
        rs, rd, rch = oracle.merge(fmt, Lh, host(p["art0"]), p["ws2"])
        assert np.array_equal(host(p["art"]), rs) and int(p["changed"].item()) == rch
        dh = host(p["ongrid_delta"])
        assert np.array_equal(np.isnan(dh), np.isnan(rd))
        assert np.array_equal(dh.view(np.uint32)[~np.isnan(dh)], rd.view(np.uint32)[~np.isnan(rd)])
        b1, m1 = h.sq_project_scales(fmt, p["latent"], p["ws2"])
        h.sq_sync()
        assert torch.equal(b1, p["bytes"]) and torch.equal(m1, p["mask"])


@pytest.mark.parametrize("key,fmt,M,N,K", [SMALL[0], SMALL[2]], ids=["c1", "mx_ragged"])
def test_merged_artifact_is_the_trained_weight(h, key, fmt, M, N, K):
    """max|dW| = 0 in weight space (Sec. 3, merge): the artifact (unchanged codes plus the
    merged scale plane) decodes to exactly the weight the training forward used (codes plus
    the projected bytes), and the kernels give bit-identical Y, dX and g on both."""
    from paper_2609_04526_gb300 import synth
    import paper_2609_04526_gb300 as pkg
    wl = _wl(key, fmt, M, N, K)
    lin = wl.linears[0]
    w = synth.gen_weight(wl, lin, device="cuda")
    X = synth.gen_act(wl, lin.x, device="cuda")
    dY = synth.gen_dy(wl, lin, device="cuda")
    L = synth.gen_latent(wl, lin, w, device="cuda")
    L[::3] *= 2                      # a step of one binade on every third row, so E8M0 bytes move too
    codes0 = w.codes.clone()
    q, mask = h.sq_project_scales(wl.fmt, L, w.ws2)
    art = w.scales.clone()
    h.sq_merge(wl.fmt, L, w.ws2, art)
    h.sq_sync()
    c = host(w.codes)
    W_train = oracle.decode_weight(fmt, c, host(q), w.ws2, N, K)
    W_art = oracle.decode_weight(fmt, c, host(art), w.ws2, N, K)
    assert np.isfinite(W_train).all()
    assert np.max(np.abs(W_art - W_train)) == 0.0
    assert not np.array_equal(host(art), host(w.scales))       # the merge did move bytes
    outs = []
    for s in (q, art):
        qw = pkg.QuantWeight(wl.fmt, N, K, w.codes, s, w.ws2)
        outs.append((h.sq_fwd(qw, X), h.sq_bwd_dx(qw, dY), h.sq_scale_grad(qw, X, dY, mask=mask)))
    h.sq_sync()
    for a, b in zip(*outs):
        assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a.view(torch.int32),
                           b.view(torch.int16) if b.dtype == torch.bfloat16 else b.view(torch.int32))
    assert torch.equal(w.codes, codes0)


@pytest.mark.parametrize("fmt,M,N,K", [(NV, 9000, 1024, 512), (MX, 8320, 520, 1024)], ids=["nv", "mx"])
def test_token_split_scale_gradient(h, fmt, M, N, K):
    """A weight with few scale-gradient tiles (8 and 12 here) cuts its tokens into
    parts, the last one ragged: the masked sum of the parts matches the oracle on
    every block of sampled rows, the query reports the split and its scratch, two
    runs give identical bits, and the unsplit launch on the first 2048 tokens (a
    single part) matches too."""
    from paper_2609_04526_gb300 import synth
    wl = synth.custom(f"split{fmt}", fmt, M, N, K, seed=11 + fmt, kind="outlier" if fmt else "gauss")
    w, X, dY = setup_linear(wl, wl.linears[0])
    G = K // (16 if fmt == NV else 32)
    splits, nbytes = h.sq_scale_grad_workspace(w, M)
    assert splits == 4 and nbytes == splits * N * G * 4
    assert h.sq_scale_grad_workspace(w, 2048) == (1, 0)
    rng = np.random.default_rng(M)
    mask = torch.from_numpy(rng.integers(0, 2, size=(N, G), dtype=np.uint8)).cuda()
    g1 = h.sq_scale_grad(w, X, dY, mask=mask)
    g2 = h.sq_scale_grad(w, X, dY, mask=mask)
    g0 = h.sq_scale_grad(w, X[:2048], dY[:2048])
    h.sq_sync()
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    rows = np.unique(np.concatenate([[0, 255, 256, N - 1], rng.integers(0, N, 20)]))
    codes = host(w.codes)
    ref = oracle.scale_grad(fmt, codes, hbits(X), hbits(dY), mask=host(mask), rows=rows)
    full = oracle.scale_grad(fmt, codes, hbits(X), hbits(dY), rows=rows)
    assert_close(f64(g1)[rows], ref, rms=float(np.sqrt(np.mean(full ** 2))), what="split g*mask")
    ref0 = oracle.scale_grad(fmt, codes, hbits(X[:2048]), hbits(dY[:2048]), rows=rows)
    assert_close(f64(g0)[rows], ref0, what="unsplit g")


def test_split_scale_gradient_in_a_cuda_graph():
    """A fresh handle refuses to grow its split scratch inside graph capture (nothing
    is enqueued); after one call outside capture, the captured split scale gradient
    replays to the same bits as the direct call."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("graph", NV, 9000, 1024, 512, seed=5)
    w, X, dY = setup_linear(wl, wl.linears[0])
    h2 = pkg.Handle()
    assert h2.sq_scale_grad_workspace(w, 9000)[0] > 1
    s = torch.cuda.Stream()
    g = torch.zeros(1024, 32, device="cuda")
    graph = torch.cuda.CUDAGraph()
    with pytest.raises(pkg.SQError) as ei:
        with torch.cuda.graph(graph, stream=s):
            h2.sq_scale_grad(w, X, dY, g=g, stream=s)
    assert ei.value.status == -2 and "outside graph capture" in str(ei.value)
    ref = h2.sq_scale_grad(w, X, dY, stream=s)      # sizes the scratch
    h2.sq_sync(s)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        h2.sq_scale_grad(w, X, dY, g=g, stream=s)
    g.zero_()
    torch.cuda.synchronize()
    graph.replay()
    torch.cuda.synchronize()
    h2.sq_sync(s)
    assert torch.equal(g.view(torch.int32), ref.view(torch.int32))


def test_captured_graph_survives_scratch_growth():
    """A graph that captured a split scale gradient keeps replaying to the direct
    call's bits after a later call on the same handle grows the split scratch (the
    captured buffer is retired, not freed), and the larger call matches the oracle."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("grow", NV, 9000, 1024, 512, seed=6)
    w, X, dY = setup_linear(wl, wl.linears[0])
    h2 = pkg.Handle()
    small, big = h2.sq_scale_grad_workspace(w, 4096), h2.sq_scale_grad_workspace(w, 9000)
    assert 1 < small[0] < big[0] and small[1] < big[1]
    s = torch.cuda.Stream()
    ref = h2.sq_scale_grad(w, X[:4096], dY[:4096], stream=s)    # sizes the scratch for the smaller split
    h2.sq_sync(s)
    g = torch.zeros(1024, 32, device="cuda")
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        h2.sq_scale_grad(w, X[:4096], dY[:4096], g=g, stream=s)
    torch.cuda.synchronize()
    g_big = h2.sq_scale_grad(w, X, dY, stream=s)                 # grows the scratch
    h2.sq_sync(s)
    g.zero_()
    torch.cuda.synchronize()
    graph.replay()
    torch.cuda.synchronize()
    h2.sq_sync(s)
    assert torch.equal(g.view(torch.int32), ref.view(torch.int32))
    rows = np.array([0, 255, 256, 511, 700, 1023])
    ref_big = oracle.scale_grad(NV, host(w.codes), hbits(X), hbits(dY), rows=rows)
    assert_close(f64(g_big)[rows], ref_big, what="grown split g")
    del graph
    h2.close()


def _edge_latents(fmt, ws2):
    rng = np.random.default_rng(99)
    vals = []
    if fmt == NV:
        grid = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).float().numpy()
        pos = grid[1:0x7F].astype(np.float64)
        mids = (pos[:-1] + pos[1:]) / 2
        cap = np.float32(448.0) * np.float32(ws2)
        vals += list(pos * ws2) + list(mids * ws2) + list(-mids * ws2)
        vals += [cap, np.nextafter(cap, np.float32(1e30)), cap * 2, -cap, -cap * 3]
        vals += [2.0 ** -10 * ws2, 2.0 ** -11 * ws2, 1e-30, -1e-30]
    else:
        e = np.arange(-130, 130)
        vals += list(np.ldexp(1.0, e)) + list(np.ldexp(np.sqrt(2.0), e)) + list(np.ldexp(1.4142135, e))
        vals += list(np.ldexp(1.4142137, e)) + [2.0 ** -149, 3e-45, 1.5 * 2.0 ** 127, 3.4e38, -1.0]
    vals += [0.0, -0.0, np.inf, -np.inf, np.nan, -np.nan]
    vals += list(rng.standard_normal(1000) * (ws2 if fmt == NV else 1e-3))
    a = np.array(vals, dtype=np.float32)
    return a  # length not a multiple of 16 on purpose


@pytest.mark.parametrize("fmt,ws2", [(NV, 1.0), (NV, 0.0123), (NV, 2.0 ** -9), (MX, 1.0)])
def test_projection_and_merge_edges_bit_exact(h, fmt, ws2):
    ws2 = float(np.float32(ws2))
    L = _edge_latents(fmt, ws2)
    n = L.size
    for count in (n, n - 5, 17, 16, 15, 1):
        Lc = L[:count].reshape(1, count)
        Ld = torch.from_numpy(Lc.copy()).cuda()
        nf = torch.full((1,), 77, dtype=torch.int32, device="cuda")
        b, m = h.sq_project_scales(fmt, Ld, ws2, nonfinite=nf)
        old = torch.from_numpy(np.random.default_rng(count).integers(0, 0x7F if fmt == NV else 255, size=(1, count),
                                                                      dtype=np.uint8)).cuda()
        sc = old.clone()
        delta = torch.empty_like(Ld)
        ch = torch.full((1,), 5, dtype=torch.int64, device="cuda")
        h.sq_merge(fmt, Ld, ws2, sc, ongrid_delta=delta, changed=ch)
        h.sq_sync()
        rb, rm, rnf = oracle.project(fmt, Lc, ws2)
        assert np.array_equal(host(b), rb), np.nonzero(host(b) != rb)
        assert np.array_equal(host(m), rm)
        assert int(nf.item()) == rnf
        rs, rd, rch = oracle.merge(fmt, Lc, host(old), ws2)
        assert np.array_equal(host(sc), rs) and int(ch.item()) == rch
        dh = host(delta)
        assert np.array_equal(np.isnan(dh), np.isnan(rd))
        ok = ~np.isnan(rd)
        assert np.array_equal(dh.view(np.uint32)[ok], rd.view(np.uint32)[ok])


def test_projection_dense_sweep_bit_exact(h):
    """2^24 latents spread over the whole E4M3 range (and past the ceiling) and a
    full fp32 binade for E8M0: every byte and mask bit equals the oracle's."""
    rng = np.random.default_rng(7)
    ws2 = float(np.float32(0.00731))
    L = (np.exp(rng.uniform(np.log(1e-7), np.log(600), size=1 << 24)) * rng.choice([-1, 1], size=1 << 24) * ws2)
    L = L.astype(np.float32).reshape(1 << 12, 1 << 12)
    b, m = h.sq_project_scales(NV, torch.from_numpy(L).cuda(), ws2)
    rb, rm, _ = oracle.project(NV, L, ws2)
    assert np.array_equal(host(b), rb) and np.array_equal(host(m), rm)
    j = np.arange(1 << 23, dtype=np.int64)
    Lm = (1.0 + j / float(1 << 23)).astype(np.float32).reshape(1 << 11, 1 << 12) * np.float32(2.0 ** -20)
    b, m = h.sq_project_scales(MX, torch.from_numpy(Lm).cuda(), 1.0)
    rb, rm, _ = oracle.project(MX, Lm, 1.0)
    assert np.array_equal(host(b), rb) and np.array_equal(host(m), rm)


@pytest.mark.parametrize("ws2", [0.00731, 1.0, 0.0123, 2.0 ** -9, 3.3e-4, 5.1e3])
def test_projection_near_e4m3_midpoints_bit_exact(h, ws2):
    """Latents whose quotient by ws2 lies at, or within 40 fp32 ulps of, every
    rounding midpoint and grid value of E4M3 (normal and subnormal range, both
    signs), each also nudged by one ulp of the latent: the projected bytes and mask
    equal the oracle's. These are the values where rounding the quotient to E4M3
    depends on its last bits."""
    ws2 = float(np.float32(ws2))
    grid = np.array([m * 2.0 ** -9 for m in range(1, 8)] +
                    [(1 + m / 8) * 2.0 ** e for e in range(-6, 9) for m in range(8)], dtype=np.float64)
    grid = grid[grid <= 448]
    mids = (grid[:-1] + grid[1:]) / 2
    t = np.concatenate([grid, mids, [2.0 ** -10]]).astype(np.float32)
    k = np.arange(-40, 41, dtype=np.int64)
    tb = (t.view(np.uint32).astype(np.int64)[:, None] + k[None, :]).ravel()
    q = tb[(tb > 0) & (tb < 0x7F800000)].astype(np.uint32).view(np.float32)
    L = (q.astype(np.float64) * ws2).astype(np.float32)
    L = np.concatenate([L, np.nextafter(L, np.float32(np.inf)), np.nextafter(L, np.float32(0))])
    L = np.concatenate([L, -L]).astype(np.float32)
    L = L[: L.size // 16 * 16].reshape(16, -1)
    b, m = h.sq_project_scales(NV, torch.from_numpy(L.copy()).cuda(), ws2)
    h.sq_sync()
    rb, rm, _ = oracle.project(NV, L, ws2)
    bad = np.nonzero(host(b) != rb)
    assert np.array_equal(host(b), rb), (L[bad][:8], host(b)[bad][:8], rb[bad][:8])
    assert np.array_equal(host(m), rm)


def test_empty_batch_and_sync(h):
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("e", NV, 4, 64, 128, seed=1)
    w, X, dY = setup_linear(wl, wl.linears[0])
    g = torch.full((64, 8), 3.0, device="cuda")
    h.sq_scale_grad(w, X[:0], dY[:0], g=g)
    Y = torch.full((0, 64), 1.0, dtype=torch.bfloat16, device="cuda")
    h.sq_fwd(w, X[:0], Y)
    h.sq_sync()
    assert (g == 0).all()


def test_bounded_wait_runs_out_and_the_context_survives(h):
    """The failure path without a fault: a wait on a barrier nothing arrives on runs
    out after its bound, the next sync reports SQ_ERR_DEVICE_TIMEOUT, the sync after
    it is clean, and the same handle and context still compute correct results."""
    import time
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    h.sq_sync()
    t0 = time.time()
    h.sq_selftest_wait_timeout()
    with pytest.raises(pkg.SQError) as info:
        h.sq_sync()
    waited = time.time() - t0
    assert info.value.status == -5 and "bounded device wait" in str(info.value)
    assert 0.5 < waited < 30, waited
    h.sq_sync()                                   # the error word was cleared
    wl = synth.custom("t", NV, 70, 136, 2080, seed=3)
    w, X, dY = setup_linear(wl, wl.linears[0])
    Y = h.sq_fwd(w, X)
    h.sq_sync()
    ref = oracle.fwd(NV, host(w.codes), host(w.scales), w.ws2, hbits(X))
    assert_close(f64(Y), ref, what="Y after a device timeout")


def test_invalid_args_on_device(h):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    wl = synth.custom("e", NV, 4, 64, 128, seed=2)
    w, X, dY = setup_linear(wl, wl.linears[0])
    bad = pkg.QuantWeight(w.fmt, 60, w.K, w.codes, w.scales, w.ws2)
    with pytest.raises(pkg.SQError):
        h.sq_fwd(bad, X)
    with pytest.raises(pkg.SQError):
        h.sq_fwd(w, X[:, 1:])  # misaligned base
