"""GPU parity of rollback, scale-only swap and the byte audit (Sec. 5 Payoff 3,
"Hot-swap", byte-level audit) against the oracle, through the C ABI: bit-exact
bytes and counts, ragged sizes, the full Llama-8B layer planes, and the code plane
audited unchanged across merge, rollback and swap."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import host

pytestmark = pytest.mark.gpu

NV, MX = 0, 1


@pytest.fixture(scope="module")
def h():
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build
    build.build()
    assert torch.cuda.is_available()
    return pkg.Handle()


def _scale(fmt, bytes_, ws2):
    if fmt == NV:
        g = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).to(torch.float32).numpy()
        return (g[bytes_] * np.float32(ws2)).astype(np.float32)
    return np.ldexp(np.float32(1.0), bytes_.astype(np.int32) - 127).astype(np.float32)


@pytest.mark.parametrize("fmt,ws2,N,G", [(NV, 0.0021, 256, 96), (NV, 1.0 / (6 * 448), 37, 48), (MX, 1.0, 129, 80),
                                         (NV, 1.0, 1, 16)])
def test_merge_rollback_round_trip_bit_exact(h, fmt, ws2, N, G):
    rng = np.random.default_rng(N * 7 + G)
    old = (rng.integers(0x10, 0x76, size=(N, G)) if fmt == NV else rng.integers(60, 190, size=(N, G))).astype(np.uint8)
    L = (_scale(fmt, old, ws2) * np.exp(rng.uniform(-0.6, 0.6, size=old.shape))).astype(np.float32)
    art = torch.from_numpy(old).cuda()
    Ld = torch.from_numpy(L).cuda()
    delta = torch.empty(N, G, dtype=torch.float32, device="cuda")
    ch = torch.zeros(1, dtype=torch.int64, device="cuda")
    h.sq_merge(fmt, Ld, ws2, art, ongrid_delta=delta, changed=ch)
    merged = art.clone()
    ch2 = torch.zeros(1, dtype=torch.int64, device="cuda")
    h.sq_rollback(fmt, delta, ws2, art, changed=ch2)
    h.sq_sync()
    rnew, rdelta, rch = oracle.merge(fmt, L, old, ws2)
    assert np.array_equal(host(merged), rnew) and int(ch.item()) == rch
    assert np.array_equal(host(delta).view(np.uint32), rdelta.view(np.uint32))
    rback, rch2 = oracle.rollback(fmt, rnew, rdelta, ws2)
    assert np.array_equal(rback, old)
    assert np.array_equal(host(art), rback) and int(ch2.item()) == rch2 == rch
    # the raw training delta: GPU and oracle agree byte for byte on what it (wrongly) restores
    raw = (L - _scale(fmt, old, ws2)).astype(np.float32)
    art2 = merged.clone()
    h.sq_rollback(fmt, torch.from_numpy(raw).cuda(), ws2, art2)
    h.sq_sync()
    rraw, _ = oracle.rollback(fmt, rnew, raw, ws2)
    assert np.array_equal(host(art2), rraw)


@pytest.mark.parametrize("count", [0, 1, 15, 16, 17, 4096 + 5, 1 << 20])
def test_swap_and_audit_match_oracle(h, count):
    rng = np.random.default_rng(count + 3)
    a = rng.integers(0, 256, size=count, dtype=np.uint8)
    b = a.copy()
    flip = rng.random(count) < 0.047
    b[flip] = (b[flip] + rng.integers(1, 256, size=int(flip.sum()))).astype(np.uint8)
    da, db = torch.from_numpy(a).cuda(), torch.from_numpy(b).cuda()
    n = h.sq_count_diff(da, db)
    ch = torch.zeros(1, dtype=torch.int64, device="cuda")
    dst = da.clone().view(1, -1) if count else torch.empty(0, 0, dtype=torch.uint8, device="cuda")
    src = db.view(1, -1) if count else torch.empty(0, 0, dtype=torch.uint8, device="cuda")
    h.sq_swap_scales(src, dst, changed=ch)
    h.sq_sync()
    assert int(n.item()) == oracle.count_diff(a, b) == int(flip.sum())
    rnew, rch = oracle.swap(b, a)
    assert np.array_equal(host(dst).reshape(-1), rnew) and int(ch.item()) == rch


def test_layer_planes_merge_rollback_swap_and_code_audit(h):
    """Every plane of the Llama-3-8B layer: merge the synthetic latents with the
    on-grid delta, audit the code plane (0 bytes differ), roll back (the base
    returns wherever the merge stayed within a factor 2, and the GPU matches the
    oracle on every byte), and swap the merged plane back in."""
    from paper_2609_04526_gb300 import synth
    wl = synth.WORKLOADS["c5"]
    for lin in wl.linears:
        w = synth.gen_weight(wl, lin, device="cuda")
        L = synth.gen_latent(wl, lin, w, device="cuda")
        codes0 = w.codes.clone()
        art = w.scales.clone()
        delta = torch.empty(L.shape, dtype=torch.float32, device="cuda")
        h.sq_merge(wl.fmt, L, w.ws2, art, ongrid_delta=delta)
        merged = art.clone()
        h.sq_rollback(wl.fmt, delta, w.ws2, art)
        code_diff = h.sq_count_diff(codes0, w.codes)
        back_diff = h.sq_count_diff(art, w.scales)
        ch = torch.zeros(1, dtype=torch.int64, device="cuda")
        h.sq_swap_scales(merged, art, changed=ch)
        h.sq_sync()
        assert int(code_diff.item()) == 0
        rnew, rdelta, _ = oracle.merge(wl.fmt, host(L), host(w.scales), w.ws2)
        assert np.array_equal(host(merged), rnew)
        rback, _ = oracle.rollback(wl.fmt, rnew, rdelta, w.ws2)
        assert int(back_diff.item()) == oracle.count_diff(rback, host(w.scales))
        s_old = _scale(wl.fmt, host(w.scales), w.ws2)
        s_new = _scale(wl.fmt, rnew, w.ws2)
        near = (s_new <= 2 * s_old) & (s_new >= s_old / 2)
        assert np.array_equal(rback[near], host(w.scales)[near])     # restored wherever Sterbenz applies
        assert torch.equal(art, merged) and int(ch.item()) == oracle.count_diff(rback, rnew)


def test_rollback_swap_audit_invalid_args(h):
    import paper_2609_04526_gb300 as pkg
    dev = "cuda"
    p = torch.zeros(8, 16, dtype=torch.uint8, device=dev)
    d = torch.zeros(8, 16, dtype=torch.float32, device=dev)
    bad = [
        lambda: h.sq_rollback(NV, d, float("nan"), p),                     # ws2
        lambda: h.sq_rollback(MX, d, 0.5, p),                              # MXFP4 ws2 != 1
        lambda: h.sq_rollback(NV, d.view(-1)[1:113].view(7, 16), 1.0, p[:7]),   # misaligned delta
        lambda: h.sq_swap_scales(p.view(-1)[1:113].view(7, 16), p[:7]),   # misaligned src
        lambda: h.sq_count_diff(p.view(-1)[1:], p.view(-1)[1:]),         # misaligned buffers
    ]
    for call in bad:
        with pytest.raises(pkg.SQError) as ei:
            call()
        assert ei.value.status == -1
