"""Byte and parameter accounting of the Llama-3-8B-shaped layer against the
paper's printed totals (Sec. 5 Payoffs 2-3, param-efficiency Pareto). Pins the
layer shapes, two codes per byte and one scale byte per 16-block."""
from conftest import read_golden

from paper_2609_04526_gb300 import synth


def test_llama8b_layer_accounting():
    gold = read_golden("llama8b_accounting.txt")
    wl = synth.WORKLOADS["c5"]
    layers = 32
    nk = sum(l.N * l.K for l in wl.linears)
    assert nk == 218_103_808
    code_bytes = layers * nk // 2
    scale_bytes = layers * nk // wl.block
    assert code_bytes == 3_489_660_928
    assert round(code_bytes / 1e9, 2) == gold["code_plane_gb"][0]
    assert code_bytes / 2 ** 20 == gold["code_plane_mib"][0]
    assert scale_bytes / 2 ** 20 == gold["scale_plane_mib"][0]
    assert 8 * scale_bytes / (layers * nk) == gold["scale_bits_per_param"][0]
    assert round(4 * scale_bytes / 1e9, 1) == gold["rollback_delta_gb"][0]
    per_rank_scale = layers * sum(l.N + l.K // wl.block for l in wl.linears)
    per_rank_qlora = layers * sum(l.N + l.K for l in wl.linears)
    assert round(per_rank_scale / 1e6, 3) == gold["scale_params_per_rank_m"][0]
    assert round(per_rank_qlora / 1e6, 3) == gold["qlora_params_per_rank_m"][0]
    assert wl.M == 16 * 2048


def test_fixture_quantizer_shapes_and_ranges():
    """The synthetic checkpoint generator emits packed codes [N, K/2], block scale
    bytes [N, K/B] and (NVFP4) a positive tensor scale; MXFP4 bytes stay finite."""
    for key in ("c1",):
        wl = synth.WORKLOADS[key]
        lin = wl.linears[0]
        w = synth.gen_weight(wl, lin)
        assert w.codes.shape == (lin.N, lin.K // 2) and w.scales.shape == (lin.N, lin.K // 16)
        assert w.ws2 > 0 and int(w.scales.max()) <= 0x7E
    wl = synth.custom("t", synth.MXFP4, 8, 64, 256, seed=9)
    w = synth.gen_weight(wl, wl.linears[0])
    assert w.scales.shape == (64, 8) and int(w.scales.max()) < 255 and w.ws2 == 1.0
