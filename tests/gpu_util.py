"""Shared helpers of the GPU parity tests: workload setup on the device, host
copies for the oracle, and the tolerance check."""
import numpy as np
import torch

from conftest import bf16_bits

# Per-element bar for floating-point outputs: relative 2e-2 plus an absolute
# floor of 1e-3 x the RMS of the oracle's output (bf16 inputs, fp32 accumulation).
RTOL = 2e-2
AFLOOR = 1e-3


def assert_close(gpu, ref, rms=None, what=""):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    rms = float(np.sqrt(np.mean(ref ** 2))) if rms is None else rms
    err = np.abs(gpu - ref)
    bound = RTOL * np.abs(ref) + AFLOOR * rms
    bad = ~(err <= bound)
    if bad.any():
        i = int(np.argmax(np.where(bad, err / np.maximum(bound, 1e-300), 0)))
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} elements outside tolerance; "
                             f"worst flat index {i}: gpu {gpu.flat[i]!r} oracle {ref.flat[i]!r} bound {bound.flat[i]!r}")


def setup_linear(wl, lin, device="cuda", M=None):
    """Returns (QuantWeight on device, X, dY on device) for one linear of a workload."""
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import synth
    w = synth.gen_weight(wl, lin, device=device)
    qw = pkg.QuantWeight(w.fmt, w.N, w.K, w.codes.contiguous(), w.scales.contiguous(), w.ws2)
    X = synth.gen_act(wl, lin.x, M=M, device=device).contiguous()
    dY = synth.gen_dy(wl, lin, M=M, device=device).contiguous()
    return qw, X, dY


def host(t):
    return t.detach().cpu().numpy()


def hbits(t):
    return bf16_bits(t)


def f64(t):
    return t.detach().float().cpu().double().numpy()
