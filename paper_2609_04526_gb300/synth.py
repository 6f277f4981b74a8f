"""Seeded synthetic workloads: Llama-3-8B-shaped NVFP4 / MXFP4 linears and activations.

This module only draws inputs. It holds none of the scale-only training step's
arithmetic (decode, contraction, grid projection, merge); both the CUDA path and
the float64 oracle consume what it returns.

The checkpoints stand in for the paper's Llama-3.1-8B NVFP4 and gpt-oss MXFP4
bases (not available offline). They are built with a round-to-nearest fixture
quantizer of a Gaussian weight (the amax/6 rule of the block-statistics appendix
for NVFP4, the HF ceil(log2(amax/6)) exponent rule for MXFP4), using torch's own
float8 cast for the E4M3 byte. The E2M1 code is the nearest element of the
printed alphabet +-{0,.5,1,1.5,2,3,4,6} (ties to the even mantissa, saturating
at 6); codes are packed two per byte, even k in the low nibble.
"""
from __future__ import annotations

import dataclasses
import zlib
from typing import Dict, List, Optional

import math

import torch

NVFP4 = 0
MXFP4 = 1
BLOCK = {NVFP4: 16, MXFP4: 32}
FMT_NAME = {NVFP4: "nvfp4", MXFP4: "mxfp4"}

# E2M1 magnitudes (printed alphabet) and the midpoints between neighbours; used
# only to pick fixture codes for a Gaussian weight.
_E2M1_MAG = (0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0)
_E2M1_MID = (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)


@dataclasses.dataclass(frozen=True)
class Linear:
    name: str
    N: int          # out features
    K: int          # in features
    x: str          # activation that feeds it


@dataclasses.dataclass(frozen=True)
class Workload:
    key: str
    title: str
    fmt: int
    M: int
    linears: tuple
    acts: tuple                 # (name, K, kind) with kind in {"gauss", "outlier", "silu"}
    seed: int
    w_std: float = 0.02
    dy_std: float = 1e-3
    # relative RMS of the latent perturbation: starting from on-grid scales, a byte
    # moves only when it exceeds half a grid step; 0.021 moves ~4.7% of NVFP4
    # bytes, the share the paper's Llama-8B merge touched (Sec. 5, Payoff 3)
    latent_rel_rms: float = 0.021
    latent_rank: int = 58           # rank of the latent perturbation (scale r58)
    above_ceiling_frac: float = 1e-3

    @property
    def block(self) -> int:
        return BLOCK[self.fmt]

    def flops(self) -> int:
        """6*M*N*K summed over linears: forward, input gradient and the dW contraction."""
        return sum(6 * self.M * l.N * l.K for l in self.linears)


def _layer(M, fmt, seed, key, title):
    d, kv, f = 4096, 1024, 14336
    lin = (
        Linear("q_proj", d, d, "x_attn"),
        Linear("k_proj", kv, d, "x_attn"),
        Linear("v_proj", kv, d, "x_attn"),
        Linear("o_proj", d, d, "x_o"),
        Linear("gate_proj", f, d, "x_mlp"),
        Linear("up_proj", f, d, "x_mlp"),
        Linear("down_proj", d, f, "x_down"),
    )
    acts = (("x_attn", d, "gauss"), ("x_o", d, "gauss"), ("x_mlp", d, "gauss"), ("x_down", f, "silu"))
    return Workload(key, title, fmt, M, lin, acts, seed)


WORKLOADS: Dict[str, Workload] = {
    "c1": Workload("c1", "tiny NVFP4 linear 64x256x512", NVFP4, 64,
                   (Linear("w", 256, 512, "x"),), (("x", 512, "gauss"),), 1001),
    "c2": Workload("c2", "Llama-3-8B q_proj 4096x4096x4096 MXFP4, 1% outlier channels x20", MXFP4, 4096,
                   (Linear("q_proj", 4096, 4096, "x"),), (("x", 4096, "outlier"),), 1002),
    "c3": Workload("c3", "Llama-3-8B gate/up_proj 8192x14336x4096 NVFP4", NVFP4, 8192,
                   (Linear("gate_proj", 14336, 4096, "x"),), (("x", 4096, "gauss"),), 1003),
    "c4": Workload("c4", "Llama-3-8B down_proj 8192x4096x14336 NVFP4, SiLU-gated input", NVFP4, 8192,
                   (Linear("down_proj", 4096, 14336, "x"),), (("x", 14336, "silu"),), 1004),
    "c5": _layer(32768, NVFP4, 1005, "c5",
                 "Llama-3-8B decoder layer (q,k,v,o,gate,up,down) NVFP4, 16x2048 tokens"),
}


def custom(key: str, fmt: int, M: int, N: int, K: int, seed: int, kind: str = "gauss") -> Workload:
    """A single-linear workload of any shape (parity cases with ragged tails)."""
    return Workload(key, f"{FMT_NAME[fmt]} {M}x{N}x{K}", fmt, M, (Linear("w", N, K, "x"),),
                    (("x", K, kind),), seed)


def _gen(seed: int, name: str, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed * 1_000_003 + zlib.crc32(name.encode()))
    return g


@dataclasses.dataclass
class Weight:
    fmt: int
    N: int
    K: int
    codes: torch.Tensor     # [N, K/2] uint8
    scales: torch.Tensor    # [N, K/B] uint8
    ws2: float


def _e2m1_index(a: torch.Tensor) -> torch.Tensor:
    """Index into _E2M1_MAG of the nearest magnitude to a >= 0 (ties to even index)."""
    mids = torch.tensor(_E2M1_MID, dtype=a.dtype, device=a.device)
    idx = torch.bucketize(a, mids)              # a == mid -> lower index
    at_mid = (idx < 7) & (a == mids[idx.clamp(max=6)])
    idx = idx + (at_mid & (idx % 2 == 1)).to(idx.dtype)
    return idx


def quantize_rtn(w: torch.Tensor, fmt: int) -> Weight:
    """Fixture RTN quantizer of an fp32 weight [N, K] into packed codes and block scales."""
    N, K = w.shape
    B = BLOCK[fmt]
    G = K // B
    wb = w.reshape(N, G, B)
    amax = wb.abs().amax(dim=2)
    if fmt == NVFP4:
        ws2 = float(w.abs().max()) / (6.0 * 448.0)
        if ws2 == 0.0:
            ws2 = 1.0
        x = (amax / (6.0 * ws2)).clamp(max=448.0)
        sb = x.to(torch.float8_e4m3fn)
        scales = sb.view(torch.uint8)
        s = sb.to(torch.float32) * ws2
    else:
        ws2 = 1.0
        x = amax / 6.0
        m, e = torch.frexp(x)
        e = torch.where(m == 0.5, e - 1, e)                 # ceil(log2 x)
        byte = (e + 127).clamp(0, 254)
        byte = torch.where(amax > 0, byte, torch.zeros_like(byte))
        scales = byte.to(torch.uint8)
        s = torch.ldexp(torch.ones_like(x), (byte - 127).to(torch.int32))
    s_full = s.unsqueeze(2)
    r = torch.where(s_full > 0, wb / s_full, torch.zeros_like(wb))
    idx = _e2m1_index(r.abs())
    sign = ((r < 0) & (idx > 0)).to(torch.uint8)
    nib = (sign << 3) | idx.to(torch.uint8)
    nib = nib.reshape(N, K)
    codes = (nib[:, 0::2] | (nib[:, 1::2] << 4)).contiguous()
    return Weight(fmt, N, K, codes, scales.contiguous(), float(ws2))


def gen_weight(wl: Workload, lin: Linear, device="cpu") -> Weight:
    g = _gen(wl.seed, "W:" + lin.name, device)
    w = torch.randn(lin.N, lin.K, generator=g, device=device, dtype=torch.float32) * wl.w_std
    return quantize_rtn(w, wl.fmt)


def gen_act(wl: Workload, name: str, M: Optional[int] = None, device="cpu") -> torch.Tensor:
    """Activation [M, K] in bf16 (fp32 draw, then a round-to-nearest-even cast)."""
    K, kind = next((k, kd) for (n, k, kd) in wl.acts if n == name)
    M = wl.M if M is None else M
    g = _gen(wl.seed, "X:" + name, device)
    if kind == "silu":
        a = torch.randn(M, K, generator=g, device=device, dtype=torch.float32)
        b = torch.randn(M, K, generator=g, device=device, dtype=torch.float32)
        x = torch.nn.functional.silu(a) * b
    else:
        x = torch.randn(M, K, generator=g, device=device, dtype=torch.float32)
        if kind == "outlier":
            n_out = round(0.01 * K)
            ch = torch.randperm(K, generator=_gen(wl.seed, "outlier:" + name, "cpu"))[:n_out]
            x[:, ch.to(device)] *= 20.0
    return x.to(torch.bfloat16)


def gen_dy(wl: Workload, lin: Linear, M: Optional[int] = None, device="cpu") -> torch.Tensor:
    M = wl.M if M is None else M
    g = _gen(wl.seed, "dY:" + lin.name, device)
    return (torch.randn(M, lin.N, generator=g, device=device, dtype=torch.float32) * wl.dy_std).to(torch.bfloat16)


def gen_latent(wl: Workload, lin: Linear, weight: Weight, device="cpu") -> torch.Tensor:
    """Latent (pre-projection) effective scales, fp32 [N, G], absolute units.

    L = s * (1 + eps): s is the checkpoint's current effective scale (decoded with
    torch's float8 cast), eps a seeded rank-r Gaussian product scaled to a relative
    RMS, so a few percent of bytes move. For NVFP4 a small fraction of latents is
    pushed above the 448*ws2 ceiling (exercises the clamp)."""
    N, G = weight.scales.shape
    g = _gen(wl.seed, "L:" + lin.name, device)
    sb = weight.scales.to(device)
    if wl.fmt == NVFP4:
        s = sb.view(torch.float8_e4m3fn).to(torch.float32) * weight.ws2
    else:
        s = torch.ldexp(torch.ones(N, G, device=device), sb.to(torch.int32) - 127)
    r = wl.latent_rank
    P = torch.randn(N, r, generator=g, device=device)
    Q = torch.randn(r, G, generator=g, device=device)
    eps = P @ Q
    eps = eps * (wl.latent_rel_rms / eps.pow(2).mean().sqrt().clamp(min=1e-30))
    L = s * (1.0 + eps)
    if wl.fmt == NVFP4 and wl.above_ceiling_frac > 0:
        cap = 448.0 * weight.ws2
        u = torch.rand(N, G, generator=g, device=device)
        hot = torch.rand(N, G, generator=g, device=device) < wl.above_ceiling_frac
        L = torch.where(hot, cap * (1.0 + 0.5 * u), L)
    return L.contiguous()


def gen_adapter(wl: Workload, lin: Linear, weight: Weight, r: int = 58, alpha: float = 16.0, device="cpu"):
    """Low-rank scale adapter factors in mid-training: B [N, r] and A [r, G] bf16 and
    alpha/r (the adapter of Sec. 3 "Scale-QLoRA forward"; r = 58 is the paper's
    Llama-8B rank). Seeded Gaussians, A ~ N(0, 1/r) and B scaled so (alpha/r) (B A)
    has the workload's latent relative RMS of the median effective scale, so a few
    percent of bytes move. Returns (B, A, alpha_over_r)."""
    N, G = weight.scales.shape
    g = _gen(wl.seed, "adapter:" + lin.name, device)
    sb = weight.scales.to(device)
    if wl.fmt == NVFP4:
        s = sb.view(torch.float8_e4m3fn).to(torch.float32) * weight.ws2
    else:
        s = torch.ldexp(torch.ones(N, G, device=device), sb.to(torch.int32) - 127)
    aor = alpha / r
    s_med = float(s.abs().float().median().clamp(min=1e-30))
    A = torch.randn(r, G, generator=g, device=device) / math.sqrt(r)
    B = torch.randn(N, r, generator=g, device=device) * (wl.latent_rel_rms * s_med / aor)
    return B.to(torch.bfloat16).contiguous(), A.to(torch.bfloat16).contiguous(), aor


def act_names(wl: Workload) -> List[str]:
    return [a[0] for a in wl.acts]


# ---------------------------------------------------------------- MoE experts
# The paper's MoE bases (Sec. 4: Qwen3-30B-A3B NVFP4; gpt-oss-120B, 128 experts,
# native MXFP4) are not available offline and the paper prints no expert shapes;
# these workloads take the experts' shapes from the public model configurations
# (Qwen3-30B-A3B: 128 experts, top-8, hidden 2048, expert intermediate 768;
# gpt-oss-120B: 128 experts, top-4, hidden 2880, intermediate 2880, its fused
# gate/up projection drawn as two linears). A batch of T tokens is routed top-k
# by a seeded router whose expert popularity is log-normal (route_sigma), so the
# per-expert token counts are ragged like a load-balanced router's; tokens are
# sorted by expert, so expert e owns rows offsets[e] .. offsets[e+1]-1.

@dataclasses.dataclass(frozen=True)
class MoEWorkload:
    key: str
    title: str
    fmt: int
    T: int                      # tokens of the batch
    top_k: int                  # experts per token
    E: int                      # experts per linear
    linears: tuple              # per-expert Linear shapes
    acts: tuple                 # (name, K, kind) as in Workload
    seed: int
    route_sigma: float = 0.3    # log-normal spread of the experts' popularity (max load ~2.2x the mean)
    counts: Optional[tuple] = None  # fixed per-expert token counts (tests); else drawn by the router
    w_std: float = 0.02
    dy_std: float = 1e-3
    latent_rel_rms: float = 0.021   # as Workload
    latent_rank: int = 54           # the paper's MoE scale rank (scale r54)
    above_ceiling_frac: float = 1e-3

    @property
    def block(self) -> int:
        return BLOCK[self.fmt]

    @property
    def M(self) -> int:
        """Routed token rows of every expert linear (each token appears top_k times)."""
        return sum(self.counts) if self.counts is not None else self.T * self.top_k

    def flops(self) -> int:
        """6 * (routed rows) * N * K summed over the expert linears."""
        return sum(6 * self.M * l.N * l.K for l in self.linears)


def _moe(key, title, fmt, T, top_k, E, hidden, inter, seed):
    lin = (Linear("gate_proj", inter, hidden, "x_moe"), Linear("up_proj", inter, hidden, "x_moe"),
           Linear("down_proj", hidden, inter, "x_moe_down"))
    acts = (("x_moe", hidden, "gauss"), ("x_moe_down", inter, "silu"))
    return MoEWorkload(key, title, fmt, T, top_k, E, lin, acts, seed)


MOE_WORKLOADS: Dict[str, MoEWorkload] = {
    "moe_qwen": _moe("moe_qwen", "Qwen3-30B-A3B-shaped MoE experts (128 x {768x2048, 2048x768}) NVFP4, "
                     "16x2048 tokens top-8", NVFP4, 32768, 8, 128, 2048, 768, 2001),
    "moe_gptoss": _moe("moe_gptoss", "gpt-oss-120B-shaped MoE experts (128 x 2880x2880) MXFP4, 16x2048 tokens top-4",
                       MXFP4, 32768, 4, 128, 2880, 2880, 2002),
}


def custom_moe(key: str, fmt: int, counts, N: int, K: int, seed: int, kind: str = "gauss") -> MoEWorkload:
    """One expert linear [N, K] over len(counts) experts with fixed token counts."""
    return MoEWorkload(key, f"{FMT_NAME[fmt]} {len(counts)} experts {N}x{K}", fmt, sum(counts), 1, len(counts),
                       (Linear("w", N, K, "x"),), (("x", K, kind),), seed, counts=tuple(int(c) for c in counts))


def gen_routing(wl: MoEWorkload) -> List[int]:
    """Tokens routed to each expert (sums to wl.M): each of the T tokens picks top_k
    distinct experts with probability proportional to the experts' popularity."""
    if wl.counts is not None:
        return list(wl.counts)
    g = _gen(wl.seed, "router", "cpu")
    pop = torch.exp(wl.route_sigma * torch.randn(wl.E, generator=g))
    picks = torch.multinomial(pop.expand(wl.T, wl.E), wl.top_k, replacement=False, generator=g)
    return torch.bincount(picks.reshape(-1), minlength=wl.E).tolist()


def offsets_of(counts) -> List[int]:
    out = [0]
    for c in counts:
        out.append(out[-1] + int(c))
    return out


@dataclasses.dataclass
class Experts:
    fmt: int
    E: int
    N: int
    K: int
    codes: torch.Tensor     # [E, N, K/2] uint8
    scales: torch.Tensor    # [E, N, K/B] uint8
    ws2: List[float]        # one tensor scale per expert


def gen_experts(wl: MoEWorkload, lin: Linear, device="cpu") -> Experts:
    """Every expert's weight drawn and RTN-quantized like gen_weight (one draw per expert)."""
    codes = torch.empty(wl.E, lin.N, lin.K // 2, dtype=torch.uint8, device=device)
    scales = torch.empty(wl.E, lin.N, lin.K // BLOCK[wl.fmt], dtype=torch.uint8, device=device)
    ws2 = []
    for e in range(wl.E):
        g = _gen(wl.seed, f"W:{lin.name}:{e}", device)
        w = torch.randn(lin.N, lin.K, generator=g, device=device, dtype=torch.float32) * wl.w_std
        q = quantize_rtn(w, wl.fmt)
        codes[e].copy_(q.codes)
        scales[e].copy_(q.scales)
        ws2.append(q.ws2)
    return Experts(wl.fmt, wl.E, lin.N, lin.K, codes, scales, ws2)


def gen_expert_latents(wl: MoEWorkload, lin: Linear, ex: Experts, device="cpu") -> torch.Tensor:
    """Latent effective scales [E, N, G] of every expert (gen_latent per expert, each
    with its own draw)."""
    out = torch.empty(ex.scales.shape, dtype=torch.float32, device=device)
    for e in range(ex.E):
        w = Weight(ex.fmt, ex.N, ex.K, ex.codes[e], ex.scales[e], ex.ws2[e])
        out[e].copy_(gen_latent(wl, dataclasses.replace(lin, name=f"{lin.name}:{e}"), w, device=device))
    return out


def gen_expert_adapters(wl: MoEWorkload, lin: Linear, ex: Experts, r: Optional[int] = None, alpha: float = 16.0,
                        device="cpu"):
    """Low-rank adapter factors of every expert (gen_adapter per expert, each with its
    own draw): B [E, N, r] and A [E, r, G] bf16 and the shared alpha/r."""
    r = wl.latent_rank if r is None else r
    G = ex.K // BLOCK[ex.fmt]
    B = torch.empty(ex.E, ex.N, r, dtype=torch.bfloat16, device=device)
    A = torch.empty(ex.E, r, G, dtype=torch.bfloat16, device=device)
    aor = alpha / r
    for e in range(ex.E):
        w = Weight(ex.fmt, ex.N, ex.K, ex.codes[e], ex.scales[e], ex.ws2[e])
        Be, Ae, aor = gen_adapter(wl, dataclasses.replace(lin, name=f"{lin.name}:{e}"), w, r=r, alpha=alpha,
                                  device=device)
        B[e].copy_(Be)
        A[e].copy_(Ae)
    return B, A, aor
