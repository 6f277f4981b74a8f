#!/usr/bin/env python
"""Benchmark of the Scale-QLoRA scale-only training step on a Llama-3-8B-shaped
NVFP4 decoder layer (q, k, v, o, gate, up, down; 16 x 2048 tokens).

One step = for every linear: grid projection of the latent scales (with STE
mask), forward, input gradient, masked block-reduced scale gradient, and the
merge of the latent into the artifact's scale plane: every row of the hot path.
Metric: fwd+dX+dScale TFLOP/s = 6*M*N*K summed over the linears / step time,
with its fraction of the measured GB300 dense-bf16 peak.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (launched by torch.distributed.run) every rank runs an independent
replica of the step (the method has no exchange on this path); rank 0 prints
the JSON line with the maximum time over ranks. `--impl reference` times the
float64 CPU oracle on a bounded sample of the same workload on the host cores.
"""
import argparse
import json
import os
import shutil
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "fwd+dX+dScale TFLOP/s per layer & fraction of GB300 bf16 tensor peak"
UNIT = "TFLOP/s"
KINDS = ("project", "fwd", "dx", "sgrad", "merge")
KINDS_LOWRANK = ("project", "fwd", "dx", "sgrad", "adapter_grad", "merge")
# GB300 datasheet figures (dense, no sparsity): the fractions against these sit beside
# the ones against the measured torch matmul / copy rates.
DATASHEET = {"bf16_tflops": 2250.0, "hbm_gbs": 7900.0}
# The tensor pipe's dense bf16 rate per GHz of SM clock: 4096 multiply-adds per SM per
# cycle (measured with tcgen05 MMAs on static operands) on 152 SMs.
TENSOR_TFLOPS_PER_GHZ = 2 * 4096 * 152 / 1e3
ADAPTER_RANK = 58  # the paper's Llama-3-8B scale rank (Sec. 5 recipe)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="c5")
    ap.add_argument("--linears", default=None,
                    help="comma-separated subset of the workload's linears (e.g. q_proj): the step runs only "
                         "these; for profiling one linear of the layer on a few GB of device memory")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-context", action="store_true",
                    help="skip the context legs (large-plane projection/merge ceiling, cuBLAS on pre-decoded weights)")
    ap.add_argument("--plane-only", action="store_true",
                    help="only the projection/merge ceiling on one 2^28-block plane (for profiling those kernels)")
    ap.add_argument("--moe", default=None,
                    help="time the grouped-expert step of an MoE workload instead (moe_qwen: Qwen3-30B-A3B-shaped "
                         "NVFP4 experts; moe_gptoss: gpt-oss-120B-shaped MXFP4 experts)")
    ap.add_argument("--lowrank", action="store_true",
                    help="the paper's exact training step: the latent comes from the low-rank adapter "
                         "(sq_project_lowrank) and the adapter gradients follow the scale gradient "
                         "(device-resident step only: no e2e or CPU-baseline legs)")
    return ap.parse_args()


def profiled_traffic(workload):
    """DRAM bytes per launch measured by ncu for each kernel kind (profiles/); a kind
    is left out when a source file of its kernel changed since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}_layer_step.json")
    if not os.path.exists(path):
        return {}
    with open(path) as f:
        prof = json.load(f)
    out = {}
    for kind, entry in prof.get("kernels", {}).items():
        srcs = [os.path.join(ROOT, "paper_2609_04526_gb300", "csrc", f) for f in entry.get("sources", [])]
        if not srcs or not all(os.path.isfile(f) for f in srcs):
            continue
        h = hashlib.sha256()
        for f in srcs:
            h.update(open(f, "rb").read())
        if h.hexdigest() == entry.get("sources_sha256"):
            out[kind] = entry
    return out


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16": float(p["bf16_tflops"]),
                "bf16_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


# --------------------------------------------------------------------- clocks

class _Nvml:
    """Read-only NVML queries through ctypes (libnvidia-ml ships with the driver):
    SM clock, its maximum, power draw and the active clock-event reasons."""
    SM = 1  # NVML_CLOCK_SM
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown"}

    def __init__(self, uuid):
        import ctypes
        self.c = ctypes
        self.lib = ctypes.CDLL("libnvidia-ml.so.1")
        if self.lib.nvmlInit_v2() != 0:
            raise RuntimeError("nvmlInit failed")
        self.dev = ctypes.c_void_p()
        if self.lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(self.dev)) != 0:
            raise RuntimeError("no NVML device for " + uuid)
        try:
            self.reasons_fn = self.lib.nvmlDeviceGetCurrentClocksEventReasons
        except AttributeError:
            self.reasons_fn = self.lib.nvmlDeviceGetCurrentClocksThrottleReasons
        v = ctypes.c_uint()
        self.max_mhz = float(v.value) if self.lib.nvmlDeviceGetMaxClockInfo(self.dev, self.SM, ctypes.byref(v)) == 0 \
            else None

    def sample(self):
        c = self.c
        mhz, mw, reasons = c.c_uint(), c.c_uint(), c.c_ulonglong()
        if self.lib.nvmlDeviceGetClockInfo(self.dev, self.SM, c.byref(mhz)) != 0:
            return None
        self.lib.nvmlDeviceGetPowerUsage(self.dev, c.byref(mw))
        self.reasons_fn(self.dev, c.byref(reasons))
        return float(mhz.value), mw.value / 1000.0, int(reasons.value)

    def close(self):
        self.lib.nvmlShutdown()


class ClockSampler:
    """SM clock, power and throttle reasons sampled every 25 ms during the timed
    region (NVML through ctypes; nvidia-smi at 50 ms where NVML is unavailable)."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")
    PERIOD_S = 0.025

    def __init__(self, device_index):
        self.proc = None
        self.thread = None
        self.samples = []
        self.source = None
        try:
            uuid = "GPU-" + str(torch.cuda.get_device_properties(device_index).uuid)
        except Exception:
            uuid = None
        if uuid:
            try:
                self.nvml = _Nvml(uuid)
                self._start_thread()
                self.source = "nvml 25 ms"
                return
            except Exception:
                self.nvml = None
        exe = shutil.which("nvidia-smi")
        if not exe:
            return
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        cmd = [exe] + (["-i", uuid] if uuid else []) + ["--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                                                         "-lms", "50"]
        self.fh = open(self.path, "w")
        self.proc = subprocess.Popen(cmd, stdout=self.fh, stderr=subprocess.DEVNULL)
        self.source = "nvidia-smi 50 ms"

    def _start_thread(self):
        import threading
        self.stop_evt = threading.Event()

        def loop():
            while not self.stop_evt.is_set():
                v = self.nvml.sample()
                if v is not None:
                    self.samples.append(v)
                self.stop_evt.wait(self.PERIOD_S)

        self.thread = threading.Thread(target=loop, daemon=True)
        self.thread.start()

    def _summary(self, sm, smax, watts, reasons):
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "sm_min_mhz": min(sm),
                "power_w_median": statistics.median(watts) if watts else None, "reasons": sorted(reasons),
                "samples": len(sm), "source": self.source}

    def stop(self):
        if self.thread is not None:
            self.stop_evt.set()
            self.thread.join(timeout=5)
            self.nvml.close()
            reasons = set()
            for _, _, r in self.samples:
                for bit, name in _Nvml.REASONS.items():
                    if r & bit:
                        reasons.add(name)
            return self._summary([m for m, _, _ in self.samples], self.nvml.max_mhz,
                                 [w for _, w, _ in self.samples], reasons)
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, smax, watts, reasons = [], [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 8:
                    continue
                try:
                    sm.append(float(parts[0]))
                    smax.append(float(parts[1]))
                    watts.append(float(parts[2]))
                except ValueError:
                    continue
                for name, v in zip(names, parts[4:8]):
                    if v.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        return self._summary(sm, max(smax) if smax else None, watts, reasons)


def per_ghz(kernels, clk):
    """Clock-normalised figures of each kernel kind: throughput per GHz of the median
    sampled SM clock, the step's share of that kind in millions of SM cycles, and for
    contractions the fraction of the tensor pipe's peak at that clock."""
    if not clk or not clk.get("sm_mhz"):
        return
    ghz = clk["sm_mhz"] / 1e3
    for k in kernels.values():
        k["per_ghz"] = k["achieved"] / ghz
        k["per_ghz_unit"] = k["unit"] + " per GHz"
        k["mcycles_per_step"] = k["ms_per_step"] * clk["sm_mhz"] / 1e3
        if k["unit"] == "TFLOP/s":
            k["frac_of_tensor_pipe_at_sampled_clock"] = k["per_ghz"] / TENSOR_TFLOPS_PER_GHZ


# --------------------------------------------------------------------- workload

class LayerState:
    """Device-resident inputs and outputs of one step of the workload."""

    def __init__(self, wl, device, lowrank=False):
        import paper_2609_04526_gb300 as pkg
        from paper_2609_04526_gb300 import synth
        self.wl = wl
        self.lowrank = lowrank
        self.lin = []
        self.acts = {name: synth.gen_act(wl, name, device=device) for name in synth.act_names(wl)
                     if any(l.x == name for l in wl.linears)}
        for lin in wl.linears:
            w = synth.gen_weight(wl, lin, device=device)
            L = synth.gen_latent(wl, lin, w, device=device)
            G = lin.K // wl.block
            st = dict(
                lin=lin, base_scales=w.scales, ws2=w.ws2, codes=w.codes, latent=L,
                codes0=w.codes.clone(),                     # the frozen code plane, to verify it is untouched
                art=w.scales.clone(),                       # artifact scale plane rewritten by the merge
                qbytes=torch.empty_like(w.scales),          # projected (on-grid) scale bytes used by the forward
                mask=torch.empty_like(w.scales),
                dY=synth.gen_dy(wl, lin, device=device),
                Y=torch.empty(wl.M, lin.N, dtype=torch.bfloat16, device=device),
                dX=torch.empty(wl.M, lin.K, dtype=torch.bfloat16, device=device),
                g=torch.empty(lin.N, G, dtype=torch.float32, device=device),
                nonfinite=torch.zeros(1, dtype=torch.int32, device=device),
                changed=torch.zeros(1, dtype=torch.int64, device=device),
            )
            st["qw"] = pkg.QuantWeight(wl.fmt, lin.N, lin.K, w.codes, st["qbytes"], w.ws2)
            if lowrank:
                st["B"], st["A"], st["aor"] = synth.gen_adapter(wl, lin, w, r=ADAPTER_RANK, device=device)
                st["dB"] = torch.empty(lin.N, ADAPTER_RANK, dtype=torch.float32, device=device)
                st["dA"] = torch.empty(ADAPTER_RANK, G, dtype=torch.float32, device=device)
            self.lin.append(st)

    def results(self):
        """(name, tensor) of the step's results read back by a user: scale gradients,
        merged scale planes and the NaN / changed-byte counters."""
        out = []
        for st in self.lin:
            out += [("g:" + st["lin"].name, st["g"]), ("art:" + st["lin"].name, st["art"]),
                    ("nf:" + st["lin"].name, st["nonfinite"]), ("ch:" + st["lin"].name, st["changed"])]
        return out


def input_set(S):
    """The step's inputs as a dict: activations by name, then dY and latent per linear."""
    return {"acts": dict(S.acts), "dY": [st["dY"] for st in S.lin], "L": [st["latent"] for st in S.lin]}


def clone_input_set(ins):
    return {"acts": {k: torch.empty_like(v) for k, v in ins["acts"].items()},
            "dY": [torch.empty_like(t) for t in ins["dY"]], "L": [torch.empty_like(t) for t in ins["L"]]}


def flat_inputs(ins):
    return list(ins["acts"].values()) + ins["dY"] + ins["L"]


def run_step(h, S, stream, timer=None, ins=None):
    """One step over every linear: grid projection (+ STE mask) of all linears' latents
    in one launch, then per linear the forward, input gradient and masked scale
    gradient, and the merge of all latents into the artifact scale planes in one
    launch. With the low-rank adapter (S.lowrank) each linear's latent is formed from
    its adapter inside its projection (and kept for the merge), and the adapter
    gradients follow the scale gradient. `timer(kind)` records an event after each
    kind's launch(es)."""
    fmt = S.wl.fmt
    ins = input_set(S) if ins is None else ins
    mark = timer if timer is not None else (lambda kind: None)
    mark(None)
    if S.lowrank:
        for i, st in enumerate(S.lin):
            h.sq_project_lowrank(fmt, st["base_scales"], st["B"], st["A"], st["ws2"], st["aor"],
                                 bytes_out=st["qbytes"], mask_out=st["mask"], nonfinite=st["nonfinite"],
                                 latent_out=ins["L"][i], stream=stream)
    else:
        h.sq_project_planes(fmt, [dict(latent=ins["L"][i], bytes=st["qbytes"], mask=st["mask"],
                                       nonfinite=st["nonfinite"], ws2=st["ws2"]) for i, st in enumerate(S.lin)],
                            stream=stream)
    mark("project")
    for i, st in enumerate(S.lin):
        X = ins["acts"][st["lin"].x]
        dY = ins["dY"][i]
        h.sq_fwd(st["qw"], X, st["Y"], stream=stream)
        mark("fwd")
        h.sq_bwd_dx(st["qw"], dY, st["dX"], stream=stream)
        mark("dx")
        h.sq_scale_grad(st["qw"], X, dY, mask=st["mask"], g=st["g"], stream=stream)
        mark("sgrad")
        if S.lowrank:
            h.sq_lowrank_grad(st["g"], st["B"], st["A"], st["aor"], dB=st["dB"], dA=st["dA"], stream=stream)
            mark("adapter_grad")
    h.sq_merge_planes(fmt, [dict(latent=ins["L"][i], bytes=st["art"], changed=st["changed"], ws2=st["ws2"])
                            for i, st in enumerate(S.lin)], stream=stream)
    mark("merge")


class StepTimer:
    """CUDA events between the kinds of a step's launches, on the launching stream."""

    def __init__(self, stream):
        self.stream = stream
        self.marks = []

    def __call__(self, kind):
        e = torch.cuda.Event(enable_timing=True)
        e.record(self.stream)
        self.marks.append((kind, e))

    def add_to(self, kind_ms, kind_launch):
        for (_, a), (kind, b) in zip(self.marks[:-1], self.marks[1:]):
            kind_ms[kind] += a.elapsed_time(b)
            kind_launch[kind] += 1


LAUNCHES_PER_STEP = 2    # the projection and the merge of all linears' planes
LAUNCHES_PER_LINEAR = 3  # fwd, dX, scale-grad (+1 where the scale gradient splits its tokens)
LAUNCHES_PER_LINEAR_LOWRANK = 8  # + the adapter projection and the adapter gradients' four kernels


def kernel_work(S):
    """Algorithmic FLOPs (contractions) and bytes (projection / merge) per kernel kind per step."""
    fl = {"fwd": 0, "dx": 0, "sgrad": 0}
    by = {"project": 0, "merge": 0}
    for st in S.lin:
        l = st["lin"]
        for k in fl:
            fl[k] += 2 * S.wl.M * l.N * l.K
        blocks = l.N * (l.K // S.wl.block)
        by["merge"] += blocks * (4 + 1 + 1)     # latent in, old byte in, new byte out
        if S.lowrank:
            r = ADAPTER_RANK
            factors = (l.N * r + r * (l.K // S.wl.block)) * 2   # B and A, bf16
            by["project"] += blocks * (1 + 1 + 1 + 4) + factors  # base byte in; byte, mask, latent out
            by["adapter_grad"] = by.get("adapter_grad", 0) + blocks * 4 + factors + factors * 2  # g in; dB, dA fp32 out
        else:
            by["project"] += blocks * (4 + 1 + 1)   # latent fp32 in, byte + mask byte out
    return fl, by


# --------------------------------------------------------------------- oracle sample

def snapshot_outputs(S, n_y, n_dx, n_rows, seed=0):
    """A seeded sample of the last timed step's outputs, read back right after the
    timed region (before any other leg reuses the buffers): Y and dX elements, full
    rows of the masked scale gradient, the projected bytes, STE mask and merged
    artifact planes, the NaN and changed-byte counters, and whether every code plane
    still equals the copy taken before the first step."""
    rng = np.random.default_rng(seed)
    out = {}
    for st in S.lin:
        l = st["lin"]
        M = S.wl.M
        ms, ns = rng.integers(0, M, n_y), rng.integers(0, l.N, n_y)
        ms2, ks = rng.integers(0, M, n_dx), rng.integers(0, l.K, n_dx)
        rows = rng.integers(0, l.N, n_rows)
        dev = st["Y"].device

        def ti(a):
            return torch.from_numpy(a).to(dev)

        out[l.name] = dict(
            ms=ms, ns=ns, ms2=ms2, ks=ks, rows=rows,
            Y=st["Y"][ti(ms), ti(ns)].double().cpu().numpy(), dX=st["dX"][ti(ms2), ti(ks)].double().cpu().numpy(),
            g=st["g"][ti(rows)].double().cpu().numpy(), qbytes=st["qbytes"].cpu().numpy(),
            mask=st["mask"].cpu().numpy(), art=st["art"].cpu().numpy(), nonfinite=int(st["nonfinite"].item()),
            changed=int(st["changed"].item()), codes_unchanged=bool(torch.equal(st["codes"], st["codes0"])))
    return out


def _err_over_bound(gpu, ref, rms):
    """Worst |gpu - ref| / (2e-2 |ref| + 1e-3 rms) over a sample (<= 1 passes), and the count above 1."""
    bound = 2e-2 * np.abs(ref) + 1e-3 * rms
    r = np.abs(gpu - ref) / np.maximum(bound, 1e-300)
    r = np.where(np.isnan(r), np.inf, r)
    return float(r.max()) if r.size else 0.0, int((r > 1).sum())


def oracle_sample(wl, host, linears, n_y, n_dx, n_rows, n_plane, seed=0):
    """Time the float64 oracle on a bounded sample of one step and extrapolate
    the full step's CPU time from each part's per-unit rate."""
    import oracle
    rng = np.random.default_rng(seed)
    t_full = 0.0
    t_spent = 0.0
    desc = []
    for lin in linears:
        d = host[lin.name]
        M, N, K = wl.M, lin.N, lin.K
        ms, ns, ks = rng.integers(0, M, n_y), rng.integers(0, N, n_y), rng.integers(0, K, n_dx)
        t0 = time.perf_counter()
        oracle.fwd_at(wl.fmt, d["codes"], d["scales"], d["ws2"], d["X"], ms, ns)
        t1 = time.perf_counter()
        oracle.dx_at(wl.fmt, d["codes"], d["scales"], d["ws2"], d["dY"], ms[:n_dx], ks)
        t2 = time.perf_counter()
        rows = rng.integers(0, N, n_rows)
        oracle.scale_grad(wl.fmt, d["codes"], d["X"], d["dY"], mask=d["mask"], rows=rows)
        t3 = time.perf_counter()
        Lp = d["latent"].reshape(-1)[:n_plane]
        oracle.project(wl.fmt, Lp, d["ws2"])
        t4 = time.perf_counter()
        oracle.merge(wl.fmt, Lp, d["scales"].reshape(-1)[:n_plane], d["ws2"], want_delta=False)
        t5 = time.perf_counter()
        blocks = N * (K // wl.block)
        t_full += ((t1 - t0) * (M * N / n_y) + (t2 - t1) * (M * K / n_dx) + (t3 - t2) * (N / n_rows)
                   + (t4 - t3 + t5 - t4) * (blocks / min(n_plane, blocks)))
        t_spent += t5 - t0
        desc.append(lin.name)
    return t_full, t_spent, (f"{n_y} Y and {n_dx} dX elements, {n_rows} full scale-gradient rows and "
                             f"{n_plane} latents through projection and merge, per linear ({', '.join(desc)}); "
                             "full-step time extrapolated from each part's measured per-element rate")


def oracle_check_sample(wl, host, linears, n_plane, snap):
    """The CPU baseline: time the float64 oracle on the sampled outputs of one step
    and extrapolate the full step's CPU time from each part's per-unit rate; the
    same sample checks the last timed step. The oracle projects each latent plane
    itself (untimed), and its own bytes and mask feed its contractions: the GPU's
    projected bytes, mask, merged plane and counters must equal the oracle's bit for
    bit, Y, dX and g rows agree within 2e-2 relative + 1e-3 x RMS, and the code
    planes must be unchanged."""
    import oracle
    t_full = 0.0
    t_spent = 0.0
    desc = []
    ver = {"ok": True, "linears": 0, "y_elements": 0, "dx_elements": 0, "g_rows": 0, "plane_bytes_bit_exact": 0,
           "code_planes_unchanged": True, "worst_err_over_bound": {"Y": 0.0, "dX": 0.0, "g": 0.0}, "failures": []}
    for lin in linears:
        d = host[lin.name]
        v = snap[lin.name]
        M, N, K = wl.M, lin.N, lin.K
        rb, rm, rnf = oracle.project(wl.fmt, d["latent"], d["ws2"])
        # the artifact plane before the last step held the previous step's merge, the same projection
        rs, _, rch = oracle.merge(wl.fmt, d["latent"], rb, d["ws2"], want_delta=False)
        planes = [("bytes", v["qbytes"], rb), ("mask", v["mask"], rm), ("merged", v["art"], rs)]
        for what, a, b in planes:
            if np.array_equal(a, b):
                ver["plane_bytes_bit_exact"] += a.size
            else:
                ver["failures"].append(f"{lin.name}: {what} plane differs in {int((a != b).sum())} bytes")
        if v["nonfinite"] != rnf or v["changed"] != rch:
            ver["failures"].append(f"{lin.name}: counters {v['nonfinite']}/{v['changed']} vs oracle {rnf}/{rch}")
        if not v["codes_unchanged"]:
            ver["code_planes_unchanged"] = False
            ver["failures"].append(f"{lin.name}: code plane changed")
        t0 = time.perf_counter()
        Yr = oracle.fwd_at(wl.fmt, d["codes"], rb, d["ws2"], d["X"], v["ms"], v["ns"])
        t1 = time.perf_counter()
        dXr = oracle.dx_at(wl.fmt, d["codes"], rb, d["ws2"], d["dY"], v["ms2"], v["ks"])
        t2 = time.perf_counter()
        gr = oracle.scale_grad(wl.fmt, d["codes"], d["X"], d["dY"], mask=rm, rows=v["rows"])
        t3 = time.perf_counter()
        Lp = d["latent"].reshape(-1)[:n_plane]
        oracle.project(wl.fmt, Lp, d["ws2"])
        t4 = time.perf_counter()
        oracle.merge(wl.fmt, Lp, d["scales"].reshape(-1)[:n_plane], d["ws2"], want_delta=False)
        t5 = time.perf_counter()
        for what, a, b in (("Y", v["Y"], Yr), ("dX", v["dX"], dXr), ("g", v["g"], gr)):
            worst, bad = _err_over_bound(a, b, float(np.sqrt(np.mean(b ** 2))))
            ver["worst_err_over_bound"][what] = max(ver["worst_err_over_bound"][what], worst)
            if bad:
                ver["failures"].append(f"{lin.name}: {bad} {what} values outside the tolerance")
        ver["linears"] += 1
        ver["y_elements"] += len(Yr)
        ver["dx_elements"] += len(dXr)
        ver["g_rows"] += len(v["rows"])
        blocks = N * (K // wl.block)
        n_y, n_dx, n_rows = len(v["ms"]), len(v["ks"]), len(v["rows"])
        t_full += ((t1 - t0) * (M * N / n_y) + (t2 - t1) * (M * K / n_dx) + (t3 - t2) * (N / n_rows)
                   + (t4 - t3 + t5 - t4) * (blocks / min(n_plane, blocks)))
        t_spent += t5 - t0
        desc.append(lin.name)
    ver["ok"] = not ver["failures"]
    n0 = snap[linears[0].name]
    return t_full, t_spent, (f"{len(n0['ms'])} Y and {len(n0['ks'])} dX elements, {len(n0['rows'])} full "
                             f"scale-gradient rows and {n_plane} latents through projection and merge, per linear "
                             f"({', '.join(desc)}); full-step time extrapolated from each part's measured per-element "
                             "rate"), ver


def host_copies(S, linears):
    out = {}
    for st in S.lin:
        l = st["lin"]
        if l not in linears:
            continue
        X = S.acts[l.x]
        out[l.name] = dict(
            codes=st["codes"].cpu().numpy(), scales=st["base_scales"].cpu().numpy(), ws2=st["ws2"],
            X=X.cpu().contiguous().view(torch.int16).numpy().view(np.uint16),
            dY=st["dY"].cpu().contiguous().view(torch.int16).numpy().view(np.uint16),
            mask=st["mask"].cpu().numpy(), latent=st["latent"].cpu().numpy())
    return out


# --------------------------------------------------------------------- arms

def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and not torch.distributed.is_initialized():
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        torch.distributed.init_process_group(backend=backend)
    return world, rank, local


def max_over_ranks(x, world):
    if world == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


PLANE_N, PLANE_G = 1 << 18, 1 << 10  # 2^28 scale blocks: far larger than the layer's planes and L2


def plane_ceiling(h, pk, stream, reps=10):
    """The plane kernels over one synthetic 2^28-block NVFP4 plane: at the layer's
    sizes these launches last a few microseconds, so this shows their HBM ceiling.
    Bytes per block: projection 4 (latent) + 1 (byte) + 1 (mask); merge 4 + 1 (old
    byte) + 1 (new byte); rollback 4 (delta) + 1 + 1; swap 1 (source) + 1 + 1;
    audit 1 + 1."""
    gen = torch.Generator(device="cuda").manual_seed(2028)
    ws2 = 1.0 / (6 * 448)
    L = torch.exp(torch.randn(PLANE_N, PLANE_G, device="cuda", generator=gen) * 2.0 - 3.0) * (448 * ws2 / 20)
    qb = torch.empty(PLANE_N, PLANE_G, dtype=torch.uint8, device="cuda")
    mask = torch.empty_like(qb)
    nonfinite = torch.zeros(1, dtype=torch.int32, device="cuda")
    art = torch.zeros_like(qb)
    changed = torch.zeros(1, dtype=torch.int64, device="cuda")
    blocks = PLANE_N * PLANE_G
    out = {"blocks": blocks, "shape": [PLANE_N, PLANE_G], "format": "nvfp4"}
    delta = torch.zeros(PLANE_N, PLANE_G, dtype=torch.float32, device="cuda")
    other = torch.empty_like(qb)
    count = torch.zeros(1, dtype=torch.int64, device="cuda")
    legs = (("project", 6, lambda: h.sq_project_scales(0, L, ws2, bytes_out=qb, mask_out=mask,
                                                      nonfinite=nonfinite, stream=stream)),
            ("merge", 6, lambda: h.sq_merge(0, L, ws2, art, changed=changed, stream=stream)),
            ("rollback", 6, lambda: h.sq_rollback(0, delta, ws2, art, changed=changed, stream=stream)),  # delta, old, new
            ("swap", 3, lambda: h.sq_swap_scales(qb, other, changed=changed, stream=stream)),           # src, old, new
            ("audit", 2, lambda: h.sq_count_diff(qb, art, count=count, stream=stream)))                # two planes
    for name, per_block, fn in legs:
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        gbs = per_block * blocks / (ms / 1e3) / 1e9
        out[name] = {"ms": ms, "bytes": per_block * blocks, "achieved": gbs, "unit": "GB/s",
                     "frac": gbs / pk["hbm_gbs"]}
    h.sq_sync(stream)
    del L, qb, mask, art, delta, other
    return out


E2M1_VALUES = (0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0, -0.0, -0.5, -1.0, -1.5, -2.0, -3.0, -4.0, -6.0)


def predecoded_weight(wl, st):
    """The decoded weight as a bf16 tensor (context leg only): codes through the E2M1
    table times the block scale (E4M3 byte x ws2, or 2^(byte-127))."""
    codes = st["codes"]
    nib = torch.stack((codes & 0xF, codes >> 4), dim=-1).reshape(codes.shape[0], -1).long()
    table = torch.tensor(E2M1_VALUES, dtype=torch.float32, device=codes.device)
    if wl.fmt == 0:
        s = st["base_scales"].view(torch.float8_e4m3fn).float() * st["ws2"]
    else:
        s = torch.exp2(st["base_scales"].float() - 127.0)
    return (table[nib] * s.repeat_interleave(wl.block, dim=1)).to(torch.bfloat16)


def adapter_leg(h, S, stream, reps=10):
    """The low-rank adapter kernels alone over the layer's linears (rank 58): the
    adapter projection (latent formed from B, A and projected, with mask and latent
    out) and the adapter gradients (dB, dA from the masked scale gradient). GB/s
    from their algorithmic bytes."""
    from paper_2609_04526_gb300 import synth
    wl = S.wl
    r = ADAPTER_RANK
    per = []
    by_proj = by_grad = 0
    for st in S.lin:
        l = st["lin"]
        G = l.K // wl.block
        w = synth.Weight(wl.fmt, l.N, l.K, st["codes"], st["base_scales"], st["ws2"])
        B, A, aor = synth.gen_adapter(wl, l, w, r=r, device="cuda")
        per.append(dict(st=st, B=B, A=A, aor=aor, L=torch.empty(l.N, G, dtype=torch.float32, device="cuda"),
                        q=torch.empty(l.N, G, dtype=torch.uint8, device="cuda"),
                        m=torch.empty(l.N, G, dtype=torch.uint8, device="cuda"),
                        dB=torch.empty(l.N, r, dtype=torch.float32, device="cuda"),
                        dA=torch.empty(r, G, dtype=torch.float32, device="cuda")))
        blocks, factors = l.N * G, (l.N * r + r * G) * 2
        by_proj += blocks * (1 + 1 + 1 + 4) + factors
        by_grad += blocks * 4 + factors + factors * 2

    def proj():
        for a in per:
            h.sq_project_lowrank(wl.fmt, a["st"]["base_scales"], a["B"], a["A"], a["st"]["ws2"], a["aor"],
                                 bytes_out=a["q"], mask_out=a["m"], latent_out=a["L"], stream=stream)

    def grad():
        for a in per:
            h.sq_lowrank_grad(a["st"]["g"], a["B"], a["A"], a["aor"], dB=a["dB"], dA=a["dA"], stream=stream)

    out = {"rank": r, "linears": len(per)}
    for name, fn, by in (("project_lowrank", proj, by_proj), ("adapter_grad", grad, by_grad)):
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        out[name] = {"us_per_layer": ms * 1e3, "bytes": by, "achieved": by / (ms / 1e3) / 1e9, "unit": "GB/s"}
    h.sq_sync(stream)
    return out


def variants_leg(h, S, pk, stream, reps=10):
    """The scale-family variant kernels on the layer's largest plane (gate_proj,
    14336 x 4096 NVFP4): the least-squares fit of a bf16 weight update (delta and both
    energies out), the group gradient at gd = 4 and the group-delta projection at gd = 4.
    Algorithmic bytes: fit 2 (dW) + 0.5 (codes) bytes per weight + 4 (delta) per block;
    group gradient 4 per block in; projection 1 (base) + 1 + 1 + 4 (byte, mask, latent) per block."""
    st = max(S.lin, key=lambda t: t["lin"].N * t["lin"].K)
    l = st["lin"]
    G = l.K // S.wl.block
    gen = torch.Generator(device="cuda").manual_seed(404)
    dW = (torch.randn(l.N, l.K, device="cuda", generator=gen) * 1e-4).to(torch.bfloat16)
    delta = torch.empty(l.N, G, device="cuda")
    cap, tot = torch.empty_like(delta), torch.empty_like(delta)
    gd = 4
    gdelta = torch.randn(l.N, gd, device="cuda", generator=gen) * st["ws2"] * 8
    gout = torch.empty(l.N, gd, device="cuda")
    qb = torch.empty(l.N, G, dtype=torch.uint8, device="cuda")
    mask, lat = torch.empty_like(qb), torch.empty_like(delta)
    blocks, weights = l.N * G, l.N * l.K
    legs = (("fit", 2.5 * weights + 4 * blocks,
             lambda: h.sq_fit_scale_delta(S.wl.fmt, st["codes"], dW, st["ws2"], want_energy=False, stream=stream)),
            ("group_grad", 4 * blocks + 4 * l.N * gd, lambda: h.sq_group_reduce(st["g"], gd, out=gout, stream=stream)),
            ("project_group_delta", 7 * blocks,
             lambda: h.sq_project_group_delta(S.wl.fmt, st["base_scales"], gdelta, st["ws2"], bytes_out=qb,
                                              mask_out=mask, latent_out=lat, stream=stream)))
    out = {"plane": [l.N, l.K], "linear": l.name, "gd": gd}
    # the full-precision multiplicative control on the same linear: W the bf16 decoded
    # weight, one coefficient per (row, block of 16); its three contractions, TFLOP/s
    Wbf = predecoded_weight(S.wl, st)
    dS = torch.randn(l.N, l.K // 16, device="cuda", generator=gen) * 0.05
    X = S.acts[l.x]
    Yc = torch.empty(S.wl.M, l.N, dtype=torch.bfloat16, device="cuda")
    dXc = torch.empty(S.wl.M, l.K, dtype=torch.bfloat16, device="cuda")
    gc = torch.empty(l.N, l.K // 16, device="cuda")
    flops = 2 * S.wl.M * l.N * l.K
    ctl = {"shape": [S.wl.M, l.N, l.K]}
    for name, fn in (("fwd", lambda: h.sq_control_fwd(Wbf, dS, X, Y=Yc, stream=stream)),
                     ("dx", lambda: h.sq_control_bwd_dx(Wbf, dS, st["dY"], dX=dXc, stream=stream)),
                     ("grad", lambda: h.sq_control_grad(Wbf, X, st["dY"], g=gc, stream=stream))):
        for _ in range(2):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        ctl[name] = {"ms": ms, "achieved": flops / (ms / 1e3) / 1e12, "unit": "TFLOP/s",
                     "frac": flops / (ms / 1e3) / 1e12 / pk["bf16_sustained"]}
    out["control"] = ctl
    del Wbf, Yc, dXc
    for name, by, fn in legs:
        for _ in range(3):
            fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        out[name] = {"us": ms * 1e3, "bytes": int(by), "achieved": by / (ms / 1e3) / 1e9, "unit": "GB/s",
                     "frac": by / (ms / 1e3) / 1e9 / pk["hbm_gbs"]}
    h.sq_sync(stream)
    return out


def cublas_context(S, stream, steps=5):
    """torch.matmul (cuBLAS, bf16 in and out, fp32 accumulation) on pre-decoded weights
    for the same three contractions per linear: context for the fused kernels, which
    decode on the fly and reduce dW to g without writing it."""
    wl = S.wl
    Ws = [predecoded_weight(wl, st) for st in S.lin]
    dWs = [torch.empty(st["lin"].N, st["lin"].K, dtype=torch.bfloat16, device="cuda") for st in S.lin]
    acts = S.acts

    def step():
        for st, W, dW in zip(S.lin, Ws, dWs):
            X = acts[st["lin"].x]
            torch.matmul(X, W.t(), out=st["Y"])
            torch.matmul(st["dY"], W, out=st["dX"])
            torch.matmul(st["dY"].t(), X, out=dW)

    for _ in range(2):
        step()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    del Ws, dWs
    return {"value": wl.flops() / (ms / 1e3) / 1e12, "unit": UNIT, "ms_per_step": ms,
            "what": "torch.matmul bf16 on pre-decoded weights (Y, dX and a materialised bf16 dW per linear); "
                    "context only, not the method"}


def run_ours(args):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build, synth
    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    build.build()
    wl = synth.WORKLOADS[args.workload]
    if args.linears:
        import dataclasses
        keep = args.linears.split(",")
        wl = dataclasses.replace(wl, linears=tuple(l for l in wl.linears if l.name in keep),
                                 title=f"{wl.title}, only {args.linears}")
        if not wl.linears:
            raise SystemExit(f"--linears {args.linears}: no such linear in {args.workload}")
    pk = peaks()
    h = pkg.Handle()
    stream = torch.cuda.current_stream()
    if args.plane_only:
        if rank == 0:
            print(json.dumps({"plane_ceiling": plane_ceiling(h, pk, stream)}), flush=True)
        return
    if args.lowrank:
        args.no_e2e = True
        args.no_cpu_baseline = True
    kinds = KINDS_LOWRANK if args.lowrank else KINDS
    S = LayerState(wl, "cuda", lowrank=args.lowrank)
    flops_step = wl.flops()

    for _ in range(args.warmup):
        run_step(h, S, stream)
    h.sq_sync(stream)

    # ---- device-resident timed region (inputs already in HBM; inputs > L2)
    nl = len(S.lin)
    timers = [StepTimer(stream) for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    t_start.record(stream)
    for k in range(args.steps):
        run_step(h, S, stream, timers[k])
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(world)
    h.sq_sync(stream)
    ms_total = max_over_ranks(t_start.elapsed_time(t_end), world)
    ms_step = ms_total / args.steps
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    n_threads = None
    if want_cpu:
        import oracle
        oracle.lib()
        n_threads = oracle.num_threads()
        snap = snapshot_outputs(S, n_y=1024, n_dx=1024, n_rows=6 * n_threads, seed=12345)

    kind_ms = {k: 0.0 for k in kinds}
    kind_launch = {k: 0 for k in kinds}
    for t in timers:
        t.add_to(kind_ms, kind_launch)
    fl, by = kernel_work(S)
    kernels = {}
    for kind in kinds:
        t = kind_ms[kind] / args.steps / 1e3  # s per step
        if kind in fl:
            ach = fl[kind] / t / 1e12
            kernels[kind] = {"ms_per_step": t * 1e3, "achieved": ach, "unit": "TFLOP/s",
                             "frac": ach / pk["bf16_sustained"]}
        else:
            ach = by[kind] / t / 1e9
            kernels[kind] = {"ms_per_step": t * 1e3, "achieved": ach, "unit": "GB/s", "frac": ach / pk["hbm_gbs"]}
    for kind, k in kernels.items():
        k["frac_vs_datasheet"] = k["achieved"] / (DATASHEET["bf16_tflops"] if k["unit"] == "TFLOP/s"
                                                  else DATASHEET["hbm_gbs"])
    per_ghz(kernels, clk)
    dom = max(("fwd", "dx", "sgrad"), key=lambda k: kind_ms[k])
    traffic = {} if (args.lowrank or args.linears) else profiled_traffic(wl.key)  # the profile is of the default step's kernels
    for kind in kinds:
        if kind in traffic:
            kernels[kind]["dram_bytes_per_launch"] = traffic[kind]["dram_bytes_per_launch"]
    value = flops_step * args.steps * world / (ms_total / 1e3) / 1e12

    # ---- end to end through the public API with host buffers: every step copies
    # its inputs from pinned host memory and reads its results back; the copies of
    # step k+1 run on a copy stream into a second input buffer set while step k
    # computes.
    e2e = None
    if not args.no_e2e:
        sets = [input_set(S), clone_input_set(input_set(S))]
        host_in = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in flat_inputs(sets[0])]
        for hst, dev in zip(host_in, flat_inputs(sets[0])):
            hst.copy_(dev)
        outs = [(t, torch.empty(t.shape, dtype=t.dtype, pin_memory=True)) for _, t in S.results()]
        h2d = sum(t.numel() * t.element_size() for t in host_in)
        d2h = sum(t.numel() * t.element_size() for t, _ in outs)
        copy_stream = torch.cuda.Stream()
        ready = [torch.cuda.Event(), torch.cuda.Event()]
        free = [torch.cuda.Event(), torch.cuda.Event()]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def issue_copy(k):
            b = k % 2
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(free[b] if k >= 2 else e0)
                for hst, dev in zip(host_in, flat_inputs(sets[b])):
                    dev.copy_(hst, non_blocking=True)
                ready[b].record(copy_stream)

        barrier(world)
        torch.cuda.synchronize()
        e0.record(stream)
        issue_copy(0)
        for k in range(args.steps):
            if k + 1 < args.steps:
                issue_copy(k + 1)
            stream.wait_event(ready[k % 2])
            run_step(h, S, stream, ins=sets[k % 2])
            free[k % 2].record(stream)
            for dev, hst in outs:
                hst.copy_(dev, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        h.sq_sync(stream)
        e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)
        e2e = {"value": flops_step * args.steps * world / (e2e_ms / 1e3) / 1e12, "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms / args.steps,
               "overlap": "inputs of step k+1 copied on a second stream while step k computes"}
        del sets, host_in

    # ---- context legs: the projection/merge HBM ceiling on a large plane, cuBLAS on pre-decoded weights
    context = {}
    if not args.no_context:
        context["plane_ceiling"] = plane_ceiling(h, pk, stream)
        context["adapter_kernels"] = adapter_leg(h, S, stream)
        context["variant_kernels"] = variants_leg(h, S, pk, stream)
        context["cublas_context"] = cublas_context(S, stream)

    # ---- CPU baseline: the oracle on a bounded sample (rank 0, N = 1 only)
    cpu = None
    verified = None
    if want_cpu:
        host = host_copies(S, list(wl.linears))
        t_full, t_spent, desc, verified = oracle_check_sample(wl, host, list(wl.linears), n_plane=1 << 18, snap=snap)
        cpu = {"value": flops_step / t_full / 1e12, "unit": UNIT, "cores": n_threads, "kind": "oracle",
               "sample": desc, "sample_seconds": round(t_spent, 2), "extrapolated_step_seconds": round(t_full, 1)}

    if rank == 0:
        k = kernels[dom]
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": f"{wl.key}: {wl.title}", "M": wl.M,
                       "linears": {l.name: [l.N, l.K] for l in wl.linears}, "format": "nvfp4" if wl.fmt == 0 else "mxfp4",
                       "l2": "inputs larger than L2 (activations + output gradients > 4 GB per step), no flush",
                       "parallelism": f"replicas x{world}", "flops_per_step": flops_step,
                       "step": (f"adapter step: latent from a rank-{ADAPTER_RANK} scale adapter, adapter gradients"
                                if args.lowrank else "latent projection")},
            "roofline": {"bound": "tensor", "kernel": dom, "achieved": k["achieved"],
                         "peak": pk["bf16_sustained"], "unit": "TFLOP/s", "frac": k["achieved"] / pk["bf16_sustained"],
                         "traffic": traffic.get(dom, {}).get("dram_bytes_per_launch"),
                         "algorithmic_bytes": traffic.get(dom, {}).get("algorithmic_bytes_per_launch"),
                         "traffic_note": "ncu dram bytes per launch, mean over the layer's 7 launches of this kernel "
                                         "(profiles/traffic_c5_layer_step.json); null if its sources changed since",
                         "peak_source": f"{pk['source']} bf16 sustained (torch.matmul 8192^3 held for 4 s)",
                         "frac_vs_datasheet": k["achieved"] / DATASHEET["bf16_tflops"],
                         "frac_of_tensor_pipe_at_sampled_clock": k.get("frac_of_tensor_pipe_at_sampled_clock"),
                         "tensor_pipe_peak_at_sampled_clock": (TENSOR_TFLOPS_PER_GHZ * clk["sm_mhz"] / 1e3
                                                               if clk and clk.get("sm_mhz") else None)},
            "fraction_of_peak": {"bf16_burst_measured_matmul": value / world / pk["bf16"],
                                 "bf16_sustained_measured_matmul": value / world / pk["bf16_sustained"],
                                 "bf16_datasheet_dense": value / world / DATASHEET["bf16_tflops"]},
            "per_ghz": ({"value": value / world / (clk["sm_mhz"] / 1e3), "unit": "TFLOP/s per GHz (median SM clock)"}
                        if clk and clk.get("sm_mhz") else None),
            "verified": verified,
            "kernels": kernels,
            "e2e": e2e, "cpu_baseline": cpu,
            "gpu_launches": (LAUNCHES_PER_STEP - (1 if args.lowrank else 0)
                             + (LAUNCHES_PER_LINEAR_LOWRANK if args.lowrank else LAUNCHES_PER_LINEAR) * nl
                             + sum(h.sq_scale_grad_workspace(st["qw"], S.wl.M)[0] > 1 for st in S.lin)) * args.steps,
            "clocks": clk,
        }
        line.update(context)
        print(json.dumps(line), flush=True)


# --------------------------------------------------------------------- MoE experts

class MoEState:
    """Device-resident inputs and outputs of one grouped-expert step: every expert
    linear (gate, up, down) of an MoE layer over the routed token rows."""

    def __init__(self, wl, device, lowrank=False):
        import paper_2609_04526_gb300 as pkg
        from paper_2609_04526_gb300 import synth
        self.wl = wl
        self.lowrank = lowrank
        self.counts = synth.gen_routing(wl)
        self.off = synth.offsets_of(self.counts)
        M = self.off[-1]
        self.acts = {name: synth.gen_act(wl, name, M=M, device=device) for name, _, _ in wl.acts
                     if any(l.x == name for l in wl.linears)}
        self.lin = []
        for lin in wl.linears:
            ex = synth.gen_experts(wl, lin, device=device)
            L = synth.gen_expert_latents(wl, lin, ex, device=device)
            st = dict(lin=lin, ex=ex, latent=L, art=ex.scales.clone(), qbytes=torch.empty_like(ex.scales),
                      mask=torch.empty_like(ex.scales), dY=synth.gen_dy(wl, lin, M=M, device=device),
                      Y=torch.empty(M, lin.N, dtype=torch.bfloat16, device=device),
                      dX=torch.empty(M, lin.K, dtype=torch.bfloat16, device=device),
                      g=torch.empty(ex.scales.shape, dtype=torch.float32, device=device),
                      nonfinite=torch.zeros(1, dtype=torch.int32, device=device),
                      changed=torch.zeros(1, dtype=torch.int64, device=device))
            # the forward and backward read the projected bytes; projection and merge read only ws2
            st["gw"] = pkg.GroupedWeight(wl.fmt, wl.E, lin.N, lin.K, ex.codes, st["qbytes"], ex.ws2)
            if lowrank:  # every expert's adapter over its frozen base plane (rank 54, the paper's MoE rank)
                st["gw_base"] = pkg.GroupedWeight(wl.fmt, wl.E, lin.N, lin.K, None, ex.scales, ex.ws2)
                st["B"], st["A"], st["aor"] = synth.gen_expert_adapters(wl, lin, ex, device=device)
                st["dB"] = torch.empty(st["B"].shape, dtype=torch.float32, device=device)
                st["dA"] = torch.empty(st["A"].shape, dtype=torch.float32, device=device)
            self.lin.append(st)

    def inputs(self):
        return {"acts": dict(self.acts), "dY": [st["dY"] for st in self.lin], "L": [st["latent"] for st in self.lin]}

    def results(self):
        out = []
        for st in self.lin:
            n = st["lin"].name
            out += [("g:" + n, st["g"]), ("art:" + n, st["art"]), ("nf:" + n, st["nonfinite"]),
                    ("ch:" + n, st["changed"])]
        return out


def run_moe_step(h, S, stream, events=None, ins=None):
    """One grouped-expert step per linear: projection of every expert's latent plane,
    forward, input gradient and masked scale gradient over all experts, merge."""
    ins = S.inputs() if ins is None else ins
    for i, st in enumerate(S.lin):
        X, dY, L = ins["acts"][st["lin"].x], ins["dY"][i], ins["L"][i]
        ev = events[i] if events is not None else None
        gw = st["gw"]
        if S.lowrank:
            project = lambda: h.sq_grouped_project_lowrank(st["gw_base"], st["B"], st["A"], st["aor"],
                                                           bytes_out=st["qbytes"], mask_out=st["mask"],
                                                           nonfinite=st["nonfinite"], latent_out=L, stream=stream)
        else:
            project = lambda: h.sq_grouped_project_scales(gw, L, bytes_out=st["qbytes"], mask_out=st["mask"],
                                                          nonfinite=st["nonfinite"], stream=stream)
        calls = [project,
                 lambda: h.sq_grouped_fwd(gw, S.off, X, Y=st["Y"], stream=stream),
                 lambda: h.sq_grouped_bwd_dx(gw, S.off, dY, dX=st["dX"], stream=stream),
                 lambda: h.sq_grouped_scale_grad(gw, S.off, X, dY, mask=st["mask"], g=st["g"], stream=stream)]
        if S.lowrank:
            calls.append(lambda: h.sq_grouped_lowrank_grad(st["g"], st["B"], st["A"], st["aor"], dB=st["dB"],
                                                           dA=st["dA"], stream=stream))
        calls.append(lambda: h.sq_grouped_merge(gw, L, st["art"], changed=st["changed"], stream=stream))
        for j, call in enumerate(calls):
            if ev:
                ev[j].record(stream)
            call()
        if ev:
            ev[len(calls)].record(stream)


def moe_context(h, S, stream, steps=3):
    """Context legs of the MoE step: (1) the same contractions as a loop of dense
    calls, one per expert (what a per-expert loop costs); (2) the dense kernels on
    one weight over all routed rows at once (the same FLOPs without ragged experts:
    the ceiling of the grouped launches)."""
    wl = S.wl
    off = S.off

    def per_expert():
        for st in S.lin:
            X = S.acts[st["lin"].x]
            for e in range(wl.E):
                a, b = off[e], off[e + 1]
                if b == a:
                    continue
                w = st["gw"].expert(e)
                if w.scales.data_ptr() % 16:
                    continue  # never for these workloads' planes (N * G is a multiple of 16)
                h.sq_fwd(w, X[a:b], Y=st["Y"][a:b], stream=stream)
                h.sq_bwd_dx(w, st["dY"][a:b], dX=st["dX"][a:b], stream=stream)
                h.sq_scale_grad(w, X[a:b], st["dY"][a:b], mask=st["mask"][e], g=st["g"][e], stream=stream)

    dense_w = [st["gw"].expert(0) for st in S.lin]

    def dense_all_rows():
        for st, w in zip(S.lin, dense_w):
            X = S.acts[st["lin"].x]
            h.sq_fwd(w, X, Y=st["Y"], stream=stream)
            h.sq_bwd_dx(w, st["dY"], dX=st["dX"], stream=stream)
            h.sq_scale_grad(w, X, st["dY"], mask=st["mask"][0], g=st["g"][0], stream=stream)

    out = {}
    for name, fn in (("per_expert_loop", per_expert), ("dense_same_rows", dense_all_rows)):
        fn()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / steps
        out[name] = {"value": wl.flops() / (ms / 1e3) / 1e12, "unit": UNIT, "ms_per_step": ms}
    out["per_expert_loop"]["what"] = ("fwd, dX and scale gradient as one dense call per expert and linear "
                                      f"({sum(1 for c in S.counts if c) * len(S.lin) * 3} launches per step)")
    out["dense_same_rows"]["what"] = ("the dense kernels on one expert's weight over all routed rows at once: the same "
                                      "FLOPs without per-expert raggedness (ceiling of the grouped launches)")
    h.sq_sync(stream)
    return out


def moe_oracle_sample(S, n_experts=2, n_y=128, n_dx=128, n_rows=None, n_plane=1 << 14, seed=0):
    """The float64 oracle on a bounded sample of the MoE step: a few experts of every
    linear through oracle_sample's per-element rates, scaled to the whole step by
    those experts' share of the step's FLOPs."""
    import oracle
    from paper_2609_04526_gb300 import synth
    wl = S.wl
    rng = np.random.default_rng(seed)
    nz = [e for e in range(wl.E) if S.counts[e]]
    experts = [int(e) for e in rng.choice(nz, min(n_experts, len(nz)), replace=False)]
    n_rows = oracle.num_threads() if n_rows is None else n_rows
    t_full = t_spent = 0.0
    flops_sampled = 0
    for st in S.lin:
        lin = st["lin"]
        X = S.acts[lin.x]
        for e in experts:
            a, b = S.off[e], S.off[e + 1]
            sub = synth.custom(f"{wl.key}:{lin.name}:{e}", wl.fmt, b - a, lin.N, lin.K, seed=0)
            sub_lin = sub.linears[0]
            host = {sub_lin.name: dict(
                codes=st["ex"].codes[e].cpu().numpy(), scales=st["ex"].scales[e].cpu().numpy(), ws2=st["ex"].ws2[e],
                X=X[a:b].cpu().contiguous().view(torch.int16).numpy().view(np.uint16),
                dY=st["dY"][a:b].cpu().contiguous().view(torch.int16).numpy().view(np.uint16),
                mask=st["mask"][e].cpu().numpy(), latent=st["latent"][e].cpu().numpy())}
            tf, ts, _ = oracle_sample(sub, host, [sub_lin], n_y=n_y, n_dx=n_dx, n_rows=n_rows, n_plane=n_plane,
                                      seed=seed + e)
            t_full += tf
            t_spent += ts
            flops_sampled += 6 * (b - a) * lin.N * lin.K
    t_step = t_full * wl.flops() / flops_sampled
    desc = (f"experts {experts} of every linear: {n_y} Y and {n_dx} dX elements, {n_rows} full scale-gradient rows "
            f"and {n_plane} latents through projection and merge per expert linear; the step's time extrapolated "
            "from per-element rates and those experts' share of the step's FLOPs")
    return t_step, t_spent, desc


def run_moe(args):
    import paper_2609_04526_gb300 as pkg
    from paper_2609_04526_gb300 import build, synth
    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    build.build()
    wl = synth.MOE_WORKLOADS[args.moe]
    if args.linears:
        import dataclasses
        keep = args.linears.split(",")
        wl = dataclasses.replace(wl, linears=tuple(l for l in wl.linears if l.name in keep),
                                 title=f"{wl.title}, only {args.linears}")
        if not wl.linears:
            raise SystemExit(f"--linears {args.linears}: no such linear in {args.moe}")
    pk = peaks()
    h = pkg.Handle()
    stream = torch.cuda.current_stream()
    if args.lowrank:
        args.no_e2e = True
        args.no_cpu_baseline = True
    S = MoEState(wl, "cuda", lowrank=args.lowrank)
    kinds = KINDS_LOWRANK if args.lowrank else KINDS
    nl = len(S.lin)
    for _ in range(args.warmup):
        run_moe_step(h, S, stream)
    h.sq_sync(stream)
    events = [[[torch.cuda.Event(enable_timing=True) for _ in range(len(kinds) + 1)] for _ in range(nl)]
              for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    t_start.record(stream)
    for k in range(args.steps):
        run_moe_step(h, S, stream, events[k])
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    barrier(world)
    h.sq_sync(stream)
    ms_total = max_over_ranks(t_start.elapsed_time(t_end), world)
    kind_ms = {k: 0.0 for k in kinds}
    for k in range(args.steps):
        for i in range(nl):
            ev = events[k][i]
            for j, kind in enumerate(kinds):
                kind_ms[kind] += ev[j].elapsed_time(ev[j + 1])
    M = S.off[-1]
    fl = {k: sum(2 * M * st["lin"].N * st["lin"].K for st in S.lin) for k in ("fwd", "dx", "sgrad")}
    blocks = sum(wl.E * st["lin"].N * (st["lin"].K // wl.block) for st in S.lin)
    by = {"project": blocks * 6, "merge": blocks * 6}
    if args.lowrank:  # as kernel_work: base byte in, byte + mask + latent out, the factors; g in, dB and dA out
        factors = sum(wl.E * (st["lin"].N + st["lin"].K // wl.block) * st["B"].shape[2] * 2 for st in S.lin)
        by["project"] = blocks * 7 + factors
        by["adapter_grad"] = blocks * 4 + factors * 3
    kernels = {}
    for kind in kinds:
        t = kind_ms[kind] / args.steps / 1e3
        if kind in fl:
            ach = fl[kind] / t / 1e12
            kernels[kind] = {"ms_per_step": t * 1e3, "achieved": ach, "unit": "TFLOP/s",
                             "frac": ach / pk["bf16_sustained"]}
        else:
            ach = by[kind] / t / 1e9
            kernels[kind] = {"ms_per_step": t * 1e3, "achieved": ach, "unit": "GB/s", "frac": ach / pk["hbm_gbs"]}
    for k in kernels.values():
        k["frac_vs_datasheet"] = k["achieved"] / (DATASHEET["bf16_tflops"] if k["unit"] == "TFLOP/s"
                                                  else DATASHEET["hbm_gbs"])
    per_ghz(kernels, clk)
    dom = max(("fwd", "dx", "sgrad"), key=lambda k: kind_ms[k])
    value = wl.flops() * args.steps * world / (ms_total / 1e3) / 1e12

    e2e = None
    if not args.no_e2e:
        sets = [S.inputs(), clone_input_set(S.inputs())]
        host_in = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in flat_inputs(sets[0])]
        for hst, dev in zip(host_in, flat_inputs(sets[0])):
            hst.copy_(dev)
        outs = [(t, torch.empty(t.shape, dtype=t.dtype, pin_memory=True)) for _, t in S.results()]
        # + per linear: three expert tables (descriptors, tile starts, rows, ws2) of the grouped
        # contractions and, for NVFP4, the experts' tensor scales for projection and merge
        tables = nl * (3 * (268 * wl.E + 4) + (8 * wl.E if wl.fmt == 0 else 0))
        h2d = sum(t.numel() * t.element_size() for t in host_in) + tables
        d2h = sum(t.numel() * t.element_size() for t, _ in outs)
        copy_stream = torch.cuda.Stream()
        ready = [torch.cuda.Event(), torch.cuda.Event()]
        free = [torch.cuda.Event(), torch.cuda.Event()]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def issue_copy(k):
            b = k % 2
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(free[b] if k >= 2 else e0)
                for hst, dev in zip(host_in, flat_inputs(sets[b])):
                    dev.copy_(hst, non_blocking=True)
                ready[b].record(copy_stream)

        barrier(world)
        torch.cuda.synchronize()
        e0.record(stream)
        issue_copy(0)
        for k in range(args.steps):
            if k + 1 < args.steps:
                issue_copy(k + 1)
            stream.wait_event(ready[k % 2])
            run_moe_step(h, S, stream, ins=sets[k % 2])
            free[k % 2].record(stream)
            for dev, hst in outs:
                hst.copy_(dev, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        h.sq_sync(stream)
        e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)
        e2e = {"value": wl.flops() * args.steps * world / (e2e_ms / 1e3) / 1e12, "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms / args.steps,
               "overlap": "inputs of step k+1 copied on a second stream while step k computes; the routing "
                          "offsets and expert tables go host to device with every grouped call"}
        del sets, host_in

    context = {} if args.no_context else moe_context(h, S, stream)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.lib()
        t_step, t_spent, desc = moe_oracle_sample(S)
        cpu = {"value": wl.flops() / t_step / 1e12, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
               "sample": desc, "sample_seconds": round(t_spent, 2), "extrapolated_step_seconds": round(t_step, 1)}
    if rank == 0:
        k = kernels[dom]
        c = np.asarray(S.counts)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_total / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": f"{wl.key}: {wl.title}", "experts": wl.E, "top_k": wl.top_k, "tokens": wl.T,
                       "routed_rows": int(M), "rows_per_expert": {"min": int(c.min()), "mean": float(c.mean()),
                                                                  "max": int(c.max()), "empty": int((c == 0).sum())},
                       "linears": {st["lin"].name: [st["lin"].N, st["lin"].K] for st in S.lin},
                       "format": "nvfp4" if wl.fmt == 0 else "mxfp4",
                       "l2": "inputs larger than L2 (routed activations + output gradients > 2 GB per step), no flush",
                       "parallelism": f"replicas x{world}", "flops_per_step": wl.flops(),
                       "step": ("grouped experts: rank-54 adapters of all experts, projection, fwd, dX, masked scale "
                                "gradient, adapter gradients, merge per linear" if args.lowrank else
                                "grouped experts: projection, fwd, dX, masked scale gradient, merge per linear")},
            "roofline": {"bound": "tensor", "kernel": dom, "achieved": k["achieved"], "peak": pk["bf16_sustained"],
                         "unit": "TFLOP/s", "frac": k["achieved"] / pk["bf16_sustained"], "traffic": None,
                         "peak_source": f"{pk['source']} bf16 sustained"},
            "fraction_of_peak": {"bf16_burst": value / world / pk["bf16"],
                                 "bf16_sustained": value / world / pk["bf16_sustained"]},
            "kernels": kernels, "e2e": e2e, "cpu_baseline": cpu,
            "gpu_launches": (LAUNCHES_PER_LINEAR_LOWRANK if args.lowrank else LAUNCHES_PER_LINEAR) * nl * args.steps,
            "clocks": clk,
        }
        line.update(context)
        print(json.dumps(line), flush=True)


def run_reference(args):
    """The float64 CPU oracle, as it stands, on bounded samples of the same workload."""
    world, rank, local = dist_setup(args)
    if rank != 0:
        return
    import oracle
    from paper_2609_04526_gb300 import synth
    oracle.lib()
    wl = synth.WORKLOADS[args.workload]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    if dev == "cuda":
        torch.cuda.set_device(local)
    host = {}
    acts = {}
    for lin in wl.linears:
        w = synth.gen_weight(wl, lin, device=dev)
        if lin.x not in acts:
            acts[lin.x] = synth.gen_act(wl, lin.x, device=dev).cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
        L = synth.gen_latent(wl, lin, w, device=dev)
        G = lin.K // wl.block
        host[lin.name] = dict(codes=w.codes.cpu().numpy(), scales=w.scales.cpu().numpy(), ws2=w.ws2, X=acts[lin.x],
                              dY=synth.gen_dy(wl, lin, device=dev).cpu().contiguous().view(torch.int16).numpy().view(np.uint16),
                              mask=np.ones((lin.N, G), dtype=np.uint8), latent=L.cpu().numpy())
        del w, L
    lins = list(wl.linears)
    per_step = []
    for k in range(args.warmup + args.steps):
        lin = lins[k % len(lins)]
        t_full, t_spent, desc = oracle_sample(wl, host, [lin], n_y=64, n_dx=64, n_rows=oracle.num_threads(),
                                              n_plane=1 << 15, seed=k)
        # scale this linear's extrapolated time to the whole layer by its FLOP share
        share = 6 * wl.M * lin.N * lin.K / wl.flops()
        if k >= args.warmup:
            per_step.append((t_full / share, t_spent))
    t_layer = statistics.median(t for t, _ in per_step)
    value = wl.flops() / t_layer / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(s for _, s in per_step), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{wl.key}: {wl.title}", "M": wl.M, "format": "nvfp4" if wl.fmt == 0 else "mxfp4",
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": "each step: one linear (cycling through the 7), 64 Y and 64 dX elements, one full "
                                   "scale-gradient row per host thread, 32768 latents through projection and merge; "
                                   "full-layer time extrapolated from per-element rates and the linear's FLOP share "
                                   "(median over steps)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.moe:
        run_moe(args)
    else:
        run_ours(args)
    if torch.distributed.is_available() and torch.distributed.is_initialized():
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
