"""Benchmark of the policy-masked MoE layer forward on GB300.

python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

A step is one full layer forward (resolve, masked router + top-k, dispatch,
grouped gate/up GEMM + SwiGLU, grouped down GEMM, combine) over one batch of
the named workload (default: the Qwen3-30B-A3B-shaped prefill layer, 4096
tokens, mixed ALLOW/DENY requests).  Prints one JSON line on rank 0.

Multi-GPU: independent replicas (the layer is token-parallel with no
exchange step); each rank runs the same workload on its own GPU, and value =
tokens processed by all ranks / max over ranks of the timed duration.
"""
from __future__ import annotations

import argparse
import json
import os
import shutil
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_06690_gb300 import inputs as inp  # noqa: E402
from paper_2608_06690_gb300.configs import CONFIGS  # noqa: E402

METRIC = "MoE-layer tokens/s (mixed allow/deny)"
L2_FLUSH_BYTES = 512 << 20   # > 129 MB L2
# After each L2 flush the GPU also spins this many cycles (~0.1 ms) before
# the timed interval opens, so the host has always enqueued the timed work
# by the time the GPU reaches it: no host gap inside a measured interval,
# also for the first interval after a synchronisation.
GPU_LEAD_CYCLES = 200_000


def flush_l2(flush):
    flush.zero_()
    torch.cuda._sleep(GPU_LEAD_CYCLES)

# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of the
# grouped GEMM launches (the persistent gate/up + down pair, and each GEMM
# launched alone), from ncu captures of the current kernels on the named
# workload; None where no capture of the current kernels exists.
# DRAM read + write bytes per launch of the dominant kernel (the persistent
# expert GEMM pair), from one ncu capture of the current kernel per workload:
# profiles/expert_gemm_tc_qwen3_prefill.md and ..._qwen3_decode.md.
NCU_TRAFFIC = {"qwen3_prefill": {"experts": 1.7942e9}, "qwen3_decode": {"experts": 1.3541e9}}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, device) -> float:
    """Maximum of a per-rank float over all ranks (identity without a process
    group); `device` is where the reduction tensor lives (cuda for NCCL, cpu
    for gloo)."""
    t = torch.tensor([x], dtype=torch.float64, device=device)
    if torch.distributed.is_available() and torch.distributed.is_initialized():
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, n_ranks: int, slowest_s: float) -> float:
    """Units processed by all ranks divided by the slowest rank's time."""
    return n_ranks * units_per_rank / slowest_s


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p.get("bf16_tflops_sustained", p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples, taken every 50 ms from
    before the warm-up until after the end-to-end leg; each sample is stamped
    on arrival so the ones inside the timed region can be counted."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self._first = threading.Event()

    def _read(self):
        for l in self.proc.stdout:
            if l.strip():
                self.lines.append((time.perf_counter(), l))
                self._first.set()

    def __enter__(self):
        cmd = ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "50"]
        if shutil.which("stdbuf"):
            cmd = ["stdbuf", "-oL"] + cmd   # one line per sample, as it is taken
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return self
        self._thread = threading.Thread(target=self._read, daemon=True)
        self._thread.start()
        self._first.wait(3.0)          # the sampler is running before the GPU work starts
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.proc.wait()
            self._thread.join(timeout=5)

    def summary(self, window=None):
        sm, mx, reasons, inside = [], None, set(), 0
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for t, l in list(self.lines):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            if window is not None and window[0] <= t <= window[1]:
                inside += 1
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        out = {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
               "samples": len(sm)}
        if window is not None:
            out["samples_in_timed_region"] = inside
        return out


class NvmlClockSampler:
    """SM clock, power and clock-event (throttle) reasons read through NVML
    (the driver's libnvidia-ml, via ctypes) every `period_s` in a background
    thread, so that even a timed region of a few milliseconds holds samples.
    Reads settings only; changes none.  Falls back to nothing (samples = 0)
    when NVML cannot be loaded; ClockSampler (nvidia-smi) runs beside it."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown"}

    def __init__(self, device_index: int, period_s: float = 0.002):
        import ctypes
        self.samples = []       # (t, sm_mhz, power_w, reasons)
        self.max_mhz = None
        self.period = period_s
        self._stop = threading.Event()
        self._thread = None
        self._h = None
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            props = torch.cuda.get_device_properties(device_index)
            bus = getattr(props, "pci_bus_id", None)
            ok = False
            if bus is not None:
                busid = f"{getattr(props, 'pci_domain_id', 0):08x}:{bus:02x}:{getattr(props, 'pci_device_id', 0):02x}.0"
                ok = lib.nvmlDeviceGetHandleByPciBusId_v2(busid.encode(), ctypes.byref(h)) == 0
            if not ok and lib.nvmlDeviceGetHandleByIndex_v2(device_index, ctypes.byref(h)) != 0:
                return
            self._lib, self._h, self._ct = lib, h, ctypes
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:   # 1 = NVML_CLOCK_SM
                self.max_mhz = float(mx.value)
            self._reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
        except Exception:
            self._h = None

    def _poll(self):
        ct, lib, h = self._ct, self._lib, self._h
        mhz, mw, rs = ct.c_uint(), ct.c_uint(), ct.c_ulonglong()
        while not self._stop.is_set():
            t = time.perf_counter()
            a = lib.nvmlDeviceGetClockInfo(h, 1, ct.byref(mhz))
            b = lib.nvmlDeviceGetPowerUsage(h, ct.byref(mw))
            c = self._reasons_fn(h, ct.byref(rs))
            if a == 0:
                self.samples.append((t, float(mhz.value), mw.value / 1e3 if b == 0 else None,
                                     int(rs.value) if c == 0 else 0))
            self._stop.wait(self.period)

    def __enter__(self):
        if self._h is not None:
            self._thread = threading.Thread(target=self._poll, daemon=True)
            self._thread.start()
        return self

    def __exit__(self, *a):
        self._stop.set()
        if self._thread is not None:
            self._thread.join(timeout=5)

    def summary(self, window):
        """Median SM clock and the reasons seen inside [t0, t1] (perf_counter)."""
        inside = [x for x in self.samples if window[0] <= x[0] <= window[1]]
        reasons = sorted({n for x in inside for bit, n in self.REASONS.items() if x[3] & bit})
        return {"sm_mhz": statistics.median([x[1] for x in inside]) if inside else None,
                "sm_max_mhz": self.max_mhz, "reasons": reasons, "samples_in_timed_region": len(inside),
                "power_w_max": max((x[2] for x in inside if x[2] is not None), default=None),
                "source": "NVML every %.0f ms" % (self.period * 1e3)}


def build_workload(cfg, device, seed_offset=0):
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed + seed_offset, device=device, skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed + seed_offset, device=device, skew=cfg.skew)
    pol = cfg.policy(s.T).to(device)
    return w, h, pol


def algorithmic_work(s, counts: np.ndarray):
    """FLOPs of the two grouped GEMMs and the least DRAM bytes of each stage,
    for one forward with the given per-expert row counts.  The gate/up tiles
    gather their rows from the hidden states (read once from DRAM; the other
    k - 1 reads of a row hit L2)."""
    R = s.T * s.k
    f_gateup = 2.0 * R * s.H * 2 * s.I + 2.0 * s.T * s.H * 2 * s.E_sh * s.I
    f_down = 2.0 * R * s.I * s.H + 2.0 * s.T * s.E_sh * s.I * s.H
    touched = int((counts > 0).sum())
    expert_w = 3 * s.I * s.H * 2
    gemm_weight_bytes = touched * expert_w + s.E_sh * expert_w
    w_gu = (touched + s.E_sh) * 2 * s.I * s.H * 2
    w_dn = (touched + s.E_sh) * s.I * s.H * 2
    act = R * s.I * 2 + s.T * s.E_sh * s.I * 2
    yb = R * s.H * 2 + (s.T * s.H * 2 if s.E_sh else 0)
    b_gateup = w_gu + s.T * s.H * 2 + act + R * 4
    b_down = w_dn + act + yb + R * 4
    b_combine = yb + s.T * s.H * 2 + R * 4
    b_route = s.T * s.H * 2 + (s.E_pub + s.E_priv) * s.H * 2 + s.T * s.k * 8 + s.T
    # the dispatch order: route log and tickets in, slot maps out
    b_permute = R * 12 + R * 12
    # the least DRAM traffic of a whole forward: the touched experts' weights
    # (and the shared experts'), both routers, hidden in and out, the route log
    b_layer_min = gemm_weight_bytes + (s.E_pub + s.E_priv) * s.H * 2 + 2 * s.T * s.H * 2 + s.T * s.k * 8 + s.T
    return dict(flops_gateup=f_gateup, flops_down=f_down, bytes_gateup=b_gateup, bytes_down=b_down,
                bytes_layer_min=b_layer_min,
                flops_experts=f_gateup + f_down, bytes_experts=b_gateup + b_down,
                bytes_route=b_route, bytes_permute=b_permute, bytes_combine=b_combine,
                touched_experts=touched, gemm_weight_bytes=gemm_weight_bytes)


def backward_flops(s, counts: np.ndarray, allow_tokens: int) -> float:
    """Algorithmic FLOPs of the private-branch backward: per private row,
    dL/da = W_down^T dout, the recomputed gate and up projections, and the
    three weight gradients (2 H I each: 12 H I); the router weight gradient
    over every token (2 T E_priv H), plus the private logits the pool softmax
    recomputes (2 E_priv H per ALLOW token)."""
    rows = float(counts[s.E_pub:].sum())
    f = 12.0 * rows * s.H * s.I + 2.0 * s.T * s.E_priv * s.H
    if not s.renormalize:
        f += 2.0 * allow_tokens * s.E_priv * s.H
    return f


def backward_input_flops(s, counts: np.ndarray, allow_tokens: int) -> float:
    """Algorithmic FLOPs of the input gradient: per routed row and per token
    of each shared expert, Z = W_down^T dout, the recomputed gate and up
    projections and dA = W_gate^T dG + W_up^T dU (10 H I); the router term
    W_router^T dz over the token's k picks (renormalised) or its whole pool,
    whose logits the pool softmax also recomputes."""
    rows = float(counts.sum()) + float(s.T * s.E_sh)
    f = 10.0 * rows * s.H * s.I
    if s.renormalize:
        f += 2.0 * s.T * s.k * s.H
    else:
        pool = allow_tokens * s.E_priv + (s.T - allow_tokens) * s.E_pub
        f += 4.0 * pool * s.H
    return f


def backward_min_bytes(s, counts: np.ndarray, allow_tokens: int, which: str) -> float:
    """Lower bound of a backward pass's DRAM bytes: every input read once and
    every output written once (the weights of the experts with rows, the
    hidden and dout rows of the tokens that reach them, the routers, and the
    FP32 outputs); intermediates and the recompute are not counted."""
    per_expert = 3.0 * s.I * s.H * 2
    if which == "private":
        touched = float((counts[s.E_pub:] > 0).sum())
        return (touched * per_expert + 2.0 * allow_tokens * s.H * 2 + s.E_priv * s.H * 2
                + 3.0 * s.E_priv * s.I * s.H * 4 + s.E_priv * s.H * 4)
    touched = float((counts > 0).sum()) + s.E_sh
    return touched * per_expert + 2.0 * s.T * s.H * 2 + s.E * s.H * 2 + s.T * s.H * 4


def cpu_baseline(cfg, w, h, pol, budget_s=12.0, max_tokens=4096):
    """The CPU oracle, as it stands, on a bounded sample of the workload's
    tokens (the first n tokens of each request, spread evenly)."""
    import oracle
    s = cfg.shape
    wc = {k: (None if v is None else v.cpu()) for k, v in w.items()}
    L = oracle.Layer(s, dict(wc, hidden=h.cpu()), pol.cpu().numpy())
    cores = len(os.sched_getaffinity(0))
    per_req = s.T // cfg.n_requests

    def sample(n):
        take = max(1, n // cfg.n_requests)
        toks = [r * per_req + i for r in range(cfg.n_requests) for i in range(min(take, per_req))]
        return np.array(toks[:max(n, 1)], dtype=np.int32)

    n = min(32, s.T)
    t0 = time.perf_counter()
    oracle.forward(L, tokens=sample(n), nthreads=cores)
    dt = time.perf_counter() - t0
    n2 = int(min(max_tokens, s.T, max(n, n * budget_s / max(dt, 1e-3))))
    toks = sample(n2)
    t0 = time.perf_counter()
    oracle.forward(L, tokens=toks, nthreads=cores)
    dt = time.perf_counter() - t0
    return {"value": len(toks) / dt, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{len(toks)} of {s.T} tokens of {cfg.name} (spread over its {cfg.n_requests} requests), "
                      f"full layer forward in fp64, OpenMP over tokens, {dt:.1f} s"}


def run_reference(args):
    """Reference arm: the CPU oracle, timed as it stands on the host cores,
    each step a bounded sample of the workload."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    import oracle
    cfg = CONFIGS[args.config]
    s = cfg.shape
    w, h, pol = build_workload(cfg, "cpu")
    L = oracle.Layer(s, dict(w, hidden=h), pol.numpy())
    cores = len(os.sched_getaffinity(0))
    per_req = s.T // cfg.n_requests
    n_tok = max(1, min(s.T, args.ref_tokens))
    take = max(1, n_tok // cfg.n_requests)
    toks = np.array([r * per_req + i for r in range(cfg.n_requests) for i in range(min(take, per_req))][:n_tok],
                    dtype=np.int32)
    for _ in range(args.warmup):
        oracle.forward(L, tokens=toks[:max(1, len(toks) // 8)], nthreads=cores)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.forward(L, tokens=toks, nthreads=cores)
    dt = time.perf_counter() - t0
    value = len(toks) * args.steps / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": cfg.name, "tokens_per_step": len(toks), "layer_tokens": s.T},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{len(toks)} of {s.T} tokens of {cfg.name} per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def roofline_of(work, stage_avg, pipeline, hbm, tf_burst, peak_src):
    """The dominant stage against the roofline its arithmetic intensity
    selects: tensor above the ridge point (peak FLOP/s / peak B/s), HBM
    below it; both fractions are given for the GEMMs."""
    dominant = max(pipeline, key=stage_avg.get)
    sec = stage_avg[dominant] / 1e3
    if dominant in ("experts", "gateup", "down"):
        tflops = work[f"flops_{dominant}"] / sec / 1e12
        gbs = work[f"bytes_{dominant}"] / sec / 1e9
        intensity = work[f"flops_{dominant}"] / work[f"bytes_{dominant}"]
        ridge = tf_burst * 1e12 / (hbm * 1e9)
        if intensity >= ridge:
            roof = {"kernel": dominant, "bound": "tensor", "achieved": tflops, "peak": tf_burst, "unit": "TFLOP/s",
                    "frac": tflops / tf_burst, "peak_source": f"{peak_src} bf16 burst"}
        else:
            roof = {"kernel": dominant, "bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s",
                    "frac": gbs / hbm, "peak_source": f"{peak_src} HBM copy"}
        roof.update({"flop_per_byte": intensity, "ridge_flop_per_byte": ridge, "tflops": tflops,
                     "tensor_frac": tflops / tf_burst, "hbm_gbs": gbs, "hbm_frac": gbs / hbm})
    else:
        achieved = work[f"bytes_{dominant}"] / sec / 1e9
        roof = {"kernel": dominant, "bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "peak_source": f"{peak_src} HBM copy"}
    return dominant, roof


def measure_forward(pmpe, cfg, w, h, pol, dev, args, ws_n, barrier, nvml, flush):
    """One workload's forward: K device-timed steps (L2 flushed before each),
    the per-stage breakdown, the audit of one forward, and the end-to-end leg
    through the public API with host buffers.  Returns the report and the
    per-expert row counts."""
    s = cfg.shape
    stream = torch.cuda.current_stream(dev)
    layer = pmpe.MoeLayer(s, w, device=dev)
    out = torch.empty_like(h)
    audit = torch.zeros(pmpe.audit_words(s.T, s.E), dtype=torch.int32, device=dev)

    def step():
        layer.forward(h, pol, out=out)

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize(dev)

    # ---- timed region: K steps, L2 flushed before each, CUDA events per step
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize(dev)
    t_wall0 = time.perf_counter()
    for e0, e1 in evs:
        flush_l2(flush)
        e0.record(stream)
        step()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    t_wall = time.perf_counter() - t_wall0
    barrier()
    step_ms = [e0.elapsed_time(e1) for e0, e1 in evs]
    total_ms = max_over_ranks(sum(step_ms), dev)
    value = whole_job_rate(s.T * args.steps, ws_n, total_ms / 1e3)
    clocks = nvml.summary((t_wall0, t_wall0 + t_wall))

    # ---- per-stage breakdown: each stage after its own L2 flush, so the GPU
    # is still busy flushing while the host enqueues the stage (no host gap
    # inside the measured interval); stages run in pipeline order on the
    # workspace the previous stage filled.  "experts" is the persistent
    # gate/up + down launch the forward runs; the two GEMMs launched one at a
    # time are reported as diagnostics.
    stages = [("route", pmpe.STAGE_ROUTE), ("permute", pmpe.STAGE_PERMUTE),
              ("experts", pmpe.STAGE_GATEUP | pmpe.STAGE_DOWN), ("combine", pmpe.STAGE_COMBINE),
              ("gateup", pmpe.STAGE_GATEUP), ("down", pmpe.STAGE_DOWN)]
    pipeline = ("route", "permute", "experts", "combine")
    stage_ms = {n: [] for n, _ in stages}
    for _ in range(args.steps):
        evs_s = []
        for n, bit in stages:
            flush_l2(flush)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            layer.forward(h, pol, out=out, stages=bit)
            b.record(stream)
            evs_s.append((n, a, b))
        torch.cuda.synchronize(dev)
        for n, a, b in evs_s:
            stage_ms[n].append(a.elapsed_time(b))
    stage_avg = {n: float(np.mean(v)) for n, v in stage_ms.items()}

    # ---- audit of one forward (exactness of the counters is a test; here: sanity + expert loads)
    pmpe.audit_reset(audit, s.T, s.E)
    layer.forward(h, pol, out=out, audit=audit)
    a = pmpe.audit_read(audit, s.T, s.E)
    counts = a["route_count"]
    work = algorithmic_work(s, counts)

    # ---- end to end through the public API with host buffers, pipelined as a
    # serving loop would run it: step i+1's inputs are copied in (copy-in
    # stream) while step i computes, and step i's result is copied out
    # (copy-out stream) while step i+1 computes; two device buffer sets.  Every
    # step's host->device and device->host copies lie inside the timed window.
    # No L2 flush here: every step streams the layer's weights (far larger
    # than L2) through it.
    h_host = h.cpu().pin_memory()
    pol_host = pol.cpu().pin_memory()
    out_host = [torch.empty(h.shape, dtype=h.dtype).pin_memory() for _ in range(2)]
    h_dev = [torch.empty_like(h) for _ in range(2)]
    pol_dev = [torch.empty_like(pol) for _ in range(2)]
    out_dev = [torch.empty_like(h) for _ in range(2)]
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    n_e2e = max(args.warmup, 3) + args.steps
    ev_in = [torch.cuda.Event() for _ in range(n_e2e)]
    ev_cmp = [torch.cuda.Event() for _ in range(n_e2e)]
    ev_out = [torch.cuda.Event() for _ in range(n_e2e)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    barrier()
    for i in range(n_e2e):
        bsel = i & 1
        if i == max(args.warmup, 3):
            torch.cuda.synchronize(dev)
            t_start.record(s_in)
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev_cmp[i - 2])   # step i-2 has consumed this input buffer
            h_dev[bsel].copy_(h_host, non_blocking=True)
            pol_dev[bsel].copy_(pol_host, non_blocking=True)
            ev_in[i].record(s_in)
        stream.wait_event(ev_in[i])
        if i >= 2:
            stream.wait_event(ev_out[i - 2])     # step i-2's result has been read out of this buffer
        layer.forward(h_dev[bsel], pol_dev[bsel], out=out_dev[bsel], stream=stream)
        ev_cmp[i].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_cmp[i])
            out_host[bsel].copy_(out_dev[bsel], non_blocking=True)
            ev_out[i].record(s_out)
    t_end.record(s_out)
    torch.cuda.synchronize(dev)
    barrier()
    e2e_ms = max_over_ranks(t_start.elapsed_time(t_end), dev)
    e2e_value = whole_job_rate(s.T * args.steps, ws_n, e2e_ms / 1e3)
    assert torch.equal(out_host[(n_e2e - 1) & 1].view(torch.int16), out.cpu().view(torch.int16)), \
        "the pipelined end-to-end result differs from the device-resident forward"

    hbm, tf_burst, tf_sus, peak_src = _peaks()
    dominant, roof = roofline_of(work, stage_avg, pipeline, hbm, tf_burst, peak_src)
    roof["traffic"] = args.traffic if (args.traffic is not None and cfg.name == args.config) \
        else NCU_TRAFFIC.get(cfg.name, {}).get(dominant)
    stage_report = {}
    for n, ms in stage_avg.items():
        d = {"ms": ms}
        if n in ("experts", "gateup", "down"):
            d["tflops"] = work[f"flops_{n}"] / (ms / 1e3) / 1e12
        d["gbs"] = work[f"bytes_{n}"] / (ms / 1e3) / 1e9
        d["hbm_frac"] = d["gbs"] / hbm
        stage_report[n] = d
    ms_step = total_ms / args.steps
    layer_bytes = work["bytes_layer_min"]
    rep = {
        "value": value, "unit": "tokens/s", "ms_per_step": ms_step, "steps": args.steps,
        "roofline": roof, "stages": stage_report,
        # the whole layer against HBM: the least DRAM traffic a forward needs
        # (the touched experts' weights, the routers, hidden in and out) over
        # the measured step time -- the decode-step figure of merit
        "layer_hbm": {"min_bytes": layer_bytes, "gbs": layer_bytes / (ms_step / 1e3) / 1e9,
                      "frac": layer_bytes / (ms_step / 1e3) / 1e9 / hbm, "peak_source": f"{peak_src} HBM copy"},
        "expert_load": {"touched": work["touched_experts"], "max_rows": int(counts.max()),
                        "mean_rows_public": float(counts[:s.E_pub].mean()),
                        "mean_rows_private": float(counts[s.E_pub:].mean())},
        "gpu_launches": pmpe.kernels_per_forward(s) * args.steps,
        "clocks": clocks,
        "wall_s_timed_region": t_wall,
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h.numel() * 2 + pol.numel(),
                "d2h_bytes_per_step": out.numel() * 2,
                "pipeline": "pinned host -> device copy-in, forward, device -> pinned host copy-out on three "
                            "streams with two device buffer sets; one window over all K steps",
                "l2": "not flushed: every step streams the layer's weights, far larger than L2"},
        "config": {"workload": cfg.name, "T": s.T, "H": s.H, "I": s.I, "E_pub": s.E_pub, "E_priv": s.E_priv,
                   "E_shared": s.E_sh, "k": s.k, "renormalize": s.renormalize, "requests": cfg.n_requests,
                   "allow_tokens": int((pol == 1).sum().item()),
                   "l2": "flushed (512 MB write) before every step, then a 0.1 ms GPU spin outside the timed interval", "parallelism": f"replicas x{ws_n}"},
    }
    return rep, layer, counts


def measure_backward(pmpe, cfg, layer, h, pol, dev, args, flush, counts):
    """The private-branch backward, the input gradient, both in one pass,
    and a training step (forward + both), each after its own L2 flush."""
    s = cfg.shape
    stream = torch.cuda.current_stream(dev)
    out = torch.empty_like(h)
    hbm, tf_burst, tf_sus, peak_src = _peaks()
    g_dout = torch.Generator(device=dev)
    g_dout.manual_seed(7)
    dout = torch.randn(h.shape, generator=g_dout, device=dev, dtype=torch.float32).to(torch.bfloat16)
    layer.forward(h, pol, out=out)

    def timed(fn, n):
        evs = []
        for _ in range(n):
            flush_l2(flush)
            a_ev, b_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a_ev.record(stream)
            fn()
            b_ev.record(stream)
            evs.append((a_ev, b_ev))
        torch.cuda.synchronize(dev)
        return float(np.mean([x.elapsed_time(y) for x, y in evs]))

    for _ in range(2):
        layer.backward_private(h, pol, dout)
    bwd_avg = timed(lambda: layer.backward_private(h, pol, dout), args.steps)
    for _ in range(2):
        layer.backward_input(h, pol, dout)
    bin_avg = timed(lambda: layer.backward_input(h, pol, dout), args.steps)
    for _ in range(2):
        layer.backward(h, pol, dout)
    bst_avg = timed(lambda: layer.backward(h, pol, dout), args.steps)

    def train_step(save):
        layer.forward(h, pol, out=out, save_for_backward=save)
        layer.backward(h, pol, dout)

    def fwd_only(save):
        layer.forward(h, pol, out=out, save_for_backward=save)

    train = {}
    for save in (True, False):
        for _ in range(2):
            train_step(save)
        key = "saved_gate_up" if save else "recomputed_gate_up"
        train[key] = {"step_ms": timed(lambda: train_step(save), args.steps),
                      "forward_ms": timed(lambda: fwd_only(save), args.steps)}
        train[key]["backward_ms"] = timed(lambda: layer.backward(h, pol, dout), args.steps)
    train["saved_bytes"] = int(pmpe._lib.pmpe_saved_gu_floats(s.T, s.I, s.E_sh, s.k)) * 4
    train["l2"] = "flushed before every step"

    allow = int((pol == 1).sum().item())
    f_bwd = backward_flops(s, counts, allow)
    backward = {"ms": bwd_avg, "flops": f_bwd, "tflops": f_bwd / (bwd_avg / 1e3) / 1e12,
                "tensor_frac": f_bwd / (bwd_avg / 1e3) / 1e12 / tf_burst, "peak_source": f"{peak_src} bf16 burst",
                "private_rows": int(counts[s.E_pub:].sum()), "launches": pmpe.kernels_per_backward_private(s),
                "l2": "flushed before every pass"}
    mb = backward_min_bytes(s, counts, allow, "private")
    backward.update({"min_dram_bytes": mb, "hbm_gbs_of_min_bytes": mb / (bwd_avg / 1e3) / 1e9,
                     "hbm_frac_of_min_bytes": mb / (bwd_avg / 1e3) / 1e9 / hbm})
    f_bin = backward_input_flops(s, counts, allow)
    backward_in = {"ms": bin_avg, "flops": f_bin, "tflops": f_bin / (bin_avg / 1e3) / 1e12,
                   "tensor_frac": f_bin / (bin_avg / 1e3) / 1e12 / tf_burst, "peak_source": f"{peak_src} bf16 burst",
                   "routed_rows": int(counts.sum()), "launches": pmpe.kernels_per_backward_input(s),
                   "l2": "flushed before every pass"}
    mb = backward_min_bytes(s, counts, allow, "input")
    backward_in.update({"min_dram_bytes": mb, "hbm_gbs_of_min_bytes": mb / (bin_avg / 1e3) / 1e9,
                        "hbm_frac_of_min_bytes": mb / (bin_avg / 1e3) / 1e9 / hbm})
    backward_step = {"ms": bst_avg, "flops": f_bwd + f_bin - 6.0 * float(counts[s.E_pub:].sum()) * s.H * s.I,
                     "separate_ms": bwd_avg + bin_avg, "launches": pmpe.kernels_per_backward_step(s),
                     "outputs": "the private gradients and d_hidden, bitwise as the two separate passes",
                     "l2": "flushed before every pass"}
    backward_step["tflops"] = backward_step["flops"] / (bst_avg / 1e3) / 1e12
    return {"backward_private": backward, "backward_input": backward_in, "backward_step": backward_step,
            "training_step": train}


# the single-layer workloads the bench also measures beside the headline one
EXTRA_WORKLOADS = ("qwen3_decode", "deepseek_v2_lite", "tiny")


def run_ours(args):
    from paper_2608_06690_gb300 import pmpe
    ws_n, rank, local = _dist()
    if ws_n > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def barrier():
        if ws_n > 1:
            torch.distributed.barrier()

    nvml = NvmlClockSampler(local).__enter__()
    clk = ClockSampler(local).__enter__()   # nvidia-smi samples through the whole run
    cfg = CONFIGS[args.config]
    w, h, pol = build_workload(cfg, dev)
    head, layer, counts = measure_forward(pmpe, cfg, w, h, pol, dev, args, ws_n, barrier, nvml, flush)
    extras = {} if args.no_backward else measure_backward(pmpe, cfg, layer, h, pol, dev, args, flush, counts)
    del layer
    others = {}
    if not args.only:
        for name in EXTRA_WORKLOADS:
            if name == cfg.name:
                continue
            c2 = CONFIGS[name]
            w2, h2, p2 = build_workload(c2, dev)
            rep2, l2, _ = measure_forward(pmpe, c2, w2, h2, p2, dev, args, ws_n, barrier, nvml, flush)
            others[name] = rep2
            del l2, w2, h2, p2
            torch.cuda.empty_cache()
    nvml.__exit__(None, None, None)
    clk.__exit__(None, None, None)

    if rank != 0:
        if ws_n > 1:
            torch.distributed.destroy_process_group()
        return

    smi = clk.summary()
    clocks = dict(head["clocks"])
    if clocks.get("sm_mhz") is None:   # NVML unavailable: the nvidia-smi samples of the whole run
        clocks.update({k: smi[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")})
    clocks["smi_whole_run"] = smi
    line = {
        "metric": METRIC, "value": head["value"], "unit": "tokens/s", "n_gpus": ws_n, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": head["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": head["config"],
        "roofline": head["roofline"],
        "stages": head["stages"],
        "layer_hbm": head["layer_hbm"],
        "expert_load": head["expert_load"],
        "gpu_launches": head["gpu_launches"],
        "clocks": clocks,
        "wall_s_timed_region": head["wall_s_timed_region"],
        "e2e": head["e2e"],
    }
    line.update(extras)
    if others:
        line["workloads"] = others
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, w, h, pol, budget_s=args.cpu_budget)
    print(json.dumps(line), flush=True)
    if ws_n > 1:
        torch.distributed.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", default="qwen3_prefill", choices=sorted(CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--ref-tokens", type=int, default=96)
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-backward", action="store_true", help="skip the backward and training-step timings")
    ap.add_argument("--only", action="store_true", help="measure only --config, not the other workloads")
    ap.add_argument("--traffic", type=float, default=None,
                    help="DRAM bytes per launch of the dominant kernel from an ncu capture of this build")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
