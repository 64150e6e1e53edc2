"""Benchmark of the slot-addressed MoE layer forward on GB300.

python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

A step is one MoE layer forward over one batch of synthetic tokens: router
(fp32 logits, softmax, top-k), histogram and permutation, expert staging into
GPU slots (LRU waves, generation-fenced) where the workload streams, grouped
SwiGLU expert FFN reading weights from slots, shared expert, combine.
Default workload (prefill32k_lru64): the Qwen3-Next-shaped layer (hidden
2048, 512 experts, top-10, intermediate 512, shared expert) over a
32,768-token prefill with a 64-slot pool: 448 of the 512 experts are staged
from pinned host windows per call in LRU waves of 32.  The same line carries
a resident pass (`resident_32k`): the same 32,768 tokens with all 512 experts
resident in a 512-slot pool, so the routed GEMMs' tensor fraction is also
measured without waves.  --workload qwen3next_4k runs 4,096 tokens with all
512 experts resident; qwen3next_32k the resident 32K step alone;
prefill32k_q4_lru64 the staged 32K step with 4-bit experts.
--workload decode48 runs one
decode step through a stack of 48 layers of the tiny shape (hidden 256, 16
experts, top-2, intermediate 128) over --batch rows, one 64-slot LRU pool
shared by the 768 objects; --predict adds next-layer prediction with the
two-bank prefetch (each call routes its rows through the next layer's router
and stages the predicted objects after its last wave).

Prints one JSON line (rank 0).  `value` is whole-job tokens/s at the median
timed step (device time, CUDA events on the compute stream around each step,
no per-kernel events inside it; the mean is beside it); a second timed pass of the same steps with an
event pair around every kernel launch gives `kernels_ms_per_step` and the
roofline kernel's launch duration; `e2e` repeats the
metric with the hidden rows copied from pinned host memory and the outputs
read back inside the timed region; `roofline` is the routed expert GEMMs'
(gate-up and down together, the dominant pair) algorithmic work per launch
pair over their event-timed duration, against the burst bf16 peak when
tensor-bound (they run at full clock inside the step) or the copy bandwidth
when HBM-bound; `h2d_roof` sets the staged bytes of a step against the
host-to-device copy rate measured in the same run; `cpu_baseline` is the fp64
oracle timed on a bounded sample on this host's cores, with the BLAS threads
it actually ran on.
Multi-GPU (torchrun): independent replicas, one per GPU, no collective in the
data path; the timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "MoE-layer prefill tokens/s"
METRIC_DECODE = "MoE decode tokens/s through a 48-layer stack"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                  "sm_max_mhz": 2070.0}
N_SMS = 152
# FP32 FFMA throughput measured on this machine's GB300 at 2,070 MHz
# (profiles/ffma_roof.md): the roof of the SIMT router
FFMA_TFLOPS_MEASURED = 82.6
FFMA_MHZ = 2070.0
L2_BYTES = 129 * 1024 * 1024

# dram__bytes_read.sum + dram__bytes_write.sum per launch from one ncu capture
# (the summaries under profiles/), keyed by (workload, kernel kind); reported
# only while the GEMM source still hashes to the value the capture was taken at.
TRAFFIC = {
    # one fused wave launch (gate-up + down of 32 experts, ~20,480 routed rows)
    ("prefill32k_lru64", "gateup+down"): {"bytes_per_launch": 293416192 + 58992128, "src_hash": "aabc8aa52af9bf27",
                                          "profile": "profiles/gemm_fused_wave_prefill32k_lru64.md"},
    # the fused launch of a 4K resident call
    ("qwen3next_4k", "gateup+down"): {"bytes_per_launch": 3388257536 + 196642816, "src_hash": "aabc8aa52af9bf27",
                                      "profile": "profiles/gemm_fused_qwen3next_4k.md"},
    # one fused 4-bit wave launch
    ("prefill32k_q4_lru64", "gateup+down"): {"bytes_per_launch": 144022272 + 54480128, "src_hash": "aabc8aa52af9bf27",
                                             "profile": "profiles/gemm_fused_wave_q4_prefill32k_q4_lru64.md"},
}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


def kernel_source_hash() -> str:
    """Hash of the grouped-GEMM source (the dominant kernels' code), comments
    and blank lines left out: a capture stays valid until the code changes."""
    import re
    h = hashlib.sha256()
    for name in ("gemm.cu", "gemm_pair.cu", "gemm_fused.cu", "gemm_fused_pair.cu", "internal.cuh"):
        with open(os.path.join(ROOT, "paper_2608_23805_gb300", "csrc", name)) as f:
            src = re.sub(r"/\*.*?\*/", "", f.read(), flags=re.S)
        for line in src.splitlines():
            code = re.sub(r"//.*", "", line).strip()
            if code:
                h.update(code.encode() + b"\n")
    return h.hexdigest()[:16]


# ---------------------------------------------------------------------------
# Distributed plumbing (replicas only)
# ---------------------------------------------------------------------------

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def aggregate(units_per_rank: float, seconds: float, world: int, backend_ready: bool):
    """Whole-job throughput for independent replicas: the units all ranks
    processed over the slowest rank's time (max over ranks)."""
    if world > 1 and backend_ready:
        import torch
        import torch.distributed as dist
        dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
        t = torch.tensor([seconds, units_per_rank], dtype=torch.float64, device=dev)
        mx = t[:1].clone()
        dist.all_reduce(mx, op=dist.ReduceOp.MAX)
        tot = t[1:].clone()
        dist.all_reduce(tot, op=dist.ReduceOp.SUM)
        return float(tot.item()) / float(mx.item()), float(mx.item())
    return units_per_rank / seconds, seconds


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", "msi_clocks_%d_%d.csv" % (os.getpid(), gpu_index))

    def start(self):
        if os.environ.get("MSI_NO_CLOCKS"):
            return
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", os.environ.get("MSI_CLOCK_MS", "20")],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
            return
        # the sampler's start-up (driver-library initialisation) must not fall
        # inside the warm-up or timed region: wait for its first sample
        t0 = time.time()
        while time.time() - t0 < 10.0 and self.proc.poll() is None:
            self.f.flush()
            if os.path.getsize(self.path) > 0:
                break
            time.sleep(0.05)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# Workload setup (synthetic, seeded)
# ---------------------------------------------------------------------------

class Workload:
    def __init__(self, name: str, batch: int | None = None, predict: bool = False, windows=None,
                 early_staging: bool = False):
        """windows: pinned host windows of an earlier workload with the same
        layer shape and weights (reused, not regenerated); early_staging:
        streamed calls copy their first misses while they route."""
        import torch

        import synth
        from paper_2608_23805_gb300 import api
        cfg = synth.config(name)
        if batch is not None and cfg.n_layers > 1:
            cfg = synth.config(name, tokens=batch)
        self.cfg = cfg
        self.name = name
        self.L = L = cfg.n_layers
        self.predict = predict and L > 1
        E, H, I, eb = cfg.n_experts, cfg.hidden, cfg.inter, cfg.extent_bytes
        if windows is not None:
            assert windows.numel() == L * E * eb
            self.windows = windows
        else:
            self.windows = torch.empty(L * E * eb, dtype=torch.uint8, pin_memory=True)
            wnp = self.windows.numpy()
            for l in range(L):
                synth.fill_extents(cfg, l, wnp[l * E * eb:(l + 1) * E * eb])
        self.routers_np = [synth.router_weight(cfg, l) for l in range(L)]
        self.routers = [torch.from_numpy(w).cuda() for w in self.routers_np]
        self.router_np, self.router = self.routers_np[0], self.routers[0]
        self.x_bits = synth.hidden(cfg)
        self.x_host = torch.from_numpy(self.x_bits.view(np.int16)).view(torch.bfloat16).pin_memory()
        self.x = self.x_host.cuda()
        shared_w = gate_w = None
        self.shared_np = self.gate_np = None
        if cfg.has_shared:
            self.shared_np = synth.shared_extent(cfg)
            self.gate_np = synth.shared_gate_weight(cfg)
            shared_w = torch.from_numpy(self.shared_np).cuda()
            gate_w = torch.from_numpy(self.gate_np[None, :].copy()).cuda()
        self.plan = api.Plan(n_layers=L, n_experts=E, top_k=cfg.top_k, hidden=H, inter=I,
                             n_slots=cfg.n_slots, host_windows=self.windows,
                             has_shared=cfg.has_shared, shared_w=shared_w, shared_gate_w=gate_w,
                             wdtype=cfg.wdtype, early_staging=early_staging)
        self.cs = torch.cuda.Stream()
        self.ss = torch.cuda.Stream()
        self.out = torch.empty_like(self.x)
        self.ev = api.RouteEvent(cfg.tokens, cfg.top_k, E)
        if L > 1:  # a layer stack: outputs alternate between two buffers
            self.outs = [self.out, torch.empty_like(self.x)]
            self.evs = [api.RouteEvent(cfg.tokens, cfg.top_k, E) for _ in range(L)]
            self.nevs = [api.RouteEvent(cfg.tokens, cfg.top_k, E) for _ in range(L)]
            self.out, self.ev = self.outs[(L - 1) % 2], self.evs[L - 1]
        self.table = self.gens = None
        if not cfg.lru:
            for e in range(E):
                self.plan.stage(e, 0, e, self.ss)
            torch.cuda.synchronize()
            self.table, self.gens = self.plan.slot_table(0)

    def step(self, x=None):
        x = self.x if x is None else x
        if self.L > 1 and not self.predict:
            # the whole stack in one call (msi_moe_forward_streamed_stack)
            self.plan.forward_streamed_stack(0, x, self.routers, self.outs[0], self.outs[1], self.evs,
                                             residual=True, stream=self.cs, stage_stream=self.ss)
            return
        if self.L > 1:
            for l in range(self.L):
                nxt = self.routers[l + 1] if self.predict and l + 1 < self.L else None
                out = self.outs[l % 2]
                self.plan.forward_streamed(l, x, self.routers[l], out=out, ev=self.evs[l],
                                           residual=True, stream=self.cs, stage_stream=self.ss,
                                           next_router_w=nxt, next_ev=self.nevs[l] if nxt is not None
                                           else None)
                x = out
            return
        if self.cfg.lru:
            self.plan.forward_streamed(0, x, self.router, out=self.out, ev=self.ev, stream=self.cs,
                                       stage_stream=self.ss)
        else:
            self.plan.forward(0, x, self.router, self.table, self.gens, out=self.out, ev=self.ev,
                              stream=self.cs)

    def step_host(self, out_host, ids_host):
        """One step end to end through the host-buffer C-ABI call: rows from
        pinned host memory in, outputs and route ids to pinned host memory
        out (copies inside the call, on the plan's copy stream)."""
        self.plan.forward_host(0, self.x_host, self.router, self.table, self.gens, out_host=out_host,
                               ids_host=ids_host, ev=self.ev, stream=self.cs, stage_stream=self.ss)


def algorithmic(cfg, kind: str, units: dict):
    """Algorithmic work per step of one kernel kind: (bound, flops, bytes).

    rows = T*k routed rows; per routed row the gate-up GEMM does 2*H*2I flops
    and the down GEMM 2*I*H; weights are read once per expert per step; the
    gate-up reads each token's row once (its re-reads for further experts are
    L2 hits, not algorithmic HBM traffic) and writes h; the down reads h and
    writes the expert outputs."""
    T, H, I, E, k = cfg.tokens, cfg.hidden, cfg.inter, cfg.n_experts, cfg.top_k
    rows = T * k
    wb = 2.0 if cfg.wdtype == 0 else 0.5625      # bytes per weight (bf16, or 4-bit + fp16 scale / 32)
    eb_w13 = 2 * I * H * wb
    eb_w2 = H * I * wb
    if kind == "gateup":
        return 2.0 * rows * H * 2 * I, E * eb_w13 + T * H * 2 + rows * I * 2
    if kind == "down":
        return 2.0 * rows * I * H, E * eb_w2 + rows * I * 2 + rows * H * 2
    if kind == "shared_gateup":
        return 2.0 * T * H * 2 * I, eb_w13 + T * H * 2 + T * I * 2
    if kind == "shared_down":
        return 2.0 * T * I * H, eb_w2 + T * I * 2 + T * H * 2
    if kind == "router":
        return 2.0 * T * H * E, T * H * 2 + E * H * 4 + T * k * 8
    if kind == "combine":
        return 2.0 * rows * H, rows * H * 2 + T * H * 2 * (2 if cfg.has_shared else 1) + T * k * 8
    if kind in ("scan", "scatter"):
        return 0.0, T * k * 4 * 3
    return 0.0, 0.0


def _bound_of(flops: float, nbytes: float, peaks: dict) -> str:
    """tensor when the work's arithmetic intensity is at or above the ridge of
    the burst bf16 peak over the copy bandwidth, else hbm."""
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    return "tensor" if flops > 0 and flops / max(nbytes, 1.0) >= ridge else "hbm"


def _part(flops_step: float, bytes_step: float, ms: float, launches: int, steps: int, peaks: dict,
          bound: str) -> dict:
    per_launch_s = ms / 1e3 / max(launches, 1)
    if bound == "tensor":
        ach = flops_step * steps / max(launches, 1) / per_launch_s / 1e12
        return {"achieved": ach, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "frac": ach / peaks["bf16_tflops"], "ms_per_launch": ms / max(launches, 1)}
    ach = bytes_step * steps / max(launches, 1) / per_launch_s / 1e9
    return {"achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": ach / peaks["hbm_gbs"], "ms_per_launch": ms / max(launches, 1)}


def roofline(cfg, kt: dict, steps: int, peaks: dict, clocks: dict, workload: str):
    """Roofline object of the routed expert GEMMs, gate-up and down together
    (the dominant pair of every step that routes rows): their algorithmic
    flops (or bytes) per launch pair over the pair's summed event-timed
    duration.  Tensor-bound work is set against the burst bf16 peak: the
    kernels run at full SM clock inside steps of milliseconds, far from the
    seconds-long power-capped loop the sustained figure comes from.  Without
    routed GEMM time (a step with no rows) the dominant kernel kind alone."""
    if "ffn" in kt or ("gateup" in kt and "down" in kt):
        # separate launches (gateup, down) and fused wave launches (ffn: both
        # projections of one wave in one kernel) may both appear in a step
        f1, b1 = algorithmic(cfg, "gateup", {})
        f2, b2 = algorithmic(cfg, "down", {})
        bound = _bound_of(f1 + f2, b1 + b2, peaks)
        ms = sum(kt[k][0] for k in ("gateup", "down", "ffn") if k in kt)
        launches = kt["ffn"][1] if "ffn" in kt else kt["gateup"][1]
        r = {"bound": bound}
        r.update(_part(f1 + f2, b1 + b2, ms, launches, steps, peaks, bound))
        r["kernel"] = "gateup+down"
        r["launches_per_step"] = launches / steps
        r["parts"] = {}
        if "gateup" in kt and "down" in kt:
            r["parts"]["gateup"] = dict(_part(f1, b1, kt["gateup"][0], kt["gateup"][1], steps, peaks, bound),
                                        flops_per_step=f1, bytes_per_step=b1)
            r["parts"]["down"] = dict(_part(f2, b2, kt["down"][0], kt["down"][1], steps, peaks, bound),
                                      flops_per_step=f2, bytes_per_step=b2)
        if "ffn" in kt:
            r["fused_waves"] = True
        kind = "gateup+down"
    else:
        kind = max(kt, key=lambda k: kt[k][0])
        ms, launches = kt[kind]
        flops, nbytes = algorithmic(cfg, kind, {})
        if kind == "router":
            mhz = clocks.get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
            peak = FFMA_TFLOPS_MEASURED * mhz / FFMA_MHZ
            per_launch_s = ms / 1e3 / max(launches, 1)
            ach = flops * steps / max(launches, 1) / per_launch_s / 1e12
            r = {"bound": "alu", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                 "frac": ach / peak, "ms_per_launch": ms / max(launches, 1)}
        else:
            bound = _bound_of(flops, nbytes, peaks)
            r = {"bound": bound}
            r.update(_part(flops, nbytes, ms, launches, steps, peaks, bound))
        r["kernel"] = kind
        r["launches_per_step"] = launches / steps
    if r["bound"] == "tensor":
        r["peak_source"] = "bf16_tflops (burst) of measured"
    elif r["bound"] == "hbm":
        r["peak_source"] = "hbm_gbs of measured"
    else:
        r["peak_source"] = "measured FP32 FFMA rate (profiles/ffma_roof.md) x median SM clock / 2070 MHz"
    t = TRAFFIC.get((workload, kind))
    r["traffic"] = t["bytes_per_launch"] if (t and t.get("src_hash") == kernel_source_hash()) else None
    if r["traffic"] is not None:
        r["traffic_source"] = t["profile"]
    return r


def blas_threads():
    """(threads, how): the BLAS threads numpy's matrix products run on (the
    oracle's time is almost all there), read from the loaded OpenBLAS."""
    import ctypes
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var]), var
    np.ones((64, 64)) @ np.ones((64, 64))          # BLAS loaded
    try:
        paths = sorted({l.split()[-1] for l in open("/proc/self/maps") if "openblas" in l.lower()
                        and l.split()[-1].startswith("/")})
    except OSError:
        paths = []
    for path in paths:
        try:
            lib = ctypes.CDLL(path)
        except OSError:
            continue
        for sym in ("scipy_openblas_get_num_threads64_", "openblas_get_num_threads64_",
                    "openblas_get_num_threads"):
            fn = getattr(lib, sym, None)
            if fn is not None:
                fn.restype = ctypes.c_int
                return int(fn()), "%s from %s" % (sym, os.path.basename(path))
    return os.cpu_count() or 1, "os.cpu_count() (no OpenBLAS found to ask)"


def h2d_probe(nbytes: int = 192 << 20, reps: int = 4):
    """Host-to-device copy rate (GB/s) of one staging run's size (32 extents
    of 6 MiB) from pinned memory: best of `reps` copies, CUDA events."""
    import torch
    src = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    dst = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    best = None
    s = torch.cuda.Stream()
    for _ in range(reps + 1):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(s)
        with torch.cuda.stream(s):
            dst.copy_(src, non_blocking=True)
        b.record(s)
        b.synchronize()
        t = a.elapsed_time(b) / 1e3
        best = t if best is None else min(best, t)
    return nbytes / best / 1e9


def cpu_baseline(w: "Workload", tokens: int):
    """The fp64 oracle, as it stands, on the first `tokens` tokens of the same
    workload, on this host's cores; tokens/s."""
    import oracle
    cfg = w.cfg
    eb = cfg.extent_bytes
    wnp = w.windows.numpy()
    kw = {}
    if cfg.has_shared:
        kw = dict(shared_extent=w.shared_np, w_sg=w.gate_np)
    if w.L > 1:
        dt = oracle_stack(cfg, w.x_bits[:tokens], w.routers_np, wnp)
        cores, how = blas_threads()
        return {"value": tokens / dt, "unit": "tokens/s", "cores": cores, "cores_source": how,
                "host_cpus": os.cpu_count(), "kind": "oracle",
                "sample": "fp64 oracle of one decode step of %d rows through all %d layers (router, "
                          "expert FFNs, combine with residual, LRU-wave plan of the shared pool), "
                          "%.2f s" % (tokens, w.L, dt)}
    t0 = time.perf_counter()
    oracle.moe_layer(w.x_bits[:tokens], w.router_np, cfg.top_k, lambda e: wnp[e * eb:(e + 1) * eb],
                     cfg.hidden, cfg.inter, cfg.wdtype, **kw)
    if cfg.lru:
        sim = oracle.LRUWaveSim(cfg.n_slots)
        sim.call(0, range(cfg.n_experts))
    dt = time.perf_counter() - t0
    cores, how = blas_threads()
    return {"value": tokens / dt, "unit": "tokens/s", "cores": cores, "cores_source": how,
            "host_cpus": os.cpu_count(), "kind": "oracle",
            "sample": "fp64 oracle forward of the first %d of %d tokens (router over all %d experts, "
                      "expert FFNs, shared expert, combine, LRU-wave plan), %.1f s" %
                      (tokens, cfg.tokens, cfg.n_experts, dt)}


def oracle_stack(cfg, x_bits, routers_np, wnp) -> float:
    """Seconds the fp64 oracle takes for one decode step through the layer
    stack (each layer's output rounded to bf16 for the next, as the GPU
    stack does; the LRU-wave plan of the shared pool alongside)."""
    import torch

    import oracle
    E, eb = cfg.n_experts, cfg.extent_bytes
    sim = oracle.LRUWaveSim(cfg.n_slots)
    t0 = time.perf_counter()
    x = x_bits
    for l, wr in enumerate(routers_np):
        r = oracle.moe_layer(x, wr, cfg.top_k,
                             lambda e, l=l: wnp[(l * E + e) * eb:(l * E + e + 1) * eb],
                             cfg.hidden, cfg.inter, cfg.wdtype, residual=True)
        sim.call(l, sorted(set(r["ids"].reshape(-1).tolist())))
        x = torch.from_numpy(r["out"]).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    return time.perf_counter() - t0


SAMPLE_TOKENS = {"prefill32k_lru64": 4096, "prefill32k_q4_lru64": 4096, "qwen3next_4k": 4096,
                 "qwen3next_32k": 4096, "tiny": 64}


# ---------------------------------------------------------------------------
# Arms
# ---------------------------------------------------------------------------

def run_ours(args):
    import torch
    world, rank, local = dist_env()
    backend = False
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", init_method="env://")
        backend = True
    else:
        torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    early = not args.no_early_staging and args.source == "none"
    w = Workload(args.workload, args.batch, args.predict, early_staging=early)
    cfg = w.cfg
    src = None
    if args.source != "none":
        if not cfg.lru:
            raise SystemExit("--source applies to the staged (LRU) workloads")
        from paper_2608_23805_gb300 import api
        path = os.path.join(os.environ.get("MSI_SOURCE_DIR", "/tmp"), "msi_extents_%d.bin" % os.getpid())
        with open(path, "wb") as f:
            f.write(w.windows.numpy().tobytes())
        src = api.Source(path, cfg.extent_bytes + 2 * 4096, n_windows=8, direct=args.source == "direct")
        os.unlink(path)  # the open file stays readable
        w.plan.set_source(src, np.arange(w.L * cfg.n_experts, dtype=np.uint64) * cfg.extent_bytes)
    peaks, peak_kind = load_peaks()

    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda")
    # the host-to-device rate of this machine, before anything is timed
    h2d_gbs = h2d_probe() if cfg.lru else None
    sampler = ClockSampler(local)
    sampler.start()
    def flush_l2(wk=None):
        # on the compute stream, so that it is ordered before the step's start
        # event and never overlaps a timed step
        with torch.cuda.stream((wk or w).cs):
            flush.zero_()

    def warm(wk):
        # warm-up immediately precedes the timed steps (an idle GPU drops its
        # clocks and link state)
        for _ in range(args.warmup):
            flush_l2(wk)
            wk.step()
        torch.cuda.synchronize()
        flush_l2(wk)                                 # one more untimed step right before timing
        wk.step()
        torch.cuda.synchronize()

    warm(w)

    def timed_steps(wk=None):
        wk = wk or w
        evs = []
        for _ in range(args.steps):
            flush_l2(wk)                             # L2 flushed between timed steps (untimed)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(wk.cs)
            wk.step()
            b.record(wk.cs)
            evs.append((a, b))
        torch.cuda.synchronize()
        return evs

    # (1) the step itself, no per-kernel events inside it: `value`
    if backend:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    launches0 = w.plan.launches()
    staged0 = w.plan.counters()["h2d_bytes"]
    wall0 = time.perf_counter()
    evs = timed_steps()
    wall = time.perf_counter() - wall0
    launches = w.plan.launches() - launches0
    staged = (w.plan.counters()["h2d_bytes"] - staged0) // args.steps
    step_ms = [a.elapsed_time(b) for a, b in evs]
    # value at the median step (a staged step that meets one of the host
    # link's periodic stalls would move a mean by tens of percent)
    dev_s = float(np.median(step_ms)) * args.steps / 1e3
    mean_ms = float(np.mean(step_ms))
    # (2) the same steps with an event pair around every kernel launch: the
    # per-kernel times and the roofline kernel's launch duration
    w.plan.timing(True)
    w.plan.timing_read(reset=True)
    evs_k = timed_steps()
    kt = w.plan.timing_read(reset=True)
    w.plan.timing(False)
    assert w.plan.status() == 0, "device status %d" % w.plan.status()

    # e2e: hidden rows from pinned host memory in, outputs and route ids out.
    # Single layers go through the host-buffer C-ABI call (the copies run
    # inside it); the layer stack copies around its device-buffer step.
    out_host = torch.empty_like(w.out, device="cpu").pin_memory()
    ids_host = torch.empty_like(w.ev.ids, device="cpu").pin_memory()
    x_dev = torch.empty_like(w.x)
    e2e_evs = []
    for _ in range(args.steps):
        flush_l2()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(w.cs)
        if w.L == 1:
            w.step_host(out_host, ids_host)
        else:
            with torch.cuda.stream(w.cs):
                x_dev.copy_(w.x_host, non_blocking=True)
            w.step(x_dev)
            with torch.cuda.stream(w.cs):
                out_host.copy_(w.out, non_blocking=True)
                ids_host.copy_(w.ev.ids, non_blocking=True)
        b.record(w.cs)
        b.synchronize()
        e2e_evs.append((a, b))
    e2e_s = float(np.median([a.elapsed_time(b) for a, b in e2e_evs])) * args.steps / 1e3

    # the same 32K tokens with all 512 experts resident (no waves, no staging):
    # the routed GEMMs' tensor fraction outside the LRU waves
    resident = None
    if args.workload == "prefill32k_lru64" and not args.no_resident_pass and world == 1:
        rwk = Workload("qwen3next_32k", windows=w.windows)
        warm(rwk)
        revs = timed_steps(rwk)
        rwk.plan.timing(True)
        rwk.plan.timing_read(reset=True)
        timed_steps(rwk)
        rkt = rwk.plan.timing_read(reset=True)
        rwk.plan.timing(False)
        assert rwk.plan.status() == 0, "device status %d" % rwk.plan.status()
        rms = float(np.median([a.elapsed_time(b) for a, b in revs]))
        resident = {
            "workload": "qwen3next_32k", "tokens": rwk.cfg.tokens, "slots": rwk.cfg.n_slots,
            "residency": "all 512 experts resident", "ms_per_step": rms,
            "value": rwk.cfg.tokens / rms * 1e3, "unit": "tokens/s",
            "roofline": roofline(rwk.cfg, {k: v for k, v in rkt.items() if v[1] > 0}, args.steps, peaks,
                                 {}, "qwen3next_32k"),
            "kernels_ms_per_step": {k: round(v[0] / args.steps, 4) for k, v in rkt.items() if v[1] > 0},
            "step_ms": [round(a.elapsed_time(b), 3) for a, b in revs]}
        rwk.plan.close()
        del rwk
    if backend:
        torch.distributed.barrier()
    clocks = sampler.stop()

    units = cfg.tokens * args.steps
    value, tmax = aggregate(units, dev_s, world, backend)
    e2e_value, _ = aggregate(units, e2e_s, world, backend)
    if rank != 0:
        return
    rl = roofline(cfg, {k: v for k, v in kt.items() if v[1] > 0}, args.steps * w.L, peaks, clocks,
                  args.workload)
    line = {
        "metric": METRIC if w.L == 1 else METRIC_DECODE, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": tmax / args.steps * 1e3, "ms_per_step_mean": mean_ms,
        "step_statistic": "median of the timed steps", "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded N(0,1) bf16 hidden rows, N(0,0.02) bf16 expert weights, "
                "N(0,0.02) fp32 router",
        "config": {"workload": args.workload, "tokens": cfg.tokens, "hidden": cfg.hidden,
                   "experts": cfg.n_experts, "top_k": cfg.top_k, "inter": cfg.inter,
                   "shared_expert": cfg.has_shared, "slots": cfg.n_slots,
                   "residency": "LRU waves of %d, staged from pinned host windows%s" % (
                       cfg.n_slots // 2, "; first misses copied early, while the call routes"
                       if early and cfg.lru and cfg.n_layers == 1 else "")
                   if cfg.lru else "all experts resident",
                   "layers": w.L,
                   "weights": "bf16" if cfg.wdtype == 0 else "q4g32",
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": "flushed between timed steps (2x L2 write, untimed)"},
        "roofline": rl,
        "e2e": {"value": e2e_value, "unit": "tokens/s",
                "h2d_bytes_per_step": int(w.x.numel() * 2),
                "d2h_bytes_per_step": int(w.out.numel() * 2 + w.ev.ids.numel() * 4),
                "staged_h2d_bytes_per_step": int(staged),
                "call": ("msi_moe_forward_streamed_host" if cfg.lru else "msi_moe_forward_host")
                if w.L == 1 else "host copies around the layer stack's device-buffer calls"},
        "gpu_launches": int(launches),
        "clocks": clocks,
        "kernels_ms_per_step": {k: round(v[0] / args.steps, 4) for k, v in kt.items() if v[1] > 0},
        "wall_s_timed": wall,
        "step_ms": [round(t, 3) for t in step_ms],
        "step_ms_kernel_timing": [round(a.elapsed_time(b), 3) for a, b in evs_k],
        "e2e_step_ms": [round(a.elapsed_time(b), 3) for a, b in e2e_evs],
        "peaks": peak_kind,
    }
    if cfg.lru and h2d_gbs:
        # the step's bytes from the host: the staged extents (and nothing else:
        # the rows are already on the device in the device-timed step)
        floor_ms = staged / (h2d_gbs * 1e9) * 1e3
        line["h2d_roof"] = {"bytes_per_step": int(staged), "measured_gbs": h2d_gbs,
                            "how": "pinned cudaMemcpyAsync of 192 MiB (one 32-extent run), best of 4",
                            "floor_ms": floor_ms, "frac": floor_ms / (tmax / args.steps * 1e3)}
    if resident is not None:
        line["resident_32k"] = resident
    if src is not None:
        ss = src.stats()
        line["config"]["source"] = {
            "kind": args.source, "windows": 8, "reads": ss["reads"], "rejected": ss["rejected"],
            "logical_gb": ss["logical_bytes"] / 1e9, "padding_mb": ss["padding_bytes"] / 1e6,
            "read_gbs_per_window": ss["logical_bytes"] / max(ss["read_seconds"], 1e-9) / 1e9,
            "max_in_flight": ss["max_in_flight"]}
        line["config"]["residency"] = "LRU waves of %d, staged from a file through the bounded " \
            "source service (%s reads)" % (cfg.n_slots // 2, args.source)
    if w.L > 1:
        c = w.plan.counters()
        line["config"]["residency"] = (
            "one %d-slot LRU pool shared by %d layers (%d objects), waves of %d, staged from pinned "
            "host windows%s" % (cfg.n_slots, w.L, w.L * cfg.n_experts, cfg.n_slots // 2,
                                "; next-layer prediction with two-bank prefetch" if w.predict else ""))
        line["config"]["prediction"] = {"on": w.predict, "prefetches": c["prefetches"],
                                        "prefetch_hits": c["prefetch_hits"], "stages": c["stages"],
                                        "hits": c["hits"]}
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, SAMPLE_TOKENS.get(args.workload, cfg.tokens))
    print(json.dumps(line), flush=True)


def run_reference(args):
    """Reference arm: the fp64 CPU oracle as it stands, each step a bounded
    sample (REF_TOKENS tokens) of the same workload, on this host's cores."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle
    import synth
    cfg = synth.config(args.workload)
    if cfg.n_layers > 1:
        cfg = synth.config(args.workload, tokens=args.batch)
        E, eb = cfg.n_experts, cfg.extent_bytes
        wnp = np.empty(cfg.n_layers * E * eb, dtype=np.uint8)
        for l in range(cfg.n_layers):
            synth.fill_extents(cfg, l, wnp[l * E * eb:(l + 1) * E * eb])
        routers = [synth.router_weight(cfg, l) for l in range(cfg.n_layers)]
        x = synth.hidden(cfg)
        for _ in range(args.warmup):
            oracle_stack(cfg, x, routers, wnp)
        dt = sum(oracle_stack(cfg, x, routers, wnp) for _ in range(args.steps))
        value = cfg.tokens * args.steps / dt
        sample = ("fp64 oracle of one decode step of %d rows through all %d layers per step"
                  % (cfg.tokens, cfg.n_layers))
        print(json.dumps({
            "impl": "reference", "metric": METRIC_DECODE, "value": value, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (same seeded inputs)",
            "config": {"workload": args.workload, "tokens": cfg.tokens, "layers": cfg.n_layers},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": blas_threads()[0],
                             "cores_source": blas_threads()[1], "host_cpus": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
        }), flush=True)
        return
    ntok = REF_TOKENS.get(args.workload, 128)
    eb = cfg.extent_bytes
    x = synth.hidden(cfg, tokens=ntok)
    wr = synth.router_weight(cfg)
    cache = {}

    def extent(e):
        if e not in cache:
            cache[e] = synth.expert_extent(cfg, 0, e)
        return cache[e]

    kw = {}
    if cfg.has_shared:
        kw = dict(shared_extent=synth.shared_extent(cfg), w_sg=synth.shared_gate_weight(cfg))
    for e in range(cfg.n_experts):
        extent(e)

    def step():
        oracle.moe_layer(x, wr, cfg.top_k, extent, cfg.hidden, cfg.inter, cfg.wdtype, **kw)
        if cfg.lru:
            oracle.LRUWaveSim(cfg.n_slots).call(0, range(cfg.n_experts))

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    value = ntok * args.steps / dt
    cores, how = blas_threads()
    sample = ("fp64 oracle forward of %d of the %d tokens per step (router over all %d experts, "
              "expert FFNs, shared expert, combine, LRU-wave plan)" % (ntok, cfg.tokens, cfg.n_experts))
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (same seeded inputs)",
        "config": {"workload": args.workload, "tokens": cfg.tokens, "sample_tokens": ntok},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "cores_source": how,
                         "host_cpus": os.cpu_count(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


REF_TOKENS = {"prefill32k_lru64": 4096, "prefill32k_q4_lru64": 4096, "qwen3next_4k": 4096,
              "qwen3next_32k": 4096, "tiny": 64}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="prefill32k_lru64",
                    choices=["prefill32k_lru64", "qwen3next_4k", "qwen3next_32k", "prefill32k_q4_lru64",
                             "tiny", "decode48"])
    ap.add_argument("--no-resident-pass", action="store_true",
                    help="prefill32k_lru64: skip the all-resident 32K pass")
    ap.add_argument("--batch", type=int, default=64, help="decode48: rows per decode step")
    ap.add_argument("--predict", action="store_true",
                    help="decode48: next-layer prediction with the two-bank prefetch")
    ap.add_argument("--no-early-staging", action="store_true",
                    help="staged workloads: no early-staging buffer (misses copied only after "
                         "the call's plan)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--source", default="none", choices=["none", "buffered", "direct"],
                    help="staged workloads: read every missing extent from a file through the "
                         "bounded source service (8 windows) instead of pinned host windows")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
