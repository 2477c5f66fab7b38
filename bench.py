#!/usr/bin/env python
"""Benchmark of one XShare MoE-layer forward on GB300.

A step is one xshare_moe_forward call: router + softmax, batch-aware expert
selection, refinement, permutation, gather, SwiGLU expert FFN over the used
experts, combine.  Default workload: the DeepSeek-R1-shaped layer (N = 256,
k = 8, d = 7168, F = 2048) at B = 32 tokens with Algorithm 2 (k0 = 1, m = 24).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints ONE JSON line on rank 0.  Multi-GPU runs (torchrun) are independent
replicas of the workload, one per GPU (the path does not shard on one layer
of this size); `value` sums all ranks' tokens over the slowest rank's time.
"""

from __future__ import annotations

import os
import sys

if "--impl" in sys.argv and "reference" in sys.argv:
    # The reference arm times the single-threaded CPU oracle: pin BLAS to one
    # thread before numpy loads.
    for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[_v] = "1"

import argparse
import ctypes
import hashlib
import json
import statistics
import subprocess
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2602_07265_gb300 import workloads as W  # noqa: E402

METRIC = "MoE-layer tokens/s and expert-weight HBM GB/s (% roofline); experts activated/batch"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
N_ROTATE = 4   # distinct input batches cycled through the timed steps
N_SINGLE = 20  # single steps timed one by one for the latency figure
L2_BYTES = 129e6


# --------------------------------------------------------------------------- setup

def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["xshare", "reference"], default="xshare")
    ap.add_argument("--workload", default="dsr1", choices=sorted(W.WORKLOADS))
    ap.add_argument("--B", type=int, default=None)
    ap.add_argument("--N", type=int, default=None, help="override the expert count (smaller profiling cases)")
    ap.add_argument("--F", type=int, default=None, help="override d_ff (smaller profiling cases)")
    ap.add_argument("--budget", type=int, default=None)
    ap.add_argument("--k0", type=int, default=None)
    ap.add_argument("--mode", default=None, choices=sorted(W.MODES))
    ap.add_argument("--tau", type=float, default=None, help="covered score-mass fraction (thresh)")
    ap.add_argument("--m-r", type=int, default=None, help="per-request budget (hier)")
    ap.add_argument("--m-g", type=int, default=None, help="per-group budget (group)")
    ap.add_argument("--sparse", action="store_true",
                    help="column scores from the top-k-masked gating values (Sec. 2.2)")
    ap.add_argument("--shared", type=int, default=0,
                    help="shared experts added to every token (DeepSeek-R1 has one)")
    ap.add_argument("--layers", type=int, default=1,
                    help="time a stack of this many residual layers, replayed from a CUDA graph")
    ap.add_argument("--weight-sets", type=int, default=2,
                    help="distinct expert-weight sets the stack's layers cycle through")
    ap.add_argument("--global-budget", type=int, default=None,
                    help="stack budget K (default: layers x the per-layer budget)")
    ap.add_argument("--unpacked", action="store_true",
                    help="read the expert weights as plain [N, F, d] matrices instead of packed tiles")
    ap.add_argument("--e2e-eager", action="store_true",
                    help="end-to-end steps as eager calls instead of CUDA-graph replays")
    ap.add_argument("--ep", action="store_true",
                    help="expert parallelism (Sec. 5): the N experts split over the ranks, one "
                         "layer per step on one shared batch, an all-reduce of the expert outputs")
    ap.add_argument("--sweep", action="append", default=[], metavar="FIELD=V1,V2,...",
                    help="sweep mode: time every combination of these workload fields (B, budget, "
                         "k0, m_r, m_g, tau, mode, tokens_per_request, sparse_scores), one JSON line "
                         "per combination with the median over --seeds")
    ap.add_argument("--seeds", default="0", help="comma-separated seeds (sweep mode)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--seed", type=int, default=0)
    return ap.parse_args(argv)


def workload_from_args(args) -> W.Workload:
    w = W.WORKLOADS[args.workload]
    kw = {}
    if args.B is not None:
        kw["B"] = args.B
    if args.N is not None:
        kw["N"] = args.N
    if args.F is not None:
        kw["F"] = args.F
    if args.budget is not None:
        kw["budget"] = args.budget
    if args.k0 is not None:
        kw["k0"] = args.k0
    if args.mode is not None:
        kw["mode"] = W.MODES[args.mode]
    if args.tau is not None:
        kw["tau"] = args.tau
    if args.m_r is not None:
        kw["m_r"] = args.m_r
    if args.m_g is not None:
        kw["m_g"] = args.m_g
    if args.sparse:
        kw["sparse_scores"] = 1
    return w.with_(**kw) if kw else w


def describe(w: W.Workload, n_shared: int = 0) -> str:
    mode = {0: "TOPK", 1: "BATCH (Algorithm 2)", 2: "GROUP (Algorithm 6)", 3: "HIER (Algorithm 4)",
            4: "THRESH (Algorithm 2, Algorithm 1 threshold)"}[w.mode]
    s = f"{w.name}: N={w.N} k={w.k} d={w.d} F={w.F} B={w.B} {mode}"
    if w.mode == W.MODE_BATCH:
        s += f" m={w.budget} k0={w.k0}"
    elif w.mode == W.MODE_HIER:
        s += f" m={w.budget} m_r={w.m_r} k0={w.k0} tokens/request={w.tokens_per_request}"
    elif w.mode == W.MODE_GROUP:
        s += f" G={w.n_groups} m_g={w.m_g} k0={w.k0}"
    elif w.mode == W.MODE_THRESH:
        s += f" tau={w.tau} k0={w.k0}"
    if w.sparse_scores:
        s += ", sparse (top-k-masked) column scores"
    if n_shared:
        s += f" + {n_shared} shared expert{'s' if n_shared > 1 else ''}"
    return s


def workload_config(w: W.Workload, n_shared: int, world: int) -> dict:
    """The `config` of the JSON line, the same for both arms: the workload and
    how the timed steps stay clear of L2."""
    return {
        "workload": describe(w, n_shared),
        "B": w.B, "N": w.N, "k": w.k, "d": w.d, "F": w.F, "shared_experts": n_shared,
        "global_batch": w.B * world,
        "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
        "l2": (f"inputs larger than L2: every step streams the weights of its used experts "
               f"({w.expert_bytes / 1e6:.1f} MB each; L2 129 MB), {N_ROTATE} rotating input batches")
        if w.N * w.expert_bytes > L2_BYTES else
        (f"all expert weights fit in L2 ({w.N * w.expert_bytes / 1e6:.0f} MB of 129 MB): "
         f"L2-warm steps, a correctness-size workload, not a bandwidth figure"),
    }


def measured_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS, "bf16_tflops": FALLBACK_BF16_TFLOPS,
                "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init_dist(world: int, backend: str):
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group(backend=backend)


def barrier(world: int):
    if world > 1:
        torch.distributed.barrier()


def reduce_max(value: float, world: int, device=None) -> float:
    """Max over ranks (the slowest rank's time)."""
    if world <= 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def reduce_sum(value: float, world: int, device=None) -> float:
    if world <= 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.SUM)
    return float(t.item())


# --------------------------------------------------------------------------- clocks

NVML_CLOCK_SM = 1
REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
           0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
           0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
           0x100: "display_clock_setting"}


class ClockSampler:
    """Samples the SM clock and the clock-event reasons through NVML (read only)
    on a background thread while the timed region runs."""

    def __init__(self, device_index: int, period_s: float = 0.005):
        self.period = period_s
        self.samples = []
        self.reasons = 0
        self.max_mhz = None
        self.ok = False
        self._stop = threading.Event()
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            props = torch.cuda.get_device_properties(device_index)
            bus = f"{props.pci_domain_id:08x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0".encode()
            h = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByPciBusId_v2(ctypes.c_char_p(bus), ctypes.byref(h)) != 0:
                if nv.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(h)) != 0:
                    return
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, NVML_CLOCK_SM, ctypes.byref(mx)) == 0:
                self.max_mhz = int(mx.value)
            self._nv, self._h = nv, h
            self._reasons_fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(nv, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.ok = True
        except (OSError, AttributeError):
            self.ok = False

    def _run(self):
        clk = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        while not self._stop.is_set():
            if self._nv.nvmlDeviceGetClockInfo(self._h, NVML_CLOCK_SM, ctypes.byref(clk)) == 0:
                self.samples.append(int(clk.value))
            if self._reasons_fn(self._h, ctypes.byref(rs)) == 0:
                self.reasons |= int(rs.value)
            time.sleep(self.period)

    def __enter__(self):
        if self.ok:
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()
        return self

    def __exit__(self, *exc):
        if self.ok:
            self._stop.set()
            self._t.join()

    def summary(self):
        if not self.ok or not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
                    "note": "NVML clock sampling unavailable"}
        names = [n for bit, n in REASONS.items() if self.reasons & bit and n != "gpu_idle"]
        return {"sm_mhz": float(statistics.median(self.samples)), "sm_max_mhz": self.max_mhz,
                "reasons": names, "samples": len(self.samples),
                "sm_mhz_min": min(self.samples)}


# --------------------------------------------------------------------------- traffic

# The source files each timed stage's kernel is built from.
KERNEL_SOURCES = {
    "ffn_gate_up": ("ffn_tc.cu", "tc_ptx.cuh", "tmap.cu", "tmap.cuh", "xs_internal.cuh"),
    "ffn_down": ("ffn_tc.cu", "tc_ptx.cuh", "tmap.cu", "tmap.cuh", "xs_internal.cuh"),
}


def kernel_source_hash(stage: str = "ffn_gate_up") -> str:
    """Hash of the sources of one stage's kernel: a recorded ncu traffic figure
    is only valid for the sources it was captured from."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2602_07265_gb300", "csrc")
    for name in KERNEL_SOURCES[stage]:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(stage: str, units: float):
    """DRAM bytes per launch from the committed ncu summary (profiles/traffic.json),
    scaled to this launch's units, or None if absent or captured from other sources."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(stage)
    except (OSError, ValueError):
        return None
    if not rec or stage not in KERNEL_SOURCES or rec.get("source_hash") != kernel_source_hash(stage):
        return None
    return float(rec["bytes_per_unit"]) * units


# --------------------------------------------------------------------------- GPU arm

def algorithmic_bytes(w: W.Workload, n_used: int, n_pairs: int, n_shared: int = 0) -> dict:
    """Bytes each stage must move at least: every weight matrix it uses once,
    plus its token rows in and out.  Shared experts count as n_shared more
    used experts with B more rows each."""
    d, F, N, B = w.d, w.F, w.N, w.B
    n_exp = n_used + n_shared
    rows = n_pairs + n_shared * B
    return {
        "router": N * d * 4 + B * d * 2 + B * N * 4,
        "ffn_gate_up": n_exp * 2 * F * d * 2 + rows * d * 2 + rows * F * 2,
        "ffn_down": n_exp * d * F * 2 + rows * F * 2 + rows * d * 4,
        "combine": rows * d * 4 + B * d * 2,
        "layer": n_exp * 6 * d * F + N * d * 4 + 2 * B * d * 2,
    }


def run_gpu(args, w: W.Workload, rank: int, world: int, local: int) -> dict:
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare as X

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(world, "nccl")
    stream = torch.cuda.current_stream()

    xs_host = [W.router_inputs(w, args.seed + 101 * rank + i)[0] for i in range(N_ROTATE)]
    _, W_g = W.router_inputs(w, args.seed)
    xs_dev = [x.to(dev) for x in xs_host]
    W_g = W_g.to(dev)
    Wg, Wu, Wd = W.expert_weights(w, args.seed, device=str(dev))
    Ns = args.shared
    shared = W.shared_expert_weights(w, Ns, args.seed, device=str(dev)) if Ns else None
    packed = not args.unpacked
    if packed:  # a layout change made once when the weights are loaded, outside the timed region
        pk = X.Packed(Wg, Wu, Wd)
        pshared = X.Packed(*shared) if shared is not None else None
        del Wg, Wu, Wd
        torch.cuda.empty_cache()
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, Ns),
                     dtype=torch.uint8, device=dev)
    y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    K, Wm = args.steps, args.warmup
    stats = torch.zeros(K, X.STATS_WORDS, dtype=torch.int32, device=dev)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(X.N_STAGES + 1)] for _ in range(K)]

    def forward(x_in, st=None, ev=None):
        if packed:
            X.xshare_moe_forward_packed(x_in, W_g, pk, w.k, w.budget, w.mode, prm, y, ws,
                                        shared=pshared, stats=st, stage_events=ev)
        else:
            X.xshare_moe_forward(x_in, W_g, Wg, Wu, Wd, w.k, w.budget, w.mode, prm, y, ws,
                                 stats=st, stage_events=ev, shared=shared)

    def step(i, st=None, ev=None):
        forward(xs_dev[i % N_ROTATE], st, ev)

    for i in range(Wm):
        step(i)
    torch.cuda.synchronize()

    # ---- timed region: device-resident inputs ----
    # Steps run back to back with no events between kernels (events would
    # serialise the programmatic launches); per-stage times come from a
    # second pass of K steps with stage events, right after.
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    with sampler:
        t0.record(stream)
        for i in range(K):
            step(i, stats[i])
        t1.record(stream)
        torch.cuda.synchronize()
        barrier(world)
        ms_local = t0.elapsed_time(t1)
        for i in range(K):
            step(i, None, events[i])
        torch.cuda.synchronize()
    ms_total = reduce_max(ms_local, world, dev)

    # The latency of one layer call: 20 single steps, each between its own
    # events with the device idle before it (no overlap with a previous
    # step), median.
    single_ms = []
    for i in range(N_SINGLE):
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_.record(stream)
        step(i)
        b_.record(stream)
        torch.cuda.synchronize()
        single_ms.append(a_.elapsed_time(b_))

    st = stats.cpu().numpy()
    if np.any(st[:, 5] != 0):
        raise RuntimeError(f"device status {st[:, 5].max()} (a bounded wait ran out)")
    stage_ms = {name: [] for name in X.STAGE_NAMES}
    for i in range(K):
        for s, name in enumerate(X.STAGE_NAMES):
            stage_ms[name].append(events[i][s].elapsed_time(events[i][s + 1]))
    n_used = st[:, 1].astype(np.float64)
    n_pairs = st[:, 4].astype(np.float64)
    mean_ms = {k: float(np.mean(v)) for k, v in stage_ms.items()}
    dominant = max(mean_ms, key=mean_ms.get)
    peaks = measured_peaks()

    # ---- algorithmic bytes and FLOPs ----
    ab = [algorithmic_bytes(w, int(n_used[i]), int(n_pairs[i]), Ns) for i in range(K)]
    dom_bytes = float(np.mean([a[dominant] for a in ab])) if dominant in ab[0] else None
    dom_ms = mean_ms[dominant]
    achieved = dom_bytes / (dom_ms * 1e-3) / 1e9 if dom_bytes else None
    layer_bytes = float(np.mean([a["layer"] for a in ab]))
    flops = float(np.mean(6 * w.d * w.F * (n_pairs + Ns * w.B) + 2 * w.B * w.N * w.d))
    step_s = ms_total / K * 1e-3
    t_roof = max(layer_bytes / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12))
    tokens_total = reduce_sum(w.B * K, world, dev)

    # ---- end to end: pinned host x in, y and stats out, every step ----
    x_pin = [x.pin_memory() for x in xs_host]
    y_pin = torch.empty(w.B, w.d, dtype=torch.bfloat16).pin_memory()
    st_pin = torch.empty(X.STATS_WORDS, dtype=torch.int32).pin_memory()
    x_in = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    st_dev = torch.zeros(X.STATS_WORDS, dtype=torch.int32, device=dev)

    def e2e_body(i):
        x_in.copy_(x_pin[i % N_ROTATE], non_blocking=True)
        forward(x_in, st_dev)
        y_pin.copy_(y, non_blocking=True)
        st_pin.copy_(st_dev, non_blocking=True)

    # By default each step replays a CUDA graph of the copy in, the forward
    # (the library's calls are capture-safe) and the copies out, one graph per
    # rotating input buffer, as a decode server would; --e2e-eager issues the
    # calls one by one every step.
    graphs = []
    if not args.e2e_eager:
        for i in range(Wm):
            e2e_body(i)
        torch.cuda.synchronize()
        for i in range(N_ROTATE):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, capture_error_mode="thread_local"):
                e2e_body(i)
            graphs.append(g)
        torch.cuda.synchronize()
        stream = torch.cuda.current_stream()

    def e2e_step(i):
        if graphs:
            graphs[i % N_ROTATE].replay()
        else:
            e2e_body(i)
        stream.synchronize()

    for i in range(Wm):
        e2e_step(i)
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(K):
        e2e_step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = reduce_max(e0.elapsed_time(e1), world, dev)

    # router, selection, [refinement: its own kernel beyond two 32-token
    # chunks], gather, gate/up, down, combine
    launches_per_step = X.N_STAGES - (1 if (w.B + 31) // 32 <= 2 else 0)
    out = {
        "metric": METRIC,
        "value": tokens_total / (ms_total * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": K,
        "warmup": Wm,
        "ms_per_step": ms_total / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": workload_config(w, Ns, world),
        "expert_weights": "packed 128 x 64 tiles (xshare_pack_experts, once at load)"
                          if packed else "plain [N, F, d] / [N, d, F] matrices",
        "weights_streamed_gb_per_step": layer_bytes / 1e9,
        "experts": {
            "selected_mean": float(st[:, 0].mean()), "used_mean": float(n_used.mean()),
            "union_topk_mean": float(st[:, 2].mean()), "max_group_load_mean": float(st[:, 3].mean()),
        },
        "layer": {
            "expert_weight_gbs": float(np.mean((n_used + Ns) * 6 * w.d * w.F)) / step_s / 1e9,
            "algorithmic_gbs": layer_bytes / step_s / 1e9,
            "roofline_frac": t_roof / step_s,
            "roofline_frac_vs_nominal_7900gbs": (layer_bytes / 7.9e12) / step_s,
            "peak_source": peaks["source"],
        },
        "stages_ms": {k: round(v, 5) for k, v in mean_ms.items()},
        "single_step_ms": {"median": float(np.median(single_ms)), "of": N_SINGLE,
                           "method": "events around each step, device idle before it"},
        "roofline": {
            "kernel": dominant,
            "bound": "hbm",
            "achieved": achieved,
            "peak": peaks["hbm_gbs"],
            "unit": "GB/s",
            "frac": (achieved / peaks["hbm_gbs"]) if achieved else None,
            "traffic": recorded_traffic(dominant, float(np.mean(n_used)) + Ns),
            "peak_source": f"{peaks['source']} (MEASURED_PEAKS.json hbm_gbs, copy)"
                           if peaks["source"] == "measured" else "fallback 6.8 TB/s",
        },
        "clocks": sampler.summary(),
        "e2e": {
            "value": tokens_total / (e2e_ms * 1e-3),
            "unit": "tokens/s",
            "h2d_bytes_per_step": w.B * w.d * 2,
            "d2h_bytes_per_step": w.B * w.d * 2 + X.STATS_WORDS * 4,
            "method": "CUDA-graph replay of copy in + xshare forward + copies out, host sync every step"
                      if graphs else "eager calls, host sync every step",
        },
        "gpu_launches": launches_per_step * K,
    }
    return out


def run_gpu_ep(args, w: W.Workload, rank: int, world: int, local: int) -> dict:
    """Expert parallelism over the ranks (Sec. 5): every rank holds the router
    and the packed weights of its N / world experts only; a step is one layer
    forward on one batch shared by all ranks (routing replicated, FFN over the
    rank's experts, NCCL all-reduce of the exchange buffer, combine)."""
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare as X

    if w.N % world != 0:
        raise SystemExit(f"--ep needs N % ranks == 0 (N = {w.N}, ranks = {world})")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(world, "nccl")
    stream = torch.cuda.current_stream()
    xs_host = [W.router_inputs(w, args.seed + i)[0] for i in range(N_ROTATE)]
    _, W_g = W.router_inputs(w, args.seed)
    xs_dev = [x.to(dev) for x in xs_host]
    W_g = W_g.to(dev)
    lo, hi = rank * (w.N // world), (rank + 1) * (w.N // world)
    full = X.Packed(*W.expert_weights(w, args.seed, device=str(dev)))
    pk = full.experts(lo, hi)                      # keep this rank's experts only
    pk.gate_up, pk.down = pk.gate_up.clone(), pk.down.clone()
    del full
    torch.cuda.empty_cache()
    Ns = args.shared
    pshared = X.Packed(*W.shared_expert_weights(w, Ns, args.seed, device=str(dev))) if Ns else None
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, Ns),
                     dtype=torch.uint8, device=dev)
    buf = X.ep_exchange_buffer(ws, w.B, w.N, w.k, w.d, w.F, w.mode, prm, Ns)
    y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    K, Wm = args.steps, args.warmup
    stats = torch.zeros(K, X.STATS_WORDS, dtype=torch.int32, device=dev)

    def step(x_in, st=None):
        X.xshare_moe_forward_ep(x_in, W_g, pk, w.k, w.budget, w.mode, prm, world, rank, ws,
                                shared=pshared, stats=st)
        if world > 1:
            torch.distributed.all_reduce(buf, op=torch.distributed.ReduceOp.SUM)
        X.xshare_ep_combine(ws, w.B, w.N, w.k, w.d, w.F, w.mode, prm, y, Ns)

    for i in range(Wm):
        step(xs_dev[i % N_ROTATE])
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    with sampler:
        t0.record(stream)
        for i in range(K):
            step(xs_dev[i % N_ROTATE], stats[i])
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms_total = reduce_max(t0.elapsed_time(t1), world, dev)
    st = stats.cpu().numpy()
    if np.any(st[:, 5] != 0):
        raise RuntimeError(f"device status {st[:, 5].max()} (a bounded wait ran out)")
    n_used, n_pairs = st[:, 1].astype(np.float64), st[:, 4].astype(np.float64)
    ab = [algorithmic_bytes(w, int(n_used[i]), int(n_pairs[i]), Ns) for i in range(K)]
    layer_bytes = float(np.mean([a["layer"] for a in ab]))
    peaks = measured_peaks()
    step_s = ms_total / K * 1e-3

    x_pin = [x.pin_memory() for x in xs_host]
    y_pin = torch.empty(w.B, w.d, dtype=torch.bfloat16).pin_memory()
    x_in = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)

    def e2e_step(i):
        x_in.copy_(x_pin[i % N_ROTATE], non_blocking=True)
        step(x_in)
        y_pin.copy_(y, non_blocking=True)
        stream.synchronize()

    for i in range(Wm):
        e2e_step(i)
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(K):
        e2e_step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = reduce_max(e0.elapsed_time(e1), world, dev)
    launches = 7 - (1 if (w.B + 31) // 32 <= 2 else 0)
    return {
        "metric": METRIC, "value": w.B * K / (ms_total * 1e-3), "unit": "tokens/s",
        "n_gpus": world, "steps": K, "warmup": Wm, "ms_per_step": ms_total / K,
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": dict(workload_config(w, Ns, 1),
                       parallelism=f"expert parallel x{world} (N / {world} experts per GPU)"),
        "experts": {"selected_mean": float(st[:, 0].mean()), "used_mean": float(n_used.mean()),
                    "union_topk_mean": float(st[:, 2].mean()),
                    "max_group_load_mean": float(st[:, 3].mean())},
        "layer": {"roofline_frac": layer_bytes / world / (peaks["hbm_gbs"] * 1e9) / step_s,
                  "note": "per-GPU share of the layer's bytes (balanced groups assumed)",
                  "peak_source": peaks["source"]},
        "roofline": {"kernel": "layer (expert-parallel step)", "bound": "hbm",
                     "achieved": layer_bytes / world / step_s / 1e9, "peak": peaks["hbm_gbs"],
                     "unit": "GB/s", "frac": layer_bytes / world / step_s / 1e9 / peaks["hbm_gbs"],
                     "traffic": None},
        "clocks": sampler.summary(),
        "e2e": {"value": w.B * K / (e2e_ms * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": w.B * w.d * 2, "d2h_bytes_per_step": w.B * w.d * 2},
        "gpu_launches": launches * K,
    }


def parse_sweep(specs) -> list:
    """[(field, [values])] from FIELD=V1,V2 strings; values typed by the field."""
    out = []
    for spec in specs:
        field, _, vals = spec.partition("=")
        if field not in ("B", "budget", "k0", "m_r", "m_g", "tau", "mode", "tokens_per_request",
                         "sparse_scores") or not vals:
            raise SystemExit(f"bad --sweep {spec!r}")
        conv = float if field == "tau" else (lambda v: W.MODES[v] if v in W.MODES else int(v)) \
            if field == "mode" else int
        out.append((field, [conv(v) for v in vals.split(",")]))
    return out


def run_sweep(args, w0: W.Workload) -> list:
    """Sweep mode (one GPU): for every seed the expert weights are drawn and
    packed once; every combination of the swept fields is timed like the
    headline (back-to-back steps, CUDA events, rotating inputs) and reported
    with the median over the seeds."""
    import itertools
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare as X

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    fields = parse_sweep(args.sweep)
    combos = [dict(zip([f for f, _ in fields], vals))
              for vals in itertools.product(*[v for _, v in fields])]
    seeds = [int(v) for v in args.seeds.split(",")]
    peaks = measured_peaks()
    K, Wm = args.steps, args.warmup
    res = {i: [] for i in range(len(combos))}
    for seed in seeds:
        pk = X.Packed(*W.expert_weights(w0, seed, device=str(dev)))
        torch.cuda.empty_cache()
        for i, kw in enumerate(combos):
            w = w0.with_(**kw)
            # Seed 0 uses the headline's input batches (0 .. N_ROTATE - 1).
            xs = [W.router_inputs(w, 101 * seed + j)[0].to(dev) for j in range(N_ROTATE)]
            W_g = W.router_inputs(w, seed)[1].to(dev)
            prm = X.route_params(**w.params())
            ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, 0),
                             dtype=torch.uint8, device=dev)
            y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
            st = torch.zeros(K, X.STATS_WORDS, dtype=torch.int32, device=dev)

            def step(j, stats=None):
                X.xshare_moe_forward_packed(xs[j % N_ROTATE], W_g, pk, w.k, w.budget, w.mode, prm, y,
                                            ws, stats=stats)
            for j in range(Wm):
                step(j)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for j in range(K):
                step(j, st[j])
            e1.record()
            torch.cuda.synchronize()
            s = st.cpu().numpy()
            if np.any(s[:, 5] != 0):
                raise RuntimeError("device status: a bounded wait ran out")
            lb = float(np.mean([algorithmic_bytes(w, int(s[j, 1]), int(s[j, 4]))["layer"] for j in range(K)]))
            ms = e0.elapsed_time(e1) / K
            res[i].append({"ms": ms, "S": float(s[:, 0].mean()), "U": float(s[:, 1].mean()),
                           "union": float(s[:, 2].mean()), "maxload": float(s[:, 3].mean()),
                           "roofline": lb / (peaks["hbm_gbs"] * 1e9) / (ms * 1e-3)})
        del pk
        torch.cuda.empty_cache()
    lines = []
    for i, kw in enumerate(combos):
        w = w0.with_(**kw)
        med = {key: float(np.median([r[key] for r in res[i]])) for key in res[i][0]}
        lines.append({"sweep": describe(w), "fields": kw, "seeds": seeds, "steps": K,
                      "ms_per_step_median": med["ms"], "ms_per_step": [r["ms"] for r in res[i]],
                      "tokens_per_s_median": w.B / (med["ms"] * 1e-3),
                      "roofline_frac_median": med["roofline"],
                      "experts_median": {"selected": med["S"], "used": med["U"],
                                         "union_topk": med["union"], "max_group_load": med["maxload"]},
                      "peak_source": peaks["source"]})
    return lines


def run_gpu_stack(args, w: W.Workload, rank: int, world: int, local: int) -> dict:
    """L residual layers (xshare_stack_graph_*): one step = one graph replay."""
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare as X

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    init_dist(world, "nccl")
    stream = torch.cuda.current_stream()
    L, P = args.layers, max(1, min(args.weight_sets, args.layers))
    K_total = args.global_budget if args.global_budget is not None else L * w.budget
    Ns = args.shared
    sets = [W.expert_weights(w, args.seed + 10 * s, device=str(dev), down_std=W.STACK_DOWN_STD)
            for s in range(P)]
    shared = [W.shared_expert_weights(w, Ns, args.seed + 10 * s, device=str(dev),
                                      down_std=W.STACK_DOWN_STD) if Ns else None
              for s in range(P)]
    if not args.unpacked:  # packed once at load, outside the timed region
        sets = [X.Packed(*ws) for ws in sets]
        shared = [X.Packed(*sh) if sh is not None else None for sh in shared]
        torch.cuda.empty_cache()
    layers = []
    for l in range(L):
        _, W_g = W.router_inputs(w, args.seed + 1000 + l)
        if args.unpacked:
            layers.append((W_g.to(dev),) + tuple(sets[l % P]) + (shared[l % P],))
        else:
            layers.append((W_g.to(dev), sets[l % P], shared[l % P]))
    x_host = W.router_inputs(w, args.seed + 101 * rank)[0]
    x = x_host.to(dev)
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, Ns),
                     dtype=torch.uint8, device=dev)
    h = torch.empty(L, w.B, w.d, dtype=torch.bfloat16, device=dev)
    st = torch.zeros(L, X.STATS_WORDS, dtype=torch.int32, device=dev)
    g = X.StackGraph(x, layers, w.k, K_total, w.mode, prm, h, ws, stats=st)
    K, Wm = args.steps, args.warmup
    for _ in range(Wm):
        g.launch(stream)
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    with sampler:
        t0.record(stream)
        for _ in range(K):
            g.launch(stream)
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms_total = reduce_max(t0.elapsed_time(t1), world, dev)
    s = st.cpu().numpy()
    if np.any(s[:, 5] != 0):
        raise RuntimeError(f"device status {s[:, 5].max()} (a bounded wait ran out)")
    n_used, n_pairs = s[:, 1], s[:, 4]
    ab = [algorithmic_bytes(w, int(n_used[l]), int(n_pairs[l]), Ns) for l in range(L)]
    stack_bytes = float(sum(a["layer"] for a in ab))
    flops = float(sum(6 * w.d * w.F * (n_pairs[l] + Ns * w.B) + 2 * w.B * w.N * w.d
                      for l in range(L)))
    peaks = measured_peaks()
    step_s = ms_total / K * 1e-3
    t_roof = max(stack_bytes / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12))
    tokens_total = reduce_sum(w.B * K, world, dev)

    # end to end: x from pinned host memory in, the last layer's output out, every step
    x_pin = x_host.pin_memory()
    y_pin = torch.empty(w.B, w.d, dtype=torch.bfloat16).pin_memory()

    def e2e_step():
        x.copy_(x_pin, non_blocking=True)
        g.launch(stream)
        y_pin.copy_(h[L - 1], non_blocking=True)
        stream.synchronize()

    for _ in range(Wm):
        e2e_step()
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = reduce_max(e0.elapsed_time(e1), world, dev)
    g.close()
    launches_per_layer = X.N_STAGES - (1 if (w.B + 31) // 32 <= 2 else 0)
    achieved = stack_bytes / step_s / 1e9
    return {
        "metric": METRIC,
        "value": tokens_total / (ms_total * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world, "steps": K, "warmup": Wm,
        "ms_per_step": ms_total / K,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {
            "workload": f"{describe(w, Ns)}; stack of {L} residual layers (x + MoE(x)), "
                        f"global budget K={K_total} (m_l = K/L), {P} expert-weight sets, "
                        "one CUDA-graph replay per step",
            "B": w.B, "N": w.N, "k": w.k, "d": w.d, "F": w.F, "layers": L, "weight_sets": P,
            "expert_weights": "plain matrices" if args.unpacked else "packed tiles",
            "global_budget": K_total, "shared_experts": Ns, "global_batch": w.B * world,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": f"inputs larger than L2: ~{stack_bytes / 1e9:.1f} GB of expert weights per step",
        },
        "experts": {"selected_per_layer": [int(v) for v in s[:, 0]],
                    "used_per_layer": [int(v) for v in n_used],
                    "union_topk_per_layer": [int(v) for v in s[:, 2]]},
        "layer": {"roofline_frac": t_roof / step_s, "algorithmic_gbs": achieved,
                  "peak_source": peaks["source"]},
        "roofline": {"kernel": "stack (whole graph replay)", "bound": "hbm", "achieved": achieved,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                     "traffic": None},
        "clocks": sampler.summary(),
        "e2e": {"value": tokens_total / (e2e_ms * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": w.B * w.d * 2, "d2h_bytes_per_step": w.B * w.d * 2},
        "gpu_launches": launches_per_layer * L * K,
    }


# --------------------------------------------------------------------------- oracle timing

class OracleStep:
    """One whole layer step of the CPU oracle on workload `w`: router logits,
    softmax, selection (Algorithms 2-6), refinement, permutation, the expert
    FFN of every routed (token, slot) pair on all F hidden units, the shared
    experts and the weighted combine, for all B tokens of one input batch, in
    fp64 with numpy.  The inputs and the bf16 weights of the experts this
    batch uses are drawn once, outside the timed calls; the oracle widens them
    to fp64 inside every step, as it stands."""

    def __init__(self, w: W.Workload, seed: int, n_shared: int = 0):
        from oracle import xshare_oracle as O
        self.O, self.w, self.n_shared = O, w, n_shared
        x, W_g = W.router_inputs(w, seed)
        self.xb, self.W_g = W.bf16_bits(x), W_g.numpy()
        p = O.softmax_scores(O.router_logits(self.xb, self.W_g))
        r = O.route(p, w.k, w.budget, w.mode, **w.params())
        self.experts = sorted(int(e) for e in r["used"])
        self.weights = {}
        if self.experts:
            Wg, Wu, Wd = W.expert_weights(w, seed, device="cpu", experts=self.experts)
            for i, e in enumerate(self.experts):
                self.weights[e] = (W.bf16_bits(Wg[i]), W.bf16_bits(Wu[i]), W.bf16_bits(Wd[i]))
            del Wg, Wu, Wd
        self.shared = []
        if n_shared:
            Sg, Su, Sd = W.shared_expert_weights(w, n_shared, seed, device="cpu")
            self.shared = [(W.bf16_bits(Sg[j]), W.bf16_bits(Su[j]), W.bf16_bits(Sd[j]))
                           for j in range(n_shared)]

    def step(self) -> float:
        """Runs one step; returns its wall-clock seconds."""
        O, w = self.O, self.w
        t0 = time.perf_counter()
        r = O.moe_forward(self.xb, self.W_g, self.weights.__getitem__, w.k, w.budget, w.mode,
                          get_shared=self.shared.__getitem__ if self.n_shared else None,
                          n_shared=self.n_shared, **w.params())
        dt = time.perf_counter() - t0
        assert r["y"].shape == (w.B, w.d)
        return dt

    def describe(self) -> str:
        sh = f" and {self.n_shared} shared" if self.n_shared else ""
        return (f"full layer steps on one {self.w.B}-token batch: router, softmax, selection, "
                f"refinement, permutation, SwiGLU FFN of all {self.w.B} tokens over its "
                f"{len(self.experts)} used experts{sh} on all {self.w.F} hidden units, combine; "
                f"numpy fp64, 1 thread")


def cpu_baseline(w: W.Workload, seed: int, n_shared: int = 0, steps: int = 2) -> dict:
    """The oracle, single-threaded, timed over `steps` whole layer steps after
    one untimed step, in a child process so that BLAS is pinned to one thread."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    kw = json.dumps(dict(B=w.B, N=w.N, F=w.F, budget=w.budget, k0=w.k0, mode=w.mode, tau=w.tau,
                         sparse_scores=w.sparse_scores, m_r=w.m_r, m_g=w.m_g))
    code = (f"import sys, json; sys.path.insert(0, {ROOT!r}); import torch; torch.set_num_threads(1); "
            f"import bench; from paper_2602_07265_gb300 import workloads as W; "
            f"w = W.WORKLOADS[{w.name!r}].with_(**{kw}); "
            f"o = bench.OracleStep(w, {seed}, {int(n_shared)}); o.step(); "
            f"t = [o.step() for _ in range({int(steps)})]; "
            f"print(json.dumps(dict(t=t, describe=o.describe())))")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=1800)
    if r.returncode != 0:
        tail = r.stderr.strip().splitlines()[-1][:200] if r.stderr.strip() else "no output"
        return {"value": None, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                "sample": "failed: " + tail}
    s = json.loads(r.stdout.strip().splitlines()[-1])
    mean_s = float(np.mean(s["t"]))
    return {"value": w.B / mean_s, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"{len(s['t'])} timed {s['describe']} (mean {mean_s:.2f} s per step)"}


def run_reference(args, w: W.Workload, rank: int, world: int) -> dict:
    """The oracle as the reference arm: W untimed and K timed whole layer steps
    of the same workload (one input batch), single-threaded on the host
    cores; ms_per_step is the measured mean of the K steps."""
    torch.set_num_threads(1)
    K, Wm = args.steps, args.warmup
    oracle = OracleStep(w, args.seed, args.shared)
    for _ in range(Wm):
        oracle.step()
    times = [oracle.step() for _ in range(K)]
    mean_s = float(np.mean(times))
    value = w.B / mean_s
    sample = f"{K} timed {oracle.describe()} (median {1e3 * float(np.median(times)):.0f} ms)"
    return {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": Wm, "ms_per_step": 1e3 * mean_s, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "impl": "reference",
        "config": workload_config(w, args.shared, world),
        "runs_on": "host cores, rank 0 only",
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    args = parse_args(argv)
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    w = workload_from_args(args)
    rank, world, local = dist_env()
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(run_reference(args, w, rank, world)))
        return 0
    if args.sweep:
        if world > 1:
            raise SystemExit("sweep mode runs on one GPU")
        for line in run_sweep(args, w):
            print(json.dumps(line), flush=True)
        return 0
    if args.ep:
        out = run_gpu_ep(args, w, rank, world, local)
        if rank == 0:
            print(json.dumps(out))
        if world > 1:
            torch.distributed.destroy_process_group()
        return 0
    if args.layers > 1:
        out = run_gpu_stack(args, w, rank, world, local)
        if rank == 0:
            print(json.dumps(out))
        if world > 1:
            torch.distributed.destroy_process_group()
        return 0
    out = run_gpu(args, w, rank, world, local)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            out["cpu_baseline"] = cpu_baseline(w, args.seed, args.shared)
        print(json.dumps(out))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
