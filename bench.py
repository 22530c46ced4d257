#!/usr/bin/env python3
"""Benchmark of the VisionPulse pruned decode step on GB300.

Workload (default): a Qwen2.5-VL-7B-shaped decoder, 28 layers of 28 query /
4 kv heads, head_dim 128, bf16 caches, batch 1, 1296 visual + 2561 text
tokens (512 prompt + 2048 generated + the current token) at the first step,
one text token appended per step.  A step is one vp_decode_step call per
layer (28 calls, each layer acting as its own anchor layer), i.e. the whole
five-stage hot path over every layer.

Prints one JSON line (rank 0).  `value` is decode steps per second with the
caches resident in HBM (per-step CUDA graphs of the 28 calls, timed with CUDA
events); `e2e` is the same metric through the C ABI with the step's query and
appended K/V copied in from pinned host memory and the results copied back.
`--impl reference` times the CPU oracle instead (rank 0, host cores).
"""

from __future__ import annotations

import argparse
import ctypes
import dataclasses
import hashlib
import json
import math
import multiprocessing as mp
import os
import statistics
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

ANCHOR_LAYER = 16  # 0-based index of the anchor layer l_a = 17 (Sec. 5.1)
METRIC = "pruned decode-attention steps/sec and achieved HBM GB/s (% of GB300 peak) on 1 GPU"
UNIT = "steps/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None, help="timed steps (default: the workload's)")
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--workload", default="qwen7b",
                    help="qwen7b (default) | qwen7b-10pct | qwen7b-anchor | qwen7b-fastv-vp | serving | long | "
                         "sweep-<N_v>-<r1|r5|r20|r50|adaptive>")
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle CPU-baseline leg")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU-baseline sample budget")
    ap.add_argument("--layer-calls", type=int, default=0,
                    help="profiling aid: N calls on one layer of the workload, no timing")
    ap.add_argument("--flush-l2", action="store_true", help="with --layer-calls: flush L2 before every call")
    return ap.parse_args(argv)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(x, world, device):
    """The largest value of x over all ranks (x itself with one rank): every
    replica's timed region is bracketed by barriers and the slowest one sets
    the job's time."""
    if world <= 1:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, steps, seconds):
    """Whole-job steps/s of `world` replicas that each ran `steps` steps in
    (at most) `seconds`."""
    return world * steps / seconds


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# --------------------------------------------------------------- algorithmic bytes

def call_bytes(r, n_visual, text_len, kept):
    """Algorithmic HBM bytes of one layer call for one sequence, split by kernel:
    score reads all visual K, text K and V and q; gather reads the kept visual
    V rows and writes out."""
    esz = 2 if r.dtype == "bf16" else 4
    row = r.kv_heads * r.head_dim * esz
    qo = r.heads * r.head_dim * esz
    score = n_visual * row + 2 * text_len * row + qo
    gather = kept * row + qo
    return score, gather


# ------------------------------------------------------------------ clock sampling

class ClockSampler:
    """Samples the SM clock and the clock-event (throttle) reasons through NVML
    in a background thread while the timed region runs."""

    REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
               0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
               0x100: "display_clock_setting"}

    def __init__(self, torch_device, interval=0.002):
        self.interval = interval
        self.samples = []
        self.err = None
        self.h = None
        try:
            self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nvml.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            import torch
            p = torch.cuda.get_device_properties(torch_device)
            bus = f"{getattr(p, 'pci_domain_id', 0):08x}:{p.pci_bus_id:02x}:{p.pci_device_id:02x}.0".encode()
            h = ctypes.c_void_p()
            if self.nvml.nvmlDeviceGetHandleByPciBusId_v2(ctypes.c_char_p(bus), ctypes.byref(h)) != 0:
                if self.nvml.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(h)) != 0:
                    raise OSError("no NVML handle")
            self.h = h
            mx = ctypes.c_uint(0)
            self.nvml.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx))
            self.max_mhz = mx.value
            fn = getattr(self.nvml, "nvmlDeviceGetCurrentClocksEventReasons", None)
            self.reasons_fn = fn or self.nvml.nvmlDeviceGetCurrentClocksThrottleReasons
        except Exception as e:  # NVML is optional: report why clocks are missing
            self.err = str(e)
        self._stop = threading.Event()
        self._t = None

    def _loop(self):
        clk = ctypes.c_uint(0)
        rs = ctypes.c_ulonglong(0)
        while not self._stop.is_set():
            if self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(clk)) == 0 and \
                    self.reasons_fn(self.h, ctypes.byref(rs)) == 0:
                self.samples.append((clk.value, rs.value))
            time.sleep(self.interval)

    def start(self):
        if self.h is not None:
            self._t = threading.Thread(target=self._loop, daemon=True)
            self._t.start()

    def stop(self):
        if self._t is None:
            return {"error": self.err or "NVML unavailable"}
        self._stop.set()
        self._t.join()
        return self.summarize(self.samples, self.max_mhz)

    @classmethod
    def summarize(cls, samples, max_mhz):
        """(SM MHz, reason bits) samples -> the JSON `clocks` object: the median
        clock and the union of the active reasons over the samples taken while
        the GPU was busy (all samples if it never was)."""
        busy = [s for s in samples if not (s[1] & 0x1)] or samples
        seen = 0
        for _, r in busy:
            seen |= r
        names = [n for bit, n in cls.REASONS.items() if seen & bit and bit != 0x1]
        return {"sm_mhz": statistics.median(c for c, _ in busy) if busy else None,
                "sm_max_mhz": max_mhz, "reasons": names, "samples": len(busy),
                "source": "NVML, 2 ms sampling during the timed region"}


# --------------------------------------------------------------------- oracle legs

def _oracle_worker(args):
    """Runs in a spawned process with single-threaded BLAS: times the oracle
    on a sample of layer calls; returns seconds per layer call."""
    recipe_name, layers, steps0, budget_s, max_calls = args
    from paper_2605_31457_gb300 import workloads as W
    from oracle import vp_oracle as O
    r = getattr(W, recipe_name)
    t_cap = r.capacity(steps0 + max_calls + 1)
    times = []
    cache = {}
    t_start = time.perf_counter()
    for n in range(max_calls):
        layer = layers[n % len(layers)]
        if layer not in cache:
            li = W.make_layer(r, layer, t_cap=t_cap)
            q = W.make_queries(r, layer, li, steps=steps0 + max_calls + 1)
            cache[layer] = (W.round_to(li.k, r.dtype).double().numpy(),
                            W.round_to(li.v, r.dtype).double().numpy(),
                            W.round_to(q, r.dtype).double().numpy())
        k, v, q = cache[layer]
        s = steps0 + n
        t0 = time.perf_counter()
        for b in range(r.batch):
            O.decode_step(q[s, b], k[b], v[b], int(r.vis_starts[b]), int(r.vis_lens[b]),
                          int(r.text_lens[b]) + s, **r.budget)
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s:
            break
    return times


def oracle_times(recipe_name, layers, steps0, budget_s, max_calls):
    env_keys = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")
    old = {k: os.environ.get(k) for k in env_keys}
    for k in env_keys:
        os.environ[k] = "1"
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(1) as pool:
            return pool.apply(_oracle_worker, ((recipe_name, layers, steps0, budget_s, max_calls),))
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    from paper_2605_31457_gb300 import workloads as W
    r = W.QWEN7B
    n = args.warmup + args.steps
    times = oracle_times("QWEN7B", list(range(4)), 0, budget_s=1e9, max_calls=n)
    timed = times[args.warmup:]
    per_call = sum(timed) / len(timed)
    ms_step = per_call * r.layers * 1e3
    value = 1e3 / ms_step
    sample = (f"each step = 1 of the {r.layers} layer calls of a decode step (layers 0-3 in turn), "
              f"scaled x{r.layers} to a full step; {len(timed)} timed calls")
    line = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(r),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def workload_config(r, nbuf=None):
    import numpy as np
    bd = r.budget
    if bd.get("mode", 0) == 0:
        btxt = f"adaptive tau={bd['tau']} clamp [{bd['r_lo_ppm'] / 1e4:g}%, {bd['r_hi_ppm'] / 1e4:g}%]"
    else:
        btxt = f"fixed ratio {bd['ratio_ppm'] / 1e4:g}%"
    tl = r.text_lens
    text = f"{int(tl[0])}" if len(set(tl.tolist())) == 1 else f"{int(tl.min())}-{int(tl.max())}"
    layout = f", paged (page {r.page_size})" if r.paged else ""
    nb = r.layers if nbuf is None else nbuf
    step_bytes = r.layers * r.batch * r.kv_heads * r.head_dim * (2 if r.dtype == "bf16" else 4) * \
        float(np.mean(r.vis_lens + 2 * r.text_lens))
    return {"workload": (f"{r.name}: {r.layers} layers x {r.heads} q / {r.kv_heads} kv heads, "
                         f"head_dim {r.head_dim}, {r.dtype}{layout}, batch {r.batch}, "
                         f"{int(r.vis_lens[0])} visual + {text} text tokens at step 0 "
                         f"(+1 text token per step), budget {btxt}"),
            "global_batch": r.batch, "layers": r.layers, "distinct_layer_caches": nb,
            "l2": f"no flush: each step streams ~{step_bytes / 1e9:.2f} GB of K/V; every layer call's "
                  f"cache is distinct from the previous one's and the per-step stream exceeds the 129 MB L2"}


# ------------------------------------------------------------------------ our arm

def pick_workload(name):
    """(recipe, default timed steps, distinct layer caches, host-generated)."""
    from paper_2605_31457_gb300 import workloads as W
    if name in ("qwen7b", "qwen7b-anchor", "qwen7b-fastv-vp"):
        return W.QWEN7B, 256, W.QWEN7B.layers, True
    if name == "qwen7b-10pct":  # the paper's 10% setting: tau = 0.4, clamp [5%, 10%]
        return dataclasses.replace(W.QWEN7B, budget=W.ADAPTIVE_10PCT), 256, W.QWEN7B.layers, True
    if name == "serving":
        return W.SERVING, 64, 4, False
    if name == "long":
        return W.LONG, 64, 4, False
    if name.startswith("sweep-"):
        _, nv, bname = name.split("-")
        budgets = {"r1": W.SWEEP_BUDGETS[0], "r5": W.SWEEP_BUDGETS[1], "r20": W.SWEEP_BUDGETS[2],
                   "r50": W.SWEEP_BUDGETS[3], "adaptive": W.SWEEP_BUDGETS[4]}
        return W.sweep_recipe(int(nv), budgets[bname]), 16, 1, False
    raise SystemExit(f"unknown workload {name}")


def run_ours(args, rank, world, local):
    import numpy as np
    import torch
    from paper_2605_31457_gb300 import build as _build
    _build.ensure_built()
    from paper_2605_31457_gb300 import vp, workloads as W

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    r, default_steps, nbuf, host_gen = pick_workload(args.workload)
    if args.steps is None:
        args.steps = default_steps
    L, B, H, Hkv, D = r.layers, r.batch, r.heads, r.kv_heads, r.head_dim
    S = args.warmup + args.steps
    t_cap = r.capacity(S + 1)
    nvs, tls = r.vis_lens.astype(np.int64), r.text_lens.astype(np.int64)
    nv_max = int(nvs.max())
    cdt = torch.bfloat16 if r.dtype == W.BF16 else torch.float32

    # Inputs: `nbuf` distinct layer caches (layer l reads cache l % nbuf; every
    # layer call's working set is far larger than L2) and per-(step, layer)
    # queries.  The default workload is drawn on the host (the generator the
    # parity tests use); the large ones on the device, same recipe.
    ks, vs_ = [], []
    q_dev = torch.empty((S, L, B, H, D), dtype=cdt, device=dev)
    focus = []
    for u in range(nbuf):
        if host_gen:
            li = W.make_layer(r, u, t_cap=t_cap)
            ks.append(W.round_to(li.k, r.dtype).to(dev))
            vs_.append(W.round_to(li.v, r.dtype).to(dev))
            focus.append(li)
        else:
            k, v, f, sk = W.make_layer_torch(r, u, t_cap, dev)
            ks.append(k)
            vs_.append(v)
            focus.append((f, sk))
    for layer in range(L):
        u = layer % nbuf
        if host_gen:
            q_dev[:, layer] = W.round_to(W.make_queries(r, layer, focus[u], steps=S), r.dtype).to(dev)
        else:
            q_dev[:, layer] = W.make_queries_torch(r, layer, S, focus[u][0], focus[u][1], dev)
    if r.paged:
        bt_np, n_pages, max_pages = W.page_table(B, t_cap, r.page_size, r.seed)
        bt = torch.from_numpy(bt_np).to(dev)
        ks = [W.scatter_pages(k, bt_np, n_pages, r.page_size) for k in ks]
        vs_ = [W.scatter_pages(v, bt_np, n_pages, r.page_size) for v in vs_]
        kc = [vp.kv_paged(k, bt) for k in ks]
        vc = [vp.kv_paged(v, bt) for v in vs_]
    else:
        kc = [vp.kv_contiguous(k) for k in ks]
        vc = [vp.kv_contiguous(v) for v in vs_]
    torch.cuda.synchronize()
    vis_start = torch.tensor(r.vis_starts, dtype=torch.int32, device=dev)
    vis_len = torch.tensor(r.vis_lens, dtype=torch.int32, device=dev)
    tl_steps = (torch.tensor(r.text_lens, dtype=torch.int32)[None, :] + torch.arange(S, dtype=torch.int32)[:, None]).to(dev)
    span = vp.span(vis_start, vis_len)
    budget = vp.make_budget(**r.budget)
    cfg = vp.make_config(B, H, Hkv, D, nv_max, int((nvs + tls).max()) + S, 
                         vp.VP_BF16 if r.dtype == W.BF16 else vp.VP_FP32, int(r.paged), r.page_size)
    ctx = vp.vp_init(cfg)
    cap = max(1, vp.vp_max_kept(budget, nv_max))
    out = torch.empty((L, B, H, D), dtype=cdt, device=dev)
    kept = torch.empty((L, B, cap), dtype=torch.int32, device=dev)
    count = torch.zeros((S, L, B), dtype=torch.int32, device=dev)
    mass = torch.empty((L, B, H), dtype=torch.float32, device=dev)
    stats = torch.empty((S, L, B, 4), dtype=torch.float32, device=dev)

    # qwen7b-anchor: the anchor-layer pipeline of the paper's FastV-VP setting
    # (Sec. 5.1, l_a = 17): layers 1-16 attend densely (the whole visual span
    # kept), layer 17 runs the VisionPulse step, layers 18-28 reuse its kept
    # set.  Every other workload treats each layer as its own anchor.
    anchor = ANCHOR_LAYER if args.workload.endswith(("-anchor", "-fastv-vp")) else None
    if anchor is not None:
        kept_all = torch.arange(nv_max, dtype=torch.int32, device=dev)[None, :].repeat(B, 1).contiguous()
        count_all = vis_len.clone()
    # qwen7b-fastv-vp: FastV at the prefill stage (the paper's appendix on
    # prefill pruning: ratio 0.5 at the pruning layer, ranked by the last
    # prompt token's head-averaged attention -- Eq. 2 with that query), then
    # the anchor pipeline over the survivors: layers from the anchor on read
    # caches compacted to the surviving visual tokens.  The prefill stage runs
    # once, before the timed decode, and is timed on its own.
    fastv = args.workload.endswith("-fastv-vp")
    kc_run, vc_run, span_run = list(kc), list(vc), [span] * L
    prefill_ms = None
    if fastv:
        fv_budget = vp.make_budget(mode=vp.VP_FIXED_RATIO, tau=0.1, ratio_ppm=500_000)
        fv_cap = max(1, vp.vp_max_kept(fv_budget, nv_max))
        fv_kept = torch.empty((B, fv_cap), dtype=torch.int32, device=dev)
        fv_count = torch.empty((B,), dtype=torch.int32, device=dev)
        fv_out = torch.empty((B, H, D), dtype=cdt, device=dev)
        fv_mass = torch.empty((B, H), dtype=torch.float32, device=dev)
        tl_all = tl_steps[S - 1]  # every row a decode step will read, appended tokens included
        comp = []
        for layer in range(anchor, L):
            shape = (B, Hkv, t_cap, D)
            comp.append((torch.zeros(shape, dtype=cdt, device=dev), torch.zeros(shape, dtype=cdt, device=dev)))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        # The last prompt token's query at the pruning layer: the recipe's
        # query for that layer (step 0), before any decode token.
        vp.vp_decode_step(ctx, B, q_dev[0, anchor], kc[anchor % nbuf], vc[anchor % nbuf], span, tl_steps[0],
                          fv_budget, fv_out, fv_kept, fv_cap, fv_count, fv_mass)
        for i, layer in enumerate(range(anchor, L)):
            for src, dst in ((kc[layer % nbuf], comp[i][0]), (vc[layer % nbuf], comp[i][1])):
                vp.vp_compact_kv(ctx, B, src, vp.kv_contiguous(dst), span, tl_all, fv_kept, fv_cap, fv_count)
        e1.record()
        torch.cuda.synchronize()
        prefill_ms = e0.elapsed_time(e1)
        vp.vp_check_errors(ctx)
        span_c = vp.span(vis_start, fv_count)
        for i, layer in enumerate(range(anchor, L)):
            kc_run[layer], vc_run[layer] = vp.kv_contiguous(comp[i][0]), vp.kv_contiguous(comp[i][1])
            span_run[layer] = span_c
        nvs_surv = fv_count.cpu().numpy().astype(np.int64)

    def step_calls(s, stream=None):
        for layer in range(L):
            kcl = kc_run[layer] if fastv else kc[layer % nbuf]
            vcl = vc_run[layer] if fastv else vc[layer % nbuf]
            spl = span_run[layer]
            if anchor is not None and layer < anchor:
                vp.vp_decode_gather(ctx, B, q_dev[s, layer], kcl, vcl, spl, tl_steps[s], kept_all, nv_max,
                                    count_all, out[layer], stream=stream)
            elif anchor is not None and layer > anchor:
                vp.vp_decode_gather(ctx, B, q_dev[s, layer], kcl, vcl, spl, tl_steps[s], kept[anchor], cap,
                                    count[s, anchor], out[layer], stream=stream)
            else:
                vp.vp_decode_step(ctx, B, q_dev[s, layer], kcl, vcl, spl, tl_steps[s], budget,
                                  out[layer], kept[layer], cap, count[s, layer], mass[layer], stats[s, layer],
                                  stream=stream)

    # One eager step loads the kernels.  Two sets of per-step CUDA graphs: the
    # first, without timing events, gives `value` (kernels chain through
    # programmatic dependent launch); the second records the library's stage
    # events around every kernel (which serialises the launches) and gives the
    # per-kernel device times for the roofline.
    step_calls(0)
    vp.vp_check_errors(ctx)
    cap_stream = torch.cuda.Stream(device=dev)

    def capture():
        gs = []
        for s in range(S):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=cap_stream):
                step_calls(s)
            gs.append(g)
        torch.cuda.synchronize()
        return gs

    graphs = capture()
    vp.vp_timing_enable(ctx, S * L)
    graphs_timed = capture()

    def timed_region(gs, sample_clocks):
        for s in range(args.warmup):
            gs[s].replay()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        sampler = ClockSampler(dev) if sample_clocks else None
        if sampler:
            sampler.start()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        ev0.record()
        for s in range(args.warmup, S):
            gs[s].replay()
        ev1.record()
        torch.cuda.synchronize()
        clk = sampler.stop() if sampler else None
        el = max_over_ranks(ev0.elapsed_time(ev1), world, dev)
        if world > 1:
            torch.distributed.barrier()
        return el, clk

    elapsed_ms, clocks = timed_region(graphs, True)
    timed_ms, _ = timed_region(graphs_timed, False)
    vp.vp_check_errors(ctx)

    # Per-stage device times of the second pass (events recorded on the calls' stream).
    per_step = L if anchor is None else 1   # vp_decode_step calls per step (the timed ones)
    stage = vp.vp_timing_read(ctx, S * L)[args.warmup * per_step:]
    counts = count.cpu().numpy()
    score_bytes = gather_bytes = other_bytes = 0
    for s in range(args.warmup, S):
        for layer in range(L):
            for b in range(B):
                if anchor is None or layer == anchor:
                    nv_read = int(nvs_surv[b]) if fastv else int(nvs[b])  # the anchor's visual span
                    a, c = call_bytes(r, nv_read, int(tls[b]) + s, int(counts[s, layer, b]))
                    score_bytes += a
                    gather_bytes += c
                else:  # the visual rows read: all of them before the anchor, the kept ones after
                    nkv = int(nvs[b]) if layer < anchor else int(counts[s, anchor, b])
                    a, c = call_bytes(r, 0, int(tls[b]) + s, 0)
                    other_bytes += a + c + 2 * nkv * r.kv_heads * r.head_dim * 2
    n_calls = args.steps * per_step
    score_ms = sum(x[0] for x in stage)
    select_ms = sum(x[1] for x in stage)
    gather_ms = sum(x[2] for x in stage)
    peak, peak_src = measured_peaks()
    achieved = score_bytes / (score_ms * 1e-3) / 1e9
    traffic = committed_traffic()
    ms_per_step = elapsed_ms / args.steps
    value = job_rate(world, args.steps, elapsed_ms * 1e-3)
    step_gbs = (score_bytes + gather_bytes + other_bytes) / (elapsed_ms * 1e-3) / 1e9
    kept_layers = list(range(L)) if anchor is None else [anchor]
    kept_frac = float(counts[args.warmup:, kept_layers].sum() / (args.steps * len(kept_layers) * nvs.sum()))

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "tokens_per_s": value * r.batch,
        "config": dict(workload_config(r, nbuf), parallelism=f"replicas x{world}" if world > 1 else "single GPU"),
        "hbm": {"achieved_gbs": step_gbs, "frac_of_measured": step_gbs / peak,
                "frac_of_nominal_8tbs": step_gbs / NOMINAL_HBM_GBS,
                "bytes_per_step": (score_bytes + gather_bytes + other_bytes) / args.steps,
                "note": "whole step: algorithmic bytes (all visual K + kept visual V + text K/V + q + out) / step time"},
        "roofline": {"kernel": "k_score", "bound": "hbm", "achieved": achieved, "peak": peak,
                     "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": traffic,
                     "avg_launch_us": score_ms * 1e3 / n_calls,
                     "algorithmic_bytes_per_launch": score_bytes / n_calls,
                     "timing": "CUDA events recorded around every score launch inside the per-step graphs of a "
                               "second timed pass over the same steps (events serialise the kernels)"},
        "stages_us_per_call": {"score": score_ms * 1e3 / n_calls, "select": select_ms * 1e3 / n_calls,
                               "gather": gather_ms * 1e3 / n_calls,
                               "timed_pass_ms_per_step": timed_ms / args.steps},
        "avg_retention": kept_frac,
        "gpu_launches": 3 * n_calls + (0 if anchor is None else 2 * args.steps * (L - 1)),
        "clocks": clocks,
    }
    if fastv:
        line["prefill_prune"] = {
            "ms": prefill_ms, "visual_kept_frac": float(nvs_surv.sum() / nvs.sum()),
            "note": (f"once before decoding: FastV selection at layer {anchor + 1} (vp_decode_step, fixed ratio 50%, "
                     f"last prompt token's query) and vp_compact_kv of the K and V caches of layers "
                     f"{anchor + 1}-{L}; not in the timed region")}
    if anchor is not None:
        line["config"]["pipeline"] = (f"anchor layer {anchor + 1} of {L}: layers 1-{anchor} dense attention "
                                      f"(vp_decode_gather, whole visual span kept), layer {anchor + 1} "
                                      f"vp_decode_step, layers {anchor + 2}-{L} vp_decode_gather on its kept set"
                                      + (f"; layers {anchor + 1}-{L} read caches holding only FastV's prefill "
                                         f"survivors (50% of the visual tokens)" if fastv else ""))
        line["roofline"]["timing"] += "; only the anchor layer's call is timed per kernel"
        line["hbm"]["note"] = ("whole step: algorithmic bytes (dense layers: all K/V; anchor layer: all visual K + "
                               "kept visual V + text K/V; later layers: kept visual K/V + text K/V; q + out) / step time")
    default = args.workload == "qwen7b"
    if not args.no_e2e and default:
        line["e2e"] = e2e_leg(args, r, vp, ctx, dev, q_dev.cpu(), ks, vs_, kc, vc, span, budget, cap, world)
    if not args.no_cpu_baseline and rank == 0 and default:
        times = oracle_times("QWEN7B", list(range(4)), args.warmup, args.cpu_seconds, 4 * L)
        per_call = sum(times) / len(times)
        line["cpu_baseline"] = {"value": 1.0 / (per_call * L), "unit": UNIT, "cores": 1, "kind": "oracle",
                                "sample": f"{len(times)} layer calls (layers 0-3, steps from {args.warmup}) "
                                          f"timed, scaled to a {L}-layer step; single-threaded numpy"}
    vp.vp_free(ctx)
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def e2e_leg(args, r, vp, ctx, dev, q_host, ks, vs_, kc, vc, span, budget, cap, world):
    """Same steps through the C ABI, fed from and read back to host memory, as
    a serving loop drives it: every step copies its queries, the appended
    token's K/V of every layer and the text lengths in from pinned memory
    (three copies into staging buffers), replays that step's CUDA graph -- the
    appends into the caches and the 28 vp_decode_step calls, captured once
    through the C ABI -- and copies the outputs, kept sets, budgets and masses
    back, with one stream synchronisation per step."""
    import torch
    L, B, H, D, Hkv = r.layers, r.batch, r.heads, r.head_dim, r.kv_heads
    S = args.warmup + args.steps
    nv0, tl0 = int(r.vis_lens[0]), int(r.text_lens[0])
    qh = q_host.pin_memory()                                           # [S, L, B, H, D]
    kvh = torch.stack([torch.stack([k[:, :, nv0 + tl0 - 1: nv0 + tl0 - 1 + S] for k in ks]),
                       torch.stack([v[:, :, nv0 + tl0 - 1: nv0 + tl0 - 1 + S] for v in vs_])])
    kvh = kvh.permute(4, 0, 1, 2, 3, 5).contiguous().cpu().pin_memory()   # [S, 2, L, B, Hkv, D]
    tlh = (torch.tensor(r.text_lens, dtype=torch.int32)[None, :] + torch.arange(S, dtype=torch.int32)[:, None]
           ).contiguous().pin_memory()                                  # [S, B]
    q_in = torch.empty((L, B, H, D), dtype=torch.bfloat16, device=dev)
    kv_in = torch.empty((2, L, B, Hkv, D), dtype=torch.bfloat16, device=dev)
    tl = torch.empty((B,), dtype=torch.int32, device=dev)
    out = torch.empty((L, B, H, D), dtype=torch.bfloat16, device=dev)
    kept = torch.empty((L, B, cap), dtype=torch.int32, device=dev)
    count = torch.empty((L, B), dtype=torch.int32, device=dev)
    mass = torch.empty((L, B, H), dtype=torch.float32, device=dev)
    stats = torch.empty((L, B, 4), dtype=torch.float32, device=dev)
    res = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in (out, kept, count, mass, stats)]
    stream = torch.cuda.Stream(device=dev)

    def calls(s):
        pos = nv0 + tl0 - 1 + s
        for layer in range(L):
            ks[layer][:, :, pos].copy_(kv_in[0, layer])
            vs_[layer][:, :, pos].copy_(kv_in[1, layer])
            vp.vp_decode_step(ctx, B, q_in[layer], kc[layer], vc[layer], span, tl, budget, out[layer],
                              kept[layer], cap, count[layer], mass[layer], stats[layer], stream=stream)

    vp.vp_timing_enable(ctx, 0)
    graphs = []
    for s in range(S):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            calls(s)
        graphs.append(g)
    torch.cuda.synchronize()

    def one(s):
        with torch.cuda.stream(stream):
            q_in.copy_(qh[s], non_blocking=True)
            kv_in.copy_(kvh[s], non_blocking=True)
            tl.copy_(tlh[s], non_blocking=True)
            graphs[s].replay()
            for dst, src in zip(res, (out, kept, count, mass, stats)):
                dst.copy_(src, non_blocking=True)
        stream.synchronize()

    for s in range(args.warmup):
        one(s)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for s in range(args.warmup, S):
        one(s)
    el = max_over_ranks(time.perf_counter() - t0, world, dev)
    h2d = sum(t[0].numel() * t.element_size() for t in (qh, kvh, tlh))
    d2h = sum(t.numel() * t.element_size() for t in (out, kept, count, mass, stats))
    return {"value": job_rate(world, args.steps, el), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": el * 1e3 / args.steps,
            "note": "host wall clock per step: pinned-host inputs copied in, the step's CUDA graph (K/V appends "
                    "+ 28 vp_decode_step calls captured through the C ABI) replayed, results copied back, "
                    "one stream sync per step"}


def run_layer_calls(args):
    """--layer-calls N: one layer of the workload, N back-to-back calls and a
    device check, for profiling a single launch of each kernel (optionally
    with the L2 flushed by a 256 MB write before every call)."""
    import torch
    from paper_2605_31457_gb300 import vp, workloads as W
    r, _, _, _ = pick_workload(args.workload)
    dev = torch.device("cuda")
    B, H, Hkv, D = r.batch, r.heads, r.kv_heads, r.head_dim
    t_cap = r.capacity(2)
    k, v, f, sk = W.make_layer_torch(r, 0, t_cap, dev)
    q = W.make_queries_torch(r, 0, 1, f, sk, dev)[0]
    if r.paged:
        bt_np, n_pages, _ = W.page_table(B, t_cap, r.page_size, r.seed)
        bt = torch.from_numpy(bt_np).to(dev)
        k = W.scatter_pages(k, bt_np, n_pages, r.page_size)
        v = W.scatter_pages(v, bt_np, n_pages, r.page_size)
        kc, vc = vp.kv_paged(k, bt), vp.kv_paged(v, bt)
    else:
        kc, vc = vp.kv_contiguous(k), vp.kv_contiguous(v)
    vs = torch.tensor(r.vis_starts, dtype=torch.int32, device=dev)
    vl = torch.tensor(r.vis_lens, dtype=torch.int32, device=dev)
    tl = torch.tensor(r.text_lens, dtype=torch.int32, device=dev)
    budget = vp.make_budget(**r.budget)
    nvm = int(r.vis_lens.max())
    cdt = torch.bfloat16 if r.dtype == W.BF16 else torch.float32
    cfg = vp.make_config(B, H, Hkv, D, nvm, int((r.vis_lens + r.text_lens).max()) + 2,
                         vp.VP_BF16 if r.dtype == W.BF16 else vp.VP_FP32, int(r.paged), r.page_size)
    ctx = vp.vp_init(cfg)
    cap = max(1, vp.vp_max_kept(budget, nvm))
    out = torch.empty((B, H, D), dtype=cdt, device=dev)
    kept = torch.empty((B, cap), dtype=torch.int32, device=dev)
    cnt = torch.empty((B,), dtype=torch.int32, device=dev)
    mass = torch.empty((B, H), dtype=torch.float32, device=dev)
    st = torch.empty((B, 4), dtype=torch.float32, device=dev)
    flush = torch.empty(64 << 20, dtype=torch.float32, device=dev) if args.flush_l2 else None
    for _ in range(args.layer_calls):
        if flush is not None:
            flush.zero_()
        vp.vp_decode_step(ctx, B, q, kc, vc, vp.span(vs, vl), tl, budget, out, kept, cap, cnt, mass, st)
    torch.cuda.synchronize()
    vp.vp_check_errors(ctx)
    vp.vp_free(ctx)
    print(json.dumps({"layer_calls": args.layer_calls, "workload": args.workload, "flush_l2": bool(args.flush_l2),
                      "kv_bytes": 2 * k.numel() * k.element_size(), "avg_kept": float(cnt.float().mean())}))
    return 0


def committed_traffic():
    """DRAM bytes per score-kernel launch from the committed ncu summary, if it
    was taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "score_kernel_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        src = open(os.path.join(ROOT, "paper_2605_31457_gb300", "csrc", "vp_kernels.cu"), "rb").read()
        if d.get("source_sha256") != hashlib.sha256(src).hexdigest():
            return None
        return d.get("dram_bytes_per_launch_full_size")
    except (OSError, ValueError):
        return None


def main(argv=None):
    args = parse_args(argv)
    rank, world, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.layer_calls:
        return run_layer_calls(args)
    if world > 1:
        import torch
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))
    try:
        return run_ours(args, rank, world, local)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
