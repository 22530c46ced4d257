#!/usr/bin/env python3
"""Benchmark of the VisionPulse pruned decode step on GB300.

Workload (default): long reasoning -- a 28-layer decoder of 28 query / 4 kv
heads, head_dim 128, bf16 caches, batch 8, 4096 visual + 16384 text tokens per
sequence at the first step (lognormal key norms), one text token appended per
step.  A step is one vp_decode_step call per layer (each layer acting as its
own anchor layer), i.e. the whole five-stage hot path over every layer and
sequence.  This is the largest of the synthetic workloads shaped like the
paper's Qwen decoders (Sec. 5.1, App. B.1); the others are measured too and
reported under `configs`.

Prints one JSON line (rank 0).  `value` is decode steps per second with the
caches resident in HBM (per-step CUDA graphs of the layer calls, timed with
CUDA events); `e2e` is the same metric through the C ABI with the step's
queries and appended K/V copied in from pinned host memory and the results
copied back; `roofline` is the score kernel's (it moves the step's bytes);
`configs` holds the same figures for the tiny fp32 reference, the B = 1
Qwen2.5-VL-7B-shaped decode, the batched paged serving batch and the 20
points of the visual-length / retention sweep, each with its own clocks;
`cpu_baseline` is the CPU oracle on the host cores over a bounded sample.
`--impl reference` times the CPU oracle instead (rank 0, host cores).
"""

from __future__ import annotations

import argparse
import ctypes
import dataclasses
import glob
import hashlib
import json
import multiprocessing as mp
import os
import shutil
import statistics
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

ANCHOR_LAYER = 16  # 0-based index of the anchor layer l_a = 17 (Sec. 5.1)
METRIC = "pruned decode-attention steps/sec and achieved HBM GB/s (% of GB300 peak) on 1 GPU"
UNIT = "steps/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129e6
DEFAULT_WORKLOAD = "long"
SWEEP_TAGS = ("r1", "r5", "r20", "r50", "adaptive")


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None, help="timed steps (default: the workload's)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    help="long (default) | qwen7b | qwen7b-10pct | qwen7b-anchor | qwen7b-fastv-vp | serving | "
                         "tiny | sweep-<N_v>-<r1|r5|r20|r50|adaptive>")
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle CPU-baseline leg")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-config table")
    ap.add_argument("--config-steps", type=int, default=16, help="timed steps of each `configs` entry")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU-baseline sample budget (wall seconds)")
    ap.add_argument("--cpu-workers", type=int, default=0, help="oracle processes (0 = every host core)")
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


def compute_dtype(r):
    """The arithmetic type of the path: bf16 caches (fp32 accumulation) or fp32."""
    return "bf16" if r.dtype == "bf16" else "f32"


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


# --------------------------------------------------------------------- workloads

def pick_workload(name):
    """(recipe, default timed steps, distinct layer caches, host-generated)."""
    from paper_2605_31457_gb300 import workloads as W
    if name in ("qwen7b", "qwen7b-anchor", "qwen7b-fastv-vp"):
        return W.QWEN7B, 256, W.QWEN7B.layers, True
    if name == "qwen7b-10pct":  # the paper's 10% setting: tau = 0.4, clamp [5%, 10%]
        return dataclasses.replace(W.QWEN7B, budget=W.ADAPTIVE_10PCT), 256, W.QWEN7B.layers, True
    if name == "tiny":
        return W.TINY, 64, 1, True
    if name == "serving":
        return W.SERVING, 64, 4, False
    if name == "long":
        return W.LONG, 64, 4, False
    if name.startswith("sweep-"):
        parts = name.split("-")
        if len(parts) != 3 or parts[2] not in SWEEP_TAGS or not parts[1].isdigit():
            raise SystemExit(f"unknown workload {name}")
        budget = W.SWEEP_BUDGETS[SWEEP_TAGS.index(parts[2])]
        return W.sweep_recipe(int(parts[1]), budget), 16, 1, False
    raise SystemExit(f"unknown workload {name}")


def config_workloads():
    """The entries of the `configs` table: the tiny fp32 reference, the B = 1
    Qwen2.5-VL-7B-shaped decode, batched paged serving, and every point of the
    sweep (4 visual spans x 5 budgets)."""
    from paper_2605_31457_gb300 import workloads as W
    names = ["tiny", "qwen7b", "serving"]
    names += [f"sweep-{nv}-{t}" for nv in W.SWEEP_VIS for t in SWEEP_TAGS]
    return names


def budget_text(bd):
    mode = bd.get("mode", 0)
    if mode == 0:
        return f"adaptive tau={bd['tau']} clamp [{bd['r_lo_ppm'] / 1e4:g}%, {bd['r_hi_ppm'] / 1e4:g}%]"
    if mode == 1:
        return f"fixed ratio {bd['ratio_ppm'] / 1e4:g}%"
    return f"mode {mode}"


def workload_config(r, nbuf=None, flush_l2=False):
    import numpy as np
    tl = r.text_lens
    text = f"{int(tl[0])}" if len(set(tl.tolist())) == 1 else f"{int(tl.min())}-{int(tl.max())}"
    layout = f", paged (page {r.page_size})" if r.paged else ""
    nb = r.layers if nbuf is None else nbuf
    step_bytes = r.layers * r.batch * r.kv_heads * r.head_dim * (2 if r.dtype == "bf16" else 4) * \
        float(np.mean(r.vis_lens + 2 * r.text_lens))
    if flush_l2:
        l2 = (f"L2 flushed (256 MB write) before every timed step: one step streams only "
              f"~{step_bytes / 1e6:.2f} MB of K/V; steps are timed one by one with CUDA events")
    else:
        l2 = (f"no flush: each step streams ~{step_bytes / 1e9:.2f} GB of K/V over {nb} distinct layer "
              f"cache(s), every one above or the set of them well above the 129 MB L2")
    return {"workload": (f"{r.name}: {r.layers} layers x {r.heads} q / {r.kv_heads} kv heads, "
                         f"head_dim {r.head_dim}, {r.dtype}{layout}, batch {r.batch}, "
                         f"{int(r.vis_lens[0])} visual + {text} text tokens at step 0 "
                         f"(+1 text token per step), budget {budget_text(r.budget)}"),
            "global_batch": r.batch, "layers": r.layers, "distinct_layer_caches": nb, "l2": l2}


def needs_l2_flush(r, nbuf):
    """Whether a step's distinct cache bytes fit in L2: such a workload is
    timed step by step with an L2 flush before every step."""
    esz = 2 if r.dtype == "bf16" else 4
    per_layer = r.batch * r.kv_heads * r.head_dim * esz * float((r.vis_lens + 2 * r.text_lens).mean())
    return per_layer * min(nbuf, r.layers) < L2_BYTES


def kernel_sources_sha256():
    """Hash of every kernel and planner source, which the committed DRAM
    traffic figures are tied to."""
    h = hashlib.sha256()
    for path in sorted(glob.glob(os.path.join(ROOT, "paper_2605_31457_gb300", "csrc", "*"))):
        if path.endswith((".cu", ".h")):
            h.update(os.path.basename(path).encode())
            h.update(open(path, "rb").read())
    return h.hexdigest()


def committed_traffic(kernel, workload, algorithmic_per_launch, path=None, sha=None):
    """DRAM bytes per launch of `kernel` on `workload`, from the committed ncu
    capture (profiles/score_kernel_traffic.json) of that kernel and workload
    on the current sources, scaled from the captured launch's algorithmic
    bytes to this run's; (None, why) when no such capture exists."""
    path = path or os.path.join(ROOT, "profiles", "score_kernel_traffic.json")
    try:
        with open(path) as f:
            caps = json.load(f).get("captures", [])
    except (OSError, ValueError):
        return None, "no committed capture"
    sha = sha or kernel_sources_sha256()
    for c in caps:
        if c.get("workload") != workload or not kernel.startswith(c.get("kernel_prefix", "\0")):
            continue
        if c.get("source_sha256") != sha:
            return None, "the committed capture predates the current kernel sources"
        dram = c["dram_bytes_per_launch"]
        mean = sum(dram) / len(dram)
        ratio = mean / c["algorithmic_bytes_per_launch"]
        return ratio * algorithmic_per_launch, (
            f"ncu dram__bytes_read.sum + dram__bytes_write.sum of {c['kernel_prefix']} on {workload} "
            f"({mean:.0f} B per launch, {ratio:.4f} x its algorithmic bytes), scaled to this run's "
            f"algorithmic bytes per launch")
    return None, f"no committed capture for {kernel} on {workload}"


# ------------------------------------------------------------ inputs on the device

@dataclasses.dataclass
class Prep:
    """One workload's inputs on the device: `nbuf` distinct layer caches and
    per-(step, layer) queries for S steps."""
    r: object
    nbuf: int
    S: int
    ks: list
    vs: list
    kc: list
    vc: list
    q: object            # [S, L, B, H, D]
    vis_start: object
    vis_len: object
    tl_steps: object     # [S, B] text lengths
    span: object
    bt: object = None    # paged block table
    bt_np: object = None


def prepare(r, nbuf, host_gen, S, dev):
    import numpy as np
    import torch
    from paper_2605_31457_gb300 import vp, workloads as W
    L, B, H, D = r.layers, r.batch, r.heads, r.head_dim
    t_cap = r.capacity(S + 1)
    cdt = torch.bfloat16 if r.dtype == W.BF16 else torch.float32
    ks, vs_, focus = [], [], []
    q_dev = torch.empty((S, L, B, H, D), dtype=cdt, device=dev)
    for u in range(nbuf):
        if host_gen:  # the generator the parity tests use
            li = W.make_layer(r, u, t_cap=t_cap)
            ks.append(W.round_to(li.k, r.dtype).to(dev))
            vs_.append(W.round_to(li.v, r.dtype).to(dev))
            focus.append(li)
        else:         # the same recipe drawn on the device (gigabytes of cache)
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
    bt = bt_np = None
    if r.paged:
        bt_np, n_pages, _ = W.page_table(B, t_cap, r.page_size, r.seed)
        bt = torch.from_numpy(bt_np).to(dev)
        ks = [W.scatter_pages(k, bt_np, n_pages, r.page_size) for k in ks]
        vs_ = [W.scatter_pages(v, bt_np, n_pages, r.page_size) for v in vs_]
        kc = [vp.kv_paged(k, bt) for k in ks]
        vc = [vp.kv_paged(v, bt) for v in vs_]
    else:
        kc = [vp.kv_contiguous(k) for k in ks]
        vc = [vp.kv_contiguous(v) for v in vs_]
    vis_start = torch.tensor(r.vis_starts, dtype=torch.int32, device=dev)
    vis_len = torch.tensor(r.vis_lens, dtype=torch.int32, device=dev)
    tl_steps = (torch.tensor(r.text_lens, dtype=torch.int32)[None, :] +
                torch.arange(S, dtype=torch.int32)[:, None]).to(dev)
    torch.cuda.synchronize()
    return Prep(r, nbuf, S, ks, vs_, kc, vc, q_dev, vis_start, vis_len, tl_steps,
                vp.span(vis_start, vis_len), bt, bt_np)


# ------------------------------------------------------------------ one measurement

def measure(prep, budget_d, warmup, steps, world, dev, pipeline=None, flush_l2=False, want_e2e=False):
    """Times `steps` decode steps (after `warmup`) of the prepared workload
    with the given budget.  Returns the figures of one bench line."""
    import numpy as np
    import torch
    from paper_2605_31457_gb300 import vp, workloads as W
    r = prep.r
    L, B, H, Hkv, D, S = r.layers, r.batch, r.heads, r.kv_heads, r.head_dim, prep.S
    assert warmup + steps <= S
    nvs, tls = r.vis_lens.astype(np.int64), r.text_lens.astype(np.int64)
    nv_max = int(nvs.max())
    cdt = prep.q.dtype
    budget = vp.make_budget(**budget_d)
    cfg = vp.make_config(B, H, Hkv, D, nv_max, int((nvs + tls).max()) + S,
                         vp.VP_BF16 if r.dtype == W.BF16 else vp.VP_FP32, int(r.paged), r.page_size)
    ctx = vp.vp_init(cfg)
    cap = max(1, vp.vp_max_kept(budget, nv_max))
    out = torch.empty((L, B, H, D), dtype=cdt, device=dev)
    kept = torch.empty((L, B, cap), dtype=torch.int32, device=dev)
    count = torch.zeros((S, L, B), dtype=torch.int32, device=dev)
    mass = torch.empty((L, B, H), dtype=torch.float32, device=dev)
    stats = torch.empty((S, L, B, 4), dtype=torch.float32, device=dev)
    kc, vc, span = prep.kc, prep.vc, prep.span
    nbuf = prep.nbuf
    extra = {}

    # Anchor-layer pipeline (Sec. 5.1, l_a = 17): layers 1-16 attend densely
    # (the whole visual span kept), layer 17 runs the VisionPulse step, layers
    # 18-28 reuse its kept set.  FastV + VisionPulse (the paper's appendix on
    # prefill pruning: ratio 0.5 at the pruning layer, ranked by the last
    # prompt token's head-averaged attention) runs the selection and the cache
    # compaction once before decoding, then the anchor pipeline over the
    # survivors.  Every other workload treats each layer as its own anchor.
    anchor = ANCHOR_LAYER if pipeline in ("anchor", "fastv") else None
    fastv = pipeline == "fastv"
    kc_run, vc_run, span_run = [kc[l % nbuf] for l in range(L)], [vc[l % nbuf] for l in range(L)], [span] * L
    nvs_surv = nvs
    if anchor is not None:
        kept_all = torch.arange(nv_max, dtype=torch.int32, device=dev)[None, :].repeat(B, 1).contiguous()
        count_all = prep.vis_len.clone()
    if fastv:
        fv_budget = vp.make_budget(mode=vp.VP_FIXED_RATIO, tau=0.1, ratio_ppm=500_000)
        fv_cap = max(1, vp.vp_max_kept(fv_budget, nv_max))
        fv_kept = torch.empty((B, fv_cap), dtype=torch.int32, device=dev)
        fv_count = torch.empty((B,), dtype=torch.int32, device=dev)
        fv_out = torch.empty((B, H, D), dtype=cdt, device=dev)
        fv_mass = torch.empty((B, H), dtype=torch.float32, device=dev)
        tl_all = prep.tl_steps[S - 1]
        t_cap = r.capacity(S + 1)
        comp = [(torch.zeros((B, Hkv, t_cap, D), dtype=cdt, device=dev),
                 torch.zeros((B, Hkv, t_cap, D), dtype=cdt, device=dev)) for _ in range(anchor, L)]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        vp.vp_decode_step(ctx, B, prep.q[0, anchor], kc[anchor % nbuf], vc[anchor % nbuf], span, prep.tl_steps[0],
                          fv_budget, fv_out, fv_kept, fv_cap, fv_count, fv_mass)
        for i, layer in enumerate(range(anchor, L)):
            for src, dst in ((kc[layer % nbuf], comp[i][0]), (vc[layer % nbuf], comp[i][1])):
                vp.vp_compact_kv(ctx, B, src, vp.kv_contiguous(dst), span, tl_all, fv_kept, fv_cap, fv_count)
        e1.record()
        torch.cuda.synchronize()
        vp.vp_check_errors(ctx)
        span_c = vp.span(prep.vis_start, fv_count)
        for i, layer in enumerate(range(anchor, L)):
            kc_run[layer], vc_run[layer] = vp.kv_contiguous(comp[i][0]), vp.kv_contiguous(comp[i][1])
            span_run[layer] = span_c
        nvs_surv = fv_count.cpu().numpy().astype(np.int64)
        extra["prefill_prune"] = {
            "ms": e0.elapsed_time(e1), "visual_kept_frac": float(nvs_surv.sum() / nvs.sum()),
            "note": (f"once before decoding: FastV selection at layer {anchor + 1} (vp_decode_step, fixed ratio "
                     f"50%, last prompt token's query) and vp_compact_kv of the K and V caches of layers "
                     f"{anchor + 1}-{L}; not in the timed region")}

    def step_calls(s, stream=None):
        for layer in range(L):
            if anchor is not None and layer < anchor:
                vp.vp_decode_gather(ctx, B, prep.q[s, layer], kc_run[layer], vc_run[layer], span_run[layer],
                                    prep.tl_steps[s], kept_all, nv_max, count_all, out[layer], stream=stream)
            elif anchor is not None and layer > anchor:
                vp.vp_decode_gather(ctx, B, prep.q[s, layer], kc_run[layer], vc_run[layer], span_run[layer],
                                    prep.tl_steps[s], kept[anchor], cap, count[s, anchor], out[layer], stream=stream)
            else:
                vp.vp_decode_step(ctx, B, prep.q[s, layer], kc_run[layer], vc_run[layer], span_run[layer],
                                  prep.tl_steps[s], budget, out[layer], kept[layer], cap, count[s, layer],
                                  mass[layer], stats[s, layer], stream=stream)

    # One eager step loads the kernels (and tells which score kernel runs).
    # Two sets of per-step CUDA graphs: the first, without timing events,
    # gives the step rate (kernels chain through programmatic dependent
    # launch); the second records the library's stage events around every
    # kernel (which serialises them) and gives the per-kernel device times.
    step_calls(0)
    vp.vp_check_errors(ctx)
    if anchor is not None:  # the launch record of the timed vp_decode_step call
        vp.vp_decode_step(ctx, B, prep.q[0, anchor], kc_run[anchor], vc_run[anchor], span_run[anchor],
                          prep.tl_steps[0], budget, out[anchor], kept[anchor], cap, count[0, anchor],
                          mass[anchor], stats[0, anchor])
        torch.cuda.synchronize()
    score_path, kernels_per_call = vp.vp_last_launch(ctx)
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
    flush = torch.empty(64 << 20, dtype=torch.float32, device=dev) if flush_l2 else None

    def timed_region(gs, sample_clocks):
        for s in range(warmup):
            gs[s].replay()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        sampler = ClockSampler(dev) if sample_clocks else None
        if sampler:
            sampler.start()
        torch.cuda.synchronize()
        if flush is None:
            ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ev0.record()
            for s in range(warmup, warmup + steps):
                gs[s].replay()
            ev1.record()
            torch.cuda.synchronize()
            el_ms = ev0.elapsed_time(ev1)
        else:  # each step timed on its own after an L2 flush outside its events
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(steps)]
            for i, s in enumerate(range(warmup, warmup + steps)):
                flush.zero_()
                evs[i][0].record()
                gs[s].replay()
                evs[i][1].record()
            torch.cuda.synchronize()
            el_ms = sum(a.elapsed_time(b) for a, b in evs)
        clk = sampler.stop() if sampler else None
        el = max_over_ranks(el_ms, world, dev)
        if world > 1:
            torch.distributed.barrier()
        return el, clk

    elapsed_ms, clocks = timed_region(graphs, True)
    timed_ms, _ = timed_region(graphs_timed, False)
    vp.vp_check_errors(ctx)

    per_step = L if anchor is None else 1   # vp_decode_step calls per step (the timed ones)
    stage = vp.vp_timing_read(ctx, S * L)[warmup * per_step:(warmup + steps) * per_step]
    counts = count.cpu().numpy()
    score_bytes = gather_bytes = other_bytes = 0
    for s in range(warmup, warmup + steps):
        for layer in range(L):
            for b in range(B):
                if anchor is None or layer == anchor:
                    a, c = call_bytes(r, int(nvs_surv[b]), int(tls[b]) + s, int(counts[s, layer, b]))
                    score_bytes += a
                    gather_bytes += c
                else:  # the visual rows read: all of them before the anchor, the kept ones after
                    nkv = int(nvs[b]) if layer < anchor else int(counts[s, anchor, b])
                    a, c = call_bytes(r, 0, int(tls[b]) + s, 0)
                    other_bytes += a + c + 2 * nkv * r.kv_heads * r.head_dim * (2 if r.dtype == W.BF16 else 4)
    n_calls = steps * per_step
    score_ms = sum(x[0] for x in stage)
    select_ms = sum(x[1] for x in stage)
    gather_ms = sum(x[2] for x in stage)
    peak, peak_src = measured_peaks()
    value = job_rate(world, steps, elapsed_ms * 1e-3)
    total_bytes = score_bytes + gather_bytes + other_bytes
    step_gbs = total_bytes / (elapsed_ms * 1e-3) / 1e9
    kept_layers = list(range(L)) if anchor is None else [anchor]
    kept_frac = float(counts[warmup:warmup + steps, kept_layers].sum() /
                      (steps * len(kept_layers) * max(int(nvs.sum()), 1)))
    kernel = "k_score_tc" if score_path == vp.VP_SCORE_TC else "k_score_tma"
    if r.dtype != W.BF16:
        kernel = "k_score_f32"
    achieved = score_bytes / (score_ms * 1e-3) / 1e9
    res = {
        "value": value, "ms_per_step": elapsed_ms / steps, "steps": steps, "warmup": warmup,
        "tokens_per_s": value * B,
        "hbm": {"achieved_gbs": step_gbs, "frac_of_measured": step_gbs / peak,
                "frac_of_nominal_8tbs": step_gbs / NOMINAL_HBM_GBS, "bytes_per_step": total_bytes / steps,
                "note": "whole step: algorithmic bytes (all visual K + kept visual V + text K/V + q + out) / step time"},
        "roofline": {"kernel": kernel, "bound": "hbm", "achieved": achieved, "peak": peak,
                     "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                     "avg_launch_us": score_ms * 1e3 / n_calls,
                     "algorithmic_bytes_per_launch": score_bytes / n_calls,
                     "timing": "CUDA events recorded by the library around every score launch inside the per-step "
                               "graphs of a second timed pass over the same steps (events serialise the kernels)"},
        "stages_us_per_call": {"score": score_ms * 1e3 / n_calls, "select": select_ms * 1e3 / n_calls,
                               "gather": gather_ms * 1e3 / n_calls,
                               "timed_pass_ms_per_step": timed_ms / steps},
        "avg_retention": kept_frac,
        "kernels_per_layer_call": kernels_per_call,
        "gpu_launches": kernels_per_call * n_calls + (0 if anchor is None else 2 * steps * (L - 1)),
        "clocks": clocks,
    }
    res.update(extra)
    if anchor is not None:
        res["pipeline"] = (f"anchor layer {anchor + 1} of {L}: layers 1-{anchor} dense attention "
                           f"(vp_decode_gather, whole visual span kept), layer {anchor + 1} "
                           f"vp_decode_step, layers {anchor + 2}-{L} vp_decode_gather on its kept set"
                           + (f"; layers {anchor + 1}-{L} read caches holding only FastV's prefill "
                              f"survivors (50% of the visual tokens)" if fastv else ""))
        res["roofline"]["timing"] += "; only the anchor layer's call is timed per kernel"
        res["hbm"]["note"] = ("whole step: algorithmic bytes (dense layers: all K/V; anchor layer: all visual K + "
                              "kept visual V + text K/V; later layers: kept visual K/V + text K/V; q + out) / step time")
    if want_e2e and anchor is None:
        res["e2e"] = e2e_leg(prep, ctx, budget, cap, warmup, steps, world, dev)
    vp.vp_free(ctx)
    return res


def e2e_leg(prep, ctx, budget, cap, warmup, steps, world, dev):
    """The same steps through the C ABI, fed from and read back to host memory,
    as a serving loop drives it: every step copies its queries, the appended
    token's K and V for every layer and the text lengths in from pinned memory
    (three copies into staging buffers), replays that step's CUDA graph -- the
    appends into the caches and the layer calls, captured once through the C
    ABI -- and copies the outputs, kept sets, budgets and masses back, with one
    stream synchronisation per step."""
    import numpy as np
    import torch
    from paper_2605_31457_gb300 import vp
    r = prep.r
    L, B, H, D, Hkv, S, nbuf = r.layers, r.batch, r.heads, r.head_dim, r.kv_heads, prep.S, prep.nbuf
    cdt = prep.q.dtype
    # Cache row of the token appended at step s: the last live row, vis_len + text_len - 1.
    rows = (r.vis_lens.astype(np.int64) + r.text_lens.astype(np.int64))[None, :] - 1 + np.arange(S)[:, None]
    if r.paged:
        i0 = torch.from_numpy(prep.bt_np[np.arange(B)[None, :], rows // r.page_size].astype(np.int64)).to(dev)
        i2 = torch.from_numpy(rows % r.page_size).to(dev)
    else:
        i0 = torch.arange(B, device=dev)[None, :].expand(S, B).contiguous()
        i2 = torch.from_numpy(rows).to(dev)
    qh = prep.q.cpu().pin_memory()                                                 # [S, L, B, H, D]
    kvh = torch.stack([torch.stack([prep.ks[l % nbuf][i0, :, i2] for l in range(L)], 1),
                       torch.stack([prep.vs[l % nbuf][i0, :, i2] for l in range(L)], 1)], 1)
    kvh = kvh.cpu().contiguous().pin_memory()                                      # [S, 2, L, B, Hkv, D]
    tlh = prep.tl_steps.cpu().contiguous().pin_memory()                            # [S, B]
    q_in = torch.empty((L, B, H, D), dtype=cdt, device=dev)
    kv_in = torch.empty((2, L, B, Hkv, D), dtype=cdt, device=dev)
    tl = torch.empty((B,), dtype=torch.int32, device=dev)
    out = torch.empty((L, B, H, D), dtype=cdt, device=dev)
    kept = torch.empty((L, B, cap), dtype=torch.int32, device=dev)
    count = torch.empty((L, B), dtype=torch.int32, device=dev)
    mass = torch.empty((L, B, H), dtype=torch.float32, device=dev)
    stats = torch.empty((L, B, 4), dtype=torch.float32, device=dev)
    res = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in (out, kept, count, mass, stats)]
    stream = torch.cuda.Stream(device=dev)

    def calls(s):
        for layer in range(L):
            prep.ks[layer % nbuf][i0[s], :, i2[s]] = kv_in[0, layer]
            prep.vs[layer % nbuf][i0[s], :, i2[s]] = kv_in[1, layer]
            vp.vp_decode_step(ctx, B, q_in[layer], prep.kc[layer % nbuf], prep.vc[layer % nbuf], prep.span, tl,
                              budget, out[layer], kept[layer], cap, count[layer], mass[layer], stats[layer],
                              stream=stream)

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

    for s in range(warmup):
        one(s)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    for s in range(warmup, warmup + steps):
        one(s)
    el = max_over_ranks(time.perf_counter() - t0, world, dev)
    vp.vp_check_errors(ctx)
    h2d = sum(t[0].numel() * t.element_size() for t in (qh, kvh, tlh))
    d2h = sum(t.numel() * t.element_size() for t in (out, kept, count, mass, stats))
    return {"value": job_rate(world, steps, el), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": el * 1e3 / steps,
            "note": (f"host wall clock per step: pinned-host inputs copied in, the step's CUDA graph (K/V appends + "
                     f"{L} vp_decode_step calls captured through the C ABI) replayed, results copied back, "
                     f"one stream sync per step")}


def free_prep(prep):
    import torch
    del prep.ks[:], prep.vs[:]
    prep.q = prep.bt = None
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


# --------------------------------------------------------------------- oracle legs

_ORACLE = {}


def _oracle_init(paths):
    """Worker start-up (spawned process, single-threaded BLAS): maps the
    shared input files read-only."""
    import numpy as np
    for key, path in paths.items():
        _ORACLE[key] = np.load(path, mmap_mode="r")


def _oracle_call(item):
    """One (layer, sequence) oracle decode step; returns its seconds."""
    import numpy as np
    from oracle import vp_oracle as O
    u, s, b, vs, nv, tl, budget = item
    q = np.asarray(_ORACLE[f"q{u}"][s, b], dtype=np.float64)
    t0 = time.perf_counter()
    O.decode_step(q, _ORACLE[f"k{u}"][b], _ORACLE[f"v{u}"][b], vs, nv, tl, **budget)
    return time.perf_counter() - t0


class OraclePool:
    """The CPU oracle on the host cores: a spawned process pool, one oracle
    call per (layer, sequence) of a decode step, the inputs (the workload's
    host generator, rounded to the cache dtype) in memory-mapped files shared
    by the workers.  A recipe whose per-layer cache would exceed `max_bytes`
    is sampled on its first sequences; a step's time is then scaled to the
    whole batch."""

    def __init__(self, r, S, n_caches, workers=0, max_bytes=1.5e9):
        import numpy as np
        from paper_2605_31457_gb300 import workloads as W
        self.r_full = r
        esz_host = 4
        per_seq = r.kv_heads * r.capacity(S + 1) * r.head_dim * esz_host * 2
        bs = max(1, min(r.batch, int(max_bytes // per_seq)))
        if bs < r.batch:
            r = W.shrink(r, batch=bs, vis_len=tuple(r.vis_lens[:bs].tolist()),
                         vis_start=tuple(r.vis_starts[:bs].tolist()), text_len=tuple(r.text_lens[:bs].tolist()),
                         planted_scale=tuple(r.planted_scale[:bs]) if r.planted_scale else ())
        self.r = r
        self.S = S
        self.n_caches = max(1, min(n_caches, r.layers))
        self.dir = tempfile.mkdtemp(prefix="vp_oracle_")
        paths = {}
        t_cap = r.capacity(S + 1)
        for u in range(self.n_caches):
            li = W.make_layer(r, u, t_cap=t_cap)
            q = W.make_queries(r, u, li, steps=S)
            for key, x in ((f"k{u}", li.k), (f"v{u}", li.v), (f"q{u}", q)):
                path = os.path.join(self.dir, key + ".npy")
                np.save(path, W.round_to(x, r.dtype).float().numpy())  # exact cache-dtype values
                paths[key] = path
            del li, q
        self.workers = workers or os.cpu_count() or 1
        env_keys = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")
        old = {k: os.environ.get(k) for k in env_keys}
        for k in env_keys:
            os.environ[k] = "1"
        try:
            self.pool = mp.get_context("spawn").Pool(self.workers, initializer=_oracle_init, initargs=(paths,))
        finally:
            for k, v in old.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
        # Warm-up: every worker maps its inputs and runs one call.
        self.pool.map(_oracle_call, [self._item(0, 0, b % r.batch) for b in range(self.workers)], chunksize=1)

    def _item(self, layer, s, b):
        r = self.r
        return (layer % self.n_caches, s, b, int(r.vis_starts[b]), int(r.vis_lens[b]),
                int(r.text_lens[b]) + s, r.budget)

    def step(self, s):
        """Wall seconds of decode step s over every layer and sampled sequence,
        scaled to the whole batch."""
        r = self.r
        items = [self._item(layer, s, b) for layer in range(r.layers) for b in range(r.batch)]
        t0 = time.perf_counter()
        self.pool.map(_oracle_call, items, chunksize=1)
        return (time.perf_counter() - t0) * self.r_full.batch / r.batch

    def sample_text(self, n_steps):
        r = self.r
        seqs = (f"all {r.batch} sequences" if r.batch == self.r_full.batch
                else f"the first {r.batch} of {self.r_full.batch} sequences, the time scaled by "
                     f"{self.r_full.batch}/{r.batch}")
        return (f"{n_steps} whole decode step(s): all {r.layers} layer calls x {seqs}, one oracle call (float64 "
                f"numpy) per (layer, sequence) on a pool of {self.workers} spawned processes; "
                f"{self.n_caches} distinct layer cache(s) from the host generator")

    def close(self):
        self.pool.terminate()
        self.pool.join()
        shutil.rmtree(self.dir, ignore_errors=True)


def cpu_caches(r, nbuf):
    return 1 if r.batch * r.kv_heads * r.capacity() * r.head_dim * 8 > 256e6 else min(nbuf, 4)


def run_reference(args, rank, world):
    """The CPU oracle on the host cores, timed over whole decode steps of the
    same workload, metric and config as our arm (rank 0 only)."""
    if rank != 0:
        return 0
    r, default_steps, nbuf, _ = pick_workload(args.workload)
    steps = args.steps if args.steps is not None else min(default_steps, 8)
    S = args.warmup + steps
    pool = OraclePool(r, S, cpu_caches(r, nbuf), args.cpu_workers)
    try:
        times = [pool.step(s) for s in range(S)]
        sample = pool.sample_text(steps) + " per timed step"
        cores = pool.workers
    finally:
        pool.close()
    timed = times[args.warmup:]
    ms_step = 1e3 * sum(timed) / len(timed)
    value = 1e3 / ms_step
    line = {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": dict(workload_config(r, nbuf, needs_l2_flush(r, nbuf)), parallelism=parallelism(world)),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def parallelism(world):
    return f"replicas x{world}" if world > 1 else "single GPU"


# ------------------------------------------------------------------------ our arm

def workload_pipeline(name):
    if name.endswith("-anchor"):
        return "anchor"
    if name.endswith("-fastv-vp"):
        return "fastv"
    return None


def run_configs(args, dev, world):
    """The `configs` table: every other workload at N = 1, a few timed steps each."""
    from paper_2605_31457_gb300 import workloads as W
    table = {}
    warmup = max(3, args.warmup)
    steps = args.config_steps
    prep_sweep = {}
    for name in config_workloads():
        if name == args.workload:
            continue
        r, _, nbuf, host_gen = pick_workload(name)
        S = warmup + steps
        key = (r.vis_lens[0], r.batch) if name.startswith("sweep-") else None
        if key is not None:
            prep = prep_sweep.get(key)
            if prep is None:
                for p in prep_sweep.values():
                    free_prep(p)
                prep_sweep.clear()
                prep = prep_sweep[key] = prepare(r, nbuf, host_gen, S, dev)
        else:
            prep = prepare(r, nbuf, host_gen, S, dev)
        flush = needs_l2_flush(r, nbuf)
        res = measure(prep, r.budget, warmup, steps, world, dev, flush_l2=flush)
        if key is None:
            free_prep(prep)
        table[name] = {
            "workload": workload_config(r, nbuf, flush)["workload"], "dtype": compute_dtype(r),
            "steps": steps, "warmup": warmup, "steps_per_s": res["value"], "ms_per_step": res["ms_per_step"],
            "tokens_per_s": res["tokens_per_s"],
            "step_hbm": {k: res["hbm"][k] for k in ("achieved_gbs", "frac_of_measured", "frac_of_nominal_8tbs")},
            "score_kernel": {k: res["roofline"][k] for k in ("kernel", "achieved", "frac", "avg_launch_us")},
            "stages_us_per_call": {k: v for k, v in res["stages_us_per_call"].items() if k != "timed_pass_ms_per_step"},
            "avg_retention": res["avg_retention"], "kernels_per_layer_call": res["kernels_per_layer_call"],
            "l2_flush": flush, "clocks": res["clocks"]}
    for p in prep_sweep.values():
        free_prep(p)
    table["note"] = ("each entry: its own per-step CUDA graphs, CUDA-event timing and NVML clock samples; "
                     "step_hbm = the whole step's algorithmic bytes / step time; score_kernel = the score "
                     "kernel's algorithmic bytes / its CUDA-event launch time, both as fractions of the "
                     "measured copy bandwidth (MEASURED_PEAKS.json)")
    return table


def run_ours(args, rank, world, local):
    import torch
    from paper_2605_31457_gb300 import build as _build
    _build.ensure_built()
    from paper_2605_31457_gb300 import vp, workloads as W  # noqa: F401  (fails loudly without libvp.so)

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    r, default_steps, nbuf, host_gen = pick_workload(args.workload)
    steps = args.steps if args.steps is not None else default_steps
    pipeline = workload_pipeline(args.workload)
    S = args.warmup + steps
    prep = prepare(r, nbuf, host_gen, S, dev)
    flush = needs_l2_flush(r, nbuf)
    res = measure(prep, r.budget, args.warmup, steps, world, dev, pipeline=pipeline, flush_l2=flush,
                  want_e2e=not args.no_e2e)
    free_prep(prep)
    traffic, traffic_note = committed_traffic(res["roofline"]["kernel"], args.workload,
                                              res["roofline"]["algorithmic_bytes_per_launch"])
    res["roofline"]["traffic"] = traffic
    res["roofline"]["traffic_source"] = traffic_note
    line = {
        "metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": compute_dtype(r), "data": "synthetic",
        "tokens_per_s": res["tokens_per_s"],
        "config": dict(workload_config(r, nbuf, flush), parallelism=parallelism(world)),
    }
    for k in ("hbm", "roofline", "stages_us_per_call", "avg_retention", "kernels_per_layer_call", "gpu_launches",
              "clocks", "e2e", "prefill_prune", "pipeline"):
        if k in res:
            line[k] = res[k]
    if "pipeline" in line:
        line["config"]["pipeline"] = line.pop("pipeline")
    if not args.no_configs and world == 1:
        line["configs"] = run_configs(args, dev, world)
    if not args.no_cpu_baseline and rank == 0 and world == 1:
        pool = OraclePool(r, S, cpu_caches(r, nbuf), args.cpu_workers)
        try:
            times, t0 = [], time.perf_counter()
            for s in range(args.warmup, S):
                times.append(pool.step(s))
                if time.perf_counter() - t0 > args.cpu_seconds:
                    break
            line["cpu_baseline"] = {"value": len(times) / sum(times), "unit": UNIT, "cores": pool.workers,
                                    "kind": "oracle", "sample": pool.sample_text(len(times))}
        finally:
            pool.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


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
    path, nk = vp.vp_last_launch(ctx)
    vp.vp_free(ctx)
    sb = 0
    for b in range(B):
        sb += call_bytes(r, int(r.vis_lens[b]), int(r.text_lens[b]), 0)[0]
    print(json.dumps({"layer_calls": args.layer_calls, "workload": args.workload, "flush_l2": bool(args.flush_l2),
                      "score_kernel": "k_score_tc" if path == vp.VP_SCORE_TC else "k_score_tma",
                      "kernels_per_call": nk, "score_algorithmic_bytes_per_launch": sb,
                      "kv_bytes": 2 * k.numel() * k.element_size(), "avg_kept": float(cnt.float().mean()),
                      "sources_sha256": kernel_sources_sha256()}))
    return 0


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
