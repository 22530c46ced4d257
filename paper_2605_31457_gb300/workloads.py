"""Seeded synthetic inputs for the VisionPulse decode step.

This module only draws inputs: cached keys/values, queries, visual spans,
text lengths and (optionally) a shuffled paged layout.  It holds none of the
method's arithmetic (no logits, softmax, mass, budget or selection), so both
the CUDA path and the CPU oracle may consume what it produces.  Everything is
drawn on the host with numpy from a fixed seed, then rounded once to the cache
dtype; the oracle widens those exact values and the GPU reads the same bytes.

Recipe (the same for every workload, with per-workload knobs):
  * keys, values and query noise are iid N(0, 1);
  * per (layer, sequence, kv-head) and focus group f, a unit "focus" vector
    u_f; a fraction ``planted_frac`` of the visual positions get keys
    c_b * sqrt(D) * (0.8 u_f + 0.6 w) with w a unit vector orthogonal to u_f
    (cosine 0.8 with the focus direction) and c_b a per-sequence scale
    (``planted_scale``, 1 by default) setting how much attention the
    sequence's visual span draws;
  * optionally a text "sink" key sqrt(D) * u_s at the first text position
    (a token every query attends to, giving a low visual-mass floor);
  * the query of head h at step s is
        sqrt(D) * (beta_v * u_f(s) + beta_s * u_s) + N(0, I),
    with beta_v drawn log-uniformly per (step, sequence, head) from
    ``beta_range`` and the focus group
    f(s) changing every ``focus_every`` steps (shifting visual focus);
  * optionally every key row is multiplied by a lognormal(0, key_sigma)
    factor (heavy-tailed key norms).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np

BF16 = "bf16"
FP32 = "fp32"


@dataclass(frozen=True)
class Recipe:
    name: str
    layers: int
    batch: int
    heads: int
    kv_heads: int
    head_dim: int
    dtype: str
    vis_len: tuple            # per sequence (len == batch) or a single value
    vis_start: tuple          # prompt tokens before the visual span, per sequence
    text_len: tuple           # text tokens at step 0, including the current token
    steps: int
    planted_frac: float
    seed: int
    n_focus: int = 1
    focus_every: int = 0      # 0 = never change focus
    beta_range: tuple = (1.0, 1.0)
    planted_scale: tuple = () # optional per-sequence multiplier c_b of the planted keys
    beta_sink: float = 0.0    # 0 = no sink token
    key_sigma: float = 0.0    # lognormal sigma of key norms (0 = off)
    paged: bool = False
    page_size: int = 16
    budget: dict = field(default_factory=dict)

    def per_seq(self, v):
        v = tuple(v) if isinstance(v, (tuple, list)) else (v,)
        return np.array(v * self.batch if len(v) == 1 else v, dtype=np.int32)

    def planted_scales(self):
        """Per-sequence multiplier of the planted keys (1 when not set)."""
        return np.asarray(self.planted_scale if self.planted_scale else (1.0,) * self.batch, dtype=np.float64)

    @property
    def vis_lens(self):
        return self.per_seq(self.vis_len)

    @property
    def vis_starts(self):
        return self.per_seq(self.vis_start)

    @property
    def text_lens(self):
        return self.per_seq(self.text_len)

    def capacity(self, steps=None):
        """Token capacity of the per-sequence cache for ``steps`` decode steps."""
        steps = self.steps if steps is None else steps
        return int((self.vis_lens + self.text_lens).max()) + max(steps - 1, 0)


def _rng(seed, *tags):
    return np.random.default_rng([int(seed)] + [int(t) for t in tags])


def _unit(rng, shape):
    x = rng.standard_normal(shape)
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def _orth_unit(rng, u):
    """Unit vectors orthogonal to the unit vectors u (same leading shape)."""
    w = rng.standard_normal(u.shape)
    w -= (w * u).sum(-1, keepdims=True) * u
    return w / np.linalg.norm(w, axis=-1, keepdims=True)


@dataclass
class LayerInputs:
    k: np.ndarray            # [B, Hkv, Tcap, D] float32 (before dtype rounding)
    v: np.ndarray            # [B, Hkv, Tcap, D]
    focus: np.ndarray        # [n_focus, B, Hkv, D] unit
    sink_dir: np.ndarray     # [B, Hkv, D] unit
    planted: list            # planted[f][b] -> visual-relative positions


def make_layer(r: Recipe, layer: int, t_cap: int | None = None) -> LayerInputs:
    """Keys and values of one layer's cache for every sequence of the batch."""
    B, Hkv, D = r.batch, r.kv_heads, r.head_dim
    t_cap = r.capacity() if t_cap is None else t_cap
    rng = _rng(r.seed, layer, 1)
    k = rng.standard_normal((B, Hkv, t_cap, D), dtype=np.float32)
    v = rng.standard_normal((B, Hkv, t_cap, D), dtype=np.float32)
    focus = _unit(rng, (r.n_focus, B, Hkv, D))
    sink_dir = _orth_unit(rng, focus[0])
    sqd = math.sqrt(D)
    vis_starts, vis_lens, text_lens = r.vis_starts, r.vis_lens, r.text_lens
    cs = r.planted_scales()
    planted = []
    for f in range(r.n_focus):
        pf = []
        for b in range(B):
            nv = int(vis_lens[b])
            n_p = min(nv, int(round(r.planted_frac * nv)))
            pos = np.sort(rng.choice(nv, size=n_p, replace=False)) if n_p else np.zeros(0, np.int64)
            pf.append(pos)
            if n_p:
                u = np.broadcast_to(focus[f, b][:, None, :], (Hkv, n_p, D))
                w = _orth_unit(rng, np.ascontiguousarray(u))
                k[b, :, vis_starts[b] + pos, :] = np.transpose(cs[b] * sqd * (0.8 * u + 0.6 * w), (1, 0, 2))
        planted.append(pf)
    if r.beta_sink > 0:
        for b in range(B):
            first_text = 0 if vis_starts[b] > 0 else int(vis_lens[b])
            k[b, :, first_text, :] = sqd * sink_dir[b]
    if r.key_sigma > 0:
        k *= np.exp(r.key_sigma * rng.standard_normal((B, Hkv, t_cap, 1))).astype(np.float32)
    return LayerInputs(k=k, v=v, focus=focus, sink_dir=sink_dir, planted=planted)


def make_queries(r: Recipe, layer: int, li: LayerInputs, steps: int | None = None) -> np.ndarray:
    """Queries [steps, B, H, D] float32 of one layer for ``steps`` decode steps."""
    steps = r.steps if steps is None else steps
    B, H, Hkv, D = r.batch, r.heads, r.kv_heads, r.head_dim
    G = H // Hkv
    rng = _rng(r.seed, layer, 2)
    lo, hi = r.beta_range
    beta = np.exp(rng.uniform(math.log(lo), math.log(hi), size=(steps, B, H)))
    noise = rng.standard_normal((steps, B, H, D))
    fidx = np.zeros(steps, dtype=np.int64)
    if r.focus_every > 0:
        fidx = (np.arange(steps) // r.focus_every) % r.n_focus
    u = li.focus[fidx]                                     # [steps, B, Hkv, D]
    u = np.repeat(u, G, axis=2)                            # [steps, B, H, D]
    us = np.repeat(li.sink_dir, G, axis=1)[None]           # [1, B, H, D]
    q = math.sqrt(D) * (beta[..., None] * u + r.beta_sink * us) + noise
    return q.astype(np.float32)


def round_to(x: np.ndarray, dtype: str):
    """Round float32 values once to the cache dtype; returns a CPU torch tensor."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x))
    return t.to(torch.bfloat16) if dtype == BF16 else t.to(torch.float32)


def page_table(batch: int, t_cap: int, page_size: int, seed: int, extra_pages: int = 3):
    """A shuffled page assignment for a paged cache of ``batch`` sequences.

    Returns (block_table [batch, max_pages] int32, n_pages, max_pages): logical
    page p of sequence b lives in pool page block_table[b, p]; a few pool pages
    are left unused.
    """
    max_pages = -(-t_cap // page_size)
    n_pages = batch * max_pages + extra_pages
    perm = _rng(seed, 7).permutation(n_pages)[: batch * max_pages].reshape(batch, max_pages)
    return perm.astype(np.int32), n_pages, max_pages


def scatter_pages(x, block_table, n_pages, page_size):
    """Copy a contiguous cache into the pool described by ``block_table``."""
    import torch
    B, Hkv, T, D = x.shape
    max_pages = block_table.shape[1]
    pad = max_pages * page_size - T
    xt = torch.as_tensor(x)
    if pad:
        xt = torch.cat([xt, xt.new_zeros(B, Hkv, pad, D)], dim=2)
    pool = xt.new_zeros(n_pages, Hkv, page_size, D)
    src = xt.reshape(B, Hkv, max_pages, page_size, D).permute(0, 2, 1, 3, 4)
    pool[torch.as_tensor(block_table.reshape(-1), dtype=torch.long)] = src.reshape(-1, Hkv, page_size, D)
    return pool


# ---------------------------------------------------------------------------
# The five workloads.  Shapes follow the Qwen-family decoders of the paper's
# experiments; budgets follow Sec. 5.2 (clamp) and App. B.1 (tau).
# ---------------------------------------------------------------------------

ADAPTIVE_5PCT = dict(mode=0, tau=0.1, r_lo_ppm=10_000, r_hi_ppm=50_000)
ADAPTIVE_10PCT = dict(mode=0, tau=0.4, r_lo_ppm=50_000, r_hi_ppm=100_000)

TINY = Recipe(
    name="tiny-ref", layers=1, batch=1, heads=8, kv_heads=2, head_dim=64, dtype=FP32,
    vis_len=576, vis_start=0, text_len=128, steps=16, planted_frac=0.05, seed=1,
    beta_range=(1.0, 1.0), budget=ADAPTIVE_5PCT)

QWEN7B = Recipe(
    name="qwen2.5-vl-7b-decode", layers=28, batch=1, heads=28, kv_heads=4, head_dim=128,
    dtype=BF16, vis_len=1296, vis_start=0, text_len=512 + 2048 + 1, steps=256,
    planted_frac=0.03, seed=2, n_focus=4, focus_every=64, beta_range=(0.3, 0.85),
    beta_sink=1.0, budget=ADAPTIVE_5PCT)


# Per-sequence planted-key scales of the batched-serving workload: c_b puts
# the visual mass that sets sequence b's budget (the head-max of the
# temperature-scaled mass at the workload's tau = 0.1) at the first decode
# step of layer 0 at the target drawn by serving_draws() (log-uniform in
# [0.01, 0.4]).  Written by tests/calibrate_serving.py, which finds each c_b
# by bisection with the CPU oracle on the host-generated layer.
SERVING_PLANTED_SCALE = (1.42711, 1.57979, 1.50723, 1.26233, 1.20460, 1.39935, 1.34273, 1.35763,
                         1.46155, 1.40012, 1.38687, 1.30919, 1.23687, 1.47727, 1.46549, 1.23615,
                         1.28423, 1.63120, 1.25340, 1.42354, 1.43298, 1.37269, 1.33983, 1.42035,
                         1.51391, 1.46188, 1.29900, 1.35225, 1.39636, 1.40571, 1.48737, 1.37757)


def serving_draws(seed=3, batch=32):
    """Text lengths (uniform in [512, 4096]) and visual-mass targets
    (log-uniform in [0.01, 0.4]) of the batched-serving sequences."""
    rng = _rng(seed, 0)
    text = tuple(int(t) for t in rng.integers(512, 4097, size=batch))
    target = tuple(float(x) for x in np.exp(rng.uniform(math.log(0.01), math.log(0.4), size=batch)))
    return text, target


def serving_recipe(seed=3, batch=32, planted_scale=None):
    text, _ = serving_draws(seed, batch)
    if planted_scale is None:
        planted_scale = SERVING_PLANTED_SCALE if (seed, batch) == (3, 32) else ()
    return Recipe(
        name="batched-serving-paged", layers=28, batch=batch, heads=28, kv_heads=4,
        head_dim=128, dtype=BF16, vis_len=2304, vis_start=0, text_len=text, steps=64,
        planted_frac=0.03, seed=seed, beta_range=(0.6, 1.0), planted_scale=tuple(planted_scale),
        beta_sink=1.6, paged=True, page_size=16, budget=ADAPTIVE_5PCT)


SERVING = serving_recipe()

LONG = Recipe(
    name="long-reasoning", layers=28, batch=8, heads=28, kv_heads=4, head_dim=128,
    dtype=BF16, vis_len=4096, vis_start=0, text_len=16384, steps=512,
    planted_frac=0.03, seed=4, beta_range=(0.3, 0.85), beta_sink=1.0, key_sigma=0.5,
    budget=ADAPTIVE_5PCT)


def sweep_recipe(vis_len: int, budget: dict, seed=5, batch=64):
    return Recipe(
        name=f"sweep-nv{vis_len}", layers=1, batch=batch, heads=32, kv_heads=8,
        head_dim=128, dtype=BF16, vis_len=vis_len, vis_start=0, text_len=1024, steps=16,
        planted_frac=0.03, seed=seed, beta_range=(0.3, 0.85), beta_sink=1.0, budget=budget)


SWEEP_VIS = (576, 2304, 6400, 16384)
SWEEP_BUDGETS = tuple(dict(mode=1, tau=0.1, ratio_ppm=r) for r in (10_000, 50_000, 200_000, 500_000)) \
    + (ADAPTIVE_5PCT,)


def shrink(r: Recipe, **kw) -> Recipe:
    """A smaller copy of a recipe (tests)."""
    return replace(r, **kw)


# ---------------------------------------------------------------------------
# The same recipe drawn on the GPU with torch's seeded generator, for the
# benchmark's large workloads (gigabytes of cache; host generation would take
# minutes).  Values differ from the host generator's; the recipe is the same.
# ---------------------------------------------------------------------------

def make_layer_torch(r: Recipe, layer: int, t_cap: int, device, dtype=None):
    """Keys and values [B, Hkv, t_cap, D] (cache dtype) plus the focus and
    sink directions [n_focus, B, Hkv, D] / [B, Hkv, D] (float32)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(int(r.seed) * 1_000_003 + int(layer) * 7_919 + 11)
    B, Hkv, D = r.batch, r.kv_heads, r.head_dim
    dt = dtype or (torch.bfloat16 if r.dtype == BF16 else torch.float32)
    k = torch.randn((B, Hkv, t_cap, D), generator=gen, device=device, dtype=torch.float32)
    v = torch.randn((B, Hkv, t_cap, D), generator=gen, device=device, dtype=torch.float32).to(dt)
    focus = torch.randn((r.n_focus, B, Hkv, D), generator=gen, device=device)
    focus = focus / focus.norm(dim=-1, keepdim=True)
    sink = torch.randn((B, Hkv, D), generator=gen, device=device)
    sink = sink - (sink * focus[0]).sum(-1, keepdim=True) * focus[0]
    sink = sink / sink.norm(dim=-1, keepdim=True)
    sqd = math.sqrt(D)
    vs, vl = r.vis_starts, r.vis_lens
    cs = r.planted_scales()
    for f in range(r.n_focus):
        for b in range(B):
            nv = int(vl[b])
            n_p = min(nv, int(round(r.planted_frac * nv)))
            if not n_p:
                continue
            pos = torch.randperm(nv, generator=gen, device=device)[:n_p] + int(vs[b])
            u = focus[f, b][:, None, :].expand(Hkv, n_p, D)
            w = torch.randn((Hkv, n_p, D), generator=gen, device=device)
            w = w - (w * u).sum(-1, keepdim=True) * u
            w = w / w.norm(dim=-1, keepdim=True)
            k[b, :, pos, :] = float(cs[b]) * sqd * (0.8 * u + 0.6 * w)
    if r.beta_sink > 0:
        for b in range(B):
            first_text = 0 if vs[b] > 0 else int(vl[b])
            k[b, :, first_text, :] = sqd * sink[b]
    if r.key_sigma > 0:
        k *= torch.exp(r.key_sigma * torch.randn((B, Hkv, t_cap, 1), generator=gen, device=device))
    return k.to(dt), v, focus, sink


def make_queries_torch(r: Recipe, layer: int, steps: int, focus, sink, device, dtype=None):
    """Queries [steps, B, H, D] in the cache dtype (same recipe as make_queries)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(int(r.seed) * 1_000_003 + int(layer) * 7_919 + 23)
    B, H, Hkv, D = r.batch, r.heads, r.kv_heads, r.head_dim
    G = H // Hkv
    lo, hi = r.beta_range
    beta = torch.exp(math.log(lo) + (math.log(hi) - math.log(lo)) *
                     torch.rand((steps, B, H), generator=gen, device=device))
    fidx = torch.zeros(steps, dtype=torch.long, device=device)
    if r.focus_every > 0:
        fidx = (torch.arange(steps, device=device) // r.focus_every) % r.n_focus
    u = focus[fidx].repeat_interleave(G, dim=2)                  # [steps, B, H, D]
    us = sink.repeat_interleave(G, dim=1)[None]
    noise = torch.randn((steps, B, H, D), generator=gen, device=device)
    q = math.sqrt(D) * (beta[..., None] * u + r.beta_sink * us) + noise
    dt = dtype or (torch.bfloat16 if r.dtype == BF16 else torch.float32)
    return q.to(dt)
