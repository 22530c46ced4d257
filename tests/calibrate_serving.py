"""Calibrates the per-sequence planted-key scales of the batched-serving
workload (``workloads.SERVING_PLANTED_SCALE``).

The serving batch should hold sequences whose visual spans draw very
different shares of the attention, so that the step-wise budgets of Eq. 7
differ across the batch.  For every sequence b this script finds, by
bisection, the scale c_b of its planted visual keys at which the visual mass
that enters Eq. 7 -- the head-max (Sec. 4.3) of the temperature-scaled mass
of Eq. 5-6 at the workload's tau = 0.1 -- at the first decode step of layer 0
equals the sequence's target from ``workloads.serving_draws`` (log-uniform
in [0.01, 0.4]).  (The plain tau = 1 mass cannot serve: set to [0.01, 0.4],
it leaves the tau = 0.1 mass of every sequence far below 1%, so every budget
sits at the clamp floor.)  The mass is computed with the CPU oracle on the
host-generated layer, with the planted rows rescaled and rounded to the cache
dtype as the generator does.

    python tests/calibrate_serving.py      # prints the tuple to paste
"""

from __future__ import annotations

import math
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import vp_oracle as O  # noqa: E402
from paper_2605_31457_gb300 import workloads as W  # noqa: E402


def head_max_mass(q, k, vis_start, vis_len, text_len, tau):
    """M_vis,max at temperature tau of one sequence (oracle arithmetic)."""
    T = vis_len + text_len
    z = O.logits(q, k[:, :T], 1.0 / math.sqrt(q.shape[1]))
    vis = np.zeros(T, dtype=bool)
    vis[vis_start:vis_start + vis_len] = True
    return O.visual_mass(O.softmax_tau(z, tau), vis)[2]


def calibrate(seed=3, batch=32, iters=40, c_hi=4.0):
    r = W.serving_recipe(seed, batch, planted_scale=())
    _, targets = W.serving_draws(seed, batch)
    li = W.make_layer(r, 0, t_cap=r.capacity(1))
    q = W.round_to(W.make_queries(r, 0, li, steps=1)[0], r.dtype).double().numpy()
    scales = []
    for b in range(batch):
        vs, nv, tl = int(r.vis_starts[b]), int(r.vis_lens[b]), int(r.text_lens[b])
        k32 = li.k[b, :, :nv + tl].copy()
        rows = vs + li.planted[0][b]
        base = k32[:, rows].astype(np.float64)

        def mass(c):
            k32[:, rows] = (c * base).astype(np.float32)
            k = W.round_to(k32, r.dtype).double().numpy()
            return head_max_mass(q[b], k, vs, nv, tl, r.budget["tau"])

        lo, hi = 0.0, c_hi
        if mass(lo) >= targets[b]:
            scales.append(0.0)
            continue
        for _ in range(iters):
            mid = 0.5 * (lo + hi)
            if mass(mid) < targets[b]:
                lo = mid
            else:
                hi = mid
        scales.append(0.5 * (lo + hi))
    return tuple(scales), targets


if __name__ == "__main__":
    sc, tg = calibrate()
    print("targets:", ", ".join(f"{t:.4f}" for t in tg))
    print("SERVING_PLANTED_SCALE = (" + ", ".join(f"{c:.5f}" for c in sc) + ")")
