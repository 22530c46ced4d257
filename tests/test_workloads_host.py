"""The synthetic workloads have the structure they are meant to have (CPU,
host generator and oracle; no GPU).

Batched serving: the planted-key scales of workloads.SERVING_PLANTED_SCALE
(calibrated by tests/calibrate_serving.py) must put every sequence's visual
mass that enters Eq. 7 -- the head-max (Sec. 4.3) of the Eq. 5-6 mass at the
workload's tau -- at the first decode step of layer 0 near its target, the
batch must span about 0.01 to 0.4, and the budgets of Eq. 7 must differ
across the batch.
"""

import numpy as np

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

from .calibrate_serving import head_max_mass


def test_serving_visual_mass_spans_the_target_range():
    r = W.SERVING
    assert len(r.planted_scale) == r.batch
    _, targets = W.serving_draws()
    li = W.make_layer(r, 0, t_cap=r.capacity(1))
    q = W.round_to(W.make_queries(r, 0, li, steps=1)[0], r.dtype).double().numpy()
    k = W.round_to(li.k, r.dtype)
    got, budgets = [], []
    for b in range(r.batch):
        vs, nv, tl = int(r.vis_starts[b]), int(r.vis_lens[b]), int(r.text_lens[b])
        kb = k[b, :, :nv + tl].double().numpy()
        m = head_max_mass(q[b], kb, vs, nv, tl, r.budget["tau"])
        got.append(m)
        budgets.append(O.budget(m, nv, O.ADAPTIVE, r.budget["r_lo_ppm"], r.budget["r_hi_ppm"]))
    got = np.array(got)
    rel = np.abs(np.log(got / np.array(targets)))
    assert rel.max() < 0.1, (got, targets)
    assert got.min() < 0.012 and got.max() > 0.33
    assert (got < 0.04).sum() >= 6 and (got > 0.1).sum() >= 6   # both decades populated
    # Eq. 7 with the clamp [1%, 5%]: masses below 5% give distinct budgets.
    assert len(set(budgets)) >= 8 and min(budgets) == 24 and max(budgets) == 115


def test_planted_scale_multiplies_only_the_planted_rows():
    base = W.shrink(W.sweep_recipe(64, W.ADAPTIVE_5PCT, batch=2), text_len=16)
    scaled = W.shrink(base, planted_scale=(1.0, 0.5))
    a = W.make_layer(base, 0, t_cap=base.capacity(1))
    b = W.make_layer(scaled, 0, t_cap=scaled.capacity(1))
    rows = a.planted[0][1]
    assert len(rows) > 0
    np.testing.assert_array_equal(a.k[0], b.k[0])
    np.testing.assert_allclose(b.k[1][:, rows], 0.5 * a.k[1][:, rows], rtol=1e-6)
    other = np.setdiff1d(np.arange(a.k.shape[2]), rows)
    np.testing.assert_array_equal(a.k[1][:, other], b.k[1][:, other])
    np.testing.assert_array_equal(a.v, b.v)
