"""GPU parity of the layers after the anchor layer (vp_decode_gather).

The anchor layer (layer 0 of a recipe) runs vp_decode_step, whose kept sets
-- checked against the oracle by the decode-step tests -- stay on the
device; a later layer (layer 1, its own caches and query) then attends over
every text token and those kept visual tokens.  The reference is the
oracle's anchor_attention with the same kept sets.
"""

import numpy as np
import pytest
import torch

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

from . import vp_harness as Hn

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vp(lib):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    return lib


def small(**kw):
    base = dict(name="small", layers=2, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                planted_frac=0.04, seed=21, beta_range=(0.3, 0.9), beta_sink=1.0,
                budget=W.ADAPTIVE_5PCT)
    base.update(kw)
    return W.Recipe(**base)


def _run(vp, r, budget, layout="bhtd", gran=None, corrupt=None):
    """Anchor at layer 0, gather at layer 1; returns (inputs of layer 1, GPU
    out of layer 1, host kept sets per sequence)."""
    budget = dict(budget)
    if gran is not None:
        budget["granularity"] = gran
    gran = budget.get("granularity", 0)
    inp_a = Hn.make_inputs(r, 0)
    inp_b = Hn.make_inputs(r, 1)
    dev_a = Hn.Device(vp, inp_a, budget, layout=layout)
    dev_b = Hn.Device(vp, inp_b, budget, layout=layout)
    try:
        ga = dev_a.run()
        kept, count = dev_a.kept, dev_a.count
        if corrupt is not None:
            kept = kept.clone()
            kept.view(-1)[0] = corrupt
        vp.vp_decode_gather(dev_b.ctx, dev_b.B, dev_b.q, dev_b.kc, dev_b.vc, dev_b.span, dev_b.tl, kept,
                            dev_a.kept_cap, count, dev_b.out, granularity=gran)
        vp.vp_check_errors(dev_b.ctx)
        torch.cuda.synchronize()
        out = dev_b.out.float().cpu().numpy()
    finally:
        dev_a.close()
        dev_b.close()
    sets = [[ga["kept"][b][g][:int(ga["count"][b][g])] for g in range(ga["kept"].shape[1])]
            for b in range(r.batch)]
    return inp_b, out, sets


def _check(inp, out, sets, seqs=None):
    tol = Hn.TOL[inp.recipe.dtype]
    err = 0.0
    for b in (range(inp.recipe.batch) if seqs is None else seqs):
        want = O.anchor_attention(inp.q[b].double().numpy(), inp.k[b].double().numpy(), inp.v[b].double().numpy(),
                                  int(inp.vis_start[b]), int(inp.vis_len[b]), int(inp.text_len[b]), sets[b])
        np.testing.assert_allclose(out[b], want, rtol=0, atol=tol, err_msg=f"seq {b}")
        err = max(err, float(np.abs(out[b] - want).max()))
    return err


@pytest.mark.parametrize("D", [128, 64])
@pytest.mark.parametrize("gran", [0, 1])
def test_anchor_gather_matches_oracle(vp, D, gran):
    r = small(head_dim=D)
    inp, out, sets = _run(vp, r, r.budget, gran=gran)
    _check(inp, out, sets)


@pytest.mark.parametrize("budget", [dict(mode=O.DENSE, tau=0.1), dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000),
                                    dict(mode=O.FIXED_K, tau=0.1, fixed_k=0)])
def test_anchor_gather_budgets(vp, budget):
    """Every visual token kept (dense attention), half kept, none kept."""
    r = small()
    inp, out, sets = _run(vp, r, budget)
    _check(inp, out, sets)


@pytest.mark.parametrize("page_size,layout", [(16, "bhtd"), (64, "bthd"), (8, "bhtd")])
def test_anchor_gather_paged(vp, page_size, layout):
    r = small(batch=4, vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0), text_len=(517, 70, 129, 33),
              paged=True, page_size=page_size)
    inp, out, sets = _run(vp, r, r.budget, layout=layout)
    _check(inp, out, sets)


@pytest.mark.parametrize("layout", ["bthd", "padded"])
def test_anchor_gather_layouts(vp, layout):
    r = small()
    inp, out, sets = _run(vp, r, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=200_000), layout=layout)
    _check(inp, out, sets)


def test_anchor_gather_edge_lengths(vp):
    """Empty visual span, one visual token, only the current text token, a
    span after the whole prompt."""
    r = small(batch=5, vis_len=(0, 1, 33, 700, 16), vis_start=(0, 0, 1, 0, 9), text_len=(5, 1, 1, 1, 9))
    for budget in (r.budget, dict(mode=O.DENSE, tau=0.1), dict(mode=O.FIXED_K, tau=0.1, fixed_k=3)):
        inp, out, sets = _run(vp, r, budget)
        _check(inp, out, sets)


def test_anchor_gather_many_sequences(vp):
    rng = np.random.default_rng(40)
    vis = tuple(int(x) for x in rng.integers(64, 700, 40))
    start = tuple(int(x) for x in rng.integers(0, 40, 40))
    text = tuple(int(s) + int(x) for s, x in zip(start, rng.integers(1, 300, 40)))
    r = small(batch=40, vis_len=vis, vis_start=start, text_len=text)
    inp, out, sets = _run(vp, r, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=100_000))
    _check(inp, out, sets, seqs=range(0, 40, 3))


def test_anchor_gather_reports_a_bad_kept_index(vp):
    """A kept index outside the visual span is skipped by the kernel and
    reported by vp_check_errors; nothing faults."""
    r = small()
    with pytest.raises(vp.VPError) as ei:
        _run(vp, r, dict(mode=O.FIXED_K, tau=0.1, fixed_k=5), corrupt=1_000_000)
    assert ei.value.status == vp.VP_ERR_DEVICE_PRECOND


def test_anchor_gather_unsupported_configurations(vp):
    """fp32 caches and layouts without a tensor-map description are refused
    before anything is enqueued."""
    for r, layout in ((small(dtype=W.FP32, head_dim=64), "bhtd"), (small(), "tbhd"),
                      (small(paged=True, page_size=4), "bhtd")):
        inp = Hn.make_inputs(r, 1)
        dev = Hn.Device(vp, inp, r.budget, layout=layout)
        try:
            st = vp.vp_decode_gather(dev.ctx, dev.B, dev.q, dev.kc, dev.vc, dev.span, dev.tl, dev.kept,
                                     dev.kept_cap, dev.count, dev.out, check=False)
            assert st == vp.VP_ERR_UNSUPPORTED, st
        finally:
            dev.close()
