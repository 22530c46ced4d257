"""GPU parity of the tcgen05 score kernel (128-row tiles, TMEM accumulators),
forced with vp_set_score_path(VP_SCORE_TC) on shapes the automatic choice
would give to the mma.sync kernels, and of the mma.sync kernels forced on a
shape the automatic choice gives to the tcgen05 kernel.  Every case is the
whole decode step against the oracle (kept sets, masses, outputs).

The cases span visual spans that start and end inside a 128-row tile (tiles
holding visual and text rows), tiles wholly inside the span (K only), ragged
last tiles, text before the span, several splits per sequence, every group
size class (G = 1, 3, 4, 7, 16), the cache layouts a tensor descriptor can
describe, pages of 8 to 256 tokens, every budget mode, and text logits that
grow along the sequence (so the text reference maximum is raised and the
TMEM accumulator rescaled)."""

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
    base = dict(name="small", layers=1, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                planted_frac=0.04, seed=31, beta_range=(0.3, 0.9), beta_sink=1.0,
                budget=W.ADAPTIVE_5PCT)
    base.update(kw)
    return W.Recipe(**base)


def tc_check(vp, r, budget=None, layout="bhtd", inp=None, seqs=None):
    inp = Hn.make_inputs(r) if inp is None else inp
    return Hn.check_all(vp, inp, r.budget if budget is None else budget, layout=layout, seqs=seqs,
                        score_path=vp.VP_SCORE_TC)


def test_tc_small_mixed_tiles(vp):
    tc_check(vp, small())


@pytest.mark.parametrize("H,Hkv", [(8, 8), (12, 4), (32, 8), (28, 4), (16, 1)])
def test_tc_group_sizes(vp, H, Hkv):
    tc_check(vp, small(heads=H, kv_heads=Hkv))


@pytest.mark.parametrize("layout", ["bhtd", "bthd", "padded"])
def test_tc_layouts(vp, layout):
    tc_check(vp, small(), layout=layout)


@pytest.mark.parametrize("page_size,layout", [(8, "bhtd"), (16, "bthd"), (32, "bhtd"), (64, "bthd"),
                                              (128, "bhtd"), (256, "bthd")])
def test_tc_paged(vp, page_size, layout):
    r = small(batch=4, vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0),
              text_len=(517, 70, 129, 33), paged=True, page_size=page_size)
    tc_check(vp, r, layout=layout)


@pytest.mark.parametrize("budget", [
    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000),
    dict(mode=O.DENSE, tau=0.4),
    dict(mode=O.FIXED_K, tau=0.1, fixed_k=7),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=300_000),
    dict(W.ADAPTIVE_5PCT, granularity=1),
    dict(W.ADAPTIVE_10PCT),
])
def test_tc_budgets(vp, budget):
    tc_check(vp, small(), budget=budget)


def test_tc_edge_lengths(vp):
    """Empty visual span, one visual token, only the current text token, a
    span after the whole prompt, spans ending exactly on a tile boundary."""
    r = small(batch=7, vis_len=(0, 1, 33, 700, 16, 128, 256), vis_start=(0, 0, 1, 0, 9, 0, 128),
              text_len=(5, 1, 1, 1, 9, 128, 131))
    for budget in (r.budget, dict(mode=O.DENSE, tau=0.1), dict(mode=O.FIXED_K, tau=0.1, fixed_k=3)):
        tc_check(vp, r, budget=budget)


def test_tc_long_sequences_many_splits(vp):
    """Thousands of rows per sequence: several splits each, splits wholly
    inside the visual span (no text rows: an empty text partial)."""
    r = small(batch=2, heads=32, kv_heads=8, vis_len=(3000, 1800), vis_start=(0, 700),
              text_len=(2500, 900), seed=32)
    tc_check(vp, r)


def test_tc_text_maximum_raised_along_the_sequence(vp):
    """Text keys aligned with the query with a norm growing along the
    sequence: later tiles pass the text reference maximum by more than
    theta, so it is raised and the O accumulator rescaled several times."""
    r = small(batch=2, heads=8, kv_heads=2, vis_len=(256, 200), vis_start=(0, 50),
              text_len=(1400, 900), seed=33)
    inp = Hn.make_inputs(r)
    k = inp.k.float()
    q = inp.q.float()
    G = r.heads // r.kv_heads
    for b in range(r.batch):
        vs, nv, tl = int(inp.vis_start[b]), int(inp.vis_len[b]), int(inp.text_len[b])
        T = nv + tl
        for g in range(r.kv_heads):
            qd = q[b, g * G:(g + 1) * G].mean(0)
            qd = qd / qd.norm()
            for t in range(vs + nv, T, 97):  # every 97th text row after the span
                k[b, g, t] = qd * (2.0 + 30.0 * t / T)
    inp.k = W.round_to(k.numpy(), r.dtype)
    gpu = tc_check(vp, r, inp=inp)
    assert np.all(np.isfinite(gpu["out"]))


def test_mma_forced_where_auto_takes_tc(vp):
    """The mma.sync kernels stay correct on a shape the automatic choice
    gives to the tcgen05 kernel (the long-reasoning shape, one sequence
    pair)."""
    r = small(batch=8, vis_len=(2304,) * 8, vis_start=(0,) * 8, text_len=(2100,) * 8, seed=34)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget, seqs=(0, 5), score_path=vp.VP_SCORE_MMA)


def test_tc_refuses_what_it_cannot_serve(vp):
    """fp32 caches, head_dim 64 and token-outermost layouts: VP_ERR_UNSUPPORTED
    before anything is enqueued; an unknown path: VP_ERR_INVALID_ARG."""
    for r, layout in ((small(dtype=W.FP32), "bhtd"), (small(head_dim=64), "bhtd"), (small(), "tbhd")):
        inp = Hn.make_inputs(r)
        dev = Hn.Device(vp, inp, r.budget, layout=layout, score_path=vp.VP_SCORE_TC)
        try:
            st = vp.vp_decode_step(dev.ctx, dev.B, dev.q, dev.kc, dev.vc, dev.span, dev.tl, dev.budget, dev.out,
                                   dev.kept, dev.kept_cap, dev.count, dev.mass, dev.stats, check=False)
            assert st == vp.VP_ERR_UNSUPPORTED, st
            with pytest.raises(vp.VPError) as ei:
                vp.vp_set_score_path(dev.ctx, 7)
            assert ei.value.status == vp.VP_ERR_INVALID_ARG
        finally:
            dev.close()


def test_tc_ragged_lengths_one_long_sequence(vp):
    """Very different lengths in one call: one long sequence among short ones
    (splits of the long one's size, empty splits for the short ones), an
    empty visual span, one-token sequences, text before the span."""
    r = small(batch=12, vis_len=(1000, 64, 300, 0, 577, 128, 900, 1, 33, 700, 256, 512),
              vis_start=(0, 5, 40, 0, 13, 0, 7, 0, 2, 0, 0, 100),
              text_len=(9000, 20, 300, 5, 70, 1500, 129, 1, 2, 40, 2500, 300), seed=33)
    tc_check(vp, r)
    tc_check(vp, r, budget=dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=200_000))


def test_tc_paged_ragged_batch(vp):
    """A paged batch with text lengths spread like batched serving's, on the
    automatic path (which picks the tcgen05 kernel) and forced."""
    rng = np.random.default_rng(34)
    text = tuple(int(t) for t in rng.integers(50, 3000, 16))
    r = small(batch=16, vis_len=640, vis_start=0, text_len=text, paged=True, page_size=16, seed=34)
    inp = Hn.make_inputs(r)
    tc_check(vp, r, inp=inp)
    Hn.check_all(vp, inp, r.budget)


@pytest.mark.parametrize("path", ["tc", "mma"])
@pytest.mark.parametrize("budget", [W.ADAPTIVE_5PCT, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000)])
def test_back_to_back_calls_on_one_stream(vp, path, budget):
    """Four layer calls on one context and stream with no host
    synchronisation.  Each call's score kernel starts while the previous
    call's select (and gather) still run and waits only before its first
    workspace write, so its text-only splits stream meanwhile.  Every output
    must be bit-identical to the same call run alone.  The 5% budget takes the
    fused select + gather, the 50% one the select and the chunk gather."""
    r = small(vis_len=(1024, 577), vis_start=(0, 40), text_len=(4000, 2600), batch=2)
    layers = range(4)
    devs = [Hn.Device(vp, Hn.make_inputs(r, layer), budget) for layer in layers]
    ctx = devs[0].ctx
    vp.vp_set_score_path(ctx, vp.VP_SCORE_TC if path == "tc" else vp.VP_SCORE_MMA)

    def call(d):
        outs = dict(out=torch.full_like(d.out, float("nan")), kept=torch.full_like(d.kept, -7),
                    count=torch.full_like(d.count, -7), mass=torch.full_like(d.mass, float("nan")),
                    stats=torch.full_like(d.stats, float("nan")))
        vp.vp_decode_step(ctx, d.B, d.q, d.kc, d.vc, d.span, d.tl, d.budget, outs["out"], outs["kept"], d.kept_cap,
                          outs["count"], outs["mass"], outs["stats"])
        return outs

    def host(o):
        return dict(out=o["out"].view(torch.int16).cpu().numpy(), kept=o["kept"].cpu().numpy(),
                    count=o["count"].cpu().numpy(), mass=o["mass"].cpu().numpy(), stats=o["stats"].cpu().numpy())

    try:
        alone = []
        for d in devs:
            o = call(d)
            vp.vp_check_errors(ctx)
            torch.cuda.synchronize()
            alone.append(host(o))
        chained = [call(d) for d in devs]
        vp.vp_check_errors(ctx)
        torch.cuda.synchronize()
        for layer, (want, o) in enumerate(zip(alone, chained)):
            got = host(o)
            for k in want:
                np.testing.assert_array_equal(got[k], want[k], err_msg=f"layer {layer} {k}")
        assert (alone[0]["count"] > 0).all()
        if path == "tc":
            assert vp.vp_last_launch(ctx)[0] == vp.VP_SCORE_TC
    finally:
        for d in devs:
            d.close()
