"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Small cases span several 32-token groups, split boundaries and ragged tails;
the full-size cases run the launch configuration the benchmark times and
compare every (or a sample of) sequence with the oracle.
"""

import dataclasses

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
                planted_frac=0.04, seed=11, beta_range=(0.3, 0.9), beta_sink=1.0,
                budget=W.ADAPTIVE_5PCT)
    base.update(kw)
    return W.Recipe(**base)


# ------------------------------------------------------------------ tiny ref

def test_tiny_reference_all_steps(vp):
    """The 16-step fp32 reference workload, every step against the oracle."""
    r = W.TINY
    li = W.make_layer(r, 0, t_cap=r.capacity())
    qs = W.make_queries(r, 0, li)
    rep = {}
    for step in range(r.steps):
        inp = Hn.make_inputs(r, 0, step, t_cap=r.capacity(), q_override=qs[step])
        Hn.check_all(vp, inp, r.budget, report=rep)
    assert rep.get("max_out_err", 0) < 1e-5


# --------------------------------------------------------- shapes and modes

@pytest.mark.parametrize("dtype,D", [(W.BF16, 128), (W.BF16, 64), (W.FP32, 128), (W.FP32, 64)])
def test_dtypes_and_head_dims(vp, dtype, D):
    r = small(dtype=dtype, head_dim=D)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget)


@pytest.mark.parametrize("H,Hkv", [(8, 8), (16, 1), (32, 8), (12, 4), (28, 4)])
def test_group_sizes(vp, H, Hkv):
    r = small(heads=H, kv_heads=Hkv)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget)


@pytest.mark.parametrize("budget", [
    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=10_000),
    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=50_000),
    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=200_000),
    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000),
    dict(mode=O.FIXED_K, tau=0.1, fixed_k=256),
    dict(mode=O.DENSE, tau=0.1),
    W.ADAPTIVE_10PCT,
    dict(mode=O.ADAPTIVE, tau=0.4, r_lo_ppm=0, r_hi_ppm=1_000_000),
    dict(mode=O.ADAPTIVE, tau=1.0, r_lo_ppm=0, r_hi_ppm=1_000_000),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=100_000),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=500_000),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=10_000),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=1_000_000),
    dict(mode=O.TOP_P, tau=0.1, ratio_ppm=0),
])
def test_budget_modes(vp, budget):
    r = small()
    Hn.check_all(vp, Hn.make_inputs(r), budget)


@pytest.mark.parametrize("budget", [dict(W.ADAPTIVE_5PCT, granularity=1),
                                    dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=200_000, granularity=1)])
def test_per_kv_head_selection(vp, budget):
    r = small()
    Hn.check_all(vp, Hn.make_inputs(r), budget)


def test_paged_cache(vp):
    r = small(batch=4, vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0),
              text_len=(517, 70, 129, 33), paged=True, page_size=16)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget)


def test_paged_cache_other_page_size(vp):
    r = small(paged=True, page_size=64, dtype=W.FP32, head_dim=64, heads=8, kv_heads=2)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget)


@pytest.mark.parametrize("layout", Hn.LAYOUTS)
@pytest.mark.parametrize("dtype,D", [(W.BF16, 128), (W.BF16, 64), (W.FP32, 128)])
def test_cache_layouts(vp, layout, dtype, D):
    """Dense, token-major, token-outermost and row-padded caches: the bulk
    tensor copies serve the first, second and fourth, the per-row copies the
    third; all must agree with the oracle."""
    r = small(dtype=dtype, head_dim=D)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget, layout=layout)


@pytest.mark.parametrize("page_size,layout", [(4, "bhtd"), (8, "bhtd"), (32, "bthd"), (64, "bhtd"),
                                              (256, "bthd"), (16, "padded")])
def test_paged_bf16_page_sizes(vp, page_size, layout):
    """Pages smaller than, equal to and larger than the 32-token tile (below
    8 tokens the per-row copies take over), in both pool layouts."""
    r = small(batch=4, vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0),
              text_len=(517, 70, 129, 33), paged=True, page_size=page_size)
    Hn.check_all(vp, Hn.make_inputs(r), r.budget, layout=layout)


def _many(batch, **kw):
    """`batch` sequences with varied lengths (seeded), for the per-chunk gather."""
    rng = np.random.default_rng(batch)
    vis = tuple(int(x) for x in rng.integers(64, 700, batch))
    start = tuple(int(x) for x in rng.integers(0, 40, batch))
    text = tuple(int(s) + int(x) for s, x in zip(start, rng.integers(1, 300, batch)))
    return small(batch=batch, vis_len=vis, vis_start=start, text_len=text, **kw)


@pytest.mark.parametrize("dtype,D,batch,budget,heads", [
    (W.FP32, 64, 3, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000), (28, 4)),
    (W.FP32, 128, 3, dict(mode=O.DENSE, tau=0.1), (28, 4)),
    (W.BF16, 128, 40, W.ADAPTIVE_5PCT, (28, 4)),
    (W.BF16, 64, 40, W.ADAPTIVE_5PCT, (28, 4)),
    (W.BF16, 128, 40, W.ADAPTIVE_5PCT, (32, 2)),
    (W.BF16, 64, 40, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=200_000), (28, 4)),
    (W.BF16, 128, 40, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000, granularity=1), (28, 4)),
    (W.BF16, 128, 40, dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000), (32, 2)),
])
def test_chunk_gather_paths(vp, dtype, D, batch, budget, heads):
    """Kept sets above 256 rows (fp32 and bf16 chunk kernels), and many
    sequences with small kept sets, which also take the chunk kernel (with a
    single ring slot when no chunk exceeds one 32-row tile per warp); up to
    8 and 16 query heads per kv-head."""
    H, Hkv = heads
    kw = dict(dtype=dtype, head_dim=D, heads=H, kv_heads=Hkv)
    r = _many(batch, **kw) if batch > 3 else small(**kw)
    Hn.check_all(vp, Hn.make_inputs(r), budget)


def test_zero_kept_capacity_on_the_chunk_gather(vp):
    """A budget that keeps nothing (fixed K = 0: kept capacity 0 and no kept
    array at all) on a shape that takes the shared-memory select and the
    chunk gather (16 sequences x 4 kv-heads, more than 4096 visual tokens):
    nothing is read from the absent list, and the output is the attention
    over the text tokens alone."""
    budget = dict(mode=O.FIXED_K, tau=0.1, fixed_k=0)
    B = 16
    rng = np.random.default_rng(B)
    vis = tuple(int(x) for x in rng.integers(4097, 4200, B))
    start = tuple(int(x) for x in rng.integers(0, 40, B))
    text = tuple(int(s) + int(x) for s, x in zip(start, rng.integers(1, 200, B)))
    inp = Hn.make_inputs(small(batch=B, vis_len=vis, vis_start=start, text_len=text))
    dev = Hn.Device(vp, inp, budget)
    try:
        assert vp.vp_max_kept(dev.budget, dev.cfg.max_visual) == 0
        vp.vp_decode_step(dev.ctx, B, dev.q, dev.kc, dev.vc, dev.span, dev.tl, dev.budget, dev.out, None, 0,
                          dev.count, dev.mass, dev.stats)
        vp.vp_check_errors(dev.ctx)
        assert vp.vp_last_launch(dev.ctx)[1] == 3, "score, select and chunk gather should serve this batch"
        torch.cuda.synchronize()
        gpu = dict(out=dev.out.float().cpu().numpy(), kept=np.full((B, 1, 1), -1, np.int32),
                   count=dev.count.cpu().numpy().reshape(B, 1), mass=dev.mass.cpu().numpy(),
                   stats=dev.stats.cpu().numpy())
        assert np.all(gpu["count"] == 0)
        for b in (0, 7, 15):
            Hn.compare_seq(inp, gpu, b, budget)
    finally:
        dev.close()


def test_explicit_logit_scale(vp):
    r = small()
    Hn.check_all(vp, Hn.make_inputs(r), dict(r.budget, scale=0.05))


# ---------------------------------------------------------------- edge cases

def test_edge_lengths(vp):
    """Empty visual span, one visual token, only the current text token,
    and a visual span starting after the whole prompt."""
    r = small(batch=5, vis_len=(0, 1, 33, 700, 16), vis_start=(0, 0, 1, 0, 9),
              text_len=(5, 1, 1, 1, 9))
    for budget in (r.budget, dict(mode=O.DENSE, tau=0.1), dict(mode=O.FIXED_K, tau=0.1, fixed_k=3)):
        Hn.check_all(vp, Hn.make_inputs(r), budget)


def test_zero_query_ties_go_to_lower_indices(vp):
    r = small()
    q = np.zeros((r.batch, r.heads, r.head_dim), dtype=np.float32)
    inp = Hn.make_inputs(r, q_override=q)
    gpu = Hn.check_all(vp, inp, dict(mode=O.FIXED_K, tau=0.1, fixed_k=17))
    for b in range(r.batch):
        k = int(gpu["count"][b][0])
        np.testing.assert_array_equal(gpu["kept"][b][0][:k], np.arange(k))


def test_planted_keys_recovered_on_gpu(vp):
    r = small(beta_range=(1.2, 1.2), beta_sink=0.0, planted_frac=0.03)
    inp = Hn.make_inputs(r)
    li = W.make_layer(r, 0, t_cap=r.capacity(1))
    budget = dict(mode=O.FIXED_K, tau=0.1, fixed_k=64)
    gpu = Hn.check_all(vp, inp, budget)
    for b in range(r.batch):
        planted = set(li.planted[0][b].tolist())
        kept = set(gpu["kept"][b][0][: int(gpu["count"][b][0])].tolist())
        assert planted <= kept


def test_batch_below_max_batch_and_repeat_calls(vp):
    """A context sized for more sequences, called twice: same results."""
    r = small()
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget, max_batch=8, max_seq=4096)
    try:
        a = dev.run()
        b = dev.run()
    finally:
        dev.close()
    for key in a:
        np.testing.assert_array_equal(a[key], b[key])
    for s in range(r.batch):
        Hn.compare_seq(inp, a, s, r.budget)


def test_device_precondition_is_reported_not_faulted(vp):
    """A visual span past the live cache is clamped and reported."""
    r = small(batch=1, vis_len=(64,), vis_start=(0,), text_len=(32,))
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget)
    try:
        dev.vs.fill_(50)          # vis_start > text_len
        dev.run(check_errors=False)
        st = vp.vp_check_errors(dev.ctx, check=False)
        assert st == vp.VP_ERR_DEVICE_PRECOND
        assert "visual span" in vp.vp_last_error(dev.ctx)
        assert vp.vp_check_errors(dev.ctx, check=False) == vp.VP_OK   # cleared
    finally:
        dev.close()


def test_capacity_and_argument_errors(vp):
    r = small(batch=1, vis_len=(64,), vis_start=(0,), text_len=(32,))
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget)
    try:
        st = vp.vp_decode_step(dev.ctx, 1, dev.q, dev.kc, dev.vc, dev.span, dev.tl, dev.budget, dev.out,
                               dev.kept, 1, dev.count, dev.mass, dev.stats, check=False)
        assert st == vp.VP_ERR_CAPACITY
        st = vp.vp_decode_step(dev.ctx, 2, dev.q, dev.kc, dev.vc, dev.span, dev.tl, dev.budget, dev.out,
                               dev.kept, dev.kept_cap, dev.count, dev.mass, dev.stats, check=False)
        assert st == vp.VP_ERR_CAPACITY
        bad = vp.make_budget(tau=-1.0)
        st = vp.vp_decode_step(dev.ctx, 1, dev.q, dev.kc, dev.vc, dev.span, dev.tl, bad, dev.out,
                               dev.kept, dev.kept_cap, dev.count, dev.mass, dev.stats, check=False)
        assert st == vp.VP_ERR_INVALID_ARG
        odd = vp.vp_kv(dev.k_t.data_ptr() + 2, dev.kc.stride_b, dev.kc.stride_h, dev.kc.stride_t, None, 0, 0)
        st = vp.vp_decode_step(dev.ctx, 1, dev.q, odd, dev.vc, dev.span, dev.tl, dev.budget, dev.out,
                               dev.kept, dev.kept_cap, dev.count, dev.mass, dev.stats, check=False)
        assert st == vp.VP_ERR_INVALID_ARG
        assert vp.vp_check_errors(dev.ctx, check=False) == vp.VP_OK
    finally:
        dev.close()


# -------------------------------------------------------------- full sizes

def test_qwen7b_full_size_layer(vp):
    """The B = 1 decode (28/4 heads, 1296 visual + 2561 text, bf16) at four
    decode steps of one layer, two of them after the first shift of the visual
    focus (every 64 steps): every output against the oracle."""
    r = W.QWEN7B
    t_cap = r.capacity(66)
    li = W.make_layer(r, 3, t_cap=t_cap)
    qs = W.make_queries(r, 3, li, steps=66)
    rep = {}
    for step in (0, 63, 64, 65):   # 64, 65: past the first shift of the visual focus
        inp = Hn.make_inputs(r, 3, step, t_cap=t_cap, q_override=qs[step])
        Hn.check_all(vp, inp, r.budget, report=rep)
        Hn.check_all(vp, inp, W.ADAPTIVE_10PCT, report=rep)


@pytest.mark.parametrize("paged", [False, True])
def test_fused_select_gather_full_width_slices(vp, paged):
    """A batch whose select clusters hold one CTA per kv-head: the fused
    select + gather then attends over the kept rows for all 128 output
    dimensions of a kv-head in one CTA (V staged as two swizzled 64-dimension
    halves, two threads per text-partial element).  Ragged spans and lengths,
    every sequence against the oracle."""
    rng = np.random.default_rng(17)
    B = 20
    vis = tuple(int(x) for x in rng.integers(64, 700, size=B))
    start = tuple(int(x) for x in rng.integers(0, 40, size=B))
    text = tuple(int(x) + start[i] for i, x in enumerate(rng.integers(40, 900, size=B)))
    r = small(batch=B, vis_len=vis, vis_start=start, text_len=text, seed=13, paged=paged, page_size=16)
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget)
    try:
        gpu = dev.run()
        assert vp.vp_last_launch(dev.ctx)[1] == 2, "the fused select + gather should serve this batch"
        for b in range(B):
            Hn.compare_seq(inp, gpu, b, r.budget)
    finally:
        dev.close()


def test_serving_paged_full_size_layer(vp):
    """Batched serving: B = 32, paged (page 16), 2304 visual, text 512..4096,
    visual mass spread over [0.01, 0.4]: every sequence against the oracle."""
    r = W.SERVING
    inp = Hn.make_inputs(r, 0, 0)
    gpu = Hn.check_all(vp, inp, r.budget)
    assert len(set(gpu["count"][:, 0].tolist())) >= 4, "budgets should differ across the batch"


@pytest.mark.parametrize("nv", [576, 2304])
def test_sweep_points(vp, nv):
    inp = Hn.make_inputs(W.sweep_recipe(nv, W.ADAPTIVE_5PCT))
    for budget in W.SWEEP_BUDGETS:
        Hn.check_all(vp, inp, budget, seqs=(0, 31, 63))


# ------------------------------------------------- full sizes, device-generated

def _device_generated(vp, r, seqs, budgets, rep, expect_tc=None):
    """One layer of `r` at full size, drawn by the benchmark's on-device
    generator and run in the launch configuration the benchmark times; the
    sampled sequences are copied to the host and checked against the oracle."""
    dev = torch.device("cuda")
    t_cap = r.capacity(1)
    k, v, f, sk = W.make_layer_torch(r, 0, t_cap, dev)
    q = W.make_queries_torch(r, 0, 1, f, sk, dev)[0]
    B, H, Hkv, D = r.batch, r.heads, r.kv_heads, r.head_dim
    nvs, tls, vss = r.vis_lens, r.text_lens, r.vis_starts
    cfg = vp.make_config(B, H, Hkv, D, int(nvs.max()), int((nvs + tls).max()), vp.VP_BF16, 0, 1)
    ctx = vp.vp_init(cfg)
    vs_d = torch.from_numpy(vss.astype(np.int32)).to(dev)  # kept alive: the span holds raw pointers
    vl_d = torch.from_numpy(nvs.astype(np.int32)).to(dev)
    span = vp.span(vs_d, vl_d)
    tl = torch.from_numpy(tls.astype(np.int32)).to(dev)
    sel = list(seqs)
    inp = Hn.Inputs(r, q[sel].cpu(), k[sel].cpu(), v[sel].cpu(), vss[sel], nvs[sel], tls[sel])
    try:
        for budget in budgets:
            bd = vp.make_budget(**budget)
            cap = max(1, vp.vp_max_kept(bd, int(nvs.max())))
            nsel = Hkv if budget.get("granularity", 0) else 1
            out = torch.empty((B, H, D), dtype=torch.bfloat16, device=dev)
            kept = torch.empty((B, nsel, cap), dtype=torch.int32, device=dev)
            count = torch.empty((B, nsel), dtype=torch.int32, device=dev)
            mass = torch.empty((B, H), dtype=torch.float32, device=dev)
            stats = torch.empty((B, 4), dtype=torch.float32, device=dev)
            vp.vp_decode_step(ctx, B, q, vp.kv_contiguous(k), vp.kv_contiguous(v), span, tl, bd, out, kept,
                              cap, count, mass, stats)
            vp.vp_check_errors(ctx)
            if expect_tc is not None:
                assert (vp.vp_last_launch(ctx)[0] == vp.VP_SCORE_TC) == expect_tc
            torch.cuda.synchronize()
            gpu = dict(out=out[sel].float().cpu().numpy(), kept=kept[sel].cpu().numpy(),
                       count=count[sel].cpu().numpy(), mass=mass[sel].cpu().numpy(), stats=stats[sel].cpu().numpy())
            for i in range(len(sel)):
                Hn.compare_seq(inp, gpu, i, budget, rep)
    finally:
        vp.vp_free(ctx)


def test_long_reasoning_full_size_layer(vp):
    """Long reasoning: B = 8, 4096 visual + 16384 text, lognormal key norms,
    in the benchmark's launch configuration (tcgen05 score kernel): every
    sequence against the oracle."""
    rep = {}
    _device_generated(vp, W.LONG, range(8), [W.LONG.budget], rep, expect_tc=True)
    assert rep.get("max_out_err", 0) < 2e-2


@pytest.mark.parametrize("nv", [6400, 16384])
def test_sweep_points_full_size(vp, nv):
    """The long visual spans of the sweep at full size (B = 64, 32/8 heads),
    every benchmarked point -- the adaptive budget and 1% / 5% / 20% / 50%
    retention (slice and chunk gathers) -- plus top-p."""
    r = W.sweep_recipe(nv, W.ADAPTIVE_5PCT)
    rep = {}
    _device_generated(vp, r, (0, 33, 63), [W.ADAPTIVE_5PCT, *W.SWEEP_BUDGETS[:4],
                                           dict(mode=O.TOP_P, tau=0.1, ratio_ppm=100_000)], rep, expect_tc=True)
