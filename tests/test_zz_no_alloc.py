"""The allocation-free entry point against the context-based one.

vp_decode_step_noalloc serves callers that cannot allocate device memory on
their inference path (a plugin host whose framework owns all device memory, a
latency-critical loop that must not pay for an allocation): its scratch sits
in a fixed device array inside the library.  Here it must reproduce
vp_decode_step on the same inputs, on two calls in a row (the second call
reuses the array the first one left behind), for every kernel family it can
reach inside its fixed scratch: the mma.sync and the tcgen05 score kernels,
contiguous and paged bf16 caches, fp32 caches.  This file is collected last.
"""

import numpy as np
import pytest
import torch

from paper_2605_31457_gb300 import workloads as W

from . import vp_harness as Hn

pytestmark = pytest.mark.gpu


def _case(kind):
    base = dict(name="noalloc", layers=1, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                planted_frac=0.04, seed=21, beta_range=(0.3, 0.9), beta_sink=1.0, budget=W.ADAPTIVE_5PCT)
    if kind == "tcgen05":   # long enough for the tensor-core score kernel (6.7 MB of scratch)
        base.update(vis_len=(2048, 1500, 700), vis_start=(0, 40, 10), text_len=(14000, 9000, 5000), seed=22)
    elif kind == "paged":
        base.update(batch=4, vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0),
                    text_len=(517, 70, 129, 33), paged=True, page_size=16, seed=23)
    elif kind == "fp32":
        base.update(dtype=W.FP32, heads=8, kv_heads=2, head_dim=64, seed=24)
    return W.Recipe(**base)


@pytest.mark.parametrize("kind", ["mma", "tcgen05", "paged", "fp32"])
def test_noalloc_matches_context_path_twice(lib, kind):
    vp = lib
    assert torch.cuda.is_available(), "GPU test"
    r = _case(kind)
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget)
    try:
        ref = dev.run()
        path, _ = vp.vp_last_launch(dev.ctx)
        assert (path == vp.VP_SCORE_TC) == (kind == "tcgen05"), f"context path took score kernel {path}"
        tol = Hn.TOL[r.dtype]
        for call in range(2):
            out = torch.full_like(dev.out, float("nan"))
            kept = torch.full_like(dev.kept, -7)
            count = torch.full_like(dev.count, -7)
            mass = torch.full_like(dev.mass, float("nan"))
            stats = torch.full_like(dev.stats, float("nan"))
            st = vp.vp_decode_step_noalloc(dev.cfg, r.batch, dev.q, dev.kc, dev.vc, dev.span, dev.tl,
                                           dev.budget, out, kept, dev.kept_cap, count, mass, stats)
            assert st == vp.VP_OK, f"call {call}: status {st}: {vp.vp_last_error(None)}"
            torch.cuda.synchronize()
            np.testing.assert_array_equal(count.cpu().numpy(), ref["count"])
            np.testing.assert_array_equal(kept.cpu().numpy(), ref["kept"])
            np.testing.assert_allclose(out.float().cpu().numpy(), ref["out"], rtol=0, atol=tol)
            np.testing.assert_allclose(mass.cpu().numpy(), ref["mass"], rtol=0, atol=tol)
            np.testing.assert_allclose(stats.cpu().numpy(), ref["stats"], rtol=0, atol=tol)
        for b in range(r.batch):
            Hn.compare_seq(inp, ref, b, r.budget)
    finally:
        dev.close()


def test_noalloc_rejects_scratch_overflow_and_bad_capacity(lib):
    vp = lib
    big = vp.make_config(64, 32, 8, 128, 16384, 17408, vp.VP_BF16)
    b = vp.make_budget()
    cap = vp.vp_max_kept(b, 16384)
    x = torch.empty(16, dtype=torch.bfloat16, device="cuda")
    kv = vp.kv_contiguous(torch.empty((1, 8, 16, 128), dtype=torch.bfloat16, device="cuda"))
    i32 = torch.zeros(64, dtype=torch.int32, device="cuda")
    sp = vp.span(i32, i32)
    kept = torch.empty((64, cap), dtype=torch.int32, device="cuda")
    f = torch.empty(64 * 32, dtype=torch.float32, device="cuda")
    st = vp.vp_decode_step_noalloc(big, 64, x, kv, kv, sp, i32, b, x, kept, cap, i32, f, f)
    assert st == vp.VP_ERR_CAPACITY
    assert "scratch bytes" in vp.vp_last_error(None)
    # A negative kept_cap is refused even when no visual token is configured.
    none = vp.make_config(1, 32, 8, 128, 0, 64, vp.VP_BF16)
    st = vp.vp_decode_step_noalloc(none, 1, x, kv, kv, sp, i32, b, x, kept, -1, i32, f, f)
    assert st == vp.VP_ERR_CAPACITY and "negative" in vp.vp_last_error(None)
