"""The allocation-free entry point against the context-based one.

vp_decode_step_noalloc serves callers that cannot allocate device memory on
their inference path (a plugin host whose framework owns all device memory, a
latency-critical loop that must not pay for an allocation): its scratch sits
in a fixed device array inside the library.  Here it must reproduce
vp_decode_step on the same inputs, on two calls in a row (the second call
reuses the array the first one left behind).  This file is collected last.
"""

import numpy as np
import pytest
import torch

from paper_2605_31457_gb300 import workloads as W

from . import vp_harness as Hn

pytestmark = pytest.mark.gpu


def _case():
    return W.Recipe(name="noalloc", layers=1, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                    vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                    planted_frac=0.04, seed=21, beta_range=(0.3, 0.9), beta_sink=1.0,
                    budget=W.ADAPTIVE_5PCT)


def test_noalloc_matches_context_path_twice(lib):
    vp = lib
    assert torch.cuda.is_available(), "GPU test"
    r = _case()
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, r.budget)
    try:
        ref = dev.run()
        tol = Hn.TOL[r.dtype]
        for call in range(2):
            out = torch.full_like(dev.out, float("nan"))
            kept = torch.full_like(dev.kept, -7)
            count = torch.full_like(dev.count, -7)
            mass = torch.full_like(dev.mass, float("nan"))
            stats = torch.full_like(dev.stats, float("nan"))
            st = vp.vp_decode_step_noalloc(dev.cfg, r.batch, dev.q, dev.kc, dev.vc, dev.span, dev.tl,
                                           dev.budget, out, kept, dev.kept_cap, count, mass, stats)
            assert st == vp.VP_OK, f"call {call}: status {st}"
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


def test_noalloc_rejects_scratch_overflow(lib):
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
