"""GPU parity of FastV prefill pruning followed by VisionPulse (the paper's
appendix "Complementarity with Prefill Pruning": FastV keeps half of the
visual tokens at the prefill stage, VisionPulse then prunes step by step
over the survivors).

* the selection: vp_decode_step with the last prompt token as the query and
  a fixed 50% ratio, against the oracle's fastv_survivors (and the decode-step
  parity rules);
* the compaction (vp_compact_kv): bit-exact against the oracle's
  compact_cache, for contiguous and paged sources, both dtypes and both head
  dimensions, spans that start after text, empty and full kept sets;
* a decode step over the compacted caches against the oracle on the
  compacted inputs.
"""

import dataclasses

import numpy as np
import pytest
import torch

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

from . import vp_harness as Hn

pytestmark = pytest.mark.gpu

FASTV = dict(mode=O.FIXED_RATIO, tau=0.1, ratio_ppm=500_000)


@pytest.fixture(scope="module")
def vp(lib):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    return lib


def small(**kw):
    base = dict(name="small", layers=1, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                planted_frac=0.04, seed=41, beta_range=(0.3, 0.9), beta_sink=1.0, budget=W.ADAPTIVE_5PCT)
    base.update(kw)
    return W.Recipe(**base)


def _compact_on_gpu(vp, dev, kept, count, cap):
    """Compacts dev's K and V caches with the given kept sets; returns CPU
    tensors [B, Hkv, Tmax, D] (rows past each sequence's length are left 0)."""
    B, Hkv, D = dev.B, dev.Hkv, dev.D
    tmax = int(dev.cfg.max_seq)
    out = []
    for src in (dev.kc, dev.vc):
        dst_t = torch.zeros((B, Hkv, tmax, D), dtype=dev.q.dtype, device="cuda")
        vp.vp_compact_kv(dev.ctx, B, src, vp.kv_contiguous(dst_t), dev.span, dev.tl, kept, cap, count)
        out.append(dst_t)
    vp.vp_check_errors(dev.ctx)
    torch.cuda.synchronize()
    return [t.cpu() for t in out]


def _bits(t):
    """Raw element bits (numpy has no bfloat16): the comparison is bit-exact."""
    return (t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)).numpy()


def _check_compaction(inp, kc, vc, kept_np, count_np):
    for b in range(inp.recipe.batch):
        K = int(count_np[b])
        vs, nv, tl = int(inp.vis_start[b]), int(inp.vis_len[b]), int(inp.text_len[b])
        kept_b = kept_np[b][:K]
        for got, full in ((kc, inp.k), (vc, inp.v)):
            want = O.compact_cache(_bits(full[b]), vs, nv, tl, kept_b)
            np.testing.assert_array_equal(_bits(got[b, :, :K + tl]), want, err_msg=f"seq {b}")


@pytest.mark.parametrize("dtype,D", [(W.BF16, 128), (W.BF16, 64), (W.FP32, 128)])
@pytest.mark.parametrize("paged,page_size", [(False, 1), (True, 16), (True, 8)])
def test_compact_matches_oracle(vp, dtype, D, paged, page_size):
    """Random ascending kept sets, K = 0 and K = N_v included."""
    r = small(dtype=dtype, head_dim=D, paged=paged, page_size=page_size, batch=4,
              vis_len=(300, 577, 64, 1000), vis_start=(0, 13, 40, 0), text_len=(517, 70, 129, 33))
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, dict(mode=O.DENSE, tau=0.1))
    try:
        rng = np.random.default_rng(7)
        cap = int(dev.cfg.max_visual)
        kept_np = np.full((r.batch, cap), -1, dtype=np.int32)
        count_np = np.zeros(r.batch, dtype=np.int32)
        for b in range(r.batch):
            nv = int(inp.vis_len[b])
            K = (0, nv, nv // 3, 1)[b]
            kept_np[b, :K] = np.sort(rng.choice(nv, size=K, replace=False))
            count_np[b] = K
        kept = torch.from_numpy(kept_np).cuda()
        count = torch.from_numpy(count_np).cuda()
        kc, vc = _compact_on_gpu(vp, dev, kept, count, cap)
    finally:
        dev.close()
    _check_compaction(inp, kc, vc, kept_np, count_np)


@pytest.mark.parametrize("paged", [False, True])
def test_fastv_then_visionpulse(vp, paged):
    """Selection with the last prompt token (50%), compaction, then a decode
    step over the compacted caches with the adaptive budget."""
    r = small(paged=paged, page_size=16)
    inp = Hn.make_inputs(r)
    # The last prompt token's query: a second seeded query of the same recipe.
    q_last = Hn.make_inputs(r, step=1).q
    pre = dataclasses.replace(inp, q=q_last)
    dev = Hn.Device(vp, pre, FASTV)
    try:
        gpu = dev.run()
        for b in range(r.batch):
            Hn.compare_seq(pre, gpu, b, FASTV)
        count_np = gpu["count"][:, 0].astype(np.int32)
        kept_np = gpu["kept"][:, 0, :].astype(np.int32)
        for b in range(r.batch):  # FastV's ratio: ceil(N_v / 2) survivors
            assert count_np[b] == -(-int(inp.vis_len[b]) // 2)
        kc, vc = _compact_on_gpu(vp, dev, dev.kept[:, 0, :].contiguous(), dev.count[:, 0].contiguous(), dev.kept_cap)
    finally:
        dev.close()
    _check_compaction(inp, kc, vc, kept_np, count_np)
    # VisionPulse over the survivors: the compacted caches, N_v' = K.
    comp = dataclasses.replace(inp, k=kc, v=vc, vis_len=count_np.astype(inp.vis_len.dtype),
                               recipe=dataclasses.replace(r, paged=False), block_table=None, n_pages=0)
    Hn.check_all(vp, comp, r.budget)


def test_compact_reports_a_bad_kept_index(vp):
    """An index outside the visual span is skipped (its row zeroed) and
    reported by vp_check_errors; nothing faults."""
    r = small()
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, dict(mode=O.DENSE, tau=0.1))
    try:
        cap = int(dev.cfg.max_visual)
        kept = torch.zeros((r.batch, cap), dtype=torch.int32, device="cuda")
        kept[:, :3] = torch.tensor([0, 5, 1_000_000], dtype=torch.int32)
        count = torch.full((r.batch,), 3, dtype=torch.int32, device="cuda")
        dst = torch.zeros((r.batch, r.kv_heads, int(dev.cfg.max_seq), r.head_dim), dtype=dev.q.dtype, device="cuda")
        vp.vp_compact_kv(dev.ctx, r.batch, dev.kc, vp.kv_contiguous(dst), dev.span, dev.tl, kept, cap, count)
        with pytest.raises(vp.VPError) as ei:
            vp.vp_check_errors(dev.ctx)
        assert ei.value.status == vp.VP_ERR_DEVICE_PRECOND
        vs = int(inp.vis_start[0])
        assert torch.count_nonzero(dst[0, :, vs + 2]).item() == 0
    finally:
        dev.close()


def test_compact_argument_errors(vp):
    r = small(paged=True, page_size=16)
    inp = Hn.make_inputs(r)
    dev = Hn.Device(vp, inp, dict(mode=O.DENSE, tau=0.1))
    try:
        cap = int(dev.cfg.max_visual)
        kept = torch.zeros((r.batch, cap), dtype=torch.int32, device="cuda")
        count = torch.zeros((r.batch,), dtype=torch.int32, device="cuda")
        # A paged destination, the source as destination, a batch above max_batch.
        for dst, batch, want in ((dev.kc, r.batch, vp.VP_ERR_INVALID_ARG),
                                 (vp.kv_contiguous(dev.k_t.reshape(-1, r.kv_heads, r.page_size, r.head_dim)),
                                  r.batch, vp.VP_ERR_INVALID_ARG),
                                 (vp.kv_contiguous(torch.zeros((r.batch + 1, r.kv_heads, 8, r.head_dim),
                                                               dtype=dev.q.dtype, device="cuda")),
                                  r.batch + 1, vp.VP_ERR_CAPACITY)):
            st = vp.vp_compact_kv(dev.ctx, batch, dev.kc, dst, dev.span, dev.tl, kept, cap, count, check=False)
            assert st == want, st
    finally:
        dev.close()


def test_compaction_then_decode_on_one_stream(vp):
    """vp_compact_kv followed at once by vp_decode_step over the compacted
    caches, on one stream with no host synchronisation in between: the decode
    step reads its caches before it waits for the previous kernel, so the
    compaction must have completed by the time it starts.  The result must be
    bit-identical to the same calls with a synchronisation between them."""
    r = small(vis_len=(1500, 577, 64), text_len=(2500, 70, 129))  # a compaction of a few MB
    inp = Hn.make_inputs(r)
    q_last = Hn.make_inputs(r, step=1).q
    dev = Hn.Device(vp, dataclasses.replace(inp, q=q_last), FASTV)
    try:
        dev.run()  # FastV's selection with the last prompt token
        kept, count = dev.kept[:, 0, :].contiguous(), dev.count[:, 0].contiguous()
        span_c = vp.span(dev.vs, count)  # the survivors form the new visual span
        decode_q = inp.q.cuda()
        bd = vp.make_budget(**r.budget)
        cap = max(1, vp.vp_max_kept(bd, dev.cfg.max_visual))
        results = []
        for sync in (True, False):
            dst = [torch.zeros_like(dev.k_t), torch.zeros_like(dev.v_t)]
            for src, d in zip((dev.kc, dev.vc), dst):
                vp.vp_compact_kv(dev.ctx, dev.B, src, vp.kv_contiguous(d), dev.span, dev.tl, kept, dev.kept_cap,
                                 count)
            if sync:
                torch.cuda.synchronize()
            out = torch.full_like(dev.out, float("nan"))
            kept2 = torch.full((dev.B, cap), -7, dtype=torch.int32, device="cuda")
            count2 = torch.full((dev.B,), -7, dtype=torch.int32, device="cuda")
            mass = torch.empty_like(dev.mass)
            stats = torch.empty_like(dev.stats)
            vp.vp_decode_step(dev.ctx, dev.B, decode_q, vp.kv_contiguous(dst[0]), vp.kv_contiguous(dst[1]), span_c,
                              dev.tl, bd, out, kept2, cap, count2, mass, stats)
            vp.vp_check_errors(dev.ctx)
            torch.cuda.synchronize()
            results.append((_bits(out.cpu()), kept2.cpu().numpy(), count2.cpu().numpy()))
    finally:
        dev.close()
    for a, b in zip(results[0], results[1]):
        np.testing.assert_array_equal(a, b)
    assert (results[0][2] > 0).all()
