"""GPU parity of the diagnostics (vp_set_diagnostics): the active visual
token count N_act(delta) of Sec. 4.3 and the OR-accumulated activity bits
behind App. B's persistent inactivity, against the oracle's active_count.

Scores near delta may be decided differently by the float32 kernel and the
float64 oracle (rounded to float32): tokens whose oracle score lies within
TIE_DELTA (relative) of delta may differ; every other token must agree.
"""

import numpy as np
import pytest
import torch

from oracle import vp_oracle as O
from paper_2605_31457_gb300 import workloads as W

from . import vp_harness as Hn

pytestmark = pytest.mark.gpu

TIE_DELTA = 1e-4


@pytest.fixture(scope="module")
def vp(lib):
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device")
    return lib


def _compare(s, delta, n_gpu, flags_gpu):
    """s: oracle scores [..., N_v]; flags_gpu: GPU flags of the same shape."""
    n_ref, flags_ref = O.active_count(s, delta)
    near = np.abs(np.asarray(s, dtype=np.float64) - delta) <= TIE_DELTA * delta
    assert not np.any((flags_ref != flags_gpu) & ~near), "activity differs away from delta"
    assert np.all(np.abs(np.asarray(n_gpu) - n_ref) <= near.sum(axis=-1))


def _bits_to_flags(bits, nv):
    b = bits.astype(np.uint32)
    return ((b[..., None] >> np.arange(32, dtype=np.uint32)) & 1).reshape(*b.shape[:-1], -1)[..., :nv].astype(bool)


@pytest.mark.parametrize("delta", [1e-3, 3e-3])
def test_active_count_and_bits_over_a_decode(vp, delta):
    """Every step of the 16-step reference workload: N_act per step, and the
    activity bits OR-ed over the steps equal the union of the oracle's flags."""
    r = W.TINY
    li = W.make_layer(r, 0, t_cap=r.capacity())
    qs = W.make_queries(r, 0, li)
    nv = int(r.vis_lens[0])
    words = (nv + 31) // 32
    bits = torch.zeros((1, words), dtype=torch.int32, device="cuda")
    n_act = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    union = np.zeros(nv, dtype=bool)
    near_any = np.zeros(nv, dtype=bool)
    for step in range(r.steps):
        inp = Hn.make_inputs(r, 0, step, t_cap=r.capacity(), q_override=qs[step])
        dev = Hn.Device(vp, inp, r.budget)
        try:
            vp.vp_set_diagnostics(dev.ctx, delta, n_act, bits)
            dev.run()
            n_gpu = int(n_act.cpu()[0])
        finally:
            dev.close()
        s = Hn.oracle_seq(inp, 0, r.budget)["s"]
        flags_step = np.asarray(s, dtype=np.float32) > np.float32(delta)
        _compare(s, delta, n_gpu, flags_step)
        union |= flags_step
        near_any |= np.abs(s - delta) <= TIE_DELTA * delta
    got = _bits_to_flags(bits.cpu().numpy().view(np.uint32)[0], nv)
    assert not np.any((got != union) & ~near_any)
    assert 0 < got.sum() < nv, "expected both active and persistently inactive tokens"


def test_active_count_per_kv_head_and_batch(vp):
    r = W.Recipe(name="small", layers=1, batch=3, heads=28, kv_heads=4, head_dim=128, dtype=W.BF16,
                 vis_len=(300, 577, 64), vis_start=(0, 13, 40), text_len=(517, 70, 129), steps=1,
                 planted_frac=0.04, seed=11, beta_range=(0.3, 0.9), beta_sink=1.0, budget=W.ADAPTIVE_5PCT)
    budget = dict(r.budget, granularity=1)
    inp = Hn.make_inputs(r)
    delta = 2e-3
    words = (577 + 31) // 32
    bits = torch.zeros((3, 4, words), dtype=torch.int32, device="cuda")
    n_act = torch.full((3, 4), -1, dtype=torch.int32, device="cuda")
    dev = Hn.Device(vp, inp, budget)
    try:
        vp.vp_set_diagnostics(dev.ctx, delta, n_act, bits)
        dev.run()
    finally:
        dev.close()
    n_gpu = n_act.cpu().numpy()
    flags = _bits_to_flags(bits.cpu().numpy().view(np.uint32), 577)
    for b in range(3):
        nv = int(inp.vis_len[b])
        s = Hn.oracle_seq(inp, b, budget)["s"]          # [Hkv, N_v]
        _compare(s, delta, n_gpu[b], flags[b][:, :nv])
        assert not flags[b][:, nv:].any()


def test_diagnostics_off_and_bad_delta(vp):
    r = W.TINY
    inp = Hn.make_inputs(r, 0, 0)
    n_act = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    dev = Hn.Device(vp, inp, r.budget)
    try:
        vp.vp_set_diagnostics(dev.ctx, 1e-3, n_act, None)
        vp.vp_set_diagnostics(dev.ctx, 0.0, None, None)       # off
        dev.run()
        assert int(n_act.cpu()[0]) == -7
        for bad in (0.0, -1.0, float("nan"), float("inf")):
            with pytest.raises(vp.VPError) as ei:
                vp.vp_set_diagnostics(dev.ctx, bad, n_act, None)
            assert ei.value.status == vp.VP_ERR_INVALID_ARG
    finally:
        dev.close()
