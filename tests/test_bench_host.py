"""Host logic of bench.py on the CPU: the algorithmic byte count of a layer
call, the workload table and the clock summary.  No GPU work runs here."""

import pytest

import bench
from paper_2605_31457_gb300 import workloads as W


def test_call_bytes_is_the_roofline_formula():
    """Per sequence and layer call: all visual K, text K and V, q and out read
    or written once; the gather reads only the kept visual V rows."""
    r = W.QWEN7B                                    # 4 kv-heads x 128 dims, bf16
    row = 4 * 128 * 2
    qo = 28 * 128 * 2
    score, gather = bench.call_bytes(r, 1296, 2561, 64)
    assert score == 1296 * row + 2 * 2561 * row + qo == 6579200
    assert gather == 64 * row + qo
    # No visual span: text only.  Dense: every visual V row.
    assert bench.call_bytes(r, 0, 10, 0) == (2 * 10 * row + qo, qo)
    assert bench.call_bytes(r, 1296, 1, 1296)[1] == 1296 * row + qo
    # fp32 caches: twice the bytes per element.
    r32 = W.TINY                                    # 2 kv-heads x 64 dims, fp32, 8 query heads
    assert bench.call_bytes(r32, 576, 129, 28) == (576 * 2 * 64 * 4 + 2 * 129 * 2 * 64 * 4 + 8 * 64 * 4,
                                                   28 * 2 * 64 * 4 + 8 * 64 * 4)


@pytest.mark.parametrize("name,batch,layers", [
    ("qwen7b", 1, 28), ("qwen7b-10pct", 1, 28), ("qwen7b-anchor", 1, 28), ("qwen7b-fastv-vp", 1, 28),
    ("serving", 32, 28), ("long", 8, 28), ("sweep-576-r1", 64, 1), ("sweep-16384-adaptive", 64, 1),
])
def test_workloads(name, batch, layers):
    r, steps, nbuf, host_gen = bench.pick_workload(name)
    assert (r.batch, r.layers) == (batch, layers) and steps > 0 and 1 <= nbuf <= r.layers
    cfg = bench.workload_config(r, nbuf)
    assert cfg["global_batch"] == batch and r.name in cfg["workload"]


def test_ten_percent_setting_uses_the_paper_budget():
    r = bench.pick_workload("qwen7b-10pct")[0]
    assert r.budget == W.ADAPTIVE_10PCT and "tau=0.4 clamp [5%, 10%]" in bench.workload_config(r)["workload"]


def test_unknown_workload_is_refused():
    with pytest.raises(SystemExit):
        bench.pick_workload("no-such-workload")


def test_clock_summary():
    # Idle samples (bit 0x1) are left out while busy ones exist; reasons are the
    # union over the busy samples, without the idle bit.
    c = bench.ClockSampler.summarize([(2070, 0x0), (1980, 0x4), (345, 0x1), (2070, 0x8)], 2070)
    assert c["sm_mhz"] == 2070 and c["samples"] == 3 and c["sm_max_mhz"] == 2070
    assert c["reasons"] == ["sw_power_cap", "hw_slowdown"]
    idle = bench.ClockSampler.summarize([(345, 0x1), (345, 0x1)], 2070)
    assert idle["samples"] == 2 and idle["reasons"] == []
    assert bench.ClockSampler.summarize([], 2070)["sm_mhz"] is None


def test_tiny_workload_and_config_table():
    r, steps, nbuf, host_gen = bench.pick_workload("tiny")
    assert r is W.TINY and nbuf == 1 and host_gen and bench.compute_dtype(r) == "f32"
    names = bench.config_workloads()
    assert names[:3] == ["tiny", "qwen7b", "serving"]
    sweep = [n for n in names if n.startswith("sweep-")]
    assert len(sweep) == 20 and len(set(sweep)) == 20
    for n in sweep:
        rr = bench.pick_workload(n)[0]
        assert rr.batch == 64 and int(rr.vis_lens[0]) in W.SWEEP_VIS
    assert bench.pick_workload("sweep-576-r20")[0].budget == W.SWEEP_BUDGETS[2]
    with pytest.raises(SystemExit):
        bench.pick_workload("sweep-576-r7")


def test_l2_flush_only_for_steps_that_fit_in_l2():
    assert bench.needs_l2_flush(W.TINY, 1)                 # 0.4 MB per step
    assert not bench.needs_l2_flush(W.QWEN7B, 28)          # 28 distinct caches, ~0.18 GB per step
    assert not bench.needs_l2_flush(W.LONG, 4)
    assert not bench.needs_l2_flush(W.sweep_recipe(576, W.ADAPTIVE_5PCT), 1)
    assert "L2 flushed" in bench.workload_config(W.TINY, 1, True)["l2"]


def test_committed_traffic_matches_workload_kernel_and_sources(tmp_path):
    p = tmp_path / "t.json"
    import json
    p.write_text(json.dumps({"captures": [
        {"kernel_prefix": "k_score_tc", "workload": "long", "source_sha256": "abc",
         "dram_bytes_per_launch": [110.0, 130.0], "algorithmic_bytes_per_launch": 100.0}]}))
    t, why = bench.committed_traffic("k_score_tc", "long", 1000.0, path=str(p), sha="abc")
    assert t == pytest.approx(1200.0) and "scaled" in why
    assert bench.committed_traffic("k_score_tc", "serving", 1000.0, path=str(p), sha="abc")[0] is None
    assert bench.committed_traffic("k_score_tma", "long", 1000.0, path=str(p), sha="abc")[0] is None
    t, why = bench.committed_traffic("k_score_tc", "long", 1000.0, path=str(p), sha="other")
    assert t is None and "predates" in why
    assert bench.committed_traffic("k_score_tc", "long", 1.0, path=str(tmp_path / "none.json"))[0] is None


@pytest.mark.timeout(300)
def test_oracle_pool_times_whole_steps():
    """The CPU baseline: every (layer, sequence) call of a step on a pool of
    spawned processes; a step's time scales to the whole batch when only its
    first sequences are sampled."""
    r = W.shrink(W.TINY, batch=3, vis_len=(64, 32, 16), vis_start=(0, 2, 5), text_len=(20, 9, 30))
    pool = bench.OraclePool(r, 2, n_caches=1, workers=2)
    try:
        t = [pool.step(s) for s in range(2)]
        assert all(x > 0 for x in t) and pool.workers == 2 and pool.r.batch == 3
        assert "2 whole decode step(s)" in pool.sample_text(2)
    finally:
        pool.close()
    small = bench.OraclePool(r, 1, n_caches=1, workers=1, max_bytes=1.0)   # one sequence fits
    try:
        assert small.r.batch == 1 and "the first 1 of 3 sequences" in small.sample_text(1)
        assert small.step(0) > 0
    finally:
        small.close()
