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
