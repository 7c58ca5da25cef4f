"""Host-side accounting of bench.py (CPU only): the algorithmic bytes and
flops behind every roofline fraction, and the clock record that decides
whether a timed region stands.

The byte and flop counts are checked against closed forms for the 7B-shaped
workload's known tree (a 48-token reuse chain from the root, an 8-node branch
off the root and one off chain node 24; ctx 4096; 28 query / 4 KV heads of
128; vocab 152064, hidden 3584).
"""
import os
import subprocess
import sys
import tempfile

import pytest

import bench
import workloads as W


@pytest.fixture(scope="module")
def w7b():
    return W.build("7b", layers=1, lm_head=False)


def test_7b_tree_is_the_stated_shape(w7b):
    par = [int(x) for x in w7b.parent]
    assert par[:48] == [-1] + list(range(47))                       # root + 47-node chain
    assert par[48] == 0 and par[49:56] == list(range(48, 55))       # branch off the root
    assert par[56] == 24 and par[57:64] == list(range(56, 63))      # branch off chain node 24
    assert int(w7b.ctx_len[0]) == 4096 and w7b.total_nodes == 64


def test_7b_algorithmic_bytes_and_flops(w7b):
    a = bench.algorithmic(w7b)
    ctx, T, n_q, n_kv, d = 4096, 64, 28, 4, 128
    kv_context = 2 * ctx * n_kv * d * 2                   # K and V, bf16: 8 MiB per layer
    assert kv_context == 8 * 2 ** 20
    assert a["attn_bytes"] == kv_context + T * n_q * d * 2 + 2 * T * n_kv * d * 2 + T * n_q * d * 4
    # keys seen per node: ctx + depth + 1; depths: chain 1..47, root branch 1..8, chain-24 branch 25..32
    sum_depth = sum(range(1, 48)) + sum(range(1, 9)) + sum(range(25, 33))
    assert sum_depth == 1392
    assert a["attn_flops"] == 4 * n_q * d * (T * (ctx + 1) + sum_depth) == 3_778_969_600
    V, H = 152064, 3584
    assert a["lm_bytes"] == V * H * 2 + T * H * 2 + T * 4 * 2
    assert V * H * 2 == 1_089_994_752                     # the LM-head weight, 1.09 GB
    assert a["lm_flops"] == 2 * T * H * V
    acc = int(w7b.planted_accept[0])
    assert a["comp_bytes"] == (acc + 1) * 1 * n_kv * d * 2 * 2 * 2   # one layer, K+V, read+write
    assert a["draft_nodes"] == T - 1


@pytest.mark.parametrize("clk,why", [
    (None, None),
    ({"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}, None),
    ({"sm_mhz": 1450.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}, None),
    ({"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["hw_slowdown"]}, "hw_slowdown"),
    ({"sm_mhz": 1900.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap", "sw_thermal_slowdown"]},
     "sw_thermal_slowdown"),
    ({"sm_mhz": 1005.0, "sm_max_mhz": 2070.0, "reasons": []}, "no reason"),
])
def test_clock_record_rejects_slowdowns_and_stuck_clocks(clk, why):
    got = bench.clocks_rejected(clk)
    if why is None:
        assert got is None
    else:
        assert got is not None and why in got


def test_clock_sampler_parses_nvidia_smi_rows():
    s = bench.ClockSampler(0)
    s.file = tempfile.NamedTemporaryFile("w+", delete=False, suffix=".csv")
    s.file.write("2026/12/02 15:20:45.100, 2070, 2070, 812.4, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n"
                 "2026/12/02 15:20:45.120, 2070, 2070, 1190.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n"
                 "2026/12/02 15:20:45.140, 1980, 2070, 1375.2, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n"
                 "2026/12/02 15:20:45.160, [N/A], 2070, [N/A], [N/A], [N/A], [N/A], [N/A], [N/A]\n")
    s.proc = subprocess.Popen(["sleep", "30"])
    clk = s.stop()                                   # no region marks: every row counts
    assert clk["samples"] == 3 and clk["sm_mhz"] == 2070.0 and clk["sm_max_mhz"] == 2070.0
    assert clk["reasons"] == ["sw_power_cap"]
    assert bench.clocks_rejected(clk) is None


def _rows(*spec):
    """nvidia-smi rows at the given local times (seconds after 15:20:45) with the given SM clock and
    hw_slowdown state."""
    out = []
    for t, mhz, slow in spec:
        ms = int(round(t * 1000))
        stamp = f"2026/12/02 15:20:{45 + ms // 1000:02d}.{ms % 1000:03d}"
        out.append([stamp, str(mhz), "2070", "900", "0x0", "Active" if slow else "Not Active",
                    "Not Active", "Not Active", "Not Active"])
    return out


def _t(sec):
    import datetime
    return datetime.datetime(2026, 12, 2, 15, 20, 45).timestamp() + sec


def test_clock_record_keeps_only_samples_inside_the_timed_region():
    """Samples before and after the timed region (here a slowdown during a
    later, untimed pass) do not count."""
    rows = _rows((0.00, 1500, False), (0.02, 2070, False), (0.04, 2070, False), (0.06, 2070, False),
                 (0.08, 1200, True))
    clk = bench.summarize_clock_rows(rows, _t(0.015), _t(0.065))
    assert clk["samples"] == 3 and clk["samples_in_region"] == 3 and clk["sm_mhz"] == 2070.0
    assert clk["reasons"] == [] and bench.clocks_rejected(clk) is None
    assert clk["region_ms"] == 50.0


def test_clock_record_of_a_region_shorter_than_the_sampling_period():
    """A 12 ms region between two 20 ms samples: the nearest sample on each
    side stands in, and the record says that none fell inside."""
    rows = _rows((0.00, 1500, False), (0.02, 2070, False), (0.04, 2070, True), (0.06, 2070, False))
    clk = bench.summarize_clock_rows(rows, _t(0.025), _t(0.037))
    assert clk["samples_in_region"] == 0 and clk["samples"] == 2
    assert clk["reasons"] == ["hw_slowdown"] and bench.clocks_rejected(clk) == "hw_slowdown"


def test_clock_sampler_without_nvidia_smi_reports_nothing():
    s = bench.ClockSampler(0)
    assert s.stop() is None


def test_reference_arm_runs_on_rank_0_only():
    """Under torchrun the reference arm (the oracle on the host cores) runs on
    rank 0 alone; every other rank exits 0 at once, without work or output."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "3"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_single_thread_oracle_baseline_runs_in_a_child():
    rec = bench.oracle_single_thread("tiny", 1, 4096, budget_s=0.5)
    assert "error" not in rec, rec
    assert rec["cores"] == 1 and rec["value"] > 0 and "one thread" in rec["sample"]
    assert "vocab rows 0..255 of 4096 (x16.0)" in rec["sample"]
