"""Host-side logic of bench.py (no GPU): the clock-record summary that decides
whether a measurement stands, and the lookup of ncu DRAM traffic keyed by the
kernel source's digest."""

import hashlib
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _line(sm, mx, active="0x0", hw="Not Active", hwt="Not Active", swt="Not Active",
          pcap="Not Active"):
    return f"0, {sm}, {mx}, 900.5, {active}, {hw}, {hwt}, {swt}, {pcap}"


def test_clock_summary_median_and_reasons():
    c = bench.ClockSampler(0)
    c.lines = [_line(2070, 2070), _line(1980, 2070, pcap="Active"), _line(2070, 2070),
               "garbage", _line(2010, 2070)]
    s = c.summary()
    assert s["samples"] == 4
    assert s["sm_mhz"] == pytest.approx(2040.0)          # median of 2070, 1980, 2070, 2010
    assert s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"]


def test_clock_summary_reports_thermal_slowdown():
    c = bench.ClockSampler(0)
    c.lines = [_line(1500, 2070, hwt="Active"), _line(1400, 2070, swt="Active", hw="Active")]
    s = c.summary()
    assert s["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]


def test_clock_summary_without_samples():
    c = bench.ClockSampler(0)
    c.lines = []
    assert c.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}


def _fake_root(tmp_path, src_text, digest_text):
    csrc = tmp_path / "paper_1710_02368_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "mlp_tc_dw.cu").write_text(src_text)
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "dram_traffic.txt").write_text(
        "# kernel_class workload bytes digest\n"
        f"backward_dw wl-a 1234 {digest_text}\n"
        f"backward_dw wl-b 99 000000000000\n")
    return str(tmp_path)


def test_traffic_lookup_matches_digest(tmp_path, monkeypatch):
    src = "// kernel source\n"
    digest = hashlib.sha256(src.encode()).hexdigest()[:12]
    monkeypatch.setattr(bench, "ROOT", _fake_root(tmp_path, src, digest))
    assert bench._traffic_for("backward_dw", "wl-a", True) == 1234.0
    assert bench._traffic_for("backward_dw", "wl-b", True) is None   # stale digest
    assert bench._traffic_for("backward_dw", "wl-c", True) is None   # no capture
    assert bench._traffic_for("gather", "wl-a", True) is None        # no source mapped


def test_traffic_lookup_ignores_a_changed_kernel(tmp_path, monkeypatch):
    src = "// kernel source\n"
    digest = hashlib.sha256(src.encode()).hexdigest()[:12]
    root = _fake_root(tmp_path, src, digest)
    (tmp_path / "paper_1710_02368_gb300" / "csrc" / "mlp_tc_dw.cu").write_text(src + "// edit\n")
    monkeypatch.setattr(bench, "ROOT", root)
    assert bench._traffic_for("backward_dw", "wl-a", True) is None


def test_committed_traffic_entries_are_well_formed():
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    assert rows
    for r in rows:
        assert len(r) == 4
        assert r[0] in ("forward", "forward_head", "backward_dx", "backward_dw", "softmax",
                        "commit")
        assert float(r[2]) > 0
        assert len(r[3]) == 12 and all(ch in "0123456789abcdef" for ch in r[3])


def test_commit_launch_grouping_and_bytes():
    """The standalone commit workload's launches (runs of <= 16 commits, cut at
    a repeated worker or past 256 pulls) and the bytes a pass must move:
    theta~ 8P per launch, 8P per commit, 4P per pull."""
    order, pulls = list(range(64)), [[1, 2, 3, 4]] * 64
    assert bench.commit_plan_launches(order, pulls) == 4
    assert bench.commit_plan_launches([0, 1, 0, 2], [[]] * 4) == 2
    assert bench.commit_plan_launches(list(range(8)), [list(range(100))] * 8) == 4
    P = 1 << 20
    assert bench.commit_pass_bytes(P, 64, 256, 4) == P * (8 * 4 + 8 * 64 + 4 * 256)


def test_method_bytes_of_the_dw_class_by_hand():
    """784-1000-1000-10 fp32, m = 128: theta_k and a_k read-modify-write,
    16 B per parameter (P = 1,796,010), plus the operands of the three layers'
    weight gradients (dZ_l and H_{l-1}, 4 B each)."""
    from agn_inputs import workloads as WL
    wl = WL.MNIST_SHAPED
    got = bench.method_bytes_per_worker_step(wl, "backward_dw")
    assert got == 16 * 1796010 + 128 * 4 * ((1000 + 784) + (1000 + 1000) + (10 + 1000))
    bf = bench.method_bytes_per_worker_step(WL.LARGE_BF16, "backward_dw")
    assert bf == 18 * 20037642 + 64 * 2 * ((4096 + 784) + (4096 + 4096) + (10 + 4096))


def test_method_bytes_of_the_forward_classes_split_at_the_fused_launch():
    """With the output layer in the last hidden layer's forward, the forward
    class covers the other hidden layers and forward_head that layer plus the
    output layer; together they count each layer once."""
    from agn_inputs import workloads as WL
    wl = WL.MNIST_SHAPED
    plain = bench.method_bytes_per_worker_step(wl, "forward")
    first = bench.method_bytes_per_worker_step(wl, "forward", fused_head=True)
    head = bench.method_bytes_per_worker_step(wl, "forward_head")
    out = bench.method_bytes_per_worker_step(wl, "softmax")
    assert first == 1000 * 784 * 4 + 4 * 1000 + 128 * (784 + 1000) * 4
    assert abs((first + head) - (plain + out)) <= 4 * 128 * 1000 + 1e-6
