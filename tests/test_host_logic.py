"""Host-side measurement logic, on the CPU: the link fraction of a set of moving events
(each event's best time on the link for its own mix of bytes out and in, summed, over the
measured time) and the whole-job aggregate over ranks.  Values worked by hand."""
import pytest

from paper_2606_22983_gb300.runner import link_summary


def test_link_summary_by_hand():
    # peaks in GB/s: 100 one way out, 200 one way in, 250 both ways at once
    peaks = {"d2h": 100.0, "h2d": 200.0, "bidir": 250.0}
    GB = 1e9
    moves = [
        # (ms, bytes out, bytes in, kind)
        (10.0, 1 * GB, 0, 8),        # offload only: best 1 GB / 100 GB/s = 10 ms -> 1.0
        (10.0, 0, 1 * GB, 7),        # reload only:  best 1 GB / 200 GB/s = 5 ms  -> 0.5
        (10.0, 1 * GB, 1 * GB, 7),   # both: max(10 ms, 5 ms, 2 GB / 250 GB/s = 8 ms) = 10 ms -> 1.0
        (16.0, 0.5 * GB, 2 * GB, 1),  # both: max(5, 10, 10) = 10 ms over 16 ms -> 0.625
    ]
    out = link_summary(moves, peaks, {1: "TURN", 7: "TURN_SCATTER", 8: "EVICT"})
    assert out["events"] == 4
    assert out["device_s"] == pytest.approx(0.046)
    assert out["link_best_s"] == pytest.approx(0.035)
    assert out["link_frac"] == pytest.approx(round(35 / 46, 3))
    assert out["gb_out"] == pytest.approx(2.5) and out["gb_in"] == pytest.approx(4.0)
    assert out["gbs"] == pytest.approx(round(6.5 / 0.046, 1))
    kinds = out["by_event_kind"]
    assert kinds["EVICT"]["link_frac"] == pytest.approx(1.0)
    assert kinds["TURN_SCATTER"]["link_best_s"] == pytest.approx(0.015)
    assert kinds["TURN_SCATTER"]["link_frac"] == pytest.approx(0.75)
    assert kinds["TURN"]["link_frac"] == pytest.approx(0.625)
    d = out["by_direction"]
    assert d["offload_only"]["events"] == 1 and d["offload_only"]["link_frac"] == pytest.approx(1.0)
    assert d["reload_only"]["events"] == 1 and d["reload_only"]["link_frac"] == pytest.approx(0.5)
    assert d["both"]["events"] == 2 and d["both"]["link_best_s"] == pytest.approx(0.020)
    assert d["both"]["link_frac"] == pytest.approx(round(20 / 26, 3))


def test_link_summary_without_moves_or_peaks():
    assert link_summary([], {"d2h": 1.0, "h2d": 1.0, "bidir": 1.0}, {}) is None
    assert link_summary([(1.0, 1, 1, 7)], {"d2h": 1.0}, {}) is None


def test_aggregate_is_all_bytes_over_the_slowest_rank():
    import importlib.util
    import os
    spec = importlib.util.spec_from_file_location(
        "bench_module", os.path.join(os.path.dirname(os.path.dirname(__file__)), "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    assert bench.aggregate([4e9, 6e9], [2.0, 2.5]) == pytest.approx(4e9)
    assert bench.aggregate([1e9], [0.0]) == 0.0
