"""Host logic of bench.py that needs no GPU: the clock sampler keeps only
the samples taken while the timed region ran, and says so when the region
was too short to catch one."""
import bench


def _line(sm, reasons=("Not Active",) * 4):
    return f"0, {sm}, 2070, 900.0, 0x0, " + ", ".join(reasons)


def test_clock_summary_uses_the_timed_window_only():
    cs = bench.ClockSampler(0)
    cs.lines = [(0.0, _line(345)), (0.10, _line(345)),           # idle, before the region
                (1.00, _line(2070)), (1.02, _line(2065)),          # during
                (1.30, _line(2070, ("Not Active",) * 3 + ("Active",)))]   # after, power capped
    res = cs.summarise(0.99, 1.03)
    assert res["window"] == "timed region"
    assert res["samples"] == 2 and res["sm_mhz"] == 2067.5
    assert res["reasons"] == [] and res["sm_max_mhz"] == 2070.0


def test_clock_summary_falls_back_and_says_so():
    cs = bench.ClockSampler(0)
    cs.lines = [(0.0, _line(2070)), (0.5, _line(2070, ("Active", "Not Active", "Not Active", "Not Active")))]
    res = cs.summarise(0.2, 0.21)
    assert res["window"].startswith("around the timed region")
    assert res["samples"] == 2 and res["reasons"] == ["hw_slowdown"]


def test_clock_summary_without_samples_is_none():
    assert bench.ClockSampler(0).summarise(0.0, 1.0) is None
