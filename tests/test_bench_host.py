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


def _args(phase):
    return dict(config=0, w=1.0, phase=phase, seed=0, max_tokens=0, structured=False)


def test_oracle_baseline_times_the_phase_it_names():
    """The CPU baseline's steady phase times steps at budget occupancy (the
    first window, full trace and eviction, runs untimed); the full-trace
    phase times the first step over the whole trace."""
    import synth
    w = synth.make_workload(0)
    full = bench._oracle_worker((_args("full"), 0, w.L, 2))
    assert len(full) == 2 and all(tok == w.n0(0) + 1 for _, _, tok in full)
    steady = bench._oracle_worker((_args("steady"), 0, w.L, 2))
    assert len(steady) == 2
    cap = w.budget_pages[0] * w.page_size
    for dec, ev, tok in steady:
        assert dec > 0 and ev > 0
        assert cap - w.page_size < tok <= cap + 1    # at the budget, not the whole trace
