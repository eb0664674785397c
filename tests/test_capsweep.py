"""The power-cap calibration (paper_2609_11133_gb300/capsweep.py) against a fake NVML.

No test here touches a GPU or its settings: the fake records every limit it is asked to set.
Covered: no limit changes without permission; the limit found on entry is restored and read back,
also after an error; caps outside the GPU's range are refused; the acceptance gate needs both the
throughput and the latency criterion (Algorithm 2); the mode ladder from a flat-then-cliff sweep
(Section 3.2, Figure 3's shape); the median reference resists one noisy repetition; a changed
engine fingerprint invalidates the result; the command line changes nothing without
--set-power-limits; static clock locks need permission and are released, also after an error;
the actuator A/B picks its lock arms by the rules of Section 5.3."""
import pytest

from paper_2609_11133_gb300 import capsweep as cs


class FakeNvml:
    def __init__(self, limit_w=1100, default_w=1400, lo_w=200, hi_w=1400, obey=True):
        self.limit = limit_w * 1000
        self.default = default_w * 1000
        self.lo, self.hi = lo_w * 1000, hi_w * 1000
        self.obey = obey
        self.sets = []

    def get_limit_mw(self):
        return self.limit

    def get_default_limit_mw(self):
        return self.default

    def get_constraints_mw(self):
        return self.lo, self.hi

    def set_limit_mw(self, mw):
        self.sets.append(mw)
        if self.obey:
            self.limit = mw

    def energy_mj(self):
        return 0


def curve(nvml, natural_w=900.0, cliff_w=430.0, t0=270000.0, p99_ok_ms=0.3, slow_below_w=0.0,
          noise=None):
    """A Measure whose results follow the fake's current limit: throughput flat down to the
    cliff and collapsing below it, draw = min(cap, natural), per-step p99 inflated below
    slow_below_w."""
    calls = {"n": 0}

    def run(reps):
        cap = nvml.limit / 1000.0
        draw = min(cap, natural_w)
        t = t0 if cap >= cliff_w else t0 * (cap / cliff_w) ** 3
        tput = [t] * reps
        if noise is not None and calls["n"] == 0:
            tput[0] = t * noise  # one slow repetition of the reference
        calls["n"] += 1
        p99 = p99_ok_ms * (3.0 if cap < slow_below_w else 1.0)
        return cs.CapPoint(None, tput, p99, draw / t, draw)

    return run


CAPS = [1000, 900, 800, 700, 600, 550, 500, 450, 400, 350]
FP = {"abi_version": "100", "kernel_sources": "abc"}


def test_no_limit_changes_without_permission():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv) as g:
        with pytest.raises(PermissionError):
            g.apply(800)
        with pytest.raises(PermissionError):
            cs.sweep(g, CAPS, curve(nv), 3)
    assert nv.sets == [] and nv.limit == 1400 * 1000


def test_sweep_restores_the_limit_it_found():
    nv = FakeNvml(limit_w=1100)  # someone else's limit, not the default
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv), 3)
    assert [p.cap_w for p in pts] == sorted(CAPS, reverse=True)
    assert ref.cap_w is None and ref.power_w == 900.0  # measured at the hardware default
    assert nv.sets[0] == 1400 * 1000 and nv.sets[1:len(CAPS) + 1] == [c * 1000 for c in pts_caps()]
    assert nv.limit == 1100 * 1000 and nv.sets[-1] == 1100 * 1000


def pts_caps():
    return sorted(CAPS, reverse=True)


def test_limit_restored_after_an_error():
    nv = FakeNvml(limit_w=1400)
    inner = curve(nv)
    n = {"i": 0}

    def failing(reps):
        n["i"] += 1
        if n["i"] == 3:
            raise RuntimeError("measurement failed")
        return inner(reps)

    with pytest.raises(RuntimeError, match="measurement failed"):
        with cs.CapGuard(nv, allow_set=True) as g:
            cs.sweep(g, CAPS, failing, 2)
    assert nv.limit == 1400 * 1000 and nv.sets[-1] == 1400 * 1000


def test_out_of_range_cap_is_refused():
    nv = FakeNvml(lo_w=200, hi_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        with pytest.raises(ValueError):
            g.apply(150)
        with pytest.raises(ValueError):
            g.apply(1500)
    assert nv.sets == []


def test_a_limit_that_does_not_read_back_is_an_error():
    nv = FakeNvml(obey=False)
    with pytest.raises(RuntimeError, match="read back"):
        with cs.CapGuard(nv, allow_set=True) as g:
            g.apply(800)


def test_gate_needs_throughput_and_latency():
    p = lambda t, l: cs.CapPoint(500.0, [t, t, t], l, 1.0, 500.0)
    assert cs.accept(p(99.0, 1.0), 100.0, 0.02, 1.0)
    assert not cs.accept(p(97.9, 1.0), 100.0, 0.02, 1.0)   # throughput below (1 - eps) T_ref
    assert not cs.accept(p(100.0, 1.01), 100.0, 0.02, 1.0)  # tail latency above the SLO
    assert not cs.accept(p(90.0, 2.0), 100.0, 0.02, 1.0)


def test_mode_ladder_from_a_flat_then_cliff_sweep():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv, natural_w=900.0, cliff_w=430.0), 3)
    art = cs.calibrate(ref, pts, 0.02, 1.0, FP)
    # caps at or above the natural draw cap nothing; 400 and 350 fall off the cliff
    assert art.accepted_w == [450.0, 500.0, 550.0, 600.0, 700.0, 800.0]
    assert art.modes == {"PERF": 900.0, "BAL": 700.0, "EFF": 450.0}  # BAL: nearest (450+900)/2
    assert art.modes["EFF"] <= art.modes["BAL"] <= art.modes["PERF"]
    assert art.min_energy_w == 450.0  # the fewest J/token sits just above the cliff
    assert art.note == ""


def test_latency_criterion_rejects_caps_throughput_alone_accepts():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv, slow_below_w=600.0), 3)
    art = cs.calibrate(ref, pts, 0.02, 0.5, FP)  # p99 0.3 ms above 600 W, 0.9 ms below
    assert art.modes["EFF"] == 600.0
    by_tput_only = [p.cap_w for p in pts if p.throughput >= 0.98 * ref.throughput]
    assert min(by_tput_only) == 450.0  # what a throughput-only gate would have picked


def test_median_reference_resists_one_noisy_repetition():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv, noise=0.7), 5)
    assert ref.throughput == 270000.0
    assert cs.calibrate(ref, pts, 0.02, 1.0, FP).modes["EFF"] == 450.0
    # a single-run reference taken on the slow repetition would move the cliff estimate
    single = cs.CapPoint(None, [ref.tput[0]], ref.p99_ms, ref.j_per_token, ref.power_w)
    assert cs.calibrate(single, pts, 0.02, 1.0, FP).modes["EFF"] == 400.0


def test_no_admissible_setting():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv, p99_ok_ms=2.0), 3)
    art = cs.calibrate(ref, pts, 0.02, 1.0, FP)
    assert art.modes == {"PERF": None, "BAL": None, "EFF": None}
    assert "SLO not met" in art.note
    nv2 = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv2, allow_set=True) as g:
        ref, pts = cs.sweep(g, [1000, 300], curve(nv2), 3)
    art = cs.calibrate(ref, pts, 0.02, 1.0, FP)
    assert art.modes == {"PERF": 900.0, "BAL": 900.0, "EFF": 900.0} and art.accepted_w == []


def test_fingerprint_change_invalidates():
    nv = FakeNvml(limit_w=1400)
    with cs.CapGuard(nv, allow_set=True) as g:
        ref, pts = cs.sweep(g, CAPS, curve(nv), 2)
    art = cs.calibrate(ref, pts, 0.02, 1.0, FP)
    assert art.valid_for(dict(FP))
    assert not art.valid_for({**FP, "kernel_sources": "def"})
    assert not art.valid_for({**FP, "launch": "graph of 8 steps"})
    assert '"EFF": 450.0' in art.to_json()


def test_command_line_changes_nothing_without_the_flag(capsys):
    nv = FakeNvml(limit_w=1400)
    assert cs.main(["--caps", "800,600", "--slo-ms", "1"], nvml=nv) is None
    assert nv.sets == []
    assert "dry run" in capsys.readouterr().out


class FakeClocks(FakeNvml):
    def __init__(self, max_mhz=2070, **kw):
        super().__init__(**kw)
        self.max_mhz = max_mhz
        self.locked = None
        self.lock_calls = []

    def max_sm_clock_mhz(self):
        return self.max_mhz

    def set_locked_clocks(self, lo, hi):
        self.lock_calls.append((lo, hi))
        self.locked = (lo, hi)

    def reset_locked_clocks(self):
        self.lock_calls.append("reset")
        self.locked = None


def lock_curve(nv, knee_mhz=1400.0, t0=270000.0, p_idle=300.0, p_max=900.0, slow_below=0.0):
    """A memory-bound step under a static lock: throughput flat above the knee and falling with
    the clock below it; draw rising with the clock squared; p99 inflated below `slow_below`."""
    def run(reps):
        f = nv.locked[0] if nv.locked else nv.max_mhz
        t = t0 * min(1.0, f / knee_mhz)
        draw = p_idle + (p_max - p_idle) * (f / nv.max_mhz) ** 2
        p99 = 0.3 * (3.0 if f < slow_below else 1.0)
        return cs.CapPoint(None, [t] * reps, p99, draw / t, draw)
    return run


def test_clock_locks_need_permission_and_are_released():
    nv = FakeClocks()
    with cs.ClockGuard(nv) as g:
        with pytest.raises(PermissionError):
            g.lock(1200)
    assert nv.lock_calls == []
    with pytest.raises(RuntimeError, match="failed"):
        with cs.ClockGuard(nv, allow_set=True) as g:
            g.lock(1200)
            raise RuntimeError("measurement failed")
    assert nv.locked is None and nv.lock_calls == [(1200, 1200), "reset"]
    with cs.ClockGuard(nv, allow_set=True) as g:
        with pytest.raises(ValueError):
            g.lock(2100)  # above the GPU's maximum SM clock


def test_actuator_ab_arms():
    nv = FakeClocks()
    run = lock_curve(nv, slow_below=800)
    ref = run(3)
    with cs.ClockGuard(nv, allow_set=True) as g:
        locks = cs.lock_sweep(g, [2070, 1800, 1400, 1200, 1000, 800, 600], run, 3)
    assert nv.locked is None and [p.lock_mhz for p in locks] == [2070, 1800, 1400, 1200, 1000, 800, 600]
    # a cap that keeps the full throughput at 600 W (the power manager's own DVFS under it)
    cap = cs.CapPoint(600.0, [270000.0] * 3, 0.3, 600.0 / 270000.0, 600.0)
    rows = {r["arm"]: r for r in cs.actuator_ab(ref, cap, locks, 0.5)}
    assert rows["clock lock, throughput-optimal"]["setting"] == "1400 MHz lock"  # lowest flat clock
    assert rows["clock lock, aggressive"]["setting"] == "800 MHz lock"  # 600 MHz breaks the SLO
    assert rows["power cap"]["d_throughput"] == 0.0
    assert rows["power cap"]["d_power"] == pytest.approx(600.0 / 900.0 - 1.0)
    assert rows["clock lock, aggressive"]["d_throughput"] == pytest.approx(800 / 1400 - 1.0)
    # tokens/J against the default: (270000 / 600) / (270000 / 900) - 1
    assert rows["power cap"]["d_tokens_per_j"] == pytest.approx(0.5)
    assert all(r["slo"] for r in rows.values())


def test_engine_fingerprint_names_the_library_and_its_kernels():
    fp = cs.engine_fingerprint({"gpu": "GB300", "launch": "one CUDA graph per step"})
    assert int(fp["abi_version"]) >= 100
    assert len(fp["kernel_sources"]) == 64 and int(fp["kernel_sources"], 16) >= 0
    assert fp["gpu"] == "GB300" and fp == cs.engine_fingerprint(
        {"gpu": "GB300", "launch": "one CUDA graph per step"})
