"""The interval controller (aloco_select_interval) against the paper and
against a separate plain-Python oracle of App. A (oracle/controller.py).
Host-only: no GPU."""
import math

import numpy as np
import pytest

import oracle as O
from oracle import controller as OC
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import build as B

C4_SCHED = dict(kind=0, peak_lr=4e-4, final_lr=4e-5, warmup_steps=1000,
                total_steps=50000)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    B.build()
    A.load()


def _lib_ctrl(H_base=500, H_min=250, H_max=750, q_H=50, warmup=1000,
              sched=C4_SCHED, **kw):
    return A.Controller(H_base, H_min, H_max, q_H, warmup,
                        A.Schedule.make(**sched), **kw)


def _orc_ctrl(H_base=500, H_min=250, H_max=750, q_H=50, warmup=1000,
              sched=C4_SCHED, **kw):
    return OC.IntervalController(
        OC.Settings(H_base, H_min, H_max, q_H, warmup, **kw),
        O.Schedule(**sched))


def _decision_tuple(d):
    if isinstance(d, OC.Decision):
        names = {None: 0, OC.SUPPORTED: 1, OC.CONSISTENT: 2, OC.MODERATE: 3,
                 OC.SEVERE: 4, OC.INVALID: 5}
        phases = {"warmup": 0, "reference": 1, "variability": 2,
                  "monitor": 3, "candidate": 4, "confirm": 5}
        return (d.H_tok, d.H_step, d.H_ref_step, names[d.assessment],
                phases[d.phase])
    return (d.H_tok, d.H_step, d.H_ref_step, d.assessment, d.phase)


def _run(ctrl, budget, stats, sched=C4_SCHED, tokens_per_step=1024.0):
    """Drive a controller over a training budget; stats(k, lam, H) gives
    (D, C) of interval k.  Returns the executed step horizons and the
    decisions."""
    so = O.Schedule(**sched)
    step, k = 0, 0
    first = ctrl.decision
    h = first.H_step
    executed, decisions = [], []
    while step < budget:
        h = min(h, budget - step)
        lam = O.lr_mass(so, step, h)
        D, C = stats(k, lam, h)
        step += h
        executed.append(h)
        d = ctrl.observe(D, C, lam, tokens_per_step * h, h, step)
        decisions.append(d)
        h = d.H_step
        k += 1
    return executed, decisions


def _ideal(k, lam, h):
    """Always-supportive statistics: displacement proportional to the
    accumulated inner learning rate (sqrt(D) ~ Lambda), steady coherence."""
    return 1e3 * lam * lam, 2.0


def _runs(seq):
    out = []
    for h in seq:
        if out and out[-1][0] == h:
            out[-1][1] += 1
        else:
            out.append([h, 1])
    return [tuple(x) for x in out]


PAPER_TRACE = [(500, 7), (550, 5), (600, 5), (650, 5), (700, 5), (750, 45),
               (250, 1)]


@pytest.mark.parametrize("make", [_lib_ctrl, _orc_ctrl],
                         ids=["library", "oracle"])
def test_executed_horizons_reproduce_the_paper_trace(make):
    """App. F.2: on the C4 recipe (H_base 500, bounds [250, 750], q_H 50,
    cosine schedule, 1000-step warm-up, 50,000 steps) AutoLoCo executes
    500x7, 550x5, 600x5, 650x5, 700x5, 750x45 and a final 250-step
    remainder.  Always-supportive statistics give exactly that sequence:
    the 1.15 exposure cap allows +50 at every proposal, and five intervals
    pass at each new horizon (candidate, three variability, one
    monitoring) after seven at the start (two warm-up/bootstrap, one more
    bootstrap, three variability, one monitoring)."""
    executed, _ = _run(make(), 50000, _ideal)
    assert _runs(executed) == PAPER_TRACE
    assert sum(executed) == 50000


def test_library_matches_oracle_on_random_runs():
    """Noisy statistics with occasional spikes and a non-finite interval
    exercise every transition; the two implementations must agree on every
    decision and on z."""
    for seed in range(12):
        rng = np.random.default_rng(seed)
        spikes = {int(i): float(rng.choice([2.0, 3.2, 6.0]))
                  for i in rng.integers(8, 120, 10)}
        nan_at = int(rng.integers(20, 120))

        def stats(k, lam, h, rng=rng, spikes=spikes, nan_at=nan_at):
            D = 1e3 * lam * lam * math.exp(rng.normal(0, 0.05))
            C = 2.0 * math.exp(rng.normal(0, 0.03))
            if k in spikes:
                D *= math.exp(0.2 * spikes[k])
                C /= math.exp(0.1 * spikes[k])
            if k == nan_at:
                D = float("nan")
            return D, C

        rng_state = rng.bit_generator.state
        lib_exec, lib_dec = _run(_lib_ctrl(), 60000, stats,
                                 tokens_per_step=1000.0)
        rng.bit_generator.state = rng_state
        orc_exec, orc_dec = _run(_orc_ctrl(), 60000, stats,
                                 tokens_per_step=1000.0)
        assert lib_exec == orc_exec, seed
        for a, b in zip(lib_dec, orc_dec):
            assert _decision_tuple(a) == _decision_tuple(b), seed
            assert a.z == pytest.approx(b.z, rel=1e-9, abs=1e-12)
        kinds = {d.assessment for d in lib_dec}
        assert {A.ASSESS_SUPPORTED, A.ASSESS_INVALID} <= kinds


def _has_reference(ctrl):
    phase = _decision_tuple(ctrl.decision)[4]
    return phase >= A.PHASE_VARIABILITY


def _to_monitor(ctrl):
    """Run intervals until the controller monitors at 500.  Once a reference
    exists every interval is made exactly consistent with it (zero
    residuals), so the residual histories are constant and the robust scale
    is the floor (1e-3).  Returns the global step reached."""
    so = O.Schedule(**C4_SCHED)
    step = 0
    while True:
        h = ctrl.decision.H_step
        lam = O.lr_mass(so, step, h)
        if _has_reference(ctrl):
            D = _D_for_residual(ctrl, 0.0, lam)
            C = math.exp(_state_ref(ctrl)[1])
        else:
            D, C = _ideal(0, lam, h)
        step += h
        ctrl.observe(D, C, lam, 1024.0 * h, h, step)
        if _decision_tuple(ctrl.decision)[4] == A.PHASE_MONITOR:
            return step


def _consistent(ctrl, lam):
    """(D, C) with zero residuals against the controller's current
    reference."""
    return _D_for_residual(ctrl, 0.0, lam), math.exp(_state_ref(ctrl)[1])


def _state_ref(ctrl):
    if isinstance(ctrl, A.Controller):
        s = ctrl.state
        return s.log_D_ref, s.log_C_ref, s.lam_ref, \
            list(s.hist_D[:s.n_hist]), list(s.hist_C[:s.n_hist])
    return (*ctrl.ref, list(ctrl.res_D), list(ctrl.res_C))


def _D_for_residual(ctrl, r_D, lam):
    log_D_ref, _, lam_ref, _, _ = _state_ref(ctrl)
    eps = 1e-8
    xi = lam / (lam_ref + eps)
    root = (math.exp(r_D) - eps) * (math.sqrt(math.exp(log_D_ref)) * xi + eps)
    return root * root


@pytest.mark.parametrize("make", [_lib_ctrl, _orc_ctrl],
                         ids=["library", "oracle"])
@pytest.mark.parametrize("z,expected", [
    (1.45, A.ASSESS_SUPPORTED), (1.55, A.ASSESS_CONSISTENT),
    (2.45, A.ASSESS_CONSISTENT), (2.55, A.ASSESS_MODERATE),
    (3.95, A.ASSESS_MODERATE), (4.05, A.ASSESS_SEVERE)])
def test_assessment_thresholds(make, z, expected):
    """Tab. adaptive-h-assessment: z < 1.5 supports an increase, [1.5, 2.5)
    is reference consistent, [2.5, 4.0) a moderate deviation, >= 4.0
    severe.  The histories hold equal residuals, so the scale is the floor
    (1e-3) and a target z maps to the residual centre + z * 1e-3."""
    ctrl = make()
    step = _to_monitor(ctrl)
    _, _, _, hist_D, _ = _state_ref(ctrl)
    centre = float(np.median(hist_D))
    so = O.Schedule(**C4_SCHED)
    lam = O.lr_mass(so, step, 500)
    r_D = centre + z * 1e-3
    D = _D_for_residual(ctrl, r_D, lam)
    C = math.exp(_state_ref(ctrl)[1])
    d = ctrl.observe(D, C, lam, 1024.0 * 500, 500, step + 500)
    got = _decision_tuple(d)[3]
    assert got == expected
    assert d.z == pytest.approx(z, rel=1e-6)


@pytest.mark.parametrize("make", [_lib_ctrl, _orc_ctrl],
                         ids=["library", "oracle"])
def test_reductions(make):
    """App. A.3: a confirmed moderate deviation (two in a row) divides the
    horizon by 1.20, a severe one by 1.50, each to the nearest admissible
    multiple of q_H strictly below; a non-finite statistic takes the severe
    path, and a second severe/invalid interval in a row falls back to
    H_min."""
    so = O.Schedule(**C4_SCHED)
    # moderate twice: 500 / 1.2 = 416.7 -> 400
    ctrl = make()
    step = _to_monitor(ctrl)
    lam = O.lr_mass(so, step, 500)
    _, _, _, hist_D, _ = _state_ref(ctrl)
    D_mod = _D_for_residual(ctrl, float(np.median(hist_D)) + 3e-3, lam)
    C = math.exp(_state_ref(ctrl)[1])
    d = ctrl.observe(D_mod, C, lam, 1024.0 * 500, 500, step + 500)
    assert d.H_tok == 500
    step += 500
    lam = O.lr_mass(so, step, 500)
    D_mod = _D_for_residual(ctrl, float(np.median(hist_D)) + 3e-3, lam)
    d = ctrl.observe(D_mod, C, lam, 1024.0 * 500, 500, step + 500)
    assert _decision_tuple(d)[3] == A.ASSESS_MODERATE
    assert d.H_tok == 400
    # severe: 500 / 1.5 = 333.3 -> 350 (nearest admissible below 500)
    ctrl = make()
    step = _to_monitor(ctrl)
    d = ctrl.observe(float("nan"), 2.0, 0.1, 1024.0 * 500, 500, step + 500)
    assert d.H_tok == 350 and _decision_tuple(d)[3] == A.ASSESS_INVALID
    # a second severe/invalid interval in a row: H_min
    d = ctrl.observe(float("inf"), 2.0, 0.1, 1024.0 * 350, 350, step + 850)
    assert d.H_tok == 250


@pytest.mark.parametrize("make", [_lib_ctrl, _orc_ctrl],
                         ids=["library", "oracle"])
def test_candidate_rejection_sets_a_bound_and_the_midpoint_rule(make):
    """App. A.2: a moderate first candidate interval rejects the candidate
    and restores the accepted horizon; the rejected horizon becomes a bound,
    and the next proposal is the admissible horizon nearest the geometric
    midpoint of accepted and bound."""
    so = O.Schedule(**C4_SCHED)
    ctrl = _lib_ctrl(H_max=1000) if make is _lib_ctrl else \
        _orc_ctrl(H_max=1000)
    step = _to_monitor(ctrl)
    # supported monitoring interval -> candidate 550
    lam = O.lr_mass(so, step, 500)
    d = ctrl.observe(*_consistent(ctrl, lam), lam, 1024.0 * 500, 500,
                     step + 500)
    step += 500
    assert d.H_tok == 550 and _decision_tuple(d)[4] == A.PHASE_CANDIDATE
    # candidate interval deviates moderately -> back to 500, bound 550
    lam = O.lr_mass(so, step, 550)
    _, _, _, hist_D, _ = _state_ref(ctrl)
    D = _D_for_residual(ctrl, float(np.median(hist_D)) + 3e-3, lam)
    d = ctrl.observe(D, math.exp(_state_ref(ctrl)[1]), lam, 1024.0 * 550,
                     550, step + 550)
    step += 550
    assert d.H_tok == 500 and _decision_tuple(d)[3] == A.ASSESS_MODERATE
    # re-estimate (1) + variability (3) + monitoring (1) at 500
    for _ in range(5):
        lam = O.lr_mass(so, step, 500)
        d = ctrl.observe(*_consistent(ctrl, lam), lam, 1024.0 * 500, 500,
                         step + 500)
        step += 500
    # the midpoint of 500 and the bound 550 (524.4) has no admissible
    # horizon strictly between them (q_H 50): no candidate while the bound
    # stands, although the exposure cap alone would allow 550
    assert _decision_tuple(d)[3] == A.ASSESS_SUPPORTED
    assert d.H_tok == 500


@pytest.mark.parametrize("make", [_lib_ctrl, _orc_ctrl],
                         ids=["library", "oracle"])
def test_bound_midpoint_and_retirement(make):
    """App. A.2 with q_H 25 and an accepted 500, where the exposure cap alone
    allows 575: an active rejected bound at 560 makes the candidate the
    admissible horizon nearest sqrt(500 * 560) = 529.2, i.e. 525; the same
    bound retires when the preview at the bound has fallen to 0.90 of the
    Lambda stored with it (here 0.85), and the cap decides again (575); a
    bound at 700 (midpoint 591.6 -> 600) leaves the cap (575) in charge."""
    so = O.Schedule(**C4_SCHED)

    def candidate(bound, stored_ratio):
        ctrl = make(q_H=25, H_min=250, H_max=1000)
        step = _to_monitor(ctrl)
        preview = O.lr_mass(so, step + 500, bound)
        stored = preview / stored_ratio
        if isinstance(ctrl, A.Controller):
            ctrl.state.bound, ctrl.state.bound_lam = bound, stored
        else:
            ctrl.bound = (bound, stored)
        lam = O.lr_mass(so, step, 500)
        d = ctrl.observe(*_consistent(ctrl, lam), lam, 1024.0 * 500, 500,
                         step + 500)
        left = ctrl.state.bound if isinstance(ctrl, A.Controller) \
            else (ctrl.bound[0] if ctrl.bound else 0)
        return d.H_tok, left

    assert candidate(560, 1.00) == (525, 560)   # active: midpoint rule
    assert candidate(560, 0.85) == (575, 0)     # retired: exposure cap
    assert candidate(700, 1.00) == (575, 700)   # midpoint above the cap


def test_token_mapper():
    """Eq. adaptive-h-token-mapping: after the first three recipe-horizon
    intervals calibrate M_base, a lower token density stretches the step
    horizon (H_step ~ M_base H_tok / (H_base n_hat)); before that the
    mapping is the identity."""
    lib, orc = _lib_ctrl(), _orc_ctrl()
    so = O.Schedule(**C4_SCHED)
    for ctrl in (lib, orc):
        step = 0
        for k in range(12):
            h = ctrl.decision.H_step
            density = 1000.0 if k < 3 else 800.0
            lam = O.lr_mass(so, step, h)
            D, C = _ideal(k, lam, h)
            step += h
            d = ctrl.observe(D, C, lam, density * h, h, step)
    assert _decision_tuple(lib.decision) == _decision_tuple(orc.decision)
    # density 1000 -> 800 with beta 0.9 over 9 intervals: n_hat = 800 +
    # 200 * 0.9^9, and the recipe horizon maps to M_base/n_hat > 500
    n_hat = 800 + 200 * 0.9 ** 9
    want = 500 * 1000 / n_hat
    assert lib.decision.H_ref_step == int(round(want / 50) * 50)
    assert lib.decision.H_ref_step > 500


def test_save_and_load_resume_identically():
    so = O.Schedule(**C4_SCHED)
    a = _lib_ctrl()
    step = 0
    for k in range(15):
        h = a.decision.H_step
        lam = O.lr_mass(so, step, h)
        step += h
        a.observe(*_ideal(k, lam, h), lam, 1024.0 * h, h, step)
    blob = a.save()
    b = _lib_ctrl()
    b.load_state(blob)
    b.decision = a.decision
    s2 = step
    for k in range(15, 40):
        h = a.decision.H_step
        lam = O.lr_mass(so, step, h)
        step += h
        da = a.observe(*_ideal(k, lam, h), lam, 1024.0 * h, h, step)
        lam2 = O.lr_mass(so, s2, b.decision.H_step)
        s2 += b.decision.H_step
        db = b.observe(*_ideal(k, lam2, h), lam2, 1024.0 * h, h, s2)
        assert _decision_tuple(da) == _decision_tuple(db)
    with pytest.raises(A.AlocoError):
        b.load_state(b"\0" * len(blob))


def test_controller_argument_errors():
    with pytest.raises(A.AlocoError):
        A.Controller(500, 600, 750, 50, 1000, A.Schedule.make())  # H_min > H_base
    with pytest.raises(A.AlocoError):
        A.Controller(510, 250, 750, 50, 1000, A.Schedule.make())  # not a multiple
    ctrl = _lib_ctrl()
    with pytest.raises(A.AlocoError):
        ctrl.observe(1.0, 1.0, 0.1, 1.0, 0, 10)                  # H_step 0
