"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these tests looks at the CUDA library.  Each one checks the oracle
against something other than its own formulas: closed forms, special cases
that reduce to a textbook routine (torch's Nesterov SGD), identities derived
in the paper's appendix, brute force, and rounds worked out by hand
(tests/golden/*.json).
"""
import glob
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
EPS = 1e-8


# --------------------------------------------------------------- schedule

def _closed_form_mass(kind, peak, final, Wu, T, t0, H):
    """sum_{s=t0}^{t0+H-1} lr(s) segment by segment in closed form:
    warm-up = arithmetic series, cosine = Lagrange's identity
    sum_{k=0}^{n-1} cos(p + k d) = sin(n d / 2) / sin(d / 2) cos(p + (n-1) d / 2),
    linear = arithmetic series, tail = constant."""
    if kind == O.SCHED_CONSTANT:
        return H * peak
    a, b = t0, t0 + H - 1
    total = 0.0
    # warm-up part: s in [a, min(b, Wu-1)]
    lo, hi = a, min(b, Wu - 1)
    if lo <= hi:
        # sum of (s+1) for s in [lo, hi] = (lo+1 + hi+1)(hi-lo+1)/2
        total += peak / Wu * (lo + 1 + hi + 1) * (hi - lo + 1) / 2.0
    # decay part: s in [max(a, Wu), min(b, T-1)]
    lo, hi = max(a, Wu), min(b, T - 1)
    if lo <= hi:
        n = hi - lo + 1
        L = T - Wu
        if kind == O.SCHED_COSINE:
            d = math.pi / L
            p = math.pi * (lo - Wu) / L
            cos_sum = math.sin(n * d / 2) / math.sin(d / 2) * \
                math.cos(p + (n - 1) * d / 2)
            total += n * final + 0.5 * (peak - final) * (n + cos_sum)
        else:
            # sum of (s - Wu) over [lo, hi]
            ssum = ((lo - Wu) + (hi - Wu)) * n / 2.0
            total += n * peak + (final - peak) * ssum / L
    # tail: s >= T
    lo = max(a, T)
    if lo <= b:
        total += (b - lo + 1) * final
    return total


@pytest.mark.parametrize("kind", [O.SCHED_COSINE, O.SCHED_LINEAR,
                                  O.SCHED_CONSTANT])
def test_lr_mass_matches_closed_form(kind):
    rng = np.random.default_rng(5)
    sched = O.Schedule(kind, 4e-4, 4e-5, 1000, 20000)
    cases = [(0, 1), (0, 1000), (990, 20), (999, 2), (1000, 1), (4000, 150),
             (4000, 100), (19950, 100), (19999, 1), (20000, 50), (0, 25000)]
    cases += [(int(rng.integers(0, 22000)), int(rng.integers(1, 3000)))
              for _ in range(60)]
    for t0, H in cases:
        got = O.lr_mass(sched, t0, H)
        want = _closed_form_mass(kind, 4e-4, 4e-5, 1000, 20000, t0, H)
        assert got == pytest.approx(want, rel=1e-12, abs=1e-18), (t0, H)


def test_lr_schedule_landmarks():
    """Tab. training settings: warm-up climbs linearly to the peak, cosine
    decays from the peak to the final value, which holds afterwards."""
    s = O.Schedule(O.SCHED_COSINE, 4e-4, 4e-5, 1000, 21000)
    assert O.lr(s, 0) == pytest.approx(4e-4 / 1000, rel=1e-15)
    assert O.lr(s, 499) == pytest.approx(2e-4, rel=1e-15)
    assert O.lr(s, 999) == 4e-4
    assert O.lr(s, 1000) == 4e-4
    assert O.lr(s, 11000) == pytest.approx((4e-4 + 4e-5) / 2, rel=1e-14)
    assert O.lr(s, 21000) == 4e-5
    assert O.lr(s, 10 ** 6) == 4e-5
    lrs = [O.lr(s, k) for k in range(1000, 21000, 37)]
    assert all(a >= b for a, b in zip(lrs, lrs[1:]))


# ------------------------------------------------------ correction scalars

@pytest.mark.parametrize("mode", [O.MODE_FULL, O.MODE_MOMENTUM_ONLY,
                                  O.MODE_NONE])
def test_correction_is_identity_at_base_horizon(mode):
    """App. D.2, Eq. fixed-horizon-ratio / fixed-horizon-correction: with
    H_step = H_ref the masses are equal, rho = 1, and the correction returns
    the base settings."""
    for step in (0, 500, 1000, 4000, 15000, 30000):
        for beta in (0.45, 0.7, 0.9):
            c = O.correction(O.Schedule(), step, 100, 100, 0.7, beta,
                             mode=mode)
            assert c.lam_sel == c.lam_base
            assert c.rho == 1.0
            assert c.mu_t == beta
            assert c.kappa_t == 1.0
            assert c.eta_out == 0.7
            assert c.inv_norm == 1.0
            cn = O.correction(O.Schedule(), step, 100, 100, 0.7, beta,
                              normalize=True, mode=mode)
            assert cn.inv_norm == pytest.approx(1.0, abs=2e-8)


def test_rho_floor_for_shorter_interval():
    """Eq. app-outer-correction-ratios: an interval whose mass does not
    exceed the base comparator uses rho = 1."""
    for step in (0, 2000, 19000):
        c = O.correction(O.Schedule(), step, 50, 100, 0.7, 0.9)
        assert c.rho_unc < 1.0
        assert c.rho == 1.0 and c.mu_t == 0.9 and c.eta_out == 0.7


def test_constant_schedule_ratio_is_horizon_ratio():
    """A constant schedule makes each mass H * lr, so rho is the horizon
    ratio up to the eps in the denominator."""
    s = O.Schedule(O.SCHED_CONSTANT, 3e-4, 3e-4, 0, 1)
    for hs, hb in ((150, 100), (300, 100), (700, 500), (750, 500)):
        c = O.correction(s, 1234, hs, hb, 0.7, 0.9)
        assert c.lam_sel == pytest.approx(hs * 3e-4, rel=1e-13)
        assert c.rho_unc == pytest.approx(hs / hb, rel=1e-6)


def test_integer_rho_equals_repeated_retention():
    """App. B.4: for integer rho the retention equals rho repeated base
    retentions.  Apply the zero-input momentum recurrence v <- mu_base v
    twice and compare the retained fraction with mu_t at rho = 2."""
    s = O.Schedule(O.SCHED_CONSTANT, 1e-3, 1e-3, 0, 1)
    beta = 0.7
    c = O.correction(s, 0, 200, 100, 1.0, beta, eps=1e-300)
    assert c.rho == pytest.approx(2.0, rel=1e-14)
    v = 1.0
    for _ in range(2):
        v = beta * v + 0.0
    assert c.mu_t == pytest.approx(v, rel=1e-13)


def test_clamps_of_momentum_and_step_scale():
    """Sec. 3.2: mu_t is clipped to [mu_min, mu_max], kappa_t = min(rho,
    kappa_max)."""
    s = O.Schedule(O.SCHED_CONSTANT, 1e-3, 1e-3, 0, 1)
    c = O.correction(s, 0, 1000, 100, 0.7, 0.9)   # rho ~ 10, 0.9^10 < 0.45
    assert c.mu_t == 0.45
    assert c.kappa_t == 1.6
    assert c.eta_out == pytest.approx(0.7 * 1.6 * 0.55 / 0.1, rel=1e-13)
    c = O.correction(s, 0, 130, 100, 0.7, 0.95, mu_max=0.9)
    assert c.mu_t == 0.9          # 0.95^1.3 = 0.9355 clipped from above


def test_outer_lr_keeps_momentum_adjusted_scale():
    """Eq. oc_scale_matching: eta_out / (1 - mu_t) equals kappa_t times the
    base ratio eta_base / (1 - mu_base)."""
    rng = np.random.default_rng(1)
    for _ in range(200):
        step = int(rng.integers(0, 40000))
        hs, hb = int(rng.integers(1, 1000)), int(rng.integers(1, 1000))
        beta = float(rng.uniform(0.5, 0.95))
        eta = float(rng.uniform(0.1, 1.0))
        c = O.correction(O.Schedule(total_steps=40000), step, hs, hb, eta,
                         beta)
        lhs = c.eta_out / (1.0 - c.mu_t)
        rhs = c.kappa_t * eta / (1.0 - beta)
        assert lhs == pytest.approx(rhs, rel=1e-13)
        assert 0.45 <= c.mu_t <= 0.90
        assert 1.0 <= c.kappa_t <= 1.6


def test_ablation_modes():
    """Tab. component ablation: 'momentum' adjusts retention only and keeps
    the base outer lr; no correction keeps both base settings."""
    full = O.correction(O.Schedule(), 4000, 250, 100, 0.7, 0.9)
    mom = O.correction(O.Schedule(), 4000, 250, 100, 0.7, 0.9,
                       mode=O.MODE_MOMENTUM_ONLY)
    none = O.correction(O.Schedule(), 4000, 250, 100, 0.7, 0.9,
                        mode=O.MODE_NONE)
    assert full.rho > 1.6
    assert mom.mu_t == full.mu_t and mom.eta_out == 0.7
    assert none.mu_t == 0.9 and none.eta_out == 0.7
    assert full.eta_out != 0.7


# ------------------------------------------------------------ round pins

def _rand_round(N, M, seed, dtype=O.F32, scale=1e-3):
    rng = np.random.default_rng(seed)
    g = rng.normal(0, 0.02, N).astype(np.float32)
    v = rng.normal(0, 1e-3, N).astype(np.float32)
    xs = [(g + rng.normal(0, scale, N)).astype(np.float32) for _ in range(M)]
    if dtype == O.BF16:
        xs = [torch.from_numpy(x).to(torch.bfloat16).view(torch.int16)
              .numpy().view(np.uint16) for x in xs]
    return g, v, xs


def _widen(x, dtype):
    return x.astype(np.float64) if dtype == O.F32 else O.bf16_bits_to_float(x)


@pytest.mark.parametrize("path", sorted(glob.glob(os.path.join(GOLDEN,
                                                                 "dyadic_round_*.json"))))
def test_hand_worked_rounds(path):
    fx = json.load(open(path))
    mode = {"none": O.MODE_NONE, "full": O.MODE_FULL}[fx["mode"]]
    g = np.array(fx["g"], np.float32)
    v = np.array(fx["v"], np.float32)
    xs = [np.array(x, np.float32) for x in fx["x"]]
    r = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, fx["H_sel"],
                     fx["H_base"], fx["eta"], fx["mu"], mode=mode, eps=EPS)
    ex = fx["expect"]
    assert r["corr"].mu_t == fx["mu"] and r["corr"].eta_out == fx["eta"]
    assert r["drift"] == ex["drift"]
    assert r["mean_sq_norm"] == ex["mean_sq_norm"]
    assert r["D"] == ex["D"]
    assert r["C"] == pytest.approx(ex["C_numerator"] / (ex["D"] + EPS),
                                   rel=1e-15)
    assert r["g"].tolist() == ex["g"]
    assert r["v"].tolist() == ex["v"]
    for xo in r["x"]:
        assert xo.tolist() == ex["g"]


def test_diloco_special_case_matches_torch_nesterov_sgd():
    """App. D.2, Eq. fixed-horizon-nesterov: at H_sel = H_base the round is
    DiLoCo's Nesterov outer step, i.e. torch.optim.SGD(nesterov=True,
    dampening=0) applied to theta with gradient Dbar and the carried
    momentum buffer."""
    N, M = 3001, 5
    g, v, xs = _rand_round(N, M, 3)
    for mode in (O.MODE_FULL, O.MODE_NONE, O.MODE_MOMENTUM_ONLY):
        r = O.sync_round(g, v, xs, O.F32, O.Schedule(), 7000, 100, 100, 0.7,
                         0.9, mode=mode)
        p = torch.tensor(g, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.SGD([p], lr=0.7, momentum=0.9, nesterov=True,
                              dampening=0.0)
        opt.state[p]["momentum_buffer"] = torch.tensor(v, dtype=torch.float64)
        ends = np.stack([x.astype(np.float64) for x in xs])
        p.grad = torch.tensor(g.astype(np.float64) - ends.mean(axis=0))
        opt.step()
        np.testing.assert_allclose(r["g"], p.detach().numpy(), rtol=0,
                                   atol=1e-15)
        np.testing.assert_allclose(
            r["v"], opt.state[p]["momentum_buffer"].numpy(), rtol=0,
            atol=1e-16)


def test_direct_model_averaging():
    """App. E.2: the baselines' direct model averaging is the round with no
    momentum and unit outer lr: theta' = mean of the local endpoints."""
    N, M = 2049, 7
    g, v, xs = _rand_round(N, M, 4)
    r = O.sync_round(g, v * 0, xs, O.F32, O.Schedule(), 100, 100, 100, 1.0,
                     0.0, mode=O.MODE_NONE)
    mean = np.stack([x.astype(np.float64) for x in xs]).mean(axis=0)
    np.testing.assert_allclose(r["g"], mean, rtol=0, atol=1e-17)


@pytest.mark.parametrize("M", [1, 2, 3, 5, 8])
def test_endpoint_disagreement_identity(M):
    """App. C.1, Eq. dc_endpoint_disagreement: the mean squared distance of
    the local endpoints from their arithmetic mean equals D - C (D+eps)/M;
    Eq. dc_ranges: 0 <= C <= M D/(D+eps) < M."""
    N = 4097
    g, v, xs = _rand_round(N, M, 10 + M)
    r = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 150, 100, 0.7, 0.9)
    ends = np.stack([x.astype(np.float64) for x in xs])
    centred = ends - ends.mean(axis=0)
    disagreement = (centred ** 2).sum(axis=1).mean()
    D, C = r["D"], r["C"]
    assert disagreement == pytest.approx(D - C * (D + EPS) / M, rel=1e-9,
                                         abs=1e-20)
    assert 0.0 <= C <= M * D / (D + EPS) * (1 + 1e-12)
    assert C < M


def test_degenerate_coherence_values():
    """App. C.1: identical updates give C = M D/(D+eps) (Eq.
    dc_identical_updates); D = 0 gives C = 0; one worker gives
    C = D/(D+eps)."""
    N = 513
    g, v, xs = _rand_round(N, 1, 20)
    same = [xs[0].copy() for _ in range(6)]
    r = O.sync_round(g, v, same, O.F32, O.Schedule(), 4000, 150, 100, 0.7,
                     0.9)
    assert r["C"] == pytest.approx(6 * r["D"] / (r["D"] + EPS), rel=1e-13)
    r1 = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 150, 100, 0.7,
                      0.9)
    assert r1["C"] == pytest.approx(r1["D"] / (r1["D"] + EPS), rel=1e-13)
    r0 = O.sync_round(g, v, [g.copy(), g.copy()], O.F32, O.Schedule(), 4000,
                      150, 100, 0.7, 0.9)
    assert r0["D"] == 0.0 and r0["C"] == 0.0 and r0["mean_sq_norm"] == 0.0


def test_coherence_of_the_noise_model():
    """Statistical sanity of the diagnostics on the shared/private noise
    model: Delta_m = -sigma (a s + b e_m) gives, for large N,
    C -> (M a^2 + b^2)/(a^2 + b^2) and D -> sigma^2 N (a^2 + b^2)."""
    w = W.toy_round()
    g = W.make_global(w)
    xs = W.fill_replicas(w, g, W.alloc_replicas(w), 0)
    r = O.sync_round(g.numpy(), W.make_momentum(w).numpy(),
                     [x.numpy() for x in xs], O.F32, O.Schedule(), 4000, 150,
                     100, 0.7, 0.9)
    a, b, M = w.noise_a, w.noise_b, w.M
    assert r["C"] == pytest.approx((M * a * a + b * b) / (a * a + b * b),
                                   rel=0.01)
    assert r["D"] == pytest.approx(1e-6 * w.numel * (a * a + b * b),
                                   rel=0.01)


def test_steady_state_response_without_normalisation():
    """App. C.3, Eqs. oc_momentum_fixed_point / oc_steady_response: with mu,
    eta and Dbar held fixed, v_k = Dbar (1 - mu^k)/(1 - mu) from v_0 = 0,
    and the step theta_k - theta_{k+1} tends to eta Dbar / (1 - mu).
    Dyadic values keep every round exact in fp32."""
    g = np.array([0.5, -0.25, 1.0, 0.0], np.float32)
    deltas = [np.array([0.25, -0.5, 0.125, 0.0], np.float32),
              np.array([0.75, 0.0, -0.125, 0.0], np.float32)]
    dbar = (deltas[0].astype(np.float64) + deltas[1]) / 2
    xs = [g - d for d in deltas]
    v = np.zeros(4, np.float32)
    mu, eta = 0.5, 0.25
    for k in range(1, 21):
        r = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 100, 100, eta,
                         mu, mode=O.MODE_NONE)
        np.testing.assert_array_equal(r["v"], dbar * (1 - mu ** k) / (1 - mu))
        v = r["v"].astype(np.float32)
        assert np.array_equal(v.astype(np.float64), r["v"])
        step = g.astype(np.float64) - r["g"]
    np.testing.assert_allclose(step, eta * dbar / (1 - mu), rtol=0,
                               atol=1e-6)


def test_normalisation_response_coefficient():
    """Sec. 4.3 / App. C.3: with normalisation the steady response to the
    averaged pseudo-gradient is eta_out / ((rho+eps)(1 - mu_t)).  Start the
    momentum at the fixed point Dtil/(1-mu_t) of the normalised recurrence:
    it must stay there, and the step must equal that coefficient times
    Dbar."""
    N, M = 1000, 3
    g, _, xs = _rand_round(N, M, 30)
    sched = O.Schedule(total_steps=40000)
    c = O.correction(sched, 15000, 250, 100, 0.7, 0.9, normalize=True)
    assert c.rho > 1.5
    ends = np.stack([x.astype(np.float64) for x in xs])
    dbar = g.astype(np.float64) - ends.mean(axis=0)
    v_fix = (dbar / (c.rho + EPS) / (1 - c.mu_t)).astype(np.float32)
    r = O.sync_round(g, v_fix, xs, O.F32, sched, 15000, 250, 100, 0.7, 0.9,
                     normalize=True)
    np.testing.assert_allclose(r["v"], v_fix, rtol=1e-6, atol=1e-12)
    coeff = c.eta_out / ((c.rho + EPS) * (1 - c.mu_t))
    np.testing.assert_allclose(g.astype(np.float64) - r["g"], coeff * dbar,
                               rtol=1e-5, atol=1e-12)


def test_replica_reset_and_slicewise_sums():
    """Algorithm 1: every replica restarts from theta_{t+1}.  Processing the
    vector in slices gives bit-identical sums to one pass."""
    N, M = 10007, 4
    for dtype in (O.F32, O.BF16):
        g, v, xs = _rand_round(N, M, 40, dtype)
        r = O.sync_round(g, v, xs, dtype, O.Schedule(), 4000, 150, 100, 0.7,
                         0.9)
        for xo in r["x"]:
            if dtype == O.F32:
                np.testing.assert_array_equal(xo, r["g"].astype(np.float32))
            else:
                want = [O.double_to_bf16_bits(val) for val in r["g"][:300]]
                assert xo[:300].tolist() == want
        acc = O.Pass1Accumulator(M)
        for s in range(0, N, 997):
            acc.add(g[s:s + 997], [x[s:s + 997] for x in xs], dtype)
        st = acc.stats(EPS)
        assert st["drift"] == r["drift"]
        assert st["mean_sq_norm"] == r["mean_sq_norm"]


def test_pseudo_gradient_sign():
    """Algorithm 1: Delta = theta_t - theta_local.  Replicas that moved
    downhill by +0.5 everywhere give Dbar = -0.5 and, with no momentum and
    unit lr, theta' = theta + 0.5 (the average of the endpoints)."""
    g = np.zeros(8, np.float32)
    xs = [np.full(8, 0.5, np.float32)] * 3
    r = O.sync_round(g, g, xs, O.F32, O.Schedule(), 0, 10, 10, 1.0, 0.0,
                     mode=O.MODE_NONE)
    assert r["g"].tolist() == [0.5] * 8
    assert r["v"].tolist() == [-0.5] * 8


def test_nonfinite_elements_are_counted():
    """App. A.2 treats a non-finite statistic as a reduction signal; the
    round propagates NaN/Inf and counts the affected elements."""
    N, M = 100, 3
    g, v, xs = _rand_round(N, M, 50)
    xs[1][7] = np.nan
    xs[2][7] = np.inf
    v[20] = np.inf
    g[33] = np.nan
    r = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 150, 100, 0.7, 0.9)
    assert r["nonfinite"] == 3
    assert not math.isfinite(r["D"])


# ------------------------------------------------------------ bf16 codec

def _bf16_neighbours_bruteforce(x):
    """Nearest bf16 by enumeration of the two bf16 values that bracket x
    (ties to the even bit pattern)."""
    f32 = np.float32(x)
    bits = int(np.array([f32]).view(np.uint32)[0])
    cand = set()
    for hi in ((bits >> 16) - 1, bits >> 16, (bits >> 16) + 1):
        hi &= 0xFFFF
        cand.add(hi)
    best = None
    for c in cand:
        val = O.bf16_bits_to_float(np.array([c], np.uint16))[0]
        if not np.isfinite(val):
            continue
        err = abs(val - x)
        key = (err, c & 1)
        if best is None or key < best[0]:
            best = (key, c)
    return best[1]


def test_bf16_rounding_bruteforce():
    rng = np.random.default_rng(8)
    vals = list(rng.normal(0, 1, 3000)) + list(rng.normal(0, 1e-3, 1000))
    vals += list(rng.uniform(-1e30, 1e30, 200))
    vals += list(np.ldexp(rng.uniform(1, 2, 200), -130))      # bf16 subnormal
    # exact ties: midpoints between consecutive bf16 values
    for k in range(200):
        base = int(rng.integers(0x3800, 0x4400))
        lo = O.bf16_bits_to_float(np.array([base], np.uint16))[0]
        hi = O.bf16_bits_to_float(np.array([base + 1], np.uint16))[0]
        vals.append((lo + hi) / 2)
        vals.append(-(lo + hi) / 2)
        vals.append((lo + hi) / 2 + (hi - lo) * 1e-9)
    for x in vals:
        got = O.double_to_bf16_bits(x)
        want = _bf16_neighbours_bruteforce(float(x))
        assert got == want, (x, hex(got), hex(want))


def test_bf16_rounding_agrees_with_torch_on_fp32_values():
    rng = np.random.default_rng(9)
    x = rng.normal(0, 1, 5000).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy() \
        .view(np.uint16)
    got = np.array([O.double_to_bf16_bits(float(t)) for t in x], np.uint16)
    np.testing.assert_array_equal(got, want)


def test_bf16_special_values():
    assert O.double_to_bf16_bits(0.0) == 0x0000
    assert O.double_to_bf16_bits(-0.0) == 0x8000
    assert O.double_to_bf16_bits(float("inf")) == 0x7F80
    assert O.double_to_bf16_bits(float("-inf")) == 0xFF80
    assert O.double_to_bf16_bits(1e39) == 0x7F80           # overflow
    assert O.double_to_bf16_bits(3.3895313892515355e38) == 0x7F7F   # max
    nan = O.double_to_bf16_bits(float("nan"))
    assert (nan & 0x7F80) == 0x7F80 and (nan & 0x7F) != 0
