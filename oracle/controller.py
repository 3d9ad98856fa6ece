"""Plain-Python oracle of the AutoLoCo interval controller (Sec. 3.1 and
App. A.1-A.3).  TEST INFRASTRUCTURE ONLY, like the rest of this package: it
shares no code with the library's C++ controller and exists to check it.

It follows the appendix's rules in the order the appendix states them, with
the same readings the library documents where the paper gives no value:
  * residual scale = 1.4826 * median absolute deviation, at least 1e-3;
  * reference diagnostics move by a log-space EMA with weight 0.1 for a new
    interval; before blending, D_ref is carried to the new interval's
    accumulated inner learning rate (sqrt(D) proportional to Lambda, the
    model behind xi), and Lambda_ref becomes the latest accepted interval's;
  * "nearest admissible horizon": ties take the smaller horizon;
  * two consecutive severe or invalid assessments fall back to H_min; only
    the first reference estimate skips non-finite intervals (App. A.1 asks
    for finite ones), elsewhere they take the severe path (App. A.2);
  * after adoption the candidate interval's own statistics initialise the
    new reference; after a return or a reduction one interval does; then
    three variability intervals and one monitoring interval follow;
  * while a rejected-horizon bound is active the candidate is the
    admissible horizon nearest sqrt(accepted * bound) (strictly between
    them), still subject to the exposure cap.

Parity status: pinned by the executed-horizon trace of App. F.2 and by
unit cases of each rule (tests/test_controller.py).
"""
from __future__ import annotations

import math
import statistics
from dataclasses import dataclass, field
from typing import List, Optional

from . import Schedule, lr_mass

SUPPORTED, CONSISTENT, MODERATE, SEVERE, INVALID = (
    "supported", "consistent", "moderate", "severe", "invalid")


@dataclass
class Settings:
    H_base: int
    H_min: int
    H_max: int
    q_H: int
    warmup_steps: int
    beta: float = 0.9
    thresholds: tuple = (1.5, 2.5, 4.0)
    exposure: float = 1.15
    divisors: tuple = (1.20, 1.50)
    retire: float = 0.90
    ema: float = 0.1
    mad_k: float = 1.4826
    floor: float = 1e-3
    eps: float = 1e-8
    mapper_intervals: int = 3
    reference_intervals: int = 2
    variability_intervals: int = 3
    history: int = 16
    fallback_after: int = 2


@dataclass
class Decision:
    H_tok: int
    H_step: int
    H_ref_step: int
    assessment: Optional[str]
    phase: str
    z: float = 0.0


class IntervalController:
    def __init__(self, cfg: Settings, schedule: Schedule):
        self.cfg = cfg
        self.schedule = schedule
        self.accepted = cfg.H_base
        self.next_h = cfg.H_base
        self.candidate = None
        self.phase = "warmup"
        self.count = 0
        self.needed = cfg.reference_intervals
        self.logs_D: List[float] = []
        self.logs_C: List[float] = []
        self.ref = None            # (log D_ref, log C_ref, Lambda_ref)
        self.res_D: List[float] = []
        self.res_C: List[float] = []
        self.moderates = 0
        self.severes = 0
        self.bound = None          # (token horizon, Lambda when set)
        self.masses: List[float] = []
        self.M_base = None
        self.n_hat = None
        self.decision = self._decide()

    # ---------------------------------------------------------- horizons
    def admissible(self):
        c = self.cfg
        return list(range(c.H_min, c.H_max + 1, c.q_H))

    def nearest(self, x, lo=None, hi=None):
        pool = [h for h in self.admissible()
                if (lo is None or h > lo) and (hi is None or h < hi)]
        if not pool:
            return None
        return min(pool, key=lambda h: (abs(h - x), h))

    def steps(self, h_tok):
        """Eq. adaptive-h-token-mapping; the identity before calibration."""
        c = self.cfg
        if self.M_base is None or not self.n_hat:
            return h_tok
        x = self.M_base * h_tok / (c.H_base * (self.n_hat + c.eps))
        below = math.floor(x / c.q_H) * c.q_H
        above = below + c.q_H
        h = below if x - below <= above - x else above
        return int(max(h, c.q_H))

    def _decide(self, assessment=None, z=0.0):
        self.decision = Decision(self.next_h, self.steps(self.next_h),
                                 self.steps(self.cfg.H_base), assessment,
                                 self.phase, z)
        return self.decision

    # --------------------------------------------------------- statistics
    def residuals(self, D, C, lam):
        """Eqs. adaptive-h-lr-mass and adaptive-h-core-residuals."""
        eps = self.cfg.eps
        log_D_ref, log_C_ref, lam_ref = self.ref
        xi = lam / (lam_ref + eps)
        r_D = math.log(math.sqrt(D) / (math.sqrt(math.exp(log_D_ref)) * xi
                                       + eps) + eps)
        r_C = -math.log(C / (math.exp(log_C_ref) + eps) + eps)
        return r_D, r_C

    def z_max(self, r_D, r_C):
        """Eq. adaptive-h-core-deviation with median / MAD over the
        residual histories."""
        def part(r, hist):
            centre = statistics.median(hist)
            mad = statistics.median([abs(h - centre) for h in hist])
            scale = max(self.cfg.mad_k * mad, self.cfg.floor)
            excess = max(r - centre, 0.0)
            return excess / scale if excess > 0 else 0.0
        if not self.res_D:
            return 0.0
        return max(part(r_D, self.res_D), part(r_C, self.res_C))

    def assess(self, z):
        """Tab. adaptive-h-assessment."""
        t_cand, t_mod, t_sev = self.cfg.thresholds
        if not math.isfinite(z):
            return INVALID
        if z < t_cand:
            return SUPPORTED
        if z < t_mod:
            return CONSISTENT
        if z < t_sev:
            return MODERATE
        return SEVERE

    def remember(self, r_D, r_C):
        self.res_D.append(r_D)
        self.res_C.append(r_C)
        self.res_D = self.res_D[-self.cfg.history:]
        self.res_C = self.res_C[-self.cfg.history:]

    def blend(self, D, C, lam):
        a, eps = self.cfg.ema, self.cfg.eps
        log_D_ref, log_C_ref, lam_ref = self.ref
        carried = log_D_ref + 2.0 * math.log((lam + eps) / (lam_ref + eps))
        self.ref = ((1 - a) * carried + a * math.log(max(D, 1e-300)),
                    (1 - a) * log_C_ref + a * math.log(max(C, 1e-300)), lam)

    # ------------------------------------------------------- transitions
    def to_reference(self, n):
        self.phase, self.count, self.needed = "reference", 0, n
        self.logs_D, self.logs_C = [], []

    def to_variability(self):
        self.phase, self.count = "variability", 0
        self.res_D, self.res_C = [], []

    def reduce(self, divisor):
        c = self.cfg
        h = self.nearest(self.accepted / divisor, hi=self.accepted)
        if h is None or self.severes >= c.fallback_after:
            h = c.H_min
        self.accepted = self.next_h = h
        self.candidate = None
        self.moderates = 0
        self.to_reference(1)

    def propose(self, position):
        c = self.cfg
        if self.bound is not None:
            h_b, lam_b = self.bound
            if lr_mass(self.schedule, position, self.steps(h_b)) <= \
                    c.retire * lam_b:
                self.bound = None
        base = lr_mass(self.schedule, position, self.steps(self.accepted))
        longer = [h for h in self.admissible() if h > self.accepted and
                  lr_mass(self.schedule, position, self.steps(h))
                  <= c.exposure * base]
        best = max(longer) if longer else None
        if best is not None and self.bound is not None:
            mid = math.sqrt(self.accepted * self.bound[0])
            h_mid = self.nearest(mid, lo=self.accepted, hi=self.bound[0])
            best = None if h_mid is None else min(best, h_mid)
        return best

    def observe(self, D, C, lam, tokens, H_step, step_end) -> Decision:
        c = self.cfg
        ran = self.next_h
        # token mapper first (App. A.3)
        if math.isfinite(tokens) and tokens >= 0:
            density = tokens / H_step
            self.n_hat = density if self.n_hat is None else \
                c.beta * self.n_hat + (1 - c.beta) * density
            if self.M_base is None and ran == c.H_base and \
                    len(self.masses) < c.mapper_intervals:
                self.masses.append(tokens)
                if len(self.masses) == c.mapper_intervals:
                    self.M_base = statistics.median(self.masses)
        finite = all(math.isfinite(x) for x in (D, C, lam)) and \
            D >= 0 and C >= 0 and lam >= 0

        if self.phase == "warmup":
            if step_end < c.warmup_steps:
                return self._decide()
            self.to_reference(c.reference_intervals)

        if self.phase == "reference":
            if not finite:
                if self.ref is not None:      # re-estimation: reduction path
                    self.severes += 1
                    self.reduce(c.divisors[1])
                return self._decide(INVALID)
            self.logs_D.append(math.log(max(D, 1e-300)))
            self.logs_C.append(math.log(max(C, 1e-300)))
            self.count += 1
            if self.count == self.needed:
                self.ref = (sum(self.logs_D) / self.needed,
                            sum(self.logs_C) / self.needed, lam)
                self.to_variability()
            return self._decide()

        if self.phase == "variability":
            if not finite:
                self.severes += 1
                self.reduce(c.divisors[1])
                return self._decide(INVALID)
            r_D, r_C = self.residuals(D, C, lam)
            self.remember(r_D, r_C)
            self.blend(D, C, lam)
            self.count += 1
            if self.count == c.variability_intervals:
                self.phase, self.count = "monitor", 0
            return self._decide()

        z = float("inf")
        if finite:
            r_D, r_C = self.residuals(D, C, lam)
            z = self.z_max(r_D, r_C)
        a = self.assess(z) if finite else INVALID
        good = a in (SUPPORTED, CONSISTENT)
        if self.phase == "monitor":
            if good:
                self.remember(r_D, r_C)
                self.blend(D, C, lam)
                self.moderates = self.severes = 0
                if a == SUPPORTED:
                    h = self.propose(step_end)
                    if h is not None and h > self.accepted:
                        self.candidate = self.next_h = h
                        self.phase = "candidate"
            elif a == MODERATE:
                self.severes = 0
                self.moderates += 1
                if self.moderates >= 2:
                    self.reduce(c.divisors[0])
            else:
                self.severes += 1
                self.reduce(c.divisors[1])
        elif self.phase in ("candidate", "confirm"):
            adopt = a == SUPPORTED or (self.phase == "confirm" and good)
            if adopt:
                self.accepted = self.next_h = self.candidate
                self.candidate = None
                if self.bound is not None and self.accepted >= self.bound[0]:
                    self.bound = None
                self.ref = (math.log(max(D, 1e-300)),
                            math.log(max(C, 1e-300)), lam)
                self.moderates = self.severes = 0
                self.to_variability()
            elif self.phase == "candidate" and a == CONSISTENT:
                self.phase = "confirm"
            else:
                self.bound = (self.candidate, lam)
                self.candidate = None
                self.next_h = self.accepted
                self.moderates = 0
                self.to_reference(1)
        return self._decide(a, z if math.isfinite(z) else 0.0)
