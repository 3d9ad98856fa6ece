"""The method's degenerate rounds on every kernel, against the oracle
(App. C.1: Eq. dc_identical_updates and the ranges of Eq. dc_ranges).

  * Zero drift: every replica equals theta, so every pseudo-gradient is 0.
    Then D = 0, ||Dbar||^2 = 0 and C = M * 0 / (0 + eps) = 0, and the outer
    step moves theta by the momentum alone: v' = mu_t v, theta' = theta -
    eta_out mu_t v'.  In the INT8-communicated round every codec block is
    all zero (scale 1, codes 0), so the decoded aggregate is 0 as well.
  * Identical replicas: every worker returns the same endpoint x != theta.
    Then every ||Delta_m||^2 is the same value, ||Dbar||^2 = D and
    C = M D / (D + eps), just below M, the top of the range 0 <= C < M
    (up to the fp32 rounding of the sum over workers).  In the INT8 round
    C comes from the decoded aggregate and D from the raw pseudo-gradients
    (App. G.1), so there C differs from M D / (D + eps) by the codec's
    error and only the oracle comparison and the equal energies apply.

Each case runs on the register, bulk-copy and tile passes of the plain
round and on both forms of the INT8 round, for both replica types, on a
vector that spans many tiles and ends in a ragged tail."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

from _parity import (RTOL_STAT, assert_rel, compare_round, oracle_corr,
                     run_oracle_round, schedule_pair, to_numpy_bits)

pytestmark = pytest.mark.gpu

N = 1_000_003
PLAIN = {"registers": A.PASS_REGISTERS, "bulk_copy": A.PASS_BULK_COPY,
         "tile": A.PASS_TILE}
INT8 = {"int8_split": A.PASS_INT8_SPLIT, "int8_fused": A.PASS_INT8_FUSED}
INT8_PARTS = [3 * 4096 + 64, 768, 5001, 12, 4096, N - (3 * 4096 + 64 + 768 +
                                                       5001 + 12 + 4096)]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _state(w, case):
    """theta (exactly representable in the replica type), a non-zero
    momentum and the replicas of the case."""
    gen = torch.Generator("cuda").manual_seed(7 + w.M)
    g = torch.empty(w.numel, device="cuda").normal_(0, 0.02, generator=gen)
    rdt = W.replica_dtype(w)
    g = g.to(rdt).float()
    v = torch.empty(w.numel, device="cuda").normal_(0, 1e-3, generator=gen)
    if case == "zero_drift":
        xs = [g.to(rdt).clone() for _ in range(w.M)]
    else:
        x = (g + torch.empty_like(g).normal_(0, 1e-3, generator=gen)).to(rdt)
        xs = [x.clone() for _ in range(w.M)]
    return g, v, xs


def _round(w, g, v, xs, pass_):
    sa, _ = schedule_pair(w.schedule)
    kw = dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step,
              schedule=sa, outer_lr=w.outer_lr, outer_beta=w.outer_beta,
              opts=A.default_opts(pass_=pass_))
    if pass_ in INT8.values():
        return A.sync_int8(g, v, xs, parts=INT8_PARTS, **kw)
    return A.sync(g, v, xs, **kw)


def _check_case(w, case, st, g_in, v_in, g, v, int8=False):
    M = w.M
    if case == "zero_drift":
        assert st["D"] == 0.0 and st["C"] == 0.0
        assert st["mean_sq_norm"] == 0.0
        assert st["drift"] == [0.0] * M
        # momentum alone: v' = mu_t v to one fp32 rounding
        mu = st["corr"]["mu_t"]
        want = mu * v_in.double()
        err = (v.double() - want).abs() / want.abs().clamp_min(1e-30)
        assert float(err.max()) <= 2.0 ** -23
    else:
        d = st["drift"]
        assert all(x == d[0] for x in d), "identical workers, unequal energies"
        assert d[0] > 0.0
        if not int8:
            assert_rel(st["C"], M * st["D"] / (st["D"] + 1e-8),
                       "C vs M D/(D+eps)", RTOL_STAT)
            assert st["C"] < M * (1 + RTOL_STAT)


@pytest.mark.parametrize("case", ["zero_drift", "identical"])
@pytest.mark.parametrize("pass_name", sorted(PLAIN))
@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("M", [1, 4, 8])
def test_plain_round_degenerate_cases(case, pass_name, dt, M):
    w = W.small(N, M, dt, seed=90 + M)
    g, v, xs = _state(w, case)
    g_in, v_in = g.clone(), v.clone()
    orc = run_oracle_round(g, v, xs, w, w.start_step, w.H_sel[0])
    st = _round(w, g, v, xs, PLAIN[pass_name])
    assert st["status"] == A.OK, A.last_error()
    assert st["pass_used"] == PLAIN[pass_name]
    compare_round(w, st, orc, g, v, xs)
    _check_case(w, case, st, g_in, v_in, g, v)


@pytest.mark.parametrize("case", ["zero_drift", "identical"])
@pytest.mark.parametrize("form", sorted(INT8))
@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("M", [1, 4, 8, 16])
def test_int8_round_degenerate_cases(case, form, dt, M):
    w = W.small(N, M, dt, seed=95 + M)
    g, v, xs = _state(w, case)
    g_in, v_in = g.clone(), v.clone()
    corr = oracle_corr(w, w.start_step, w.H_sel[0])
    odt = O.F32 if dt == "f32" else O.BF16
    orc = O.int8_round(g.cpu().numpy(), v.cpu().numpy(),
                       [to_numpy_bits(x) for x in xs], odt, INT8_PARTS,
                       corr.mu_t, corr.eta_out, corr.inv_norm)
    orc["corr"] = corr
    st = _round(w, g, v, xs, INT8[form])
    assert st["status"] == A.OK, A.last_error()
    assert st["pass_used"] == INT8[form]
    compare_round(w, st, orc, g, v, xs)
    _check_case(w, case, st, g_in, v_in, g, v, int8=True)
