"""Whole AutoLoCo intervals on one GPU (Algorithm 1): every interval runs H
inner AdamW steps on each worker's replica (Sec. 2), then the outer round
(Sec. 3.3) and the interval controller (Sec. 3.1; App. A) picks the next
H.  The library's chain (aloco_adamw_step, aloco_sync, aloco_select_interval)
is compared with an independent oracle chain (the fp64 AdamW step and round,
and the Python oracle of the controller), both storing fp32 state between
steps.

The workers minimise seeded quadratics f_m(x) = 1/2 sum a (x - c - d_m)^2
with shared gradient noise: g_m = a (x_m - c - d_m) + s xi, xi drawn once
per step on the host and given to both chains, so only rounding separates
them."""
import numpy as np
import pytest
import torch

import oracle as O
from oracle import controller as OC
from paper_2609_36662_gb300 import aloco as A
from _parity import RTOL_FIELD, assert_field_after_chain

pytestmark = pytest.mark.gpu

SCHED = dict(kind=0, peak_lr=4e-3, final_lr=4e-4, warmup_steps=50,
             total_steps=1200)
# H_base 50 in [25, 100] on multiples of 5: a +5 step raises the interval's
# learning-rate mass by about 10 %, inside the 1.15 exposure cap (App. A)
CTRL = (50, 25, 100, 5)
ADAM = dict(beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1,
            max_grad_norm=1.0)
OUTER_LR, OUTER_BETA = 0.7, 0.9


def _objective(N, M, seed):
    r = np.random.default_rng(seed)
    a = (0.5 + r.random(N)).astype(np.float32)              # curvatures
    c = (r.standard_normal(N) * 0.05).astype(np.float32)    # shared optimum
    d = [(r.standard_normal(N) * 0.01).astype(np.float32) for _ in range(M)]
    targets = [(c + dm).astype(np.float32) for dm in d]
    return a, targets


def _grad_np(a, x, target, s, xi):
    return (a * (x - target) + s * xi).astype(np.float32)


def test_intervals_with_controller_match_the_oracle_chain():
    N, M, budget, s_noise = 32_771, 4, 1200, np.float32(0.01)
    a, targets = _objective(N, M, 1)
    theta0 = (np.random.default_rng(2).standard_normal(N) * 0.02).astype(np.float32)
    noise = np.random.default_rng(3)

    # GPU side
    dev = "cuda"
    a_d = torch.from_numpy(a).to(dev)
    t_d = [torch.from_numpy(t).to(dev) for t in targets]
    g_d = torch.from_numpy(theta0).to(dev)
    v_d = torch.zeros(N, device=dev)
    x_d = [g_d.clone() for _ in range(M)]
    grads_d = [torch.empty(N, device=dev) for _ in range(M)]
    m1_d = [torch.zeros(N, device=dev) for _ in range(M)]
    m2_d = [torch.zeros(N, device=dev) for _ in range(M)]
    sa = A.Schedule.make(**SCHED)
    ctrl = A.Controller(*CTRL, SCHED["warmup_steps"], sa)

    # oracle side
    so = O.Schedule(**SCHED)
    octrl = OC.IntervalController(OC.Settings(*CTRL, SCHED["warmup_steps"]), so)
    g_h, v_h = theta0.copy(), np.zeros(N, np.float32)
    x_h = [theta0.copy() for _ in range(M)]
    m1_h = [np.zeros(N, np.float32) for _ in range(M)]
    m2_h = [np.zeros(N, np.float32) for _ in range(M)]

    step, k, executed, assessed = 0, 0, [], 0
    h = ctrl.decision.H_step
    assert h == octrl.decision.H_step
    while step < budget:
        h = min(h, budget - step)
        for i in range(h):
            xi = [noise.standard_normal(N).astype(np.float32) for _ in range(M)]
            lr = O.lr(so, step + i)
            cfg = dict(ADAM, lr=lr, step=step + i + 1)
            for m in range(M):
                xi_d = torch.from_numpy(xi[m]).to(dev)
                torch.add(a_d * (x_d[m] - t_d[m]), s_noise * xi_d, out=grads_d[m])
            A.adamw_step(x_d, grads_d, m1_d, m2_d, A.adamw_cfg(**cfg),
                         want_stats=False)
            gs = [_grad_np(a, x_h[m], targets[m], s_noise, xi[m]) for m in range(M)]
            o = O.adamw_step(x_h, O.F32, gs, O.F32, m1_h, m2_h, lr, ADAM["beta1"],
                             ADAM["beta2"], ADAM["eps"], ADAM["weight_decay"],
                             ADAM["max_grad_norm"], step + i + 1)
            x_h = o["x_store"]
            m1_h = [z.astype(np.float32) for z in o["m1"]]
            m2_h = [z.astype(np.float32) for z in o["m2"]]
        H_base = ctrl.decision.H_ref_step
        assert H_base == octrl.decision.H_ref_step
        st = A.sync(g_d, v_d, x_d, H_sel=h, H_base=H_base, step=step,
                    schedule=sa, outer_lr=OUTER_LR, outer_beta=OUTER_BETA)
        orc = O.sync_round(g_h, v_h, x_h, O.F32, so, step, h, H_base, OUTER_LR,
                           OUTER_BETA)
        g_h, v_h = orc["g"].astype(np.float32), orc["v"].astype(np.float32)
        x_h = orc["x"]
        # the chains differ only by rounding; the statistics drive the
        # controller, whose decisions must be identical
        done = step + h
        assert st["D"] == pytest.approx(orc["D"], rel=1e-4), k
        assert st["C"] == pytest.approx(orc["C"], rel=1e-4), k
        lam = st["corr"]["lam_sel"]
        assert lam == pytest.approx(orc["corr"].lam_sel, rel=1e-12)
        d = ctrl.observe(st["D"], st["C"], lam, 1024.0 * h, h, done)
        od = octrl.observe(orc["D"], orc["C"], orc["corr"].lam_sel, 1024.0 * h,
                           h, done)
        assert (d.H_tok, d.H_step, d.H_ref_step) == \
            (od.H_tok, od.H_step, od.H_ref_step), k
        executed.append(h)
        assessed += d.assessment != A.ASSESS_NONE
        step, k, h = done, k + 1, d.H_step
    # the controller left its warm-up and assessed intervals on both sides
    assert sum(executed) == budget and assessed >= 5, (executed, assessed)
    print("executed horizons:", executed)
    # final global model after `budget` inner steps of fp32 storage
    assert_field_after_chain(g_d.cpu().numpy(), g_h.astype(np.float64),
                             g_h.astype(np.float64), budget, "theta",
                             rtol=RTOL_FIELD * 10)
