"""Pins of the oracle's inner AdamW step (Sec. 2, Eq. diloco-local-trajectory;
Tab. training settings) against a library routine and closed forms."""
import numpy as np
import pytest
import torch

import oracle as O

C4 = dict(beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1, max_norm=1.0)
SFT = dict(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, max_norm=1.0)


def _f32(rng, n, scale):
    return (rng.standard_normal(n) * scale).astype(np.float32)


def _torch_step(x, g, m1, m2, step, lr, beta1, beta2, eps, weight_decay,
                max_norm):
    """One step of torch.optim.AdamW (single-tensor path, fp64) from a given
    state, after torch.nn.utils.clip_grad_norm_."""
    p = torch.nn.Parameter(torch.from_numpy(x.astype(np.float64)))
    p.grad = torch.from_numpy(g.astype(np.float64))
    if max_norm > 0:
        torch.nn.utils.clip_grad_norm_([p], max_norm)
    opt = torch.optim.AdamW([p], lr=lr, betas=(beta1, beta2), eps=eps,
                            weight_decay=weight_decay, foreach=False)
    opt.state[p] = {"step": torch.tensor(float(step - 1), dtype=torch.float64),
                    "exp_avg": torch.from_numpy(m1.astype(np.float64)),
                    "exp_avg_sq": torch.from_numpy(m2.astype(np.float64))}
    opt.step()
    st = opt.state[p]
    return (p.detach().numpy(), st["exp_avg"].numpy(),
            st["exp_avg_sq"].numpy())


@pytest.mark.parametrize("cfg", [C4, SFT], ids=["c4", "sft"])
def test_matches_torch_adamw_over_a_chain(cfg):
    """Five steps on three replicas with different gradient scales (one far
    above the clipping threshold, one below): every step from the same
    fp32-stored state agrees with torch.optim.AdamW + clip_grad_norm_ to
    fp64 rounding."""
    rng = np.random.default_rng(5)
    n, M = 1000, 3
    xs = [_f32(rng, n, 0.02) for _ in range(M)]
    m1 = [np.zeros(n, np.float32) for _ in range(M)]
    m2 = [np.zeros(n, np.float32) for _ in range(M)]
    gscale = [1.0, 0.01, 3e-4]   # norms ~32, ~0.3, ~0.01
    for step in range(1, 6):
        lr = 4e-4 * step / 5
        gs = [_f32(rng, n, s) for s in gscale]
        orc = O.adamw_step(xs, O.F32, gs, O.F32, m1, m2, lr=lr, step=step,
                           **cfg)
        for k in range(M):
            tx, tm1, tm2 = _torch_step(xs[k], gs[k], m1[k], m2[k], step, lr,
                                       **cfg)
            # torch updates the first moment as a lerp: the two fp64
            # rounding orders differ by ~1e-16 of the field's scale
            for got, ref in ((orc["x"][k], tx), (orc["m1"][k], tm1),
                             (orc["m2"][k], tm2)):
                np.testing.assert_allclose(got, ref, rtol=1e-13,
                                           atol=1e-14 * np.abs(ref).max())
            assert orc["norms"][k] == pytest.approx(
                float(np.linalg.norm(gs[k].astype(np.float64))), rel=1e-14)
        xs = orc["x_store"]
        m1 = [a.astype(np.float32) for a in orc["m1"]]
        m2 = [a.astype(np.float32) for a in orc["m2"]]


def test_first_step_closed_form():
    """From zero moments at t = 1 the bias corrections give m^ = g and
    v^ = g^2, so (no decay, no clipping) x' = x - lr g / (|g| + eps)."""
    rng = np.random.default_rng(1)
    x = _f32(rng, 257, 0.02)
    g = _f32(rng, 257, 1e-3)
    z = np.zeros(257, np.float32)
    lr, eps = 1e-3, 1e-8
    orc = O.adamw_step([x], O.F32, [g], O.F32, [z], [z], lr, 0.9, 0.95, eps,
                       0.0, 0.0, 1)
    gd = g.astype(np.float64)
    want = x.astype(np.float64) - lr * gd / (np.abs(gd) + eps)
    np.testing.assert_allclose(orc["x"][0], want, rtol=1e-12, atol=1e-20)
    np.testing.assert_allclose(orc["m1"][0], 0.1 * gd, rtol=1e-12)
    np.testing.assert_allclose(orc["m2"][0], 0.05 * gd * gd, rtol=1e-12)


def test_zero_gradient_is_pure_decoupled_decay():
    """g = 0 and zero moments: only the decoupled weight decay acts,
    x' = x (1 - lr wd); a zero norm leaves the clipping factor at 1."""
    rng = np.random.default_rng(2)
    x = _f32(rng, 100, 1.0)
    z = np.zeros(100, np.float32)
    orc = O.adamw_step([x], O.F32, [z], O.F32, [z], [z], 1e-2, 0.9, 0.95,
                       1e-8, 0.1, 1.0, 7)
    np.testing.assert_allclose(orc["x"][0], x.astype(np.float64) * (1 - 1e-3),
                               rtol=1e-15)
    assert orc["norms"] == [0.0]


def test_clipping_scales_the_gradient_to_the_threshold():
    """A gradient of norm 10 with threshold 1 acts like g (1 / (10 + 1e-6));
    a gradient below the threshold is untouched."""
    rng = np.random.default_rng(3)
    n = 400
    g = _f32(rng, n, 1.0)
    g = (g / np.linalg.norm(g.astype(np.float64)) * 10).astype(np.float32)
    norm = float(np.linalg.norm(g.astype(np.float64)))
    x = _f32(rng, n, 0.02)
    m1 = _f32(rng, n, 1e-3)
    m2 = np.abs(_f32(rng, n, 1e-4))
    args = (0.9, 0.95, 1e-8, 0.1)
    clipped = O.adamw_step([x], O.F32, [g], O.F32, [m1], [m2], 1e-3, *args,
                           1.0, 4)
    scaled = (g.astype(np.float64) / (norm + 1e-6))
    # the same step with the pre-scaled gradient and no clipping, in fp64:
    # compare the moment updates directly
    np.testing.assert_allclose(clipped["m1"][0],
                               0.9 * m1.astype(np.float64) + 0.1 * scaled,
                               rtol=1e-12)
    np.testing.assert_allclose(clipped["m2"][0],
                               0.95 * m2.astype(np.float64) + 0.05 * scaled ** 2,
                               rtol=1e-12)
    small = (g / np.float32(100)).astype(np.float32)      # norm 0.1 < 1
    a = O.adamw_step([x], O.F32, [small], O.F32, [m1], [m2], 1e-3, *args, 1.0, 4)
    b = O.adamw_step([x], O.F32, [small], O.F32, [m1], [m2], 1e-3, *args, 0.0, 4)
    np.testing.assert_array_equal(a["x"][0], b["x"][0])


def test_update_is_invariant_to_gradient_scale():
    """Without clipping and decay, and with eps negligible, the first step's
    update does not depend on the gradient's scale."""
    rng = np.random.default_rng(4)
    x = _f32(rng, 64, 0.02)
    g = _f32(rng, 64, 1.0)
    z = np.zeros(64, np.float32)
    a = O.adamw_step([x], O.F32, [g], O.F32, [z], [z], 1e-3, 0.9, 0.95, 1e-30,
                     0.0, 0.0, 1)
    b = O.adamw_step([x], O.F32, [(g * np.float32(1024)).astype(np.float32)],
                     O.F32, [z], [z], 1e-3, 0.9, 0.95, 1e-30, 0.0, 0.0, 1)
    np.testing.assert_allclose(a["x"][0], b["x"][0], rtol=1e-15)


def test_bf16_inputs_are_widened_and_the_result_rounded_to_nearest_even():
    """bf16 replicas and gradients enter exactly; x' is stored by
    round-to-nearest-even of the fp64 result (checked against torch)."""
    rng = np.random.default_rng(6)
    n = 300
    xb = torch.from_numpy(_f32(rng, n, 0.02)).to(torch.bfloat16)
    gb = torch.from_numpy(_f32(rng, n, 1e-3)).to(torch.bfloat16)
    bits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
    z = np.zeros(n, np.float32)
    orc = O.adamw_step([bits(xb)], O.BF16, [bits(gb)], O.BF16, [z], [z],
                       4e-4, step=3, **C4)
    ref = O.adamw_step([xb.float().numpy()], O.F32, [gb.float().numpy()],
                       O.F32, [z], [z], 4e-4, step=3, **C4)
    np.testing.assert_array_equal(orc["x"][0], ref["x"][0])
    want = torch.from_numpy(ref["x"][0]).to(torch.bfloat16)
    np.testing.assert_array_equal(orc["x_store"][0], bits(want))


def test_given_norms_reproduce_the_whole_replica_step_on_a_slice():
    """A slice stepped with the whole replica's norm equals that slice of
    the whole step (the clipping factor is the only coupling)."""
    rng = np.random.default_rng(8)
    n = 5000
    x, g = _f32(rng, n, 0.02), _f32(rng, n, 0.1)
    m1, m2 = _f32(rng, n, 1e-3), np.abs(_f32(rng, n, 1e-4))
    whole = O.adamw_step([x], O.F32, [g], O.F32, [m1], [m2], 1e-3, step=6, **C4)
    sl = slice(1234, 3456)
    part = O.adamw_step([x[sl]], O.F32, [g[sl]], O.F32, [m1[sl]], [m2[sl]], 1e-3,
                        step=6, norms=whole["norms"], **C4)
    assert whole["norms"][0] > 1.0            # clipping active
    for k in ("x", "m1", "m2"):
        np.testing.assert_array_equal(part[k][0], whole[k][0][sl])
    assert part["norms"] == whole["norms"]
