"""GPU parity of the inner AdamW step (Sec. 2, Eq. diloco-local-trajectory;
Tab. training settings) against the fp64 oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import (RTOL_STAT, assert_bf16_replica, assert_field,
                     assert_field_after_chain, to_numpy_bits)

pytestmark = pytest.mark.gpu

C4 = dict(beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1, max_grad_norm=1.0)
SFT = dict(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, max_grad_norm=1.0)
TDT = {O.F32: torch.float32, O.BF16: torch.bfloat16}


def _state(N, M, pdt, gdt, seed, gscales=None, offset=0):
    """Replicas, gradients and moments on the GPU (each buffer `offset`
    elements into a larger allocation when offset > 0)."""
    g = torch.Generator("cuda").manual_seed(seed)

    def mk(dt, scale, positive=False):
        base = torch.empty(N + offset, dtype=torch.float32, device="cuda")
        base.normal_(0, 1, generator=g)
        if positive:
            base.abs_()
        base.mul_(scale)
        return base.to(dt)[offset:]
    gscales = gscales or [10.0 ** (-1 - 2 * (m % 3)) for m in range(M)]
    xs = [mk(TDT[pdt], 0.02) for _ in range(M)]
    gs = [mk(TDT[gdt], s / max(N, 1) ** 0.5 * 30) for s in gscales]
    m1 = [mk(torch.float32, 1e-3) for _ in range(M)]
    m2 = [mk(torch.float32, 1e-6, positive=True) for _ in range(M)]
    return xs, gs, m1, m2


def _host(ts):
    return [to_numpy_bits(t) for t in ts]


def _oracle(xs, gs, m1, m2, pdt, gdt, cfg):
    return O.adamw_step(_host(xs), pdt, _host(gs), gdt,
                        [t.cpu().numpy() for t in m1], [t.cpu().numpy() for t in m2],
                        cfg["lr"], cfg["beta1"], cfg["beta2"], cfg["eps"],
                        cfg["weight_decay"], cfg["max_grad_norm"], cfg["step"])


def _compare(xs, m1, m2, st, orc, pdt, name=""):
    M = len(xs)
    for m in range(M):
        if pdt == O.F32:
            assert_field(xs[m].cpu().numpy(), orc["x"][m], f"{name}x'[{m}]")
        else:
            assert_bf16_replica(to_numpy_bits(xs[m]), orc["x_store"][m],
                                orc["x"][m], f"{name}x'[{m}]")
        assert_field(m1[m].cpu().numpy(), orc["m1"][m], f"{name}m'[{m}]")
        assert_field(m2[m].cpu().numpy(), orc["m2"][m], f"{name}v'[{m}]")
        if st is not None:
            assert st["grad_norm"][m] == pytest.approx(orc["norms"][m], rel=RTOL_STAT,
                                                       abs=1e-30)
            want_c = min(1.0, 1.0 / (orc["norms"][m] + 1e-6))
            assert st["clip"][m] == pytest.approx(want_c, rel=RTOL_STAT)


@pytest.mark.parametrize("pdt,gdt", [(O.F32, O.F32), (O.BF16, O.BF16),
                                     (O.F32, O.BF16), (O.BF16, O.F32)],
                         ids=["p32g32", "p16g16", "p32g16", "p16g32"])
@pytest.mark.parametrize("N", [1, 7, 4097, 1_000_003])
@pytest.mark.parametrize("M", [1, 3, 8, 32])
def test_step_matches_oracle(pdt, gdt, N, M):
    """One step from a random state; the workers' gradient norms straddle
    the clipping threshold (about 3, 0.03 and 3e-4)."""
    if N == 1_000_003 and M == 32 and pdt != gdt:
        pytest.skip("covered by the matching-dtype cases")
    xs, gs, m1, m2 = _state(N, M, pdt, gdt, seed=N + M)
    cfg = dict(C4, lr=4e-4, step=7)
    orc = _oracle(xs, gs, m1, m2, pdt, gdt, cfg)
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**cfg))
    assert st["status"] == A.OK
    _compare(xs, m1, m2, st, orc, pdt)
    assert any(c < 1.0 for c in st["clip"]) or N < 4097


@pytest.mark.parametrize("cfg", [C4, SFT], ids=["c4", "sft"])
@pytest.mark.parametrize("pdt", [O.F32, O.BF16], ids=["p32", "p16"])
def test_chain_of_steps_from_zero_state(cfg, pdt):
    """Eight steps from zero moments, the state carried on both sides (fp32
    storage between steps), under a linear warm-up of the learning rate."""
    N, M, R = 100_003, 4, 8
    xs, gs, m1, m2 = _state(N, M, pdt, pdt, seed=11)
    for t in m1 + m2:
        t.zero_()
    h = dict(x=_host(xs), m1=[t.cpu().numpy() for t in m1],
             m2=[t.cpu().numpy() for t in m2])
    gen = torch.Generator("cuda").manual_seed(3)
    for step in range(1, R + 1):
        for g in gs:
            g.copy_(torch.randn(N, generator=gen, device="cuda").mul_(
                3e-3 * step).to(g.dtype))
        c = dict(cfg, lr=4e-4 * step / R, step=step)
        orc = O.adamw_step(h["x"], pdt, _host(gs), pdt, h["m1"], h["m2"],
                           c["lr"], c["beta1"], c["beta2"], c["eps"],
                           c["weight_decay"], c["max_grad_norm"], step)
        A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**c), want_stats=False)
        h = dict(x=orc["x_store"], m1=[a.astype(np.float32) for a in orc["m1"]],
                 m2=[a.astype(np.float32) for a in orc["m2"]])
    torch.cuda.synchronize()
    for m in range(M):
        if pdt == O.F32:
            assert_field_after_chain(xs[m].cpu().numpy(), orc["x"][m], orc["x"][m],
                                     R, f"x'[{m}]")
        else:
            assert_bf16_replica(to_numpy_bits(xs[m]), orc["x_store"][m],
                                orc["x"][m], f"x'[{m}]",
                                extra_abs=R * 2.0 ** -8 * np.abs(orc["x"][m]))
        assert_field_after_chain(m1[m].cpu().numpy(), orc["m1"][m], orc["m1"][m],
                                 R, f"m'[{m}]")
        assert_field_after_chain(m2[m].cpu().numpy(), orc["m2"][m], orc["m2"][m],
                                 R, f"v'[{m}]")


def test_unaligned_buffers_and_a_shared_gradient():
    """Buffers one element off 16-byte alignment take the element loop; one
    gradient tensor may serve every replica."""
    N, M = 50_001, 3
    xs, gs, m1, m2 = _state(N, M, O.F32, O.F32, seed=5, offset=1)
    shared = [gs[0]] * M
    cfg = dict(SFT, lr=5e-6, step=2)
    orc = _oracle(xs, shared, m1, m2, O.F32, O.F32, cfg)
    st = A.adamw_step(xs, shared, m1, m2, A.adamw_cfg(**cfg))
    _compare(xs, m1, m2, st, orc, O.F32)


def test_no_clipping_and_no_decay():
    N, M = 20_000, 2
    xs, gs, m1, m2 = _state(N, M, O.F32, O.F32, seed=9, gscales=[10.0, 10.0])
    cfg = dict(C4, lr=1e-3, step=1, max_grad_norm=0.0, weight_decay=0.0)
    orc = _oracle(xs, gs, m1, m2, O.F32, O.F32, cfg)
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**cfg))
    assert st["clip"] == [1.0, 1.0] and st["grad_norm"][0] > 1.0
    for m in range(M):
        assert_field(xs[m].cpu().numpy(), orc["x"][m], "x'")


def test_repeated_steps_are_bit_identical_and_async_matches():
    """The same step twice from the same state gives identical bits, with
    and without waiting for the statistics; a side stream works."""
    N, M = 300_001, 5
    outs = []
    for want, use_stream in ((True, False), (True, False), (False, True)):
        xs, gs, m1, m2 = _state(N, M, O.BF16, O.F32, seed=21)
        s = torch.cuda.Stream() if use_stream else None
        A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(step=4), stream=s,
                     want_stats=want)
        torch.cuda.synchronize()
        outs.append([t.clone() for t in xs + m1 + m2])
    for other in outs[1:]:
        for a, b in zip(outs[0], other):
            assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16
                               else a.view(torch.int32),
                               b.view(torch.int16) if b.dtype == torch.bfloat16
                               else b.view(torch.int32))


def test_host_memory_is_rejected():
    """A gradient in host memory is refused before any kernel runs; the
    parameters are left as they were."""
    N = 1000
    xs = [torch.ones(N, device="cuda")]
    gs = [torch.zeros(N)]
    with pytest.raises(A.AlocoError) as ei:
        A.adamw_step(xs, gs, [torch.zeros(N, device="cuda")],
                     [torch.zeros(N, device="cuda")], A.adamw_cfg())
    assert ei.value.status == A.ERR_ARG and "grads[0]" in str(ei.value)
    assert torch.equal(xs[0], torch.ones(N, device="cuda"))


def test_full_size_llama150m_eight_fp32_workers():
    """The 150M set with 8 fp32 replicas in the benchmark's launch
    configuration: every element of every replica against the oracle (one
    replica at a time)."""
    w = W.llama_150m()
    N, M = w.numel, w.M
    xs, gs, m1, m2 = _state(N, M, O.F32, O.F32, seed=150)
    cfg = dict(C4, lr=3e-4, step=1200)
    host = [(to_numpy_bits(xs[m]), to_numpy_bits(gs[m]), m1[m].cpu().numpy(),
             m2[m].cpu().numpy()) for m in range(M)]
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**cfg))
    for m in range(M):
        x, g, a, b = host[m]
        orc = O.adamw_step([x], O.F32, [g], O.F32, [a], [b], cfg["lr"],
                           cfg["beta1"], cfg["beta2"], cfg["eps"],
                           cfg["weight_decay"], cfg["max_grad_norm"], cfg["step"])
        assert_field(xs[m].cpu().numpy(), orc["x"][0], f"x'[{m}]")
        assert_field(m1[m].cpu().numpy(), orc["m1"][0], f"m'[{m}]")
        assert_field(m2[m].cpu().numpy(), orc["m2"][0], f"v'[{m}]")
        assert st["grad_norm"][m] == pytest.approx(orc["norms"][0], rel=RTOL_STAT)
        del orc


@pytest.mark.parametrize("pdt,gdt", [(O.F32, O.F32), (O.BF16, O.BF16), (O.BF16, O.F32)],
                         ids=["p32g32", "p16g16", "p16g32"])
def test_normed_step_equals_the_two_pass_step(pdt, gdt):
    """Given the norms the two-pass step computed, the one-pass step forms
    the same clipping factors and writes the same bits."""
    N, M = 1_000_003, 5
    a = _state(N, M, pdt, gdt, seed=77)
    b = _state(N, M, pdt, gdt, seed=77)
    cfg = A.adamw_cfg(**dict(C4, lr=4e-4, step=9))
    st1 = A.adamw_step(*a, cfg)
    st2 = A.adamw_step(*b, cfg, grad_norms=st1["grad_norm"])
    assert st2["grad_norm"] == st1["grad_norm"]
    assert st2["clip"] == st1["clip"] and min(st1["clip"]) < 1.0
    for x, y in zip(sum(a[:1] + a[2:], []), sum(b[:1] + b[2:], [])):
        bits = torch.int16 if x.dtype == torch.bfloat16 else torch.int32
        assert torch.equal(x.view(bits), y.view(bits))


def test_normed_step_matches_the_oracle():
    """The oracle's norms in, the oracle's step out (fields within 1e-5)."""
    N, M = 300_007, 3
    xs, gs, m1, m2 = _state(N, M, O.F32, O.F32, seed=78)
    cfg = dict(C4, lr=3e-4, step=5)
    orc = _oracle(xs, gs, m1, m2, O.F32, O.F32, cfg)
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**cfg), grad_norms=orc["norms"])
    _compare(xs, m1, m2, st, orc, O.F32)
