"""Parity of the CUDA round (through the C ABI) with the fp64 oracle on the
same seeded inputs, at sizes the oracle finishes in seconds: several
thousand blocks' worth of packs, ragged tails, unaligned buffers, every
worker count from 1 to 32, both replica types, all correction modes."""
import glob
import json
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

from _parity import (RTOL_STAT, assert_corr, assert_field, assert_field_after_chain,
                     assert_stats, compare_round, gpu_inputs,
                     oracle_chain_replicas,
                     run_gpu_round, run_oracle_round, schedule_pair,
                     to_numpy_bits)

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    yield
    A.shutdown()


@pytest.mark.parametrize("path", sorted(glob.glob(os.path.join(
    GOLDEN, "dyadic_round_*.json"))))
@pytest.mark.parametrize("rdt", [torch.float32, torch.bfloat16])
def test_hand_worked_rounds_bit_exact(path, rdt):
    """Dyadic inputs make every fp32 step exact: the GPU must reproduce the
    hand-worked values bit for bit."""
    fx = json.load(open(path))
    g = torch.tensor(fx["g"], dtype=torch.float32, device="cuda")
    v = torch.tensor(fx["v"], dtype=torch.float32, device="cuda")
    xs = [torch.tensor(x, dtype=torch.float32, device="cuda").to(rdt)
          for x in fx["x"]]
    mode = {"none": A.CORR_NONE, "full": A.CORR_FULL}[fx["mode"]]
    st = A.sync(g, v, xs, H_sel=fx["H_sel"], H_base=fx["H_base"], step=4000,
                schedule=A.Schedule.make(), outer_lr=fx["eta"],
                outer_beta=fx["mu"], opts=A.default_opts(mode=mode))
    ex = fx["expect"]
    assert st["status"] == A.OK
    assert g.cpu().tolist() == ex["g"]
    assert v.cpu().tolist() == ex["v"]
    for x in xs:
        assert x.float().cpu().tolist() == ex["g"]
    assert st["drift"] == ex["drift"]
    assert st["mean_sq_norm"] == ex["mean_sq_norm"]
    assert st["D"] == ex["D"]
    assert st["C"] == pytest.approx(ex["C_numerator"] / (ex["D"] + 1e-8),
                                    rel=1e-15)


SMALL = [(n, m, dt) for n in (1, 7, 4097) for m in (1, 2, 3, 5, 8, 13, 16,
                                                    17, 32)
         for dt in ("f32", "bf16")]
MEDIUM = [(1_000_003, m, dt) for m in (1, 3, 4, 8, 16, 17, 32)
          for dt in ("f32", "bf16")]


PASSES = [A.PASS_REGISTERS, A.PASS_BULK_COPY, A.PASS_TILE]
PASS_IDS = ["registers", "bulk_copy", "tile"]


@pytest.mark.parametrize("pass_", PASSES, ids=PASS_IDS)
@pytest.mark.parametrize("N,M,dt", SMALL + MEDIUM)
def test_round_matches_oracle(N, M, dt, pass_):
    """Every fused pass against the oracle.  The bulk-copy pass serves M <=
    16 with 16-byte aligned buffers and at least one whole tile, the tile
    pass M <= 16 with aligned buffers and N >= 4096; other rounds fall back
    to the register-streaming pass."""
    w = W.small(N, M, dt, seed=N % 97 + M)
    g, v, xs = gpu_inputs(w)
    gen = torch.Generator(device=v.device).manual_seed(7919 * N + 31 * M + len(dt))
    v.normal_(0, 1e-3, generator=gen)  # carried momentum
    orc = run_oracle_round(g, v, xs, w, w.start_step, w.H_sel[0])
    st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0],
                       opts=A.default_opts(pass_=pass_))
    assert st["status"] == A.OK
    runs = {A.PASS_REGISTERS: True,
            A.PASS_BULK_COPY: M <= 16 and N * (4 if dt == "f32" else 2) >= 256 * 16,
            A.PASS_TILE: M <= 16 and N >= 4096}[pass_]
    assert st["pass_used"] == (pass_ if runs else A.PASS_REGISTERS)
    compare_round(w, st, orc, g, v, xs)


def test_toy_round_matches_oracle():
    """The 2^20-parameter, 4-worker fp32 round at step 4000 (H_sel 150,
    H_base 100, cosine 4e-4 -> 4e-5 over 20000 steps)."""
    w = W.toy_round()
    g, v, xs = gpu_inputs(w)
    orc = run_oracle_round(g, v, xs, w, w.start_step, w.H_sel[0])
    st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0])
    assert st["status"] == A.OK
    compare_round(w, st, orc, g, v, xs)
    assert st["corr"]["rho"] == pytest.approx(1.4985573577339066, rel=1e-12)


@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("offset", [1, 2, 3])
def test_unaligned_buffers(dt, offset):
    """Buffers that are not 16-byte aligned take the element-wise path."""
    N, M = 100_003, 5
    w = W.small(N + 8, M, dt, seed=offset)
    g0, v0, xs0 = gpu_inputs(w)
    g, v = g0[offset:offset + N], v0[offset + 1:offset + 1 + N]
    xs = [x[offset:offset + N] for x in xs0]
    wN = W.small(N, M, dt, seed=offset)
    orc = run_oracle_round(g, v, xs, wN, wN.start_step, wN.H_sel[0])
    st = run_gpu_round(g, v, xs, wN, wN.start_step, wN.H_sel[0])
    assert st["status"] == A.OK
    compare_round(wN, st, orc, g, v, xs)


@pytest.mark.parametrize("pass_", [A.PASS_TILE, A.PASS_BULK_COPY], ids=["tile", "bulk_copy"])
def test_bulk_passes_fall_back_on_unaligned_buffers(pass_):
    """The bulk-copy passes need 16-byte aligned buffers: asked for on a
    misaligned one, the round runs the register pass and still matches the
    oracle."""
    N, M = 300_007, 4
    w = W.small(N + 8, M, "f32", seed=21)
    g0, v0, xs0 = gpu_inputs(w)
    g, v = g0[1:1 + N], v0[:N]
    xs = [x[:N] for x in xs0]
    wN = W.small(N, M, "f32", seed=21)
    orc = run_oracle_round(g, v, xs, wN, wN.start_step, wN.H_sel[0])
    st = run_gpu_round(g, v, xs, wN, wN.start_step, wN.H_sel[0],
                       opts=A.default_opts(pass_=pass_))
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_REGISTERS
    compare_round(wN, st, orc, g, v, xs)


@pytest.mark.parametrize("mode", [A.CORR_FULL, A.CORR_MOMENTUM_ONLY,
                                  A.CORR_NONE])
@pytest.mark.parametrize("normalize", [0, 1])
def test_modes_and_normalisation(mode, normalize):
    w = W.small(300_001, 6, "f32", seed=3, H_sel=400, H_base=100)
    g, v, xs = gpu_inputs(w)
    v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(3))
    orc = run_oracle_round(g, v, xs, w, 9000, 400, normalize=bool(normalize),
                           mode=mode)
    st = run_gpu_round(g, v, xs, w, 9000, 400,
                       opts=A.default_opts(mode=mode, normalize=normalize))
    compare_round(w, st, orc, g, v, xs)


def test_direct_averaging_gives_the_mean_of_endpoints():
    """No momentum, unit outer lr, no correction: theta' is the average of
    the workers' endpoints (the baselines' direct model averaging)."""
    w = W.small(65_537, 4, "f32", seed=12)
    g, v, xs = gpu_inputs(w)
    mean = torch.stack([x.double() for x in xs]).mean(0)
    sa, _ = schedule_pair(w.schedule)
    A.sync(g, v, xs, H_sel=100, H_base=100, step=0, schedule=sa, outer_lr=1.0,
           outer_beta=0.0, opts=A.default_opts(mode=A.CORR_NONE))
    assert_field(g.cpu().numpy(), mean.cpu().numpy(), "mean")


@pytest.mark.parametrize("pass_", PASSES, ids=PASS_IDS)
def test_repeated_rounds_are_bit_identical(pass_):
    w = W.small(2_000_003, 8, "bf16", seed=5)
    results = []
    for _ in range(5):
        g, v, xs = gpu_inputs(w)
        v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(1))
        st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0],
                           opts=A.default_opts(pass_=pass_))
        results.append((st["D"], st["C"], tuple(st["drift"]),
                        st["mean_sq_norm"], g.cpu().numpy().tobytes(),
                        v.cpu().numpy().tobytes(),
                        to_numpy_bits(xs[3]).tobytes()))
    assert all(r == results[0] for r in results[1:])


@pytest.mark.parametrize("pass_", PASSES, ids=PASS_IDS)
@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_guard_bands_untouched(dt, pass_):
    """Only [0, N) of each buffer is written: 64 sentinel elements on both
    sides of every buffer stay intact.  (pad is 64 elements, so for fp32 the
    buffers stay 16-byte aligned and the bulk-copy pass runs.)"""
    N, M, pad = 123_457, 3, 64
    w = W.small(N, M, dt, seed=9)
    g, v, xs = gpu_inputs(w)
    def padded(t, fill):
        big = torch.full((N + 2 * pad,), fill, dtype=t.dtype, device="cuda")
        big[pad:pad + N] = t
        return big
    gb, vb = padded(g, 7.0), padded(v, -7.0)
    xb = [padded(x, 3.0) for x in xs]
    st = run_gpu_round(gb[pad:pad + N], vb[pad:pad + N],
                       [x[pad:pad + N] for x in xb], w, w.start_step,
                       w.H_sel[0], opts=A.default_opts(pass_=pass_))
    assert st["status"] == A.OK
    for t, fill in [(gb, 7.0), (vb, -7.0)] + [(x, 3.0) for x in xb]:
        assert torch.all(t[:pad] == fill) and torch.all(t[-pad:] == fill)


def test_nonfinite_inputs_are_reported():
    """NaN/Inf in the inputs propagate through the round; the status says so
    and the count of affected elements matches the oracle's."""
    w = W.small(50_000, 4, "f32", seed=21)
    g, v, xs = gpu_inputs(w)
    xs[1][100] = float("nan")
    xs[2][100] = float("inf")
    v[4000] = float("inf")
    g[49_999] = float("nan")
    xs[0][777] = float("-inf")
    orc = run_oracle_round(g, v, xs, w, w.start_step, w.H_sel[0])
    st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0])
    assert st["status"] == A.ERR_NONFINITE
    assert st["nonfinite"] == orc["nonfinite"] == 4
    assert "non-finite" in A.last_error()
    # the remaining elements are still updated like the oracle's
    mask = np.ones(50_000, bool)
    mask[[100, 4000, 49_999, 777]] = False
    assert_field(g.cpu().numpy()[mask], orc["g"][mask], "theta'")


def test_host_memory_is_rejected():
    w = W.small(1000, 2, "f32")
    g, v, xs = gpu_inputs(w)
    host = torch.zeros(1000, dtype=torch.float32)
    sa, _ = schedule_pair(w.schedule)
    rc, _ = A.sync_ptrs(host.data_ptr(), v.data_ptr(),
                        [x.data_ptr() for x in xs], 1000, A.F32, 150, 100,
                        4000, sa, 0.7, 0.9, raise_on_error=False)
    assert rc == A.ERR_ARG and "device memory" in A.last_error()
    assert torch.all(host == 0)


def test_side_stream_and_kernel_timing():
    w = W.small(4_000_000, 4, "bf16", seed=2)
    g, v, xs = gpu_inputs(w)
    orc = run_oracle_round(g, v, xs, w, w.start_step, w.H_sel[0])
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0],
                       opts=A.default_opts(time_kernel=1), stream=s)
    assert st["kernel_ms"] > 0.0
    compare_round(w, st, orc, g, v, xs)


def _chain_workload(dt):
    base = W.llama_150m()
    return W.Workload("chain", 600_011, 8, dt, None, 0.6, 0.8, 1e-3, False,
                      base.schedule, base.start_step, base.H_base, base.H_sel,
                      7)


def test_consecutive_rounds_track_an_independent_oracle_chain():
    """Twenty fp32 rounds with momentum carried across them and horizons
    drawn by seed; each round's endpoints are drawn around the chain's own
    theta (workers restart from the synchronised model, Algorithm 1).  The
    oracle runs its own chain -- theta and v stored in fp32 between rounds,
    like the paper's FP32 master weights and outer state -- and nothing of
    the GPU chain enters it.  The final state allows for the two chains'
    independent fp32 storage of theta."""
    w = _chain_workload("f32")
    g, v, xs = gpu_inputs(w)
    g_o = g.cpu().numpy().copy()
    v_o = v.cpu().numpy().copy()
    rounds = W.steps_of_rounds(w)
    for k, (step, hsel) in enumerate(rounds):
        if k > 0:
            W.fill_replicas(w, g, xs, k)
        x_o = oracle_chain_replicas(w, g_o, k)
        orc = run_oracle_round(g_o, v_o, x_o, w, step, hsel)
        st = run_gpu_round(g, v, xs, w, step, hsel)
        assert st["status"] == A.OK
        assert_corr(st["corr"], orc["corr"])
        assert_stats(st, orc, w.M)
        g_o = orc["g"].astype(np.float32)
        v_o = orc["v"].astype(np.float32)
    R = len(rounds)
    assert_field_after_chain(g.cpu().numpy(), orc["g"], orc["g"], R,
                             "theta after 20 rounds")
    assert_field_after_chain(v.cpu().numpy(), orc["v"], orc["g"], R,
                             "v after 20 rounds")


@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_momentum_carried_across_rounds(dt):
    """Twenty rounds that carry the outer momentum while theta and the
    endpoints are drawn afresh from the seed every round, so both sides see
    bit-identical theta and endpoints and only v is each side's own state.
    The momentum recurrence contracts (mu_t < 1), so the two chains' v stay
    within the per-round tolerance; D_t and C_t are compared at 1e-6 in
    every round.  (With bf16 endpoints around a carried fp32 theta the
    pseudo-gradient would contain theta's sub-bf16 bits, and the outer step
    would amplify any rounding difference between two chains by
    |1 - eta_out (1 + mu_t)| per round.)"""
    w = _chain_workload(dt)
    v = W.make_momentum(w, "cuda")
    xs = W.alloc_replicas(w, "cuda")
    v_o = v.cpu().numpy().copy()
    for k, (step, hsel) in enumerate(W.steps_of_rounds(w)):
        g = W.make_global(w, "cuda", draw=k)
        W.fill_replicas(w, g, xs, k)
        orc = run_oracle_round(g, v_o, xs, w, step, hsel)
        st = run_gpu_round(g, v, xs, w, step, hsel)
        assert st["status"] == A.OK
        assert_corr(st["corr"], orc["corr"])
        assert_stats(st, orc, w.M)
        assert_field(g.cpu().numpy(), orc["g"], f"theta' round {k}")
        assert_field(v.cpu().numpy(), orc["v"], f"v' round {k}")
        v_o = orc["v"].astype(np.float32)


@pytest.mark.parametrize("M", [1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 12, 16])
@pytest.mark.parametrize("dt", ["f32", "bf16"])
def test_tile_pass_equals_register_pass_bit_for_bit(M, dt):
    """The tile pass runs the register pass's per-element arithmetic:
    theta', v' and every replica agree bit for bit, on whole blocks and on
    the element-wise tail; the statistics agree within their tolerance.
    Covers every shape: 1024-thread (fp32 M <= 8), 256- and 512-thread
    (bf16), and one 512-thread CTA per SM (fp32 M > 8)."""
    w = W.small(3 * 2048 * 37 + 1234, M, dt, seed=40 + M)
    out = []
    for p in (A.PASS_TILE, A.PASS_REGISTERS):
        g, v, xs = gpu_inputs(w)
        v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(2))
        st = run_gpu_round(g, v, xs, w, w.start_step, w.H_sel[0],
                           opts=A.default_opts(pass_=p))
        assert st["status"] == A.OK and st["pass_used"] == p
        out.append((st, g, v, xs))
    (s1, g1, v1, x1), (s2, g2, v2, x2) = out
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))
    for a_, b_ in zip(x1, x2):
        assert torch.equal(a_.view(torch.int16) if dt == "bf16" else a_.view(torch.int32),
                           b_.view(torch.int16) if dt == "bf16" else b_.view(torch.int32))
    assert s1["D"] == pytest.approx(s2["D"], rel=RTOL_STAT)
    assert s1["mean_sq_norm"] == pytest.approx(s2["mean_sq_norm"], rel=RTOL_STAT)
    for m in range(M):
        assert s1["drift"][m] == pytest.approx(s2["drift"][m], rel=RTOL_STAT)


def test_auto_pass_choice():
    """AUTO runs the tile pass from 2^27 parameters for fp32 with M = 1 or
    5..16 and for bf16 with M <= 12, and the register pass elsewhere (fp32
    M = 2..4, bf16 M >= 13, smaller rounds).  The buffers are zeros: only
    the choice is checked."""
    big, small = (1 << 27) + 4096, (1 << 27) - 4096
    sched = A.Schedule.make()
    cases = [(big, 8, torch.float32, A.PASS_TILE), (big, 1, torch.float32, A.PASS_TILE),
             (big, 3, torch.float32, A.PASS_REGISTERS), (big, 4, torch.bfloat16, A.PASS_TILE),
             (big, 13, torch.bfloat16, A.PASS_REGISTERS), (small, 8, torch.float32, A.PASS_REGISTERS)]
    for n, M, dt, want in cases:
        g = torch.zeros(n, device="cuda")
        v = torch.zeros(n, device="cuda")
        xs = [torch.zeros(n, dtype=dt, device="cuda") for _ in range(M)]
        st = A.sync(g, v, xs, H_sel=150, H_base=100, step=4000, schedule=sched,
                    outer_lr=0.7, outer_beta=0.9)
        assert st["status"] == A.OK and st["pass_used"] == want, (n, M, dt, st["pass_used"])
        del g, v, xs
        torch.cuda.empty_cache()
