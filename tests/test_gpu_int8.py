"""INT8 pseudo-gradient communication (App. G.1) on the GPU against the
oracle: the codec bit for bit (codes, scales and decoded values decide
integers in FP32 on both sides), and the INT8-communicated round."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

from _parity import (RTOL_STAT, assert_bf16_replica, assert_corr, assert_field,
                     assert_stats, compare_int8_whole_vector, gpu_inputs,
                     oracle_corr, schedule_pair, to_numpy_bits)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


PARTS = {
    "one_part": None,
    "ragged": [3 * 4096 + 64, 768, 5001, 12, 4096, 7],
    "llama_like": [32000 * 64, 64, 64 * 64, 64 * 16, 64 * 16, 64 * 64, 64,
                   64 * 172, 64 * 172, 172 * 64, 64],
}


def _vec(n, seed, kind="normal"):
    rng = np.random.default_rng(seed)
    y = rng.normal(0, 1e-3, n).astype(np.float32)
    if kind == "special":
        y[:4096] = 0.0                       # an all-zero block
        y[5000] = np.float32(3e38)           # near the top of fp32
        y[12288:16384] = np.float32(1e-42)   # a block of subnormals only
        y[20000] = np.nan
        y[30000] = np.inf
    return y


def _same_bits(a, b):
    """Bit-identical fp32 values, except that any NaN matches any NaN (the
    payload of a NaN produced by arithmetic differs between CPU and GPU)."""
    na, nb = np.isnan(a), np.isnan(b)
    np.testing.assert_array_equal(na, nb)
    np.testing.assert_array_equal(a[~na].view(np.uint32),
                                  b[~nb].view(np.uint32))


@pytest.mark.parametrize("parts_name", sorted(PARTS))
@pytest.mark.parametrize("kind", ["normal", "special"])
def test_codec_bit_exact(parts_name, kind):
    parts = PARTS[parts_name]
    N = sum(parts) if parts else 3 * 4096 + 1000
    if kind == "special" and N < 40000:
        N = 40000 if parts is None else N
    y = _vec(N, 3, kind if N >= 40000 else "normal")
    codes, scales, dec = A.int8_encode(torch.from_numpy(y).cuda(), parts)
    oc, osc, odec = O.int8_encode(y, parts)
    np.testing.assert_array_equal(codes.cpu().numpy(), oc)
    _same_bits(scales.cpu().numpy(), osc)
    _same_bits(dec.cpu().numpy(), odec)
    back = A.int8_decode(codes, scales, parts)
    _same_bits(back.cpu().numpy(), odec)
    assert A.int8_num_blocks(parts or [N]) == O.int8_blocks(parts or [N])


def _int8_oracle(w, g, v, xs, parts, step, hsel):
    corr = oracle_corr(w, step, hsel)
    dt = O.F32 if w.dtype == "f32" else O.BF16
    return corr, O.int8_round(g.cpu().numpy(), v.cpu().numpy(),
                              [to_numpy_bits(x) for x in xs], dt, parts,
                              corr.mu_t, corr.eta_out, corr.inv_norm)


def _compare(w, st, corr, orc, g, v, xs):
    assert st["status"] == A.OK
    assert_corr(st["corr"], corr)
    assert_stats(st, orc, w.M)
    assert_field(g.cpu().numpy(), orc["g"], "theta'")
    assert_field(v.cpu().numpy(), orc["v"], "v'")
    for m, x in enumerate(xs):
        if w.dtype == "f32":
            assert_field(x.cpu().numpy(), orc["x"][m], f"replica {m}")
        else:
            assert_bf16_replica(to_numpy_bits(x), orc["x"][m], orc["g"],
                                f"replica {m}")


def _fits_fused(dt, M):
    return M <= 16


FORMS = {"split": A.PASS_INT8_SPLIT, "fused": A.PASS_INT8_FUSED}


@pytest.mark.parametrize("form", sorted(FORMS))
@pytest.mark.parametrize("dt", ["f32", "bf16"])
@pytest.mark.parametrize("M", [1, 2, 3, 4, 5, 6, 7, 8, 9, 12, 13, 16])
@pytest.mark.parametrize("parts_name", ["one_part", "ragged", "llama_like"])
def test_int8_round_matches_oracle(dt, M, parts_name, form):
    """Every worker count whose fused shape differs: one and two CTAs per
    SM, theta and v staged or read directly, fp32 worker groups, and for
    bf16 above 8 workers the mixed-precision subtraction, the energies
    summed per block over rows padded to a power of two, and (13, 16) the
    L2 prefetch; every drift energy is checked against the oracle."""
    if form == "fused" and not _fits_fused(dt, M):
        pytest.skip("the fused form holds M <= 16")
    parts = PARTS[parts_name]
    N = sum(parts) if parts else 5 * 4096 + 333
    w = W.small(N, M, dt, seed=40 + M)
    g, v, xs = gpu_inputs(w)
    v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(M))
    corr, orc = _int8_oracle(w, g, v, xs, parts, w.start_step, w.H_sel[0])
    sa, _ = schedule_pair(w.schedule)
    st = A.sync_int8(g, v, xs, parts=parts, H_sel=w.H_sel[0], H_base=w.H_base,
                     step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                     outer_beta=w.outer_beta,
                     opts=A.default_opts(pass_=FORMS[form]))
    assert st["pass_used"] == FORMS[form]
    _compare(w, st, corr, orc, g, v, xs)


@pytest.mark.parametrize("dt,M", [("f32", 1), ("f32", 4), ("f32", 7), ("bf16", 2),
                                  ("bf16", 5), ("bf16", 8), ("bf16", 9), ("bf16", 12),
                                  ("bf16", 16), ("f32", 9), ("f32", 12), ("f32", 16)])
def test_int8_forms_agree_bit_for_bit(dt, M):
    """The forms take the same decisions in the same arithmetic: theta', v'
    and the replicas are bit-identical; the statistics agree within the
    statistics tolerance (the forms group each thread's fp32 partial
    energies differently)."""
    parts = PARTS["llama_like"]
    w = W.small(sum(parts), M, dt, seed=70 + M)
    sa, _ = schedule_pair(w.schedule)
    out = {}
    for form, p in FORMS.items():
        g, v, xs = gpu_inputs(w)
        v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(M))
        st = A.sync_int8(g, v, xs, parts=parts, H_sel=w.H_sel[0],
                         H_base=w.H_base, step=w.start_step, schedule=sa,
                         outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                         opts=A.default_opts(pass_=p))
        out[form] = (st, g, v, xs)
    (s1, g1, v1, x1), (s2, g2, v2, x2) = out["fused"], out["split"]
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))
    for a, b in zip(x1, x2):
        assert torch.equal(a, b)
    for key in ("D", "C", "mean_sq_norm"):
        assert s1[key] == pytest.approx(s2[key], rel=RTOL_STAT), key
    assert s1["nonfinite"] == s2["nonfinite"] == 0


def test_int8_auto_form():
    """AUTO takes the fused form at every worker count the INT8 round
    takes (fp32 above 8 workers stages each block's replicas in groups)."""
    for dt, M, want in (("bf16", 8, A.PASS_INT8_FUSED),
                        ("bf16", 9, A.PASS_INT8_FUSED),
                        ("bf16", 16, A.PASS_INT8_FUSED),
                        ("f32", 8, A.PASS_INT8_FUSED),
                        ("f32", 9, A.PASS_INT8_FUSED),
                        ("f32", 16, A.PASS_INT8_FUSED)):
        w = W.small(3 * 4096 + 5, M, dt, seed=3)
        g, v, xs = gpu_inputs(w)
        sa, _ = schedule_pair(w.schedule)
        st = A.sync_int8(g, v, xs, H_sel=w.H_sel[0], H_base=w.H_base,
                         step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                         outer_beta=w.outer_beta)
        assert st["pass_used"] == want, (dt, M)


def test_int8_round_with_normalisation_and_nonfinite():
    parts = PARTS["ragged"]
    N = sum(parts)
    w = W.small(N, 4, "f32", seed=50, H_sel=400)
    g, v, xs = gpu_inputs(w)
    xs[2][100] = float("nan")
    sa, _ = schedule_pair(w.schedule)
    corr = O.correction(O.Schedule(), w.start_step, 400, w.H_base, w.outer_lr,
                        w.outer_beta, normalize=True)
    orc = O.int8_round(g.cpu().numpy(), v.cpu().numpy(),
                       [x.cpu().numpy() for x in xs], O.F32, parts,
                       corr.mu_t, corr.eta_out, corr.inv_norm)
    st = A.sync_int8(g, v, xs, parts=parts, H_sel=400, H_base=w.H_base,
                     step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                     outer_beta=w.outer_beta,
                     opts=A.default_opts(normalize=1))
    assert st["status"] == A.ERR_NONFINITE
    assert st["nonfinite"] == orc["nonfinite"] > 0
    finite = np.isfinite(orc["g"])
    assert_field(g.cpu().numpy()[finite], orc["g"][finite], "theta'")


def test_int8_round_full_size_llama150m():
    """The 150M layout (111 tensor parts, 8 fp32 workers) in one INT8 round:
    every element against the oracle's INT8 round, run slice by slice (whole
    codec blocks each) on a device snapshot of the inputs, and the full
    statistics from the slices' sums."""
    w = W.llama_150m()
    parts = W.tensor_sizes(w)
    g, v, xs = gpu_inputs(w)
    g_in, v_in = g.clone(), v.clone()
    x_in = [x.clone() for x in xs]
    step, hsel = W.steps_of_rounds(w)[0]
    corr = oracle_corr(w, step, hsel)
    sa, _ = schedule_pair(w.schedule)
    st = A.sync_int8(g, v, xs, parts=parts, H_sel=hsel, H_base=w.H_base,
                     step=step, schedule=sa, outer_lr=w.outer_lr,
                     outer_beta=w.outer_beta)
    assert st["status"] == A.OK
    assert_corr(st["corr"], corr)
    gi = g.view(torch.int32)
    assert all(torch.equal(x.view(torch.int32), gi) for x in xs)
    orc = compare_int8_whole_vector(w, parts, g_in, v_in, x_in, g, v, xs, corr)
    assert_stats(st, orc, w.M)


def test_codec_decisions_at_rounding_ties():
    """The GPU divides by the block scale with a correctly rounded reciprocal
    and two exact-residual corrections; the oracle uses IEEE division.  Put
    values on, and one ulp either side of, half-integer multiples of the
    scale in 4096 blocks with scales spread over 2^-60 .. 2^60, plus random
    values: every code must agree."""
    rng = np.random.default_rng(123)
    nb = 4096
    y = np.empty(nb * 4096, np.float32)
    for b in range(nb):
        s_target = np.float32(2.0 ** rng.uniform(-60, 60))
        amax = np.float32(s_target * 127)
        blk = np.empty(4096, np.float32)
        blk[0] = amax                                   # fixes the scale
        s = np.float32(amax / np.float32(127))
        k = rng.integers(-126, 126, 4095)
        half = ((k + 0.5) * s.astype(np.float64)).astype(np.float32)
        which = rng.integers(0, 4, 4095)
        blk[1:] = np.where(which == 0, half,
                  np.where(which == 1, np.nextafter(half, np.float32(np.inf)),
                  np.where(which == 2, np.nextafter(half, np.float32(-np.inf)),
                           (rng.uniform(-127, 127, 4095) * s).astype(np.float32))))
        y[b * 4096:(b + 1) * 4096] = blk
    codes, scales, _ = A.int8_encode(torch.from_numpy(y).cuda())
    oc, osc, _ = O.int8_encode(y)
    np.testing.assert_array_equal(scales.cpu().numpy().view(np.uint32),
                                  osc.view(np.uint32))
    np.testing.assert_array_equal(codes.cpu().numpy(), oc)
