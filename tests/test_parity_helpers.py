"""The helpers behind the full-size parity tests, pinned on the CPU. The GPU
tests compare whole vectors slice by slice: a streaming form of the field
tolerance, the oracle's statistics summed over slices, and the oracle's
elementwise update run on slices in threads. Here the "GPU outputs" are the
oracle's own results rounded to fp32, so every check must pass; a planted
error in theta', v' or replica 0 must fail it."""
import numpy as np
import pytest
import torch

import oracle as O
from _parity import (RTOL_FIELD, _FieldCheck, _abs_diff, compare_whole_vector,
                     field_error, oracle_stats_threaded)
from paper_2609_36662_gb300 import workloads as W


def _streamed(gpu, orc, slice_elems):
    fc = _FieldCheck("f")
    for s in range(0, len(orc), slice_elems):
        e = min(len(orc), s + slice_elems)
        fc.add(_abs_diff(gpu[s:e], orc[s:e]), orc[s:e], s)
    fc.check()


@pytest.mark.parametrize("slice_elems", [7, 1000, 1 << 20])
def test_streaming_field_check_agrees_with_the_whole_field(slice_elems):
    rng = np.random.default_rng(1)
    orc = rng.standard_normal(5000)
    orc[17] = 1e-9                       # an element far below the rms
    gpu = orc * (1 + 0.5 * RTOL_FIELD * rng.uniform(-1, 1, orc.size))
    gpu[17] = orc[17] + 0.5 * RTOL_FIELD  # within rtol of the rms, not of itself
    assert field_error(gpu, orc) <= RTOL_FIELD
    _streamed(gpu, orc, slice_elems)
    bad = gpu.copy()
    bad[4321] = orc[4321] * (1 + 3 * RTOL_FIELD) + 3 * RTOL_FIELD
    assert field_error(bad, orc) > RTOL_FIELD
    with pytest.raises(AssertionError):
        _streamed(bad, orc, slice_elems)


def _inputs(N, M, dtype, seed):
    rng = np.random.default_rng(seed)
    g = rng.standard_normal(N).astype(np.float32)
    v = (1e-3 * rng.standard_normal(N)).astype(np.float32)
    xs = [(g + 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(M)]
    if dtype == "bf16":  # inputs only: bf16 bit patterns (fp32 bits truncated)
        xt = [torch.from_numpy((x.view(np.uint32) >> 16).astype(np.uint16).view(np.int16))
              .view(torch.bfloat16) for x in xs]
    else:
        xt = [torch.from_numpy(x) for x in xs]
    return torch.from_numpy(g), torch.from_numpy(v), xt


def _bits(x):
    if x.dtype == torch.bfloat16:
        return x.view(torch.int16).numpy().view(np.uint16)
    return x.numpy()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_threaded_statistics_equal_the_whole_vector(dtype):
    g, v, xs = _inputs(10_007, 3, dtype, 2)
    odt = O.F32 if dtype == "f32" else O.BF16
    acc = O.Pass1Accumulator(3)
    acc.add(g.numpy(), [_bits(x) for x in xs], odt)
    whole = acc.stats(1e-8)
    st = oracle_stats_threaded(g, xs, 1e-8, slice_elems=1000, threads=4)
    for k in ("D", "C", "mean_sq_norm"):
        assert st[k] == pytest.approx(whole[k], rel=1e-12), k
    assert st["drift"] == pytest.approx(whole["drift"], rel=1e-12)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("plant", [None, "theta", "v", "replica"])
def test_whole_vector_comparison_passes_the_oracle_and_catches_a_plant(dtype, plant):
    N, M = 10_007, 3
    w = W.small(N, M, dtype, seed=4)
    g_in, v_in, x_in = _inputs(N, M, dtype, 3)
    odt = O.F32 if dtype == "f32" else O.BF16
    corr = O.Correction(1.0, 1.0, 1.0, 1.0, 0.8, 1.0, 0.7, 1.0)
    go, vo, xo, _ = O.pass2(g_in.numpy(), v_in.numpy(), [_bits(x) for x in x_in], odt,
                            corr.mu_t, corr.eta_out, corr.inv_norm)
    g = torch.from_numpy(go.astype(np.float32))
    v = torch.from_numpy(vo.astype(np.float32))
    if dtype == "f32":
        xs = [torch.from_numpy(x.copy()) for x in xo]
    else:
        xs = [torch.from_numpy(x.view(np.int16).copy()).view(torch.bfloat16) for x in xo]
    k = 6001
    if plant == "theta":
        g[k] = g[k] * (1 + 1e-3)
    elif plant == "v":
        v[k] = v[k] * (1 + 1e-3) + 1e-6
    elif plant == "replica":
        xs[0][k] = (xs[0][k].float() * 1.01).to(xs[0].dtype)
    args = (w, g_in, v_in, x_in, g, v, xs, corr)
    if plant is None:
        compare_whole_vector(*args, slice_elems=1000, threads=4)
    else:
        with pytest.raises(AssertionError):
            compare_whole_vector(*args, slice_elems=1000, threads=4)
