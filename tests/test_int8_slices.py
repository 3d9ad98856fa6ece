"""The slicing behind the whole-vector INT8 comparisons (int8_slices): the
INT8 round's codec blocks restart at every tensor part (App. G.1), so
slices that lie inside one part and start at a multiple of 4096 from its
start hold whole blocks. Then the oracle's INT8 round run slice by slice
reproduces the round over the whole vector: theta', v' and the replicas
bit for bit, and the summed statistics to rounding."""
import numpy as np
import pytest

import oracle as O
from _parity import int8_slices

PART_SETS = {
    "one_part": [5 * 4096 + 333],
    "ragged": [4096 * 3 + 17, 100, 9000, 4096, 1, 4096 * 2 - 1],
    "small_parts": [7, 4095, 4097, 12, 8192],
}


@pytest.mark.parametrize("name", sorted(PART_SETS))
@pytest.mark.parametrize("slice_elems", [4096, 8192, 1 << 24])
def test_slices_cover_the_vector_in_whole_blocks(name, slice_elems):
    parts = PART_SETS[name]
    slices = int8_slices(parts, slice_elems)
    starts = np.cumsum([0] + parts)
    covered = np.zeros(sum(parts), np.int32)
    for s, n in slices:
        assert n > 0
        covered[s:s + n] += 1
        p = int(np.searchsorted(starts, s, side="right")) - 1
        assert s + n <= starts[p + 1], "a slice crosses a part boundary"
        assert (s - starts[p]) % 4096 == 0, "a slice starts inside a codec block"
        assert n <= max(4096, slice_elems // 4096 * 4096)
    assert (covered == 1).all()


@pytest.mark.parametrize("dt", [O.F32, O.BF16], ids=["f32", "bf16"])
@pytest.mark.parametrize("name", sorted(PART_SETS))
def test_sliced_oracle_round_equals_the_whole_round(dt, name):
    parts = PART_SETS[name]
    N, M = sum(parts), 3
    rng = np.random.default_rng(len(parts) + dt)
    g = rng.standard_normal(N).astype(np.float32)
    v = (1e-3 * rng.standard_normal(N)).astype(np.float32)
    xs = [(g + 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(M)]
    if dt == O.BF16:  # inputs only: any bf16 bit patterns (fp32 bits truncated)
        xs = [(x.view(np.uint32) >> 16).astype(np.uint16) for x in xs]
    mu, eta, inv = 0.8, 0.7, 1.0
    whole = O.int8_round(g, v, xs, dt, parts, mu, eta, inv)
    gs, vs = np.empty(N), np.empty(N)
    xo = [np.empty_like(whole["x"][m]) for m in range(M)]
    drift, sq = np.zeros(M), 0.0
    for s, n in int8_slices(parts, 4096):
        r = O.int8_round(g[s:s + n], v[s:s + n], [x[s:s + n] for x in xs], dt, [n],
                         mu, eta, inv)
        gs[s:s + n], vs[s:s + n] = r["g"], r["v"]
        for m in range(M):
            xo[m][s:s + n] = r["x"][m]
        drift += np.asarray(r["drift"])
        sq += r["mean_sq_norm"]
    assert np.array_equal(gs, whole["g"]) and np.array_equal(vs, whole["v"])
    for m in range(M):
        assert np.array_equal(xo[m], whole["x"][m])
    assert drift == pytest.approx(whole["drift"], rel=1e-12)
    assert sq == pytest.approx(whole["mean_sq_norm"], rel=1e-12)


def test_a_slice_inside_a_block_would_not_equal_the_whole_round():
    """The pin has teeth: cutting one part at an offset that is not a
    multiple of 4096 splits a codec block, and the codes change."""
    rng = np.random.default_rng(3)
    N = 8192
    g = rng.standard_normal(N).astype(np.float32)
    v = np.zeros(N, np.float32)
    xs = [(g + 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(2)]
    whole = O.int8_round(g, v, xs, O.F32, [N], 0.8, 0.7, 1.0)
    cut = 2048
    a = O.int8_round(g[:cut], v[:cut], [x[:cut] for x in xs], O.F32, [cut], 0.8, 0.7, 1.0)
    b = O.int8_round(g[cut:], v[cut:], [x[cut:] for x in xs], O.F32, [N - cut], 0.8, 0.7, 1.0)
    assert not np.array_equal(np.concatenate([a["g"], b["g"]]), whole["g"])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("plant", [None, "theta", "v", "replica"])
def test_int8_whole_vector_comparison_passes_the_oracle_and_catches_a_plant(dtype, plant):
    """compare_int8_whole_vector with the oracle's own INT8 round as the
    outputs: it passes and returns the whole round's statistics; a planted
    error in theta', v' or replica 0 fails it."""
    import torch

    from _parity import compare_int8_whole_vector
    from paper_2609_36662_gb300 import workloads as W

    parts = PART_SETS["ragged"]
    N, M = sum(parts), 3
    w = W.small(N, M, dtype, seed=5)
    rng = np.random.default_rng(6)
    g = rng.standard_normal(N).astype(np.float32)
    v = (1e-3 * rng.standard_normal(N)).astype(np.float32)
    xf = [(g + 1e-3 * rng.standard_normal(N)).astype(np.float32) for _ in range(M)]
    odt = O.F32 if dtype == "f32" else O.BF16
    xb = xf if dtype == "f32" else [(x.view(np.uint32) >> 16).astype(np.uint16) for x in xf]
    corr = O.Correction(1.0, 1.0, 1.0, 1.0, 0.8, 1.0, 0.7, 1.0)
    whole = O.int8_round(g, v, xb, odt, parts, corr.mu_t, corr.eta_out, corr.inv_norm)

    def tensor(bits):
        if dtype == "f32":
            return torch.from_numpy(np.array(bits, np.float32))
        return torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16)

    g_in, v_in = torch.from_numpy(g), torch.from_numpy(v)
    x_in = [tensor(x) for x in xb]
    go = torch.from_numpy(whole["g"].astype(np.float32))
    vo = torch.from_numpy(whole["v"].astype(np.float32))
    xo = [tensor(x) for x in whole["x"]]
    k = 13_000
    if plant == "theta":
        go[k] = go[k] * (1 + 1e-3)
    elif plant == "v":
        vo[k] = vo[k] * (1 + 1e-3) + 1e-6
    elif plant == "replica":
        xo[0][k] = (xo[0][k].float() * 1.01).to(xo[0].dtype)
    args = (w, parts, g_in, v_in, x_in, go, vo, xo, corr)
    if plant is None:
        st = compare_int8_whole_vector(*args, slice_elems=4096, threads=4)
        assert st["D"] == pytest.approx(whole["D"], rel=1e-12)
        assert st["C"] == pytest.approx(whole["C"], rel=1e-12)
        assert st["mean_sq_norm"] == pytest.approx(whole["mean_sq_norm"], rel=1e-12)
    else:
        with pytest.raises(AssertionError):
            compare_int8_whole_vector(*args, slice_elems=4096, threads=4)
