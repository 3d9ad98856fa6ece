"""Pins of the oracle's INT8 pseudo-gradient communication (App. G.1)
against the paper's numbers and the codec's definition."""
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2609_36662_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_payload_per_sync_matches_the_paper():
    """Sec. 4.2 / Tab. ultrachat_int8: Llama-3.1-8B moves 16.061 GB per sync
    in BF16 and 8.038 GB in INT8 (one byte per element plus one FP32 scale
    per block of at most 4,096 elements of each tensor part)."""
    parts = [n for _, n, _ in W.LLAMA31_8B.tensors()]
    N = sum(parts)
    assert round(2 * N / 1e9, 3) == 16.061
    assert round(O.int8_payload_bytes(parts) / 1e9, 3) == 8.038


def test_hand_worked_block():
    fx = json.load(open(os.path.join(GOLDEN, "int8_codec_block.json")))
    y = np.array(fx["y"], np.float32)
    codes, scales, dec = O.int8_encode(y)
    assert codes.tolist() == fx["codes"]
    assert scales.tolist() == [fx["scale"]]
    np.testing.assert_array_equal(dec, np.array(fx["codes"], np.float32))
    c0, s0, d0 = O.int8_encode(np.zeros(100, np.float32))
    assert s0.tolist() == [fx["zero_block_scale"]] and not c0.any()


def test_blocks_restart_at_every_part():
    """Blocks of at most 4096 elements start at each tensor part."""
    assert O.int8_blocks([5000, 3000]) == 3
    assert O.int8_blocks([4096, 4096, 1]) == 3
    y = np.zeros(8000, np.float32)
    y[4095] = 2.0      # block 0 of part 0: scale 2/127
    y[4096] = 1.0      # block 1 of part 0 (904 elements): scale 1/127
    y[5000] = 4.0      # block 0 of part 1: scale 4/127
    _, scales, dec = O.int8_encode(y, [5000, 3000])
    np.testing.assert_array_equal(
        scales, np.float32([np.float32(2) / np.float32(127),
                            np.float32(1) / np.float32(127),
                            np.float32(4) / np.float32(127)]))
    assert dec[4095] == 2.0 and dec[4096] == 1.0 and dec[5000] == 4.0


def test_codec_error_bound_and_range():
    """|y - decode(encode(y))| <= scale / 2 (plus the fp32 rounding of the
    decode); codes stay in [-127, 127] and the block maximum maps to +-127."""
    rng = np.random.default_rng(0)
    for scale_mag in (1e-30, 1e-6, 1.0, 1e20):
        y = (rng.standard_normal(3 * 4096 + 17) * scale_mag).astype(np.float32)
        codes, scales, dec = O.int8_encode(y)
        assert codes.min() >= -127 and codes.max() <= 127
        s = np.repeat(scales, 4096)[:y.size].astype(np.float64)
        err = np.abs(y.astype(np.float64) - dec.astype(np.float64))
        assert np.all(err <= 0.5 * s * (1 + 1e-6) + np.abs(y) * 2 ** -23)
        for b in range(scales.size):
            blk = codes[b * 4096:(b + 1) * 4096]
            assert np.abs(blk).max() == 127


def test_grid_values_are_lossless_so_int8_round_equals_plain_round():
    """Pseudo-gradients that already lie on the INT8 grid of their block,
    identical for every worker, survive encoding exactly; the mean of equal
    decoded contributions is that value again.  Then the INT8 round equals
    the plain round (App. G.1 changes only what is communicated)."""
    rng = np.random.default_rng(1)
    N, M = 3 * 4096, 3
    g = rng.normal(0, 0.02, N).astype(np.float32)
    q = rng.integers(-127, 128, N)
    q[::4096] = 127                                   # every block hits 127
    step = np.float32(2.0 ** -14)
    g = (np.rint(g / step) * step).astype(np.float32)  # theta on the grid too
    delta = (q * step).astype(np.float32)
    x = (g - delta).astype(np.float32)
    assert np.array_equal(g - x, delta)               # exact in fp32
    xs = [x.copy() for _ in range(M)]
    v = rng.normal(0, 1e-3, N).astype(np.float32)
    plain = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 150, 100, 0.7,
                         0.9)
    c = plain["corr"]
    i8 = O.int8_round(g, v, xs, O.F32, None, c.mu_t, c.eta_out, c.inv_norm)
    assert i8["D"] == plain["D"] and i8["drift"] == plain["drift"]
    assert i8["mean_sq_norm"] == plain["mean_sq_norm"]
    np.testing.assert_array_equal(i8["g"], plain["g"])
    np.testing.assert_array_equal(i8["v"], plain["v"])


def test_quantised_aggregate_and_prequantisation_drift():
    """App. G.1: D is measured on the local pseudo-gradients before
    quantisation (identical to the plain round's D), C on the decoded
    aggregate; the aggregate is the decoded mean of the decoded worker
    contributions, encoded once."""
    rng = np.random.default_rng(2)
    N, M = 2 * 4096 + 100, 4
    g = rng.normal(0, 0.02, N).astype(np.float32)
    xs = [(g + rng.normal(0, 1e-3, N)).astype(np.float32) for _ in range(M)]
    v = np.zeros(N, np.float32)
    plain = O.sync_round(g, v, xs, O.F32, O.Schedule(), 4000, 150, 100, 0.7,
                         0.9, mode=O.MODE_NONE)
    i8 = O.int8_round(g, v, xs, O.F32, None, 0.9, 0.7, 1.0)
    assert i8["D"] == plain["D"]
    # rebuild the aggregate from the codec alone
    dec = [O.int8_encode((g - x).astype(np.float32))[2] for x in xs]
    acc = dec[0].copy()
    for d in dec[1:]:
        acc = (acc + d).astype(np.float32)
    mean = (acc / np.float32(M)).astype(np.float32)
    agg = O.int8_encode(mean)[2].astype(np.float64)
    assert i8["mean_sq_norm"] == pytest.approx(float(np.sum(agg * agg)),
                                               rel=1e-12)
    # with v = 0 and mu = 0.9: v' = agg, theta' = g - eta (agg + mu agg)
    np.testing.assert_allclose(i8["v"], agg, rtol=0, atol=0)
    # quantisation changes C only slightly on this smooth noise
    assert i8["C"] == pytest.approx(plain["C"], rel=0.05)
