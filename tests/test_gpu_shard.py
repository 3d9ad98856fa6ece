"""Sharded rounds on one GPU (the synchronisation block of Algorithm 1 over
a parameter vector cut into contiguous shards), and the two ways a round
call can wait for its kernel.

Every element of the round depends only on its own inputs and the round's
scalars, so each shard runs the fused pass on its own elements
(aloco_sync_shard); the shards' partial sums are combined in shard order
(aloco_combine_partials).  Running the G shards of a round one after
another on one GPU must give theta', v' and the replica reset of the
unsharded round bit for bit, and D_t, C_t and the drift energies of the
oracle over the whole vector within the statistics tolerance.  The
exchange of partials between ranks is tested on CPU ranks
(test_shard_combine.py)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

from _parity import (RTOL_STAT, assert_corr, assert_rel, assert_stats,
                     gpu_inputs, oracle_corr, schedule_pair, to_numpy_bits)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _kw(w, opts=None):
    sa, _ = schedule_pair(w.schedule)
    return dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step,
                schedule=sa, outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                opts=opts)


def _inputs(w, seed):
    g, v, xs = gpu_inputs(w)
    v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(seed))
    return g, v, xs


def _oracle_stats(w, g, xs):
    acc = O.Pass1Accumulator(w.M)
    acc.add(g.cpu().numpy(), [to_numpy_bits(x) for x in xs],
            O.F32 if w.dtype == "f32" else O.BF16)
    return acc.stats(1e-8)


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


def _assert_same_outputs(a, b):
    for x, y in zip(a, b):
        assert torch.equal(_bits(x), _bits(y))


def _cuts(N, G, kind):
    if kind == "aligned":
        q = 4096
        return [0] + [(N * k // G) // q * q for k in range(1, G)] + [N]
    # ragged: not multiples of a 16-byte pack, so those shards take the
    # element path
    return [0] + [N * k // G + 2 * k + 1 for k in range(1, G)] + [N]


@pytest.mark.parametrize("cut", ["aligned", "ragged"])
@pytest.mark.parametrize("G", [2, 3, 8])
@pytest.mark.parametrize("dt,M", [("f32", 1), ("f32", 8), ("bf16", 5),
                                  ("bf16", 8), ("f32", 17)])
def test_shards_equal_the_unsharded_round(dt, M, G, cut):
    N = 3_000_017
    w = W.small(N, M, dt, seed=60 + M)
    g, v, xs = _inputs(w, M)
    orc = _oracle_stats(w, g, xs)
    g0, v0, xs0 = g.clone(), v.clone(), [x.clone() for x in xs]
    st0 = A.sync(g0, v0, xs0, **_kw(w))
    assert st0["status"] == A.OK
    cuts = _cuts(N, G, cut)
    parts = []
    for a, b in zip(cuts[:-1], cuts[1:]):
        rc, p = A.sync_shard(g[a:b], v[a:b], [x[a:b] for x in xs], **_kw(w))
        assert rc == A.OK, A.last_error()
        assert p.n == b - a and p.M == M
        parts.append(p)
    st = A.combine_partials(parts)
    assert st["status"] == A.OK
    _assert_same_outputs([g, v, *xs], [g0, v0, *xs0])
    assert_stats(st, orc, M)
    for k in ("D", "C", "mean_sq_norm"):
        assert_rel(st[k], st0[k], k, RTOL_STAT)
    assert_corr(st["corr"], oracle_corr(w, w.start_step, w.H_sel[0]))
    assert st["grid"] == G


def test_large_shards_take_the_tile_pass():
    """Two shards of 2^27 + 2^20 bf16 parameters each run the tile pass, as
    the unsharded round of that size does."""
    N = 2 * ((1 << 27) + (1 << 20))
    w = W.small(N, 8, "bf16", seed=69)
    g, v, xs = _inputs(w, 3)
    orc = _oracle_stats(w, g, xs)
    g0, v0, xs0 = g.clone(), v.clone(), [x.clone() for x in xs]
    st0 = A.sync(g0, v0, xs0, **_kw(w))
    half = N // 2
    parts = []
    for a, b in ((0, half), (half, N)):
        rc, p = A.sync_shard(g[a:b], v[a:b], [x[a:b] for x in xs], **_kw(w))
        assert rc == A.OK and p.pass_used == A.PASS_TILE
        parts.append(p)
    st = A.combine_partials(parts)
    _assert_same_outputs([g, v, *xs], [g0, v0, *xs0])
    assert_stats(st, orc, w.M)
    assert st0["pass_used"] == A.PASS_TILE


def test_empty_and_nonfinite_shards():
    N = 200_003
    w = W.small(N, 3, "f32", seed=61)
    g, v, xs = _inputs(w, 5)
    xs[2][150_000] = float("nan")
    orc_n = N
    rc0, p0 = A.sync_shard(g[:0], v[:0], [x[:0] for x in xs], **_kw(w))
    assert rc0 == A.OK and p0.n == 0 and p0.pass_used == 0
    rc1, p1 = A.sync_shard(g[:100_000], v[:100_000], [x[:100_000] for x in xs],
                           **_kw(w))
    rc2, p2 = A.sync_shard(g[100_000:], v[100_000:], [x[100_000:] for x in xs],
                           **_kw(w), raise_on_error=False)
    assert rc1 == A.OK and rc2 == A.ERR_NONFINITE and p2.nonfinite == 1
    st = A.combine_partials([p0, p1, p2], raise_on_error=False)
    assert st["status"] == A.ERR_NONFINITE and st["nonfinite"] == 1
    assert p0.n + p1.n + p2.n == orc_n


PARTS = [32000 * 64, 64, 64 * 64, 64 * 16, 64 * 16, 64 * 64, 64, 64 * 172,
         64 * 172, 172 * 64, 64, 4096 * 5 + 77]


@pytest.mark.parametrize("form", [A.PASS_INT8_FUSED, A.PASS_INT8_SPLIT],
                         ids=["fused", "split"])
@pytest.mark.parametrize("dt,M", [("f32", 4), ("bf16", 8), ("bf16", 16)])
def test_int8_shards_at_part_boundaries(dt, M, form):
    """Shards made of whole tensor parts encode the blocks of the unsharded
    INT8 round, so theta', v' and the replicas are bit-identical; D_t and
    C_t match the oracle's INT8 round over the whole vector."""
    N = sum(PARTS)
    w = W.small(N, M, dt, seed=62 + M)
    g, v, xs = _inputs(w, M)
    corr = oracle_corr(w, w.start_step, w.H_sel[0])
    orc = O.int8_round(g.cpu().numpy(), v.cpu().numpy(),
                       [to_numpy_bits(x) for x in xs],
                       O.F32 if dt == "f32" else O.BF16, PARTS, corr.mu_t,
                       corr.eta_out, corr.inv_norm)
    opts = A.default_opts(pass_=form)
    g0, v0, xs0 = g.clone(), v.clone(), [x.clone() for x in xs]
    st0 = A.sync_int8(g0, v0, xs0, parts=PARTS, **_kw(w, opts))
    assert st0["status"] == A.OK
    groups = [PARTS[:1], PARTS[1:6], PARTS[6:10], PARTS[10:]]
    off, shards = 0, []
    for grp in groups:
        n = sum(grp)
        rc, p = A.sync_shard(g[off:off + n], v[off:off + n],
                             [x[off:off + n] for x in xs], parts=grp,
                             int8=True, **_kw(w, A.default_opts(pass_=form)))
        assert rc == A.OK, A.last_error()
        assert p.pass_used == form and p.sq_scale == 1.0
        shards.append(p)
        off += n
    st = A.combine_partials(shards)
    _assert_same_outputs([g, v, *xs], [g0, v0, *xs0])
    assert_stats(st, orc, M)


@pytest.mark.parametrize("int8", [False, True], ids=["plain", "int8"])
@pytest.mark.parametrize("dt,M", [("f32", 8), ("bf16", 8)])
def test_blocking_wait_equals_spin_wait(dt, M, int8):
    """ALOCO_WAIT_BLOCK sleeps on an event instead of polling the published
    statistics: the outputs and the statistics are the same bits."""
    N = 4_000_037
    w = W.small(N, M, dt, seed=64 + M)
    out = {}
    for mode in (A.WAIT_SPIN, A.WAIT_BLOCK):
        g, v, xs = _inputs(w, 9)
        opts = A.default_opts(wait=mode, time_kernel=1)
        if int8:
            st = A.sync_int8(g, v, xs, parts=None, **_kw(w, opts))
        else:
            st = A.sync(g, v, xs, **_kw(w, opts))
        assert st["status"] == A.OK
        assert st["kernel_ms"] > 0
        out[mode] = (st, [g, v, *xs])
    (s0, t0), (s1, t1) = out[A.WAIT_SPIN], out[A.WAIT_BLOCK]
    _assert_same_outputs(t0, t1)
    for k in ("D", "C", "mean_sq_norm", "drift", "corr", "nonfinite",
              "pass_used", "grid"):
        assert s0[k] == s1[k], k


def test_blocking_wait_behind_queued_work():
    """A round queued behind other work on its stream, waited for with
    ALOCO_WAIT_BLOCK, still sees its own inputs and publishes its own
    statistics."""
    w = W.small(2_000_003, 4, "f32", seed=66)
    g, v, xs = _inputs(w, 11)
    g0, v0, xs0 = g.clone(), v.clone(), [x.clone() for x in xs]
    ref = A.sync(g0, v0, xs0, **_kw(w))
    s = torch.cuda.Stream()
    big = torch.empty(1 << 28, device="cuda")
    with torch.cuda.stream(s):
        for _ in range(8):
            big.mul_(1.0001)           # queued ahead of the round
    st = A.sync(g, v, xs, **_kw(w, A.default_opts(wait=A.WAIT_BLOCK)), stream=s)
    assert st["status"] == A.OK
    _assert_same_outputs([g, v, *xs], [g0, v0, *xs0])
    assert (st["D"], st["C"]) == (ref["D"], ref["C"])


def test_unknown_wait_mode_is_rejected():
    w = W.small(10_000, 2, "f32", seed=67)
    g, v, xs = _inputs(w, 1)
    st = A.sync(g, v, xs, **_kw(w, A.default_opts(wait=7)),
                raise_on_error=False)
    assert st["status"] == A.ERR_ARG and "wait" in A.last_error()


def test_bench_shard_mode_matches_the_unsharded_round(capsys):
    """bench.py --shards 3 on one GPU: three shards in sequence and the
    combine, one timed round; its D_t and C_t equal the unsharded round's on
    the same seeded inputs within the statistics tolerance."""
    import json
    import bench
    # four 2^24-element generator chunks: three non-empty shards
    name = "flat50343000_m4_bf16"
    assert bench.main(["--shards", "3", "--workload", name, "--steps", "1",
                       "--warmup", "0"]) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["status_ok"] and line["scaling"] == "strong"
    assert sum(line["config"]["shard_elems"]) == 50_343_000
    assert all(n > 0 for n in line["config"]["shard_elems"])
    w = bench.parse_flat(name)
    g, v, xs = gpu_inputs(w)
    step, hsel = W.steps_of_rounds(w, 1)[0]
    sa, _ = schedule_pair(w.schedule)
    st = A.sync(g, v, xs, H_sel=hsel, H_base=w.H_base, step=step, schedule=sa,
                outer_lr=w.outer_lr, outer_beta=w.outer_beta)
    assert_rel(line["D_last"], st["D"], "D", RTOL_STAT)
    assert_rel(line["C_last"], st["C"], "C", RTOL_STAT)
