"""The combine step of a sharded round, on the CPU (no GPU).

A round over a vector cut into contiguous shards runs the fused pass on
each shard and returns that shard's partial sums (aloco_sync_shard); D_t and
C_t (Eq. adaptive-h-core-diagnostics) are sums over the whole vector, so the
shards' partials are exchanged and combined in a fixed shard order by
aloco_combine_partials, a host function.  Here the shard partials come from
the oracle's pass-1 sums over each shard, the library combines them, and the
result must equal the oracle's statistics over the whole vector.  A
world-size-2 gloo job exchanges the partials the way bench.py's sharded mode
does and checks that both ranks obtain the same statistics."""
import ctypes
import os
import socket
import subprocess

import numpy as np
import pytest
import torch.multiprocessing as mp

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import build as B
from paper_2609_36662_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
EPS = 1e-8


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    return A.load()


def _inputs(N, M, dtype, seed):
    w = W.small(N, M, dtype, seed=seed)
    g = W.make_global(w, "cpu")
    xs = W.fill_replicas(w, g, W.alloc_replicas(w, "cpu"), 0)
    gh = g.numpy()
    if dtype == "f32":
        xh = [x.numpy() for x in xs]
    else:
        import torch
        xh = [x.view(torch.int16).numpy().view(np.uint16) for x in xs]
    return w, gh, xh


def _corr(w):
    s = w.schedule
    sched = O.Schedule(s.kind, s.peak_lr, s.final_lr, s.warmup_steps,
                       s.total_steps)
    c = O.correction(sched, w.start_step, w.H_sel[0], w.H_base, w.outer_lr,
                     w.outer_beta)
    return A.Correction(c.lam_sel, c.lam_base, c.rho_unc, c.rho, c.mu_t,
                        c.kappa_t, c.eta_out, c.inv_norm)


def _oracle_partials(w, gh, xh, a, b, corr, dt):
    """The oracle's pass-1 sums over elements [a, b) as a shard's partials
    (the oracle sums ||Dbar||^2 itself, so its aggregate scale is 1)."""
    acc = O.Pass1Accumulator(w.M)
    if b > a:
        acc.add(gh[a:b], [x[a:b] for x in xh], dt)
    p = A.Partials()
    for m in range(w.M):
        p.drift[m] = acc.E[m]
    p.sum_sq = acc.B.value
    p.sq_scale = 1.0
    p.eps = EPS
    p.corr = corr
    p.n = b - a
    p.M = w.M
    p.pass_used = A.PASS_REGISTERS if b > a else 0
    p.kernel_ms = -1.0
    return p


def _whole(w, gh, xh, dt):
    acc = O.Pass1Accumulator(w.M)
    acc.add(gh, xh, dt)
    return acc.stats(EPS)


def _assert_close(st, ref, M, rtol=1e-12):
    for k in ("D", "C", "mean_sq_norm"):
        assert abs(st[k] - ref[k]) <= rtol * abs(ref[k]), (k, st[k], ref[k])
    for m in range(M):
        assert abs(st["drift"][m] - ref["drift"][m]) <= \
            rtol * abs(ref["drift"][m]), m


def test_partials_layout_matches_c(tmp_path):
    src = tmp_path / "probe.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "aloco.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu %zu\n", sizeof(aloco_partials_t),
         offsetof(aloco_partials_t, sum_sq), offsetof(aloco_partials_t, corr),
         offsetof(aloco_partials_t, nonfinite), offsetof(aloco_partials_t, M),
         offsetof(aloco_partials_t, kernel_ms), offsetof(aloco_opts_t, wait));
  return 0;
}
''')
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True)
    got = list(map(int, subprocess.run([str(exe)], capture_output=True,
                                       text=True, check=True).stdout.split()))
    assert got == [ctypes.sizeof(A.Partials), A.Partials.sum_sq.offset,
                   A.Partials.corr.offset, A.Partials.nonfinite.offset,
                   A.Partials.M.offset, A.Partials.kernel_ms.offset,
                   A.Opts.wait.offset]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shards", [1, 2, 3, 8])
def test_combined_shards_equal_the_whole_vector(dtype, shards):
    w, gh, xh = _inputs(300_007, 5, dtype, seed=41)
    dt = O.F32 if dtype == "f32" else O.BF16
    corr = _corr(w)
    # ragged cut points, not multiples of a vector pack
    cuts = [0] + [w.numel * k // shards + (k % 3) for k in range(1, shards)] \
        + [w.numel]
    parts = [_oracle_partials(w, gh, xh, a, b, corr, dt)
             for a, b in zip(cuts[:-1], cuts[1:])]
    st = A.combine_partials(parts)
    assert st["status"] == A.OK
    ref = _whole(w, gh, xh, dt)
    _assert_close(st, ref, w.M)
    assert st["grid"] == shards and st["M"] == w.M
    assert st["corr"] == corr.as_dict()
    # the combine is deterministic: the same partials in the same order give
    # the same bits
    st2 = A.combine_partials(parts)
    assert (st2["D"], st2["C"], st2["drift"]) == (st["D"], st["C"],
                                                  st["drift"])


def test_empty_shards_contribute_nothing():
    w, gh, xh = _inputs(50_000, 3, "f32", seed=42)
    corr = _corr(w)
    n = w.numel
    parts = [_oracle_partials(w, gh, xh, 0, 0, corr, O.F32),
             _oracle_partials(w, gh, xh, 0, n // 2, corr, O.F32),
             _oracle_partials(w, gh, xh, n // 2, n // 2, corr, O.F32),
             _oracle_partials(w, gh, xh, n // 2, n, corr, O.F32)]
    st = A.combine_partials(parts)
    _assert_close(st, _whole(w, gh, xh, O.F32), w.M)
    assert st["pass_used"] == A.PASS_REGISTERS


def test_zero_drift_and_identical_replicas_reach_the_degenerate_values():
    """App. C.1: all Delta = 0 gives D = C = 0; identical replicas give
    C = M D / (D + eps), whatever the sharding."""
    w, gh, xh = _inputs(40_000, 4, "f32", seed=43)
    corr = _corr(w)
    same = [gh.copy() for _ in range(w.M)]
    parts = [_oracle_partials(w, gh, same, a, b, corr, O.F32)
             for a, b in ((0, 10_000), (10_000, 40_000))]
    st = A.combine_partials(parts)
    assert st["D"] == 0.0 and st["C"] == 0.0 and st["mean_sq_norm"] == 0.0
    ident = [xh[0].copy() for _ in range(w.M)]
    parts = [_oracle_partials(w, gh, ident, a, b, corr, O.F32)
             for a, b in ((0, 12_345), (12_345, 40_000))]
    st = A.combine_partials(parts)
    want = w.M * st["D"] / (st["D"] + EPS)
    assert abs(st["C"] - want) <= 1e-12 * want


def test_mismatched_shards_are_rejected():
    w, gh, xh = _inputs(20_000, 3, "f32", seed=44)
    corr = _corr(w)
    a = _oracle_partials(w, gh, xh, 0, 10_000, corr, O.F32)
    b = _oracle_partials(w, gh, xh, 10_000, 20_000, corr, O.F32)
    for field, val in (("M", 4), ("eps", 1e-6), ("sq_scale", 0.5)):
        c = A.Partials.from_bytes(b.to_bytes())
        setattr(c, field, val)
        st = A.combine_partials([a, c], raise_on_error=False)
        assert st["status"] == A.ERR_ARG, field
        assert "shard 1" in A.last_error()
    c = A.Partials.from_bytes(b.to_bytes())
    c.corr.mu_t = c.corr.mu_t * (1 + 2 ** -50)
    assert A.combine_partials([a, c], raise_on_error=False)["status"] == A.ERR_ARG
    assert A.combine_partials([], raise_on_error=False)["status"] == A.ERR_ARG


def test_nonfinite_shard_is_reported():
    w, gh, xh = _inputs(20_000, 2, "f32", seed=45)
    corr = _corr(w)
    a = _oracle_partials(w, gh, xh, 0, 10_000, corr, O.F32)
    b = _oracle_partials(w, gh, xh, 10_000, 20_000, corr, O.F32)
    b.nonfinite = 3
    st = A.combine_partials([a, b], raise_on_error=False)
    assert st["status"] == A.ERR_NONFINITE and st["nonfinite"] == 3


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # every rank draws the same seeded vector and keeps its own shard
        w, gh, xh = _inputs(123_457, 6, "bf16", seed=46)
        corr = _corr(w)
        a, b = w.numel * rank // world, w.numel * (rank + 1) // world
        mine = _oracle_partials(w, gh, xh, a, b, corr, O.BF16)
        blobs = bench.gather_partials(mine.to_bytes(), world)
        st = A.combine_partials([A.Partials.from_bytes(x) for x in blobs])
        out[rank] = (st["D"], st["C"], st["mean_sq_norm"], tuple(st["drift"]),
                     [A.Partials.from_bytes(x).n for x in blobs])
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_gloo_ranks_exchange_and_combine_the_same_statistics(world):
    port = _free_port()
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
    first = out[0]
    for r in range(1, world):
        assert out[r] == first        # bit for bit on every rank
    w, gh, xh = _inputs(123_457, 6, "bf16", seed=46)
    ref = _whole(w, gh, xh, O.BF16)
    st = {"D": first[0], "C": first[1], "mean_sq_norm": first[2],
          "drift": list(first[3])}
    _assert_close(st, ref, w.M)
    assert sum(first[4]) == w.numel
