"""Rounds from several host threads on one device, each on its own stream.

The library serialises calls per device, numbers every round it launches,
and each call returns once its own round has published its statistics (the
kernel may still be retiring on its stream).  Every thread's statistics and
outputs must then equal those of the same rounds run one after another."""
import threading

import pytest
import torch

from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import gpu_inputs, schedule_pair

pytestmark = pytest.mark.gpu

ROUNDS = 6


def _rounds(w, g, v, xs, stream, pass_):
    sa, _ = schedule_pair(w.schedule)
    out = []
    for k in range(ROUNDS):
        st = A.sync(g, v, xs, H_sel=w.H_sel[0] + 10 * k, H_base=w.H_base,
                    step=w.start_step + 100 * k, schedule=sa,
                    outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                    opts=A.default_opts(pass_=pass_), stream=stream)
        assert st["status"] == A.OK
        out.append((st["D"], st["C"], st["mean_sq_norm"], tuple(st["drift"])))
    return out


def _workloads():
    return [W.small(1_000_003 + 4096 * i, 3 + i, "f32" if i % 2 == 0 else "bf16",
                    seed=80 + i) for i in range(3)]


@pytest.mark.parametrize("pass_", [A.PASS_AUTO, A.PASS_TILE, A.PASS_REGISTERS],
                         ids=["auto", "tile", "registers"])
def test_threads_on_separate_streams_match_sequential_rounds(pass_):
    ws = _workloads()
    sequential = []
    for w in ws:
        g, v, xs = gpu_inputs(w)
        s = torch.cuda.Stream()
        stats = _rounds(w, g, v, xs, s, pass_)
        s.synchronize()
        sequential.append((stats, g.clone(), v.clone(), [x.clone() for x in xs]))

    bufs = [gpu_inputs(w) for w in ws]
    torch.cuda.synchronize()
    results = [None] * len(ws)
    errors = []

    def worker(i):
        try:
            g, v, xs = bufs[i]
            s = torch.cuda.Stream()
            results[i] = _rounds(ws[i], g, v, xs, s, pass_)
            s.synchronize()
        except Exception as e:  # reported below, on the test's thread
            errors.append(e)

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(len(ws))]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    torch.cuda.synchronize()
    for i, (stats, g0, v0, x0) in enumerate(sequential):
        g, v, xs = bufs[i]
        assert results[i] == stats, i
        assert torch.equal(g, g0) and torch.equal(v, v0)
        for a, b in zip(xs, x0):
            assert torch.equal(a, b)


def test_consecutive_rounds_on_two_streams_see_each_others_outputs():
    """A round on stream B that waits on stream A (an event) reads the
    outputs of A's round, although A's call may return before its kernel
    has retired."""
    w = W.small(2_000_003, 4, "f32", seed=90)
    sa, _ = schedule_pair(w.schedule)
    kw = dict(H_base=w.H_base, schedule=sa, outer_lr=w.outer_lr,
              outer_beta=w.outer_beta)

    def two_rounds(g, v, xs, s1, s2):
        st1 = A.sync(g, v, xs, H_sel=150, step=4000, stream=s1, **kw)
        ev = torch.cuda.Event()
        ev.record(s1)
        s2.wait_event(ev)
        st2 = A.sync(g, v, xs, H_sel=200, step=4150, stream=s2, **kw)
        s2.synchronize()
        return st1, st2

    g1, v1, x1 = gpu_inputs(w)
    s = torch.cuda.current_stream()
    a1, a2 = two_rounds(g1, v1, x1, s, s)
    g2, v2, x2 = gpu_inputs(w)
    b1, b2 = two_rounds(g2, v2, x2, torch.cuda.Stream(), torch.cuda.Stream())
    assert (a1["D"], a2["D"], a2["C"]) == (b1["D"], b2["D"], b2["C"])
    assert torch.equal(g1, g2) and torch.equal(v1, v2)
