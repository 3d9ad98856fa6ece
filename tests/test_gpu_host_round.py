"""The outer round on host-resident state (aloco_sync_host): theta, v and the
replicas in page-locked host memory, streamed through the GPU in chunks.
Per-element results must equal the device round's bit for bit.  The
statistics agree within the statistics tolerance: chunking changes which
elements share a thread's fp32 partial sum before it is added in fp64."""
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import RTOL_STAT, assert_field, gpu_inputs, schedule_pair

pytestmark = pytest.mark.gpu


def _pinned(t):
    return t.detach().cpu().pin_memory()


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def _rounds(w, chunk, stream=None):
    g, v, xs = gpu_inputs(w)
    v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(w.M))
    gh, vh, xh = _pinned(g), _pinned(v), [_pinned(x) for x in xs]
    x_before = [x.clone() for x in xh]
    sa, _ = schedule_pair(w.schedule)
    kw = dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step, schedule=sa,
              outer_lr=w.outer_lr, outer_beta=w.outer_beta)
    st_d = A.sync(g, v, xs, **kw)
    st_h = A.sync_host(gh, vh, xh, chunk_elems=chunk, stream=stream, **kw)
    return g, v, xs, gh, vh, xh, x_before, st_d, st_h


@pytest.mark.parametrize("dt,M,N,chunk", [
    ("f32", 1, 1000, 0),                 # one chunk shorter than a pack row
    ("f32", 3, 1_000_003, 65_536),       # many chunks, ragged tail
    ("bf16", 8, 1_000_003, 100_000),
    ("bf16", 5, 300_001, 8),             # the smallest chunk: 37,501 chunks
    ("f32", 8, 4_194_309, 0),            # default chunk, one chunk
    ("bf16", 16, 2_000_000, 1 << 20),
    ("f32", 32, 50_000, 4096),
    ("f32", 4, 40_000_001, 0),           # default chunk, three chunks
])
def test_host_round_equals_device_round(dt, M, N, chunk):
    w = W.small(N, M, dt, seed=60 + M)
    g, v, xs, gh, vh, xh, x_before, st_d, st_h = _rounds(w, chunk)
    assert st_h["status"] == A.OK
    assert torch.equal(_bits(gh), _bits(g.cpu()))
    assert torch.equal(_bits(vh), _bits(v.cpu()))
    for a, b in zip(xh, x_before):          # host replicas are inputs only
        assert torch.equal(_bits(a), _bits(b))
    for key in ("D", "C", "mean_sq_norm"):
        assert st_h[key] == pytest.approx(st_d[key], rel=RTOL_STAT), key
    for a, b in zip(st_h["drift"][:M], st_d["drift"][:M]):
        assert a == pytest.approx(b, rel=RTOL_STAT)
    assert st_h["nonfinite"] == st_d["nonfinite"] == 0
    assert st_h["corr"] == st_d["corr"]


def test_host_round_matches_the_oracle():
    w = W.small(777_777, 4, "f32", seed=3)
    g, v, xs = gpu_inputs(w)
    gh, vh, xh = _pinned(g), _pinned(v), [_pinned(x) for x in xs]
    sa, so = schedule_pair(w.schedule)
    orc = O.sync_round(gh.numpy(), vh.numpy(), [x.numpy() for x in xh], O.F32,
                       so, w.start_step, w.H_sel[0], w.H_base,
                       w.outer_lr, w.outer_beta)
    st = A.sync_host(gh, vh, xh, H_sel=w.H_sel[0], H_base=w.H_base,
                     step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                     outer_beta=w.outer_beta, chunk_elems=100_000)
    assert_field(gh.numpy(), orc["g"], "theta'")
    assert_field(vh.numpy(), orc["v"], "v'")
    for key in ("D", "C"):
        assert st[key] == pytest.approx(orc[key], rel=RTOL_STAT)


def test_side_stream_and_nonfinite_counts():
    w = W.small(500_000, 3, "bf16", seed=8)
    g, v, xs = gpu_inputs(w)
    xs[1][12345] = float("nan")
    xs[2][499_999] = float("inf")
    gh, vh, xh = _pinned(g), _pinned(v), [_pinned(x) for x in xs]
    sa, _ = schedule_pair(w.schedule)
    kw = dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step, schedule=sa,
              outer_lr=w.outer_lr, outer_beta=w.outer_beta)
    st_d = A.sync(g, v, xs, **kw)
    s = torch.cuda.Stream()
    st_h = A.sync_host(gh, vh, xh, chunk_elems=65_536, stream=s,
                       opts=A.default_opts(time_kernel=1), **kw)
    assert st_d["status"] == st_h["status"] == A.ERR_NONFINITE
    assert st_h["nonfinite"] == st_d["nonfinite"] == 2
    assert st_h["kernel_ms"] > 0
    assert torch.equal(_bits(gh), _bits(g.cpu()))


def test_pageable_memory_and_bulk_copy_are_rejected():
    w = W.small(10_000, 2, "f32", seed=1)
    g, v, xs = gpu_inputs(w)
    sa, _ = schedule_pair(w.schedule)
    kw = dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step, schedule=sa,
              outer_lr=w.outer_lr, outer_beta=w.outer_beta)
    pageable = g.cpu()
    with pytest.raises(A.AlocoError) as ei:
        A.sync_host(pageable, _pinned(v), [_pinned(x) for x in xs], **kw)
    assert ei.value.status == A.ERR_ARG and "page-locked" in str(ei.value)
    with pytest.raises(A.AlocoError) as ei:                  # device memory
        A.sync_host(g, v, xs, **kw)
    assert ei.value.status == A.ERR_ARG
    with pytest.raises(A.AlocoError) as ei:
        A.sync_host(_pinned(g), _pinned(v), [_pinned(x) for x in xs],
                    opts=A.default_opts(pass_=A.PASS_BULK_COPY), **kw)
    assert ei.value.status == A.ERR_ARG
