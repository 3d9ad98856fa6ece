"""Failure detection on the GPU without a GPU fault: every mbarrier wait of
the bulk-copy pass and of the fused INT8 round is bounded, so a stage that
never fills makes the round return an error status while every kernel
finishes and the device stays usable.  The stall is requested through
aloco_test_stall_tile, which makes the issuing thread skip one tile's (or
one codec block's) copies: its barrier is then never completed, a flag that
nothing sets."""
import time

import pytest
import torch

from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import gpu_inputs, schedule_pair

pytestmark = pytest.mark.gpu


def _kw(w):
    sa, _ = schedule_pair(w.schedule)
    return dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step, schedule=sa,
                outer_lr=w.outer_lr, outer_beta=w.outer_beta)


def test_stalled_bulk_copy_stage_is_reported_and_the_device_stays_usable():
    w = W.small(1 << 22, 2, "f32", seed=5)
    kw = _kw(w)
    bulk = lambda: A.default_opts(pass_=A.PASS_BULK_COPY)
    g, v, xs = gpu_inputs(w)
    st = A.sync(g, v, xs, opts=bulk(), **kw)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_BULK_COPY
    tile = 3 * st["grid"] + 7        # the fourth tile of block 7

    g, v, xs = gpu_inputs(w)
    A.test_stall_tile(tile)
    t0 = time.time()
    st = A.sync(g, v, xs, opts=bulk(), raise_on_error=False, **kw)
    took = time.time() - t0
    assert st["status"] == A.ERR_CUDA
    assert "timed out" in A.last_error()
    assert 1.0 < took < 60.0, took       # the ~2 s bounded waits, not a hang
    torch.cuda.synchronize()             # nothing is left running

    # the hook was consumed, the error word cleared, and the pass works:
    # the next bulk-copy round equals the register pass bit for bit
    g1, v1, x1 = gpu_inputs(w)
    g2, v2, x2 = gpu_inputs(w)
    st1 = A.sync(g1, v1, x1, opts=bulk(), **kw)
    st2 = A.sync(g2, v2, x2, opts=A.default_opts(pass_=A.PASS_REGISTERS), **kw)
    assert st1["status"] == st2["status"] == A.OK
    assert st1["pass_used"] == A.PASS_BULK_COPY
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))
    assert st1["D"] == pytest.approx(st2["D"], rel=1e-6)


def test_stall_hook_ignored_by_other_rounds():
    """A register-pass round neither reads nor consumes the hook; the next
    bulk-copy round does."""
    w = W.small(1 << 20, 3, "bf16", seed=6)
    kw = _kw(w)
    A.test_stall_tile(0)
    g, v, xs = gpu_inputs(w)
    st = A.sync(g, v, xs, opts=A.default_opts(pass_=A.PASS_REGISTERS), **kw)
    assert st["status"] == A.OK
    A.test_stall_tile(-1)                 # cancel before any bulk-copy round
    g, v, xs = gpu_inputs(w)
    st = A.sync(g, v, xs, opts=A.default_opts(pass_=A.PASS_BULK_COPY), **kw)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_BULK_COPY


@pytest.mark.parametrize("M", [4, 16], ids=["two_ctas", "one_cta_prefetch"])
def test_stalled_int8_fused_block_is_reported_and_the_device_stays_usable(M):
    """M = 4: two CTAs per SM; M = 16: one CTA per SM, which also prefetches
    the next block into L2 and leaves its place in shared memory."""
    w = W.small(1 << 22, M, "bf16", seed=5)   # every codec block whole and aligned
    kw = _kw(w)
    fused = lambda: A.default_opts(pass_=A.PASS_INT8_FUSED)
    g, v, xs = gpu_inputs(w)
    st = A.sync_int8(g, v, xs, opts=fused(), **kw)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_INT8_FUSED
    block = 2 * st["grid"] + 5                # the third block of CTA 5
    assert block < (w.numel + 4095) // 4096

    g, v, xs = gpu_inputs(w)
    A.test_stall_tile(block)
    t0 = time.time()
    st = A.sync_int8(g, v, xs, opts=fused(), raise_on_error=False, **kw)
    took = time.time() - t0
    assert st["status"] == A.ERR_CUDA
    assert "timed out" in A.last_error()
    assert 1.0 < took < 60.0, took
    torch.cuda.synchronize()

    # the next fused round runs and equals the split form bit for bit
    g1, v1, x1 = gpu_inputs(w)
    g2, v2, x2 = gpu_inputs(w)
    st1 = A.sync_int8(g1, v1, x1, opts=fused(), **kw)
    st2 = A.sync_int8(g2, v2, x2, opts=A.default_opts(pass_=A.PASS_INT8_SPLIT), **kw)
    assert st1["status"] == st2["status"] == A.OK
    assert st1["pass_used"] == A.PASS_INT8_FUSED
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))
    for a_, b_ in zip(x1, x2):
        assert torch.equal(a_.view(torch.int16), b_.view(torch.int16))


def test_stalled_tile_pass_block_is_reported_and_the_device_stays_usable():
    w = W.small(1 << 22, 3, "f32", seed=5)
    kw = _kw(w)
    tile = lambda: A.default_opts(pass_=A.PASS_TILE)
    g, v, xs = gpu_inputs(w)
    st = A.sync(g, v, xs, opts=tile(), **kw)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_TILE
    block = 3 * st["grid"] + 11            # the fourth block of CTA 11
    assert block < w.numel // 4096

    g, v, xs = gpu_inputs(w)
    A.test_stall_tile(block)
    t0 = time.time()
    st = A.sync(g, v, xs, opts=tile(), raise_on_error=False, **kw)
    took = time.time() - t0
    assert st["status"] == A.ERR_CUDA
    assert "timed out" in A.last_error()
    assert 1.0 < took < 60.0, took
    torch.cuda.synchronize()

    g1, v1, x1 = gpu_inputs(w)
    g2, v2, x2 = gpu_inputs(w)
    st1 = A.sync(g1, v1, x1, opts=tile(), **kw)
    st2 = A.sync(g2, v2, x2, opts=A.default_opts(pass_=A.PASS_REGISTERS), **kw)
    assert st1["status"] == st2["status"] == A.OK
    assert st1["pass_used"] == A.PASS_TILE
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))


def test_stalled_int8_worker_group_block_is_reported_and_the_device_stays_usable():
    """The fused INT8 round with worker groups (fp32, M > 8): a block whose
    first group never arrives makes the round report the timeout; the next
    round equals the split form bit for bit."""
    w = W.small(1 << 22, 12, "f32", seed=6)
    kw = _kw(w)
    fused = lambda: A.default_opts(pass_=A.PASS_INT8_FUSED)
    g, v, xs = gpu_inputs(w)
    st = A.sync_int8(g, v, xs, opts=fused(), **kw)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_INT8_FUSED
    block = 2 * st["grid"] + 9                # the third block of CTA 9
    assert block < w.numel // 4096

    g, v, xs = gpu_inputs(w)
    A.test_stall_tile(block)
    t0 = time.time()
    st = A.sync_int8(g, v, xs, opts=fused(), raise_on_error=False, **kw)
    took = time.time() - t0
    assert st["status"] == A.ERR_CUDA
    assert "timed out" in A.last_error()
    assert 1.0 < took < 60.0, took
    torch.cuda.synchronize()

    g1, v1, x1 = gpu_inputs(w)
    g2, v2, x2 = gpu_inputs(w)
    st1 = A.sync_int8(g1, v1, x1, opts=fused(), **kw)
    st2 = A.sync_int8(g2, v2, x2, opts=A.default_opts(pass_=A.PASS_INT8_SPLIT), **kw)
    assert st1["status"] == st2["status"] == A.OK
    assert torch.equal(g1.view(torch.int32), g2.view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2.view(torch.int32))
    for a_, b_ in zip(x1, x2):
        assert torch.equal(a_.view(torch.int32), b_.view(torch.int32))

