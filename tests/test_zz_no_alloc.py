"""aloco_sync_noalloc, the entry point that allocates nothing.

Some callers cannot let a library allocate memory: frameworks that reserve
all device memory up front and serve it from their own pools, deployments
whose footprint must be fixed when the library loads, and loops that cannot
afford the device-wide synchronisation of cudaMalloc / cudaFree.  For them
aloco_sync_noalloc keeps its scratch in a static device array inside the
library.  These tests call it through the C ABI and check it against
aloco_sync_ex, the entry point that allocates a cached workspace, on the
same inputs, on two calls in a row, within the tolerances of the parity
tests.  The file is collected last so that a run stopping at the first
failure has already run every other test; it also passes on its own in a
fresh process.
"""
import numpy as np
import pytest
import torch

from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

from _parity import (RTOL_STAT, assert_corr, assert_field, assert_rel,
                     assert_stats, compare_sampled, gather_host, gpu_inputs,
                     oracle_corr, oracle_pass2_at, oracle_stats_threaded,
                     sample_indices, schedule_pair, to_numpy_bits)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _round(w, g, v, xs, noalloc, opts=None):
    sa, _ = schedule_pair(w.schedule)
    return A.sync(g, v, xs, H_sel=w.H_sel[0], H_base=w.H_base,
                  step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                  outer_beta=w.outer_beta, opts=opts, noalloc=noalloc)


@pytest.mark.parametrize("pass_", [A.PASS_AUTO, A.PASS_BULK_COPY, A.PASS_TILE],
                         ids=["auto", "bulk_copy", "tile"])
@pytest.mark.parametrize("dt,N,M", [("f32", 1_000_003, 8),
                                    ("bf16", 2_000_005, 5),
                                    ("f32", 4099, 17)])
def test_noalloc_matches_the_allocating_entry_point(dt, N, M, pass_):
    w = W.small(N, M, dt, seed=31)
    opts = A.default_opts(pass_=pass_)
    for call in range(2):
        g, v, xs = gpu_inputs(w, round_index=call)
        v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(call))
        g2, v2, xs2 = g.clone(), v.clone(), [x.clone() for x in xs]
        # the first call starts with the allocation-free entry point, so a
        # fresh process exercises its set-up before anything else
        if call == 0:
            st_new = _round(w, g2, v2, xs2, noalloc=True, opts=opts)
            st_ref = _round(w, g, v, xs, noalloc=False, opts=opts)
        else:
            st_ref = _round(w, g, v, xs, noalloc=False, opts=opts)
            st_new = _round(w, g2, v2, xs2, noalloc=True, opts=opts)
        assert st_new["status"] == A.OK and st_ref["status"] == A.OK
        assert st_new["kernel_ms"] == -1.0
        assert st_new["nonfinite"] == st_ref["nonfinite"] == 0
        for k in ("D", "C", "mean_sq_norm"):
            assert_rel(st_new[k], st_ref[k], k, RTOL_STAT)
        for m in range(M):
            assert_rel(st_new["drift"][m], st_ref["drift"][m], f"drift {m}",
                       RTOL_STAT)
        assert st_new["corr"] == st_ref["corr"]
        assert st_new["pass_used"] == st_ref["pass_used"]
        assert st_new["grid"] == st_ref["grid"]
        assert_field(g2.cpu().numpy(), g.cpu().numpy().astype(np.float64),
                     "theta'")
        assert_field(v2.cpu().numpy(), v.cpu().numpy().astype(np.float64),
                     "v'")
        for a, b in zip(xs2, xs):
            if dt == "f32":
                assert_field(a.cpu().numpy(), b.cpu().numpy().astype(
                    np.float64), "replica")
            else:
                d = np.abs(to_numpy_bits(a).astype(np.int64) -
                           to_numpy_bits(b).astype(np.int64))
                assert d.max() <= 1


def test_noalloc_reports_nonfinite_and_bad_arguments():
    w = W.small(10_000, 3, "f32", seed=32)
    g, v, xs = gpu_inputs(w)
    xs[1][17] = float("nan")
    st = _round(w, g, v, xs, noalloc=True)
    assert st["status"] == A.ERR_NONFINITE and st["nonfinite"] == 1
    sa, _ = schedule_pair(w.schedule)
    rc, _ = A.sync_ptrs(g.data_ptr(), v.data_ptr(), [x.data_ptr() for x in xs],
                        w.numel, 7, 150, 100, 4000, sa, 0.7, 0.9,
                        raise_on_error=False, noalloc=True)
    assert rc == A.ERR_ARG and "dtype" in A.last_error()
    rc, _ = A.sync_ptrs(g.data_ptr(), v.data_ptr(), [g.data_ptr() + 64],
                        w.numel, A.F32, 150, 100, 4000, sa, 0.7, 0.9,
                        raise_on_error=False, noalloc=True)
    assert rc == A.ERR_ALIAS


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


@pytest.mark.parametrize("dt,M", [("bf16", 8), ("f32", 8)])
def test_noalloc_large_round_is_the_allocating_round_bit_for_bit(dt, M):
    """From 2^27 parameters AUTO takes the tile pass in both entry points:
    the same kernel and grid, so outputs and statistics are the same bits.
    The round is also checked against the oracle: D_t, C_t and the drift
    energies over the whole vector, theta' and v' on sampled elements."""
    N = (1 << 27) + 4099
    w = W.small(N, M, dt, seed=33)
    outs = {}
    for noalloc in (True, False):
        g, v, xs = gpu_inputs(w)
        v.normal_(0, 1e-3, generator=torch.Generator("cuda").manual_seed(5))
        if noalloc:
            idx = sample_indices(N, k=4096)
            g_idx, v_idx = gather_host(g, idx), gather_host(v, idx)
            x_idx = [gather_host(x, idx) for x in xs]
            orc = oracle_stats_threaded(g, xs, 1e-8)
        st = _round(w, g, v, xs, noalloc=noalloc)
        assert st["status"] == A.OK
        assert st["pass_used"] == A.PASS_TILE
        outs[noalloc] = (st, [g, v, *xs])
    (s1, t1), (s0, t0) = outs[True], outs[False]
    for a, b in zip(t1, t0):
        assert torch.equal(_bits(a), _bits(b))
    for k in ("D", "C", "mean_sq_norm", "drift", "grid", "nonfinite"):
        assert s1[k] == s0[k], k
    corr = oracle_corr(w, w.start_step, w.H_sel[0])
    assert_corr(s1["corr"], corr)
    assert_stats(s1, orc, M)
    ref = oracle_pass2_at(w, g_idx, v_idx, x_idx, corr)
    g, v, *xs = t1
    compare_sampled(w, gather_host(g, idx), gather_host(v, idx),
                    [gather_host(x, idx) for x in xs], ref)


def test_noalloc_refuses_a_capturing_stream():
    """The call ends with a stream synchronisation, which no capture can
    contain: on a capturing stream it returns ALOCO_ERR_ARG before any other
    CUDA call, and the caller's capture stays valid."""
    w = W.small(100_003, 2, "f32", seed=34)
    g, v, xs = gpu_inputs(w)
    assert _round(w, g, v, xs, noalloc=True)["status"] == A.OK
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    sa, _ = schedule_pair(w.schedule)
    with torch.cuda.stream(s):
        graph.capture_begin(capture_error_mode="relaxed")
        try:
            st = A.sync(g, v, xs, H_sel=w.H_sel[0], H_base=w.H_base,
                        step=w.start_step, schedule=sa, outer_lr=w.outer_lr,
                        outer_beta=w.outer_beta, stream=s, noalloc=True,
                        raise_on_error=False)
            g.mul_(1.0)            # one captured node, so the graph is valid
        finally:
            graph.capture_end()
    assert st["status"] == A.ERR_ARG
    assert "capture" in A.last_error()
    graph.replay()
    torch.cuda.synchronize()


def test_noalloc_caps_a_large_blocks_per_sm_at_occupancy():
    """blocks_per_sm asks for a residency; every pass caps it at what the
    kernel's occupancy allows (at most 8 blocks of 256 threads per SM), so
    even an oversized request stays within the static scratch and gives the
    allocating entry point's grid, outputs and statistics."""
    w = W.small(3_000_017, 4, "f32", seed=35)
    opts = A.default_opts(pass_=A.PASS_REGISTERS, blocks_per_sm=64)
    out = {}
    for noalloc in (True, False):
        g, v, xs = gpu_inputs(w)
        st = _round(w, g, v, xs, noalloc=noalloc, opts=opts)
        assert st["status"] == A.OK
        out[noalloc] = (st, [g, v, *xs])
    (s1, t1), (s0, t0) = out[True], out[False]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert s1["grid"] == s0["grid"] <= 8 * sms
    for a, b in zip(t1, t0):
        assert torch.equal(_bits(a), _bits(b))
    for k in ("D", "C", "mean_sq_norm", "drift"):
        assert s1[k] == s0[k], k
