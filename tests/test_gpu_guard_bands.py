"""Guard bands: every kernel writes only [0, N) of its buffers.  Each
buffer sits inside a larger allocation with sentinel elements on both sides
(64 elements, so 16-byte alignment is kept and the vector paths run, or 1
element, so the buffers are misaligned and the element paths run); after
the call the sentinels must be intact."""
import pytest
import torch

from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import gpu_inputs, schedule_pair

pytestmark = pytest.mark.gpu

PARTS = [3 * 4096 + 5, 17, 4096, 8191, 64]


def _padded(t, pad, fill, device="cuda", pin=False):
    big = torch.full((t.numel() + 2 * pad,), fill, dtype=t.dtype, device=device)
    if pin:
        big = big.pin_memory()
    big[pad:pad + t.numel()] = t.to(device)
    return big, big[pad:pad + t.numel()]


def _intact(big, pad, fill):
    return bool(torch.all(big[:pad] == fill)) and bool(torch.all(big[-pad:] == fill))


def _kw(w):
    sa, _ = schedule_pair(w.schedule)
    return dict(H_sel=w.H_sel[0], H_base=w.H_base, step=w.start_step, schedule=sa,
                outer_lr=w.outer_lr, outer_beta=w.outer_beta)


@pytest.mark.parametrize("pad", [64, 1])
@pytest.mark.parametrize("form", [A.PASS_INT8_FUSED, A.PASS_INT8_SPLIT],
                         ids=["fused", "split"])
@pytest.mark.parametrize("dt,M", [("f32", 3), ("bf16", 8), ("f32", 8), ("bf16", 5),
                                  ("bf16", 16)])
def test_int8_round(dt, M, form, pad):
    N = sum(PARTS)
    w = W.small(N, M, dt, seed=31)
    g, v, xs = gpu_inputs(w)
    gb, gi = _padded(g, pad, 7.0)
    vb, vi = _padded(v, pad, -7.0)
    xb = [_padded(x, pad, 3.0) for x in xs]
    st = A.sync_int8(gi, vi, [x[1] for x in xb], parts=PARTS,
                     opts=A.default_opts(pass_=form), **_kw(w))
    assert st["status"] == A.OK and st["pass_used"] == form
    assert _intact(gb, pad, 7.0) and _intact(vb, pad, -7.0)
    assert all(_intact(x[0], pad, 3.0) for x in xb)


@pytest.mark.parametrize("pad", [64, 1])
def test_int8_codec(pad):
    N = sum(PARTS)
    y = torch.randn(N, device="cuda", generator=torch.Generator("cuda").manual_seed(pad)) * 1e-3
    yb, yi = _padded(y, pad, 5.0)
    nb = A.int8_num_blocks(PARTS)
    cb = torch.full((N + 2 * pad,), 99, dtype=torch.int8, device="cuda")
    sb = torch.full((nb + 2 * pad,), 5.0, device="cuda")
    db = torch.full((N + 2 * pad,), 5.0, device="cuda")
    ci, si, di = cb[pad:pad + N], sb[pad:pad + nb], db[pad:pad + N]
    import ctypes
    lib = A.load()
    arr = (ctypes.c_int64 * len(PARTS))(*PARTS)
    s = torch.cuda.current_stream().cuda_stream
    assert lib.aloco_int8_encode(yi.data_ptr(), N, arr, len(PARTS), ci.data_ptr(),
                                 si.data_ptr(), di.data_ptr(), s) == A.OK
    assert lib.aloco_int8_decode(ci.data_ptr(), si.data_ptr(), N, arr, len(PARTS),
                                 di.data_ptr(), s) == A.OK
    torch.cuda.synchronize()
    assert _intact(yb, pad, 5.0) and _intact(db, pad, 5.0) and _intact(sb, pad, 5.0)
    assert bool(torch.all(cb[:pad] == 99)) and bool(torch.all(cb[-pad:] == 99))


@pytest.mark.parametrize("pad", [64, 1])
@pytest.mark.parametrize("pdt,gdt", [(torch.float32, torch.float32),
                                     (torch.bfloat16, torch.bfloat16),
                                     (torch.float32, torch.bfloat16),
                                     (torch.bfloat16, torch.float32)])
def test_adamw(pdt, gdt, pad):
    N, M = 100_003, 3
    gen = torch.Generator("cuda").manual_seed(4)
    mk = lambda dt, sc: (torch.randn(N, generator=gen, device="cuda") * sc).to(dt)
    bufs = {"x": [_padded(mk(pdt, 0.02), pad, 2.0) for _ in range(M)],
            "g": [_padded(mk(gdt, 1e-2), pad, -2.0) for _ in range(M)],
            "m1": [_padded(mk(torch.float32, 1e-3), pad, 9.0) for _ in range(M)],
            "m2": [_padded(mk(torch.float32, 1e-6).abs(), pad, -9.0) for _ in range(M)]}
    st = A.adamw_step(*[[b[1] for b in bufs[k]] for k in ("x", "g", "m1", "m2")],
                      A.adamw_cfg(step=3))
    assert st["status"] == A.OK
    for k, fill in (("x", 2.0), ("g", -2.0), ("m1", 9.0), ("m2", -9.0)):
        assert all(_intact(b[0], pad, fill) for b in bufs[k]), k


@pytest.mark.parametrize("pad", [64, 1])
def test_host_round(pad):
    N, M = 300_007, 3
    w = W.small(N, M, "bf16", seed=12)
    g, v, xs = gpu_inputs(w)
    gb, gi = _padded(g, pad, 7.0, device="cpu", pin=True)
    vb, vi = _padded(v, pad, -7.0, device="cpu", pin=True)
    xb = [_padded(x, pad, 3.0, device="cpu", pin=True) for x in xs]
    st = A.sync_host(gi, vi, [x[1] for x in xb], chunk_elems=65_536, **_kw(w))
    assert st["status"] == A.OK
    assert _intact(gb, pad, 7.0) and _intact(vb, pad, -7.0)
    assert all(_intact(x[0], pad, 3.0) for x in xb)
