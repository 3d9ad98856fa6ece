"""The inner AdamW step (Sec. 2; Tab. training settings) at the bench's
full size with bf16 replicas: the Llama-style 1B set, 4 workers, in the
launch configuration bench.py --mode adamw times.  The clipping norm of each
replica is summed on the host in float64 over the whole gradient; sampled
elements are checked against the oracle given those norms (every element
depends only on its own inputs and its replica's clipping factor)."""
import concurrent.futures as cf

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import (RTOL_STAT, assert_bf16_replica, assert_field,
                     sample_indices, to_numpy_bits)

pytestmark = pytest.mark.gpu


def _norm_host(t, slice_elems=1 << 24):
    """||t|| in float64 over the whole vector, slices added in order."""
    n = t.numel()
    bounds = [(s, min(n, s + slice_elems)) for s in range(0, n, slice_elems)]

    def part(b):
        s, e = b
        x = t[s:e].float().cpu().numpy().astype(np.float64)
        return float(np.dot(x, x))
    with cf.ThreadPoolExecutor(8) as ex:
        sq = list(ex.map(part, bounds))
    return float(np.sqrt(sum(sq)))


def test_adamw_full_size_llama1b_bf16():
    w = W.llama_1b()
    N, M = w.numel, w.M
    gen = torch.Generator("cuda").manual_seed(101)

    def draw(scale, dt, positive=False):
        t = torch.empty(N, device="cuda")
        t.normal_(0, 1, generator=gen)
        if positive:
            t.abs_()
        return t.mul_(scale).to(dt)
    xs = [draw(0.02, torch.bfloat16) for _ in range(M)]
    gs = [draw(3.0 / N ** 0.5 * (1 + m), torch.bfloat16) for m in range(M)]
    m1 = [draw(1e-4, torch.float32) for _ in range(M)]
    m2 = [draw(1e-8, torch.float32, True) for _ in range(M)]
    norms = [_norm_host(g) for g in gs]
    idx = sample_indices(N, W.tensor_boundaries(w), k=8192, seed=5)
    before = [(to_numpy_bits(xs[m][idx.cuda()]), to_numpy_bits(gs[m][idx.cuda()]),
               m1[m][idx.cuda()].cpu().numpy(), m2[m][idx.cuda()].cpu().numpy())
              for m in range(M)]
    cfg = dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1,
               max_grad_norm=1.0, step=1200)
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(**cfg))
    assert st["status"] == A.OK
    for m in range(M):
        assert st["grad_norm"][m] == pytest.approx(norms[m], rel=RTOL_STAT)
        x, g, a, b = before[m]
        orc = O.adamw_step([x], O.BF16, [g], O.BF16, [a], [b], cfg["lr"],
                           cfg["beta1"], cfg["beta2"], cfg["eps"],
                           cfg["weight_decay"], cfg["max_grad_norm"], cfg["step"],
                           norms=[norms[m]])
        assert_bf16_replica(to_numpy_bits(xs[m][idx.cuda()]), orc["x_store"][0],
                            orc["x"][0], f"x'[{m}]")
        assert_field(m1[m][idx.cuda()].cpu().numpy(), orc["m1"][0], f"m'[{m}]")
        assert_field(m2[m][idx.cuda()].cpu().numpy(), orc["m2"][0], f"v'[{m}]")
    assert min(st["clip"]) < 1.0
