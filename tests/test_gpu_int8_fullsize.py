"""The INT8-communicated round (App. G.1) at the benchmark's full sizes, in
the launch configuration bench.py times (AUTO form): the Llama-style 1B set
with 4 bf16 workers and the 3B set with 8.  Every codec block is
self-contained (its scale, its mean and its outputs depend on that block
alone), so the oracle checks sampled whole blocks one by one; D_t comes from
the pre-quantisation pseudo-gradients, which the oracle sums over the whole
vector; the replica reset is checked everywhere."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import (RTOL_STAT, assert_bf16_replica, assert_field, gpu_inputs,
                     oracle_corr, oracle_stats_threaded, schedule_pair,
                     to_numpy_bits)

pytestmark = pytest.mark.gpu


def _blocks(parts):
    """(start, length) of every codec block, part by part."""
    out, off = [], 0
    for p in parts:
        for b in range(0, p, 4096):
            out.append((off + b, min(4096, p - b)))
        off += p
    return out


@pytest.mark.parametrize("make", [W.llama_1b, W.llama_3b], ids=["llama1b", "llama3b"])
def test_int8_round_full_size_sampled_blocks(make):
    w = make()
    parts = W.tensor_sizes(w)
    g, v, xs = gpu_inputs(w)
    step, hsel = W.steps_of_rounds(w)[0]
    corr = oracle_corr(w, step, hsel)
    pre = oracle_stats_threaded(g, xs, 1e-8)

    blocks = _blocks(parts)
    rng = np.random.default_rng(7)
    pick = set(rng.choice(len(blocks), 160, replace=False).tolist())
    starts = np.cumsum([0] + parts[:-1])
    for p in rng.choice(len(parts), 16, replace=False):   # ends of some tensors
        first = int(np.searchsorted([b[0] for b in blocks], starts[p]))
        pick.update([first, first + (parts[p] - 1) // 4096])
    pick.update([0, len(blocks) - 1])
    chosen = [blocks[i] for i in sorted(pick)]
    saved = [(g[s:s + n].cpu().numpy(), v[s:s + n].cpu().numpy(),
              [to_numpy_bits(x[s:s + n]) for x in xs]) for s, n in chosen]

    sa, _ = schedule_pair(w.schedule)
    st = A.sync_int8(g, v, xs, parts=parts, H_sel=hsel, H_base=w.H_base, step=step,
                     schedule=sa, outer_lr=w.outer_lr, outer_beta=w.outer_beta)
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_INT8_FUSED

    for (s, n), (gh, vh, xh) in zip(chosen, saved):
        orc = O.int8_round(gh, vh, xh, O.BF16, [n], corr.mu_t, corr.eta_out,
                           corr.inv_norm)
        assert_field(g[s:s + n].cpu().numpy(), orc["g"], f"theta' block @{s}")
        assert_field(v[s:s + n].cpu().numpy(), orc["v"], f"v' block @{s}")
        assert_bf16_replica(to_numpy_bits(xs[0][s:s + n]), orc["x"][0], orc["g"],
                            f"replica block @{s}")
    # D_t from the pre-quantisation pseudo-gradients over the whole vector
    assert st["D"] == pytest.approx(pre["D"], rel=RTOL_STAT)
    for m in range(w.M):
        assert st["drift"][m] == pytest.approx(pre["drift"][m], rel=RTOL_STAT)
    # every replica is theta' rounded to bf16
    want = g.to(torch.bfloat16)
    for x in xs:
        assert torch.equal(x.view(torch.int16), want.view(torch.int16))
