"""The INT8-communicated round (App. G.1) at the benchmark's full sizes, in
the launch configuration bench.py times (AUTO form): the Llama-style 1B set
with 4 bf16 workers and the 3B set with 8, and the 1B layout with the
paper's 16 INT8 workers (one CTA per SM, the L2 prefetch of the next block,
the mixed-precision subtraction and the per-block energy sums).  Every element of theta', v' and
the replica reset is compared with the oracle's INT8 round, which runs slice
by slice (whole codec blocks each: the blocks restart at every tensor part)
on host copies of a device snapshot of the inputs; the slices' sums give the
whole round's D_t (pre-quantisation pseudo-gradients), ||Dbar||^2 and C_t
(decoded aggregate), compared at the statistics tolerance; every replica is
checked on the device to equal theta' rounded to bf16."""
import dataclasses
import gc

import pytest
import torch

from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W
from _parity import (assert_corr, assert_stats, compare_int8_whole_vector,
                     gpu_inputs, oracle_corr, schedule_pair)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _llama_1b_16_workers():
    return dataclasses.replace(W.llama_1b(), name="llama1b_m16_bf16", M=16)


@pytest.mark.parametrize("make", [W.llama_1b, W.llama_3b, _llama_1b_16_workers],
                         ids=["llama1b", "llama3b", "llama1b_m16"])
def test_int8_round_full_size_whole_vector(make):
    w = make()
    parts = W.tensor_sizes(w)
    g, v, xs = gpu_inputs(w)
    g_in, v_in = g.clone(), v.clone()
    x_in = [x.clone() for x in xs]
    step, hsel = W.steps_of_rounds(w)[0]
    corr = oracle_corr(w, step, hsel)
    sa, _ = schedule_pair(w.schedule)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    st = A.sync_int8(g, v, xs, parts=parts, H_sel=hsel, H_base=w.H_base, step=step,
                     schedule=sa, outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                     opts=A.default_opts(time_kernel=1), stream=stream)
    torch.cuda.synchronize()
    assert st["status"] == A.OK and st["pass_used"] == A.PASS_INT8_FUSED
    assert_corr(st["corr"], corr)
    # every replica is theta' rounded to bf16
    want = g.to(torch.bfloat16)
    for x in xs:
        assert torch.equal(x.view(torch.int16), want.view(torch.int16))
    orc = compare_int8_whole_vector(w, parts, g_in, v_in, x_in, g, v, xs, corr)
    assert_stats(st, orc, w.M)
    del g, v, xs, g_in, v_in, x_in
    gc.collect()
    torch.cuda.empty_cache()
