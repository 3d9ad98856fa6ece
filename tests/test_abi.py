"""CPU-side checks of the C ABI: the library loads, exports every function
that include/aloco.h declares, the ctypes structures match the C layout,
and the host-only entry points (schedule mass, correction context,
argument validation) agree with the oracle.  No GPU is needed: nothing here
launches a kernel."""
import ctypes
import math
import os
import re
import subprocess

import numpy as np
import pytest

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "aloco.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return A.load()


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"\b(aloco_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


def test_every_declared_function_is_exported(lib):
    declared = _declared_functions()
    assert declared, "no declarations parsed"
    assert sorted(A.EXPORTS) == declared
    for name in declared:
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", A.library_path()],
                         capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (aloco_\w+)", out))
    assert set(declared) <= exported


def test_struct_layout_matches_c(tmp_path):
    """Compile a probe against the public header and compare sizeof and
    offsetof with the ctypes mirrors used by the binding."""
    src = tmp_path / "probe.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "aloco.h"
int main(void) {
  printf("%zu %zu %zu %zu\n", sizeof(aloco_schedule_t), sizeof(aloco_opts_t),
         sizeof(aloco_correction_t), sizeof(aloco_stats_t));
  printf("%zu %zu %zu %zu %zu %zu\n", sizeof(aloco_ctrl_cfg_t),
         sizeof(aloco_ctrl_state_t), sizeof(aloco_interval_obs_t),
         sizeof(aloco_ctrl_decision_t), offsetof(aloco_ctrl_state_t, hist_C),
         offsetof(aloco_ctrl_state_t, referenced));
  printf("%zu %zu %zu %zu %zu %zu %zu\n", offsetof(aloco_opts_t, pass), offsetof(aloco_opts_t, stream),
         offsetof(aloco_stats_t, corr), offsetof(aloco_stats_t, nonfinite),
         offsetof(aloco_stats_t, kernel_ms), offsetof(aloco_schedule_t, peak_lr),
         offsetof(aloco_schedule_t, total_steps));
  printf("%zu %zu %zu %zu %zu\n", sizeof(aloco_adamw_cfg_t),
         sizeof(aloco_adamw_stats_t), offsetof(aloco_adamw_cfg_t, step),
         offsetof(aloco_adamw_stats_t, clip), offsetof(aloco_adamw_stats_t, kernel_ms));
  return 0;
}
''')
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe)], check=True)
    lines = subprocess.run([str(exe)], capture_output=True, text=True,
                           check=True).stdout.split("\n")
    sizes = list(map(int, lines[0].split()))
    ctrl = list(map(int, lines[1].split()))
    offs = list(map(int, lines[2].split()))
    assert ctrl == [ctypes.sizeof(A.CtrlCfg), ctypes.sizeof(A.CtrlState),
                    ctypes.sizeof(A.IntervalObs), ctypes.sizeof(A.CtrlDecision),
                    A.CtrlState.hist_C.offset, A.CtrlState.referenced.offset]
    assert sizes == [ctypes.sizeof(A.Schedule), ctypes.sizeof(A.Opts),
                     ctypes.sizeof(A.Correction), ctypes.sizeof(A.Stats)]
    adam = list(map(int, lines[3].split()))
    assert adam == [ctypes.sizeof(A.AdamwCfg), ctypes.sizeof(A.AdamwStats),
                    A.AdamwCfg.step.offset, A.AdamwStats.clip.offset,
                    A.AdamwStats.kernel_ms.offset]
    assert offs == [A.Opts.pass_.offset, A.Opts.stream.offset,
                    A.Stats.corr.offset,
                    A.Stats.nonfinite.offset, A.Stats.kernel_ms.offset,
                    A.Schedule.peak_lr.offset, A.Schedule.total_steps.offset]


def test_default_opts_are_the_papers_settings(lib):
    """Tab. AutoLoCo configuration: momentum bounds [0.45, 0.90], maximum
    outer-step scale 1.6."""
    o = A.default_opts()
    assert (o.mu_min, o.mu_max, o.kappa_max) == (0.45, 0.90, 1.6)
    assert o.eps == 1e-8 and o.normalize == 0 and o.mode == A.CORR_FULL
    assert o.stream is None and o.time_kernel == 0
    assert o.pass_ == A.PASS_AUTO and o.blocks_per_sm == 0


@pytest.mark.parametrize("kind", [0, 1, 2])
def test_lr_accum_matches_oracle(lib, kind):
    rng = np.random.default_rng(kind)
    sa = A.Schedule.make(kind, 4e-4, 4e-5, 1000, 40000)
    so = O.Schedule(kind, 4e-4, 4e-5, 1000, 40000)
    cases = [(0, 0), (0, 1), (999, 1), (999, 2), (39990, 30), (50000, 7),
             (15000, 250), (4000, 150)]
    cases += [(int(rng.integers(0, 45000)), int(rng.integers(0, 5000)))
              for _ in range(100)]
    for t0, H in cases:
        want = O.lr_mass(so, t0, H)
        got = A.inner_lr_accum(sa, t0, H)
        assert got == pytest.approx(want, rel=1e-12, abs=1e-300), (t0, H)


def test_lr_accum_rejects_bad_arguments(lib):
    s = A.Schedule.make()
    assert math.isnan(A.inner_lr_accum(s, -1, 5))
    assert math.isnan(A.inner_lr_accum(s, 0, -5))
    bad = A.Schedule.make(warmup_steps=500, total_steps=500)
    assert math.isnan(A.inner_lr_accum(bad, 0, 5))
    assert "warmup" in A.last_error()
    assert math.isnan(A.inner_lr_accum(A.Schedule.make(kind=7), 0, 5))
    assert math.isnan(A.inner_lr_accum(A.Schedule.make(peak_lr=-1.0), 0, 5))


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("normalize", [0, 1])
def test_correction_matches_oracle(lib, mode, normalize):
    rng = np.random.default_rng(10 * mode + normalize)
    for _ in range(150):
        total = int(rng.integers(2000, 60000))
        sa = A.Schedule.make(0, 4e-4, 4e-5, 1000, total)
        so = O.Schedule(0, 4e-4, 4e-5, 1000, total)
        step = int(rng.integers(0, total + 1000))
        hs, hb = int(rng.integers(1, 2000)), int(rng.integers(1, 1000))
        eta = float(rng.uniform(0.1, 1.5))
        beta = float(rng.uniform(0.3, 0.95))
        opts = A.default_opts(mode=mode, normalize=normalize)
        c = A.correction(sa, step, hs, hb, eta, beta, opts).as_dict()
        oc = O.correction(so, step, hs, hb, eta, beta, normalize=normalize,
                          mode=mode)
        for k, v in c.items():
            assert v == pytest.approx(getattr(oc, k), rel=1e-12), k


def test_correction_argument_errors(lib):
    s = A.Schedule.make()
    cases = [dict(H_sel=0), dict(H_base=0), dict(step=-1),
             dict(outer_beta=1.0), dict(outer_beta=0.0),
             dict(outer_lr=float("nan")),
             dict(opts=A.default_opts(eps=0.0)),
             dict(opts=A.default_opts(mu_min=0.9, mu_max=0.5)),
             dict(opts=A.default_opts(kappa_max=0.5)),
             dict(opts=A.default_opts(mode=9)),
             dict(opts=A.default_opts(pass_=7)),
             dict(opts=A.default_opts(blocks_per_sm=-1))]
    for kw in cases:
        args = dict(schedule=s, step=4000, H_sel=150, H_base=100,
                    outer_lr=0.7, outer_beta=0.9, opts=None)
        args.update(kw)
        with pytest.raises(A.AlocoError) as ei:
            A.correction(**args)
        assert ei.value.status == A.ERR_ARG, kw
    # beta = 0 is allowed without correction (direct averaging)
    A.correction(s, 4000, 150, 100, 1.0, 0.0, A.default_opts(mode=A.CORR_NONE))


def test_sync_argument_errors_before_any_device_work(lib):
    """Validation happens before the library touches CUDA: fake addresses
    are never dereferenced."""
    s = A.Schedule.make()
    base = 1 << 40
    xs = [base + (k + 2) * (1 << 20) for k in range(4)]
    rc, _ = A.sync_ptrs(base, base + (1 << 20), xs, 1000, A.F32, 150, 100,
                        4000, s, 0.7, 0.9, raise_on_error=False)
    assert rc in (A.ERR_CUDA, A.ERR_ARG)   # no device here
    # M out of range
    rc, _ = A.sync_ptrs(base, base + 8192, [], 10, A.F32, 150, 100, 4000, s,
                        0.7, 0.9, raise_on_error=False)
    assert rc == A.ERR_ARG
    rc, _ = A.sync_ptrs(base, base + 8192, [base + 16384 * (k + 1)
                                            for k in range(33)],
                        10, A.F32, 150, 100, 4000, s, 0.7, 0.9,
                        raise_on_error=False)
    assert rc == A.ERR_ARG
    # overlapping replica and global
    rc, _ = A.sync_ptrs(base, base + (1 << 20), [base + 64], 1000, A.F32,
                        150, 100, 4000, s, 0.7, 0.9, raise_on_error=False)
    assert rc == A.ERR_ALIAS and "overlap" in A.last_error()
    # two replicas that overlap
    rc, _ = A.sync_ptrs(base, base + (1 << 20), [base + (2 << 20),
                                                 base + (2 << 20) + 400],
                        1000, A.BF16, 150, 100, 4000, s, 0.7, 0.9,
                        raise_on_error=False)
    assert rc == A.ERR_ALIAS
    # misaligned fp32 buffer
    rc, _ = A.sync_ptrs(base + 2, base + (1 << 20), [base + (2 << 20)], 1000,
                        A.F32, 150, 100, 4000, s, 0.7, 0.9,
                        raise_on_error=False)
    assert rc == A.ERR_ARG
    # bad horizons / dtype / NULL
    for kw in (dict(H_sel=0), dict(H_base=-3), dict(dtype=5)):
        a = dict(g_ptr=base, v_ptr=base + (1 << 20), x_ptrs=[base + (2 << 20)],
                 N=100, dtype=A.F32, H_sel=150, H_base=100, step=4000,
                 schedule=s, outer_lr=0.7, outer_beta=0.9,
                 raise_on_error=False)
        a.update(kw)
        rc, _ = A.sync_ptrs(**a)
        assert rc == A.ERR_ARG, kw
    rc, _ = A.sync_ptrs(0, base, [base + (2 << 20)], 100, A.F32, 150, 100,
                        4000, s, 0.7, 0.9, raise_on_error=False)
    assert rc == A.ERR_ARG


def test_pass_values_are_checked_against_the_round(lib):
    """The INT8 forms are rejected by the plain round (and its allocation-free
    entry point), the plain round's passes by the INT8 round, and the fused
    INT8 form where its worker count does not fit; all before any device
    work."""
    import ctypes
    s = A.Schedule.make()
    base = 1 << 40
    xs = [base + (k + 2) * (1 << 22) for k in range(2)]
    for p in (A.PASS_INT8_SPLIT, A.PASS_INT8_FUSED, 6, -1):
        for noalloc in (False, True):
            rc, _ = A.sync_ptrs(base, base + (1 << 22), xs, 1000, A.F32, 150,
                                100, 4000, s, 0.7, 0.9,
                                opts=A.default_opts(pass_=p), noalloc=noalloc,
                                raise_on_error=False)
            assert rc == A.ERR_ARG, (p, noalloc)
            assert "pass" in A.last_error()

    def int8(M, dtype, p):
        ptrs = (ctypes.c_void_p * M)(*[base + (k + 2) * (1 << 22)
                                       for k in range(M)])
        st = A.Stats()
        return lib.aloco_sync_int8(base, base + (1 << 22), ptrs, 1000, M,
                                   dtype, 150, 100, 4000, ctypes.byref(s),
                                   0.7, 0.9, None, 0,
                                   ctypes.byref(A.default_opts(pass_=p)),
                                   ctypes.byref(st))
    for p in (A.PASS_REGISTERS, A.PASS_BULK_COPY, A.PASS_TILE):
        assert int8(2, A.F32, p) == A.ERR_ARG
    # the fused form takes every worker count the INT8 round takes (M <= 16)
    for dt in (A.F32, A.BF16):
        assert int8(16, dt, A.PASS_INT8_FUSED) in (A.ERR_CUDA, A.ERR_ARG)
        assert "fused" not in A.last_error()
    assert int8(17, A.BF16, A.PASS_INT8_FUSED) == A.ERR_ARG
    # accepted combinations get past argument checks (no device here)
    assert int8(4, A.F32, A.PASS_INT8_FUSED) in (A.ERR_CUDA, A.ERR_ARG)
    assert "fused" not in A.last_error()


def test_empty_round_needs_no_device(lib):
    """N = 0 is a valid round: no kernel runs, the statistics are zero and
    the correction context is still reported."""
    s = A.Schedule.make()
    rc, st = A.sync_ptrs(0, 0, [0, 0], 0, A.F32, 150, 100, 4000, s, 0.7, 0.9)
    assert rc == A.OK
    d = st.as_dict()
    assert d["D"] == 0.0 and d["C"] == 0.0 and d["nonfinite"] == 0
    oc = O.correction(O.Schedule(), 4000, 150, 100, 0.7, 0.9)
    assert d["corr"]["rho"] == pytest.approx(oc.rho, rel=1e-12)


def test_int8_block_count_gives_the_papers_payload(lib):
    """Host-only block count of the library (aloco_int8_num_blocks): the
    Llama-3.1-8B parameter set moves 8.038 GB per INT8 synchronisation
    (App. G.1; one byte per element plus one FP32 scale per block), the
    same count as the oracle's; bad part lists are rejected."""
    from paper_2609_36662_gb300 import workloads as W
    parts = [n for _, n, _ in W.LLAMA31_8B.tensors()]
    nb = A.int8_num_blocks(parts)
    assert nb == O.int8_blocks(parts)
    assert round((sum(parts) + 4 * nb) / 1e9, 3) == 8.038
    assert A.int8_num_blocks([4096, 1, 4097]) == 1 + 1 + 2
    for bad in ([0], [5, -1]):
        with pytest.raises(A.AlocoError):
            A.int8_num_blocks(bad)


def test_adamw_defaults_and_argument_errors(lib):
    """Default settings are the C4 pre-training recipe (Tab. training
    settings); bad settings, NULLs and overlapping buffers are rejected
    before any device work."""
    import ctypes
    c = A.adamw_cfg()
    assert (c.lr, c.beta1, c.beta2, c.eps, c.weight_decay, c.max_grad_norm,
            c.step) == (4e-4, 0.9, 0.95, 1e-8, 0.1, 1.0, 1)
    base = 1 << 40
    MB = 1 << 20

    def call(cfg=None, N=1000, M=2, pdt=A.F32, gdt=A.F32, ptrs=None):
        cfg = cfg or A.adamw_cfg()
        p = ptrs or {k: [base + (4 * m + i) * MB for m in range(M)]
                     for i, k in enumerate(("x", "g", "m1", "m2"))}
        arr = lambda v: (ctypes.c_void_p * M)(*v)
        return lib.aloco_adamw_step(arr(p["x"]), arr(p["g"]), arr(p["m1"]),
                                    arr(p["m2"]), N, M, pdt, gdt,
                                    ctypes.byref(cfg), None, None)
    for kw in (dict(lr=-1.0), dict(beta1=1.0), dict(beta2=-0.1), dict(eps=0.0),
               dict(weight_decay=-0.1), dict(max_grad_norm=float("nan")),
               dict(step=0)):
        assert call(A.adamw_cfg(**kw)) == A.ERR_ARG, kw
    assert call(M=0) == A.ERR_ARG
    assert call(M=33) == A.ERR_ARG
    assert call(pdt=7) == A.ERR_ARG
    # a moment buffer overlapping a parameter buffer
    p = {"x": [base, base + MB], "g": [base + 2 * MB, base + 3 * MB],
         "m1": [base + 4 * MB, base + 100], "m2": [base + 6 * MB, base + 7 * MB]}
    assert call(ptrs=p) == A.ERR_ALIAS
    # a gradient overlapping an updated buffer
    p = {"x": [base, base + MB], "g": [base + 8, base + 3 * MB],
         "m1": [base + 4 * MB, base + 5 * MB], "m2": [base + 6 * MB, base + 7 * MB]}
    assert call(ptrs=p) == A.ERR_ALIAS
    # one gradient shared by both replicas passes the argument checks
    p = {"x": [base, base + MB], "g": [base + 2 * MB] * 2,
         "m1": [base + 4 * MB, base + 5 * MB], "m2": [base + 6 * MB, base + 7 * MB]}
    assert call(ptrs=p) in (A.ERR_CUDA, A.ERR_ARG)
    assert "overlap" not in A.last_error()
    # N = 0 needs no device
    assert call(N=0) == A.OK
    # given norms must be finite and non-negative
    def normed(norms):
        p = {k: [base + (4 * m + i) * MB for m in range(2)]
             for i, k in enumerate(("x", "g", "m1", "m2"))}
        arr = lambda v: (ctypes.c_void_p * 2)(*v)
        nrm = (ctypes.c_double * 2)(*norms)
        return lib.aloco_adamw_step_normed(arr(p["x"]), arr(p["g"]), arr(p["m1"]),
                                           arr(p["m2"]), 1000, 2, A.F32, A.F32,
                                           ctypes.byref(A.adamw_cfg()), nrm, None, None)
    for bad in ([1.0, float("nan")], [-1.0, 2.0], [float("inf"), 1.0]):
        assert normed(bad) == A.ERR_ARG and "grad_norms" in A.last_error()
    assert lib.aloco_adamw_step_normed(None, None, None, None, 0, 1, A.F32, A.F32,
                                       ctypes.byref(A.adamw_cfg()), None, None,
                                       None) == A.ERR_ARG


def test_binding_constants_match_the_header():
    """Every enumerator the binding mirrors has the header's value."""
    import re
    header = open(os.path.join(ROOT, "include", "aloco.h")).read()
    values = {name: int(val) for name, val in
              re.findall(r"\b(ALOCO_[A-Z0-9_]+)\s*=\s*(-?\d+)", header)}
    mirror = {
        "ALOCO_F32": A.F32, "ALOCO_BF16": A.BF16,
        "ALOCO_OK": A.OK, "ALOCO_ERR_ARG": A.ERR_ARG, "ALOCO_ERR_CUDA": A.ERR_CUDA,
        "ALOCO_ERR_NONFINITE": A.ERR_NONFINITE, "ALOCO_ERR_ALIAS": A.ERR_ALIAS,
        "ALOCO_ERR_NOMEM": A.ERR_NOMEM,
        "ALOCO_PASS_AUTO": A.PASS_AUTO, "ALOCO_PASS_REGISTERS": A.PASS_REGISTERS,
        "ALOCO_PASS_BULK_COPY": A.PASS_BULK_COPY, "ALOCO_PASS_INT8_SPLIT": A.PASS_INT8_SPLIT,
        "ALOCO_PASS_INT8_FUSED": A.PASS_INT8_FUSED, "ALOCO_PASS_TILE": A.PASS_TILE,
        "ALOCO_WAIT_SPIN": A.WAIT_SPIN, "ALOCO_WAIT_BLOCK": A.WAIT_BLOCK,
        "ALOCO_CORR_FULL": A.CORR_FULL, "ALOCO_CORR_MOMENTUM_ONLY": A.CORR_MOMENTUM_ONLY,
        "ALOCO_CORR_NONE": A.CORR_NONE,
        "ALOCO_SCHED_COSINE": A.SCHED_COSINE, "ALOCO_SCHED_CONSTANT": A.SCHED_CONSTANT,
        "ALOCO_SCHED_LINEAR": A.SCHED_LINEAR,
    }
    for name, val in mirror.items():
        assert values.get(name) == val, (name, values.get(name), val)
