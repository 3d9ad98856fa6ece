"""Plain fp64 CPU oracle for the AutoLoCo outer synchronization round.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The product library
never imports this package, and this package imports nothing from the
product.  The arithmetic lives in ``aloco_oracle.c`` (plain C, double
precision, no FMA contraction); this module compiles it with gcc and wraps
it with ctypes and numpy.

What each function follows in the paper (arxiv 2609.36662):
  * ``lr`` / ``lr_mass``  -- the inner schedule and the accumulated inner
    learning rate, Eq. app-outer-correction-lr-masses (App. B.2);
  * ``correction``       -- rho, mu_t, kappa_t, eta_out,
    Eqs. outer-correction-ratio, app-outer-step-scale,
    adjusted-outer-learning-rate (Sec. 3.2, App. B.4);
  * ``sync_round``       -- Algorithm 1 synchronisation block:
    pseudo-gradients, average, D_t and C_t
    (Eq. adaptive-h-core-diagnostics), the corrected Nesterov step
    (Eq. autoloco-corrected-nesterov) and the replica reset.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "aloco_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

SCHED_COSINE, SCHED_CONSTANT, SCHED_LINEAR = 0, 1, 2
MODE_FULL, MODE_MOMENTUM_ONLY, MODE_NONE = 0, 1, 2
F32, BF16 = 0, 1

_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so next to its source (gcc, -O2, no FP contraction)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    i64, dbl, i32 = ctypes.c_int64, ctypes.c_double, ctypes.c_int
    vp, dp = ctypes.c_void_p, ctypes.POINTER(ctypes.c_double)
    lib.orc_lr.restype = dbl
    lib.orc_lr.argtypes = [i32, dbl, dbl, i64, i64, i64]
    lib.orc_lr_mass.restype = dbl
    lib.orc_lr_mass.argtypes = [i32, dbl, dbl, i64, i64, i64, i64]
    lib.orc_correction.restype = None
    lib.orc_correction.argtypes = [i32, dbl, dbl, i64, i64, i64, i64, i64,
                                   dbl, dbl, dbl, dbl, dbl, dbl, i32, i32, dp]
    lib.orc_double_to_bf16.restype = ctypes.c_uint16
    lib.orc_double_to_bf16.argtypes = [dbl]
    lib.orc_pass1.restype = None
    lib.orc_pass1.argtypes = [vp, vp, i32, i64, i32, dp, dp]
    lib.orc_pass2.restype = i64
    lib.orc_pass2.argtypes = [vp, vp, vp, i32, i64, i32, dbl, dbl, dbl,
                              vp, vp, vp]
    lib.orc_stats.restype = None
    lib.orc_stats.argtypes = [dp, dbl, i32, dbl, dp]
    lib.orc_int8_blocks.restype = i64
    lib.orc_int8_blocks.argtypes = [vp, i32]
    lib.orc_int8_encode.restype = None
    lib.orc_int8_encode.argtypes = [vp, vp, i32, vp, vp, vp]
    lib.orc_int8_round.restype = i64
    lib.orc_int8_round.argtypes = [vp, vp, vp, i32, vp, i32, i32, dbl, dbl,
                                   dbl, vp, vp, vp, dp, dp]
    lib.orc_adamw_step.restype = None
    lib.orc_adamw_step.argtypes = [vp, i32, vp, i32, vp, vp, i64, i32, dbl,
                                   dbl, dbl, dbl, dbl, dbl, i64, vp, vp, vp,
                                   vp, dp, vp]
    _lib = lib
    return lib


@dataclass
class Schedule:
    """Inner learning-rate schedule (Tab. training settings: cosine with a
    linear warm-up).  ``total_steps`` counts the warm-up."""
    kind: int = SCHED_COSINE
    peak_lr: float = 4e-4
    final_lr: float = 4e-5
    warmup_steps: int = 1000
    total_steps: int = 20000

    def args(self):
        return (self.kind, self.peak_lr, self.final_lr, self.warmup_steps,
                self.total_steps)


@dataclass
class Correction:
    lam_sel: float
    lam_base: float
    rho_unc: float
    rho: float
    mu_t: float
    kappa_t: float
    eta_out: float
    inv_norm: float


def lr(schedule: Schedule, s: int) -> float:
    return _load().orc_lr(*schedule.args(), s)


def lr_mass(schedule: Schedule, t0: int, H: int) -> float:
    return _load().orc_lr_mass(*schedule.args(), t0, H)


def correction(schedule: Schedule, step: int, H_sel: int, H_base: int,
               outer_lr: float, outer_beta: float, mu_min=0.45, mu_max=0.90,
               kappa_max=1.6, eps=1e-8, normalize=False,
               mode=MODE_FULL) -> Correction:
    out = (ctypes.c_double * 8)()
    _load().orc_correction(*schedule.args(), step, H_sel, H_base, outer_lr,
                           outer_beta, mu_min, mu_max, kappa_max, eps,
                           int(bool(normalize)), mode, out)
    return Correction(*list(out))


def double_to_bf16_bits(x: float) -> int:
    return int(_load().orc_double_to_bf16(float(x)))


def bf16_bits_to_float(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _check_inputs(g, v, xs, dtype):
    g = np.ascontiguousarray(g, dtype=np.float32)
    v = np.ascontiguousarray(v, dtype=np.float32)
    rdt = np.float32 if dtype == F32 else np.uint16
    xs = [np.ascontiguousarray(x, dtype=rdt) for x in xs]
    N = g.shape[0]
    assert g.ndim == 1 and v.shape == (N,)
    assert all(x.shape == (N,) for x in xs)
    return g, v, xs, N


class Pass1Accumulator:
    """Running pass-1 sums over consecutive slices of one long vector; the
    summation order is that of one call over the whole vector."""

    def __init__(self, M: int):
        self.M = M
        self.E = (ctypes.c_double * M)()
        self.B = ctypes.c_double(0.0)

    def add(self, g, xs, dtype):
        g, _, xs, N = _check_inputs(g, np.zeros_like(g), xs, dtype)
        assert len(xs) == self.M
        ptrs = (ctypes.c_void_p * self.M)(*[_ptr(x) for x in xs])
        _load().orc_pass1(_ptr(g), ptrs, dtype, N, self.M, self.E,
                          ctypes.byref(self.B))

    def stats(self, eps: float):
        out = (ctypes.c_double * 2)()
        _load().orc_stats(self.E, self.B.value, self.M, eps, out)
        return {"D": out[0], "C": out[1], "mean_sq_norm": self.B.value,
                "drift": list(self.E)}


def pass2(g, v, xs, dtype, mu_t, eta_out, inv_norm, want_replicas=True):
    """Elementwise update of a (slice of the) vector; returns
    (g_out float64, v_out float64, [x_out per replica] or None, nonfinite)."""
    g, v, xs, N = _check_inputs(g, v, xs, dtype)
    M = len(xs)
    g_out = np.empty(N, np.float64)
    v_out = np.empty(N, np.float64)
    rdt = np.float32 if dtype == F32 else np.uint16
    x_out = [np.empty(N, rdt) for _ in range(M)] if want_replicas else None
    ptrs = (ctypes.c_void_p * M)(*[_ptr(x) for x in xs])
    optrs = (ctypes.c_void_p * M)(*([_ptr(x) for x in x_out]
                                    if want_replicas else [None] * M))
    nf = _load().orc_pass2(_ptr(g), _ptr(v), ptrs, dtype, N, M, mu_t,
                           eta_out, inv_norm, _ptr(g_out), _ptr(v_out), optrs)
    return g_out, v_out, x_out, int(nf)


def sync_round(g, v, xs, dtype, schedule: Schedule, step: int, H_sel: int,
               H_base: int, outer_lr: float, outer_beta: float, mu_min=0.45,
               mu_max=0.90, kappa_max=1.6, eps=1e-8, normalize=False,
               mode=MODE_FULL):
    """One outer synchronisation round over whole vectors (Algorithm 1).

    g, v: float32 [N]; xs: M arrays of float32, or of bf16 bit patterns
    (uint16) when dtype == BF16.  Returns a dict with the updated global
    weights and momentum (float64, unrounded), the reset replicas (in their
    storage type), the statistics and the correction context."""
    corr = correction(schedule, step, H_sel, H_base, outer_lr, outer_beta,
                      mu_min, mu_max, kappa_max, eps, normalize, mode)
    acc = Pass1Accumulator(len(xs))
    acc.add(g, xs, dtype)
    st = acc.stats(eps)
    g_out, v_out, x_out, nf = pass2(g, v, xs, dtype, corr.mu_t, corr.eta_out,
                                    corr.inv_norm)
    st.update(g=g_out, v=v_out, x=x_out, nonfinite=nf, corr=corr)
    return st


# ------------------------------------------------ INT8 communication (App. G.1)

INT8_BLOCK = 4096


def _parts(parts, N):
    p = np.ascontiguousarray([N] if parts is None else parts, dtype=np.int64)
    assert int(p.sum()) == N, "parts must add up to the vector length"
    return p


def int8_blocks(parts) -> int:
    p = np.ascontiguousarray(parts, dtype=np.int64)
    return int(_load().orc_int8_blocks(_ptr(p), len(p)))


def int8_payload_bytes(parts) -> int:
    """Logical bytes one worker sends per sync: one int8 per element and one
    fp32 scale per block."""
    return int(np.sum(parts)) + 4 * int8_blocks(parts)


def int8_encode(y, parts=None):
    """Blockwise INT8 codec of an fp32 vector: (codes int8, scales float32
    per block, decoded float32)."""
    y = np.ascontiguousarray(y, dtype=np.float32)
    p = _parts(parts, y.shape[0])
    nb = int8_blocks(p)
    codes = np.empty(y.shape[0], np.int8)
    scales = np.empty(nb, np.float32)
    dec = np.empty(y.shape[0], np.float32)
    _load().orc_int8_encode(_ptr(y), _ptr(p), len(p), _ptr(codes),
                            _ptr(scales), _ptr(dec))
    return codes, scales, dec


def int8_round(g, v, xs, dtype, parts, mu_t, eta_out, inv_norm, eps=1e-8):
    """The outer round with INT8-communicated pseudo-gradients: D from the
    pre-quantisation pseudo-gradients, C from the decoded aggregate."""
    g, v, xs, N = _check_inputs(g, v, xs, dtype)
    p = _parts(parts, N)
    M = len(xs)
    g_out = np.empty(N, np.float64)
    v_out = np.empty(N, np.float64)
    rdt = np.float32 if dtype == F32 else np.uint16
    x_out = [np.empty(N, rdt) for _ in range(M)]
    E = (ctypes.c_double * M)()
    B = ctypes.c_double(0.0)
    ptrs = (ctypes.c_void_p * M)(*[_ptr(x) for x in xs])
    optrs = (ctypes.c_void_p * M)(*[_ptr(x) for x in x_out])
    nf = _load().orc_int8_round(_ptr(g), _ptr(v), ptrs, dtype, _ptr(p),
                                len(p), M, mu_t, eta_out, inv_norm,
                                _ptr(g_out), _ptr(v_out), optrs, E,
                                ctypes.byref(B))
    out = (ctypes.c_double * 2)()
    _load().orc_stats(E, B.value, M, eps, out)
    return {"D": out[0], "C": out[1], "mean_sq_norm": B.value,
            "drift": list(E), "g": g_out, "v": v_out, "x": x_out,
            "nonfinite": int(nf)}


# ------------------------------------------------ inner AdamW step (Sec. 2)

def adamw_step(xs, x_dtype, grads, g_dtype, m1s, m2s, lr, beta1, beta2, eps,
               weight_decay, max_norm, step, norms=None):
    """One AdamW step (decoupled weight decay, per-replica gradient-norm
    clipping) on each replica.  xs / grads: float32 arrays, or bf16 bit
    patterns (uint16) for dtype BF16; m1s, m2s: float32.  norms (optional):
    the gradients' norms over their whole replicas, for a slice.  Returns the
    unrounded float64 results, x' in its storage type and the pre-clipping
    gradient norms."""
    M = len(xs)
    xdt = np.float32 if x_dtype == F32 else np.uint16
    gdt = np.float32 if g_dtype == F32 else np.uint16
    xs = [np.ascontiguousarray(a, dtype=xdt) for a in xs]
    grads = [np.ascontiguousarray(a, dtype=gdt) for a in grads]
    m1s = [np.ascontiguousarray(a, dtype=np.float32) for a in m1s]
    m2s = [np.ascontiguousarray(a, dtype=np.float32) for a in m2s]
    N = xs[0].shape[0]
    for a in xs + grads + m1s + m2s:
        assert a.shape == (N,)
    x_out = [np.empty(N, np.float64) for _ in range(M)]
    m1_out = [np.empty(N, np.float64) for _ in range(M)]
    m2_out = [np.empty(N, np.float64) for _ in range(M)]
    x_store = [np.empty(N, xdt) for _ in range(M)]
    out_norms = (ctypes.c_double * M)()
    given = None if norms is None else (ctypes.c_double * M)(*[float(x) for x in norms])

    def arr(lst):
        return (ctypes.c_void_p * M)(*[_ptr(a) for a in lst])
    _load().orc_adamw_step(arr(xs), x_dtype, arr(grads), g_dtype, arr(m1s),
                           arr(m2s), N, M, lr, beta1, beta2, eps,
                           weight_decay, max_norm, step, arr(x_out),
                           arr(m1_out), arr(m2_out), arr(x_store), out_norms,
                           given)
    return {"x": x_out, "m1": m1_out, "m2": m2_out, "x_store": x_store,
            "norms": list(out_norms)}
