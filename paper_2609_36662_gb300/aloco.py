"""ctypes binding of libaloco (include/aloco.h).

Argument marshalling only: every step of the round runs inside the
library's CUDA kernels.  If the compiled library is missing this module
raises on first use; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional, Sequence

MAX_WORKERS = 32

F32, BF16 = 0, 1
SCHED_COSINE, SCHED_CONSTANT, SCHED_LINEAR = 0, 1, 2
CORR_FULL, CORR_MOMENTUM_ONLY, CORR_NONE = 0, 1, 2
PASS_AUTO, PASS_REGISTERS, PASS_BULK_COPY = 0, 1, 2
PASS_INT8_SPLIT, PASS_INT8_FUSED = 3, 4
PASS_TILE = 5
WAIT_SPIN, WAIT_BLOCK = 0, 1

OK = 0
ERR_ARG = -1
ERR_CUDA = -2
ERR_NONFINITE = -3
ERR_ALIAS = -4
ERR_NOMEM = -5

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                         "libaloco.so")

# Names declared in include/aloco.h (checked by the ABI test).
EXPORTS = ("aloco_default_opts", "aloco_inner_lr_accum", "aloco_correction",
           "aloco_sync", "aloco_sync_ex", "aloco_sync_noalloc", "aloco_sync_host",
           "aloco_sync_shard", "aloco_sync_int8_shard", "aloco_combine_partials",
           "aloco_sync_int8", "aloco_int8_num_blocks", "aloco_int8_encode",
           "aloco_int8_decode", "aloco_adamw_default_cfg", "aloco_adamw_step",
           "aloco_adamw_step_normed",
           "aloco_ctrl_default_cfg", "aloco_ctrl_init", "aloco_select_interval",
           "aloco_ctrl_state_bytes", "aloco_ctrl_save", "aloco_ctrl_load",
           "aloco_test_stall_tile", "aloco_last_error", "aloco_shutdown",
           "aloco_version")

CTRL_HISTORY = 16
ASSESS_NONE, ASSESS_SUPPORTED, ASSESS_CONSISTENT, ASSESS_MODERATE, \
    ASSESS_SEVERE, ASSESS_INVALID = range(6)
PHASE_WARMUP, PHASE_REFERENCE, PHASE_VARIABILITY, PHASE_MONITOR, \
    PHASE_CANDIDATE, PHASE_CONFIRM = range(6)


class Schedule(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("peak_lr", ctypes.c_double), ("final_lr", ctypes.c_double),
                ("warmup_steps", ctypes.c_int64),
                ("total_steps", ctypes.c_int64)]

    @classmethod
    def make(cls, kind=SCHED_COSINE, peak_lr=4e-4, final_lr=4e-5,
             warmup_steps=1000, total_steps=20000):
        return cls(kind, 0, peak_lr, final_lr, warmup_steps, total_steps)


class Opts(ctypes.Structure):
    _fields_ = [("mu_min", ctypes.c_double), ("mu_max", ctypes.c_double),
                ("kappa_max", ctypes.c_double), ("eps", ctypes.c_double),
                ("normalize", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("time_kernel", ctypes.c_int32),
                ("blocks_per_sm", ctypes.c_int32),
                ("stream", ctypes.c_void_p), ("pass_", ctypes.c_int32),
                ("wait", ctypes.c_int32)]


class AdamwCfg(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("beta1", ctypes.c_double),
                ("beta2", ctypes.c_double), ("eps", ctypes.c_double),
                ("weight_decay", ctypes.c_double),
                ("max_grad_norm", ctypes.c_double), ("step", ctypes.c_int64)]


class AdamwStats(ctypes.Structure):
    _fields_ = [("grad_norm", ctypes.c_double * MAX_WORKERS),
                ("clip", ctypes.c_double * MAX_WORKERS),
                ("M", ctypes.c_int32), ("grid", ctypes.c_int32),
                ("kernel_ms", ctypes.c_float), ("reserved", ctypes.c_int32)]

    def as_dict(self):
        return {"grad_norm": list(self.grad_norm[:self.M]),
                "clip": list(self.clip[:self.M]), "M": self.M,
                "grid": self.grid, "kernel_ms": self.kernel_ms}


class Correction(ctypes.Structure):
    _fields_ = [(n, ctypes.c_double) for n in
                ("lam_sel", "lam_base", "rho_unc", "rho", "mu_t", "kappa_t",
                 "eta_out", "inv_norm")]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class Stats(ctypes.Structure):
    _fields_ = [("D", ctypes.c_double), ("C", ctypes.c_double),
                ("mean_sq_norm", ctypes.c_double),
                ("drift", ctypes.c_double * MAX_WORKERS),
                ("corr", Correction), ("nonfinite", ctypes.c_int64),
                ("M", ctypes.c_int32), ("grid", ctypes.c_int32),
                ("kernel_ms", ctypes.c_float), ("pass_used", ctypes.c_int32)]

    def as_dict(self):
        return {"D": self.D, "C": self.C, "mean_sq_norm": self.mean_sq_norm,
                "drift": list(self.drift[:self.M]),
                "corr": self.corr.as_dict(), "nonfinite": self.nonfinite,
                "M": self.M, "grid": self.grid, "kernel_ms": self.kernel_ms,
                "pass_used": self.pass_used}


class Partials(ctypes.Structure):
    """aloco_partials_t: one shard's partial sums of a round."""
    _fields_ = [("drift", ctypes.c_double * MAX_WORKERS),
                ("sum_sq", ctypes.c_double), ("sq_scale", ctypes.c_double),
                ("eps", ctypes.c_double), ("corr", Correction),
                ("nonfinite", ctypes.c_int64), ("n", ctypes.c_int64),
                ("M", ctypes.c_int32), ("pass_used", ctypes.c_int32),
                ("kernel_ms", ctypes.c_float), ("reserved", ctypes.c_int32)]

    def to_bytes(self) -> bytes:
        return ctypes.string_at(ctypes.addressof(self), ctypes.sizeof(self))

    @classmethod
    def from_bytes(cls, blob: bytes) -> "Partials":
        if len(blob) != ctypes.sizeof(cls):
            raise ValueError(f"partials blob of {len(blob)} bytes, want "
                             f"{ctypes.sizeof(cls)}")
        return cls.from_buffer_copy(blob)


_i64, _i32, _dbl = ctypes.c_int64, ctypes.c_int32, ctypes.c_double


class CtrlCfg(ctypes.Structure):
    _fields_ = [("H_base", _i64), ("H_min", _i64), ("H_max", _i64),
                ("q_H", _i64), ("warmup_steps", _i64), ("beta_tok", _dbl),
                ("thr_candidate", _dbl), ("thr_moderate", _dbl),
                ("thr_severe", _dbl), ("exposure_mult", _dbl),
                ("div_moderate", _dbl), ("div_severe", _dbl),
                ("retire_frac", _dbl), ("ref_ema", _dbl), ("mad_scale", _dbl),
                ("scale_floor", _dbl), ("eps", _dbl),
                ("mapper_bootstrap", _i32), ("ref_bootstrap", _i32),
                ("variability_intervals", _i32), ("severe_fallback", _i32)]


class CtrlState(ctypes.Structure):
    _fields_ = [("version", _i32), ("phase", _i32), ("intervals", _i64),
                ("H_acc", _i64), ("H_next", _i64), ("H_cand", _i64),
                ("bound", _i64), ("bound_lam", _dbl), ("phase_count", _i32),
                ("ref_needed", _i32), ("moderate_run", _i32),
                ("severe_run", _i32), ("log_D_ref", _dbl),
                ("log_C_ref", _dbl), ("lam_ref", _dbl), ("sum_log_D", _dbl),
                ("sum_log_C", _dbl), ("n_hist", _i32), ("head", _i32),
                ("hist_D", _dbl * CTRL_HISTORY),
                ("hist_C", _dbl * CTRL_HISTORY), ("mapper_n", _i32),
                ("calibrated", _i32), ("mapper_mass", _dbl * 8),
                ("M_base", _dbl), ("n_hat", _dbl), ("last_z", _dbl),
                ("last_r_D", _dbl), ("last_r_C", _dbl),
                ("last_assessment", _i32), ("referenced", _i32)]


class IntervalObs(ctypes.Structure):
    _fields_ = [("D", _dbl), ("C", _dbl), ("lam", _dbl), ("tokens", _dbl),
                ("H_step", _i64), ("step_end", _i64)]


class CtrlDecision(ctypes.Structure):
    _fields_ = [("H_tok", _i64), ("H_step", _i64), ("H_ref_step", _i64),
                ("assessment", _i32), ("phase", _i32), ("z", _dbl),
                ("r_D", _dbl), ("r_C", _dbl)]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class AlocoError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"aloco status {status}: {message}")
        self.status = status


_lib = None


def library_path() -> str:
    return _LIB_PATH


def load():
    """Load libaloco.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise ImportError(
            f"{_LIB_PATH} is missing: build it with "
            "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(_LIB_PATH)
    vp, i64, i32, dbl = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, \
        ctypes.c_double
    lib.aloco_default_opts.argtypes = [ctypes.POINTER(Opts)]
    lib.aloco_default_opts.restype = None
    lib.aloco_inner_lr_accum.argtypes = [ctypes.POINTER(Schedule), i64, i64]
    lib.aloco_inner_lr_accum.restype = dbl
    lib.aloco_correction.argtypes = [ctypes.POINTER(Schedule), i64, i64, i64,
                                     dbl, dbl, ctypes.POINTER(Opts),
                                     ctypes.POINTER(Correction)]
    lib.aloco_correction.restype = i32
    sync_args = [vp, vp, ctypes.POINTER(vp), ctypes.c_size_t, i32, i32, i64,
                 i64, i64, ctypes.POINTER(Schedule), dbl, dbl]
    lib.aloco_sync.argtypes = sync_args + [ctypes.POINTER(Stats)]
    lib.aloco_sync.restype = i32
    lib.aloco_sync_ex.argtypes = sync_args + [ctypes.POINTER(Opts),
                                              ctypes.POINTER(Stats)]
    lib.aloco_sync_ex.restype = i32
    lib.aloco_sync_noalloc.argtypes = sync_args + [ctypes.POINTER(Opts),
                                                   ctypes.POINTER(Stats)]
    lib.aloco_sync_noalloc.restype = i32
    P = ctypes.POINTER
    lib.aloco_sync_int8.argtypes = sync_args + [vp, i32, P(Opts), P(Stats)]
    lib.aloco_sync_int8.restype = i32
    lib.aloco_adamw_default_cfg.argtypes = [P(AdamwCfg)]
    lib.aloco_adamw_default_cfg.restype = None
    lib.aloco_adamw_step.argtypes = [vp, vp, vp, vp, ctypes.c_size_t, i32,
                                     i32, i32, P(AdamwCfg), P(Opts),
                                     P(AdamwStats)]
    lib.aloco_adamw_step.restype = i32
    lib.aloco_adamw_step_normed.argtypes = [vp, vp, vp, vp, ctypes.c_size_t, i32,
                                            i32, i32, P(AdamwCfg), vp, P(Opts),
                                            P(AdamwStats)]
    lib.aloco_adamw_step_normed.restype = i32
    lib.aloco_sync_host.argtypes = sync_args + [ctypes.c_size_t, P(Opts), P(Stats)]
    lib.aloco_sync_host.restype = i32
    lib.aloco_sync_shard.argtypes = sync_args + [P(Opts), P(Partials)]
    lib.aloco_sync_shard.restype = i32
    lib.aloco_sync_int8_shard.argtypes = sync_args + [vp, i32, P(Opts), P(Partials)]
    lib.aloco_sync_int8_shard.restype = i32
    lib.aloco_combine_partials.argtypes = [vp, i32, P(Stats)]
    lib.aloco_combine_partials.restype = i32
    lib.aloco_test_stall_tile.argtypes = [i64]
    lib.aloco_test_stall_tile.restype = None
    lib.aloco_int8_num_blocks.argtypes = [vp, i32]
    lib.aloco_int8_num_blocks.restype = i64
    lib.aloco_int8_encode.argtypes = [vp, ctypes.c_size_t, vp, i32, vp, vp, vp,
                                      vp]
    lib.aloco_int8_encode.restype = i32
    lib.aloco_int8_decode.argtypes = [vp, vp, ctypes.c_size_t, vp, i32, vp, vp]
    lib.aloco_int8_decode.restype = i32
    lib.aloco_ctrl_default_cfg.argtypes = [P(CtrlCfg), i64, i64, i64, i64,
                                           i64]
    lib.aloco_ctrl_default_cfg.restype = None
    lib.aloco_ctrl_init.argtypes = [P(CtrlState), P(CtrlCfg),
                                    P(CtrlDecision)]
    lib.aloco_ctrl_init.restype = i32
    lib.aloco_select_interval.argtypes = [P(CtrlState), P(CtrlCfg),
                                          P(IntervalObs), P(Schedule),
                                          P(CtrlDecision)]
    lib.aloco_select_interval.restype = i32
    lib.aloco_ctrl_state_bytes.argtypes = []
    lib.aloco_ctrl_state_bytes.restype = ctypes.c_size_t
    lib.aloco_ctrl_save.argtypes = [P(CtrlState), vp, ctypes.c_size_t]
    lib.aloco_ctrl_save.restype = i32
    lib.aloco_ctrl_load.argtypes = [P(CtrlState), vp, ctypes.c_size_t]
    lib.aloco_ctrl_load.restype = i32
    lib.aloco_last_error.argtypes = []
    lib.aloco_last_error.restype = ctypes.c_char_p
    lib.aloco_shutdown.argtypes = []
    lib.aloco_shutdown.restype = None
    lib.aloco_version.argtypes = []
    lib.aloco_version.restype = i32
    _lib = lib
    return lib


def last_error() -> str:
    return load().aloco_last_error().decode()


def default_opts(**kw) -> Opts:
    o = Opts()
    load().aloco_default_opts(ctypes.byref(o))
    for k, val in kw.items():
        setattr(o, k, val)
    return o


def inner_lr_accum(schedule: Schedule, t0: int, H: int) -> float:
    return load().aloco_inner_lr_accum(ctypes.byref(schedule), t0, H)


def correction(schedule: Schedule, step: int, H_sel: int, H_base: int,
               outer_lr: float, outer_beta: float,
               opts: Optional[Opts] = None) -> Correction:
    out = Correction()
    rc = load().aloco_correction(ctypes.byref(schedule), step, H_sel, H_base,
                                 outer_lr, outer_beta,
                                 ctypes.byref(opts) if opts else None,
                                 ctypes.byref(out))
    if rc != OK:
        raise AlocoError(rc, last_error())
    return out


def sync_ptrs(g_ptr: int, v_ptr: int, x_ptrs: Sequence[int], N: int,
              dtype: int, H_sel: int, H_base: int, step: int,
              schedule: Schedule, outer_lr: float, outer_beta: float,
              opts: Optional[Opts] = None, raise_on_error: bool = True,
              noalloc: bool = False):
    """aloco_sync_ex (or, with noalloc=True, aloco_sync_noalloc) on raw
    device addresses.  Returns (status, Stats)."""
    M = len(x_ptrs)
    arr = (ctypes.c_void_p * max(M, 1))(*x_ptrs)
    st = Stats()
    fn = load().aloco_sync_noalloc if noalloc else load().aloco_sync_ex
    rc = fn(g_ptr, v_ptr, arr, N, M, dtype, H_sel, H_base,
                              step, ctypes.byref(schedule), outer_lr,
                              outer_beta,
                              ctypes.byref(opts) if opts is not None else None,
                              ctypes.byref(st))
    if raise_on_error and rc not in (OK, ERR_NONFINITE):
        raise AlocoError(rc, last_error())
    return rc, st


def sync(global_, momentum, locals_, *, H_sel: int, H_base: int, step: int,
         schedule: Schedule, outer_lr: float, outer_beta: float,
         opts: Optional[Opts] = None, stream=None, raise_on_error=True,
         noalloc: bool = False):
    """One outer synchronisation round on torch CUDA tensors, in place.

    global_, momentum: contiguous float32 [N]; locals_: M contiguous tensors
    [N] of float32 or bfloat16.  The round runs on `stream` (default: the
    current torch stream).  noalloc=True calls aloco_sync_noalloc, the entry
    point that allocates nothing (its scratch is a static device array)."""
    import torch
    if global_.dtype != torch.float32 or momentum.dtype != torch.float32:
        raise TypeError("global and momentum must be float32")
    N = global_.numel()
    if momentum.numel() != N or any(x.numel() != N for x in locals_):
        raise ValueError("all buffers must have the same number of elements")
    if not locals_:
        raise ValueError("need at least one replica")
    rdt = locals_[0].dtype
    if any(x.dtype != rdt for x in locals_):
        raise TypeError("replicas must share one dtype")
    if rdt == torch.float32:
        dtype = F32
    elif rdt == torch.bfloat16:
        dtype = BF16
    else:
        raise TypeError(f"unsupported replica dtype {rdt}")
    for t in (global_, momentum, *locals_):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("buffers must be contiguous CUDA tensors")
    if opts is None:
        opts = default_opts()
    s = stream if stream is not None else torch.cuda.current_stream(
        global_.device)
    opts.stream = s.cuda_stream
    with torch.cuda.device(global_.device):
        rc, st = sync_ptrs(global_.data_ptr(), momentum.data_ptr(),
                           [x.data_ptr() for x in locals_], N, dtype, H_sel,
                           H_base, step, schedule, outer_lr, outer_beta, opts,
                           raise_on_error, noalloc)
    return st.as_dict() | {"status": rc}


def shutdown():
    if _lib is not None:
        _lib.aloco_shutdown()


# ------------------------------------------------------------ sharded rounds

def _replica_dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported replica dtype {t.dtype}")


def sync_shard(global_, momentum, locals_, *, H_sel: int, H_base: int,
               step: int, schedule: Schedule, outer_lr: float,
               outer_beta: float, opts: Optional[Opts] = None, stream=None,
               raise_on_error=True, parts=None, int8: bool = False):
    """One shard of a round on torch CUDA tensors (views of the shard's
    elements), in place: aloco_sync_shard, or aloco_sync_int8_shard with
    int8=True (parts: the shard's tensor parts).  Returns (status,
    Partials)."""
    import torch
    N = global_.numel()
    if momentum.numel() != N or any(x.numel() != N for x in locals_):
        raise ValueError("all buffers must have the same number of elements")
    for t in (global_, momentum, *locals_):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("buffers must be contiguous CUDA tensors")
    dtype = _replica_dtype_code(locals_[0])
    if opts is None:
        opts = default_opts()
    s = stream if stream is not None else torch.cuda.current_stream(
        global_.device)
    opts.stream = s.cuda_stream
    M = len(locals_)
    ptrs = (ctypes.c_void_p * M)(*[x.data_ptr() for x in locals_])
    out = Partials()
    with torch.cuda.device(global_.device):
        if int8:
            arr, n = _parts_array(parts)
            rc = load().aloco_sync_int8_shard(
                global_.data_ptr(), momentum.data_ptr(), ptrs, N, M, dtype,
                H_sel, H_base, step, ctypes.byref(schedule), outer_lr,
                outer_beta, arr, n, ctypes.byref(opts), ctypes.byref(out))
        else:
            rc = load().aloco_sync_shard(
                global_.data_ptr(), momentum.data_ptr(), ptrs, N, M, dtype,
                H_sel, H_base, step, ctypes.byref(schedule), outer_lr,
                outer_beta, ctypes.byref(opts), ctypes.byref(out))
    if raise_on_error and rc not in (OK, ERR_NONFINITE):
        raise AlocoError(rc, last_error())
    return rc, out


def combine_partials(shards: Sequence[Partials], raise_on_error=True):
    """aloco_combine_partials over the shards in the given order (host
    only).  Returns the statistics dict with "status"."""
    n = len(shards)
    arr = (Partials * max(n, 1))(*shards)
    st = Stats()
    rc = load().aloco_combine_partials(arr if n else None, n,
                                       ctypes.byref(st))
    if raise_on_error and rc not in (OK, ERR_NONFINITE):
        raise AlocoError(rc, last_error())
    return st.as_dict() | {"status": rc}


class Controller:
    """The host interval controller (aloco_select_interval) with its state
    and settings."""

    def __init__(self, H_base: int, H_min: int, H_max: int, q_H: int,
                 warmup_steps: int, schedule: Schedule, **overrides):
        lib = load()
        self.cfg = CtrlCfg()
        lib.aloco_ctrl_default_cfg(ctypes.byref(self.cfg), H_base, H_min,
                                   H_max, q_H, warmup_steps)
        for k, val in overrides.items():
            setattr(self.cfg, k, val)
        self.schedule = schedule
        self.state = CtrlState()
        d = CtrlDecision()
        rc = lib.aloco_ctrl_init(ctypes.byref(self.state),
                                 ctypes.byref(self.cfg), ctypes.byref(d))
        if rc != OK:
            raise AlocoError(rc, last_error())
        self.decision = d

    def observe(self, D: float, C: float, lam: float, tokens: float,
                H_step: int, step_end: int) -> CtrlDecision:
        obs = IntervalObs(D, C, lam, tokens, H_step, step_end)
        d = CtrlDecision()
        rc = load().aloco_select_interval(
            ctypes.byref(self.state), ctypes.byref(self.cfg),
            ctypes.byref(obs), ctypes.byref(self.schedule), ctypes.byref(d))
        if rc != OK:
            raise AlocoError(rc, last_error())
        self.decision = d
        return d

    def save(self) -> bytes:
        n = load().aloco_ctrl_state_bytes()
        buf = ctypes.create_string_buffer(n)
        rc = load().aloco_ctrl_save(ctypes.byref(self.state), buf, n)
        if rc != OK:
            raise AlocoError(rc, last_error())
        return buf.raw

    def load_state(self, blob: bytes):
        buf = ctypes.create_string_buffer(blob, len(blob))
        rc = load().aloco_ctrl_load(ctypes.byref(self.state), buf, len(blob))
        if rc != OK:
            raise AlocoError(rc, last_error())


# ------------------------------------------------ INT8 communication (App. G.1)

def _parts_array(parts):
    if parts is None:
        return None, 0
    arr = (ctypes.c_int64 * len(parts))(*[int(p) for p in parts])
    return arr, len(parts)


def int8_num_blocks(parts) -> int:
    arr, n = _parts_array(parts)
    nb = load().aloco_int8_num_blocks(arr, n)
    if nb < 0:
        raise AlocoError(ERR_ARG, last_error())
    return nb


def int8_payload_bytes(parts) -> int:
    """Bytes one worker sends per sync: the codes plus one fp32 scale per
    block."""
    return int(sum(parts)) + 4 * int8_num_blocks(parts)


def int8_encode(x, parts=None, want_decoded=True, stream=None):
    """Blockwise INT8 codec of a contiguous float32 CUDA tensor; returns
    (codes int8, scales float32, decoded float32 or None)."""
    import torch
    if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous():
        raise TypeError("x must be a contiguous float32 CUDA tensor")
    N = x.numel()
    nb = int8_num_blocks(parts if parts is not None else [N])
    codes = torch.empty(N, dtype=torch.int8, device=x.device)
    scales = torch.empty(nb, dtype=torch.float32, device=x.device)
    dec = torch.empty_like(x) if want_decoded else None
    s = stream if stream is not None else torch.cuda.current_stream(x.device)
    arr, n = _parts_array(parts)
    with torch.cuda.device(x.device):
        rc = load().aloco_int8_encode(x.data_ptr(), N, arr, n,
                                      codes.data_ptr(), scales.data_ptr(),
                                      dec.data_ptr() if dec is not None
                                      else None, s.cuda_stream)
    if rc != OK:
        raise AlocoError(rc, last_error())
    return codes, scales, dec


def int8_decode(codes, scales, parts=None, stream=None):
    import torch
    N = codes.numel()
    out = torch.empty(N, dtype=torch.float32, device=codes.device)
    s = stream if stream is not None else torch.cuda.current_stream(
        codes.device)
    arr, n = _parts_array(parts)
    with torch.cuda.device(codes.device):
        rc = load().aloco_int8_decode(codes.data_ptr(), scales.data_ptr(), N,
                                      arr, n, out.data_ptr(), s.cuda_stream)
    if rc != OK:
        raise AlocoError(rc, last_error())
    return out


def sync_host(global_, momentum, locals_, *, H_sel: int, H_base: int,
              step: int, schedule: Schedule, outer_lr: float,
              outer_beta: float, chunk_elems: int = 0,
              opts: Optional[Opts] = None, stream=None, raise_on_error=True):
    """aloco_sync_host on page-locked torch CPU tensors (theta, v updated in
    place; the replicas are read only)."""
    import torch
    N = global_.numel()
    dtype = F32 if locals_[0].dtype == torch.float32 else BF16
    if opts is None:
        opts = default_opts()
    s = stream if stream is not None else torch.cuda.current_stream()
    opts.stream = s.cuda_stream
    M = len(locals_)
    ptrs = (ctypes.c_void_p * M)(*[x.data_ptr() for x in locals_])
    st = Stats()
    rc = load().aloco_sync_host(global_.data_ptr(), momentum.data_ptr(), ptrs, N,
                                M, dtype, H_sel, H_base, step,
                                ctypes.byref(schedule), outer_lr, outer_beta,
                                chunk_elems, ctypes.byref(opts), ctypes.byref(st))
    if raise_on_error and rc not in (OK, ERR_NONFINITE):
        raise AlocoError(rc, last_error())
    return st.as_dict() | {"status": rc}


def sync_int8(global_, momentum, locals_, *, parts=None, H_sel: int,
              H_base: int, step: int, schedule: Schedule, outer_lr: float,
              outer_beta: float, opts: Optional[Opts] = None, stream=None,
              raise_on_error=True):
    """One outer round with INT8-communicated pseudo-gradients (in place on
    torch CUDA tensors, like sync())."""
    import torch
    N = global_.numel()
    rdt = locals_[0].dtype
    dtype = F32 if rdt == torch.float32 else BF16
    if opts is None:
        opts = default_opts()
    s = stream if stream is not None else torch.cuda.current_stream(
        global_.device)
    opts.stream = s.cuda_stream
    M = len(locals_)
    ptrs = (ctypes.c_void_p * M)(*[x.data_ptr() for x in locals_])
    arr, n = _parts_array(parts)
    st = Stats()
    with torch.cuda.device(global_.device):
        rc = load().aloco_sync_int8(global_.data_ptr(), momentum.data_ptr(),
                                    ptrs, N, M, dtype, H_sel, H_base, step,
                                    ctypes.byref(schedule), outer_lr,
                                    outer_beta, arr, n, ctypes.byref(opts),
                                    ctypes.byref(st))
    if raise_on_error and rc not in (OK, ERR_NONFINITE):
        raise AlocoError(rc, last_error())
    return st.as_dict() | {"status": rc}


# ----------------------------------------------------- inner AdamW (Sec. 2)

def adamw_cfg(**kw) -> AdamwCfg:
    """The library's default AdamW settings (C4 pre-training) with the given
    fields replaced."""
    c = AdamwCfg()
    load().aloco_adamw_default_cfg(ctypes.byref(c))
    for k, v in kw.items():
        if not hasattr(c, k):
            raise TypeError(f"unknown AdamW setting {k!r}")
        setattr(c, k, v)
    return c


def adamw_step(params, grads, exp_avg, exp_avg_sq, cfg: AdamwCfg,
               opts: Optional[Opts] = None, stream=None, want_stats=True,
               raise_on_error=True, grad_norms=None):
    """One AdamW step on every replica, in place (lists of torch CUDA tensors
    of one device: params and grads fp32 or bf16, moments fp32).  With
    grad_norms (M floats, the gradients' norms) the step takes them instead
    of computing them (aloco_adamw_step_normed).  Returns the per-replica
    gradient norms and clipping factors (want_stats), else None without
    waiting for the GPU."""
    import torch
    M = len(params)
    if not (len(grads) == len(exp_avg) == len(exp_avg_sq) == M):
        raise ValueError("params, grads and moments need one tensor per replica")
    N = params[0].numel()
    pdt = F32 if params[0].dtype == torch.float32 else BF16
    gdt = F32 if grads[0].dtype == torch.float32 else BF16
    if opts is None:
        opts = default_opts()
    s = stream if stream is not None else torch.cuda.current_stream(
        params[0].device)
    opts.stream = s.cuda_stream

    def arr(ts):
        return (ctypes.c_void_p * M)(*[t.data_ptr() for t in ts])
    st = AdamwStats() if want_stats else None
    with torch.cuda.device(params[0].device):
        if grad_norms is None:
            rc = load().aloco_adamw_step(arr(params), arr(grads), arr(exp_avg),
                                         arr(exp_avg_sq), N, M, pdt, gdt,
                                         ctypes.byref(cfg), ctypes.byref(opts),
                                         ctypes.byref(st) if st is not None else None)
        else:
            norms = (ctypes.c_double * M)(*[float(x) for x in grad_norms])
            rc = load().aloco_adamw_step_normed(
                arr(params), arr(grads), arr(exp_avg), arr(exp_avg_sq), N, M, pdt,
                gdt, ctypes.byref(cfg), norms, ctypes.byref(opts),
                ctypes.byref(st) if st is not None else None)
    if raise_on_error and rc != OK:
        raise AlocoError(rc, last_error())
    if st is None:
        return rc if not raise_on_error else None
    return st.as_dict() | {"status": rc}


def test_stall_tile(tile: int):
    """Testing only: the next bulk-copy round on this thread skips the copies
    of one tile, so that its bounded wait runs out (aloco_test_stall_tile)."""
    load().aloco_test_stall_tile(int(tile))
