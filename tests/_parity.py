"""Helpers shared by the parity tests: run the CUDA path and the oracle on the
same seeded inputs and compare them.

Tolerances (written here, used by every parity test):
  * theta' and v' (fp32 on the GPU, fp64 in the oracle):
        |gpu - oracle| <= 1e-5 * max(|oracle|, rms(oracle field))
  * fp32 replicas: the same bound (they hold theta');
  * bf16 replicas: |gpu - oracle| <= 1 bf16 ulp (at the oracle's value)
    plus theta's own field tolerance.  The GPU rounds its fp32 theta' to
    bf16, the oracle its fp64 theta': the two roundings can differ by one
    step, and by more only where theta' itself differs by more than a bf16
    step, which happens where theta - eta d cancels to a value far below the
    field's scale.  In addition, every GPU bf16 replica must be exactly the
    round-to-nearest-even of the GPU's own theta' (a property, not a
    comparison with the oracle);
  * D, C, ||Dbar||^2 and each ||Delta_m||^2: relative 1e-6;
  * correction scalars (both fp64, on the host): relative 1e-12;
  * integer outputs (non-finite count): exact.
"""
from __future__ import annotations

import concurrent.futures as cf

import numpy as np
import torch

import oracle as O
from paper_2609_36662_gb300 import aloco as A
from paper_2609_36662_gb300 import workloads as W

RTOL_FIELD = 1e-5
RTOL_STAT = 1e-6
RTOL_SCALAR = 1e-12


def to_numpy_bits(x: torch.Tensor) -> np.ndarray:
    """Host copy of a replica: float32 values or bf16 bit patterns."""
    if x.dtype == torch.bfloat16:
        return x.detach().cpu().view(torch.int16).numpy().view(np.uint16)
    return x.detach().cpu().numpy()


def oracle_dtype(t: torch.dtype) -> int:
    return O.F32 if t == torch.float32 else O.BF16


def schedule_pair(spec: W.ScheduleSpec):
    return (A.Schedule.make(spec.kind, spec.peak_lr, spec.final_lr,
                            spec.warmup_steps, spec.total_steps),
            O.Schedule(spec.kind, spec.peak_lr, spec.final_lr,
                       spec.warmup_steps, spec.total_steps))


def field_error(gpu: np.ndarray, orc: np.ndarray, terms=None) -> float:
    """Largest error relative to max(|oracle|, rms of the oracle field, and,
    where given, the magnitude of the terms the value is formed from)."""
    gpu = np.asarray(gpu, np.float64)
    orc = np.asarray(orc, np.float64)
    if orc.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(orc * orc)))
    scale = np.maximum(np.abs(orc), max(rms, 1e-300))
    if terms is not None:
        scale = np.maximum(scale, np.asarray(terms, np.float64))
    err = np.abs(gpu - orc) / scale
    err[(gpu == orc)] = 0.0
    return float(err.max())


def assert_field(gpu, orc, name, rtol=RTOL_FIELD, terms=None):
    e = field_error(gpu, orc, terms)
    assert e <= rtol, f"{name}: max scaled error {e:.3e} > {rtol:.0e}"


def step_terms(g, v, xs, dtype, mu_t, eta_out, inv_norm):
    """Per element, the magnitudes of the terms of the corrected Nesterov
    step (Eq. autoloco-corrected-nesterov): v' = mu v + Dtil with Dtil =
    inv_norm S / M, S = sum_m (theta - x_m), and theta' = theta - eta (Dtil +
    mu v').  Evaluated in fp32, each result carries rounding errors of the
    size of its terms (S alone rounds M - 1 times), so where the terms
    cancel (a vector of a few elements has no rms to fall back on) the
    tolerance scales with them: |mu v| + |inv_norm / M| sum_m |theta - x_m|
    for v', and |theta| + |eta| (that + mu (that)) for theta'."""
    g = np.asarray(g, np.float64)
    v = np.asarray(v, np.float64)
    a = np.zeros_like(g)
    for x in xs:
        xf = (O.bf16_bits_to_float(x) if dtype == O.BF16 else np.asarray(x)).astype(np.float64)
        a += np.abs(g - xf)
    dt = abs(inv_norm) / len(xs) * a
    tv = abs(mu_t) * np.abs(v) + dt
    tg = np.abs(g) + abs(eta_out) * (dt + abs(mu_t) * tv)
    return tg, tv


def fp32_ulp(values) -> np.ndarray:
    """Spacing of fp32 numbers at |values|."""
    a = np.abs(np.asarray(values, np.float64))
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return np.exp2(np.maximum(e, -126) - 23)


def assert_field_after_chain(gpu, orc, theta_orc, rounds, name,
                             rtol=RTOL_FIELD):
    """Final state of two independent multi-round chains.  Each chain stores
    theta in fp32 between rounds; where the two roundings of theta differ
    (one fp32 step), the next round's pseudo-gradients differ by that step,
    and the state carries it on with gain at most one per round.  So on top
    of the per-round field tolerance each element may differ by up to
    `rounds` fp32 steps of its theta; the whole-vector relative L2 error
    must still be within the field tolerance."""
    gpu = np.asarray(gpu, np.float64)
    orc = np.asarray(orc, np.float64)
    rms = float(np.sqrt(np.mean(orc * orc)))
    tol = rtol * np.maximum(np.abs(orc), rms) + rounds * fp32_ulp(theta_orc)
    bad = np.abs(gpu - orc) > tol
    assert not bad.any(), (f"{name}: {int(bad.sum())} elements beyond the "
                           f"chain tolerance, e.g. index {int(np.argmax(bad))}")
    l2 = float(np.linalg.norm(gpu - orc) / max(np.linalg.norm(orc), 1e-300))
    assert l2 <= rtol, f"{name}: relative L2 error {l2:.3e}"


def bf16_order_key(bits: np.ndarray) -> np.ndarray:
    b = bits.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def bf16_ulp(values: np.ndarray) -> np.ndarray:
    """Spacing of bf16 numbers at |values| (8 significant bits)."""
    a = np.abs(np.asarray(values, np.float64))
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return np.exp2(np.maximum(e, -126) - 7)


def assert_bf16_replica(gpu_bits, orc_bits, orc_theta, name,
                        rtol=RTOL_FIELD, extra_abs=0.0):
    gv = O.bf16_bits_to_float(gpu_bits)
    ov = O.bf16_bits_to_float(orc_bits)
    orc_theta = np.asarray(orc_theta, np.float64)
    rms = float(np.sqrt(np.mean(orc_theta * orc_theta))) if orc_theta.size \
        else 0.0
    tol = bf16_ulp(ov) + rtol * np.maximum(np.abs(orc_theta), rms) + extra_abs
    bad = np.abs(gv - ov) > tol
    assert not bad.any(), (f"{name}: {int(bad.sum())} bf16 replicas beyond one "
                           f"ulp + field tolerance, e.g. index "
                           f"{int(np.argmax(bad))}")


def assert_bf16_is_rounded_theta(gpu_bits, gpu_theta: torch.Tensor, name):
    want = gpu_theta.detach().cpu().to(torch.bfloat16).view(torch.int16) \
        .numpy().view(np.uint16)
    assert np.array_equal(gpu_bits, want), \
        f"{name} is not the bf16 rounding of theta'"


def assert_rel(gpu, orc, name, rtol):
    if orc == 0.0:
        assert gpu == 0.0 or abs(gpu) < 1e-300, f"{name}: {gpu} vs 0"
        return
    r = abs(gpu - orc) / abs(orc)
    assert r <= rtol, f"{name}: {gpu!r} vs {orc!r} (rel {r:.3e} > {rtol:.0e})"


def assert_stats(st: dict, orc: dict, M: int):
    assert_rel(st["D"], orc["D"], "D", RTOL_STAT)
    assert_rel(st["C"], orc["C"], "C", RTOL_STAT)
    assert_rel(st["mean_sq_norm"], orc["mean_sq_norm"], "||Dbar||^2",
               RTOL_STAT)
    for m in range(M):
        assert_rel(st["drift"][m], orc["drift"][m], f"||Delta_{m}||^2",
                   RTOL_STAT)


def assert_corr(corr: dict, oc: O.Correction):
    for k in ("lam_sel", "lam_base", "rho_unc", "rho", "mu_t", "kappa_t",
              "eta_out", "inv_norm"):
        assert_rel(corr[k], getattr(oc, k), k, RTOL_SCALAR)


def oracle_stats_threaded(g: torch.Tensor, xs, eps: float, slice_elems=1 << 24,
                          threads: int = 16):
    """Pass-1 sums of the oracle over a long device-resident vector: slices
    are copied to the host and summed by oracle threads (ctypes releases the
    GIL); the per-slice sums are then added in slice order."""
    N = g.numel()
    M = len(xs)
    dt = oracle_dtype(xs[0].dtype)
    bounds = [(s, min(N, s + slice_elems)) for s in range(0, N, slice_elems)]
    accs = [O.Pass1Accumulator(M) for _ in bounds]

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        futs = []
        for k, (s, e) in enumerate(bounds):
            gh = g[s:e].cpu().numpy()
            xh = [to_numpy_bits(x[s:e]) for x in xs]
            futs.append(ex.submit(accs[k].add, gh, xh, dt))
            if len(futs) >= 2 * threads:
                futs.pop(0).result()
        for f in futs:
            f.result()
    E = [0.0] * M
    B = 0.0
    for acc in accs:
        for m in range(M):
            E[m] += acc.E[m]
        B += acc.B.value
    Dsum = 0.0
    for m in range(M):
        Dsum += E[m]
    D = Dsum / M
    return {"D": D, "C": M * B / (D + eps), "mean_sq_norm": B, "drift": E}


def sample_indices(N: int, boundaries=(), k: int = 4096, seed: int = 0):
    """Indices to compare at full size: random ones, both ends, and the
    first/last element of every tensor of the layout."""
    rng = np.random.default_rng(seed)
    idx = set(rng.integers(0, N, size=min(k, N)).tolist())
    idx.update([0, 1, N - 2, N - 1])
    for b in boundaries:
        for j in (b - 1, b, b + 1):
            if 0 <= j < N:
                idx.add(j)
    return torch.tensor(sorted(idx), dtype=torch.int64)


# ------------------------------------------------------------ round runners

def gpu_inputs(w: W.Workload, device="cuda", round_index=0):
    g = W.make_global(w, device)
    v = W.make_momentum(w, device)
    xs = W.fill_replicas(w, g, W.alloc_replicas(w, device), round_index)
    return g, v, xs


def run_gpu_round(g, v, xs, w: W.Workload, step: int, H_sel: int,
                  opts=None, stream=None):
    sa, _ = schedule_pair(w.schedule)
    return A.sync(g, v, xs, H_sel=H_sel, H_base=w.H_base, step=step,
                  schedule=sa, outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                  opts=opts, stream=stream, raise_on_error=False)


def run_oracle_round(g, v, xs, w: W.Workload, step: int, H_sel: int,
                     normalize=False, mode=O.MODE_FULL, eps=1e-8):
    """Oracle round on host copies (taken before the GPU overwrites them)."""
    _, so = schedule_pair(w.schedule)
    gh = g.cpu().numpy() if isinstance(g, torch.Tensor) else g
    vh = v.cpu().numpy() if isinstance(v, torch.Tensor) else v
    xh = [to_numpy_bits(x) if isinstance(x, torch.Tensor) else x for x in xs]
    dt = O.F32 if w.dtype == "f32" else O.BF16
    orc = O.sync_round(gh, vh, xh, dt, so, step, H_sel, w.H_base, w.outer_lr,
                       w.outer_beta, eps=eps, normalize=normalize, mode=mode)
    c = orc["corr"]
    orc["g_terms"], orc["v_terms"] = step_terms(gh, vh, xh, dt, c.mu_t, c.eta_out,
                                                c.inv_norm)
    return orc


def compare_round(w, st, orc, g, v, xs):
    """Element-by-element comparison of a whole round."""
    assert st["nonfinite"] == orc["nonfinite"]
    assert_corr(st["corr"], orc["corr"])
    assert_stats(st, orc, w.M)
    assert_field(g.cpu().numpy(), orc["g"], "theta'", terms=orc.get("g_terms"))
    assert_field(v.cpu().numpy(), orc["v"], "v'", terms=orc.get("v_terms"))
    gg = g.cpu().numpy()
    for m, x in enumerate(xs):
        if w.dtype == "f32":
            xh = x.cpu().numpy()
            assert np.array_equal(xh.view(np.uint32), gg.view(np.uint32)), \
                f"replica {m} is not theta'"
            assert_field(xh, orc["x"][m], f"replica {m}")
        else:
            bits = to_numpy_bits(x)
            assert_bf16_is_rounded_theta(bits, g, f"replica {m}")
            assert_bf16_replica(bits, orc["x"][m], orc["g"], f"replica {m}")


def oracle_chain_endpoints(w: W.Workload, g_host: np.ndarray, round_index,
                           device="cuda"):
    """The oracle chain's own endpoints for a round: the same generator,
    applied to the oracle's theta (uploaded chunk by chunk).  Returns the
    fp32 values before storage and the stored replicas (fp32, or bf16 bit
    patterns rounded to nearest even)."""
    y = [np.empty(w.numel, np.float32) for _ in range(w.M)]
    for c in range(W.n_chunks(w)):
        s, e = c * W.CHUNK, min(w.numel, (c + 1) * W.CHUNK)
        gc = torch.from_numpy(g_host[s:e]).to(device)
        for m, x in enumerate(W.replica_chunk(w, gc, round_index, c)):
            y[m][s:e] = x.cpu().numpy()
    if w.dtype == "f32":
        return y, y
    return y, [to_bf16_bits(t) for t in y]


def oracle_chain_replicas(w: W.Workload, g_host: np.ndarray, round_index,
                          device="cuda"):
    return oracle_chain_endpoints(w, g_host, round_index, device)[1]


def to_bf16_bits(y: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(y, np.float32)) \
        .to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def gather_host(t: torch.Tensor, idx: torch.Tensor) -> np.ndarray:
    return to_numpy_bits(t[idx.to(t.device)])


def oracle_pass2_at(w: W.Workload, g_idx, v_idx, x_idx, corr: O.Correction):
    """The oracle's elementwise update at sampled elements (each element
    depends only on its own inputs and the round's scalars)."""
    dt = O.F32 if w.dtype == "f32" else O.BF16
    return O.pass2(g_idx, v_idx, x_idx, dt, corr.mu_t, corr.eta_out,
                   corr.inv_norm)


def oracle_corr(w: W.Workload, step, hsel, normalize=False, mode=O.MODE_FULL):
    _, so = schedule_pair(w.schedule)
    return O.correction(so, step, hsel, w.H_base, w.outer_lr, w.outer_beta,
                        normalize=normalize, mode=mode)


def compare_sampled(w, g_gpu_idx, v_gpu_idx, x_gpu_idx, ref,
                    prior_rounds: int = 0):
    """Sampled elements of a round.  In the k-th round of two independent
    chains (prior_rounds = k) the inputs already differ by the chains' fp32
    storage of theta; see assert_field_after_chain."""
    g_o, v_o, x_o, _ = ref
    if prior_rounds == 0:
        assert_field(g_gpu_idx, g_o, "theta' (sampled)")
        assert_field(v_gpu_idx, v_o, "v' (sampled)")
    else:
        assert_field_after_chain(g_gpu_idx, g_o, g_o, prior_rounds + 1,
                                 "theta' (sampled)")
        assert_field_after_chain(v_gpu_idx, v_o, g_o, prior_rounds + 1,
                                 "v' (sampled)")
    for m in range(w.M):
        if w.dtype == "f32":
            if prior_rounds == 0:
                assert_field(x_gpu_idx[m], x_o[m], f"replica {m} (sampled)")
            else:
                assert_field_after_chain(x_gpu_idx[m], x_o[m], g_o,
                                         prior_rounds + 1,
                                         f"replica {m} (sampled)")
        else:
            assert_bf16_replica(x_gpu_idx[m], x_o[m], g_o,
                                f"replica {m} (sampled)",
                                extra_abs=(prior_rounds + 1) * fp32_ulp(g_o)
                                if prior_rounds else 0.0)


def oracle_pass2_threaded(w: W.Workload, g_h, v_h, x_h, corr,
                          slice_elems=1 << 22, threads=16):
    """Oracle update over whole host vectors, slices run by threads.
    Returns fp64 theta', v'."""
    N = g_h.shape[0]
    g_out = np.empty(N, np.float64)
    v_out = np.empty(N, np.float64)
    dt = O.F32 if w.dtype == "f32" else O.BF16

    def work(s):
        e = min(N, s + slice_elems)
        go, vo, _, _ = O.pass2(g_h[s:e], v_h[s:e], [x[s:e] for x in x_h], dt,
                               corr.mu_t, corr.eta_out, corr.inv_norm,
                               want_replicas=False)
        g_out[s:e] = go
        v_out[s:e] = vo

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(work, range(0, N, slice_elems)))
    return g_out, v_out


def oracle_stats_host_threaded(w: W.Workload, g_h, x_h, eps=1e-8,
                               slice_elems=1 << 22, threads=16):
    N = g_h.shape[0]
    dt = O.F32 if w.dtype == "f32" else O.BF16
    starts = list(range(0, N, slice_elems))
    accs = [O.Pass1Accumulator(w.M) for _ in starts]

    def work(k):
        s = starts[k]
        e = min(N, s + slice_elems)
        accs[k].add(g_h[s:e], [x[s:e] for x in x_h], dt)

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(work, range(len(starts))))
    E = [0.0] * w.M
    B = 0.0
    for acc in accs:
        for m in range(w.M):
            E[m] += acc.E[m]
        B += acc.B.value
    D = sum(E) / w.M
    return {"D": D, "C": w.M * B / (D + eps), "mean_sq_norm": B, "drift": E}



class _FieldCheck:
    """Streaming form of the field tolerance over a vector seen slice by
    slice: the bound excess <= rtol * max(|field|, rms(field)) needs the
    whole field's rms, so elements whose excess is above rtol * |field| are
    kept as candidates and judged against the rms once every slice has been
    seen."""

    def __init__(self, name, rtol=RTOL_FIELD):
        self.name, self.rtol = name, rtol
        self.sq, self.n = 0.0, 0
        self.excess, self.ref, self.index = [], [], []

    def add(self, excess, field, offset):
        field = np.asarray(field, np.float64)
        self.sq += float(np.dot(field, field))
        self.n += field.size
        a = np.abs(field)
        c = np.nonzero(excess > self.rtol * a)[0]
        self.excess.append(excess[c])
        self.ref.append(a[c])
        self.index.append(c + offset)

    def check(self) -> int:
        """Assert the bound; returns the number of elements that needed the
        rms part of it."""
        rms = np.sqrt(self.sq / max(self.n, 1))
        ex = np.concatenate(self.excess)
        ref = np.concatenate(self.ref)
        idx = np.concatenate(self.index)
        bad = ex > self.rtol * np.maximum(ref, rms)
        assert not bad.any(), (f"{self.name}: {int(bad.sum())} elements beyond "
                               f"the field tolerance, e.g. index "
                               f"{int(idx[np.argmax(bad)])}")
        return int(ex.size)


def _abs_diff(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    d = np.abs(a - b)
    d[a == b] = 0.0
    return d


def compare_whole_vector(w: W.Workload, g_in, v_in, x_in, g, v, xs, corr,
                         slice_elems=1 << 24, threads=16):
    """theta', v' and the replica reset of a round against the oracle's
    elementwise update over the WHOLE vector (not a sample), slice by slice:
    each slice of the device snapshot of the inputs and of the GPU's outputs
    is copied to the host, the oracle's pass 2 runs on it in threads, and
    every element is held to the tolerances of compare_round.  Host memory
    stays at a few slices whatever the vector's size.  The replica reset is
    compared with the oracle through replica 0; the caller checks on the
    device that every replica equals it (the reset writes one value)."""
    N = w.numel
    dt = O.F32 if w.dtype == "f32" else O.BF16
    fg, fv, fx = (_FieldCheck("theta'"), _FieldCheck("v'"),
                  _FieldCheck("replica 0"))
    sub = max(1, slice_elems // threads)
    for s in range(0, N, slice_elems):
        e = min(N, s + slice_elems)
        gh = g_in[s:e].cpu().numpy()
        vh = v_in[s:e].cpu().numpy()
        xh = [to_numpy_bits(x[s:e]) for x in x_in]
        go = np.empty(e - s, np.float64)
        vo = np.empty(e - s, np.float64)
        xo = np.empty(e - s, np.float32 if dt == O.F32 else np.uint16)

        def work(a):
            b = min(e - s, a + sub)
            r = O.pass2(gh[a:b], vh[a:b], [x[a:b] for x in xh], dt,
                        corr.mu_t, corr.eta_out, corr.inv_norm,
                        want_replicas=True)
            go[a:b], vo[a:b], xo[a:b] = r[0], r[1], r[2][0]

        with cf.ThreadPoolExecutor(max_workers=threads) as ex:
            list(ex.map(work, range(0, e - s, sub)))
        fg.add(_abs_diff(g[s:e].cpu().numpy(), go), go, s)
        fv.add(_abs_diff(v[s:e].cpu().numpy(), vo), vo, s)
        x0 = to_numpy_bits(xs[0][s:e])
        if dt == O.F32:
            fx.add(_abs_diff(x0, xo), xo, s)
        else:
            # one bf16 ulp at the oracle's value, then theta's own bound
            ov = O.bf16_bits_to_float(xo)
            fx.add(_abs_diff(O.bf16_bits_to_float(x0), ov) - bf16_ulp(ov),
                   go, s)
    return {"theta_candidates": fg.check(), "v_candidates": fv.check(),
            "replica_candidates": fx.check()}


def int8_slices(parts, slice_elems=1 << 24):
    """(start, length) slices of a vector made of tensor parts, each inside
    one part and starting at a multiple of 4096 from that part's start, so
    every slice holds whole codec blocks (they restart at every part)."""
    step = max(4096, slice_elems // 4096 * 4096)
    out, off = [], 0
    for p in parts:
        for o in range(0, p, step):
            out.append((off + o, min(step, p - o)))
        off += p
    return out


def compare_int8_whole_vector(w: W.Workload, parts, g_in, v_in, x_in, g, v, xs,
                              corr, eps=1e-8, slice_elems=1 << 24, threads=16):
    """The INT8-communicated round against the oracle over the WHOLE vector:
    slice by slice (whole codec blocks each), the oracle's INT8 round runs on
    host copies of the device snapshot in threads, and every element of
    theta', v' and replica 0 is held to the tolerances of compare_round; the
    slices' drift energies and squared decoded aggregates are added in slice
    order into the whole round's statistics, which are returned (D from the
    pre-quantisation pseudo-gradients, C from the decoded aggregate)."""
    dt = O.F32 if w.dtype == "f32" else O.BF16
    fg, fv, fx = (_FieldCheck("theta'"), _FieldCheck("v'"),
                  _FieldCheck("replica 0"))
    E = [0.0] * w.M
    B = 0.0
    slices = int8_slices(parts, slice_elems)

    def work(s, n, gh, vh, xh):
        return O.int8_round(gh, vh, xh, dt, [n], corr.mu_t, corr.eta_out,
                            corr.inv_norm, eps)

    def check(s, n, r):
        nonlocal B
        e = s + n
        fg.add(_abs_diff(g[s:e].cpu().numpy(), r["g"]), r["g"], s)
        fv.add(_abs_diff(v[s:e].cpu().numpy(), r["v"]), r["v"], s)
        x0 = to_numpy_bits(xs[0][s:e])
        if dt == O.F32:
            fx.add(_abs_diff(x0, r["x"][0]), r["x"][0], s)
        else:
            ov = O.bf16_bits_to_float(r["x"][0])
            fx.add(_abs_diff(O.bf16_bits_to_float(x0), ov) - bf16_ulp(ov),
                   r["g"], s)
        for m in range(w.M):
            E[m] += r["drift"][m]
        B += r["mean_sq_norm"]

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        pending = []
        for s, n in slices:
            e = s + n
            fut = ex.submit(work, s, n, g_in[s:e].cpu().numpy(),
                            v_in[s:e].cpu().numpy(),
                            [to_numpy_bits(x[s:e]) for x in x_in])
            pending.append((s, n, fut))
            if len(pending) >= 2 * threads:
                s0, n0, f0 = pending.pop(0)
                check(s0, n0, f0.result())
        for s0, n0, f0 in pending:
            check(s0, n0, f0.result())
    fg.check()
    fv.check()
    fx.check()
    D = sum(E) / w.M
    return {"D": D, "C": w.M * B / (D + eps), "mean_sq_norm": B, "drift": E}
