#!/usr/bin/env python3
"""Benchmark of the fused AutoLoCo outer-sync round on GB300.

A step is one outer synchronisation round (Algorithm 1: pseudo-gradients,
average, D_t / C_t, corrected Nesterov step, replica reset) over one batch
of synthetic worker endpoints, called through the C ABI.  The default
workload is the largest parameter set that fits one GPU: the Llama-style 3B
set (26 layers, d 3072, 8 KV heads, untied; N = 2,814,016,512) with 8 bf16
worker replicas and fp32 global weights and momentum (67.5 GB resident),
over consecutive rounds whose horizons rise from 100 to 400 steps along a
40k-step cosine schedule, momentum carried across rounds.

Between timed rounds the replicas are refilled with new endpoints (this
stands in for the workers' inner loops and is not timed); each round is
bracketed by CUDA events on the launch stream, and the whole loop by a
barrier and device synchronisation.  The reported step time is the median
over the timed rounds.  A round of the default workload reads and writes
135 GB, far more than the 129 MB L2; rounds whose buffers are smaller than
four times the L2 are preceded by an untimed write of a buffer twice the
L2's size, so that no round starts with its inputs in L2.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 oracle on the host

Multi-GPU: the round does not shard across GPUs; with N > 1 every rank runs
an independent replica of the workload on its own GPU ("replicas only") and
the value is the total rounds/s of the job.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("outer-sync rounds/s and achieved HBM GB/s (fraction of GB300 "
          "roofline) at N params × M workers")
UNIT = "rounds/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
PASSES = {"auto": 0, "registers": 1, "bulk_copy": 2, "int8_split": 3,
          "int8_fused": 4, "tile": 5}
WAITS = {"spin": 0, "block": 1}


def workloads_by_name():
    from paper_2609_36662_gb300 import workloads as W
    out = {w.name: w for w in W.all_configs()}
    return out


def parse_flat(name: str):
    """flat<N>_m<M>_<f32|bf16>: a flat vector of N parameters (used for the
    small profiling cases)."""
    import re
    from paper_2609_36662_gb300 import workloads as W
    m = re.fullmatch(r"flat(\d+)_m(\d+)_(f32|bf16)", name)
    if not m:
        return None
    return W.small(int(m.group(1)), int(m.group(2)), m.group(3), seed=4,
                   H_sel=200, H_base=100)


def default_workload_name():
    from paper_2609_36662_gb300 import workloads as W
    return W.llama_3b().name


L2_FALLBACK_BYTES = 129 * 1024 * 1024


def l2_bytes(device) -> int:
    import torch
    try:
        n = int(torch.cuda.get_device_properties(device).L2_cache_size)
        return n if n > 0 else L2_FALLBACK_BYTES
    except Exception:
        return L2_FALLBACK_BYTES


def needs_l2_flush(footprint_bytes: int, l2: int) -> bool:
    """Whether a round's buffers are small enough that part of them could
    still sit in L2 from the previous round (then each timed round is
    preceded by an untimed write of a buffer twice the L2's size)."""
    return footprint_bytes < 4 * l2


def host_memory():
    """Physical and available host memory in bytes (None where unknown),
    and the cgroup limit if one is set."""
    out = {"host_ram_bytes": None, "mem_available_bytes": None,
           "cgroup_limit_bytes": None}
    try:
        out["host_ram_bytes"] = os.sysconf("SC_PAGE_SIZE") * \
            os.sysconf("SC_PHYS_PAGES")
    except Exception:
        pass
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    out["mem_available_bytes"] = int(line.split()[1]) * 1024
    except Exception:
        pass
    for path in ("/sys/fs/cgroup/memory.max",
                 "/sys/fs/cgroup/memory/memory.limit_in_bytes"):
        try:
            with open(path) as f:
                txt = f.read().strip()
            if txt.isdigit() and int(txt) < (1 << 60):
                out["cgroup_limit_bytes"] = int(txt)
            break
        except Exception:
            continue
    return out


def pinned_budget(mem, ranks_on_host: int = 1) -> int:
    """Pinned host bytes one rank's e2e leg may take: half of what is
    available (and of the cgroup limit), shared by the ranks on this host,
    so the host keeps room for the rest."""
    cands = [v for v in (mem.get("mem_available_bytes"),
                         mem.get("cgroup_limit_bytes"),
                         mem.get("host_ram_bytes")) if v]
    if not cands:
        return 0
    return int(0.5 * min(cands) / max(1, ranks_on_host))


def ranks_on_host() -> int:
    """Ranks of this job on this host (torchrun's LOCAL_WORLD_SIZE)."""
    try:
        return max(1, int(os.environ.get("LOCAL_WORLD_SIZE", "1")))
    except ValueError:
        return 1


def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# the sources each timed kernel is compiled from; a recorded ncu traffic
# figure stays valid only while these files are unchanged
KERNEL_SOURCES = {
    "sync_kernel": ("aloco_sync_kernel.cuh", "aloco_sync_f32.cu",
                    "aloco_sync_bf16.cu"),
    "sync_tile_kernel": ("aloco_sync_kernel.cuh", "aloco_bulk.cuh", "aloco_sync_tile.cu"),
    "sync_tma_kernel": ("aloco_sync_kernel.cuh", "aloco_bulk.cuh", "aloco_sync_tma.cuh",
                        "aloco_sync_tma_f32.cu", "aloco_sync_tma_bf16.cu"),
    "int8_split_kernels": ("aloco_sync_kernel.cuh", "aloco_int8.cuh",
                           "aloco_int8.cu"),
    "int8_fused_kernel": ("aloco_sync_kernel.cuh", "aloco_bulk.cuh", "aloco_int8.cuh",
                          "aloco_int8_fused.cu"),
    "adamw_kernels": ("aloco_sync_kernel.cuh", "aloco_adamw.cu"),
}


def kernel_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_36662_gb300", "csrc")
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def recorded_entry(workload: str, kernel: str):
    """The committed ncu record of this kernel on this workload, if it was
    taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except Exception:
        return None
    entry = rec.get(f"{workload}/{kernel}")
    if not entry or entry.get("kernel_hash") != kernel_source_hash(kernel):
        return None
    return entry


def recorded_traffic(workload: str, kernel: str):
    """DRAM bytes per launch of the fused pass from the committed ncu
    summary, if it was taken on the current kernel source."""
    entry = recorded_entry(workload, kernel)
    return entry.get("dram_bytes_per_launch") if entry else None


def recorded_occupancy(workload: str, kernel: str):
    """Achieved occupancy (ncu sm__warps_active, % of the SM's warp slots)
    from the same record, with the case it was measured on."""
    entry = recorded_entry(workload, kernel)
    if not entry or entry.get("warps_active_pct") is None:
        return None
    return {"warps_active_pct": entry["warps_active_pct"],
            "measured_on": entry["measured_on"].split(":")[0]}


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed
    region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        time.sleep(0.2)
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
        return False

    def summary(self):
        rows = []
        for line in (self.out or "").splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[4:8]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows
                          for i, f in enumerate(flags) if f.lower() == "active"})
        mx = max(r[1] for r in rows)
        loaded = [r[0] for r in rows if r[0] >= 0.5 * mx] or [r[0] for r in rows]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx,
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------- distributed

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reduce_max(value: float, world: int, device=None) -> float:
    """Max over ranks (identity for one rank)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def gather_partials(blob: bytes, world: int, device=None):
    """Every rank's partial-sums blob (aloco_partials_t bytes), in rank
    order: an all-gather of one fixed-size byte string per rank over the
    process group (identity for one rank)."""
    if world <= 1:
        return [bytes(blob)]
    import torch
    import torch.distributed as dist
    t = torch.frombuffer(bytearray(blob), dtype=torch.uint8)
    if device is not None:
        t = t.to(device)
    out = [torch.empty_like(t) for _ in range(world)]
    dist.all_gather(out, t)
    return [o.cpu().numpy().tobytes() for o in out]


def job_value(units_per_rank: float, seconds_max: float, world: int) -> float:
    """Whole-job throughput: the units every rank processed over the slowest
    rank's time."""
    return units_per_rank * world / seconds_max


# ------------------------------------------------------------ CPU oracle

def prefix_parts(parts, n: int):
    """The tensor parts of the first n elements (the last one cut short)."""
    out, acc = [], 0
    for p in parts:
        if acc >= n:
            break
        take = min(p, n - acc)
        out.append(take)
        acc += take
    return out


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def slice_cuts(n: int, k: int, starts=None):
    """Cut points of k contiguous slices of [0, n); with `starts` (sorted
    codec block starts) every cut falls on a block start."""
    import bisect
    cuts = [0]
    for i in range(1, k):
        c = n * i // k
        if starts is not None:
            j = bisect.bisect_left(starts, c)
            c = starts[j] if j < len(starts) else n
        if cuts[-1] < c < n:
            cuts.append(c)
    return cuts + [n]


def parts_between(parts, a: int, b: int):
    """The tensor parts of elements [a, b), cut at both ends."""
    out, off = [], 0
    for p in parts:
        lo, hi = max(off, a), min(off + p, b)
        if lo < hi:
            out.append(hi - lo)
        off += p
    return out


def run_sliced(fn, cuts, threads: int):
    """fn(a, b) over the slices, on `threads` host threads (the oracle's C
    calls release the interpreter lock)."""
    pairs = list(zip(cuts[:-1], cuts[1:]))
    if threads <= 1 or len(pairs) == 1:
        for a, b in pairs:
            fn(a, b)
        return
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(lambda ab: fn(*ab), pairs))


def oracle_sample(w, g, v, xs, elems: int, step: int, H_sel: int,
                  comm: str = "fp32", threads: int = 1):
    """Time the oracle, as it stands, on the first `elems` elements of the
    round (the INT8-communicated round when comm is "int8", with the codec's
    blocks cut at the same tensor boundaries).  With threads > 1 the sample
    is cut into that many contiguous slices (at codec block starts for INT8)
    run concurrently.  Returns (seconds, elements)."""
    import numpy as np
    import torch
    import oracle as O
    n = min(elems, w.numel)
    gh = g[:n].cpu().numpy()
    vh = v[:n].cpu().numpy()
    if w.dtype == "f32":
        xh = [x[:n].cpu().numpy() for x in xs]
    else:
        xh = [x[:n].cpu().view(torch.int16).numpy().view(np.uint16)
              for x in xs]
    s = w.schedule
    sched = O.Schedule(s.kind, s.peak_lr, s.final_lr, s.warmup_steps,
                       s.total_steps)
    dt = O.F32 if w.dtype == "f32" else O.BF16
    if comm == "int8":
        from paper_2609_36662_gb300 import workloads as W
        parts = prefix_parts(W.tensor_sizes(w), n)
        starts, off = [], 0
        for p in parts:
            starts.extend(range(off, off + p, 4096))
            off += p
        cuts = slice_cuts(n, threads, starts)
        corr = O.correction(sched, step, H_sel, w.H_base, w.outer_lr,
                            w.outer_beta)

        def fn(a, b):
            O.int8_round(gh[a:b], vh[a:b], [x[a:b] for x in xh], dt,
                         parts_between(parts, a, b), corr.mu_t, corr.eta_out,
                         corr.inv_norm)
    else:
        cuts = slice_cuts(n, threads)

        def fn(a, b):
            O.sync_round(gh[a:b], vh[a:b], [x[a:b] for x in xh], dt, sched,
                         step, H_sel, w.H_base, w.outer_lr, w.outer_beta)
    t0 = time.perf_counter()
    run_sliced(fn, cuts, threads)
    return time.perf_counter() - t0, n


def calibrated_sample(w, g, v, xs, step, H_sel, target_s, comm="fp32"):
    """Pick a sample size whose oracle run takes about target_s seconds."""
    probe = min(w.numel, 1 << 20)
    t, n = oracle_sample(w, g, v, xs, probe, step, H_sel, comm)
    per_elem = t / n
    want = int(target_s / max(per_elem, 1e-12))
    want = max(1 << 16, min(w.numel, want))
    return want


# ------------------------------------------------------------- main arms

def run_reference(args, w):
    """The fp64 oracle on the host cores, timed per step on a bounded
    sample of the workload (rank 0 only)."""
    import torch
    from paper_2609_36662_gb300 import workloads as W
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    rounds = W.steps_of_rounds(w, args.warmup + args.steps)
    step0, h0 = rounds[0]

    def inputs(n_chunks):
        # the first n_chunks generator chunks of theta, v and the endpoints
        # (a prefix of the workload's own vectors)
        n = min(w.numel, n_chunks * W.CHUNK)
        g = W.make_global(w, "cpu", upto=n)
        v = W.make_momentum(w, "cpu", upto=n)
        xs = [torch.empty(n, dtype=W.replica_dtype(w)) for _ in range(w.M)]
        W.fill_replicas(w, g, xs, 0, 0, W.n_chunks_upto(n))
        return g, v, xs

    # calibrate on the first chunk, then draw only the chunks the sample needs
    g, v, xs = inputs(1)
    sample = calibrated_sample(w, g, v, xs, step0, h0, args.ref_step_seconds,
                               args.comm)
    need = W.n_chunks_upto(sample)
    if need > 1:
        g, v, xs = inputs(need)
    cores = host_cores()
    times = []
    for k, (step, hsel) in enumerate(rounds):
        t, n = oracle_sample(w, g, v, xs, sample, step, hsel, args.comm,
                             threads=cores)
        if k >= args.warmup:
            times.append(t)
    sec_per_round = statistics.median(times) * w.numel / sample
    value = 1.0 / sec_per_round
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sec_per_round * 1e3, "ms_per_step_stat": "median",
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64",
        "replica_dtype": w.dtype, "data": "synthetic",
        "config": dict(config_block(w), comm=args.comm),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores,
                         "kind": "oracle",
                         "sample": f"first {sample} of {w.numel} parameters "
                                   f"x {w.M} workers per step, in {cores} "
                                   f"concurrent slices, scaled to a full "
                                   f"round"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def footprint_bytes(w) -> int:
    """Bytes of the buffers one round reads (each is also written)."""
    return w.bytes_per_round() // 2


def l2_note(w, l2: int = L2_FALLBACK_BYTES) -> str:
    if needs_l2_flush(footprint_bytes(w), l2):
        return (f"L2 flushed before each timed round: the round's buffers "
                f"({footprint_bytes(w) / 1e6:.0f} MB) are smaller than four "
                f"times the L2, so an untimed write of {2 * l2 / 1e6:.0f} MB "
                f"precedes each round")
    return (f"no flush: each round moves {w.bytes_per_round() / 1e9:.1f} GB "
            f"> 129 MB L2")


def config_block(w):
    from paper_2609_36662_gb300 import workloads as W
    return {"workload": w.name, "N": w.numel, "M": w.M,
            "replica_dtype": w.dtype, "outer_state_dtype": "f32",
            "shape": (None if w.shape is None else
                      {"layers": w.shape.layers, "d_model": w.shape.d_model,
                       "heads": w.shape.heads, "kv_heads": w.shape.kv_heads,
                       "ffn": w.shape.ffn, "vocab": w.shape.vocab,
                       "tied": w.shape.tied}),
            "bytes_per_round": w.bytes_per_round(),
            "l2": l2_note(w),
            "H_base": w.H_base, "start_step": w.start_step,
            "parallelism": "replicas only"}


def run_cuda(args, w):
    import numpy as np
    import torch
    from paper_2609_36662_gb300 import aloco as A
    from paper_2609_36662_gb300 import workloads as W

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", torch.cuda.current_device())
    A.load()

    rounds = W.steps_of_rounds(w, args.warmup + args.steps)
    g = W.make_global(w, device)
    v = W.make_momentum(w, device)
    xs = W.fill_replicas(w, g, W.alloc_replicas(w, device), 0)
    s = w.schedule
    sched = A.Schedule.make(s.kind, s.peak_lr, s.final_lr, s.warmup_steps,
                            s.total_steps)
    stream = torch.cuda.Stream(device)

    # CPU baseline: the oracle on a bounded sample of the first outer round (rank 0, N=1)
    cpu_baseline = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        step0, h0 = rounds[0]
        sample = calibrated_sample(w, g, v, xs, step0, h0, args.cpu_seconds,
                                   args.comm)
        t1, n = oracle_sample(w, g, v, xs, sample, step0, h0, args.comm)
        cores = host_cores()
        t, n = oracle_sample(w, g, v, xs, sample, step0, h0, args.comm,
                             threads=cores)
        cpu_baseline = {"value": (n / w.numel) / t, "unit": UNIT, "cores": cores,
                        "kind": "oracle",
                        "sample": f"first {n} of {w.numel} parameters x "
                                  f"{w.M} workers of one round in {cores} "
                                  f"concurrent slices ({t:.2f} s), scaled to "
                                  f"a full round",
                        "single_core": {"value": (n / w.numel) / t1,
                                        "sample": f"the same {n} parameters "
                                                  f"on one thread ({t1:.1f} s)"}}

    opts = A.default_opts(time_kernel=1, pass_=PASSES[args.pass_],
                          wait=WAITS[args.wait])
    parts = W.tensor_sizes(w)
    step_ms, kern_ms, statuses = [], [], []
    ev = [(torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in rounds]

    l2 = l2_bytes(device)
    flush_buf = None
    if needs_l2_flush(footprint_bytes(w), l2):
        flush_buf = torch.empty(2 * l2 // 4, dtype=torch.float32, device=device)

    def one_round(k):
        step, hsel = rounds[k]
        if k > 0:
            with torch.cuda.stream(stream):
                W.fill_replicas(w, g, xs, k)      # untimed: the inner loops
        if flush_buf is not None:
            with torch.cuda.stream(stream):
                flush_buf.fill_(float(k))         # untimed: evict the L2
        ev[k][0].record(stream)
        if args.comm == "int8":
            st = A.sync_int8(g, v, xs, parts=parts, H_sel=hsel,
                             H_base=w.H_base, step=step, schedule=sched,
                             outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                             opts=opts, stream=stream)
        else:
            st = A.sync(g, v, xs, H_sel=hsel, H_base=w.H_base, step=step,
                        schedule=sched, outer_lr=w.outer_lr,
                        outer_beta=w.outer_beta, opts=opts, stream=stream)
        ev[k][1].record(stream)
        return st

    for k in range(args.warmup):
        one_round(k)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    st_first = None
    with ClockSampler(device.index) as clocks:
        for k in range(args.warmup, args.warmup + args.steps):
            st = one_round(k)
            st_first = st_first or st
            statuses.append(st["status"])
            kern_ms.append(st["kernel_ms"])
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    for k in range(args.warmup, args.warmup + args.steps):
        step_ms.append(ev[k][0].elapsed_time(ev[k][1]))

    kernel_name = {2: "sync_tma_kernel", 3: "int8_split_kernels",
                   4: "int8_fused_kernel", 5: "sync_tile_kernel"}.get(st_first.get("pass_used"),
                                               "sync_kernel")
    # median over the timed rounds (each rank), then the slowest rank
    ms_step_mean = reduce_max(statistics.mean(step_ms), world, device)
    ms_step = reduce_max(statistics.median(step_ms), world, device)
    ms_kern = reduce_max(statistics.median(kern_ms), world, device)
    value = job_value(1.0, ms_step / 1e3, world)
    peak, peak_kind = hbm_peak()
    achieved = w.bytes_per_round() / (ms_kern / 1e3) / 1e9

    # end to end through the C ABI with host buffers: H2D of the round's
    # inputs from pinned memory, the round, D2H of theta' and v'
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, w, g, v, xs, sched, stream, rounds, world, device,
                      parts if args.comm == "int8" else None)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms_step, "ms_per_step_stat": "median",
            "ms_per_step_mean": ms_step_mean, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None,
            # arithmetic type of the path; the replicas are stored as below
            "dtype": "f32", "replica_dtype": w.dtype,
            "data": "synthetic (seeded; Llama-shaped parameter set, "
                    "shared/private drift noise)",
            "config": dict(config_block(w), comm=args.comm,
                           l2=l2_note(w, l2), wait=args.wait),
            "rounds_per_s_per_gpu": 1e3 / ms_step,
            "elem_per_s": value * w.numel * w.M,
            "kernel_ms": ms_kern, "kernel_ms_stat": "median",
            "hbm_gbs": achieved,
            "frac_of_nominal_8000": achieved / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak,
                         "peak_source": peak_kind,
                         "traffic": recorded_traffic(w.name, kernel_name),
                         "kernel": kernel_name,
                         "occupancy": recorded_occupancy(w.name, kernel_name),
                         "algorithmic_bytes_per_launch": w.bytes_per_round()},
            "cpu_baseline": cpu_baseline,
            "e2e": e2e,
            # the split INT8 round is two kernels (block scales, then apply)
            "gpu_launches": args.steps * (2 if kernel_name == "int8_split_kernels"
                                          else 1),
            "clocks": clocks.summary(),
            "status_ok": all(s_ in (A.OK,) for s_ in statuses),
            "wall_s_timed_loop": t_wall,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_e2e(args, w, g, v, xs, sched, stream, rounds, world, device,
            int8_parts=None):
    """The metric end to end with the state in pinned host memory.  The
    plain round goes through aloco_sync_host (the library streams theta, v
    and the endpoints to the GPU and theta', v' back in overlapped chunks);
    the INT8 round copies the inputs in, calls aloco_sync_int8 and copies
    theta', v' out."""
    import torch
    from paper_2609_36662_gb300 import aloco as A
    from paper_2609_36662_gb300 import workloads as W
    rbytes = w.replica_bytes()
    h2d = w.numel * (8 + w.M * rbytes)
    d2h = w.numel * 8
    # pinned host state: theta, v and the endpoints (theta', v' come back
    # into theta, v); the INT8 leg copies theta', v' out to two more arrays
    pinned = h2d + (d2h if int8_parts is not None else 0)
    mem = host_memory()
    local = ranks_on_host()
    budget = pinned_budget(mem, local)
    # every rank decides the same way, so all take the e2e leg or none do
    skip = 1.0 if (budget and pinned > budget) else 0.0
    if world > 1:
        skip = reduce_max(skip, world, device)
    if skip:
        return {"value": None, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "pinned_bytes": pinned, **mem,
                "ranks_on_host": local,
                "skipped": f"the pinned host state ({pinned / 1e9:.1f} GB per "
                           f"rank) exceeds this rank's share of half of the "
                           f"host memory available ({budget / 1e9:.1f} GB)"}
    t_pin = time.perf_counter()
    hg = torch.empty(w.numel, dtype=torch.float32, pin_memory=True)
    hv = torch.empty(w.numel, dtype=torch.float32, pin_memory=True)
    hx = [torch.empty(w.numel, dtype=W.replica_dtype(w), pin_memory=True)
          for _ in range(w.M)]
    if int8_parts is not None:
        og = torch.empty(w.numel, dtype=torch.float32, pin_memory=True)
        ov = torch.empty(w.numel, dtype=torch.float32, pin_memory=True)
    t_pin = time.perf_counter() - t_pin
    W.fill_replicas(w, g, xs, 0)
    hg.copy_(g)
    hv.copy_(v)
    for a, b in zip(hx, xs):
        a.copy_(b)
    ms = []
    n_total = args.e2e_warmup + args.e2e_steps
    for k in range(n_total):
        step, hsel = rounds[k % len(rounds)]
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        if int8_parts is None:
            # theta' and v' come back into hg, hv (the next round's inputs)
            A.sync_host(hg, hv, hx, H_sel=hsel, H_base=w.H_base, step=step,
                        schedule=sched, outer_lr=w.outer_lr,
                        outer_beta=w.outer_beta, stream=stream)
        else:
            with torch.cuda.stream(stream):
                g.copy_(hg, non_blocking=True)
                v.copy_(hv, non_blocking=True)
                for a, b in zip(xs, hx):
                    a.copy_(b, non_blocking=True)
            A.sync_int8(g, v, xs, parts=int8_parts, H_sel=hsel,
                        H_base=w.H_base, step=step, schedule=sched,
                        outer_lr=w.outer_lr, outer_beta=w.outer_beta,
                        stream=stream)
            with torch.cuda.stream(stream):
                og.copy_(g, non_blocking=True)
                ov.copy_(v, non_blocking=True)
        e1.record(stream)
        e1.synchronize()
        if k >= args.e2e_warmup:
            ms.append(e0.elapsed_time(e1))
    m = reduce_max(statistics.median(ms), world, device)
    out = {"value": job_value(1.0, m / 1e3, world), "unit": UNIT,
           "ms_per_step": m, "ms_per_step_stat": "median",
           "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h + 8 * (w.M + 2),
           "steps": args.e2e_steps,
           "api": "aloco_sync_host" if int8_parts is None else
                  "copies + aloco_sync_int8",
           "pinned_bytes": pinned, "pin_alloc_s": t_pin,
           "host_ram_bytes": mem["host_ram_bytes"]}
    del hg, hv, hx
    return out


# ----------------------------------------------------------- sharded mode

def run_shard(args, w):
    """The round over a vector cut into contiguous shards at generator-chunk
    boundaries (aloco_sync_shard on each, aloco_combine_partials in shard
    order).  One process: --shards G shards run one after another on the one
    GPU.  Under torchrun: rank r holds and runs shard r of WORLD_SIZE shards,
    and the ranks all-gather their partials (one small struct each) over
    NCCL before combining them, so every rank obtains the same D_t and C_t.
    A step is one whole round: every shard this rank holds and the exchange,
    timed with CUDA events on the launch stream (the all-gather is enqueued
    on it), then the host combine; the value is whole rounds per second
    (total work fixed as ranks are added: strong scaling)."""
    import torch
    from paper_2609_36662_gb300 import aloco as A
    from paper_2609_36662_gb300 import workloads as W

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", torch.cuda.current_device())
    A.load()
    G = world if world > 1 else max(1, args.shards)
    mine = [rank] if world > 1 else list(range(G))
    rounds = W.steps_of_rounds(w, args.warmup + args.steps)
    pieces = []
    for k in mine:
        c_lo, c_hi = W.shard_chunks(w, G, k)
        g = W.make_global(w, device, chunks=(c_lo, c_hi))
        v = torch.zeros_like(g)
        xs = [torch.empty(g.numel(), dtype=W.replica_dtype(w), device=device)
              for _ in range(w.M)]
        W.fill_replicas(w, g, xs, 0, c_lo, c_hi)
        pieces.append((c_lo, c_hi, g, v, xs))
    s = w.schedule
    sched = A.Schedule.make(s.kind, s.peak_lr, s.final_lr, s.warmup_steps,
                            s.total_steps)
    stream = torch.cuda.Stream(device)
    opts = A.default_opts(time_kernel=1, pass_=PASSES[args.pass_],
                          wait=WAITS[args.wait])
    step_ms, host_ms, kern_ms, statuses, D, C = [], [], [], [], [], []

    def one_round(k):
        step, hsel = rounds[k]
        if k > 0:
            with torch.cuda.stream(stream):
                for c_lo, c_hi, g, v, xs in pieces:
                    W.fill_replicas(w, g, xs, k, c_lo, c_hi)   # untimed
        stream.synchronize()
        if world > 1:
            torch.distributed.barrier()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        e0.record(stream)
        blobs, ms = [], 0.0
        for _, _, g, v, xs in pieces:
            rc, part = A.sync_shard(g, v, xs, H_sel=hsel, H_base=w.H_base,
                                    step=step, schedule=sched,
                                    outer_lr=w.outer_lr,
                                    outer_beta=w.outer_beta, opts=opts,
                                    stream=stream)
            blobs.append(part.to_bytes())
            ms += max(part.kernel_ms, 0.0)
        if world > 1:
            with torch.cuda.stream(stream):
                blobs = gather_partials(blobs[0], world, device)
        e1.record(stream)
        e1.synchronize()
        st = A.combine_partials([A.Partials.from_bytes(b) for b in blobs])
        t1 = time.perf_counter()
        return e0.elapsed_time(e1), (t1 - t0) * 1e3, ms, st

    for k in range(args.warmup):
        one_round(k)
    torch.cuda.synchronize()
    with ClockSampler(device.index) as clocks:
        for k in range(args.warmup, args.warmup + args.steps):
            t, th, ms, st = one_round(k)
            step_ms.append(t)
            host_ms.append(th)
            kern_ms.append(ms)
            statuses.append(st["status"])
            D.append(st["D"])
            C.append(st["C"])
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    ms_step = reduce_max(statistics.median(step_ms), world, device)
    ms_kern = reduce_max(statistics.median(kern_ms), world, device)
    peak, peak_kind = hbm_peak()
    # bytes this rank's shards move in one round, over their kernel time
    my_bytes = sum(g.numel() for _, _, g, _, _ in pieces) * \
        (2 * (8 + w.M * w.replica_bytes()))
    achieved = my_bytes / (ms_kern / 1e3) / 1e9 if ms_kern > 0 else None
    if rank == 0:
        line = {
            "metric": METRIC, "value": 1e3 / ms_step, "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms_step, "ms_per_step_stat": "median",
            "ms_per_step_host": statistics.median(host_ms),
            "higher_is_better": True, "scaling": "strong",
            "vs_baseline": None, "dtype": "f32", "replica_dtype": w.dtype,
            "data": "synthetic (seeded; Llama-shaped parameter set, "
                    "shared/private drift noise)",
            "config": dict(config_block(w), comm="fp32",
                           parallelism=(f"shard{G}" if world > 1 else
                                        f"{G} shards in sequence on one GPU"),
                           shard_elems=[g.numel() for _, _, g, _, _ in pieces]
                           if world == 1 else None),
            "kernel_ms": ms_kern, "kernel_ms_stat": "median",
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                         "unit": "GB/s",
                         "frac": achieved / peak if achieved else None,
                         "peak_source": peak_kind, "traffic": None,
                         "kernel": "shard kernels (rank 0)",
                         "algorithmic_bytes_per_launch": my_bytes},
            "cpu_baseline": None, "e2e": None,
            "gpu_launches": args.steps * len(pieces),
            "clocks": clocks.summary(),
            "status_ok": all(x == A.OK for x in statuses),
            "D_last": D[-1], "C_last": C[-1],
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


# ------------------------------------------------------ inner AdamW mode

ADAMW_METRIC = ("inner AdamW steps/s (all M replicas) and achieved HBM GB/s "
                "(fraction of GB300 roofline) at N params × M replicas")
ADAMW_UNIT = "steps/s"
ADAMW_LR, ADAMW_STEP0 = 3e-4, 1200   # a mid-run step of the C4 schedule


def adamw_bytes(w) -> int:
    """Algorithmic HBM bytes of one inner step: per element and replica the
    parameter (read + write), the gradient (read once) and the two fp32
    moments (read + write).  Gradients have the replicas' dtype."""
    r = w.replica_bytes()
    return w.numel * w.M * (3 * r + 16)


def adamw_inputs(w, device, seed=7):
    """Replicas, gradients (the replicas' dtype; norms about 3, so the
    C4 threshold of 1.0 clips them) and moments, drawn on `device`."""
    import torch
    from paper_2609_36662_gb300 import workloads as W
    dt = W.replica_dtype(w)
    gen = torch.Generator(device).manual_seed(seed)
    sc = 3.0 / max(w.numel, 1) ** 0.5

    def draw(scale, dtype, positive=False):
        t = torch.empty(w.numel, dtype=torch.float32, device=device)
        t.normal_(0, 1, generator=gen)
        if positive:
            t.abs_()
        return t.mul_(scale).to(dtype)
    xs = [draw(0.02, dt) for _ in range(w.M)]
    gs = [draw(sc, dt) for _ in range(w.M)]
    m1 = [draw(1e-3 * sc * 30, torch.float32) for _ in range(w.M)]
    m2 = [draw((sc * 30) ** 2 * 1e-3, torch.float32, True) for _ in range(w.M)]
    return xs, gs, m1, m2


def adamw_oracle_sample(w, xs, gs, m1, m2, elems, threads: int = 1):
    """Time the oracle's AdamW step, as it stands, on the first `elems`
    elements of every replica; with threads > 1 in that many concurrent
    slices (each clipping by its own slice's norm: the same work).  Returns
    (seconds, elements)."""
    import numpy as np
    import torch
    import oracle as O
    n = min(elems, w.numel)

    def host(t):
        t = t[:n].cpu()
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().view(np.uint16)
        return t.numpy()
    dt = O.F32 if w.dtype == "f32" else O.BF16
    hx, hg = [host(t) for t in xs], [host(t) for t in gs]
    h1, h2 = [host(t) for t in m1], [host(t) for t in m2]

    def fn(a, b):
        O.adamw_step([x[a:b] for x in hx], dt, [x[a:b] for x in hg], dt,
                     [x[a:b] for x in h1], [x[a:b] for x in h2], ADAMW_LR, 0.9,
                     0.95, 1e-8, 0.1, 1.0, ADAMW_STEP0)
    t0 = time.perf_counter()
    run_sliced(fn, slice_cuts(n, threads), threads)
    return time.perf_counter() - t0, n


def adamw_calibrated(w, xs, gs, m1, m2, target_s):
    t, n = adamw_oracle_sample(w, xs, gs, m1, m2, min(w.numel, 1 << 18))
    want = int(target_s / max(t / n, 1e-12))
    return max(1 << 14, min(w.numel, want))


def adamw_config(w):
    from paper_2609_36662_gb300 import workloads as W
    return {"workload": w.name, "mode": "adamw", "N": w.numel, "M": w.M,
            "param_dtype": w.dtype, "grad_dtype": w.dtype,
            "moment_dtype": "f32",
            "settings": "C4: lr 3e-4 at step 1200, betas (0.9, 0.95), eps 1e-8, "
                        "weight decay 0.1, clipping 1.0",
            "bytes_per_step": adamw_bytes(w),
            "l2": f"no flush: each step moves {adamw_bytes(w) / 1e9:.1f} GB "
                  "> 129 MB L2",
            "parallelism": "replicas only"}


def run_adamw_reference(args, w):
    from paper_2609_36662_gb300 import workloads as W
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    import torch
    small = W.small(min(w.numel, 1 << 22), w.M, w.dtype)
    xs, gs, m1, m2 = adamw_inputs(small, "cpu")
    sample = adamw_calibrated(small, xs, gs, m1, m2, args.ref_step_seconds)
    cores = host_cores()
    times = []
    for k in range(args.warmup + args.steps):
        t, n = adamw_oracle_sample(small, xs, gs, m1, m2, sample, threads=cores)
        if k >= args.warmup:
            times.append(t)
    sec = statistics.median(times) * w.numel / sample
    value = 1.0 / sec
    line = {"impl": "reference", "metric": ADAMW_METRIC, "value": value,
            "unit": ADAMW_UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": sec * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "replica_dtype": w.dtype, "data": "synthetic",
            "config": adamw_config(w),
            "cpu_baseline": {"value": value, "unit": ADAMW_UNIT, "cores": cores,
                             "kind": "oracle",
                             "sample": f"first {sample} elements of each of "
                                       f"{w.M} replicas per step in {cores} "
                                       f"concurrent slices, scaled to "
                                       f"{w.numel}"},
            "e2e": {"value": value, "unit": ADAMW_UNIT,
                    "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_adamw(args, w):
    """Time inner AdamW steps on all replicas (the same gradients every
    step; parameters and moments evolve)."""
    import torch
    from paper_2609_36662_gb300 import aloco as A
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", torch.cuda.current_device())
    A.load()
    xs, gs, m1, m2 = adamw_inputs(w, device)
    stream = torch.cuda.Stream(device)
    cpu_baseline = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = adamw_calibrated(w, xs, gs, m1, m2, args.cpu_seconds)
        t1, n = adamw_oracle_sample(w, xs, gs, m1, m2, sample)
        cores = host_cores()
        t, n = adamw_oracle_sample(w, xs, gs, m1, m2, sample, threads=cores)
        cpu_baseline = {"value": (n / w.numel) / t, "unit": ADAMW_UNIT,
                        "cores": cores, "kind": "oracle",
                        "sample": f"first {n} of {w.numel} elements of each of "
                                  f"{w.M} replicas in {cores} concurrent "
                                  f"slices ({t:.2f} s), scaled to a full step",
                        "single_core": {"value": (n / w.numel) / t1,
                                        "sample": f"the same elements on one "
                                                  f"thread ({t1:.1f} s)"}}
    opts = A.default_opts()
    ev = [(torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True))
          for _ in range(args.warmup + args.steps)]
    # "given": the gradients' norms are known to the caller (taken once from
    # a regular step here), and the one-pass aloco_adamw_step_normed runs
    norms = None
    if args.adamw_norms == "given":
        norms = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(lr=ADAMW_LR,
                                                         step=ADAMW_STEP0),
                             opts=opts, stream=stream)["grad_norm"]

    def one_step(k):
        cfg = A.adamw_cfg(lr=ADAMW_LR, step=ADAMW_STEP0 + k)
        ev[k][0].record(stream)
        A.adamw_step(xs, gs, m1, m2, cfg, opts=opts, stream=stream,
                     want_stats=False, grad_norms=norms)
        ev[k][1].record(stream)

    for k in range(args.warmup):
        one_step(k)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(device.index) as clocks:
        for k in range(args.warmup, args.warmup + args.steps):
            one_step(k)
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    ms = statistics.median(ev[k][0].elapsed_time(ev[k][1])
                           for k in range(args.warmup, args.warmup + args.steps))
    ms = reduce_max(ms, world, device)
    st = A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(lr=ADAMW_LR, step=ADAMW_STEP0),
                      opts=opts, stream=stream)
    value = job_value(1.0, ms / 1e3, world)
    peak, peak_kind = hbm_peak()
    achieved = adamw_bytes(w) / (ms / 1e3) / 1e9

    e2e = None
    if not args.no_e2e:
        # the step's inputs from pinned host memory (the M gradients), the
        # step, and the per-replica norms read back
        hg = [torch.empty_like(g, device="cpu").pin_memory() for g in gs]
        for a, b in zip(hg, gs):
            a.copy_(b)
        times = []
        for k in range(args.e2e_warmup + args.e2e_steps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            with torch.cuda.stream(stream):
                for a, b in zip(gs, hg):
                    a.copy_(b, non_blocking=True)
            A.adamw_step(xs, gs, m1, m2, A.adamw_cfg(lr=ADAMW_LR,
                                                     step=ADAMW_STEP0 + k),
                         opts=opts, stream=stream)
            e1.record(stream)
            e1.synchronize()
            if k >= args.e2e_warmup:
                times.append(e0.elapsed_time(e1))
        m_e = reduce_max(statistics.median(times), world, device)
        e2e = {"value": job_value(1.0, m_e / 1e3, world), "unit": ADAMW_UNIT,
               "ms_per_step": m_e,
               "h2d_bytes_per_step": sum(g.numel() * g.element_size() for g in gs),
               "d2h_bytes_per_step": 16 * 32, "steps": args.e2e_steps}
    if rank == 0:
        line = {
            "metric": ADAMW_METRIC, "value": value, "unit": ADAMW_UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms, "ms_per_step_stat": "median",
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "replica_dtype": w.dtype,
            "data": "synthetic (seeded replicas, gradients and moments)",
            "config": adamw_config(w),
            "elem_per_s": value * w.numel * w.M,
            "hbm_gbs": achieved,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak,
                         "peak_source": peak_kind,
                         "traffic": (recorded_traffic(w.name, "adamw_kernels")
                                     if norms is None else None),
                         "kernel": ("adamw_kernels" if norms is None
                                    else "adamw_update_kernel"),
                         "occupancy": (recorded_occupancy(w.name, "adamw_kernels")
                                       if norms is None else None),
                         "algorithmic_bytes_per_launch": adamw_bytes(w)},
            "grad_norms": st["grad_norm"], "clip": st["clip"],
            "cpu_baseline": cpu_baseline, "e2e": e2e,
            # two kernels per step (gradient norms, then the update), or the
            # update alone with given norms
            "gpu_launches": (2 if norms is None else 1) * args.steps,
            "grad_norms_source": "computed" if norms is None else "given",
            "clocks": clocks.summary(),
        }
        print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------- whole-interval mode

INTERVAL_METRIC = ("inner steps/s of whole AutoLoCo intervals (H AdamW steps on "
                   "all M replicas, the outer round and the controller) and the "
                   "outer round's share of the interval time")


def run_interval(args, w):
    """Whole intervals on one GPU: the C4 recipe's controller (H_base 500 in
    [250, 750], q_H 50) picks each interval's horizon; an interval is that
    many aloco_adamw_step calls (the same synthetic gradients every step),
    then aloco_sync with the statistics, then aloco_select_interval.  Each
    interval's inner loop and round are timed with CUDA events."""
    import torch
    from paper_2609_36662_gb300 import aloco as A
    from paper_2609_36662_gb300 import workloads as W
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", torch.cuda.current_device())
    A.load()
    xs, gs, m1, m2 = adamw_inputs(w, device)
    g = W.make_global(w, device)
    v = W.make_momentum(w, device)
    for x in xs:
        x.copy_(g.to(x.dtype))
    sched = A.Schedule.make(0, 4e-4, 4e-5, 1000, 50_000)
    ctrl = A.Controller(500, 250, 750, 50, 1000, sched)
    stream = torch.cuda.Stream(device)
    opts = A.default_opts()
    step = 2000                      # past the warm-up of the schedule
    inner_ms, round_ms, hs = [], [], []
    for k in range(args.warmup + args.steps):
        h = ctrl.decision.H_step
        e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        e0.record(stream)
        for i in range(h):
            A.adamw_step(xs, gs, m1, m2,
                         A.adamw_cfg(lr=A.inner_lr_accum(sched, step + i, 1),
                                     step=step + i + 1),
                         opts=opts, stream=stream, want_stats=False)
        e1.record(stream)
        st = A.sync(g, v, xs, H_sel=h, H_base=ctrl.decision.H_ref_step,
                    step=step, schedule=sched, outer_lr=0.7, outer_beta=0.9,
                    opts=opts, stream=stream, raise_on_error=False)
        ctrl.observe(st["D"], st["C"], st["corr"]["lam_sel"], 1024.0 * h, h,
                     step + h)
        e2.record(stream)
        e2.synchronize()
        step += h
        if k >= args.warmup:
            inner_ms.append(e0.elapsed_time(e1))
            round_ms.append(e1.elapsed_time(e2))
            hs.append(h)
    tot_ms = sum(inner_ms) + sum(round_ms)
    tot_ms = reduce_max(tot_ms, world, device)
    value = job_value(float(sum(hs)), tot_ms / 1e3, world)
    if rank == 0:
        line = {
            "metric": INTERVAL_METRIC, "value": value, "unit": "inner steps/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": tot_ms / len(hs), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "replica_dtype": w.dtype,
            "data": "synthetic (seeded replicas, fixed synthetic gradients)",
            "config": dict(adamw_config(w), mode="interval",
                           controller="C4 recipe: H_base 500 in [250, 750], "
                                      "q_H 50, cosine 4e-4 -> 4e-5, warm-up 1000"),
            "intervals": [{"H": h, "inner_ms": a, "round_ms": b}
                          for h, a, b in zip(hs, inner_ms, round_ms)],
            "round_share": sum(round_ms) / (sum(inner_ms) + sum(round_ms)),
            "ms_per_inner_step": sum(inner_ms) / sum(hs),
            "gpu_launches": 2 * sum(hs) + len(hs),
            "cpu_baseline": None, "e2e": None,
        }
        print(json.dumps(line), flush=True)
    return 0


def main(argv=None):
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["cuda", "reference"], default="cuda")
    p.add_argument("--workload", default=None,
                   help="workload name (default: the Llama-style 3B set, "
                        "8 bf16 workers)")
    p.add_argument("--cpu-seconds", type=float, default=10.0)
    p.add_argument("--ref-step-seconds", type=float, default=3.0)
    p.add_argument("--e2e-steps", type=int, default=5)
    p.add_argument("--e2e-warmup", type=int, default=2)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--pass", dest="pass_", choices=sorted(PASSES),
                   default="auto", help="which fused kernel runs the round")
    p.add_argument("--comm", choices=["fp32", "int8"], default="fp32",
                   help="int8: the round with INT8-communicated "
                        "pseudo-gradients (App. G.1)")
    p.add_argument("--mode", choices=["round", "adamw", "interval"],
                   default="round",
                   help="adamw: time the workers' inner AdamW step; interval: "
                        "whole intervals (inner steps, round, controller)")
    p.add_argument("--adamw-norms", choices=["computed", "given"],
                   default="computed",
                   help="--mode adamw: compute the clipping norms (two "
                        "passes) or take them from the caller (one pass)")
    p.add_argument("--wait", choices=sorted(WAITS), default="spin",
                   help="how the round call waits for its kernel: poll the "
                        "published statistics (spin) or sleep on a "
                        "blocking-sync event (block)")
    p.add_argument("--shards", type=int, default=0,
                   help="run the round as shards (aloco_sync_shard + "
                        "aloco_combine_partials): G shards in sequence on "
                        "one GPU, or one shard per rank under torchrun")
    p.add_argument("--list", action="store_true")
    args = p.parse_args(argv)
    table = workloads_by_name()
    if args.list:
        for name, w in table.items():
            print(name, w.numel, w.M, w.dtype, w.bytes_per_round())
        return 0
    if args.warmup < 3 and args.impl == "cuda":
        print("warning: fewer than 3 warm-up rounds", file=sys.stderr)
    name = args.workload or default_workload_name()
    w = table.get(name) or parse_flat(name)
    if w is None:
        p.error(f"unknown workload {name}; --list shows them, or use "
                "flat<N>_m<M>_<f32|bf16>")
    if args.mode == "adamw":
        return (run_adamw_reference(args, w) if args.impl == "reference"
                else run_adamw(args, w))
    if args.mode == "interval":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable":
                              "the interval mode has no reference arm; "
                              "--mode adamw and --mode round do"}))
            return 0
        return run_interval(args, w)
    if args.impl == "reference":
        return run_reference(args, w)
    if args.shards > 0:
        return run_shard(args, w)
    return run_cuda(args, w)


if __name__ == "__main__":
    sys.exit(main())
