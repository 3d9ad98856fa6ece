"""Seeded synthetic inputs for the outer synchronisation round.

This module only draws inputs: parameter-set layouts shaped like the
paper's Llama-style models, the global weights, and worker replicas that
have drifted from them.  It contains none of the round's arithmetic and is
shared by the CUDA path's tests/benchmark and by the oracle's tests.

Noise model for a replica m of a tensor at layer l:
    x_m = g + sigma_l * (a * s + b * e_m),   s, e_m ~ N(0, 1) per element,
with s shared by all workers and e_m private to worker m.  The shared/
private mix (a, b) sets the aggregation coherence of the round.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import torch

# ------------------------------------------------------------------ layouts


@dataclass(frozen=True)
class LlamaShape:
    layers: int
    d_model: int
    heads: int
    kv_heads: int
    ffn: int
    vocab: int
    tied: bool

    def tensors(self) -> List[Tuple[str, int, int]]:
        """(name, numel, layer index for the noise scale) in packing order:
        embed, [attn_norm, wq, wk, wv, wo, mlp_norm, w_gate, w_up, w_down]
        per layer, final_norm, lm_head (untied only)."""
        d = self.d_model
        head_dim = d // self.heads
        kv = self.kv_heads * head_dim
        out = [("embed", self.vocab * d, 0)]
        for l in range(self.layers):
            out += [
                (f"l{l}.attn_norm", d, l),
                (f"l{l}.wq", d * d, l),
                (f"l{l}.wk", d * kv, l),
                (f"l{l}.wv", d * kv, l),
                (f"l{l}.wo", d * d, l),
                (f"l{l}.mlp_norm", d, l),
                (f"l{l}.w_gate", d * self.ffn, l),
                (f"l{l}.w_up", d * self.ffn, l),
                (f"l{l}.w_down", self.ffn * d, l),
            ]
        out.append(("final_norm", d, self.layers - 1))
        if not self.tied:
            out.append(("lm_head", self.vocab * d, self.layers - 1))
        return out

    def numel(self) -> int:
        return sum(n for _, n, _ in self.tensors())


LLAMA_150M = LlamaShape(layers=12, d_model=768, heads=12, kv_heads=12,
                        ffn=3072, vocab=32000, tied=True)
LLAMA_1B = LlamaShape(layers=22, d_model=2048, heads=32, kv_heads=4,
                      ffn=5632, vocab=32000, tied=False)
LLAMA_3B = LlamaShape(layers=26, d_model=3072, heads=24, kv_heads=8,
                      ffn=8192, vocab=32000, tied=False)
# Llama-3.1-8B (the paper's fine-tuning model) for payload accounting.
LLAMA31_8B = LlamaShape(layers=32, d_model=4096, heads=32, kv_heads=8,
                        ffn=14336, vocab=128256, tied=False)


@dataclass(frozen=True)
class ScheduleSpec:
    kind: int = 0            # 0 cosine + linear warm-up, 1 constant, 2 linear
    peak_lr: float = 4e-4
    final_lr: float = 4e-5
    warmup_steps: int = 1000
    total_steps: int = 20000


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: layout, worker count, replica dtype, noise
    model, inner schedule and the horizons of its rounds."""
    name: str
    numel: int
    M: int
    dtype: str                       # "f32" or "bf16" (replica storage)
    shape: Optional[LlamaShape]      # None for a flat vector
    noise_a: float
    noise_b: float
    sigma: float                     # base noise scale
    per_layer_sigma: bool            # sigma_l = sigma * (l + 1) / layers
    schedule: ScheduleSpec
    start_step: int
    H_base: int
    H_sel: Tuple[int, ...]           # horizon of each round, in order
    seed: int
    outer_lr: float = 0.7
    outer_beta: float = 0.9

    @property
    def rounds(self) -> int:
        return len(self.H_sel)

    def replica_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def bytes_per_round(self) -> int:
        """Algorithmic HBM bytes of one round: global and momentum (fp32)
        and the M replicas, each read once and written once."""
        return 2 * self.numel * (8 + self.M * self.replica_bytes())


def _draw_h_sel(seed: int, rounds: int, choices=(50, 100, 150, 200, 300)):
    gen = torch.Generator().manual_seed(seed)
    idx = torch.randint(0, len(choices), (rounds,), generator=gen)
    return tuple(int(choices[i]) for i in idx.tolist())


def _rising_h_sel(rounds: int = 10):
    # 100 -> 400 in steps of 50 across the rounds
    return tuple(100 + 50 * round(6 * k / (rounds - 1)) for k in range(rounds))


SCHED_20K = ScheduleSpec(0, 4e-4, 4e-5, 1000, 20000)
SCHED_40K = ScheduleSpec(0, 4e-4, 4e-5, 1000, 40000)


def toy_round() -> Workload:
    """2^20 fp32 params, 4 replicas, one round at step 4000."""
    return Workload("toy_2p20_m4_f32", 1 << 20, 4, "f32", None, 0.6, 0.8,
                    1e-3, False, SCHED_20K, 4000, 100, (150,), 0)


def llama_150m(rounds: int = 20) -> Workload:
    """Llama-style 150M set (12 x 768, tied), 8 fp32 replicas, consecutive
    rounds with H_sel drawn by seed from {50, 100, 150, 200, 300}."""
    return Workload("llama150m_m8_f32", LLAMA_150M.numel(), 8, "f32",
                    LLAMA_150M, 0.6, 0.8, 1e-3, True, SCHED_20K, 4000, 100,
                    _draw_h_sel(2, rounds), 2)


def llama_1b() -> Workload:
    """Llama-style 1.1B set, 4 bf16 replicas, low coherence (0.3/0.95)."""
    return Workload("llama1b_m4_bf16", LLAMA_1B.numel(), 4, "bf16", LLAMA_1B,
                    0.3, 0.95, 1e-3, False, SCHED_40K, 15000, 100, (250,), 3)


def flat_500m(M: int) -> Workload:
    """Flat 5e8 fp32 vector, M in {2, 4, 8, 16} replicas."""
    return Workload(f"flat500m_m{M}_f32", 500_000_000, M, "f32", None, 0.6,
                    0.8, 1e-3, False, SCHED_20K, 4000, 100, (200,), 4)


def llama_3b(rounds: int = 10) -> Workload:
    """Llama-style 3B set, 8 bf16 replicas, rounds with H_sel 100 -> 400."""
    return Workload("llama3b_m8_bf16", LLAMA_3B.numel(), 8, "bf16", LLAMA_3B,
                    0.6, 0.8, 1e-3, False, SCHED_40K, 10000, 100,
                    _rising_h_sel(rounds), 5)


def small(numel: int, M: int, dtype: str = "f32", seed: int = 11,
          H_sel: int = 150, H_base: int = 100, a=0.6, b=0.8) -> Workload:
    """A flat vector of arbitrary size for parity tests."""
    return Workload(f"flat{numel}_m{M}_{dtype}", numel, M, dtype, None, a, b,
                    1e-3, False, SCHED_20K, 4000, H_base, (H_sel,), seed)


def all_configs() -> List[Workload]:
    return [toy_round(), llama_150m(), llama_1b()] + \
        [flat_500m(M) for M in (2, 4, 8, 16)] + [llama_3b()]


# --------------------------------------------------------------- generators


def _segments(w: Workload):
    """(start, numel, sigma, is_norm) for each tensor of the layout."""
    if w.shape is None:
        return [(0, w.numel, w.sigma, False)]
    segs, off = [], 0
    for name, n, layer in w.shape.tensors():
        sig = w.sigma * (layer + 1) / w.shape.layers if w.per_layer_sigma \
            else w.sigma
        segs.append((off, n, sig, name.endswith("norm")))
        off += n
    return segs


CHUNK = 1 << 24   # elements per generator chunk (bounds scratch memory)


def _chunk_gen(device, *key):
    """A generator whose seed depends only on `key`, so any chunk of any
    round can be drawn on its own."""
    seed = 0
    for k in key:
        seed = (seed * 1_000_003 + int(k) + 17) % (1 << 62)
    return torch.Generator(device=device).manual_seed(seed)


def n_chunks(w: Workload) -> int:
    return (w.numel + CHUNK - 1) // CHUNK


def make_global(w: Workload, device="cpu", draw: int = 0,
                upto: Optional[int] = None, chunks: Optional[Tuple[int, int]] = None):
    """theta_global ~ N(0, 0.02) (fp32); norm vectors set to 1.0.  `draw`
    selects an independent draw of the same distribution.  With `upto`,
    only the whole generator chunks that cover elements [0, upto) are drawn
    (a prefix of the same vector); with `chunks` = (c_lo, c_hi), only the
    elements of generator chunks c_lo .. c_hi - 1 (a contiguous piece of the
    same vector, starting at element c_lo * CHUNK)."""
    if chunks is None:
        c_lo = 0
        c_hi = n_chunks(w) if upto is None else min(n_chunks(w), n_chunks_upto(upto))
    else:
        c_lo, c_hi = chunks
    base = c_lo * CHUNK
    end = min(w.numel, c_hi * CHUNK)
    g = torch.empty(max(end - base, 0), dtype=torch.float32, device=device)
    key = 0 if draw == 0 else 10_000 + draw
    for c in range(c_lo, c_hi):
        s, e = c * CHUNK, min(w.numel, (c + 1) * CHUNK)
        g[s - base:e - base].normal_(0.0, 0.02,
                                     generator=_chunk_gen(device, w.seed, key, c))
    if w.shape is not None:
        for off, k, _, is_norm in _segments(w):
            lo, hi = max(off, base), min(off + k, end)
            if is_norm and lo < hi:
                g[lo - base:hi - base] = 1.0
    return g


def n_chunks_upto(upto: int) -> int:
    """Generator chunks that cover elements [0, upto)."""
    return (max(upto, 1) + CHUNK - 1) // CHUNK


def make_momentum(w: Workload, device="cpu", upto: Optional[int] = None):
    n = w.numel if upto is None else min(w.numel, n_chunks_upto(upto) * CHUNK)
    return torch.zeros(n, dtype=torch.float32, device=device)


def shard_chunks(w: Workload, shards: int, k: int) -> Tuple[int, int]:
    """Generator chunks [c_lo, c_hi) of shard k when the vector is cut into
    `shards` contiguous pieces at chunk boundaries (near-equal chunk counts;
    a shard may be empty when there are more shards than chunks)."""
    nc = n_chunks(w)
    return nc * k // shards, nc * (k + 1) // shards


def replica_dtype(w: Workload):
    return torch.float32 if w.dtype == "f32" else torch.bfloat16


def alloc_replicas(w: Workload, device="cpu"):
    dt = replica_dtype(w)
    return [torch.empty(w.numel, dtype=dt, device=device) for _ in range(w.M)]


def replica_chunk(w: Workload, g_chunk: torch.Tensor, round_index: int,
                  c: int):
    """The M endpoints of chunk c (elements [c*CHUNK, ...)) for round
    `round_index`, as fp32: x_m = g + sigma_l (a s + b e_m)."""
    device = g_chunk.device
    s = c * CHUNK
    n = g_chunk.numel()
    gen = _chunk_gen(device, w.seed, round_index + 1, c)
    sigma = _sigma_slice(_segments(w), s, s + n, device)
    shared = torch.randn(n, generator=gen, device=device, dtype=torch.float32)
    shared.mul_(w.noise_a)
    out = []
    for _ in range(w.M):
        priv = torch.randn(n, generator=gen, device=device,
                           dtype=torch.float32)
        priv.mul_(w.noise_b).add_(shared).mul_(sigma).add_(g_chunk)
        out.append(priv)
    return out


def fill_replicas(w: Workload, g: torch.Tensor, replicas, round_index: int,
                  c_lo: int = 0, c_hi: Optional[int] = None):
    """Write the endpoints of chunks [c_lo, c_hi) of round `round_index` into
    the replica buffers (stored in the replica dtype; bf16 by round to
    nearest even).  `g` and the buffers cover the same element range, which
    starts at chunk c_lo."""
    c_hi = n_chunks(w) if c_hi is None else c_hi
    base = c_lo * CHUNK
    for c in range(c_lo, c_hi):
        s, e = c * CHUNK, min(w.numel, (c + 1) * CHUNK)
        xs = replica_chunk(w, g[s - base:e - base], round_index, c)
        for x, r in zip(xs, replicas):
            r[s - base:e - base].copy_(x)
    return replicas


def _sigma_slice(segs, s, e, device):
    """Per-element noise scale over [s, e) as a tensor (or a float when one
    scale covers the slice)."""
    parts = []
    for off, n, sig, _ in segs:
        lo, hi = max(off, s), min(off + n, e)
        if lo < hi:
            parts.append((hi - lo, sig))
    if len({p[1] for p in parts}) == 1:
        return float(parts[0][1])
    return torch.cat([torch.full((k,), sig, dtype=torch.float32,
                                 device=device) for k, sig in parts])


def tensor_sizes(w: Workload) -> List[int]:
    """Sizes of the tensor parts of the layout (one part for a flat
    vector)."""
    return [n for _, n, _, _ in _segments(w)]


def tensor_boundaries(w: Workload) -> List[int]:
    """Start offsets of every tensor of the layout (for boundary sampling)."""
    return [off for off, _, _, _ in _segments(w)]


def steps_of_rounds(w: Workload, rounds: Optional[int] = None):
    """Scheduler position s_t and H_sel of each round: s advances by the
    executed horizon."""
    out, s = [], w.start_step
    hs = w.H_sel if rounds is None else tuple(
        w.H_sel[k % len(w.H_sel)] for k in range(rounds))
    for h in hs:
        out.append((s, h))
        s += h
    return out
