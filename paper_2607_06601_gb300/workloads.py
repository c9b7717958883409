"""Seeded synthetic workloads shaped like the TriRoute paper's 160M-1.3B decoders.

This module holds none of the method's arithmetic.  It only draws random numbers
(numpy PCG64, seeded per layer / sequence so that any slice can be regenerated on its
own), rounds inputs to bf16 bit patterns, and describes the five workloads:

  tiny      1 layer, B=2, 4 q / 2 kv heads, d=64, contexts 37 and 130, bits and modes
            uniform, window 32, seed 0 (sequential decode: every position is a query)
  160m      MHA 12x64, 12 layers, B=32, contexts 2048, 1% outlier channels x8,
            bits {16:.10, 8:.30, 4:.40, 2:.20}, modes {full .30, local W=256 .50, skip .20}
  1p3b      MHA 32x64, B=64, contexts ~U[1024, 8192], bits {16:.05, 8:.25, 4:.45, 2:.25}
            plus a 16-bit token at position 0 and every U{10..30} positions after it,
            modes {full .25, local W=512 .55, skip .20}
  gqa_long  32 q / 8 kv heads, d=128, G=64, B=16, contexts 32768,
            bits {16:.05, 4:.45, 2:.50}, modes {full .15, local W=1024 .70, skip .15}
  sweep     24 layers, MHA 32x64, contexts 4096, per-layer maps as 160m, batch 1/8/64/256

The paper's own workloads are Pile / RedPajama decoding with trained 160M-1.3B models
(Sec. 4, Table 2); those datasets and weights are not used.  These tensors stand in
for them with the same shapes: K/V/Q ~ N(0, 1) rounded to bf16, per-token bit-widths
and modes drawn i.i.d. from the stated mixes.  Router decisions are inputs.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

MODE_SKIP, MODE_LOCAL, MODE_FULL = 0, 1, 2
BITS = (2, 4, 8, 16)


def bf16_bits(x) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return the uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    # in 32-bit arithmetic: no finite value or infinity carries out of the word (the
    # largest, 0xFF7FFFFF + 0x8000, stays below 2^32); NaNs are set below
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    out = rounded.astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_to_f32(bits) -> np.ndarray:
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    num_layers: int
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    group_size: int
    window: int
    contexts: tuple            # ("fixed", n) | ("uniform", lo, hi) | ("list", (n0, n1, ...))
    bits_p: tuple              # probabilities of b = 2, 4, 8, 16
    modes_p: tuple             # probabilities of skip, local, full
    seed: int
    outlier_frac: float = 0.0  # fraction of (kv head, dim) channels scaled in K and V
    outlier_scale: float = 8.0
    forced16_gap: tuple | None = None  # (lo, hi): 16-bit renewal process gaps

    def with_(self, **kw) -> "Spec":
        return dataclasses.replace(self, **kw)

    @property
    def max_context(self) -> int:
        kind = self.contexts[0]
        if kind == "fixed":
            return int(self.contexts[1])
        if kind == "uniform":
            return int(self.contexts[2])
        return int(max(self.contexts[1]))


SPECS = {
    "tiny": Spec("tiny", 1, 2, 4, 2, 64, 32, 32, ("list", (37, 130)),
                 (0.25, 0.25, 0.25, 0.25), (1 / 3, 1 / 3, 1 / 3), seed=0),
    "160m": Spec("160m", 12, 32, 12, 12, 64, 32, 256, ("fixed", 2048),
                 (0.20, 0.40, 0.30, 0.10), (0.20, 0.50, 0.30), seed=1, outlier_frac=0.01),
    "1p3b": Spec("1p3b", 1, 64, 32, 32, 64, 32, 512, ("uniform", 1024, 8192),
                 (0.25, 0.45, 0.25, 0.05), (0.20, 0.55, 0.25), seed=2, forced16_gap=(10, 30)),
    "gqa_long": Spec("gqa_long", 1, 16, 32, 8, 128, 64, 1024, ("fixed", 32768),
                     (0.50, 0.45, 0.0, 0.05), (0.15, 0.70, 0.15), seed=3),
    "sweep": Spec("sweep", 24, 64, 32, 32, 64, 32, 256, ("fixed", 4096),
                  (0.20, 0.40, 0.30, 0.10), (0.20, 0.50, 0.30), seed=4, outlier_frac=0.01),
}


def _rng(*key: int) -> np.random.Generator:
    return np.random.default_rng([int(k) for k in key])


def contexts(spec: Spec) -> np.ndarray:
    """Context length (number of positions 0..n-1) of every sequence."""
    kind = spec.contexts[0]
    if kind == "fixed":
        return np.full(spec.batch, spec.contexts[1], dtype=np.int64)
    if kind == "list":
        return np.array(spec.contexts[1], dtype=np.int64)
    lo, hi = spec.contexts[1], spec.contexts[2]
    return _rng(spec.seed, 99).integers(lo, hi + 1, size=spec.batch).astype(np.int64)


def policy(spec: Spec, layer: int, seq: int, n: int | None = None):
    """Per-token (bits, modes) of positions 0..n-1 of one sequence at one layer."""
    n = spec.max_context if n is None else n
    r = _rng(spec.seed, layer, seq, 0)
    bits = np.array(BITS, dtype=np.uint8)[r.choice(4, size=spec.max_context, p=spec.bits_p)]
    modes = r.choice(3, size=spec.max_context, p=spec.modes_p).astype(np.uint8)
    if spec.forced16_gap is not None:
        lo, hi = spec.forced16_gap
        gaps = r.integers(lo, hi + 1, size=spec.max_context // lo + 1)
        starts = np.concatenate([[0], np.cumsum(gaps)])
        bits[starts[starts < spec.max_context]] = 16
    return bits[:n].copy(), modes[:n].copy()


def head_policy(spec: Spec, layer: int, seq: int, n: int | None = None):
    """Per-token bits and per-(token, query head) modes [n][Hq] of positions 0..n-1 (the
    paper's default granularity, Sec. 3.2(A)): bits as policy(), every head's mode drawn
    i.i.d. from the workload's mode mix."""
    n = spec.max_context if n is None else n
    bits, _ = policy(spec, layer, seq, n)
    r = _rng(spec.seed, layer, seq, 3)
    modes = r.choice(3, size=(spec.max_context, spec.num_q_heads), p=spec.modes_p).astype(np.uint8)
    return bits, modes[:n].copy()


def outlier_channels(spec: Spec, layer: int) -> np.ndarray:
    """Flat (kv head * d + dim) indices of the outlier channels of a layer."""
    if spec.outlier_frac <= 0:
        return np.zeros(0, dtype=np.int64)
    total = spec.num_kv_heads * spec.head_dim
    count = math.ceil(spec.outlier_frac * total)
    return np.sort(_rng(spec.seed, layer, 7).choice(total, size=count, replace=False))


def kv(spec: Spec, layer: int, seq: int, p0: int, p1: int):
    """bf16 bits of K and V rows [p1-p0][Hkv][d] for positions p0..p1-1."""
    r = _rng(spec.seed, layer, seq, 1)
    shape = (spec.max_context, spec.num_kv_heads * spec.head_dim)
    k = r.standard_normal(shape, dtype=np.float32)[p0:p1]
    v = r.standard_normal(shape, dtype=np.float32)[p0:p1]
    ch = outlier_channels(spec, layer)
    if ch.size:
        k[:, ch] *= spec.outlier_scale
        v[:, ch] *= spec.outlier_scale
    rs = (p1 - p0, spec.num_kv_heads, spec.head_dim)
    return bf16_bits(k).reshape(rs), bf16_bits(v).reshape(rs)


def q(spec: Spec, layer: int, seq: int, p0: int, p1: int) -> np.ndarray:
    """bf16 bits of query rows [p1-p0][Hq][d] for positions p0..p1-1."""
    r = _rng(spec.seed, layer, seq, 2)
    x = r.standard_normal((spec.max_context, spec.num_q_heads * spec.head_dim),
                          dtype=np.float32)[p0:p1]
    return bf16_bits(x).reshape(p1 - p0, spec.num_q_heads, spec.head_dim)


def q_kv_fast(spec: Spec, layer: int, seq: int, p0: int, p1: int):
    """Like (q, kv) but drawn only for positions p0..p1-1 (a separate stream, so the
    values differ from kv()/q(); used where whole-context draws would be too slow)."""
    r = _rng(spec.seed, layer, seq, 5, p0)
    n = p1 - p0
    k = r.standard_normal((n, spec.num_kv_heads * spec.head_dim), dtype=np.float32)
    v = r.standard_normal((n, spec.num_kv_heads * spec.head_dim), dtype=np.float32)
    qq = r.standard_normal((n, spec.num_q_heads * spec.head_dim), dtype=np.float32)
    ch = outlier_channels(spec, layer)
    if ch.size:
        k[:, ch] *= spec.outlier_scale
        v[:, ch] *= spec.outlier_scale
    rs = (n, spec.num_kv_heads, spec.head_dim)
    return (bf16_bits(qq).reshape(n, spec.num_q_heads, spec.head_dim),
            bf16_bits(k).reshape(rs), bf16_bits(v).reshape(rs))


def pages_needed(spec: Spec, page_size: int, extra_tokens: int = 0, skip_writes_kv: int = 0):
    """Pages each width class needs to hold every sequence of every layer (from the
    actual seeded maps) plus `extra_tokens` more per sequence and class."""
    ctx = contexts(spec)
    need = np.zeros(4, dtype=np.int64)
    for layer in range(spec.num_layers):
        for s in range(spec.batch):
            bits, modes = policy(spec, layer, s, int(ctx[s]))
            stored = np.ones_like(modes, dtype=bool) if skip_writes_kv else modes != MODE_SKIP
            for c, b in enumerate(BITS):
                cnt = int(np.count_nonzero(stored & (bits == b))) + extra_tokens
                need[c] += -(-cnt // page_size)
    return [int(x) for x in need]
