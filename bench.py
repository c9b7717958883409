#!/usr/bin/env python
"""Decode-attention effective HBM GB/s of the TriRoute serving path on GB300.

One step = one decode step of the whole hot path for one batch: at every layer, the
batch's new tokens are appended (quantise-on-write at each token's bit-width) and each
token's query attends in its own mode (skip / local / full) over the mixed-precision
paged cache.  Default workload: the 160M-scale decoder (12 layers, MHA 12 x 64,
batch 32, 2048-token contexts, window 256, seeded bit / mode mixes).

The cache holds R replicas of the batch (R * 32 sequences with their own seeded maps);
step i serves replica i % R, so each sequence grows by at most 32 tokens over the run
and consecutive steps never re-read the same cache lines (every step moves more bytes
than L2 holds).  Steps are captured as CUDA graphs; the timed region replays K of them.

value  = algorithmic attention bytes of the K steps / device time of the K steps
         (codes + fp16 scale/zero + slot positions + page-table entries of the stored
         keys in each non-skip query's range, plus Q and O rows)
e2e    = the same, through the C ABI with host buffers: pinned H2D of every step's
         inputs and D2H of every step's outputs inside the timed region (each step a
         CUDA graph of copies and API calls; `eager_value`: the same steps called one by
         one from Python)
roofline: the dominant kernel is the trr_decode_attn call (one attention kernel);
         achieved = its algorithmic bytes per call / its average duration from CUDA
         event nodes placed around each call in a second, instrumented replay.
routed : the same step driven by router logits (Sec. 3.8 hard decisions): per layer
         trr_route_decisions (cost totals of the executed policy, Sec. 3.5),
         trr_kv_append_routed and trr_decode_attn_routed, with logits whose arg max is
         the workload's seeded bits and modes; plus one prefill-sized
         trr_route_decisions call (2^22 tokens) against the HBM roofline.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import math
import os
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-attention effective HBM GB/s and % of GB300 peak; attended KV tokens/s"
UNIT = "GB/s"
PAGE = 32  # default page size (tokens); --page-size overrides
BITS = (2, 4, 8, 16)


# --------------------------------------------------------------------------- bytes --

def token_bytes(d, G):
    """Bytes of one stored token of one KV head (K + V) per width class."""
    return [2 * (d * b // 8) + 2 * (d // G) * 4 for b in BITS[:3]] + [4 * d]


class Accounting:
    """Algorithmic bytes / attended keys of decode queries, from the seeded maps."""

    def __init__(self, spec, d, G, Hq, Hkv, window, P=PAGE, skip_writes_kv=0):
        self.tokb = np.array(token_bytes(d, G), dtype=np.int64)
        self.Hq, self.Hkv, self.d, self.window, self.P = Hq, Hkv, d, window, P
        self.swk = int(skip_writes_kv)  # 1: skip tokens store KV too

    def query(self, bits_row, modes_row, t):
        """(bytes, attended keys, pages) of one query at position t of one sequence
        (the token at t already appended)."""
        m = int(modes_row[t])
        qo = 2 * self.Hq * self.d
        if m == 0:
            return qo, 0, 0                           # only the zero O row is written
        lo = 0 if m == 2 else max(0, t - self.window + 1)
        stored = (modes_row[:t + 1] != 0) | bool(self.swk)
        b_row = bits_row[:t + 1]
        total, keys, pages = 2 * qo, 0, 0
        for c, b in enumerate(BITS):
            sel = stored & (b_row == b)
            before = int(np.count_nonzero(sel[:lo]))
            n_in = int(np.count_nonzero(sel[lo:]))
            if n_in:
                i0, i1 = before, before + n_in
                pages += (i1 - 1) // self.P - i0 // self.P + 1
            keys += n_in
            total += n_in * (int(self.tokb[c]) * self.Hkv + 4)
        total += 4 * pages
        return total, keys, pages

    def query_heads(self, bits_row, modes_rows, t):
        """(bytes, attended keys, pages) of one query with per-head modes (modes_rows
        [T][Hq]): per KV head, the payload of the keys that store it in the widest range
        of its reading heads; once per key in the query's widest range its slot position,
        per page its page-table entry and the presence masks of the KV heads read; Q rows
        of the heads that read, every O row.  Keys are counted per KV head / Hkv."""
        mrow = modes_rows[t]
        g = self.Hq // self.Hkv
        qo = 2 * self.Hq * self.d
        if not mrow.any():
            return qo, 0, 0
        lo_q = 0 if (mrow == 2).any() else max(0, t - self.window + 1)
        b_row = bits_row[:t + 1]
        stored = (modes_rows[:t + 1] != 0).reshape(t + 1, self.Hkv, g).any(2) | bool(self.swk)  # [t+1][Hkv]
        took = stored.any(1)
        total = qo + 2 * self.d * int(np.count_nonzero(mrow))
        keys = pages = nkv = 0
        for j in range(self.Hkv):
            mj = mrow[j * g:(j + 1) * g]
            if not mj.any():
                continue
            nkv += 1
            lo = 0 if (mj == 2).any() else max(0, t - self.window + 1)
            for c, b in enumerate(BITS):
                n_in = int(np.count_nonzero(stored[lo:, j] & (b_row[lo:] == b)))
                keys += n_in
                total += n_in * int(self.tokb[c])
        for c, b in enumerate(BITS):
            sel = took & (b_row == b)
            before = int(np.count_nonzero(sel[:lo_q]))
            n_in = int(np.count_nonzero(sel[lo_q:]))
            if n_in:
                i0, i1 = before, before + n_in
                pages += (i1 - 1) // self.P - i0 // self.P + 1
            total += 4 * n_in
        total += pages * (4 + 8 * nkv)
        return total, keys / self.Hkv, pages


# ------------------------------------------------------------------ clocks (NVML) --

class ClockSampler:
    """Samples SM clock and clock-event reasons of this GPU while running."""
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, uuid: str | None, period_s=0.002):
        self.samples, self.reasons, self.max_mhz = [], set(), None
        self.period, self.ok = period_s, False
        self._stop = threading.Event()
        try:
            self.nv = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nv.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if uuid:
                r = self.nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(self.h))
            else:
                r = self.nv.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(self.h))
            if r != 0:
                return
            mx = ctypes.c_uint()
            if self.nv.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = int(mx.value)
            self.ok = True
        except OSError:
            pass

    def _run(self):
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        get_rs = getattr(self.nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            self.nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if self.nv.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(clk)) == 0:
                self.samples.append(int(clk.value))
            if get_rs(self.h, ctypes.byref(rs)) == 0:
                for bit, name in self.REASONS.items():
                    if rs.value & bit:
                        self.reasons.add(name)
            time.sleep(self.period)

    def __enter__(self):
        if self.ok:
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()
        return self

    def __exit__(self, *a):
        if self.ok:
            self._stop.set()
            self._t.join()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                    "samples": 0}
        return {"sm_mhz": float(statistics.median(self.samples)), "sm_max_mhz": self.max_mhz,
                "reasons": sorted(self.reasons), "samples": len(self.samples)}


# ------------------------------------------------------- CUDA event nodes (cudart) --

class CudaRt:
    """cudaEventRecordWithFlags(External) places timing events inside captured graphs."""

    def __init__(self):
        lib = None
        for name in ("libcudart.so.13", "libcudart.so", "/usr/local/cuda/lib64/libcudart.so"):
            try:
                lib = ctypes.CDLL(name)
                break
            except OSError:
                continue
        if lib is None:
            raise RuntimeError("libcudart not found")
        self.lib = lib
        lib.cudaEventCreateWithFlags.argtypes = [ctypes.POINTER(ctypes.c_void_p), ctypes.c_uint]
        lib.cudaEventRecordWithFlags.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint]
        lib.cudaEventElapsedTime.argtypes = [ctypes.POINTER(ctypes.c_float), ctypes.c_void_p, ctypes.c_void_p]
        lib.cudaEventDestroy.argtypes = [ctypes.c_void_p]

    def event(self):
        e = ctypes.c_void_p()
        assert self.lib.cudaEventCreateWithFlags(ctypes.byref(e), 0) == 0
        return e

    def record_external(self, ev, stream_handle):
        assert self.lib.cudaEventRecordWithFlags(ev, ctypes.c_void_p(stream_handle), 1) == 0

    def elapsed_ms(self, a, b):
        ms = ctypes.c_float()
        assert self.lib.cudaEventElapsedTime(ctypes.byref(ms), a, b) == 0
        return float(ms.value)


# ------------------------------------------------------------------- the workload --

def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def l2_cache_bytes():
    """L2 size of the current device (cudaDevAttrL2CacheSize)."""
    import torch
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    size = getattr(props, "L2_cache_size", 0)
    if size:
        return int(size)
    rt = CudaRt()
    v = ctypes.c_int()
    rt.lib.cudaDeviceGetAttribute(ctypes.byref(v), 89, torch.cuda.current_device())
    return int(v.value)


def expected_step_bytes(spec, ctx, P, swk=0, chunk=1):
    """Expected algorithmic attention bytes of one step (every layer, every sequence) from
    the workload's bit and mode mixes: the replica count is sized from it."""
    tokb = np.array(token_bytes(spec.head_dim, spec.group_size), dtype=np.float64)
    p_bits = np.array(spec.bits_p, dtype=np.float64)
    p_skip, p_local, p_full = spec.modes_p
    stored = 1.0 if swk else 1.0 - p_skip
    per_pos = stored * (float(p_bits @ tokb) * spec.num_kv_heads + 4)
    keys = p_full * ctx.astype(np.float64) + p_local * np.minimum(ctx, spec.window)
    qo = 2 * spec.num_q_heads * spec.head_dim
    per_layer = float(np.sum(keys * per_pos)) + len(ctx) * (qo * (2 - p_skip))
    return per_layer * spec.num_layers * chunk


def expected_cache_bytes(spec, ctx, P, swk=0):
    """Expected page bytes of one replica of the batch over every layer."""
    tokb = np.array(token_bytes(spec.head_dim, spec.group_size), dtype=np.float64)
    stored = 1.0 if swk else 1.0 - spec.modes_p[0]
    per_tok = stored * float(np.array(spec.bits_p) @ tokb) * spec.num_kv_heads
    return float(np.sum(ctx)) * per_tok * spec.num_layers * 1.1


def kernel_source_digest():
    """sha256 (16 hex digits) of the library's CUDA sources (every .cu and .cuh of csrc,
    in name order), with comments and blank space removed (a change of wording does not
    change a kernel)."""
    import glob
    import hashlib
    import re
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_06601_gb300", "csrc")
    for path in sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cuh"))):
        src = open(path).read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


def ncu_traffic(workload):
    """Per-launch DRAM bytes of the attention kernel from the committed ncu summary,
    if it was taken on the current kernel sources (else None)."""
    digest = kernel_source_digest()
    path = os.path.join(ROOT, "profiles", f"attn_kernel_{workload}_traffic.txt")
    try:
        kv = dict(line.split(":", 1) for line in open(path) if ":" in line)
    except OSError:
        return None
    if kv.get("source_sha256_16", "").strip() != digest:
        return None
    try:
        return float(kv["dram_bytes_per_call"])
    except (KeyError, ValueError):
        return None


def rank_spec(spec, rank):
    """Each rank serves its own batches (weak scaling): a rank-specific seed."""
    return spec.with_(seed=spec.seed + 1000 * rank)


def across_ranks(dist, device, ms, *units):
    """The job's time and work over one process per GPU: the MAX of the ranks' timed
    milliseconds and the SUM of their work units (bytes, keys).  No data-path
    collective exists; this is bookkeeping after the timed region."""
    if dist is None:
        return (float(ms), *[float(u) for u in units])
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    u = torch.tensor([float(x) for x in units], dtype=torch.float64, device=device)
    if len(units):
        dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return (float(t.item()), *[float(x) for x in u.tolist()])


def _mix(*xs):
    """A deterministic 31-bit seed from small integers."""
    h = 0x9E3779B9
    for x in xs:
        h = (h * 1000003 + int(x) + 1) & 0xFFFFFFFFFFFF
    return h & 0x7FFFFFFF


class Bench:
    def __init__(self, args, rank=0, world=1):
        import torch
        from paper_2607_06601_gb300 import trr, workloads as wl
        self.torch, self.trr, self.wl = torch, trr, wl
        spec = wl.SPECS[args.workload]
        if args.batch:
            spec = spec.with_(batch=args.batch)
        if args.layers:
            spec = spec.with_(num_layers=args.layers)
        self.spec = rank_spec(spec, rank)
        self.args, self.rank, self.world = args, rank, world
        s = self.spec
        self.L, self.B, self.Hq, self.Hkv, self.d, self.G = (
            s.num_layers, s.batch, s.num_q_heads, s.num_kv_heads, s.head_dim, s.group_size)
        self.window = s.window
        self.head_modes = int(getattr(args, "head_modes", False))
        self.swk = int(getattr(args, "skip_writes_kv", False))
        self.e2e_warm, self.e2e_steps = 2, 2 * min(args.steps, 10)
        # the routed step decides per token: not run with per-head modes
        self.routed_warm, self.routed_steps = (0, 0) if self.head_modes else (2, min(args.steps, 10))
        # the same steps as separate trr_kv_append / trr_decode_attn calls, for comparison
        self.sep_warm, self.sep_steps = 2, min(args.steps, 10)
        if getattr(args, "light", False):  # timed steps and per-call attribution only
            self.e2e_warm = self.e2e_steps = self.routed_warm = self.routed_steps = 0
            self.sep_warm = self.sep_steps = 0
        self.total_steps = (args.warmup + 2 * args.steps + self.e2e_warm + self.e2e_steps + self.routed_warm +
                            self.routed_steps + self.sep_warm + self.sep_steps)
        self.C = max(1, int(getattr(args, "chunk", 1)))  # new tokens (and queries) per sequence per step
        if self.B * self.C > 1024:
            raise SystemExit("batch x chunk must be at most 1024 (one append call per layer)")
        self.grow = 32                                   # tokens a sequence may grow
        self.P = args.page_size or PAGE
        self.acct = Accounting(s, self.d, self.G, self.Hq, self.Hkv, self.window, self.P, self.swk)
        self.ctx = wl.contexts(s)                       # prebuilt context per sequence
        # Replicas: enough that a sequence grows by at most `grow` tokens over the run, and
        # that the steps between two visits of a replica read at least 3 x L2, so that no
        # step finds its bytes in L2 (capped by device memory; a workload too small for
        # that is reported as such).
        self.l2_bytes = l2_cache_bytes()
        self.est_step_bytes = expected_step_bytes(s, self.ctx, self.P, self.swk, self.C)
        r_grow = max(1, math.ceil(self.total_steps * self.C / self.grow))
        r_l2 = math.ceil(3 * self.l2_bytes / max(1.0, self.est_step_bytes))
        cache_per_replica = max(1.0, expected_cache_bytes(s, self.ctx, self.P, self.swk))
        r_mem = max(1, int(getattr(args, "cache_budget_gb", 120.0) * 1e9 // cache_per_replica))
        self.R = max(r_grow, min(r_l2, r_mem, 64))
        self.maxctx = int(self.ctx.max()) + math.ceil(self.total_steps / self.R) * self.C + 1
        self.dev = torch.device("cuda", torch.cuda.current_device())

    # ---- maps
    def maps(self, layer, r):
        wl = self.wl
        bits = np.empty((self.B, self.maxctx), dtype=np.uint8)
        shape = (self.B, self.maxctx, self.Hq) if self.head_modes else (self.B, self.maxctx)
        modes = np.empty(shape, dtype=np.uint8)
        spec = self.spec.with_(contexts=("fixed", self.maxctx))
        draw = wl.head_policy if self.head_modes else wl.policy
        for s in range(self.B):
            bits[s], modes[s] = draw(spec, layer, r * self.B + s, self.maxctx)
        return bits, modes

    def setup(self):
        torch, trr = self.torch, self.trr
        L, B, R = self.L, self.B, self.R
        S = R * B
        self.all_maps = [[self.maps(l, r) for r in range(R)] for l in range(L)]
        caps = np.zeros(4, dtype=np.int64)
        for l in range(L):
            for r in range(R):
                bits, modes = self.all_maps[l][r]
                for s in range(B):
                    stored = (modes[s] != 0).any(-1) if self.head_modes else modes[s] != 0
                    stored = stored | bool(self.swk)
                    for c, b in enumerate(BITS):
                        caps[c] += -(-int(np.count_nonzero(stored & (bits[s] == b))) // self.P) + 1
        self.cache = trr.Cache(L, S, self.Hq, self.Hkv, self.d, self.G, self.P, self.maxctx,
                               [int(c) for c in caps], max_append=1024, max_queries=max(B * self.C, 64),
                               split_bytes=self.args.split_bytes, head_modes=self.head_modes,
                               skip_writes_kv=self.swk)
        # prebuild every sequence's context (untimed), K/V drawn on the device
        gen = torch.Generator(device=self.dev)
        self.prebuild_calls = 0
        for l in range(L):
            chl = torch.tensor(self.wl.outlier_channels(self.spec, l), dtype=torch.long, device=self.dev)
            bits_d = torch.from_numpy(np.concatenate([self.all_maps[l][r][0] for r in range(R)])).to(self.dev)
            modes_d = torch.from_numpy(np.concatenate([self.all_maps[l][r][1] for r in range(R)])).to(self.dev)
            ctx = np.tile(self.ctx, R)
            for p0 in range(0, int(ctx.max()), max(1, 1024 // S)):
                p1 = min(int(ctx.max()), p0 + max(1, 1024 // S))
                pos = torch.arange(p0, p1, device=self.dev, dtype=torch.int32)
                seqs = torch.arange(S, device=self.dev, dtype=torch.int32)
                pp, ss = torch.meshgrid(pos, seqs, indexing="ij")
                keep = pp < torch.from_numpy(ctx).to(self.dev)[ss.long()]
                pp, ss = pp[keep].contiguous(), ss[keep].contiguous()
                for e0 in range(0, pp.numel(), 1024):
                    e1 = min(pp.numel(), e0 + 1024)
                    sp, ps = ss[e0:e1].contiguous(), pp[e0:e1].contiguous()
                    gen.manual_seed(_mix(self.spec.seed, 1, l, p0, e0))
                    k, v = self._kv(e1 - e0, gen, chl)
                    self.cache.append(l, sp, ps, k, v, bits_d[sp.long(), ps.long()].contiguous(),
                                      modes_d[sp.long(), ps.long()].contiguous())
                    self.prebuild_calls += 1
        torch.cuda.synchronize()
        st = self.cache.status()
        if st != 0:
            raise RuntimeError(f"cache build failed: status {st}")
        self.prebuild_launches = 2 * self.prebuild_calls + 1  # + the status kernel
        print(f"prebuild_launches={self.prebuild_launches}", file=sys.stderr, flush=True)
        self.steps = [self._stage(i) for i in range(self.total_steps)]

    def _kv(self, n, gen, ch):
        torch = self.torch
        shape = (n, self.Hkv * self.d)
        k = torch.randn(shape, generator=gen, device=self.dev)
        v = torch.randn(shape, generator=gen, device=self.dev)
        if ch.numel():
            k[:, ch] *= self.spec.outlier_scale
            v[:, ch] *= self.spec.outlier_scale
        return (k.view(n, self.Hkv, self.d).to(torch.bfloat16).contiguous(),
                v.view(n, self.Hkv, self.d).to(torch.bfloat16).contiguous())

    def _stage(self, i):
        """Device inputs and host byte accounting of global step i."""
        torch = self.torch
        r, grow = i % self.R, i // self.R
        gen = torch.Generator(device=self.dev)
        layers = []
        nbytes = keys = 0
        n = self.B * self.C  # entries (and queries) per layer: C consecutive tokens per sequence
        srow = np.repeat(np.arange(self.B), self.C)
        for l in range(self.L):
            bits, modes = self.all_maps[l][r]
            pos = (self.ctx[srow] + grow * self.C + np.tile(np.arange(self.C), self.B)).astype(np.int32)
            seqs = (r * self.B + srow).astype(np.int32)
            b = bits[srow, pos]
            m = modes[srow, pos]
            gen.manual_seed(_mix(self.spec.seed, 2, i, l))
            chl = torch.tensor(self.wl.outlier_channels(self.spec, l), dtype=torch.long, device=self.dev)
            k, v = self._kv(n, gen, chl)
            q = torch.randn((n, self.Hq, self.d), generator=gen, device=self.dev).to(torch.bfloat16)
            acct = self.acct.query_heads if self.head_modes else self.acct.query
            for e in range(n):  # every query sees the chunk's tokens up to its own position
                nb, nk, _ = acct(bits[srow[e]], modes[srow[e]], int(pos[e]))
                nbytes += nb
                keys += nk
            # router logits whose arg max is the seeded decision (the routed step)
            ml = torch.rand((n, 3), generator=gen, device=self.dev) - 2.0
            bl = torch.rand((n, 4), generator=gen, device=self.dev) - 2.0
            if not self.head_modes:
                ml[torch.arange(n, device=self.dev), torch.from_numpy(m.astype(np.int64)).to(self.dev)] = 1.0
            bcls = np.array([BITS.index(int(x)) for x in b], dtype=np.int64)
            bl[torch.arange(n, device=self.dev), torch.from_numpy(bcls).to(self.dev)] = 1.0
            layers.append(dict(
                seqs=torch.from_numpy(seqs).to(self.dev), pos=torch.from_numpy(pos).to(self.dev),
                bits=torch.from_numpy(b).to(self.dev), modes=torch.from_numpy(np.ascontiguousarray(m)).to(self.dev),
                k=k, v=v, q=q, ml=ml.contiguous(), bl=bl.contiguous(),
                out=torch.empty((n, self.Hq, self.d), dtype=torch.bfloat16, device=self.dev)))
        attn_bytes_per_layer = nbytes / self.L
        return dict(layers=layers, bytes=nbytes, keys=keys, attn_bytes_per_layer=attn_bytes_per_layer)

    # ---- one step through the C ABI
    def run_step(self, st, events=None, stream=None, separate=False):
        """Every layer's decode step: one trr_decode_step call (append and attention in
        one kernel), or with `separate` trr_kv_append then trr_decode_attn.  `events`
        brackets the attention of every layer (the whole decode-step call)."""
        c = self.cache
        n = 0
        fused = not separate and self.C == 1 and not self.head_modes and self.B <= 256
        for l, x in enumerate(st["layers"]):
            if fused:
                if events is not None:
                    events[0](l)
                c.decode_step(l, x["seqs"], x["pos"], x["k"], x["v"], x["bits"], x["modes"], x["q"],
                              window_scalar=self.window, out=x["out"], stream=stream)
                n += c.launches()
            else:
                c.append(l, x["seqs"], x["pos"], x["k"], x["v"], x["bits"], x["modes"], stream=stream)
                n += c.launches()
                if events is not None:
                    events[0](l)
                c.decode_attn(l, x["seqs"], x["pos"], x["q"], x["modes"], window_scalar=self.window,
                              out=x["out"], stream=stream)
                n += c.launches()
            if events is not None:
                events[1](l)
        return n

    def run_routed_step(self, st, totals, stream=None):
        """The step driven by router logits: decisions and their cost, then the routed
        append and attention, which take the same decisions in their own kernels."""
        c, trr = self.cache, self.trr
        n = 0
        for l, x in enumerate(st["layers"]):
            trr.trr_route_decisions(x["ml"], x["bl"], x["pos"], self.window, self.Hq, self.d, self.Hkv,
                                    skip_writes_kv=self.swk, totals=totals, stream=stream)
            c.append_routed(l, x["seqs"], x["pos"], x["k"], x["v"], x["bl"], x["ml"], stream=stream)
            n += 1 + c.launches()
            c.decode_attn_routed(l, x["seqs"], x["pos"], x["q"], x["ml"], window_scalar=self.window,
                                 out=x["out"], stream=stream)
            n += c.launches()
        return n

    def capture(self, idx, instrument=None, totals=None, separate=False):
        torch = self.torch
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            with torch.cuda.graph(g, stream=s):
                if totals is not None:
                    launches = self.run_routed_step(self.steps[idx], totals)
                else:
                    launches = self.run_step(self.steps[idx], instrument(idx, s) if instrument else None,
                                             separate=separate)
        torch.cuda.current_stream().wait_stream(s)
        return g, launches


def run_separate(bench, dist, r0):
    """The same decode steps as separate trr_kv_append and trr_decode_attn calls (two
    kernels per layer instead of one trr_decode_step kernel)."""
    if not bench.sep_steps:
        return None
    torch = bench.torch
    graphs = [bench.capture(i, separate=True) for i in range(r0, r0 + bench.sep_warm + bench.sep_steps)]
    for g, _ in graphs[:bench.sep_warm]:
        g.replay()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for g, _ in graphs[bench.sep_warm:]:
        g.replay()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    idx = range(r0 + bench.sep_warm, r0 + bench.sep_warm + bench.sep_steps)
    nbytes = sum(bench.steps[i]["bytes"] for i in idx)
    ms, nbytes = across_ranks(dist, "cuda", ms, nbytes)
    launches = graphs[0][1]
    del graphs
    return {"value": round(nbytes / (ms * 1e-3) / 1e9, 2), "unit": UNIT,
            "ms_per_step": round(ms / bench.sep_steps, 5), "steps": bench.sep_steps,
            "gpu_launches": launches * bench.sep_steps,
            "how": "per layer trr_kv_append then trr_decode_attn (two kernels) instead of one trr_decode_step"}


def run_routed(bench, dist, r0):
    """The routed step (decisions from logits) timed over its own steps, and one
    prefill-sized trr_route_decisions call against the HBM roofline."""
    torch, trr = bench.torch, bench.trr
    totals = torch.zeros(4, dtype=torch.int64, device=bench.dev)
    graphs = [bench.capture(i, totals=totals) for i in range(r0, r0 + bench.routed_warm + bench.routed_steps)]
    launches = graphs[0][1]
    for g, _ in graphs[:bench.routed_warm]:
        g.replay()
    torch.cuda.synchronize()
    totals.zero_()
    if dist:
        dist.barrier()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for g, _ in graphs[bench.routed_warm:]:
        g.replay()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    idx = range(r0 + bench.routed_warm, r0 + bench.routed_warm + bench.routed_steps)
    nbytes = sum(bench.steps[i]["bytes"] for i in idx)
    ms, nbytes = across_ranks(dist, "cuda", ms, nbytes)
    tot = totals.cpu().tolist()
    del graphs

    # one prefill-sized decision call: 2^22 tokens (210 MB of inputs and outputs)
    n = 1 << 22
    gen = torch.Generator(device=bench.dev)
    gen.manual_seed(_mix(bench.spec.seed, 3))
    ml = torch.randn((n, 3), generator=gen, device=bench.dev)
    bl = torch.randn((n, 4), generator=gen, device=bench.dev)
    pos = torch.randint(0, 8192, (n,), generator=gen, device=bench.dev, dtype=torch.int32)
    out = dict(modes=torch.empty(n, dtype=torch.uint8, device=bench.dev),
               bits=torch.empty(n, dtype=torch.uint8, device=bench.dev),
               attn_flops=torch.empty(n, dtype=torch.int64, device=bench.dev),
               kv_bits=torch.empty(n, dtype=torch.int64, device=bench.dev))
    ptot = torch.zeros(4, dtype=torch.int64, device=bench.dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=bench.dev)

    def call():
        trr.trr_route_decisions(ml, bl, pos, bench.window, bench.Hq, bench.d, bench.Hkv, totals=ptot, **out)

    # one call captured as a graph, so that the timed region holds no host marshalling
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            call()
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(3):
        graph.replay()
    times = []
    for _ in range(10):
        flush.fill_(1)  # evict the inputs from L2 between calls (and keep the GPU busy)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        graph.replay()
        b.record()
        torch.cuda.synchronize()
        times.append(a.elapsed_time(b))
    del flush, graph
    us = statistics.median(times) * 1e3
    per_token = 3 * 4 + 4 * 4 + 4 + 1 + 1 + 8 + 8  # logits, position in; decisions, costs out
    gbs = n * per_token / (us * 1e-6) / 1e9
    peak, _ = measured_peaks()
    return {
        "value": round(nbytes / (ms * 1e-3) / 1e9, 2), "unit": UNIT,
        "ms_per_step": round(ms / bench.routed_steps, 5), "steps": bench.routed_steps,
        "gpu_launches": launches * bench.routed_steps,
        "budget": {"attn_flops_frac": round(tot[0] / tot[2], 4) if tot[2] else None,
                   "kv_bits_frac": round(tot[1] / tot[3], 4) if tot[3] else None,
                   "note": "executed cost / dense cost of the timed steps' tokens (Sec. 3.5, App. C)"},
        "route_decisions": {"tokens": n, "us_per_call": round(us, 2), "bytes_per_token": per_token,
                            "achieved_gbs": round(gbs, 1), "peak": peak, "frac": round(gbs / peak, 4),
                            "l2": "256 MB buffer written between calls"},
    }


# The other workloads measured beside the headline (160m) in the default run: name and
# batch (0: the workload's own).
PER_WORKLOAD = (("tiny", 0), ("1p3b", 0), ("gqa_long", 0), ("sweep", 1), ("sweep", 8), ("sweep", 64),
                ("sweep", 256))


def per_workload(args, local):
    """Every other workload's decode steps, timed like the headline: step throughput and
    the trr_decode_attn call against the HBM roofline."""
    import copy
    import gc
    import torch
    peak, peak_kind = measured_peaks()
    out = {}
    for name, batch in PER_WORKLOAD:
        a = copy.copy(args)
        a.workload, a.batch, a.layers, a.light = name, batch, 0, True
        a.steps, a.warmup = args.per_workload_steps, 3
        b = Bench(a)
        b.setup()
        core = timed_steps(b, a.warmup, a.steps, None, local)
        value = core["job_bytes"] / (core["ms"] * 1e-3) / 1e9
        avg_bytes, avg_ms = float(np.mean(core["call_bytes"])), float(np.mean(core["call_ms"]))
        in_stream = core["launches_per_step"] == b.L  # as for the headline
        launch_ms = (core["ms"] / a.steps) / b.L if in_stream else avg_ms
        if in_stream:
            avg_bytes = core["rank_bytes"] / a.steps / b.L
        achieved = avg_bytes / (launch_ms * 1e-3) / 1e9
        key = name if name != "sweep" else f"sweep_b{b.B}"
        out[key] = {
            "workload": f"{b.spec.name}: {b.L} layers, MHA/GQA {b.Hq}/{b.Hkv} x {b.d}, batch {b.B}, contexts "
                        f"{describe_ctx(b)}, window {b.window}, group {b.G}, page {b.P}",
            "value": round(value, 2), "unit": UNIT, "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": round(core["ms"] / a.steps, 5), "bytes_per_step": int(core["job_bytes"] / a.steps),
            "kv_tokens_per_s": round(core["job_keys"] / (core["ms"] * 1e-3), 1),
            "pct_of_8tbs": round(100 * value / 8000.0, 2),
            "gpu_launches": core["launches_per_step"] * a.steps,
            "roofline": {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak, "unit": "GB/s",
                         "frac": round(achieved / peak, 4), "peak_kind": peak_kind,
                         "bytes_per_call": round(avg_bytes), "us_per_call": round(launch_ms * 1e3, 3),
                         "timing": "timed region / launches (one launch per layer)" if in_stream
                         else "event nodes around each call",
                         "us_per_call_bracketed": round(avg_ms * 1e3, 3)},
            "replicas": b.R, "l2": l2_note(b, core["rank_bytes"] / a.steps),
            "clocks": core["clocks"].summary(),
        }
        print(f"per_workload {key}: {out[key]['value']} GB/s, call {launch_ms * 1e3:.2f} us "
              f"({achieved / peak:.3f} of peak)", file=sys.stderr, flush=True)
        del b, core
        gc.collect()
        torch.cuda.empty_cache()
    return out


def device_uuid(local):
    import torch
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        return None


def timed_steps(bench, W, K, dist, local):
    """W warm-up and K timed step graphs (the timed region: CUDA events on the stream,
    clocks sampled during it), then K more steps with event nodes around every
    trr_decode_attn call (the per-call attribution of the roofline)."""
    import torch
    rt = CudaRt()
    graphs = [bench.capture(i) for i in range(W + K)]
    launches_per_step = graphs[0][1]
    for i in range(W):
        graphs[i][0].replay()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(device_uuid(local)) as clocks:
        torch.cuda.synchronize()
        t0.record()
        for i in range(W, W + K):
            graphs[i][0].replay()
        t1.record()
        torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    step_bytes = sum(bench.steps[i]["bytes"] for i in range(W, W + K))
    step_keys = sum(bench.steps[i]["keys"] for i in range(W, W + K))
    ms, job_bytes, job_keys = across_ranks(dist, "cuda", ms, step_bytes, step_keys)
    del graphs

    evs = {}

    def instrument(idx, s):
        def before(l):
            e = rt.event()
            rt.record_external(e, s.cuda_stream)
            evs[(idx, l, 0)] = e

        def after(l):
            e = rt.event()
            rt.record_external(e, s.cuda_stream)
            evs[(idx, l, 1)] = e
        return before, after

    base = W + K
    igraphs = [bench.capture(i, instrument) for i in range(base, base + K)]
    torch.cuda.synchronize()
    for g, _ in igraphs:
        g.replay()
    torch.cuda.synchronize()
    call_ms, call_bytes = [], []
    for i in range(base, base + K):
        for l in range(bench.L):
            call_ms.append(rt.elapsed_ms(evs[(i, l, 0)], evs[(i, l, 1)]))
            call_bytes.append(bench.steps[i]["attn_bytes_per_layer"])
    del igraphs
    return dict(ms=ms, job_bytes=job_bytes, job_keys=job_keys, rank_bytes=step_bytes,
                launches_per_step=launches_per_step, clocks=clocks, call_ms=call_ms, call_bytes=call_bytes)


def l2_note(bench, rank_bytes_per_step):
    """How the timed steps relate to L2: the bytes read between two visits of a replica."""
    rot = bench.R * rank_bytes_per_step
    mb = bench.l2_bytes / 1e6
    if rot >= 3 * bench.l2_bytes:
        return (f"inputs larger than L2: {bench.R} replicas rotate, {rank_bytes_per_step / 1e6:.0f} MB per step, "
                f"{rot / 1e6:.0f} MB between visits of a replica = {rot / bench.l2_bytes:.1f} x L2 ({mb:.0f} MB)")
    return (f"NOT larger than L2: {bench.R} replicas x {rank_bytes_per_step / 1e6:.1f} MB per step = "
            f"{rot / 1e6:.1f} MB between visits of a replica, {rot / bench.l2_bytes:.2f} x L2 ({mb:.0f} MB); "
            "the workload is latency-bound and partly served from L2")


def run_gpu(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.distributed.is_nccl_available() else "gloo")
    bench = Bench(args, rank, world)
    bench.setup()
    W, K = args.warmup, args.steps
    core = timed_steps(bench, W, K, dist, local)
    ms, job_bytes, job_keys = core["ms"], core["job_bytes"], core["job_keys"]
    rank_bytes, launches_per_step, clocks = core["rank_bytes"], core["launches_per_step"], core["clocks"]
    call_ms, call_bytes = core["call_ms"], core["call_bytes"]
    base = W + K

    # e2e: the public API with host buffers.  Each step's inputs (every layer's entries,
    # K/V rows and queries) sit in one pinned host buffer that is copied to the device in
    # one H2D copy, and every layer's output rows come back in one D2H copy: the step as
    # a serving loop that stages a decode step's inputs would run it.
    e0 = base + K
    in_keys = ("seqs", "pos", "bits", "modes", "k", "v", "q")

    def pack(tensors):
        """One device buffer holding the tensors (256-byte aligned segments), views into
        it in the tensors' dtypes and shapes, and a pinned host copy of its bytes."""
        offs, total = [], 0
        for t in tensors:
            offs.append(total)
            total += -(-t.numel() * t.element_size() // 256) * 256
        dbuf = torch.empty(total, dtype=torch.uint8, device=bench.dev)
        views = []
        for t, o in zip(tensors, offs):
            nb = t.numel() * t.element_size()
            v = dbuf[o:o + nb].view(t.dtype).view(t.shape)
            v.copy_(t)
            views.append(v)
        return dbuf, views, dbuf.cpu().pin_memory()

    packed = []
    for i in range(e0, e0 + bench.e2e_warm + bench.e2e_steps):
        st = bench.steps[i]
        ins = [x[k] for x in st["layers"] for k in in_keys]
        din, vin, hin = pack(ins)
        dout, vout, hout = pack([x["out"] for x in st["layers"]])
        layers = []
        for li in range(len(st["layers"])):
            lay = {k: vin[li * len(in_keys) + j] for j, k in enumerate(in_keys)}
            lay["out"] = vout[li]
            layers.append(lay)
        packed.append(dict(layers=layers, din=din, hin=hin, dout=dout, hout=hout))
    h2d = packed[0]["hin"].numel()
    d2h = packed[0]["hout"].numel()

    def e2e_step(j):
        ps = packed[j]
        ps["din"].copy_(ps["hin"], non_blocking=True)
        bench.run_step(dict(layers=ps["layers"]))
        ps["hout"].copy_(ps["dout"], non_blocking=True)

    # each step as a serving engine runs it: captured once as a CUDA graph holding the
    # H2D copy, the step's public API calls and the D2H copy, then replayed per step
    ne = bench.e2e_warm + bench.e2e_steps
    half = bench.e2e_warm + bench.e2e_steps // 2
    egraphs = []
    for j in range(half):
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side):
                e2e_step(j)
        torch.cuda.current_stream().wait_stream(side)
        egraphs.append(g)
    for j in range(bench.e2e_warm):
        egraphs[j].replay()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a0.record()
    for j in range(bench.e2e_warm, half):
        egraphs[j].replay()
    a1.record()
    torch.cuda.synchronize()
    e2e_ms = a0.elapsed_time(a1)
    e2e_bytes = sum(bench.steps[e0 + j]["bytes"] for j in range(bench.e2e_warm, half))
    e2e_ms, e2e_bytes = across_ranks(dist, "cuda", e2e_ms, e2e_bytes)
    del egraphs
    # the same steps issued call by call from Python (no graph): host-launch bound
    b0, b1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    b0.record()
    for j in range(half, ne):
        e2e_step(j)
    b1.record()
    torch.cuda.synchronize()
    eager_ms = b0.elapsed_time(b1)
    eager_bytes = sum(bench.steps[e0 + j]["bytes"] for j in range(half, ne))
    eager_ms, eager_bytes = across_ranks(dist, "cuda", eager_ms, eager_bytes)
    r0 = e0 + bench.e2e_warm + bench.e2e_steps
    routed = None if bench.head_modes else run_routed(bench, dist, r0)
    separate = run_separate(bench, dist, r0 + bench.routed_warm + bench.routed_steps)
    status = bench.cache.status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the run")

    peak, peak_kind = measured_peaks()
    avg_bytes = float(np.mean(call_bytes))
    avg_ms = float(np.mean(call_ms))  # event nodes around each call (no overlap with its neighbours)
    # A step of one launch per layer (the decode-step kernel alone) gives the kernel's
    # average launch duration over the timed region itself: the step's time over its
    # launches, with programmatic dependent launch overlapping each launch's start with
    # the previous one's end as in serving.  Otherwise the bracketed calls.
    in_stream = launches_per_step == bench.L
    launch_ms = (ms / K) / bench.L if in_stream else avg_ms
    if in_stream:  # the timed steps' own bytes (modes differ from step to step)
        avg_bytes = rank_bytes / K / bench.L
    achieved = avg_bytes / (launch_ms * 1e-3) / 1e9
    value = job_bytes / (ms * 1e-3) / 1e9
    result = None
    if rank == 0:
        cpu = (cpu_baseline(bench) if (world == 1 and not args.no_cpu_baseline and not bench.head_modes
                                       and not bench.swk and bench.C == 1) else None)
        result = {
            "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
            "steps": K, "warmup": W, "ms_per_step": round(ms / K, 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {
                "workload": f"{bench.spec.name}: {bench.L} layers, MHA/GQA {bench.Hq}/{bench.Hkv} x {bench.d}, "
                            f"batch {bench.B}/GPU, contexts {describe_ctx(bench)}, window {bench.window}, "
                            f"group {bench.G}, page {bench.P}",
                "kv_storage": "per-token 2/4/8-bit codes + fp16 scale/zero, or bf16; fp32 accumulation",
                "modes": "per (token, query head), presence mask per KV head" if bench.head_modes
                         else "per token",
                "skip_tokens_store_kv": bool(bench.swk),
                "queries_per_seq": bench.C,
                "global_batch": bench.B * world, "replicas": bench.R,
                "l2": l2_note(bench, rank_bytes / K), "l2_bytes": bench.l2_bytes,
                "parallelism": f"replicas{world}" if world > 1 else "single",
                "bytes_per_step": int(job_bytes / K),
                "split_bytes": args.split_bytes or "default",
            },
            "kv_tokens_per_s": round(job_keys / (ms * 1e-3), 1),
            "pct_of_8tbs": round(100 * value / world / 8000.0, 2),
            "gpu_launches": launches_per_step * K,
            "e2e": {"value": round(e2e_bytes / (e2e_ms * 1e-3) / 1e9, 2), "unit": UNIT,
                    "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                    "how": "per step one CUDA graph of: pinned H2D copy of the step's inputs, the step's "
                           "API calls (trr_decode_step per layer), D2H copy of every output row",
                    "eager_value": round(eager_bytes / (eager_ms * 1e-3) / 1e9, 2),
                    "eager_how": "the same steps called one by one from Python, no graph (host-launch bound)"},
            "roofline": {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak,
                         "unit": "GB/s", "frac": round(achieved / peak, 4),
                         "traffic": None if (bench.head_modes or bench.swk or bench.C > 1)
                         else ncu_traffic(args.workload),
                         "peak_kind": peak_kind,
                         "kernel": "trr_decode_step call (attn_kernel: append and attention, one launch)" if bench.C == 1
                         and not bench.head_modes else "trr_decode_attn call (attn_kernel, one launch)",
                         "bytes_per_call": round(avg_bytes), "us_per_call": round(launch_ms * 1e3, 3),
                         "timing": "timed region / launches (one launch per layer)" if in_stream
                         else "event nodes around each call",
                         "us_per_call_bracketed": round(avg_ms * 1e3, 3)},
            "clocks": clocks.summary(),
        }
        if routed is not None:
            result["routed"] = routed
        if separate is not None:
            result["separate_calls"] = separate
        if cpu is not None:
            result["cpu_baseline"] = cpu
    if (rank == 0 and world == 1 and not args.no_per_workload and not bench.head_modes and not bench.swk
            and bench.C == 1 and args.workload == "160m" and not args.batch and not args.layers):
        import gc
        del bench
        gc.collect()
        torch.cuda.empty_cache()
        result["per_workload"] = per_workload(args, local)
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return result


def describe_ctx(bench):
    c = bench.ctx
    lo, hi = int(c.min()), int(c.max())
    grow = math.ceil(bench.total_steps / bench.R) * bench.C
    base = f"{lo}" if lo == hi else f"{lo}-{hi}"
    return f"{base} (+ up to {grow} decoded)"


# ----------------------------------------------------------- the oracle on the CPU --

class OracleSample:
    """A bounded sample of the workload for the CPU oracle: layer 0 of the first n_seqs
    sequences with their full prebuilt contexts; the queries are those sequences' last
    positions, newest first, each with its own seeded mode."""

    def __init__(self, spec, n_seqs, window, layer=0):
        import oracle
        from paper_2607_06601_gb300 import workloads as wl
        self.ctx = wl.contexts(spec)
        self.n_seqs = n_seqs = min(n_seqs, spec.batch)
        self.window = window
        maxctx = int(self.ctx[:n_seqs].max())
        caps = [n_seqs * (maxctx // PAGE + 2)] * 4
        self.o = oracle.OracleCache(1, n_seqs, spec.num_q_heads, spec.num_kv_heads, spec.head_dim,
                                    spec.group_size, PAGE, maxctx, caps)
        self.acct = Accounting(spec, spec.head_dim, spec.group_size, spec.num_q_heads,
                               spec.num_kv_heads, window)
        self.maps = []
        for s in range(n_seqs):
            n = int(self.ctx[s])
            bits, modes = wl.policy(spec, layer, s, n)
            q, k, v = wl.q_kv_fast(spec, layer, s, 0, n)
            for p0 in range(0, n, 1024):
                p1 = min(n, p0 + 1024)
                assert self.o.append(0, [s] * (p1 - p0), np.arange(p0, p1), k[p0:p1], v[p0:p1],
                                     bits[p0:p1], modes[p0:p1]) == 0
            self.maps.append((bits, modes, q))
        self.n_queries = min(4096, int(self.ctx[:n_seqs].min()) * n_seqs)

    def query(self, j):
        """Runs query j on the oracle; returns its (algorithmic bytes, attended keys)."""
        s = j % self.n_seqs
        t = int(self.ctx[s]) - 1 - (j // self.n_seqs)
        bits, modes, q = self.maps[s]
        st, _ = self.o.decode_attn(0, [s], [t], q[t:t + 1], [modes[t]], window_scalar=self.window)
        assert st == 0
        nb, nk, _ = self.acct.query(bits, modes, t)
        return nb, nk

    def run(self, budget_s, threads=1):
        """Queries 0, 1, 2, ... until budget_s of wall time, on `threads` host threads
        (the oracle's decode call reads the cache only, and ctypes lets go of the
        interpreter lock while it runs, so the threads run the C code side by side).
        Returns (bytes, keys, queries, wall seconds)."""
        import itertools
        import threading
        nxt = itertools.count()
        lock = threading.Lock()
        tot = [0, 0, 0]
        deadline = time.perf_counter() + budget_s

        def worker():
            nb = nk = nq = 0
            while time.perf_counter() < deadline:
                j = next(nxt)
                if j >= self.n_queries:
                    break
                b, k = self.query(j)
                nb, nk, nq = nb + b, nk + k, nq + 1
            with lock:
                tot[0] += nb
                tot[1] += nk
                tot[2] += nq

        t0 = time.perf_counter()
        if threads == 1:
            worker()
        else:
            ts = [threading.Thread(target=worker) for _ in range(threads)]
            for t in ts:
                t.start()
            for t in ts:
                t.join()
        return tot[0], tot[1], tot[2], time.perf_counter() - t0


def host_threads():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def timed_legs(sample, budget_s, threads, repeats=3):
    """Median over `repeats` runs of about budget_s each: (GB/s, kv tokens/s, queries)."""
    runs = []
    for _ in range(repeats):
        nb, nk, nq, wall = sample.run(budget_s, threads)
        runs.append((nb / wall / 1e9, nk / wall, nq))
    runs.sort()
    return runs[len(runs) // 2]


def cpu_baseline(bench):
    """The fp64 C oracle on the host: one thread and every core of this process's
    affinity, median of three runs of each."""
    sample = OracleSample(bench.spec, 4, bench.window)
    n = host_threads()
    one = timed_legs(sample, 3.0, 1)
    every = timed_legs(sample, 3.0, n)
    return {"value": round(every[0], 4), "unit": UNIT, "cores": n, "kind": "oracle",
            "kv_tokens_per_s": round(every[1], 1),
            "single_thread": {"value": round(one[0], 4), "cores": 1, "kv_tokens_per_s": round(one[1], 1)},
            "sample": f"decode queries of layer 0, sequences 0-3 at their last positions (seeded modes), "
                      f"fp64 C oracle; {n} threads: {every[2]} queries per run, 1 thread: {one[2]}; "
                      f"median of 3 runs of about 3 s each"}


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, on the same metric and workload."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return None
    from paper_2607_06601_gb300 import workloads as wl
    import oracle
    oracle.build()
    spec = wl.SPECS[args.workload]
    if args.batch:
        spec = spec.with_(batch=args.batch)
    per_step = max(0.5, min(5.0, 150.0 / max(1, args.steps + args.warmup)))
    n = host_threads()
    sample = OracleSample(spec, 4, spec.window)
    for _ in range(args.warmup):
        sample.run(per_step / 4, n)
    tot_b = tot_k = 0
    tot_t = 0.0
    for _ in range(args.steps):
        nb, nk, nq, wall = sample.run(per_step, n)
        tot_b += nb
        tot_k += nk
        tot_t += wall
    value = tot_b / tot_t / 1e9
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
        "n_gpus": int(os.environ.get("WORLD_SIZE", "1")), "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * tot_t / max(1, args.steps), 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{spec.name} (same maps and shapes as the GPU arm), oracle sample per step"},
        "kv_tokens_per_s": round(tot_k / tot_t, 1),
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": n, "kind": "oracle",
                         "sample": "each step: decode queries of sequences 0-3 at their last positions, "
                                   f"layer 0, about {per_step:.1f} s of wall time on {n} host threads"},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="160m", choices=["tiny", "160m", "1p3b", "gqa_long", "sweep"])
    ap.add_argument("--batch", type=int, default=0)
    ap.add_argument("--layers", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="skip the other workloads (1p3b, gqa_long, tiny, sweep at batch 1/8/64/256)")
    ap.add_argument("--per-workload-steps", type=int, default=10)
    ap.add_argument("--cache-budget-gb", type=float, default=120.0,
                    help="device memory the replicas of one workload's cache may take")
    ap.add_argument("--page-size", type=int, default=0, choices=[0, 16, 32, 64],
                    help="tokens per cache page (0: 32)")
    ap.add_argument("--split-bytes", type=int, default=0,
                    help="target KV bytes per split-K work item (0: the library default)")
    ap.add_argument("--chunk", type=int, default=1,
                    help="new tokens and queries per sequence per step (chunked decode / speculative "
                         "verification: each query attends up to its own position); no CPU baseline")
    ap.add_argument("--skip-writes-kv", action="store_true",
                    help="skip tokens store their KV too (the paper's Principle 1 reading; default: "
                         "they store nothing); no CPU baseline")
    ap.add_argument("--head-modes", action="store_true",
                    help="a mode per (token, query head), drawn from the workload's mode mix "
                         "(Sec. 3.2(A)); no routed step and no CPU baseline")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        res = run_reference(args)
    else:
        import __graft_entry__
        __graft_entry__.build()
        res = run_gpu(args)
    if res is not None:
        print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
