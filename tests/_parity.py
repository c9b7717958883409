"""Helpers of the GPU parity tests: drive the CUDA library and the CPU oracle with the
same seeded inputs and compare what they produce (bit-exact for the cache, within the
stated tolerance for attention)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2607_06601_gb300 import trr

ATOL = 2e-2       # max |gpu - oracle| over every element
ROW_RTOL = 5e-3   # per (query, head) row: max |gpu - oracle| / max |oracle|

REGION_NAMES = ("last_pos", "ntok", "presence", "page_table", "page_first", "page_last", "next_page")


def dev(a, dtype):
    """numpy array (bf16 passed as uint16 bits) -> CUDA tensor of `dtype`."""
    t = torch.from_numpy(np.ascontiguousarray(a))
    return t.cuda().view(dtype)


class Pair:
    """A GPU cache and an oracle cache with one configuration, fed the same calls."""

    def __init__(self, L, S, Hq, Hkv, d, G, P, maxctx, caps, skip_writes_kv=0, max_append=1024,
                 max_queries=1024, split_bytes=0, oracle_pool=True, head_modes=0):
        self.gpu = trr.Cache(L, S, Hq, Hkv, d, G, P, maxctx, caps, max_append=max_append,
                             max_queries=max_queries, split_bytes=split_bytes,
                             skip_writes_kv=skip_writes_kv, zero_pool=True, head_modes=head_modes)
        # zero_pool: unused slots read back as zeros, as the oracle's calloc
        self.orc = oracle.OracleCache(L, S, Hq, Hkv, d, G, P, maxctx, caps,
                                      skip_writes_kv=skip_writes_kv, no_pool=not oracle_pool,
                                      head_modes=head_modes)
        self.head_modes = head_modes
        self.Hq, self.Hkv, self.d, self.P = Hq, Hkv, d, P

    def append(self, layer, seqs, pos, k, v, bits, modes, expect=0):
        seqs = np.asarray(seqs, dtype=np.int32)
        pos = np.asarray(pos, dtype=np.int32)
        bits = np.asarray(bits, dtype=np.uint8)
        modes = np.asarray(modes, dtype=np.uint8)
        self.gpu.append(layer, dev(seqs, torch.int32), dev(pos, torch.int32), dev(k, torch.bfloat16),
                        dev(v, torch.bfloat16), dev(bits, torch.uint8), dev(modes, torch.uint8))
        st_o = self.orc.append(layer, seqs, pos, k, v, bits, modes)
        st_g = self.gpu.status()
        assert st_o == expect, f"oracle append status {st_o}, expected {expect}"
        assert st_g == st_o, f"gpu append status {st_g} != oracle {st_o}"

    def attend(self, layer, seqs, ts, q, modes, windows=None, window_scalar=0, scale=0.0, expect=0):
        seqs = np.asarray(seqs, dtype=np.int32)
        ts = np.asarray(ts, dtype=np.int32)
        modes = np.asarray(modes, dtype=np.uint8)
        win = None if windows is None else dev(np.asarray(windows, dtype=np.int32), torch.int32)
        out = self.gpu.decode_attn(layer, dev(seqs, torch.int32), dev(ts, torch.int32),
                                   dev(q, torch.bfloat16), dev(modes, torch.uint8), win,
                                   window_scalar, scale)
        st_o, ref = self.orc.decode_attn(layer, seqs, ts, q, modes, windows, window_scalar, scale)
        st_g = self.gpu.status()
        assert st_o == expect, f"oracle attention status {st_o}, expected {expect}"
        assert st_g == st_o, f"gpu attention status {st_g} != oracle {st_o}"
        got = out.float().cpu().numpy().astype(np.float64)
        # skip rows must be bit-zero: per query, or per (query, head) with head modes
        check_attention(got, ref, modes.reshape(len(seqs), self.Hq) if self.head_modes else modes)
        return got, ref

    def step(self, layer, seqs, pos, k, v, bits, modes, q, windows=None, window_scalar=0, scale=0.0):
        """trr_decode_step on the GPU against the oracle's append of the same entries
        followed by its attention with their queries at the same positions and modes."""
        seqs = np.asarray(seqs, dtype=np.int32)
        pos = np.asarray(pos, dtype=np.int32)
        bits = np.asarray(bits, dtype=np.uint8)
        modes = np.asarray(modes, dtype=np.uint8)
        win = None if windows is None else dev(np.asarray(windows, dtype=np.int32), torch.int32)
        out = self.gpu.decode_step(layer, dev(seqs, torch.int32), dev(pos, torch.int32), dev(k, torch.bfloat16),
                                   dev(v, torch.bfloat16), dev(bits, torch.uint8), dev(modes, torch.uint8),
                                   dev(q, torch.bfloat16), win, window_scalar, scale)
        st_g = self.gpu.status()
        st_a = self.orc.append(layer, seqs, pos, k, v, bits, modes)
        assert st_a == 0, f"oracle append status {st_a}"
        st_o, ref = self.orc.decode_attn(layer, seqs, pos, q, modes, windows, window_scalar, scale)
        assert st_o == 0, f"oracle attention status {st_o}"
        assert st_g == 0, f"gpu decode-step status {st_g}"
        got = out.float().cpu().numpy().astype(np.float64)
        check_attention(got, ref, modes)
        return got, ref

    def check_regions(self, pools=True):
        compare_regions(self.gpu, self.orc, pools)


def bf16_half_ulp(x):
    """Half a bf16 unit in the last place at |x| (8 significant bits): the most that
    rounding a value of that size to bf16 moves it."""
    e = np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** -126)))
    return 2.0 ** (e - 8)


def check_attention(got, ref, modes=None):
    """The stated bar: max abs error 2e-2 and per-row relative error <= 5e-3; rows of
    skip queries (and rows with nothing in range) are exact zeros.  The rows are bf16
    (round to nearest even), so the absolute bound holds on top of that rounding:
    |gpu - oracle| <= 2e-2 + half a bf16 ulp of the oracle value (for |o| >= 8 the
    rounding alone reaches 2^-5 > 2e-2)."""
    assert got.shape == ref.shape
    diff = np.abs(got - ref)
    excess = diff - (ATOL + bf16_half_ulp(ref))
    assert excess.max(initial=-1.0) <= 0, f"max abs err {diff.max():.3e} (beyond the bound by {excess.max():.3e})"
    den = np.abs(ref).max(axis=-1)
    num = diff.max(axis=-1)
    zero_rows = den == 0
    assert (num[zero_rows] == 0).all(), "a row the oracle leaves at zero is not zero"
    if (~zero_rows).any():
        rel = num[~zero_rows] / den[~zero_rows]
        assert rel.max() <= ROW_RTOL, f"row-relative err {rel.max():.3e}"
    if modes is not None:
        skip = np.asarray(modes) == 0
        assert (got[skip] == 0).all() and not np.signbit(got[skip]).any()


def compare_regions(gpu: trr.Cache, orc: oracle.OracleCache, pools=True):
    torch.cuda.synchronize()
    for name in REGION_NAMES:
        g = gpu.region(name).cpu().numpy()
        o = orc.region(name)
        assert g.shape == o.shape, name
        if not np.array_equal(g, o):
            bad = np.nonzero(g != o)[0]
            raise AssertionError(f"region {name} differs at {bad.size} bytes, first at {bad[:8]}")
    if not pools:
        return
    nextp = orc.region("next_page").view(np.int32)
    for c, b in enumerate((2, 4, 8, 16)):
        used = int(nextp[c]) * orc.page_bytes(c)
        g = gpu.region(f"pool{b}")[:used].cpu().numpy()
        o = orc.region(f"pool{b}")[:used]
        if not np.array_equal(g, o):
            bad = np.nonzero(g != o)[0]
            pb = orc.page_bytes(c)
            raise AssertionError(f"pool{b} differs at {bad.size} bytes; first page {bad[0] // pb}, "
                                 f"offset {bad[0] % pb}")


def logical_pages(cache_pt, ntok, P, seq, c, MP):
    """Page ids of (seq, class c) in position order."""
    np_ = -(-int(ntok[seq, c]) // P)
    return cache_pt[seq, c, :np_]
