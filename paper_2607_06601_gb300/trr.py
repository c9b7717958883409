"""Python binding of the C ABI in include/trr.h (argument marshalling only).

Every step of the serving path runs in the CUDA library ``_build/libtrr.so``; this
module only checks tensor dtypes / devices / shapes, passes raw device pointers and the
current CUDA stream, and turns status codes into exceptions.  There is no fallback: if
the library is missing, loading it raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

STATUS = {0: "OK", 1: "INVALID_ARG", 2: "OUT_OF_MEMORY", 3: "OUT_OF_PAGES", 4: "BAD_POSITION",
          5: "CUDA", 6: "UNSUPPORTED", 7: "BAD_VALUE", 8: "TIMEOUT"}
MODE_SKIP, MODE_LOCAL, MODE_FULL = 0, 1, 2
REGIONS = {"last_pos": 0, "ntok": 1, "presence": 2, "page_table": 3, "page_first": 4,
           "page_last": 5, "next_page": 6, "pool2": 7, "pool4": 8, "pool8": 9, "pool16": 10}


class TrrError(RuntimeError):
    def __init__(self, where: str, code: int):
        super().__init__(f"{where}: {STATUS.get(code, code)}")
        self.code = code


class trr_cache_config(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("group_size", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_context", ctypes.c_int32),
                ("pages_per_class", ctypes.c_int32 * 4), ("max_append", ctypes.c_int32),
                ("max_queries", ctypes.c_int32), ("split_bytes", ctypes.c_int32),
                ("skip_writes_kv", ctypes.c_int32), ("head_modes", ctypes.c_int32),
                ("pool", ctypes.c_void_p),
                ("pool_bytes", ctypes.c_uint64)]


EXPORTS = ("trr_cache_required_bytes", "trr_create_cache", "trr_kv_append", "trr_decode_attn",
           "trr_decode_step", "trr_decode_attn_static", "trr_route_decisions", "trr_kv_append_routed",
           "trr_decode_attn_routed", "trr_destroy", "trr_get_status", "trr_set_wait_limit", "trr_reset",
           "trr_get_region",
           "trr_last_launch_count")

_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False) -> ctypes.CDLL:
    """Load libtrr.so (built by __graft_entry__.build()); raise if it is not there."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(f"CUDA library {path} is missing: run __graft_entry__.build() first")
        _build.build()
    L = ctypes.CDLL(path)
    P, I32, U64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64
    L.trr_cache_required_bytes.argtypes = [ctypes.POINTER(trr_cache_config), ctypes.POINTER(U64)]
    L.trr_create_cache.argtypes = [ctypes.POINTER(trr_cache_config), ctypes.POINTER(P)]
    L.trr_kv_append.argtypes = [P, I32, I32, P, P, P, P, P, P, P]
    L.trr_decode_attn.argtypes = [P, I32, I32, P, P, P, P, P, I32, ctypes.c_float, P, P]
    L.trr_decode_attn_static.argtypes = [P, I32, I32, P, P, P, P, P, I32, ctypes.c_float, P, P]
    L.trr_decode_step.argtypes = [P, I32, I32, P, P, P, P, P, P, P, P, I32, ctypes.c_float, P, P]
    L.trr_route_decisions.argtypes = [I32, P, P, P, I32, I32, I32, I32, I32, P, P, P, P, P, P]
    L.trr_kv_append_routed.argtypes = [P, I32, I32, P, P, P, P, P, P, P]
    L.trr_decode_attn_routed.argtypes = [P, I32, I32, P, P, P, P, P, I32, ctypes.c_float, P, P]
    L.trr_destroy.argtypes = [P]
    L.trr_get_status.argtypes = [P, P]
    L.trr_set_wait_limit.argtypes = [P, U64]
    L.trr_reset.argtypes = [P, P]
    L.trr_get_region.argtypes = [P, I32, ctypes.POINTER(P), ctypes.POINTER(U64)]
    L.trr_last_launch_count.argtypes = [P]
    for name in EXPORTS:
        getattr(L, name).restype = I32
    _lib = L
    return L


def _check(where, code):
    if code != 0:
        raise TrrError(where, code)


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dev(t: torch.Tensor, dtype, name):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def make_config(num_layers, max_seqs, num_q_heads, num_kv_heads, head_dim, group_size,
                page_size, max_context, pages_per_class, max_append=1024, max_queries=1024,
                split_bytes=0, skip_writes_kv=0, head_modes=0) -> trr_cache_config:
    cfg = trr_cache_config()
    cfg.num_layers, cfg.max_seqs = num_layers, max_seqs
    cfg.num_q_heads, cfg.num_kv_heads = num_q_heads, num_kv_heads
    cfg.head_dim, cfg.group_size, cfg.page_size = head_dim, group_size, page_size
    cfg.max_context = max_context
    for i in range(4):
        cfg.pages_per_class[i] = int(pages_per_class[i])
    cfg.max_append, cfg.max_queries = max_append, max_queries
    cfg.split_bytes, cfg.skip_writes_kv = split_bytes, skip_writes_kv
    cfg.head_modes = head_modes
    return cfg


def trr_cache_required_bytes(cfg: trr_cache_config) -> int:
    out = ctypes.c_uint64()
    _check("trr_cache_required_bytes", load().trr_cache_required_bytes(ctypes.byref(cfg), ctypes.byref(out)))
    return int(out.value)


def trr_create_cache(cfg: trr_cache_config, pool: torch.Tensor | None = None) -> ctypes.c_void_p:
    if pool is not None:
        cfg.pool = ctypes.c_void_p(pool.data_ptr())
        cfg.pool_bytes = pool.numel() * pool.element_size()
    h = ctypes.c_void_p()
    _check("trr_create_cache", load().trr_create_cache(ctypes.byref(cfg), ctypes.byref(h)))
    return h


def trr_kv_append(cache, layer, seq_ids, positions, k, v, bits, modes, stream=None):
    n = seq_ids.numel()
    _check("trr_kv_append", load().trr_kv_append(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"), _dev(positions, torch.int32, "positions"),
        _dev(k, torch.bfloat16, "k"), _dev(v, torch.bfloat16, "v"), _dev(bits, torch.uint8, "bits"),
        _dev(modes, torch.uint8, "modes"), _stream(stream)))


def trr_decode_attn(cache, layer, seq_ids, q_positions, q, modes, windows, window_scalar,
                    softmax_scale, out, stream=None):
    n = seq_ids.numel()
    win = None if windows is None else _dev(windows, torch.int32, "windows")
    _check("trr_decode_attn", load().trr_decode_attn(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"),
        _dev(q_positions, torch.int32, "q_positions"), _dev(q, torch.bfloat16, "q"),
        _dev(modes, torch.uint8, "modes"), win, int(window_scalar), float(softmax_scale),
        _dev(out, torch.bfloat16, "out"), _stream(stream)))


def trr_decode_step(cache, layer, seq_ids, positions, k, v, bits, modes, q, windows, window_scalar,
                    softmax_scale, out, stream=None):
    """One decode step of one layer in one kernel: the append of every entry's token, then
    every entry's query at the same position and mode (see include/trr.h)."""
    n = seq_ids.numel()
    win = None if windows is None else _dev(windows, torch.int32, "windows")
    _check("trr_decode_step", load().trr_decode_step(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"), _dev(positions, torch.int32, "positions"),
        _dev(k, torch.bfloat16, "k"), _dev(v, torch.bfloat16, "v"), _dev(bits, torch.uint8, "bits"),
        _dev(modes, torch.uint8, "modes"), _dev(q, torch.bfloat16, "q"), win, int(window_scalar),
        float(softmax_scale), _dev(out, torch.bfloat16, "out"), _stream(stream)))


def trr_decode_attn_static(cache, layer, seq_ids, q_positions, q, modes, windows, window_scalar,
                           softmax_scale, out, stream=None):
    """trr_decode_attn with its scratch in the library's static device array: no
    allocation anywhere on the way (see include/trr.h)."""
    n = seq_ids.numel()
    win = None if windows is None else _dev(windows, torch.int32, "windows")
    _check("trr_decode_attn_static", load().trr_decode_attn_static(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"),
        _dev(q_positions, torch.int32, "q_positions"), _dev(q, torch.bfloat16, "q"),
        _dev(modes, torch.uint8, "modes"), win, int(window_scalar), float(softmax_scale),
        _dev(out, torch.bfloat16, "out"), _stream(stream)))


def _opt(t, dtype, name):
    return None if t is None else _dev(t, dtype, name)


def trr_route_decisions(mode_logits, bit_logits, positions=None, window=1, num_q_heads=1, head_dim=1,
                        num_kv_heads=1, skip_writes_kv=0, modes=None, bits=None, attn_flops=None,
                        kv_bits=None, totals=None, stream=None):
    """Hard decisions of n tokens (and, with positions, their cost) into the given
    device tensors; ``totals`` (int64[4]) is added to."""
    n = mode_logits.shape[0] if mode_logits.dim() else 0
    if mode_logits.numel() != 3 * n or bit_logits.numel() != 4 * n:
        raise ValueError("mode_logits must be [n][3] and bit_logits [n][4]")
    for t, k, name in ((modes, n, "modes"), (bits, n, "bits"), (attn_flops, n, "attn_flops"),
                       (kv_bits, n, "kv_bits"), (positions, n, "positions"), (totals, 4, "totals")):
        if t is not None and t.numel() != k:
            raise ValueError(f"{name} must have {k} elements")
    _check("trr_route_decisions", load().trr_route_decisions(
        n, _dev(mode_logits, torch.float32, "mode_logits"), _dev(bit_logits, torch.float32, "bit_logits"),
        _opt(positions, torch.int32, "positions"), int(window), int(num_q_heads), int(head_dim),
        int(num_kv_heads), int(skip_writes_kv), _opt(modes, torch.uint8, "modes"),
        _opt(bits, torch.uint8, "bits"), _opt(attn_flops, torch.int64, "attn_flops"),
        _opt(kv_bits, torch.int64, "kv_bits"), _opt(totals, torch.int64, "totals"), _stream(stream)))


def trr_kv_append_routed(cache, layer, seq_ids, positions, k, v, bit_logits, mode_logits, stream=None):
    n = seq_ids.numel()
    if bit_logits.numel() != 4 * n or mode_logits.numel() != 3 * n:
        raise ValueError("bit_logits must be [n][4] and mode_logits [n][3]")
    _check("trr_kv_append_routed", load().trr_kv_append_routed(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"), _dev(positions, torch.int32, "positions"),
        _dev(k, torch.bfloat16, "k"), _dev(v, torch.bfloat16, "v"),
        _dev(bit_logits, torch.float32, "bit_logits"), _dev(mode_logits, torch.float32, "mode_logits"),
        _stream(stream)))


def trr_decode_attn_routed(cache, layer, seq_ids, q_positions, q, mode_logits, windows, window_scalar,
                           softmax_scale, out, stream=None):
    n = seq_ids.numel()
    if mode_logits.numel() != 3 * n:
        raise ValueError("mode_logits must be [n][3]")
    win = None if windows is None else _dev(windows, torch.int32, "windows")
    _check("trr_decode_attn_routed", load().trr_decode_attn_routed(
        cache, layer, n, _dev(seq_ids, torch.int32, "seq_ids"),
        _dev(q_positions, torch.int32, "q_positions"), _dev(q, torch.bfloat16, "q"),
        _dev(mode_logits, torch.float32, "mode_logits"), win, int(window_scalar), float(softmax_scale),
        _dev(out, torch.bfloat16, "out"), _stream(stream)))


def trr_destroy(cache):
    _check("trr_destroy", load().trr_destroy(cache))


def trr_get_status(cache, stream=None) -> int:
    return int(load().trr_get_status(cache, _stream(stream)))


def trr_reset(cache, stream=None):
    _check("trr_reset", load().trr_reset(cache, _stream(stream)))


def trr_get_region(cache, region) -> tuple[int, int]:
    p, nb = ctypes.c_void_p(), ctypes.c_uint64()
    _check("trr_get_region", load().trr_get_region(cache, REGIONS.get(region, region),
                                                   ctypes.byref(p), ctypes.byref(nb)))
    return int(p.value or 0), int(nb.value)


def trr_last_launch_count(cache) -> int:
    return int(load().trr_last_launch_count(cache))


class Cache:
    """A cache on the current CUDA device whose memory is one caller-owned uint8 tensor."""

    def __init__(self, num_layers, max_seqs, num_q_heads, num_kv_heads, head_dim, group_size,
                 page_size, max_context, pages_per_class, max_append=1024, max_queries=1024,
                 split_bytes=0, skip_writes_kv=0, device=None, zero_pool=False, head_modes=0):
        self.cfg = make_config(num_layers, max_seqs, num_q_heads, num_kv_heads, head_dim,
                               group_size, page_size, max_context, pages_per_class, max_append,
                               max_queries, split_bytes, skip_writes_kv, head_modes)
        self.head_modes = int(head_modes)
        self.nbytes = trr_cache_required_bytes(self.cfg)
        alloc = torch.zeros if zero_pool else torch.empty
        self.pool = alloc(self.nbytes, dtype=torch.uint8, device=device or torch.cuda.current_device())
        self.handle = trr_create_cache(self.cfg, self.pool)
        self.L, self.S, self.Hq, self.Hkv = num_layers, max_seqs, num_q_heads, num_kv_heads
        self.d, self.G, self.P, self.max_context = head_dim, group_size, page_size, max_context

    def _check_modes(self, modes, n):
        want = n * (self.Hq if self.head_modes else 1)
        if modes.numel() != want:
            raise ValueError(f"modes must have {want} elements "
                             f"({'[n][Hq]' if self.head_modes else '[n]'}), got {modes.numel()}")

    def append(self, layer, seq_ids, positions, k, v, bits, modes, stream=None):
        self._check_modes(modes, seq_ids.numel())
        trr_kv_append(self.handle, layer, seq_ids, positions, k, v, bits, modes, stream)

    def decode_attn(self, layer, seq_ids, q_positions, q, modes, windows=None, window_scalar=0,
                    softmax_scale=0.0, out=None, stream=None):
        self._check_modes(modes, seq_ids.numel())
        if out is None:
            out = torch.empty((seq_ids.numel(), self.Hq, self.d), dtype=torch.bfloat16, device=q.device)
        trr_decode_attn(self.handle, layer, seq_ids, q_positions, q, modes, windows, window_scalar,
                        softmax_scale, out, stream)
        return out

    def decode_step(self, layer, seq_ids, positions, k, v, bits, modes, q, windows=None, window_scalar=0,
                    softmax_scale=0.0, out=None, stream=None):
        self._check_modes(modes, seq_ids.numel())
        if out is None:
            out = torch.empty((seq_ids.numel(), self.Hq, self.d), dtype=torch.bfloat16, device=q.device)
        trr_decode_step(self.handle, layer, seq_ids, positions, k, v, bits, modes, q, windows, window_scalar,
                        softmax_scale, out, stream)
        return out

    def append_routed(self, layer, seq_ids, positions, k, v, bit_logits, mode_logits, stream=None):
        trr_kv_append_routed(self.handle, layer, seq_ids, positions, k, v, bit_logits, mode_logits, stream)

    def decode_attn_routed(self, layer, seq_ids, q_positions, q, mode_logits, windows=None,
                           window_scalar=0, softmax_scale=0.0, out=None, stream=None):
        if out is None:
            out = torch.empty((seq_ids.numel(), self.Hq, self.d), dtype=torch.bfloat16, device=q.device)
        trr_decode_attn_routed(self.handle, layer, seq_ids, q_positions, q, mode_logits, windows,
                               window_scalar, softmax_scale, out, stream)
        return out

    def status(self, stream=None) -> int:
        return trr_get_status(self.handle, stream)

    def set_wait_limit(self, nanoseconds: int):
        """Bound of every in-kernel wait of this cache's calls (0: the default, 2 s)."""
        _check("trr_set_wait_limit", load().trr_set_wait_limit(self.handle, int(nanoseconds)))

    def reset(self, stream=None):
        trr_reset(self.handle, stream)

    def region(self, name) -> torch.Tensor:
        """A uint8 view (no copy) of one layout region inside the cache memory."""
        ptr, nb = trr_get_region(self.handle, name)
        off = ptr - self.pool.data_ptr()
        return self.pool[off:off + nb]

    def launches(self) -> int:
        return trr_last_launch_count(self.handle)

    def close(self):
        if getattr(self, "handle", None) is not None and self.handle.value:
            trr_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
