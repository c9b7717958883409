"""Plain fp64 CPU oracle of the TriRoute serving path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline /
reference leg may import this package.  The product path (the CUDA library under
``paper_2607_06601_gb300``) never loads it and shares no code with it.

The arithmetic lives in ``trr_oracle.c`` (quantiser of Sec. 3.2(C) Eq. 4, mode-routed
attention of Sec. 3.2(A) Eq. 2, paged storage of Sec. 3.8 / Sec. 7); this module only
compiles it with gcc and marshals numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "trr_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle_trr.so")

STATUS = {0: "OK", 1: "INVALID_ARG", 2: "OUT_OF_MEMORY", 3: "OUT_OF_PAGES",
          4: "BAD_POSITION", 6: "UNSUPPORTED", 7: "BAD_VALUE"}


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, IEEE semantics: no fast-math, no contraction)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    tmp = _LIB + f".{os.getpid()}.tmp"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                           "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB)
    return _LIB


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        P, I, I64, U64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint64
        L.orc_create.argtypes = [P, ctypes.POINTER(P)]
        L.orc_create.restype = I
        L.orc_destroy.argtypes = [P]
        L.orc_destroy.restype = None
        L.orc_append.argtypes = [P, I, I, P, P, P, P, P, P]
        L.orc_append.restype = I
        L.orc_decode_attn.argtypes = [P, I, I, P, P, P, P, P, I, ctypes.c_double, U64, P]
        L.orc_decode_attn.restype = I
        L.orc_region.argtypes = [P, I, ctypes.POINTER(P)]
        L.orc_region.restype = I64
        L.orc_layout.argtypes = [P, I]
        L.orc_layout.restype = I64
        L.orc_dequant_token.argtypes = [P, I, I, I, I, P, P]
        L.orc_dequant_token.restype = I
        L.orc_quantize_group.argtypes = [P, I, I, P, P, P]
        L.orc_quantize_group.restype = I
        L.orc_pack_codes.argtypes = [P, I, I, P]
        L.orc_pack_codes.restype = None
        L.orc_f16_to_double.argtypes = [ctypes.c_uint16]
        L.orc_f16_to_double.restype = ctypes.c_double
        L.orc_double_to_f16.argtypes = [ctypes.c_double]
        L.orc_double_to_f16.restype = ctypes.c_uint16
        L.orc_bf16_to_double.argtypes = [ctypes.c_uint16]
        L.orc_bf16_to_double.restype = ctypes.c_double
        L.orc_argmax.argtypes = [P, I]
        L.orc_argmax.restype = I
        L.orc_route_decisions.argtypes = [I, P, P, P, I, I, I, I, I, P, P, P, P, P]
        L.orc_route_decisions.restype = I
        _lib = L
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


REGIONS = {"last_pos": 0, "ntok": 1, "presence": 2, "page_table": 3, "page_first": 4,
           "page_last": 5, "next_page": 6, "pool2": 7, "pool4": 8, "pool8": 9, "pool16": 10}


class OracleCache:
    """The oracle's own paged cache (host memory), same documented layout."""

    def __init__(self, num_layers, max_seqs, num_q_heads, num_kv_heads, head_dim,
                 group_size, page_size, max_context, pages_per_class,
                 skip_writes_kv=0, no_pool=False, head_modes=0):
        cfg = np.array([num_layers, max_seqs, num_q_heads, num_kv_heads, head_dim, group_size,
                        page_size, max_context, *pages_per_class, skip_writes_kv,
                        int(no_pool), int(head_modes)], dtype=np.int32)
        self.head_modes = int(head_modes)
        self.Hq, self.Hkv, self.d = num_q_heads, num_kv_heads, head_dim
        self.L, self.S, self.P, self.max_context = num_layers, max_seqs, page_size, max_context
        self._h = ctypes.c_void_p()
        st = lib().orc_create(_ptr(cfg), ctypes.byref(self._h))
        if st != 0:
            lib().orc_destroy(self._h)
            raise RuntimeError(f"orc_create failed: {STATUS.get(st, st)}")

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _lib is not None:
            _lib.orc_destroy(h)
            self._h = None

    def append(self, layer, seq_ids, positions, k_bits, v_bits, bits, modes) -> int:
        """k_bits / v_bits: uint16 bf16 bit patterns [n][Hkv][d]."""
        seq_ids, positions = _c(seq_ids, np.int32), _c(positions, np.int32)
        k, v = _c(k_bits, np.uint16), _c(v_bits, np.uint16)
        bits, modes = _c(bits, np.uint8), _c(modes, np.uint8)
        n = seq_ids.shape[0]
        assert k.size == n * self.Hkv * self.d and v.size == k.size
        assert modes.size == n * (self.Hq if self.head_modes else 1)
        return lib().orc_append(self._h, layer, n, _ptr(seq_ids), _ptr(positions), _ptr(k),
                                _ptr(v), _ptr(bits), _ptr(modes))

    def decode_attn(self, layer, seq_ids, q_positions, q_bits, modes, windows=None,
                    window_scalar=0, scale=0.0, order_seed=0):
        """Returns (status, out) with out float64 [n][Hq][d]."""
        seq_ids, q_positions = _c(seq_ids, np.int32), _c(q_positions, np.int32)
        q, modes = _c(q_bits, np.uint16), _c(modes, np.uint8)
        win = None if windows is None else _c(windows, np.int32)
        n = seq_ids.shape[0]
        assert q.size == n * self.Hq * self.d
        assert modes.size == n * (self.Hq if self.head_modes else 1)
        out = np.zeros((n, self.Hq, self.d), dtype=np.float64)
        st = lib().orc_decode_attn(self._h, layer, n, _ptr(seq_ids), _ptr(q_positions), _ptr(q),
                                   _ptr(modes), _ptr(win), int(window_scalar), float(scale),
                                   int(order_seed), _ptr(out))
        return st, out

    def region(self, name) -> np.ndarray:
        """A copy of one layout region as raw bytes (uint8)."""
        p = ctypes.c_void_p()
        nbytes = lib().orc_region(self._h, REGIONS[name], ctypes.byref(p))
        if nbytes <= 0 or not p.value:
            return np.zeros(0, dtype=np.uint8)
        return np.ctypeslib.as_array((ctypes.c_uint8 * nbytes).from_address(p.value)).copy()

    def layout(self, which: int) -> int:
        return int(lib().orc_layout(self._h, which))

    @property
    def hdr_bytes(self):
        return self.layout(0)

    def slice_bytes(self, c):
        return self.layout(1 + c)

    def page_bytes(self, c):
        return self.layout(5 + c)

    @property
    def mask_bytes(self):
        return self.layout(9)

    def dequant_token(self, layer, seq, pos, kv_head):
        """(class index or -1, k float64[d], v float64[d]) of a stored token; -1 also when
        (with head_modes) the token does not store KV head kv_head."""
        k = np.zeros(self.d, dtype=np.float64)
        v = np.zeros(self.d, dtype=np.float64)
        c = lib().orc_dequant_token(self._h, layer, seq, pos, kv_head, _ptr(k), _ptr(v))
        return c, k, v


def quantize_group(x_bits: np.ndarray, b: int):
    """Eq. 4 on one group of bf16 values: (s16 bits, z16 bits, codes uint8[G], bad)."""
    x = _c(x_bits, np.uint16)
    codes = np.zeros(x.shape[0], dtype=np.uint8)
    s = np.zeros(1, dtype=np.uint16)
    z = np.zeros(1, dtype=np.uint16)
    bad = lib().orc_quantize_group(_ptr(x), x.shape[0], b, _ptr(s), _ptr(z), _ptr(codes))
    return int(s[0]), int(z[0]), codes, bool(bad)


def pack_codes(codes, b: int) -> bytes:
    codes = _c(codes, np.uint8)
    out = np.zeros(codes.shape[0] * b // 8, dtype=np.uint8)
    lib().orc_pack_codes(_ptr(codes), codes.shape[0], b, _ptr(out))
    return out.tobytes()


def f16_to_double(h: int) -> float:
    return lib().orc_f16_to_double(h)


def double_to_f16(x: float) -> int:
    return lib().orc_double_to_f16(x)


def bf16_to_double(h: int) -> float:
    return lib().orc_bf16_to_double(h)


def argmax(z) -> int:
    """The hard decision of one controller head (Sec. 3.8): first maximum, NaN never."""
    z = _c(z, np.float32)
    return int(lib().orc_argmax(_ptr(z), z.shape[0]))


def route_decisions(mode_logits, bit_logits, positions, window, num_q_heads, head_dim,
                    num_kv_heads, skip_writes_kv=0, totals=None):
    """Hard decisions of n tokens and their cost (Sec. 3.5 / 3.8, Appendix C).

    Returns (modes uint8[n], bits uint8[n], attn_flops int64[n], kv_bits int64[n],
    totals int64[4]); ``totals`` (if given) is added to, as the C function does."""
    ml, bl = _c(mode_logits, np.float32), _c(bit_logits, np.float32)
    pos = _c(positions, np.int32)
    n = pos.shape[0]
    assert ml.size == 3 * n and bl.size == 4 * n
    modes = np.zeros(n, dtype=np.uint8)
    bits = np.zeros(n, dtype=np.uint8)
    flops = np.zeros(n, dtype=np.int64)
    mem = np.zeros(n, dtype=np.int64)
    tot = np.zeros(4, dtype=np.int64) if totals is None else _c(totals, np.int64).copy()
    st = lib().orc_route_decisions(n, _ptr(ml), _ptr(bl), _ptr(pos), int(window), int(num_q_heads),
                                   int(head_dim), int(num_kv_heads), int(skip_writes_kv),
                                   _ptr(modes), _ptr(bits), _ptr(flops), _ptr(mem), _ptr(tot))
    if st != 0:
        raise ValueError(f"orc_route_decisions: {STATUS.get(st, st)}")
    return modes, bits, flops, mem, tot
