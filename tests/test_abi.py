"""The C-ABI library loads on a machine without a GPU, exports every entry point that
include/trr.h declares, and validates configurations on the host."""
import ctypes
import os
import re

import pytest

from paper_2607_06601_gb300 import build, trr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    text = open(os.path.join(ROOT, "include", "trr.h")).read()
    return sorted(set(re.findall(r"^\s*(?:TRR_API\s+)?(?:trr_status|int32_t)\s+(trr_\w+)\s*\(", text, re.M)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return trr.load()


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 9
    for name in names:
        assert hasattr(lib, name), name
    assert set(names) == set(trr.EXPORTS)


def test_library_has_only_sm103a_code():
    path = build.build()
    assert path.endswith("libtrr.so") and os.path.getsize(path) > 0
    assert "arch=compute_103a,code=sm_103a" in " ".join(build.NVCC_FLAGS)


def test_host_validation_without_gpu(lib):
    ok = trr.make_config(2, 8, 8, 2, 64, 32, 16, 1024, [10, 20, 30, 40])
    need = trr.trr_cache_required_bytes(ok)
    # the pools alone: cap * roundup(128 + Hkv * P * tokb, 128) per class
    tokb = [2 * (64 * b // 8) + 2 * 2 * 4 for b in (2, 4, 8)] + [4 * 64]
    pools = sum(cap * (-(-(128 + 2 * 16 * t) // 128) * 128) for cap, t in zip([10, 20, 30, 40], tokb))
    assert need > pools
    bad = [
        (dict(head_dim=96), 6), (dict(group_size=16), 6), (dict(group_size=128), 6),
        (dict(page_size=8), 6), (dict(num_q_heads=6, num_kv_heads=4), 6),
        (dict(max_append=2048), 6), (dict(num_layers=0), 1), (dict(max_context=0), 1),
    ]
    base = dict(num_layers=2, max_seqs=8, num_q_heads=8, num_kv_heads=2, head_dim=64,
                group_size=32, page_size=16, max_context=1024, pages_per_class=[10] * 4)
    for change, code in bad:
        kw = dict(base, **change)
        cfg = trr.make_config(**kw)
        out = ctypes.c_uint64()
        assert lib.trr_cache_required_bytes(ctypes.byref(cfg), ctypes.byref(out)) == code, change
    # calls on a NULL cache fail on the host without touching CUDA
    assert lib.trr_destroy(None) == 0
    assert lib.trr_kv_append(None, 0, 0, None, None, None, None, None, None, None) == 1
    assert lib.trr_decode_attn(None, 0, 0, None, None, None, None, None, 0, 0.0, None, None) == 1
    assert lib.trr_last_launch_count(None) == 0


def test_per_head_layout_matches_the_oracle(lib):
    """With head_modes the library's pages grow by the presence masks exactly as the
    oracle lays them out (16 bytes per KV head slice, pages rounded to 128): the required
    bytes differ from the per-token cache's by the pools' difference alone."""
    import oracle
    base = dict(num_layers=2, max_seqs=8, num_q_heads=12, num_kv_heads=4, head_dim=64,
                group_size=32, page_size=32, max_context=1024, pages_per_class=[10, 20, 30, 40])
    tok = trr.trr_cache_required_bytes(trr.make_config(**base))
    hed = trr.trr_cache_required_bytes(trr.make_config(**base, head_modes=1))
    o0 = oracle.OracleCache(1, 1, 12, 4, 64, 32, 32, 64, [1] * 4, no_pool=True)
    o1 = oracle.OracleCache(1, 1, 12, 4, 64, 32, 32, 64, [1] * 4, no_pool=True, head_modes=1)
    grow = sum(cap * (o1.page_bytes(c) - o0.page_bytes(c)) for c, cap in enumerate(base["pages_per_class"]))
    assert grow > 0 and o1.slice_bytes(0) == o0.slice_bytes(0) + 16
    # the pools are 256-byte aligned regions: the difference is the pools' own up to that
    assert abs((hed - tok) - grow) < 4 * 256
    cfg = trr.make_config(**base, head_modes=2)
    out = ctypes.c_uint64()
    assert lib.trr_cache_required_bytes(ctypes.byref(cfg), ctypes.byref(out)) == 6  # not a mode setting
