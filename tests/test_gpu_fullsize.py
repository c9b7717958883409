"""GPU parity at the workloads' full sizes, in the cache configuration bench.py times
(page 32, default split size): the whole batch of one layer is built through
trr_kv_append, then one decode step appends the next token of every sequence and
attends with every sequence's query.

- All metadata (last positions, counts, presence, page tables, page first/last
  positions, next page ids) is compared bit for bit with a metadata-only oracle fed the
  same calls.
- For sampled sequences (one full, one local and one skip query where the seeded maps
  have them) the oracle builds that sequence alone: every page of the sequence, taken in
  page-table order, must be byte-identical, and the sequence's attention row must meet
  the stated tolerance.
- Every skip row is exactly zero.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_06601_gb300 import trr, workloads as wl
from tests._parity import REGION_NAMES, check_attention, dev

pytestmark = pytest.mark.gpu

P = 32
SKIP, LOCAL, FULL = 0, 1, 2


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def _build(spec, layer=0, batch=None):
    """GPU cache + metadata-only oracle of one layer, contexts prebuilt with the last
    position held back for the decode step."""
    B = batch or spec.batch
    ctx = wl.contexts(spec)[:B]
    maxctx = int(ctx.max())
    pols = [wl.policy(spec, layer, s, int(ctx[s])) for s in range(B)]
    caps = [0, 0, 0, 0]
    for bits, modes in pols:
        for c, b in enumerate((2, 4, 8, 16)):
            caps[c] += -(-int(np.count_nonzero((modes != SKIP) & (bits == b))) // P) + 1
    Hq, Hkv, d, G = spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size
    gpu = trr.Cache(1, B, Hq, Hkv, d, G, P, maxctx, caps, max_append=1024, max_queries=max(B, 64),
                    zero_pool=True)
    meta = oracle.OracleCache(1, B, Hq, Hkv, d, G, P, maxctx, caps, no_pool=True)
    kvs = {}
    per = max(1, 1024 // B)
    for p0 in range(0, maxctx - 1, per):
        ent = [(s, p) for p in range(p0, min(maxctx - 1, p0 + per)) for s in range(B) if p < ctx[s] - 1]
        if not ent:
            continue
        for s in {e[0] for e in ent}:
            if s not in kvs:
                kvs[s] = wl.kv(spec, layer, s, 0, int(ctx[s]))
        seqs = np.array([e[0] for e in ent], dtype=np.int32)
        pos = np.array([e[1] for e in ent], dtype=np.int32)
        k = np.stack([kvs[s][0][p] for s, p in ent])
        v = np.stack([kvs[s][1][p] for s, p in ent])
        bits = np.array([pols[s][0][p] for s, p in ent], dtype=np.uint8)
        modes = np.array([pols[s][1][p] for s, p in ent], dtype=np.uint8)
        gpu.append(layer, dev(seqs, torch.int32), dev(pos, torch.int32), dev(k, torch.bfloat16),
                   dev(v, torch.bfloat16), dev(bits, torch.uint8), dev(modes, torch.uint8))
        assert meta.append(layer, seqs, pos, k, v, bits, modes) == 0
    for s in range(B):
        if s not in kvs:
            kvs[s] = wl.kv(spec, layer, s, 0, int(ctx[s]))
    return gpu, meta, ctx, pols, kvs


def _decode_step(spec, gpu, meta, ctx, pols, kvs, layer=0):
    B = len(ctx)
    t = (ctx - 1).astype(np.int32)
    seqs = np.arange(B, dtype=np.int32)
    k = np.stack([kvs[s][0][t[s]] for s in range(B)])
    v = np.stack([kvs[s][1][t[s]] for s in range(B)])
    bits = np.array([pols[s][0][t[s]] for s in range(B)], dtype=np.uint8)
    modes = np.array([pols[s][1][t[s]] for s in range(B)], dtype=np.uint8)
    gpu.append(layer, dev(seqs, torch.int32), dev(t, torch.int32), dev(k, torch.bfloat16),
               dev(v, torch.bfloat16), dev(bits, torch.uint8), dev(modes, torch.uint8))
    assert meta.append(layer, seqs, t, k, v, bits, modes) == 0
    q = np.stack([wl.q(spec, layer, s, int(t[s]), int(t[s]) + 1)[0] for s in range(B)])
    out = gpu.decode_attn(layer, dev(seqs, torch.int32), dev(t, torch.int32), dev(q, torch.bfloat16),
                          dev(modes, torch.uint8), window_scalar=spec.window)
    assert gpu.status() == 0
    return t, modes, q, out.float().cpu().numpy().astype(np.float64)


def _sample(modes):
    picks = []
    for m in (FULL, LOCAL, SKIP):
        idx = np.nonzero(modes == m)[0]
        if idx.size:
            picks.append(int(idx[0]))
    return picks


def _check_sequence(spec, gpu, ctx, pols, kvs, s, t, mode, q, got_row, layer=0):
    """Oracle of sequence s alone: page bytes in page-table order, and attention."""
    n = int(ctx[s])
    bits, modes = pols[s]
    Hq, Hkv, d, G = spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size
    caps = [-(-int(np.count_nonzero((modes != SKIP) & (bits == b))) // P) + 1 for b in (2, 4, 8, 16)]
    o = oracle.OracleCache(1, 1, Hq, Hkv, d, G, P, n, caps)
    for p0 in range(0, n, 4096):
        p1 = min(n, p0 + 4096)
        assert o.append(0, [0] * (p1 - p0), np.arange(p0, p1), kvs[s][0][p0:p1], kvs[s][1][p0:p1],
                        bits[p0:p1], modes[p0:p1]) == 0
    MPg = -(-gpu.max_context // P)
    ntok = gpu.region("ntok").cpu().numpy().view(np.int32).reshape(-1, 4)[s]
    pt_g = gpu.region("page_table").cpu().numpy().view(np.int32).reshape(-1, 4, MPg)[s]
    ntok_o = o.region("ntok").view(np.int32).reshape(4)
    pt_o = o.region("page_table").view(np.int32).reshape(4, -1)
    assert np.array_equal(ntok, ntok_o)
    for c, b in enumerate((2, 4, 8, 16)):
        pb = o.page_bytes(c)
        pool_g = gpu.region(f"pool{b}")
        pool_o = o.region(f"pool{b}")
        for kk in range(-(-int(ntok[c]) // P)):
            gid, oid = int(pt_g[c, kk]), int(pt_o[c, kk])
            g_bytes = pool_g[gid * pb:(gid + 1) * pb].cpu().numpy()
            o_bytes = pool_o[oid * pb:(oid + 1) * pb]
            if not np.array_equal(g_bytes, o_bytes):
                bad = np.nonzero(g_bytes != o_bytes)[0]
                raise AssertionError(f"seq {s} class {b} page {kk}: {bad.size} bytes differ, first at {bad[0]}")
    st, ref = o.decode_attn(0, [0], [t], q[None], [mode], window_scalar=spec.window)
    assert st == 0
    check_attention(got_row[None], ref, [mode])


def _full_size_case(spec, batch=None):
    gpu, meta, ctx, pols, kvs = _build(spec, batch=batch)
    t, modes, q, out = _decode_step(spec, gpu, meta, ctx, pols, kvs)
    torch.cuda.synchronize()
    for name in REGION_NAMES:
        assert np.array_equal(gpu.region(name).cpu().numpy(), meta.region(name)), name
    assert (out[modes == SKIP] == 0).all()
    for s in _sample(modes):
        _check_sequence(spec, gpu, ctx, pols, kvs, s, int(t[s]), int(modes[s]), q[s], out[s])
    # the sampled sequences under the other modes too
    for s in _sample(modes)[:1]:
        for m in (LOCAL, FULL):
            qs = dev(q[s:s + 1], torch.bfloat16)
            row = gpu.decode_attn(0, dev(np.array([s], np.int32), torch.int32),
                                  dev(np.array([t[s]], np.int32), torch.int32), qs,
                                  dev(np.array([m], np.uint8), torch.uint8), window_scalar=spec.window)
            _check_sequence(spec, gpu, ctx, pols, kvs, s, int(t[s]), m, q[s],
                            row.float().cpu().numpy().astype(np.float64)[0])


def test_160m_decode_step_full_size():
    _full_size_case(wl.SPECS["160m"])


def test_1p3b_ragged_decode_step_full_size():
    _full_size_case(wl.SPECS["1p3b"])


def test_gqa_long_context_decode_step_full_size():
    _full_size_case(wl.SPECS["gqa_long"])


def test_sweep_layer_batch8_full_size():
    _full_size_case(wl.SPECS["sweep"], batch=8)


@pytest.mark.parametrize("b", [16, 2])
def test_sweep_edge_runs_uniform_width_all_full(b):
    """Edge runs of the 24-layer sweep at context 4096: every token at one width, every
    query full.  All-16 must equal dense bf16 attention (torch SDPA, fp32 on the GPU)."""
    spec = wl.SPECS["sweep"]
    B, n = 4, 4096
    Hq, d = spec.num_q_heads, spec.head_dim
    rng = np.random.default_rng(100 + b)
    caps = [B * (n // P + 2)] * 4
    gpu = trr.Cache(1, B, Hq, Hq, d, spec.group_size, P, n, caps, max_append=1024, zero_pool=True)
    K = rng.standard_normal((B, n, Hq, d), dtype=np.float32)
    V = rng.standard_normal((B, n, Hq, d), dtype=np.float32)
    for s in range(B):
        for p0 in range(0, n, 1024):
            gpu.append(0, dev(np.full(1024, s, np.int32), torch.int32), dev(np.arange(p0, p0 + 1024, dtype=np.int32), torch.int32),
                       dev(wl.bf16_bits(K[s, p0:p0 + 1024]), torch.bfloat16), dev(wl.bf16_bits(V[s, p0:p0 + 1024]), torch.bfloat16),
                       dev(np.full(1024, b, np.uint8), torch.uint8), dev(np.full(1024, FULL, np.uint8), torch.uint8))
    q = wl.bf16_bits(rng.standard_normal((B, Hq, d), dtype=np.float32))
    t = np.full(B, n - 1, np.int32)
    out = gpu.decode_attn(0, dev(np.arange(B, dtype=np.int32), torch.int32), dev(t, torch.int32),
                          dev(q, torch.bfloat16), dev(np.full(B, FULL, np.uint8), torch.uint8))
    assert gpu.status() == 0
    got = out.float().cpu().numpy().astype(np.float64)
    s = 1
    o = oracle.OracleCache(1, 1, Hq, Hq, d, spec.group_size, P, n, [n // P + 2] * 4)
    assert o.append(0, [0] * n, np.arange(n), wl.bf16_bits(K[s]), wl.bf16_bits(V[s]), [b] * n, [FULL] * n) == 0
    st, ref = o.decode_attn(0, [0], [n - 1], q[s:s + 1], [FULL])
    check_attention(got[s:s + 1], ref, [FULL])
    if b == 16:
        for s in range(B):
            kb = torch.from_numpy(wl.bf16_bits(K[s])).view(torch.bfloat16).cuda().float().permute(1, 0, 2)
            vb = torch.from_numpy(wl.bf16_bits(V[s])).view(torch.bfloat16).cuda().float().permute(1, 0, 2)
            qb = torch.from_numpy(q[s]).view(torch.bfloat16).cuda().float()[:, None, :]
            sdpa = torch.nn.functional.scaled_dot_product_attention(qb, kb, vb)[:, 0]
            check_attention(got[s], sdpa.double().cpu().numpy())
