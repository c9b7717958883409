"""GPU parity at the workloads' full sizes, in the cache configuration bench.py times
(page 32, default split size), on every row.

A decode step of one layer (or of every layer of the 24-layer sweep) is built the way a
server builds it: each sequence's context goes into the cache through trr_kv_append,
then one call appends the next token of every sequence and one call attends with every
sequence's query in its seeded mode; two more calls query every sequence in full and in
local mode.

- All metadata (last positions, counts, presence, page tables, page first/last
  positions, next page ids) is compared bit for bit with a metadata-only oracle fed the
  same calls.
- Every sequence is rebuilt alone in the oracle (in worker processes: the oracle's
  per-sequence work is independent): every page of every sequence, taken in page-table
  order, must be byte-identical (compared by 128-bit digests), and every attention row
  of the three calls must meet the stated tolerance.  Skip rows are exact zeros.
"""
import concurrent.futures as cf
import hashlib
import multiprocessing as mp
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_06601_gb300 import trr, workloads as wl
from tests._parity import REGION_NAMES, check_attention, dev

pytestmark = pytest.mark.gpu

P = 32
SKIP, LOCAL, FULL = 0, 1, 2
BITS = (2, 4, 8, 16)


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


@pytest.fixture(scope="module")
def workers():
    """Oracle worker processes (spawned: a forked child of a CUDA process can hang)."""
    n = max(1, min(16, (os.cpu_count() or 2) - 1))
    with cf.ProcessPoolExecutor(n, mp_context=mp.get_context("spawn")) as ex:
        yield ex


def _digest(b: bytes) -> bytes:
    return hashlib.blake2b(b, digest_size=16).digest()


def _caps(bits, modes):
    return [-(-int(np.count_nonzero((modes != SKIP) & (bits == b))) // P) + 1 for b in BITS]


def _oracle_sequence(job):
    """One sequence alone in the oracle: its page digests per class in page-table order,
    its token counts, and its decode query's rows in the seeded mode, full and local."""
    name, batch, layer, s, n, q_row = job
    spec = wl.SPECS[name].with_(batch=batch)
    bits, modes = wl.policy(spec, layer, s, n)
    k, v = wl.kv(spec, layer, s, 0, n)
    o = oracle.OracleCache(1, 1, spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size,
                           P, n, _caps(bits, modes))
    for p0 in range(0, n, 4096):
        p1 = min(n, p0 + 4096)
        assert o.append(0, [0] * (p1 - p0), np.arange(p0, p1), k[p0:p1], v[p0:p1], bits[p0:p1],
                        modes[p0:p1]) == 0
    ntok = o.region("ntok").view(np.int32).reshape(4).copy()
    pt = o.region("page_table").view(np.int32).reshape(4, -1)
    digests = []
    for c, b in enumerate(BITS):
        pb = o.page_bytes(c)
        pool = o.region(f"pool{b}")
        digests.append([_digest(pool[int(i) * pb:(int(i) + 1) * pb].tobytes())
                        for i in pt[c, :-(-int(ntok[c]) // P)]])
    t = n - 1
    rows = []
    for m in (int(modes[t]), FULL, LOCAL):
        st, ref = o.decode_attn(0, [0], [t], q_row[None], [m], window_scalar=spec.window)
        assert st == 0
        rows.append(ref[0])
    return s, ntok, digests, np.stack(rows)


def _inputs(spec, layer, s, n):
    bits, modes = wl.policy(spec, layer, s, n)
    k, v = wl.kv(spec, layer, s, 0, n)
    q = wl.q(spec, layer, s, n - 1, n)[0]
    return bits, modes, k, v, q


def _in_order(fn, items, threads=8, window=24):
    """fn over items on a thread pool (numpy's generators release the GIL), results in
    order, at most `window` held at a time."""
    items = list(items)
    with cf.ThreadPoolExecutor(threads) as ex:
        futs = [ex.submit(fn, *it) for it in items[:window]]
        for i in range(len(items)):
            if i + window < len(items):
                futs.append(ex.submit(fn, *items[i + window]))
            yield futs[i].result()
            futs[i] = None


def _gpu_pages(pt_all, pools, page_bytes, s, layer, ntok):
    """Digests of sequence s's pages at `layer` in the GPU cache's page table and pools
    (copied to the host), per class, in page order."""
    pt = pt_all[layer, s]
    out = []
    for c in range(4):
        pb = page_bytes[c]
        pool = pools[c]
        out.append([_digest(pool[int(i) * pb:(int(i) + 1) * pb].tobytes())
                    for i in pt[c, :-(-int(ntok[c]) // P)]])
    return out


def _full_size(name, workers, batch=None, layers=1, step=True):
    """step: the decode step is one trr_decode_step call (append and attention in the
    seeded modes); else trr_kv_append then trr_decode_attn."""
    spec = wl.SPECS[name]
    B = batch or spec.batch
    spec = spec.with_(batch=B)
    ctx = wl.contexts(spec)
    maxctx = int(ctx.max())
    Hq, Hkv, d, G = spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size
    caps = [0, 0, 0, 0]
    for layer in range(layers):
        for s in range(B):
            bits, modes = wl.policy(spec, layer, s, int(ctx[s]))
            caps = [a + b for a, b in zip(caps, _caps(bits, modes))]
    gpu = trr.Cache(layers, B, Hq, Hkv, d, G, P, maxctx, caps, max_append=1024, max_queries=max(B, 64),
                    zero_pool=True)
    meta = oracle.OracleCache(layers, B, Hq, Hkv, d, G, P, maxctx, caps, no_pool=True)
    steps = []
    for layer in range(layers):
        last = []
        # each sequence's context but its last token, one sequence at a time
        for s, (bits, modes, k, v, q) in enumerate(
                _in_order(_inputs, [(spec, layer, s, int(ctx[s])) for s in range(B)])):
            n = int(ctx[s])
            for p0 in range(0, n - 1, 1024):
                p1 = min(n - 1, p0 + 1024)
                seqs, pos = np.full(p1 - p0, s, np.int32), np.arange(p0, p1, dtype=np.int32)
                gpu.append(layer, dev(seqs, torch.int32), dev(pos, torch.int32), dev(k[p0:p1], torch.bfloat16),
                           dev(v[p0:p1], torch.bfloat16), dev(bits[p0:p1], torch.uint8),
                           dev(modes[p0:p1], torch.uint8))
                assert meta.append(layer, seqs, pos, k[p0:p1], v[p0:p1], bits[p0:p1], modes[p0:p1]) == 0
            last.append((k[n - 1], v[n - 1], bits[n - 1], modes[n - 1], q))
        # the decode step: every sequence's next token, then every query
        t = (ctx - 1).astype(np.int32)
        seqs = np.arange(B, dtype=np.int32)
        k1 = np.stack([x[0] for x in last])
        v1 = np.stack([x[1] for x in last])
        b1 = np.array([x[2] for x in last], dtype=np.uint8)
        m1 = np.array([x[3] for x in last], dtype=np.uint8)
        q = np.stack([x[4] for x in last])
        outs = []
        if step:
            out = gpu.decode_step(layer, dev(seqs, torch.int32), dev(t, torch.int32), dev(k1, torch.bfloat16),
                                  dev(v1, torch.bfloat16), dev(b1, torch.uint8), dev(m1, torch.uint8),
                                  dev(q, torch.bfloat16), window_scalar=spec.window)
            outs.append(out.float().cpu().numpy().astype(np.float64))
        else:
            gpu.append(layer, dev(seqs, torch.int32), dev(t, torch.int32), dev(k1, torch.bfloat16),
                       dev(v1, torch.bfloat16), dev(b1, torch.uint8), dev(m1, torch.uint8))
        assert meta.append(layer, seqs, t, k1, v1, b1, m1) == 0
        for mm in ([] if step else [m1]) + [np.full(B, FULL, np.uint8), np.full(B, LOCAL, np.uint8)]:
            out = gpu.decode_attn(layer, dev(seqs, torch.int32), dev(t, torch.int32), dev(q, torch.bfloat16),
                                  dev(mm, torch.uint8), window_scalar=spec.window)
            outs.append(out.float().cpu().numpy().astype(np.float64))
        assert gpu.status() == 0
        steps.append((layer, m1, q, np.stack(outs, axis=1)))  # [B][3][Hq][d]
    torch.cuda.synchronize()
    for name_ in REGION_NAMES:
        assert np.array_equal(gpu.region(name_).cpu().numpy(), meta.region(name_)), name_
    pools = [gpu.region(f"pool{b}").cpu().numpy() for b in BITS]
    page_bytes = [meta.page_bytes(c) for c in range(4)]
    ntok_all = gpu.region("ntok").cpu().numpy().view(np.int32).reshape(layers, B, 4)
    pt_all = gpu.region("page_table").cpu().numpy().view(np.int32).reshape(layers, B, 4, -(-maxctx // P))
    for layer, m1, q, got in steps:
        assert (got[m1 == SKIP, 0] == 0).all()
        jobs = [(name, B, layer, s, int(ctx[s]), q[s]) for s in range(B)]
        for s, ntok, digests, ref in workers.map(_oracle_sequence, jobs):
            assert np.array_equal(ntok_all[layer, s], ntok), (layer, s)
            gd = _gpu_pages(pt_all, pools, page_bytes, s, layer, ntok)
            for c in range(4):
                if gd[c] != digests[c]:
                    bad = [i for i, (x, y) in enumerate(zip(gd[c], digests[c])) if x != y]
                    raise AssertionError(f"layer {layer} seq {s} class {BITS[c]}: pages {bad[:8]} differ")
            check_attention(got[s], ref, [int(m1[s]), FULL, LOCAL])


def test_160m_decode_step_full_size(workers):
    _full_size("160m", workers)


def test_160m_separate_append_and_attention_full_size(workers):
    _full_size("160m", workers, step=False)


def test_1p3b_ragged_decode_step_full_size(workers):
    _full_size("1p3b", workers)


def test_gqa_long_context_decode_step_full_size(workers):
    _full_size("gqa_long", workers)


@pytest.mark.parametrize("batch", [1, 8, 64, 256])
def test_sweep_layer_full_size(workers, batch):
    """The sweep's batch points at context 4096, one layer."""
    _full_size("sweep", workers, batch=batch)


def test_sweep_24_layer_step(workers):
    """A whole 24-layer sweep step (independent seeded maps per layer) at batch 8."""
    _full_size("sweep", workers, batch=8, layers=24)


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
    for s in range(B):
        o = oracle.OracleCache(1, 1, Hq, Hq, d, spec.group_size, P, n, [n // P + 2] * 4)
        assert o.append(0, [0] * n, np.arange(n), wl.bf16_bits(K[s]), wl.bf16_bits(V[s]), [b] * n, [FULL] * n) == 0
        st, ref = o.decode_attn(0, [0], [n - 1], q[s:s + 1], [FULL])
        assert st == 0
        check_attention(got[s:s + 1], ref, [FULL])
    if b == 16:
        for s in range(B):
            kb = torch.from_numpy(wl.bf16_bits(K[s])).view(torch.bfloat16).cuda().float().permute(1, 0, 2)
            vb = torch.from_numpy(wl.bf16_bits(V[s])).view(torch.bfloat16).cuda().float().permute(1, 0, 2)
            qb = torch.from_numpy(q[s]).view(torch.bfloat16).cuda().float()[:, None, :]
            sdpa = torch.nn.functional.scaled_dot_product_attention(qb, kb, vb)[:, 0]
            check_attention(got[s], sdpa.double().cpu().numpy())
