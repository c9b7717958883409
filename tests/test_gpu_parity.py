"""GPU parity: trr_kv_append must be bit-exact against the oracle (codes, scales, page
tables, presence, headers), and trr_decode_attn within max abs 2e-2 / row-relative
5e-3 of the fp64 oracle, on seeded inputs spanning several pages, work items and a
ragged tail.  Every call goes through the C ABI (libtrr.so)."""
import numpy as np
import pytest
import torch

from paper_2607_06601_gb300 import workloads as wl
from tests._parity import Pair, check_attention, dev

pytestmark = pytest.mark.gpu

SKIP, LOCAL, FULL = 0, 1, 2


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def test_library_is_the_cuda_path():
    from paper_2607_06601_gb300 import trr
    lib = trr.load()
    assert lib._name.endswith("libtrr.so")


def test_tiny_sequential_decode():
    """The tiny workload exactly: append token p, then attend with query p, for every
    position of both sequences (contexts 37 and 130)."""
    spec = wl.SPECS["tiny"]
    ctx = wl.contexts(spec)
    B, P = spec.batch, 16
    maxctx = int(ctx.max())
    caps = [B * (maxctx // P + 2)] * 4
    pair = Pair(1, B, spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size, P,
                maxctx, caps, max_append=64, max_queries=64)
    pols = [wl.policy(spec, 0, s, int(ctx[s])) for s in range(B)]
    kvs = [wl.kv(spec, 0, s, 0, int(ctx[s])) for s in range(B)]
    qs = [wl.q(spec, 0, s, 0, int(ctx[s])) for s in range(B)]
    for p in range(maxctx):
        seqs = [s for s in range(B) if p < ctx[s]]
        bits = [pols[s][0][p] for s in seqs]
        modes = [pols[s][1][p] for s in seqs]
        pair.append(0, seqs, [p] * len(seqs), np.stack([kvs[s][0][p] for s in seqs]),
                    np.stack([kvs[s][1][p] for s in seqs]), bits, modes)
        pair.attend(0, seqs, [p] * len(seqs), np.stack([qs[s][p] for s in seqs]), modes,
                    window_scalar=spec.window)
        if p % 16 == 15 or p == maxctx - 1:
            pair.check_regions()


CONFIGS = [  # d, G, P, Hq, Hkv
    (64, 32, 16, 4, 2),
    (64, 64, 32, 4, 4),
    (64, 32, 64, 2, 1),
    (128, 64, 16, 8, 2),
    (128, 128, 64, 4, 1),
    (128, 32, 16, 4, 4),
]


def _random_setup(rng, d, G, P, Hq, Hkv, ctxs, bits_p=(0.25, 0.25, 0.25, 0.25),
                  modes_p=(0.2, 0.4, 0.4), skip_writes_kv=0, per_call=1024, split_bytes=0, max_queries=1024):
    S = len(ctxs)
    maxctx = max(ctxs) + 8
    caps = [S * (maxctx // P + 2)] * 4
    pair = Pair(1, S, Hq, Hkv, d, G, P, maxctx, caps, skip_writes_kv=skip_writes_kv,
                split_bytes=split_bytes, max_queries=max_queries)
    ent = [(s, p) for p in range(max(ctxs)) for s in range(S) if p < ctxs[s]]
    bits = {(s, p): int(rng.choice([2, 4, 8, 16], p=bits_p)) for s, p in ent}
    modes = {(s, p): int(rng.choice(3, p=modes_p)) for s, p in ent}
    K = {e: rng.standard_normal((Hkv, d), dtype=np.float32) for e in ent}
    V = {e: rng.standard_normal((Hkv, d), dtype=np.float32) for e in ent}
    for i in range(0, len(ent), per_call):
        ch = ent[i:i + per_call]
        pair.append(0, [e[0] for e in ch], [e[1] for e in ch],
                    wl.bf16_bits(np.stack([K[e] for e in ch])), wl.bf16_bits(np.stack([V[e] for e in ch])),
                    [bits[e] for e in ch], [modes[e] for e in ch])
    return pair, ent, bits, modes


@pytest.mark.parametrize("d,G,P,Hq,Hkv", CONFIGS)
def test_ragged_contexts_all_layouts(d, G, P, Hq, Hkv):
    rng = np.random.default_rng(d + G + P + Hq)
    ctxs = [1, 17, 100, 257, 611]
    pair, ent, bits, modes = _random_setup(rng, d, G, P, Hq, Hkv, ctxs)
    pair.check_regions()
    # every sequence queried at many positions, modes and windows mixed, in one call
    seqs, ts, ms, ws = [], [], [], []
    for s, n in enumerate(ctxs):
        for t in sorted(set([0, n - 1, n // 2, max(0, n - 3)] + list(rng.integers(0, n, 6)))):
            for m in (SKIP, LOCAL, FULL):
                seqs.append(s)
                ts.append(t)
                ms.append(m)
                ws.append(int(rng.choice([1, 2, 5, 16, 33, 100, 1000])))
    q = wl.bf16_bits(rng.standard_normal((len(seqs), Hq, d), dtype=np.float32))
    pair.attend(0, seqs, ts, q, ms, windows=ws)


def test_many_splits_and_small_split_bytes():
    """Small split_bytes forces many split-K items per (query, head) and the
    last-arriver merge; queries with one split write their rows directly."""
    rng = np.random.default_rng(12)
    ctxs = [900, 1500, 40]
    pair, ent, _, _ = _random_setup(rng, 64, 32, 16, 4, 4, ctxs, split_bytes=1024)
    q = wl.bf16_bits(rng.standard_normal((6, 4, 64), dtype=np.float32))
    for _ in range(3):  # repeated calls reuse the arrival counters
        pair.attend(0, [0, 1, 2, 0, 1, 2], [899, 1499, 39, 500, 1000, 20],
                    q, [FULL, FULL, FULL, LOCAL, LOCAL, LOCAL], window_scalar=300)


def test_calls_above_one_launch_of_queries_and_an_error_in_the_second():
    """More queries than one launch takes (1024): the call runs as several launches,
    each with its own work units and merges, and an invalid query in the second one is
    reported with its index in the whole call (the lowest failing index)."""
    rng = np.random.default_rng(31)
    ctxs = [70, 260, 130, 33]
    for Hq, Hkv in ((4, 4), (8, 2)):  # CUDA-core and tensor-core consumers
        pair, ent, _, _ = _random_setup(rng, 64, 32, 16, Hq, Hkv, ctxs, split_bytes=1024, max_queries=2048)
        nq = 1100
        seqs = rng.integers(0, len(ctxs), nq)
        ts = np.array([rng.integers(0, ctxs[s]) for s in seqs])
        ms = rng.choice(3, size=nq)
        ws = rng.choice([1, 5, 40, 300], size=nq)
        q = wl.bf16_bits(rng.standard_normal((nq, Hq, 64), dtype=np.float32))
        pair.attend(0, seqs, ts, q, ms, windows=ws)
        bad = ms.copy()
        bad[1050] = 7  # not a mode
        got, ref = pair.attend(0, seqs, ts, q, bad, windows=ws, expect=1)
        assert (got[1050] == 0).all()


def test_bulk_append_with_repeated_sequences_equals_incremental():
    rng = np.random.default_rng(5)
    S, n, d = 3, 300, 64
    a = Pair(1, S, 2, 2, d, 32, 16, n, [S * 30] * 4)
    b = Pair(1, S, 2, 2, d, 32, 16, n, [S * 30] * 4)
    bits = rng.choice([2, 4, 8, 16], size=(S, n))
    modes = rng.choice(3, size=(S, n))
    K = wl.bf16_bits(rng.standard_normal((S, n, 2, d), dtype=np.float32))
    V = wl.bf16_bits(rng.standard_normal((S, n, 2, d), dtype=np.float32))
    ent = [(s, p) for p in range(n) for s in range(S)]
    rng.shuffle(ent)
    ent.sort(key=lambda e: e[1])       # positions increase per sequence, seqs interleaved
    for i in range(0, len(ent), 700):  # 700 entries per call, many per sequence
        ch = ent[i:i + 700]
        ss, pp = [e[0] for e in ch], [e[1] for e in ch]
        a.append(0, ss, pp, K[ss, pp], V[ss, pp], bits[ss, pp], modes[ss, pp])
    for s, p in ent:
        b.append(0, [s], [p], K[s, p:p + 1], V[s, p:p + 1], [bits[s, p]], [modes[s, p]])
    a.check_regions()
    b.check_regions()
    for name in ("page_table", "ntok", "presence", "next_page", "pool2", "pool4", "pool8", "pool16"):
        assert torch.equal(a.gpu.region(name), b.gpu.region(name)), name


def test_edge_cases_and_error_contract():
    rng = np.random.default_rng(3)
    d, Hq, Hkv = 64, 2, 1
    pair = Pair(1, 3, Hq, Hkv, d, 32, 16, 64, [2, 2, 2, 2], max_append=64, max_queries=64)
    K = wl.bf16_bits(rng.standard_normal((40, Hkv, d), dtype=np.float32))
    q = wl.bf16_bits(rng.standard_normal((8, Hq, d), dtype=np.float32))
    # empty calls are no-ops
    pair.append(0, [], [], K[:0], K[:0], [], [])
    pair.attend(0, [], [], q[:0], [])
    # nothing stored yet: every mode gives a zero row
    pair.attend(0, [0, 1, 2], [0, 5, 63], q[:3], [SKIP, LOCAL, FULL], window_scalar=4)
    # skips store nothing
    pair.append(0, [0, 0, 0], [0, 1, 2], K[:3], K[:3], [2, 4, 8], [SKIP, SKIP, SKIP])
    pair.attend(0, [0, 0], [2, 2], q[:2], [LOCAL, FULL], window_scalar=4)
    pair.append(0, [0] * 10, list(range(3, 13)), K[:10], K[10:20], [2, 4, 8, 16, 2, 4, 8, 16, 2, 2],
                [FULL, LOCAL] * 5)
    # windows of 1 (only the query's own position), wider than the context, huge
    pair.attend(0, [0] * 6, [12, 12, 12, 3, 7, 12], q[:6], [LOCAL] * 6, windows=[1, 2, 100, 1, 3, 1 << 30])
    # a query at an older position sees only keys up to it; beyond the last one, all
    pair.attend(0, [0, 0, 0], [5, 9, 63], q[:3], [FULL, LOCAL, FULL], window_scalar=3)
    pair.check_regions()
    # invalid appends: state unchanged, the lowest failing entry's code recorded
    before = {k: pair.gpu.region(k).clone() for k in ("ntok", "page_table", "last_pos", "presence")}
    pair.append(0, [1, 9], [0, 0], K[:2], K[:2], [2, 2], [FULL, FULL], expect=1)
    pair.append(0, [1, 1], [0, 1], K[:2], K[:2], [2, 3], [FULL, FULL], expect=1)
    pair.append(0, [1, 1], [0, 1], K[:2], K[:2], [2, 2], [FULL, 7], expect=1)
    pair.append(0, [1, 1], [5, 5], K[:2], K[:2], [2, 2], [FULL, FULL], expect=4)
    pair.append(0, [1], [64], K[:1], K[:1], [2], [FULL], expect=4)
    pair.append(0, [0], [12], K[:1], K[:1], [2], [FULL], expect=4)
    for k, v in before.items():
        assert torch.equal(v, pair.gpu.region(k)), k
    pair.check_regions()
    # invalid queries: zero rows, the lowest failing index decides the code
    pair.attend(0, [0, 7, 0, 0], [12, 3, 99, 12], q[:4], [FULL, FULL, FULL, 9], expect=1)
    pair.attend(0, [0, 0], [12, 12], q[:2], [LOCAL, FULL], windows=[0, 5], expect=1)
    pair.attend(0, [0, 0], [64, 12], q[:2], [FULL, FULL], expect=4)
    # explicit softmax scale
    pair.attend(0, [0, 0], [12, 12], q[:2], [FULL, LOCAL], window_scalar=5, scale=0.3)
    # pool exhaustion: 2 pages per class; seq 1 and 2 open the remaining 4-bit page, then fail
    pair.append(0, [1] * 16, list(range(16)), K[:16], K[16:32], [4] * 16, [FULL] * 16)
    pair.append(0, [2] * 17, list(range(17)), K[:17], K[17:34], [4] * 17, [FULL] * 17, expect=3)
    pair.check_regions()
    # a non-finite value: that group stored as zeros, BAD_VALUE recorded, the rest applied
    Kn = K[:2].copy()
    Kn[0, 0, 40] = 0x7FC0  # NaN in group 1 of entry 0
    Kn[1, 0, 3] = 0x7F80   # +inf in group 0 of entry 1
    pair.append(0, [2, 2], [0, 1], Kn, K[2:4], [8, 16], [FULL, FULL], expect=7)
    pair.check_regions()


def test_append_rounds_the_exact_quotient_near_half_way_points():
    """Groups built so that (x - z) / s lies on, or within 2^-60 of, a half-way point c + 1/2
    (z = -(c + 1/2), s = 1, x = 0 or +-tiny), mixed with groups of small integers and
    quarter-integers that put exact ties everywhere: the codes must follow the exact
    quotient, bit for bit with the oracle."""
    rng = np.random.default_rng(21)
    d, G, Hkv = 64, 32, 2
    tiny = 2.0 ** -60
    rows, bits = [], []
    for b, cs in ((2, range(3)), (4, range(15)), (8, [127])):
        levels = (1 << b) - 1
        for c in cs:
            tok = np.empty((Hkv, d), dtype=np.float32)
            for h in range(Hkv):
                for g in range(d // G):
                    grp = rng.choice([tiny, -tiny, 0.0, -0.0, 2.0 ** -100, -(2.0 ** -126)], size=G)
                    at = rng.choice(G, size=2, replace=False)
                    grp[at[0]], grp[at[1]] = -(c + 0.5), levels - c - 0.5
                    tok[h, g * G:(g + 1) * G] = grp
            rows.append(tok)
            bits.append(b)
    for _ in range(24):
        b = int(rng.choice([2, 4, 8]))
        rows.append((rng.integers(-40, 40, size=(Hkv, d)) / rng.choice([1, 2, 4])).astype(np.float32))
        bits.append(b)
    n = len(rows)
    K = wl.bf16_bits(np.stack(rows))
    V = wl.bf16_bits(-np.stack(rows[::-1]))
    pair = Pair(1, 1, 2, Hkv, d, G, 16, 128, [8, 8, 8, 8], max_append=128)
    pair.append(0, [0] * n, list(range(n)), K, V, bits, [FULL] * n)
    pair.check_regions()


def test_skip_writes_kv_variant():
    rng = np.random.default_rng(8)
    pair, ent, bits, modes = _random_setup(rng, 64, 32, 16, 2, 2, [50, 200], skip_writes_kv=1)
    pair.check_regions()
    q = wl.bf16_bits(rng.standard_normal((4, 2, 64), dtype=np.float32))
    pair.attend(0, [0, 1, 1, 1], [49, 199, 150, 60], q, [FULL, FULL, LOCAL, SKIP], window_scalar=40)


def _uniform_pair(rng, b, S=4, n=300, Hq=8, Hkv=4, d=64):
    pair = Pair(1, S, Hq, Hkv, d, 32, 16, n, [S * (n // 16 + 2)] * 4)
    K = rng.standard_normal((S, n, Hkv, d), dtype=np.float32)
    V = rng.standard_normal((S, n, Hkv, d), dtype=np.float32)
    for s in range(S):
        for p0 in range(0, n, 256):
            p1 = min(n, p0 + 256)
            pair.append(0, [s] * (p1 - p0), list(range(p0, p1)), wl.bf16_bits(K[s, p0:p1]),
                        wl.bf16_bits(V[s, p0:p1]), [b] * (p1 - p0), [FULL] * (p1 - p0))
    return pair, K, V


def test_all16_full_matches_dense_bf16_attention():
    """Edge run: every token 16-bit and every query full is dense causal attention on
    the bf16 values; checked against torch SDPA (fp32 on the GPU) and the oracle."""
    rng = np.random.default_rng(16)
    S, n, Hq, Hkv, d = 4, 300, 8, 4, 64
    pair, K, V = _uniform_pair(rng, 16, S, n, Hq, Hkv, d)
    pair.check_regions()
    ts = np.array([299, 150, 17, 0])
    q = wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32))
    got, ref = pair.attend(0, range(S), ts, q, [FULL] * S)
    for s in range(S):
        kb = torch.from_numpy(wl.bf16_bits(K[s, :ts[s] + 1])).view(torch.bfloat16).cuda().float()
        vb = torch.from_numpy(wl.bf16_bits(V[s, :ts[s] + 1])).view(torch.bfloat16).cuda().float()
        qb = torch.from_numpy(q[s]).view(torch.bfloat16).cuda().float()
        kx = kb.repeat_interleave(Hq // Hkv, dim=1).permute(1, 0, 2)
        vx = vb.repeat_interleave(Hq // Hkv, dim=1).permute(1, 0, 2)
        sdpa = torch.nn.functional.scaled_dot_product_attention(qb[:, None, :], kx, vx)[:, 0]
        check_attention(got[s], sdpa.double().cpu().numpy())


def test_all2_full():
    rng = np.random.default_rng(2)
    pair, _, _ = _uniform_pair(rng, 2)
    pair.check_regions()
    q = wl.bf16_bits(rng.standard_normal((4, 8, 64), dtype=np.float32))
    pair.attend(0, range(4), [299, 200, 100, 0], q, [FULL] * 4)


def test_chunked_decode_several_queries_per_sequence():
    """Several queries of one sequence in one call (chunked decode, speculative
    verification): each sequence appends a chunk of C tokens in one call, then its C
    queries attend in one call, each up to its own position (causal inside the chunk),
    with mixed modes and windows; chunks repeat so later ones see earlier ones."""
    rng = np.random.default_rng(88)
    S, Hq, Hkv, d, P, C = 4, 8, 8, 64, 32, 8
    ctxs = [300, 64, 129, 1]
    maxctx = max(ctxs) + 3 * C
    pair = Pair(1, S, Hq, Hkv, d, 32, P, maxctx, [S * (maxctx // P + 2)] * 4)

    def chunk(pos_of):  # one append call of every sequence's positions, then their queries
        seqs = np.concatenate([[s] * len(pos_of[s]) for s in range(S)]).astype(np.int32)
        pos = np.concatenate([pos_of[s] for s in range(S)]).astype(np.int32)
        n = len(seqs)
        modes = rng.choice(3, size=n, p=[0.2, 0.4, 0.4])
        pair.append(0, seqs, pos, wl.bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)),
                    wl.bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)),
                    rng.choice([2, 4, 8, 16], size=n), modes)
        return seqs, pos, modes

    chunk([np.arange(c) for c in ctxs])  # the prefilled contexts
    nxt = list(ctxs)
    for _ in range(3):
        seqs, pos, modes = chunk([np.arange(nxt[s], nxt[s] + C) for s in range(S)])
        q = wl.bf16_bits(rng.standard_normal((len(seqs), Hq, d), dtype=np.float32))
        pair.attend(0, seqs, pos, q, modes, windows=rng.choice([1, 3, 8, 40, 500], size=len(seqs)))
        nxt = [x + C for x in nxt]
    pair.check_regions()
