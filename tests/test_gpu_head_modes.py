"""GPU parity of per-head attention modes (Sec. 3.2(A): a mode per head by default; the
router's mode logits are [B, T, H, |A|] in Appendix C).  A cache created with
head_modes takes modes[n][Hq] in trr_kv_append and trr_decode_attn: a token stores KV
head j when a query head reading it does not skip, and every page carries a 64-bit
presence mask per KV head.  Against the oracle (head_modes=1): the append bit-exact
(metadata, page bytes, presence masks) and attention within max abs 2e-2 / row-relative
5e-3, skip heads bit-zero.  Every call goes through the C ABI (libtrr.so)."""
import numpy as np
import pytest
import torch

from paper_2607_06601_gb300 import trr
from paper_2607_06601_gb300 import workloads as wl
from tests._parity import Pair, check_attention, dev

pytestmark = pytest.mark.gpu

SKIP, LOCAL, FULL = 0, 1, 2


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def test_tiny_sequential_decode_per_head():
    """The tiny workload (4 query / 2 KV heads) with a mode per (token, head): append
    token p, then attend with query p, for every position of both sequences."""
    spec = wl.SPECS["tiny"]
    ctx = wl.contexts(spec)
    B, P, Hq = spec.batch, 16, spec.num_q_heads
    maxctx = int(ctx.max())
    pair = Pair(1, B, Hq, spec.num_kv_heads, spec.head_dim, spec.group_size, P, maxctx,
                [B * (maxctx // P + 2)] * 4, max_append=64, max_queries=64, head_modes=1)
    pols = [wl.head_policy(spec, 0, s, int(ctx[s])) for s in range(B)]
    kvs = [wl.kv(spec, 0, s, 0, int(ctx[s])) for s in range(B)]
    qs = [wl.q(spec, 0, s, 0, int(ctx[s])) for s in range(B)]
    for p in range(maxctx):
        seqs = [s for s in range(B) if p < ctx[s]]
        hm = np.stack([pols[s][1][p] for s in seqs])
        pair.append(0, seqs, [p] * len(seqs), np.stack([kvs[s][0][p] for s in seqs]),
                    np.stack([kvs[s][1][p] for s in seqs]), [pols[s][0][p] for s in seqs], hm)
        pair.attend(0, seqs, [p] * len(seqs), np.stack([qs[s][p] for s in seqs]), hm,
                    window_scalar=spec.window)
        if p % 16 == 15 or p == maxctx - 1:
            pair.check_regions()


# d, G, P, Hq, Hkv: MHA and query groups, including blocks of 4 query heads whose first
# KV head is odd (g = 4 and g = 3) and 16-bit pages whose KV heads take one stage each
# (d 128, P 64)
LAYOUTS = [
    (64, 32, 16, 4, 2),
    (64, 32, 32, 12, 12),
    (64, 32, 16, 8, 2),
    (64, 64, 32, 12, 4),
    (128, 64, 64, 8, 8),
    (128, 128, 16, 4, 1),
]


def _setup(rng, d, G, P, Hq, Hkv, ctxs, per_call, skip_p=0.3, skip_writes_kv=0, split_bytes=0):
    S = len(ctxs)
    maxctx = max(ctxs) + 8
    pair = Pair(1, S, Hq, Hkv, d, G, P, maxctx, [S * (maxctx // P + 2)] * 4,
                skip_writes_kv=skip_writes_kv, split_bytes=split_bytes, head_modes=1)
    ent = [(s, p) for p in range(max(ctxs)) for s in range(S) if p < ctxs[s]]
    mp = ((skip_p, (1 - skip_p) / 2, (1 - skip_p) / 2))
    bits = {e: int(rng.choice([2, 4, 8, 16])) for e in ent}
    hmod = {e: rng.choice(3, size=Hq, p=mp).astype(np.uint8) for e in ent}
    for e in ent[::7]:
        hmod[e][:] = SKIP  # tokens no head reads: no slot at all
    K = {e: rng.standard_normal((Hkv, d), dtype=np.float32) for e in ent}
    V = {e: rng.standard_normal((Hkv, d), dtype=np.float32) for e in ent}
    for i in range(0, len(ent), per_call):
        ch = ent[i:i + per_call]
        pair.append(0, [e[0] for e in ch], [e[1] for e in ch],
                    wl.bf16_bits(np.stack([K[e] for e in ch])), wl.bf16_bits(np.stack([V[e] for e in ch])),
                    [bits[e] for e in ch], np.stack([hmod[e] for e in ch]))
    return pair


def _queries(rng, ctxs, Hq):
    seqs, ts, hm, ws = [], [], [], []
    for s, n in enumerate(ctxs):
        for t in sorted(set([0, n - 1, n // 2, max(0, n - 3)] + list(rng.integers(0, n, 5)))):
            for kind in range(4):
                seqs.append(s)
                ts.append(t)
                if kind == 0:
                    hm.append(rng.choice(3, size=Hq).astype(np.uint8))  # mixed heads
                elif kind == 1:
                    hm.append(np.full(Hq, LOCAL, dtype=np.uint8))  # all local
                elif kind == 2:
                    m = np.full(Hq, SKIP, dtype=np.uint8)  # one head reads, the rest skip
                    m[rng.integers(Hq)] = FULL
                    hm.append(m)
                else:
                    hm.append(np.full(Hq, SKIP, dtype=np.uint8))  # every head skips
                ws.append(int(rng.choice([1, 2, 5, 16, 33, 100, 1000])))
    return seqs, ts, np.stack(hm), ws


@pytest.mark.parametrize("per_call", [1024, 200])  # the two-kernel and the one-kernel append
@pytest.mark.parametrize("d,G,P,Hq,Hkv", LAYOUTS)
def test_ragged_contexts_per_head(d, G, P, Hq, Hkv, per_call):
    rng = np.random.default_rng(d + G + P + Hq + Hkv + per_call)
    ctxs = [1, 17, 100, 257, 611]
    pair = _setup(rng, d, G, P, Hq, Hkv, ctxs, per_call)
    pair.check_regions()
    seqs, ts, hm, ws = _queries(rng, ctxs, Hq)
    q = wl.bf16_bits(rng.standard_normal((len(seqs), Hq, d), dtype=np.float32))
    pair.attend(0, seqs, ts, q, hm, windows=ws)


def test_many_splits_per_head():
    """Small split_bytes: long queries cut into many splits whose head blocks have
    different key ranges (a full head beside local and skip heads)."""
    rng = np.random.default_rng(44)
    ctxs = [900, 1500, 40]
    pair = _setup(rng, 64, 32, 16, 8, 8, ctxs, 1024, split_bytes=1024)
    hm = np.array([[FULL, LOCAL, SKIP, LOCAL, SKIP, SKIP, SKIP, SKIP],
                   [LOCAL] * 4 + [FULL] * 4,
                   [SKIP, FULL, SKIP, SKIP, LOCAL, LOCAL, SKIP, FULL],
                   [FULL] * 8, [LOCAL] * 8, [SKIP] * 7 + [LOCAL]], dtype=np.uint8)
    q = wl.bf16_bits(rng.standard_normal((6, 8, 64), dtype=np.float32))
    for _ in range(3):  # repeated calls reuse the arrival counters
        pair.attend(0, [0, 1, 2, 1, 0, 1], [899, 1499, 39, 1000, 500, 1200], q, hm, window_scalar=300)


def test_skip_writes_kv_with_head_modes():
    rng = np.random.default_rng(9)
    pair = _setup(rng, 64, 32, 16, 4, 2, [50, 200], 1024, skip_writes_kv=1)
    pair.check_regions()
    q = wl.bf16_bits(rng.standard_normal((3, 4, 64), dtype=np.float32))
    hm = np.array([[FULL, SKIP, LOCAL, FULL], [SKIP] * 4, [LOCAL, LOCAL, SKIP, FULL]], dtype=np.uint8)
    pair.attend(0, [0, 1, 1], [49, 199, 150], q, hm, window_scalar=40)


def test_per_head_error_contract():
    rng = np.random.default_rng(4)
    Hq, Hkv, d = 4, 2, 64
    pair = Pair(1, 2, Hq, Hkv, d, 32, 16, 40, [8] * 4, max_append=64, max_queries=64, head_modes=1)
    K = wl.bf16_bits(rng.standard_normal((4, Hkv, d), dtype=np.float32))
    before = {k: pair.gpu.region(k).clone() for k in ("ntok", "page_table", "last_pos", "presence")}
    pair.append(0, [0], [0], K[:1], K[:1], [4], [[FULL, SKIP, 3, LOCAL]], expect=1)  # not a mode
    for k, v in before.items():
        assert torch.equal(v, pair.gpu.region(k)), k
    pair.append(0, [0, 0, 1], [0, 1, 0], K[:3], K[1:4], [4, 2, 16],
                [[FULL, SKIP, SKIP, LOCAL], [SKIP] * 4, [SKIP, SKIP, LOCAL, SKIP]])
    pair.check_regions()
    q = wl.bf16_bits(rng.standard_normal((3, Hq, d), dtype=np.float32))
    # a local head with a window below 1 fails its query (zero row); the others compute
    pair.attend(0, [0, 0], [1, 1], q[:2], [[FULL] * 4, [LOCAL, SKIP, FULL, SKIP]], window_scalar=0,
                expect=1)
    # a value that is not a mode in any head fails the query
    pair.attend(0, [0, 1], [1, 0], q[:2], [[FULL, 4, FULL, FULL], [FULL] * 4], window_scalar=3, expect=1)
    # head 1 reads KV head 0 (stored by token 0, head 0 full): a row; the skip heads: zeros
    got, _ = pair.attend(0, [0, 1], [1, 0], q[:2], [[SKIP, FULL, SKIP, SKIP], [SKIP, SKIP, SKIP, LOCAL]],
                         window_scalar=2)
    assert got[0, 1].any() and got[1, 3].any()
    # router decisions are per token: the routed calls refuse a per-head cache
    n = 1
    with pytest.raises(trr.TrrError) as ei:
        pair.gpu.decode_attn_routed(0, dev(np.zeros(n, np.int32), torch.int32), dev(np.ones(n, np.int32), torch.int32),
                                    dev(q[:1], torch.bfloat16), torch.zeros((n, 3), device="cuda"),
                                    window_scalar=2)
    assert ei.value.code == 6
    with pytest.raises(trr.TrrError) as ei:
        pair.gpu.append_routed(0, dev(np.zeros(n, np.int32), torch.int32), dev(np.full(n, 5, np.int32), torch.int32),
                               dev(K[:1], torch.bfloat16), dev(K[:1], torch.bfloat16),
                               torch.zeros((n, 4), device="cuda"), torch.zeros((n, 3), device="cuda"))
    assert ei.value.code == 6
    # a modes array of the per-token shape is refused by the binding
    with pytest.raises(ValueError):
        pair.gpu.decode_attn(0, dev(np.zeros(2, np.int32), torch.int32), dev(np.ones(2, np.int32), torch.int32),
                             dev(q[:2], torch.bfloat16), dev(np.full(2, FULL, np.uint8), torch.uint8))


def test_160m_shape_per_head():
    """The 160m decode step's shape (MHA 12 x 64, window 256, its bit and mode mixes) at
    batch 8 and context 2048, with a mode per (token, head): the cache built by prefill
    appends, then one decode step (append position 2047, attend) checked whole."""
    spec = wl.SPECS["160m"]
    B, P, ctx, Hq = 8, 32, 2048, spec.num_q_heads
    pols = [wl.head_policy(spec, 0, s, ctx) for s in range(B)]
    need = [0, 0, 0, 0]
    for bits, hm in pols:
        took = (hm != SKIP).any(1)
        for c, b in enumerate((2, 4, 8, 16)):
            need[c] += -(-int(np.count_nonzero(took & (bits == b))) // P)
    pair = Pair(1, B, Hq, spec.num_kv_heads, spec.head_dim, spec.group_size, P, ctx, need,
                head_modes=1)
    kvs = [wl.kv(spec, 0, s, 0, ctx) for s in range(B)]
    for s in range(B):
        for p0 in range(0, ctx - 1, 1023):
            p1 = min(ctx - 1, p0 + 1023)
            pair.append(0, [s] * (p1 - p0), range(p0, p1), kvs[s][0][p0:p1], kvs[s][1][p0:p1],
                        pols[s][0][p0:p1], pols[s][1][p0:p1])
    last = ctx - 1
    hm = np.stack([pols[s][1][last] for s in range(B)])
    pair.append(0, range(B), [last] * B, np.stack([kvs[s][0][last] for s in range(B)]),
                np.stack([kvs[s][1][last] for s in range(B)]), [pols[s][0][last] for s in range(B)], hm)
    pair.check_regions()
    q = np.stack([wl.q(spec, 0, s, last, ctx)[0] for s in range(B)])
    pair.attend(0, range(B), [last] * B, q, hm, window_scalar=spec.window)


def test_static_scratch_entry_with_head_modes():
    """trr_decode_attn_static on a per-head cache: the oracle's rows within tolerance and
    the same bits as trr_decode_attn, on two calls in a row."""
    rng = np.random.default_rng(61)
    ctxs = [300, 120]
    pair = _setup(rng, 64, 32, 16, 8, 4, ctxs, 1024)
    seqs, ts, hm, ws = _queries(rng, ctxs, 8)
    q = wl.bf16_bits(rng.standard_normal((len(seqs), 8, 64), dtype=np.float32))
    got, ref = pair.attend(0, seqs, ts, q, hm, windows=ws)
    args = (dev(np.asarray(seqs, np.int32), torch.int32), dev(np.asarray(ts, np.int32), torch.int32),
            dev(q, torch.bfloat16), dev(hm, torch.uint8), dev(np.asarray(ws, np.int32), torch.int32))
    for _ in range(2):
        out = torch.full((len(seqs), 8, 64), float("nan"), dtype=torch.bfloat16, device="cuda")
        trr.trr_decode_attn_static(pair.gpu.handle, 0, *args, 0, 0.0, out)
        st = out.float().cpu().numpy().astype(np.float64)
        check_attention(st, ref, hm)
        assert np.array_equal(st, got)
    assert pair.gpu.status() == 0
