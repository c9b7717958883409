"""GPU parity of trr_decode_step (one kernel: the append of every entry's token, then
every entry's query at the same position and mode) against the oracle's append
followed by its attention: page bytes and metadata bit-exact, attention rows within
max abs 2e-2 / row-relative 5e-3.  Covers every tested layout (both consumers), first
tokens of a sequence, tokens that open pages, skip tokens with and without stored KV,
calls whose layer was touched by one of the two calls before them (the kernel waits
before reading the cache) and calls on a settled layer (it reads the cache and issues
its page copies first), and the call-level errors, after which nothing is stored and
every row is zero."""
import numpy as np
import pytest
import torch

from paper_2607_06601_gb300 import trr, workloads as wl
from tests._parity import Pair, compare_regions, dev

pytestmark = pytest.mark.gpu

SKIP, LOCAL, FULL = 0, 1, 2
BITS = (2, 4, 8, 16)


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def test_step_tiny_sequential_decode():
    """The tiny workload as decode steps: at every position, one call appends each
    sequence's token and attends with its query (contexts 37 and 130)."""
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
        pair.step(0, seqs, [p] * len(seqs), np.stack([kvs[s][0][p] for s in seqs]),
                  np.stack([kvs[s][1][p] for s in seqs]), [pols[s][0][p] for s in seqs],
                  [pols[s][1][p] for s in seqs], np.stack([qs[s][p] for s in seqs]), window_scalar=spec.window)
        if p % 16 == 15 or p == maxctx - 1:
            pair.check_regions()


CONFIGS = [  # d, G, P, Hq, Hkv: CUDA-core (g = 1) and tensor-core (query groups) consumers
    (64, 32, 16, 4, 2),
    (64, 64, 32, 4, 4),
    (64, 32, 64, 2, 1),
    (128, 64, 16, 8, 2),
    (128, 128, 64, 4, 1),
    (128, 32, 16, 4, 4),
    (64, 32, 32, 12, 12),
]


def _prefill(pair, rng, ctxs, Hkv, d, layer=0, skip_p=0.2):
    """Contexts through trr_kv_append (seeded widths and modes)."""
    ent = [(s, p) for p in range(max(ctxs, default=0)) for s in range(len(ctxs)) if p < ctxs[s]]
    for i in range(0, len(ent), 1024):
        ch = ent[i:i + 1024]
        pair.append(layer, [e[0] for e in ch], [e[1] for e in ch],
                    wl.bf16_bits(rng.standard_normal((len(ch), Hkv, d), dtype=np.float32)),
                    wl.bf16_bits(rng.standard_normal((len(ch), Hkv, d), dtype=np.float32)),
                    rng.choice(BITS, size=len(ch)), rng.choice(3, size=len(ch), p=[skip_p, 0.4, 0.6 - skip_p]))


def _steps(pair, rng, ctxs, Hq, Hkv, d, nsteps, layer=0, windows=(1, 2, 5, 16, 33, 100, 1000)):
    """nsteps decode steps of every sequence (each one token further), random widths,
    modes and windows; returns the positions reached."""
    S = len(ctxs)
    pos = list(ctxs)
    for _ in range(nsteps):
        seqs = list(rng.permutation(S))  # any order of the entries
        p = [pos[s] for s in seqs]
        pair.step(layer, seqs, p, wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32)),
                  wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32)), rng.choice(BITS, size=S),
                  rng.choice(3, size=S), wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32)),
                  windows=rng.choice(windows, size=S))
        for s in seqs:
            pos[s] += 1
    return pos


@pytest.mark.parametrize("d,G,P,Hq,Hkv", CONFIGS)
def test_step_ragged_contexts_all_layouts(d, G, P, Hq, Hkv):
    """Contexts from empty (the first token of a sequence comes in a step) to several
    pages; 40 steps cross page boundaries of every class."""
    rng = np.random.default_rng(1000 + d + G + P + Hq)
    ctxs = [0, 1, 17, 100, 257, 611, 31]
    maxctx = max(ctxs) + 64
    caps = [len(ctxs) * (maxctx // P + 2)] * 4
    pair = Pair(1, len(ctxs), Hq, Hkv, d, G, P, maxctx, caps)
    _prefill(pair, rng, ctxs, Hkv, d)
    _steps(pair, rng, ctxs, Hq, Hkv, d, 40)
    pair.check_regions()


@pytest.mark.parametrize("swk", [0, 1])
def test_step_skip_tokens(swk):
    """Skip entries: a zero row; their KV stored only with skip_writes_kv."""
    rng = np.random.default_rng(77 + swk)
    ctxs = [5, 64, 130]
    d, G, P, Hq, Hkv = 64, 32, 16, 4, 4
    maxctx = 300
    caps = [len(ctxs) * (maxctx // P + 2)] * 4
    pair = Pair(1, len(ctxs), Hq, Hkv, d, G, P, maxctx, caps, skip_writes_kv=swk)
    _prefill(pair, rng, ctxs, Hkv, d)
    pos = list(ctxs)
    for i in range(20):
        m = [SKIP if (i + s) % 3 == 0 else FULL for s in range(3)]
        pair.step(0, [0, 1, 2], pos, wl.bf16_bits(rng.standard_normal((3, Hkv, d), dtype=np.float32)),
                  wl.bf16_bits(rng.standard_normal((3, Hkv, d), dtype=np.float32)), rng.choice(BITS, size=3), m,
                  wl.bf16_bits(rng.standard_normal((3, Hq, d), dtype=np.float32)), window_scalar=8)
        pos = [p + 1 for p in pos]
    pair.check_regions()


@pytest.mark.parametrize("d,G,P,Hq,Hkv", [(64, 32, 32, 12, 12), (128, 64, 16, 8, 2)])
def test_step_layers_in_turn(d, G, P, Hq, Hkv):
    """A three-layer cache stepped layer by layer, as a decoder runs: after the first
    calls every call's layer is settled (the kernel reads its cache state and issues its
    page copies before the previous kernel ends); calls on one layer twice in a row,
    and an append or attention call in between, make it wait first."""
    rng = np.random.default_rng(5 + d)
    L, ctxs = 3, [40, 300, 7, 129]
    maxctx = max(ctxs) + 64
    caps = [L * len(ctxs) * (maxctx // P + 2)] * 4
    pair = Pair(L, len(ctxs), Hq, Hkv, d, G, P, maxctx, caps)
    for layer in range(L):
        _prefill(pair, rng, ctxs, Hkv, d, layer=layer)
    pos = {layer: list(ctxs) for layer in range(L)}
    order = [0, 1, 2] * 4 + [1, 1, 2, 0, 0, 2, 1]
    for i, layer in enumerate(order):
        S = len(ctxs)
        pair.step(layer, list(range(S)), pos[layer],
                  wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32)),
                  wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32)), rng.choice(BITS, size=S),
                  rng.choice(3, size=S), wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32)),
                  window_scalar=int(rng.choice([4, 50, 1000])))
        pos[layer] = [p + 1 for p in pos[layer]]
        if i == 14:  # a plain attention call on another layer in between
            other = (layer + 1) % L
            pair.attend(other, list(range(S)), [p - 1 for p in pos[other]],
                        wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32)), [FULL] * S)
    pair.check_regions()


def _error_case(pair, seqs, pos, bits, modes, windows, expect, Hq, Hkv, d, rng):
    before = {k: pair.gpu.region(k).cpu().numpy().copy() for k in ("last_pos", "ntok", "page_table", "next_page")}
    n = len(seqs)
    out = pair.gpu.decode_step(0, dev(np.asarray(seqs, np.int32), torch.int32), dev(np.asarray(pos, np.int32), torch.int32),
                               dev(wl.bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)), torch.bfloat16),
                               dev(wl.bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)), torch.bfloat16),
                               dev(np.asarray(bits, np.uint8), torch.uint8), dev(np.asarray(modes, np.uint8), torch.uint8),
                               dev(wl.bf16_bits(rng.standard_normal((n, Hq, d), dtype=np.float32)), torch.bfloat16),
                               dev(np.asarray(windows, np.int32), torch.int32), 0)
    assert pair.gpu.status() == expect
    got = out.float().cpu().numpy()
    assert (got == 0).all() and not np.signbit(got).any(), "an erroneous call writes zero rows"
    for k, v in before.items():
        assert np.array_equal(pair.gpu.region(k).cpu().numpy(), v), f"{k} changed by an erroneous call"


def test_step_errors_store_nothing():
    rng = np.random.default_rng(9)
    d, G, P, Hq, Hkv = 64, 32, 16, 4, 2
    ctxs = [20, 33, 64]
    maxctx = 128
    pair = Pair(1, 3, Hq, Hkv, d, G, P, maxctx, [3 * (maxctx // P + 2)] * 4)
    _prefill(pair, rng, ctxs, Hkv, d)
    ok = dict(seqs=[0, 1, 2], pos=[20, 33, 64], bits=[2, 4, 8], modes=[FULL, LOCAL, FULL], windows=[4, 4, 4])
    cases = [
        (dict(seqs=[0, 1, 0]), 1),                                  # a sequence named twice
        (dict(pos=[20, 33, 64 - 1]), 4),                            # not above the last position
        (dict(pos=[20, 33, maxctx]), 4),                            # outside [0, max_context)
        (dict(bits=[2, 3, 8]), 1),                                  # bit-width not allowed
        (dict(modes=[FULL, 3, FULL]), 1),                           # mode not allowed
        (dict(windows=[4, 0, 4]), 1),                               # local window below 1
        (dict(seqs=[0, 5, 2]), 1),                                  # sequence id out of range
    ]
    for change, code in cases:
        args = dict(ok, **change)
        _error_case(pair, args["seqs"], args["pos"], args["bits"], args["modes"], args["windows"], code, Hq, Hkv, d,
                    rng)
    # after all that, the same cache still steps correctly
    pair.step(0, ok["seqs"], ok["pos"], wl.bf16_bits(rng.standard_normal((3, Hkv, d), dtype=np.float32)),
              wl.bf16_bits(rng.standard_normal((3, Hkv, d), dtype=np.float32)), ok["bits"], ok["modes"],
              wl.bf16_bits(rng.standard_normal((3, Hq, d), dtype=np.float32)), windows=ok["windows"])
    pair.check_regions()


def test_step_out_of_pages_stores_nothing():
    """A pool with no page left for a token that opens one: OUT_OF_PAGES (known only
    after the wait on the previous kernel), zero rows, nothing stored."""
    rng = np.random.default_rng(10)
    d, G, P, Hq, Hkv = 64, 32, 16, 4, 4
    caps = [1, 1, 1, 1]
    pair = Pair(1, 2, Hq, Hkv, d, G, P, 64, caps)
    k = wl.bf16_bits(rng.standard_normal((16, Hkv, d), dtype=np.float32))
    pair.append(0, [0] * 16, list(range(16)), k, k, [4] * 16, [FULL] * 16)  # class 4 pool now full
    _error_case(pair, [0, 1], [16, 0], [8, 4], [FULL, FULL], [1, 1], 3, Hq, Hkv, d, rng)
    pair.step(0, [0, 1], [16, 0], wl.bf16_bits(rng.standard_normal((2, Hkv, d), dtype=np.float32)),
              wl.bf16_bits(rng.standard_normal((2, Hkv, d), dtype=np.float32)), [8, 16], [FULL, LOCAL],
              wl.bf16_bits(rng.standard_normal((2, Hq, d), dtype=np.float32)), window_scalar=3)
    pair.check_regions()


def test_step_matches_separate_calls_on_a_full_batch():
    """The decode step of the 160m shape (12 heads x 64, batch 32, 2048-token contexts)
    against trr_kv_append + trr_decode_attn on a second cache built the same way: the
    same metadata and page bytes, bit for bit, and the same rows within the tolerance
    (each compared with the oracle in the full-size tests)."""
    spec = wl.SPECS["160m"]
    B, P, n = 32, 32, 512
    Hq, Hkv, d, G = spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.group_size
    rng = np.random.default_rng(3)
    caps = [B * (n // P + 2)] * 4
    a = trr.Cache(1, B, Hq, Hkv, d, G, P, n, caps, max_append=1024, max_queries=64, zero_pool=True)
    b = trr.Cache(1, B, Hq, Hkv, d, G, P, n, caps, max_append=1024, max_queries=64, zero_pool=True)
    ctx = n - 8
    ent_s = np.repeat(np.arange(B, dtype=np.int32), ctx)
    ent_p = np.tile(np.arange(ctx, dtype=np.int32), B)
    bits = rng.choice(BITS, size=B * ctx).astype(np.uint8)
    modes = rng.choice(3, size=B * ctx, p=[0.2, 0.5, 0.3]).astype(np.uint8)
    K = wl.bf16_bits(rng.standard_normal((B * ctx, Hkv, d), dtype=np.float32))
    V = wl.bf16_bits(rng.standard_normal((B * ctx, Hkv, d), dtype=np.float32))
    for c in (a, b):
        for i in range(0, B * ctx, 1024):
            sl = slice(i, i + 1024)
            c.append(0, dev(ent_s[sl], torch.int32), dev(ent_p[sl], torch.int32), dev(K[sl], torch.bfloat16),
                     dev(V[sl], torch.bfloat16), dev(bits[sl], torch.uint8), dev(modes[sl], torch.uint8))
    for t in range(ctx, n):
        seqs = dev(np.arange(B, dtype=np.int32), torch.int32)
        pos = dev(np.full(B, t, np.int32), torch.int32)
        k1 = dev(wl.bf16_bits(rng.standard_normal((B, Hkv, d), dtype=np.float32)), torch.bfloat16)
        v1 = dev(wl.bf16_bits(rng.standard_normal((B, Hkv, d), dtype=np.float32)), torch.bfloat16)
        b1 = dev(rng.choice(BITS, size=B).astype(np.uint8), torch.uint8)
        m1 = dev(rng.choice(3, size=B).astype(np.uint8), torch.uint8)
        q1 = dev(wl.bf16_bits(rng.standard_normal((B, Hq, d), dtype=np.float32)), torch.bfloat16)
        out_a = a.decode_step(0, seqs, pos, k1, v1, b1, m1, q1, window_scalar=256)
        b.append(0, seqs, pos, k1, v1, b1, m1)
        out_b = b.decode_attn(0, seqs, pos, q1, m1, window_scalar=256)
        ga, gb = out_a.float().cpu().numpy(), out_b.float().cpu().numpy()
        assert np.abs(ga - gb).max() <= 4e-2
    assert a.status() == 0 and b.status() == 0
    for name in ("last_pos", "ntok", "presence", "page_table", "page_first", "page_last", "next_page",
                 "pool2", "pool4", "pool8", "pool16"):
        assert torch.equal(a.region(name), b.region(name)), name
