"""Pins of the oracle's mode-routed attention (Sec. 3.2(A), Eq. 2) over its paged
mixed-precision cache, against definitions that do not go through the oracle's page
walk: dense softmax attention (numpy, and torch's SDPA in fp64), an explicit T x T
mask built from the modes, brute-force enumeration of every per-token policy on tiny
contexts, and the window length fixed by the paper's cost model (golden file)."""
import itertools
import os

import numpy as np
import pytest

import oracle
from paper_2607_06601_gb300.workloads import bf16_bits, bf16_to_f32

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SKIP, LOCAL, FULL = 0, 1, 2


def _cache(S=1, Hq=2, Hkv=1, d=64, G=32, P=16, maxctx=64, cap=64, swk=0):
    return oracle.OracleCache(1, S, Hq, Hkv, d, G, P, maxctx, [cap] * 4, skip_writes_kv=swk)


def _dense(q, K, V, mask, scale):
    """Softmax attention of one query over the rows of K/V selected by mask."""
    if not mask.any():
        return np.zeros(V.shape[1])
    sc = scale * (K[mask] @ q)
    p = np.exp(sc - sc.max())
    return (p[:, None] * V[mask]).sum(0) / p.sum()


def test_all16_full_equals_dense_sdpa():
    """b = 16 is native precision, so all-16 / all-full is plain causal attention."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    ctxs, Hq, Hkv, d = [5, 40, 70], 4, 2, 64
    o = _cache(S=3, Hq=Hq, Hkv=Hkv, maxctx=80, cap=40)
    K = {s: bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)) for s, n in enumerate(ctxs)}
    V = {s: bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32)) for s, n in enumerate(ctxs)}
    Q = {s: bf16_bits(rng.standard_normal((n, Hq, d), dtype=np.float32)) for s, n in enumerate(ctxs)}
    for p in range(max(ctxs)):  # sequences interleaved position by position
        for s in range(3):
            if p < ctxs[s]:
                assert o.append(0, [s], [p], K[s][p:p + 1], V[s][p:p + 1], [16], [FULL]) == 0
    scale = 1 / np.sqrt(d)
    for s, n in enumerate(ctxs):
        ts = np.arange(n)
        st, out = o.decode_attn(0, [s] * n, ts, Q[s], [FULL] * n)
        assert st == 0
        Kf, Vf, Qf = (bf16_to_f32(x).astype(np.float64) for x in (K[s], V[s], Q[s]))
        for t in ts:
            for h in range(Hq):
                kvh = h // (Hq // Hkv)
                ref = _dense(Qf[t, h], Kf[:, kvh], Vf[:, kvh], np.arange(n) <= t, scale)
                assert np.abs(out[t, h] - ref).max() < 1e-12
        # the same rows from torch's SDPA, fp64 on the CPU
        tq = torch.from_numpy(Qf).permute(1, 0, 2)[None]
        tk = torch.from_numpy(np.repeat(Kf, Hq // Hkv, axis=1)).permute(1, 0, 2)[None]
        tv = torch.from_numpy(np.repeat(Vf, Hq // Hkv, axis=1)).permute(1, 0, 2)[None]
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True)
        assert np.abs(out - ref[0].permute(1, 0, 2).numpy()).max() < 1e-12


def test_local_equals_full_on_truncated_window():
    rng = np.random.default_rng(6)
    n, w, d = 60, 9, 64
    bits = rng.choice([2, 4, 8, 16], size=n)
    keep = rng.random(n) > 0.25              # some tokens in the window are skipped
    K = bf16_bits(rng.standard_normal((n, 1, d), dtype=np.float32))
    V = bf16_bits(rng.standard_normal((n, 1, d), dtype=np.float32))
    q = bf16_bits(rng.standard_normal((1, 2, d), dtype=np.float32))
    for t in (0, 3, w - 1, w, 33, n - 1):
        a = _cache(maxctx=n)
        modes_a = np.where(keep, LOCAL, SKIP)
        assert a.append(0, [0] * (t + 1), np.arange(t + 1), K[:t + 1], V[:t + 1],
                        bits[:t + 1], modes_a[:t + 1]) == 0
        st, out_local = a.decode_attn(0, [0], [t], q, [LOCAL], window_scalar=w)
        assert st == 0
        b = _cache(maxctx=n)
        lo = max(0, t - w + 1)
        idx = [j for j in range(lo, t + 1) if keep[j]]
        assert b.append(0, [0] * len(idx), idx, K[idx], V[idx], bits[idx], [FULL] * len(idx)) == 0
        st, out_full = b.decode_attn(0, [0], [t], q, [FULL])
        assert st == 0
        assert np.abs(out_local - out_full).max() < 1e-12


def test_skip_reads_nothing_and_writes_nothing():
    rng = np.random.default_rng(7)
    d = 64
    K = bf16_bits(rng.standard_normal((4, 1, d), dtype=np.float32))
    q = bf16_bits(rng.standard_normal((1, 2, d), dtype=np.float32))
    o = _cache()
    assert o.append(0, [0, 0, 0], [0, 1, 2], K[:3], K[:3], [4, 2, 8], [FULL, SKIP, LOCAL]) == 0
    ntok = o.region("ntok").view(np.int32)
    assert list(ntok[:4]) == [0, 1, 1, 0]                      # the skipped 2-bit token is absent
    assert o.region("presence").view(np.uint32)[0] == 0b101
    assert o.region("last_pos").view(np.int32)[0] == 2         # but its position is consumed
    assert list(o.region("next_page").view(np.int32)) == [0, 1, 1, 0]
    st, out = o.decode_attn(0, [0], [2], q, [SKIP])
    assert st == 0 and (out == 0).all() and not np.signbit(out).any()
    # with skip_writes_kv = 1 (Principle 1: a lazy reader can still be a source)
    o2 = _cache(swk=1)
    assert o2.append(0, [0, 0], [0, 1], K[:2], K[:2], [4, 2], [FULL, SKIP]) == 0
    assert o2.region("presence").view(np.uint32)[0] == 0b11
    st, out = o2.decode_attn(0, [0], [1], q, [SKIP])
    assert (out == 0).all()


def _random_cache(rng, S, n, Hq=4, Hkv=2, d=64, G=32, P=16, order=None):
    o = oracle.OracleCache(1, S, Hq, Hkv, d, G, P, n, [S * (n // P + 2)] * 4)
    bits = rng.choice([2, 4, 8, 16], size=(S, n))
    modes = rng.choice([SKIP, LOCAL, FULL], size=(S, n))
    K = bf16_bits(rng.standard_normal((S, n, Hkv, d), dtype=np.float32))
    V = bf16_bits(rng.standard_normal((S, n, Hkv, d), dtype=np.float32))
    if order is None:  # position by position, sequences interleaved
        for p in range(n):
            for s in range(S):
                assert o.append(0, [s], [p], K[s, p:p + 1], V[s, p:p + 1], [bits[s, p]],
                                [modes[s, p]]) == 0
    else:              # one whole sequence after another, in the given order
        for s in order:
            assert o.append(0, [s] * n, np.arange(n), K[s], V[s], bits[s], modes[s]) == 0
    return o, bits, modes


def test_invariant_to_page_order_and_page_location():
    S, n, Hq, d = 3, 90, 4, 64
    rng = np.random.default_rng(8)
    a, _, _ = _random_cache(np.random.default_rng(8), S, n)
    b, _, _ = _random_cache(np.random.default_rng(8), S, n, order=[2, 0, 1])
    assert not np.array_equal(a.region("page_table"), b.region("page_table"))
    q = bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32))
    seqs, ts = np.arange(S), np.array([n - 1, 50, 17])
    for mode in (LOCAL, FULL):
        st, ref = a.decode_attn(0, seqs, ts, q, [mode] * S, window_scalar=20)
        assert st == 0 and np.abs(ref).max() > 0
        st, moved = b.decode_attn(0, seqs, ts, q, [mode] * S, window_scalar=20)
        assert np.array_equal(ref, moved)        # same visiting order, other page ids
        for seed in (1, 2, 3):
            st, perm = a.decode_attn(0, seqs, ts, q, [mode] * S, window_scalar=20, order_seed=seed)
            assert np.abs(perm - ref).max() <= 1e-12 * np.abs(ref).max()


def _policy_cases(T):
    pol = list(itertools.product([2, 4, 8, 16], [SKIP, LOCAL, FULL]))
    return itertools.product(pol, repeat=T)


def _brute(T, cases, w=2, d=64):
    """Sequential decode (append token t, then query t) under every policy; compare
    with an explicit mask over the stored tokens' dequantised K/V."""
    rng = np.random.default_rng(100 + T)
    K = bf16_bits(rng.standard_normal((T, 1, d), dtype=np.float32) * 2)
    V = bf16_bits(rng.standard_normal((T, 1, d), dtype=np.float32))
    Q = bf16_bits(rng.standard_normal((T, 1, d), dtype=np.float32) * 2)
    Qf = bf16_to_f32(Q).astype(np.float64)
    scale = 1 / np.sqrt(d)
    count = 0
    for case in cases:
        bits = [c[0] for c in case]
        modes = [c[1] for c in case]
        o = oracle.OracleCache(1, 1, 1, 1, d, 32, 16, T, [4, 4, 4, 4])
        outs = []
        for t in range(T):
            assert o.append(0, [0], [t], K[t:t + 1], V[t:t + 1], [bits[t]], [modes[t]]) == 0
            st, out = o.decode_attn(0, [0], [t], Q[t:t + 1], [modes[t]], window_scalar=w)
            assert st == 0
            outs.append(out[0, 0])
        Kh = np.zeros((T, d))
        Vh = np.zeros((T, d))
        present = np.zeros(T, dtype=bool)
        for j in range(T):
            c, kk, vv = o.dequant_token(0, 0, j, 0)
            present[j] = c >= 0
            assert present[j] == (modes[j] != SKIP)
            if present[j]:
                assert [2, 4, 8, 16][c] == bits[j]
                Kh[j], Vh[j] = kk, vv
        j = np.arange(T)
        for t in range(T):
            if modes[t] == SKIP:
                ref = np.zeros(d)
            else:
                mask = present & (j <= t) & ((modes[t] == FULL) | (j >= t - w + 1))
                ref = _dense(Qf[t, 0], Kh, Vh, mask, scale)
            assert np.abs(outs[t] - ref).max() < 1e-12, (case, t)
        # querying every position after the whole context is stored gives the same
        st, late = o.decode_attn(0, [0] * T, np.arange(T), Q, modes, window_scalar=w)
        assert np.abs(late[:, 0] - np.array(outs)).max() < 1e-12
        count += 1
    return count


def test_brute_force_every_policy_up_to_three_tokens():
    assert sum(_brute(T, _policy_cases(T)) for T in (1, 2, 3)) == 12 + 144 + 1728


@pytest.mark.slow
def test_brute_force_four_token_policies_sampled():
    rng = np.random.default_rng(44)
    allc = list(_policy_cases(4))
    pick = [allc[i] for i in rng.choice(len(allc), size=1500, replace=False)]
    assert _brute(4, pick) == 1500


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                rows.append([int(x) for x in line.split()])
    return rows


def test_golden_local_window_key_count():
    """A local query at 0-indexed position t reads min(t+1, w) keys when every token is
    stored: the cost model's kappa_local = 2 d min(t, w) over 1-indexed positions."""
    d = 64
    for t, w, expect in _read_golden("local_window_keys.txt"):
        n = t + 1
        o = oracle.OracleCache(1, 1, 1, 1, d, 32, 16, n, [64] * 4)
        K = bf16_bits(np.zeros((n, 1, d), dtype=np.float32))   # equal scores
        V = np.zeros((n, 1, d), dtype=np.float32)
        V[:, 0, 0] = 1.0
        V[:, 0, 1] = np.arange(n)                              # the key's own position
        assert o.append(0, [0] * n, np.arange(n), K, bf16_bits(V), [16] * n, [LOCAL] * n) == 0
        q = bf16_bits(np.ones((1, 1, d), dtype=np.float32))
        st, out = o.decode_attn(0, [0], [t], q, [LOCAL], window_scalar=w)
        assert st == 0 and abs(out[0, 0, 0] - 1) < 1e-12
        # uniform weights over positions t-expect+1 .. t average to t - (expect-1)/2
        assert abs(out[0, 0, 1] - (t - (expect - 1) / 2)) < 1e-9, (t, w, expect)


def test_golden_memory_cost_per_token():
    """The stored payload of one token at width b < 16 is the cost model's 2 d_kv b bits
    (Sec. 3.5, c^mem) plus one binary16 (scale, zero) pair per group for K and for V."""
    for b, hkv, d, G, bits_per_token in _read_golden("mem_cost_bits.txt"):
        o = oracle.OracleCache(1, 1, hkv, hkv, d, G, 16, 16, [1] * 4)
        c = [2, 4, 8, 16].index(b)
        tokb = o.slice_bytes(c) // 16          # bytes of one token of one KV head
        overhead = 0 if b == 16 else 2 * (d // G) * 4
        assert (tokb - overhead) * 8 * hkv == bits_per_token
