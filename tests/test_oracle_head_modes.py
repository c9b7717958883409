"""Pins of the oracle's per-head attention modes (Sec. 3.2(A): a mode per head by
default; Appendix C's router emits modes of shape [B, T, H, |A|]).  A cache with
head_modes takes modes[n][Hq]; KV head j of a token is stored when one of the query
heads reading it (h / (Hq / Hkv) = j) does not skip (or when skip tokens store KV), and
every KV head's slice of a page ends with 16 bytes holding its 64-bit presence mask.
Pinned against: the per-token cache (all heads of a token with one mode give the same
results and bytes), an explicit per-head mask over dequantised K/V for every per-head
policy of tiny contexts, the presence bits read straight from the page bytes, and the
error contract."""
import itertools

import numpy as np
import pytest

import oracle
from paper_2607_06601_gb300.workloads import bf16_bits, bf16_to_f32

SKIP, LOCAL, FULL = 0, 1, 2


def _dense(q, K, V, mask, scale):
    if not mask.any():
        return np.zeros(V.shape[1])
    sc = scale * (K[mask] @ q)
    p = np.exp(sc - sc.max())
    return (p[:, None] * V[mask]).sum(0) / p.sum()


def _heads_store(hmodes, Hq, Hkv, swk=0):
    """[n][Hkv] whether each token stores each KV head (any reading head not skip)."""
    g = Hq // Hkv
    hm = np.asarray(hmodes).reshape(-1, Hq)
    return np.stack([(hm[:, j * g:(j + 1) * g] != SKIP).any(1) | bool(swk) for j in range(Hkv)], 1)


def _permuted(Hq, Hkv, d, G, head_modes):
    """The documented rule: 8- and 16-bit code rows keep a permuted chunk order in every
    cache except those of query groups g >= 2 whose g * (d / G) columns fit 8, without
    per-head modes (the tensor-core path's)."""
    g = Hq // Hkv
    return not (not head_modes and g >= 2 and g * (d // G) <= 8)


def _logical(sl, b, code_bytes):
    """A slice's bytes with its K and V code regions (the first code_bytes) back in
    logical order: line n keeps logical chunk k at chunk k ^ (n % 8)."""
    out = sl.copy()
    if b < 8:
        return out
    for n in range(code_bytes // 128):
        for k in range(8):
            src = n * 128 + (k ^ (n % 8)) * 16
            out[n * 128 + k * 16:n * 128 + k * 16 + 16] = sl[src:src + 16]
    return out


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (4, 4), (8, 1)])
def test_equal_head_modes_match_the_per_token_cache(Hq, Hkv):
    rng = np.random.default_rng(Hq * 10 + Hkv)
    S, n, d, P = 3, 150, 64, 16
    tok = oracle.OracleCache(1, S, Hq, Hkv, d, 32, P, n, [S * 12] * 4)
    hed = oracle.OracleCache(1, S, Hq, Hkv, d, 32, P, n, [S * 12] * 4, head_modes=1)
    bits = rng.choice([2, 4, 8, 16], size=(S, n))
    modes = rng.choice(3, size=(S, n), p=[0.3, 0.35, 0.35])
    for p in range(n):
        K = bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32))
        V = bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32))
        m = modes[:, p]
        assert tok.append(0, np.arange(S), [p] * S, K, V, bits[:, p], m) == 0
        assert hed.append(0, np.arange(S), [p] * S, K, V, bits[:, p], np.repeat(m, Hq)) == 0
    for name in ("last_pos", "ntok", "presence", "page_table", "page_first", "page_last", "next_page"):
        assert np.array_equal(tok.region(name), hed.region(name)), name
    assert tok.mask_bytes == 0 and hed.mask_bytes == 16
    ntok = hed.region("ntok").view(np.int32).reshape(S, 4)
    for c, b in enumerate((2, 4, 8, 16)):
        pt, ph = tok.region(f"pool{b}"), hed.region(f"pool{b}")
        sl_t = tok.slice_bytes(c)
        assert hed.slice_bytes(c) == sl_t + 16
        for pid in range(int(hed.region("next_page").view(np.int32)[c])):
            a0, b0 = pid * tok.page_bytes(c), pid * hed.page_bytes(c)
            assert np.array_equal(pt[a0:a0 + tok.hdr_bytes], ph[b0:b0 + hed.hdr_bytes]), (b, pid)
            masks = []
            code_bytes = 2 * P * (d * b // 8 if b < 16 else 2 * d)
            for j in range(Hkv):  # each KV head's slice: the same bytes, then its mask, 8 zeros
                sa = pt[a0 + tok.hdr_bytes + j * sl_t:][:sl_t]
                sb = ph[b0 + hed.hdr_bytes + j * (sl_t + 16):][:sl_t + 16]
                if _permuted(Hq, Hkv, d, 32, 0):
                    sa = _logical(sa, b, code_bytes)
                assert np.array_equal(sa, _logical(sb[:sl_t], b, code_bytes)), (b, pid, j)
                masks.append(int(sb[sl_t:sl_t + 8].view(np.uint64)[0]))
                assert not sb[sl_t + 8:].any()
            fill = bin(masks[0]).count("1")
            assert fill >= 1 and all(x == (1 << fill) - 1 for x in masks)  # every head, every slot
    assert ntok.sum() > 0
    q = bf16_bits(rng.standard_normal((3 * S, Hq, d), dtype=np.float32))
    seqs = np.tile(np.arange(S), 3)
    ts = np.array([n - 1] * S + [60] * S + [7] * S)
    qm = rng.choice(3, size=3 * S)
    st1, out1 = tok.decode_attn(0, seqs, ts, q, qm, window_scalar=24)
    st2, out2 = hed.decode_attn(0, seqs, ts, q, np.repeat(qm, Hq), window_scalar=24)
    assert st1 == st2 == 0 and np.array_equal(out1, out2) and np.abs(out1).max() > 0


def _head_cases(T, Hq):
    pol = list(itertools.product([2, 4, 8, 16], itertools.product([SKIP, LOCAL, FULL], repeat=Hq)))
    return itertools.product(pol, repeat=T)


def _brute(T, Hq, Hkv, cases, w=2, d=64, swk=0):
    """Sequential decode under per-head policies, against an explicit per-head mask."""
    rng = np.random.default_rng(200 + T + Hq + Hkv)
    K = bf16_bits(rng.standard_normal((T, Hkv, d), dtype=np.float32) * 2)
    V = bf16_bits(rng.standard_normal((T, Hkv, d), dtype=np.float32))
    Q = bf16_bits(rng.standard_normal((T, Hq, d), dtype=np.float32) * 2)
    Qf = bf16_to_f32(Q).astype(np.float64)
    scale, g = 1 / np.sqrt(d), Hq // Hkv
    count = 0
    for case in cases:
        bits = [c[0] for c in case]
        hm = np.array([c[1] for c in case], dtype=np.uint8)  # [T][Hq]
        o = oracle.OracleCache(1, 1, Hq, Hkv, d, 32, 16, T, [4, 4, 4, 4], skip_writes_kv=swk, head_modes=1)
        outs = []
        for t in range(T):
            assert o.append(0, [0], [t], K[t:t + 1], V[t:t + 1], [bits[t]], hm[t]) == 0
            st, out = o.decode_attn(0, [0], [t], Q[t:t + 1], hm[t], window_scalar=w)
            assert st == 0
            outs.append(out[0])
        stores = _heads_store(hm, Hq, Hkv, swk)
        Kh = np.zeros((Hkv, T, d))
        Vh = np.zeros((Hkv, T, d))
        for j in range(T):
            for kv in range(Hkv):
                c, kk, vv = o.dequant_token(0, 0, j, kv)
                assert (c >= 0) == stores[j, kv], (case, j, kv)
                if c >= 0:
                    assert [2, 4, 8, 16][c] == bits[j]
                    Kh[kv, j], Vh[kv, j] = kk, vv
        j = np.arange(T)
        for t in range(T):
            for h in range(Hq):
                m = hm[t, h]
                if m == SKIP:
                    ref = np.zeros(d)
                else:
                    mask = stores[:, h // g] & (j <= t) & ((m == FULL) | (j >= t - w + 1))
                    ref = _dense(Qf[t, h], Kh[h // g], Vh[h // g], mask, scale)
                assert np.abs(outs[t][h] - ref).max() < 1e-12, (case, t, h)
        count += 1
    return count


def test_brute_force_per_head_policies_gqa():
    """Two query heads sharing one KV head: every per-head policy of 1-2 token contexts."""
    assert sum(_brute(T, 2, 1, _head_cases(T, 2)) for T in (1, 2)) == 36 + 36 ** 2


def test_brute_force_per_head_policies_mha_and_sampled_three_tokens():
    assert _brute(2, 2, 2, _head_cases(2, 2)) == 36 ** 2
    rng = np.random.default_rng(7)
    allc = list(_head_cases(3, 2))
    pick = [allc[i] for i in rng.choice(len(allc), size=400, replace=False)]
    assert _brute(3, 2, 1, pick) == 400
    assert _brute(3, 2, 1, pick[:100], swk=1) == 100


def test_brute_force_per_head_policies_two_query_groups():
    """Four query heads over two KV heads (groups of 2): sampled per-head policies of
    2-3 token contexts, so that a head's KV head (h // 2) differs from h and from h % 2."""
    rng = np.random.default_rng(11)
    pol = list(itertools.product([2, 4, 8, 16], itertools.product([SKIP, LOCAL, FULL], repeat=4)))
    for T, n in ((2, 300), (3, 150)):
        cases = [tuple(pol[i] for i in rng.choice(len(pol), size=T)) for _ in range(n)]
        assert _brute(T, 4, 2, cases) == n


def test_presence_bits_follow_the_reading_heads():
    """The page's mask bits, read from its bytes: set for the KV heads that a
    non-skip query head reads, for every stored token, and for nothing else."""
    rng = np.random.default_rng(3)
    Hq, Hkv, d, P, n = 8, 4, 64, 16, 120
    o = oracle.OracleCache(1, 1, Hq, Hkv, d, 32, P, n, [20] * 4, head_modes=1)
    bits = rng.choice([2, 4, 8, 16], size=n)
    hm = rng.choice(3, size=(n, Hq), p=[0.6, 0.2, 0.2]).astype(np.uint8)
    hm[5] = SKIP  # a token no head reads: no slot at all
    K = bf16_bits(rng.standard_normal((n, Hkv, d), dtype=np.float32))
    assert o.append(0, [0] * n, np.arange(n), K, K, bits, hm) == 0
    stores = _heads_store(hm, Hq, Hkv)
    took = stores.any(1)
    assert not took[5]
    ntok = o.region("ntok").view(np.int32)
    pres = o.region("presence").view(np.uint32)
    for p in range(n):
        assert bool((pres[p // 32] >> (p % 32)) & 1) == took[p]
    for c, b in enumerate((2, 4, 8, 16)):
        pos = np.arange(n)[took & (bits == b)]
        assert ntok[c] == pos.size
        pool = o.region(f"pool{b}")
        pt = o.region("page_table").view(np.int32).reshape(4, -1)
        slb = o.slice_bytes(c)
        for k in range(-(-pos.size // P)):
            base = int(pt[c, k]) * o.page_bytes(c)
            slots = pool[base:base + 4 * P].view(np.int32)
            # KV head j's mask: the first 8 of the 16 bytes that end its slice
            masks = [pool[base + o.hdr_bytes + (j + 1) * slb - 16:][:8].view(np.uint64)[0] for j in range(Hkv)]
            for sl in range(min(P, pos.size - k * P)):
                assert slots[sl] == pos[k * P + sl]
                for j in range(Hkv):
                    assert bool((int(masks[j]) >> sl) & 1) == stores[pos[k * P + sl], j]
            for j in range(Hkv):
                assert int(masks[j]) >> min(P, pos.size - k * P) == 0


def test_per_head_error_contract():
    Hq, Hkv, d = 4, 2, 64
    o = oracle.OracleCache(1, 2, Hq, Hkv, d, 32, 16, 40, [8] * 4, head_modes=1)
    K = bf16_bits(np.ones((1, Hkv, d), dtype=np.float32))
    assert o.append(0, [0], [0], K, K, [4], [FULL, SKIP, 3, LOCAL]) == 1   # a mode that is not one
    assert o.region("last_pos").view(np.int32)[0] == -1                      # nothing happened
    assert o.append(0, [0], [0], K, K, [4], [FULL, SKIP, SKIP, LOCAL]) == 0
    q = bf16_bits(np.ones((2, Hq, d), dtype=np.float32))
    st, out = o.decode_attn(0, [0, 0], [0, 0], q, [FULL] * 4 + [LOCAL, SKIP, FULL, SKIP], window_scalar=0)
    assert st == 1 and not out[1].any() and out[0].any()   # local head with w < 1: that query fails
    st, out = o.decode_attn(0, [0, 0], [0, 0], q, [FULL] * 4 + [FULL, SKIP, LOCAL, SKIP], window_scalar=0)
    assert st == 1 and not out[1].any() and out[0].any()   # the local head need not be the first
    st, out = o.decode_attn(0, [0], [0], q[:1], [SKIP, FULL, SKIP, SKIP], window_scalar=0)
    # head 1 reads KV head 0, which token 0 stores (head 0 full): a row; skip heads: zeros
    assert st == 0 and out[0, 1].any() and not out[0, [0, 2, 3]].any()
