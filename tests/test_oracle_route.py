"""Pins of the oracle's hard decisions and their cost (Sec. 3.5 cost model, Sec. 3.8
hard arg max at inference, Appendix C expected_cost): numpy's nanargmax, hand-worked
costs on the paper's model shapes (golden file), closed forms of the dense
normalisers, and the keys / bits that the oracle's own attention and cache actually
read and store for the same decisions."""
import os

import numpy as np

import oracle
from paper_2607_06601_gb300.workloads import bf16_bits

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SKIP, LOCAL, FULL = 0, 1, 2
BITS = [2, 4, 8, 16]


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                rows.append([int(x) for x in line.split()])
    return rows


def _one_hot_logits(idx, k, rng=None):
    z = np.full((len(idx), k), -1.0, dtype=np.float32)
    z[np.arange(len(idx)), idx] = 1.0
    return z


def test_argmax_hand_rows():
    nan, inf = np.nan, np.inf
    cases = [([0.0, 1.0, 0.5], 1), ([2.0, 2.0, 1.0], 0), ([1.0, 3.0, 3.0], 1),
             ([nan, 0.0, -1.0], 1), ([nan, nan, nan], 0), ([nan, -inf, nan], 1),
             ([-inf, -inf, -inf], 0), ([1.0, inf, inf], 1), ([0.0, -0.0, 0.0], 0),
             ([-0.0, 0.0, 1e-45], 2), ([1.0, 2.0, 3.0, 4.0], 3), ([4.0, nan, 4.0, 5.0], 3),
             ([nan, nan, nan, 7.0], 3), ([3.0, 3.0, 3.0, 3.0], 0)]
    for z, expect in cases:
        assert oracle.argmax(z) == expect, (z, expect)


def test_argmax_equals_numpy_nanargmax():
    """np.nanargmax: index of the first maximum ignoring NaN (independent routine).  It
    reads NaN as -inf, so where every number of a row is -inf the reading differs: there
    the first -inf is taken (a NaN is never the decision)."""
    rng = np.random.default_rng(9)
    for k in (3, 4):
        z = rng.integers(-3, 4, size=(4000, k)).astype(np.float32)   # many ties
        z[rng.random(z.shape) < 0.15] = np.nan
        z[rng.random(z.shape) < 0.05] = np.inf
        z[rng.random(z.shape) < 0.05] = -np.inf
        z[0] = np.nan
        for row in z:
            if np.isnan(row).all():
                expect = 0
            elif np.nanmax(row) == -np.inf:
                expect = int(np.flatnonzero(~np.isnan(row))[0])
            else:
                expect = int(np.nanargmax(row))
            assert oracle.argmax(row) == expect, row


def test_option_order_modes_and_widths():
    """Mode options in the order skip, local, full; width options b = 2, 4, 8, 16."""
    n = 12
    mi, bi = np.arange(n) % 3, np.arange(n) % 4
    modes, bits, *_ = oracle.route_decisions(_one_hot_logits(mi, 3), _one_hot_logits(bi, 4),
                                             np.arange(n), 8, 2, 64, 1)
    assert modes.tolist() == mi.tolist()
    assert bits.tolist() == [BITS[i] for i in bi]


def test_golden_costs_on_paper_shapes():
    for Hq, d, Hkv, w, p, mode, b, swk, flops, kvb in _read_golden("route_cost.txt"):
        ml = _one_hot_logits([mode], 3)
        bl = _one_hot_logits([BITS.index(b)], 4)
        m, bb, f, mem, tot = oracle.route_decisions(ml, bl, [p], w, Hq, d, Hkv, swk)
        assert (m[0], bb[0], f[0], mem[0]) == (mode, b, flops, kvb), (Hq, d, Hkv, w, p, mode, b)
        assert tot[0] == flops and tot[1] == kvb


def test_dense_normalisers_closed_form_and_budget_bounds():
    """C_dense of Appendix C: sum over t = 1..T of Hq 2 d t and of 2 d_kv 16; a policy
    never costs more than dense, and all-full / all-16 costs exactly dense."""
    rng = np.random.default_rng(3)
    T, Hq, d, Hkv, w = 700, 12, 64, 3, 256
    pos = np.arange(T)
    ml = rng.standard_normal((T, 3)).astype(np.float32)
    bl = rng.standard_normal((T, 4)).astype(np.float32)
    m, b, f, mem, tot = oracle.route_decisions(ml, bl, pos, w, Hq, d, Hkv)
    assert tot[2] == Hq * 2 * d * T * (T + 1) // 2
    assert tot[3] == T * 2 * Hkv * d * 16
    assert tot[0] == f.sum() and tot[1] == mem.sum()
    assert (f <= Hq * 2 * d * (pos + 1)).all() and (mem <= 2 * Hkv * d * 16).all()
    full = oracle.route_decisions(_one_hot_logits([FULL] * T, 3), _one_hot_logits([3] * T, 4),
                                  pos, w, Hq, d, Hkv)
    assert full[4][0] == full[4][2] and full[4][1] == full[4][3]
    # totals accumulate across calls (layers)
    again = oracle.route_decisions(ml, bl, pos, w, Hq, d, Hkv, totals=tot)[4]
    assert (again == 2 * tot).all()


def test_attention_cost_counts_the_keys_the_oracle_attention_reads():
    """Every token stored at width 16: the keys a query's mode makes the attention read
    (counted through uniform softmax weights over the key positions) are the cost's
    kappa, and a skip query reads nothing (zero row)."""
    rng = np.random.default_rng(21)
    d, T = 64, 90
    o = oracle.OracleCache(1, 1, 1, 1, d, 32, 16, T, [16] * 4)
    K = bf16_bits(np.zeros((T, 1, d), dtype=np.float32))
    V = np.zeros((T, 1, d), dtype=np.float32)
    V[:, 0, 0] = 1.0
    V[:, 0, 1] = np.arange(T)
    assert o.append(0, [0] * T, np.arange(T), K, bf16_bits(V), [16] * T, [FULL] * T) == 0
    q = bf16_bits(np.ones((1, 1, d), dtype=np.float32))
    for _ in range(60):
        p, w = int(rng.integers(0, T)), int(rng.integers(1, 40))
        ml = rng.standard_normal((1, 3)).astype(np.float32)
        m, _, f, _, _ = oracle.route_decisions(ml, np.zeros((1, 4), np.float32), [p], w, 1, d, 1)
        st, out = o.decode_attn(0, [0], [p], q, [int(m[0])], window_scalar=w)
        assert st == 0
        if m[0] == SKIP:
            assert f[0] == 0 and not out.any()
            continue
        keys = round(2 * (p - out[0, 0, 1]) + 1)     # mean of positions p-k+1 .. p
        assert f[0] == 2 * d * keys, (p, w, int(m[0]))


def test_memory_cost_equals_the_payload_the_oracle_cache_stores():
    """Charged bits = code bits the oracle's append stores for the same decisions (its
    per-group binary16 scale/zero pairs excluded, as the cost model has none)."""
    rng = np.random.default_rng(8)
    Hq, Hkv, d, G, P, T = 4, 2, 64, 32, 16, 150
    for swk in (0, 1):
        o = oracle.OracleCache(1, 1, Hq, Hkv, d, G, P, T, [64] * 4, skip_writes_kv=swk)
        ml = rng.standard_normal((T, 3)).astype(np.float32)
        bl = rng.standard_normal((T, 4)).astype(np.float32)
        m, b, f, mem, tot = oracle.route_decisions(ml, bl, np.arange(T), 32, Hq, d, Hkv, swk)
        K = bf16_bits(rng.standard_normal((T, Hkv, d), dtype=np.float32))
        V = bf16_bits(rng.standard_normal((T, Hkv, d), dtype=np.float32))
        assert o.append(0, [0] * T, np.arange(T), K, V, b, m) == 0
        ntok = o.region("ntok").view(np.int32)
        stored = 0
        for c in range(4):
            tokb = o.slice_bytes(c) // P
            overhead = 0 if c == 3 else 2 * (d // G) * 4
            stored += int(ntok[c]) * (tokb - overhead) * 8 * Hkv
        assert stored == tot[1], swk
