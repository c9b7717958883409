"""The bench's algorithmic-byte accounting (the numerator of every GB/s it reports),
checked against a brute-force count over the cache layout on small random maps: per
stored key in a query's range its K+V payload with fp16 scale/zero for every KV head
that reads it and 4 bytes of slot position; per page in range 4 bytes of page table
(and with per-head modes 8 bytes of presence mask per KV head read); the Q rows of the
heads that read and every O row."""
import itertools
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402
from paper_2607_06601_gb300 import workloads as wl  # noqa: E402

BITS = (2, 4, 8, 16)


def _tok_bytes(d, G, b):
    return d * 2 * 2 if b == 16 else 2 * (d * b // 8) + 2 * (d // G) * 4


def _brute(bits, hmodes, t, Hq, Hkv, d, G, P, w, swk):
    """(bytes without presence masks, pages in range, keys per KV head, KV heads read) of
    query t (modes per head [T][Hq]), by enumeration."""
    g = Hq // Hkv
    m = hmodes[t]
    O = 2 * Hq * d
    if not m.any():
        return O, set(), 0.0, 0
    total = O + 2 * d * int(np.count_nonzero(m))
    stores = np.array([[swk or hmodes[p, j * g:(j + 1) * g].any() for j in range(Hkv)]
                       for p in range(t + 1)])
    took = stores.any(1)
    lo_q = 0 if (m == 2).any() else max(0, t - w + 1)
    keys = 0
    for j in range(Hkv):
        mj = m[j * g:(j + 1) * g]
        if not mj.any():
            continue
        lo = 0 if (mj == 2).any() else max(0, t - w + 1)
        for p in range(lo, t + 1):
            if stores[p, j]:
                total += _tok_bytes(d, G, bits[p])
                keys += 1
    pages = set()
    for p in range(lo_q, t + 1):
        if took[p]:
            total += 4
            c = BITS.index(bits[p])
            pages.add((c, int(np.count_nonzero(took[:p] & (bits[:p] == bits[p]))) // P))
    return total, pages, keys / Hkv, sum(1 for j in range(Hkv) if m[j * g:(j + 1) * g].any())


@pytest.mark.parametrize("Hq,Hkv,swk", [(4, 4, 0), (4, 2, 0), (6, 3, 1), (2, 1, 0)])
def test_per_head_accounting_matches_enumeration(Hq, Hkv, swk):
    rng = np.random.default_rng(Hq * 7 + Hkv + swk)
    d, G, P, w, T = 64, 32, 16, 9, 70
    spec = wl.SPECS["tiny"]
    acct = bench.Accounting(spec, d, G, Hq, Hkv, w, P, swk)
    for trial in range(40):
        bits = rng.choice(BITS, size=T)
        hm = rng.choice(3, size=(T, Hq), p=[0.4, 0.3, 0.3]).astype(np.uint8)
        if trial % 8 == 0:
            hm[T // 2] = 0  # a query no head of which reads: its zero O rows only
        t = T // 2 if trial % 8 == 0 else int(rng.integers(0, T))
        got = acct.query_heads(bits, hm, t)
        total, pages, keys, nkv_read = _brute(bits, hm, t, Hq, Hkv, d, G, P, w, swk)
        assert got[1] == pytest.approx(keys)
        assert got[2] == len(pages)
        assert got[0] == total + len(pages) * (4 + 8 * nkv_read)


@pytest.mark.parametrize("swk", [0, 1])
def test_per_token_accounting_is_per_head_with_equal_heads(swk):
    """One mode for all heads of a token: the per-token count equals the per-head count
    less the presence masks (which a per-token cache does not have)."""
    spec = wl.SPECS["160m"]
    Hq = Hkv = 12
    a = bench.Accounting(spec, 64, 32, Hq, Hkv, 256, 32, swk)
    bits, modes = wl.policy(spec, 0, 0, 2048)
    hm = np.repeat(modes[:, None], Hq, 1)
    for t in itertools.chain([0, 1, 2047], np.random.default_rng(1).integers(0, 2048, 30)):
        x = a.query(bits, modes, int(t))
        y = a.query_heads(bits, hm, int(t))
        assert x[1] == y[1] and x[2] == y[2]
        assert y[0] - x[0] == (8 * Hkv * y[2] if modes[t] else 0)


def test_threaded_oracle_baseline_runs_the_same_queries():
    """The CPU baseline's oracle sample: with a budget that lets every query of the
    sample run, one thread and four threads process the same queries (same algorithmic
    bytes, keys and count), each query's bytes being the accounting's."""
    spec = wl.SPECS["tiny"]
    sample = bench.OracleSample(spec, 4, spec.window)
    assert sample.n_queries == int(wl.contexts(spec).min()) * sample.n_seqs
    one = sample.run(60.0, threads=1)
    four = sample.run(60.0, threads=4)
    assert one[2] == four[2] == sample.n_queries
    assert one[:3] == four[:3]
    total = 0
    for j in range(sample.n_queries):
        nb, _ = sample.query(j)
        total += nb
    assert total == one[0]
