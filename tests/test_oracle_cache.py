"""Pins of the oracle's paged cache (Sec. 3.8: KV stored at the chosen width, paged;
Sec. 7: tokens grouped by precision): allocation invariants, bulk == incremental
append, the error contract, the byte layout checked by hand, and the stored values
against the quantiser pinned in test_oracle_quantizer.py."""
import numpy as np
import pytest

import oracle
from paper_2607_06601_gb300.workloads import bf16_bits, bf16_to_f32

SKIP, LOCAL, FULL = 0, 1, 2
BITS = [2, 4, 8, 16]


def _fill(o, rng, S, n, layer=0, per_call=1):
    bits = rng.choice(BITS, size=(S, n))
    modes = rng.choice([SKIP, LOCAL, FULL], size=(S, n))
    K = bf16_bits(rng.standard_normal((S, n, o.Hkv, o.d), dtype=np.float32))
    V = bf16_bits(rng.standard_normal((S, n, o.Hkv, o.d), dtype=np.float32))
    ent = [(s, p) for p in range(n) for s in range(S)]
    for i in range(0, len(ent), per_call):
        chunk = ent[i:i + per_call]
        ss = [e[0] for e in chunk]
        pp = [e[1] for e in chunk]
        st = o.append(layer, ss, pp, K[ss, pp], V[ss, pp], bits[ss, pp], modes[ss, pp])
        assert st == 0
    return bits, modes, K, V


def _regions(o):
    return {k: o.region(k) for k in oracle.REGIONS}


def test_allocation_invariants():
    rng = np.random.default_rng(21)
    L, S, n, P = 2, 5, 150, 16
    o = oracle.OracleCache(L, S, 4, 2, 64, 32, P, n, [200] * 4)
    maps = [_fill(o, rng, S, n, layer=l) for l in range(L)]
    MP = -(-n // P)
    ntok = o.region("ntok").view(np.int32).reshape(L, S, 4)
    pres = o.region("presence").view(np.uint32).reshape(L, S, -1)
    pt = o.region("page_table").view(np.int32).reshape(L, S, 4, MP)
    pf = o.region("page_first").view(np.int32).reshape(L, S, 4, MP)
    pl = o.region("page_last").view(np.int32).reshape(L, S, 4, MP)
    nextp = o.region("next_page").view(np.int32)
    used = [set() for _ in range(4)]
    for l in range(L):
        bits, modes, _, _ = maps[l]
        for s in range(S):
            stored = modes[s] != SKIP
            # presence == the non-skip tokens, bit p of word p // 32
            bitsset = [(pres[l, s, p // 32] >> (p % 32)) & 1 for p in range(n)]
            assert np.array_equal(np.array(bitsset, dtype=bool), stored)
            for c, b in enumerate(BITS):
                want = np.nonzero(stored & (bits[s] == b))[0]
                assert ntok[l, s, c] == len(want)
                npg = -(-len(want) // P)
                got = []
                for k in range(npg):
                    pid = pt[l, s, c, k]
                    assert pid not in used[c]
                    used[c].add(pid)
                    page = o.region(f"pool{b}")[pid * o.page_bytes(c):(pid + 1) * o.page_bytes(c)]
                    fill = min(P, len(want) - k * P)
                    pos = page[:4 * fill].view(np.int32)
                    assert pf[l, s, c, k] == pos[0] and pl[l, s, c, k] == pos[-1]
                    got += list(pos)
                assert (pt[l, s, c, npg:] == -1).all()
                assert np.array_equal(got, want)         # each stored token once, in order
    for c in range(4):
        assert used[c] == set(range(nextp[c]))          # ids 0 .. next_page-1, each once


def test_bulk_append_equals_incremental():
    rng_a, rng_b = np.random.default_rng(3), np.random.default_rng(3)
    S, n = 4, 100
    a = oracle.OracleCache(1, S, 2, 2, 64, 32, 16, n, [64] * 4)
    b = oracle.OracleCache(1, S, 2, 2, 64, 32, 16, n, [64] * 4)
    _fill(a, rng_a, S, n, per_call=1)
    _fill(b, rng_b, S, n, per_call=S * n)
    ra, rb = _regions(a), _regions(b)
    for k in ra:
        assert np.array_equal(ra[k], rb[k]), k


def test_byte_layout_by_hand():
    """One 4-bit token, d = 64, G = 32, P = 16, 2 KV heads: every byte at the place the
    documented layout puts it."""
    d, G, P, Hkv = 64, 32, 16, 2
    o = oracle.OracleCache(1, 1, 2, Hkv, d, G, P, 32, [2] * 4)
    hdr = 128
    tokb = 2 * (d * 4 // 8) + 2 * (d // G) * 4            # 80 bytes per token and head
    assert o.hdr_bytes == hdr and o.slice_bytes(1) == P * tokb
    assert o.page_bytes(1) == hdr + Hkv * P * tokb        # 2688, a multiple of 128
    x = np.zeros((1, Hkv, d), dtype=np.float32)
    x[0, 1, :32] = np.arange(32) % 16                     # head 1, group 0: 0..15 twice
    x[0, 1, 32:] = 7.0                                     # head 1, group 1: constant
    xv = -x
    st = o.append(0, [0, 0], [5, 9], np.concatenate([bf16_bits(x)] * 2),
                  np.concatenate([bf16_bits(xv)] * 2), [4, 4], [FULL, LOCAL])
    assert st == 0
    page = o.region("pool4")[:o.page_bytes(1)]
    assert list(page[:8].view(np.int32)) == [5, 9]
    sl = page[hdr + P * tokb:]                             # head 1
    kc = sl[:P * 32].reshape(P, 32)                        # K codes [P][d*b/8]
    vc = sl[P * 32:2 * P * 32].reshape(P, 32)
    ksz = sl[2 * P * 32:2 * P * 32 + P * 8].view(np.uint16).reshape(P, 2, 2)
    vsz = sl[2 * P * 32 + P * 8:2 * P * 32 + 2 * P * 8].view(np.uint16).reshape(P, 2, 2)
    ramp = np.arange(32) % 16
    assert list(kc[1, :16]) == [int(ramp[2 * j]) | (int(ramp[2 * j + 1]) << 4) for j in range(16)]
    assert (kc[1, 16:] == 0).all()                         # constant group -> code 0
    assert list(ksz[1, 0]) == [int(np.float16(1).view(np.uint16)), 0]      # s = 1, z = 0
    assert list(ksz[1, 1]) == [0, int(np.float16(7).view(np.uint16))]      # s = 0, z = 7
    assert list(vsz[1, 0]) == [int(np.float16(1).view(np.uint16)),
                               int(np.float16(-15).view(np.uint16))]
    assert list(vc[1, :16]) == [int(15 - ramp[2 * j]) | (int(15 - ramp[2 * j + 1]) << 4)
                                for j in range(16)]


@pytest.mark.parametrize("Hq,Hkv,permuted", [(2, 2, True), (4, 2, False), (16, 2, True)])
def test_chunk_order_of_wide_rows_by_hand(Hq, Hkv, permuted):
    """One 8-bit and one 16-bit token at slot 3, d = 64, G = 32, P = 16: where every
    16-byte chunk of their K rows is stored.  In a cache read by the CUDA-core path (MHA;
    query groups too wide for one 8-column mma tile) line n of a slice keeps logical chunk
    k at chunk k ^ (n % 8); in a tensor-core cache (g = 2: 4 columns) rows are plain."""
    d, G, P, slot = 64, 32, 16, 3
    o = oracle.OracleCache(1, 2, Hq, Hkv, d, G, P, 32, [2] * 4)
    rng = np.random.default_rng(3)
    K = bf16_bits(rng.standard_normal((2, Hkv, d), dtype=np.float32))
    V = bf16_bits(rng.standard_normal((2, Hkv, d), dtype=np.float32))
    for p in range(slot + 1):  # the fourth token of each sequence lands in slot 3
        assert o.append(0, [0, 1], [p, p], K, V, [16, 8], [FULL, FULL]) == 0
    for b, c, seq in ((16, 3, 0), (8, 2, 1)):
        rowb = d * b // 8
        page = o.region(f"pool{b}")[:o.page_bytes(c)]
        sl = page[o.hdr_bytes:o.hdr_bytes + o.slice_bytes(c)]     # KV head 0
        if b == 16:
            logical = K[seq, 0].view(np.uint8)
        else:  # 8-bit codes: one byte each, in element order
            _, _, c0, _ = oracle.quantize_group(K[seq, 0][:32], 8)
            _, _, c1, _ = oracle.quantize_group(K[seq, 0][32:], 8)
            logical = np.concatenate([c0, c1]).astype(np.uint8)
        assert logical.size == rowb
        for k in range(rowb // 16):
            x = slot * rowb + 16 * k                       # logical offset in the slice
            n, ch = x // 128, (x // 16) % 8
            at = n * 128 + ((ch ^ (n % 8)) if permuted else ch) * 16
            assert np.array_equal(sl[at:at + 16], logical[16 * k:16 * k + 16]), (b, k)


def test_stored_values_are_the_quantiser_output():
    rng = np.random.default_rng(9)
    o = oracle.OracleCache(1, 2, 4, 2, 128, 64, 16, 40, [16] * 4)
    bits, modes, K, V = _fill(o, rng, 2, 40)
    for s in range(2):
        for p in range(40):
            for h in range(2):
                c, kk, vv = o.dequant_token(0, s, p, h)
                if modes[s, p] == SKIP:
                    assert c == -1
                    continue
                b = bits[s, p]
                for ref_bits, got in ((K[s, p, h], kk), (V[s, p, h], vv)):
                    if b == 16:
                        assert np.array_equal(bf16_to_f32(ref_bits).astype(np.float64), got)
                        continue
                    for g in range(2):
                        s16, z16, codes, _ = oracle.quantize_group(ref_bits[g * 64:(g + 1) * 64], b)
                        sf = float(np.uint16(s16).view(np.float16))
                        zf = float(np.uint16(z16).view(np.float16))
                        assert np.array_equal(zf + codes * sf, got[g * 64:(g + 1) * 64])


def _snapshot(o):
    return {k: v.copy() for k, v in _regions(o).items()}


def test_error_contract_leaves_state_unchanged():
    rng = np.random.default_rng(4)
    o = oracle.OracleCache(1, 2, 2, 1, 64, 32, 16, 64, [2, 1, 1, 1])
    K = bf16_bits(rng.standard_normal((8, 1, 64), dtype=np.float32))
    assert o.append(0, [0, 1], [0, 0], K[:2], K[:2], [2, 4], [FULL, FULL]) == 0
    snap = _snapshot(o)
    cases = [
        (([0, 5], [1, 1], [2, 2], [1, 1]), 1),      # sequence id out of range
        (([0, 1], [1, 1], [2, 3], [1, 1]), 1),      # bits not in {2,4,8,16}
        (([0, 1], [1, 1], [2, 2], [1, 3]), 1),      # mode not in {0,1,2}
        (([0, 1], [1, 64], [2, 2], [1, 1]), 4),     # position >= max_context
        (([0, 1], [1, 0], [2, 2], [1, 1]), 4),      # position not above the last one
        (([0, 0], [3, 2], [2, 2], [1, 1]), 4),      # decreasing inside one call
        (([1, 1], [1, 2], [4, 8], [2, 2]), 0),      # fine (checked below separately)
    ]
    for (seqs, pos, bits, modes), want in cases[:-1]:
        assert o.append(0, seqs, pos, K[:2], K[:2], bits, modes) == want
        now = _snapshot(o)
        for k in snap:
            assert np.array_equal(snap[k], now[k]), (k, seqs, pos, bits, modes)
    # the lowest failing index decides the code
    assert o.append(0, [0, 0], [0, 99], K[:2], K[:2], [2, 2], [1, 1]) == 4
    assert o.append(0, [7, 0], [1, 0], K[:2], K[:2], [2, 2], [1, 1]) == 1
    # class pool exhaustion: 2 pages of 2-bit, both can be opened, a third cannot
    assert o.append(0, [1], [1], K[:1], K[:1], [2], [FULL]) == 0     # opens 2-bit page 1
    snap = _snapshot(o)
    big = 40
    Kb = bf16_bits(rng.standard_normal((big, 1, 64), dtype=np.float32))
    assert o.append(0, [0] * big, np.arange(2, 2 + big), Kb, Kb, [2] * big, [FULL] * big) == 3
    now = _snapshot(o)
    for k in snap:
        assert np.array_equal(snap[k], now[k]), k
    # several pages opened inside one call: the capacity check counts each of them
    fresh = oracle.OracleCache(1, 2, 2, 1, 64, 32, 16, 64, [1, 1, 1, 1])
    n17 = 17
    Kc = bf16_bits(rng.standard_normal((n17, 1, 64), dtype=np.float32))
    snap = _snapshot(fresh)
    assert fresh.append(0, [0] * n17, np.arange(n17), Kc, Kc, [4] * n17, [FULL] * n17) == 3
    now = _snapshot(fresh)
    for k in snap:
        assert np.array_equal(snap[k], now[k]), k
    assert fresh.append(0, [0] * 16, np.arange(16), Kc[:16], Kc[:16], [4] * 16, [FULL] * 16) == 0
    # a non-finite value: the group is stored as zeros, the rest of the call applies
    Kn = K[:1].copy()
    Kn[0, 0, 3] = 0x7F80                                   # +inf in group 0
    assert o.append(0, [1], [2], Kn, K[:1], [8], [FULL]) == 7
    c, kk, vv = o.dequant_token(0, 1, 2, 0)
    assert c == 2 and (kk[:32] == 0).all() and np.abs(kk[32:]).max() > 0
