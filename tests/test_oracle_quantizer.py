"""Pins of the oracle's number formats and quantiser (Sec. 3.2(C), Eq. 4) against
facts that do not come from the oracle itself: numpy's IEEE conversions, the exact
nearest-level definition enumerated over all 2^b levels, the closed-form error bound,
hand-packed bytes, and special cases with known answers."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2607_06601_gb300.workloads import bf16_bits


def test_bf16_decode_all_patterns():
    pats = np.arange(65536, dtype=np.uint32)
    ref = (pats << 16).view(np.float32).astype(np.float64)
    for h in range(0, 65536, 97):
        got = oracle.bf16_to_double(h)
        if np.isnan(ref[h]):
            assert np.isnan(got)
        else:
            assert got == ref[h], h


def test_f16_decode_all_patterns():
    ref = np.arange(65536, dtype=np.uint16).view(np.float16).astype(np.float64)
    for h in range(65536):
        got = oracle.f16_to_double(h)
        if np.isnan(ref[h]):
            assert np.isnan(got)
        else:
            assert got == ref[h], h


def test_f16_encode_matches_numpy_rne():
    rng = np.random.default_rng(11)
    xs = np.concatenate([
        rng.standard_normal(20000) * 10.0 ** rng.uniform(-9, 4.8, 20000),
        # exact ties between neighbouring binary16 values, normal and subnormal
        (np.arange(1, 2000, dtype=np.float64) + 0.5) * 2.0 ** -24,
        (np.arange(1024, 3000, dtype=np.float64) + 0.5) * 2.0 ** -10,
        [0.0, -0.0, 65504.0, -65504.0, 2.0 ** -14, 2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26],
    ])
    xs = xs[np.abs(xs) <= 65504]
    ref = xs.astype(np.float16).view(np.uint16)
    for x, r in zip(xs, ref):
        assert oracle.double_to_f16(float(x)) == int(r), x


def test_pack_hand_examples():
    # element j at byte floor(j*b/8), bit (j*b) % 8, least significant bits first
    assert oracle.pack_codes([1, 2, 3, 0], 2) == bytes([0x39])
    assert oracle.pack_codes([3, 0, 0, 0, 0, 0, 0, 2], 2) == bytes([0x03, 0x80])
    assert oracle.pack_codes([0xA, 0x5], 4) == bytes([0x5A])
    assert oracle.pack_codes([7, 200, 255, 0], 8) == bytes([7, 200, 255, 0])


def _exact_nearest_ok(x, z, s, c, levels):
    xf, zf, sf = Fraction(x), Fraction(z), Fraction(s)
    d = abs(xf - (zf + c * sf))
    for nb in (c - 1, c + 1):
        if 0 <= nb <= levels:
            dn = abs(xf - (zf + nb * sf))
            if dn < d or (dn == d and c % 2 == 1):
                return False
    return True


def _groups(rng, G, count):
    out = [rng.standard_normal(G).astype(np.float32) for _ in range(count)]
    out += [(rng.standard_normal(G) * 8).astype(np.float32) for _ in range(count // 4)]
    out += [(rng.standard_normal(G) * 1e-3 + 5).astype(np.float32) for _ in range(count // 8)]
    out += [rng.uniform(-60000, 60000, G).astype(np.float32) for _ in range(count // 8)]
    out += [(rng.standard_normal(G) * 1e-6).astype(np.float32) for _ in range(count // 8)]
    return [bf16_bits(g) for g in out]


@pytest.mark.parametrize("b", [2, 4, 8])
@pytest.mark.parametrize("G", [32, 64, 128])
def test_quantizer_nearest_level_and_bound(b, G):
    """codes are the nearest level z + c*s (all 2^b levels enumerated), ties to the even
    code, decided in exact rational arithmetic; every element meets the closed-form bound
    of Eq. 4 with binary16 s and z."""
    rng = np.random.default_rng(1000 * b + G)
    levels = (1 << b) - 1
    for xb in _groups(rng, G, 60):
        s16, z16, codes, bad = oracle.quantize_group(xb, b)
        assert not bad
        x = (xb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        mn, mx = x.min(), x.max()
        # scale/zero as the paper defines them, rounded the documented way (numpy IEEE)
        assert z16 == int(np.float16(mn).view(np.uint16))
        s_ref = np.float32(np.float32(mx - mn) / np.float32(levels))
        assert s16 == int(np.float16(s_ref).view(np.uint16))
        z = float(np.uint16(z16).view(np.float16))
        s = float(np.uint16(s16).view(np.float16))
        assert codes.max() <= levels
        if s == 0:
            assert (codes == 0).all()
            continue
        lv = z + np.arange(levels + 1) * s             # exact in float64
        dist = np.abs(x[:, None] - lv[None, :])
        best = dist.min(axis=1)
        chosen = dist[np.arange(G), codes]
        assert (chosen <= best * (1 + 1e-9) + 1e-300).all()
        # exactly: |x - level| is convex in the code, so the chosen code beats both
        # neighbours (strictly, or equal with the chosen code even)
        for xi, c in zip(x, codes):
            assert _exact_nearest_ok(xi, z, s, int(c), levels), (xi, z, s, c)
        xhat = z + codes * s
        bound = max(s / 2 * (1 + 1e-5), z - mn, mx - lv[-1], 0.0)
        assert (np.abs(x - xhat) <= bound + 1e-300).all()


def test_quantizer_special_cases():
    # constant group: s = 0, every code 0, and x is recovered exactly
    xb = bf16_bits(np.full(32, 1.5, dtype=np.float32))
    s16, z16, codes, bad = oracle.quantize_group(xb, 4)
    assert (s16, bad) == (0, False) and (codes == 0).all()
    assert float(np.uint16(z16).view(np.float16)) == 1.5
    # integer ramp spanning exactly 2^b levels: s = 1, z = 0, codes = x
    for b in (2, 4, 8):
        vals = np.resize(np.arange(1 << b), 32 if b < 8 else 256)[:128].astype(np.float32)
        vals[0], vals[1] = 0, (1 << b) - 1
        s16, z16, codes, bad = oracle.quantize_group(bf16_bits(vals), b)
        assert float(np.uint16(s16).view(np.float16)) == 1.0
        assert float(np.uint16(z16).view(np.float16)) == 0.0
        assert (codes == vals).all()
    # half-way points go to the even code: x = z + (c + 1/2) s
    vals = np.array([0, 3, 0.5, 1.5, 2.5, 1, 2, 3] * 4, dtype=np.float32)
    s16, z16, codes, _ = oracle.quantize_group(bf16_bits(vals), 2)
    assert list(codes[:8]) == [0, 3, 0, 2, 2, 1, 2, 3]


def test_quantizer_rounds_the_exact_quotient():
    """Near a half-way point the code follows the exact quotient (x - z) / s, not a
    rounded one: with z = -2.5 and s = 1, x = +-2^-60 gives quotients 2.5 +- 2^-60, which
    round to 3 and 2, although binary32 (or binary64) arithmetic would see a tie at 2.5."""
    tiny = 2.0 ** -60
    vals = np.array([-2.5, 0.5, tiny, -tiny, 0.0, 2.0 ** -30, -(2.0 ** -30), 0.5] * 4, dtype=np.float32)
    s16, z16, codes, bad = oracle.quantize_group(bf16_bits(vals), 2)
    assert not bad
    assert float(np.uint16(s16).view(np.float16)) == 1.0
    assert float(np.uint16(z16).view(np.float16)) == -2.5
    assert list(codes[:8]) == [0, 3, 3, 2, 2, 3, 2, 3]
    # the same at every half-way point c + 1/2 that bf16 inputs can put a tie on:
    # z = -(c + 1/2), s = 1, x in {+tiny, -tiny, 0}
    for b, cs in ((2, range(3)), (4, range(15)), (8, [127])):
        levels = (1 << b) - 1
        for c in cs:
            grp = np.array([-(c + 0.5), levels - c - 0.5] + [tiny, -tiny, 0.0] * 10, dtype=np.float32)
            s16, z16, codes, bad = oracle.quantize_group(bf16_bits(grp), b)
            assert float(np.uint16(s16).view(np.float16)) == 1.0
            assert float(np.uint16(z16).view(np.float16)) == -(c + 0.5)
            assert list(codes[2:5]) == [c + 1, c, c + (c % 2)], (b, c)


def test_quantizer_rejects_unrepresentable_values():
    for bad_val in (np.nan, np.inf, -np.inf, 70000.0, -1e6):
        vals = np.zeros(32, dtype=np.float32)
        vals[5] = bad_val
        s16, z16, codes, bad = oracle.quantize_group(bf16_bits(vals), 4)
        assert bad and s16 == 0 and z16 == 0 and (codes == 0).all()
    vals = np.zeros(32, dtype=np.float32)
    vals[3] = 65280.0  # the largest bf16 value <= 65504 is accepted
    assert not oracle.quantize_group(bf16_bits(vals), 8)[3]
