"""GPU parity of the router's hard decisions (Sec. 3.8) and their cost (Sec. 3.5,
Appendix C): trr_route_decisions against the oracle, bit-exact (decisions and costs are
integers, and both sides compare the same binary32 logits); the routed append and
attention, which take the decisions inside their own kernels, against the oracle cache
fed the oracle's decisions, and against the plain calls fed trr_route_decisions'
output.  Every call goes through the C ABI (libtrr.so)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_06601_gb300 import trr
from paper_2607_06601_gb300 import workloads as wl
from tests._parity import Pair, check_attention, dev

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def _logits(rng, n, k, ties=True):
    """Router logits with many exact ties, NaN and infinities mixed in."""
    if ties:
        z = rng.integers(-3, 4, size=(n, k)).astype(np.float32)
    else:
        z = rng.standard_normal((n, k)).astype(np.float32)
    z[rng.random(z.shape) < 0.08] = np.nan
    z[rng.random(z.shape) < 0.03] = np.inf
    z[rng.random(z.shape) < 0.03] = -np.inf
    z[: min(n, 3)] = np.nan  # rows of NaN only
    return z


def _gpu_route(ml, bl, pos, w, Hq, d, Hkv, swk, totals0):
    n = ml.shape[0]
    out = {"modes": torch.full((n,), 255, dtype=torch.uint8, device="cuda"),
           "bits": torch.full((n,), 255, dtype=torch.uint8, device="cuda"),
           "attn_flops": torch.full((n,), -1, dtype=torch.int64, device="cuda"),
           "kv_bits": torch.full((n,), -1, dtype=torch.int64, device="cuda")}
    tot = torch.tensor(totals0, dtype=torch.int64, device="cuda")
    trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32), dev(pos, torch.int32), w, Hq,
                            d, Hkv, swk, totals=tot, **out)
    torch.cuda.synchronize()
    return [out[k].cpu().numpy() for k in ("modes", "bits", "attn_flops", "kv_bits")] + [tot.cpu().numpy()]


@pytest.mark.parametrize("Hq,d,Hkv,w", [(12, 64, 3, 256), (16, 128, 4, 128), (32, 64, 32, 512)])
@pytest.mark.parametrize("swk", [0, 1])
def test_route_decisions_match_oracle(Hq, d, Hkv, w, swk):
    rng = np.random.default_rng(Hq + d + w + swk)
    n = 3001
    ml, bl = _logits(rng, n, 3), _logits(rng, n, 4, ties=False)
    pos = rng.integers(-5, 40000, size=n).astype(np.int32)
    pos[5:10] = [0, 1, w - 1, w, w + 1]
    totals0 = [5, 7, 11, 13]
    got = _gpu_route(ml, bl, pos, w, Hq, d, Hkv, swk, totals0)
    ref = oracle.route_decisions(ml, bl, pos, w, Hq, d, Hkv, swk, totals=totals0)
    for name, g, r in zip(("modes", "bits", "attn_flops", "kv_bits", "totals"), got, ref):
        assert np.array_equal(g, r), f"{name} differs at {np.nonzero(g != r)[0][:8]}"


def test_route_decisions_optional_outputs():
    rng = np.random.default_rng(4)
    n = 777
    ml, bl = _logits(rng, n, 3), _logits(rng, n, 4)
    ref = oracle.route_decisions(ml, bl, np.arange(n), 64, 8, 64, 2)
    modes = torch.zeros(n, dtype=torch.uint8, device="cuda")
    trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32), modes=modes)
    bits = torch.zeros(n, dtype=torch.uint8, device="cuda")
    trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32), bits=bits)
    tot = torch.zeros(4, dtype=torch.int64, device="cuda")
    trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32),
                            dev(np.arange(n, dtype=np.int32), torch.int32), 64, 8, 64, 2, totals=tot)
    torch.cuda.synchronize()
    assert np.array_equal(modes.cpu().numpy(), ref[0])
    assert np.array_equal(bits.cpu().numpy(), ref[1])
    assert np.array_equal(tot.cpu().numpy(), ref[4])
    # cost outputs need positions and a window of at least 1; nothing is launched
    with pytest.raises(trr.TrrError):
        trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32), totals=tot)
    with pytest.raises(trr.TrrError):
        trr.trr_route_decisions(dev(ml, torch.float32), dev(bl, torch.float32),
                                dev(np.arange(n, dtype=np.int32), torch.int32), 0, 8, 64, 2, totals=tot)
    trr.trr_route_decisions(torch.zeros((0, 3), device="cuda"), torch.zeros((0, 4), device="cuda"))


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 1023])
def test_route_decisions_unaligned_arrays_and_short_calls(n):
    """Arrays off the 16-byte grid take the token-by-token path; every n mod 4."""
    rng = np.random.default_rng(n)
    ml, bl = _logits(rng, n + 1, 3), _logits(rng, n + 1, 4)
    pos = rng.integers(0, 5000, size=n + 1).astype(np.int32)
    mt, bt, pt = dev(ml, torch.float32), dev(bl, torch.float32), dev(pos, torch.int32)
    out = {"modes": torch.zeros(n + 1, dtype=torch.uint8, device="cuda"),
           "bits": torch.zeros(n + 1, dtype=torch.uint8, device="cuda"),
           "attn_flops": torch.zeros(n + 1, dtype=torch.int64, device="cuda"),
           "kv_bits": torch.zeros(n + 1, dtype=torch.int64, device="cuda")}
    tot = torch.zeros(4, dtype=torch.int64, device="cuda")
    trr.trr_route_decisions(mt[1:], bt[1:], pt[1:], 100, 12, 64, 3, 1, totals=tot,
                            **{k: v[1:] for k, v in out.items()})
    torch.cuda.synchronize()
    ref = oracle.route_decisions(ml[1:], bl[1:], pos[1:], 100, 12, 64, 3, 1)
    for (name, t), r in zip(out.items(), ref[:4]):
        g = t.cpu().numpy()
        assert g[0] == 0 and np.array_equal(g[1:], r), name
    assert np.array_equal(tot.cpu().numpy(), ref[4])


def test_route_decisions_two_million_tokens():
    """More tokens than one wave of CTAs (the grid-stride loop), every output checked."""
    rng = np.random.default_rng(12)
    n = 1 << 21
    ml = rng.standard_normal((n, 3)).astype(np.float32)
    bl = rng.standard_normal((n, 4)).astype(np.float32)
    ml[rng.random(n) < 0.01, 1] = np.nan
    pos = rng.integers(0, 300, size=n).astype(np.int32)
    got = _gpu_route(ml, bl, pos, 32, 12, 64, 12, 0, [0, 0, 0, 0])
    ref = oracle.route_decisions(ml, bl, pos, 32, 12, 64, 12, 0)
    for name, g, r in zip(("modes", "bits", "attn_flops", "kv_bits", "totals"), got, ref):
        assert np.array_equal(g, r), name


@pytest.mark.parametrize("d,G,P,Hq,Hkv,per_call", [(64, 32, 16, 12, 12, 1024), (64, 32, 16, 12, 12, 97),
                                                   (128, 64, 16, 32, 8, 1024), (128, 64, 32, 8, 4, 200)])
def test_routed_append_and_attention(d, G, P, Hq, Hkv, per_call):
    """Routed calls (decisions from logits inside the kernels) equal the oracle fed the
    oracle's decisions: cache bytes bit-exact, attention within the stated bar; and the
    plain calls fed trr_route_decisions' modes give the same bf16 rows bit for bit."""
    rng = np.random.default_rng(d + P + Hq + per_call)
    ctxs = [3, 40, 170, 333]
    S, maxctx, w = len(ctxs), max(ctxs) + 8, 24
    caps = [S * (maxctx // P + 2)] * 4
    pair = Pair(1, S, Hq, Hkv, d, G, P, maxctx, caps)
    ent = [(s, p) for p in range(max(ctxs)) for s in range(S) if p < ctxs[s]]
    ml, bl = _logits(rng, len(ent), 3, ties=False), _logits(rng, len(ent), 4)
    modes, bits, *_ = oracle.route_decisions(ml, bl, [p for _, p in ent], w, Hq, d, Hkv)
    K = wl.bf16_bits(rng.standard_normal((len(ent), Hkv, d), dtype=np.float32))
    V = wl.bf16_bits(rng.standard_normal((len(ent), Hkv, d), dtype=np.float32))
    for i in range(0, len(ent), per_call):
        sl = slice(i, i + per_call)
        seqs = np.array([e[0] for e in ent[sl]], dtype=np.int32)
        pos = np.array([e[1] for e in ent[sl]], dtype=np.int32)
        pair.gpu.append_routed(0, dev(seqs, torch.int32), dev(pos, torch.int32), dev(K[sl], torch.bfloat16),
                               dev(V[sl], torch.bfloat16), dev(bl[sl], torch.float32), dev(ml[sl], torch.float32))
        assert pair.orc.append(0, seqs, pos, K[sl], V[sl], bits[sl], modes[sl]) == 0
        assert pair.gpu.status() == 0
    pair.check_regions()

    nq = 300
    qs = rng.integers(0, S, size=nq).astype(np.int32)
    qt = np.array([rng.integers(0, ctxs[s]) for s in qs], dtype=np.int32)
    qml = _logits(rng, nq, 3, ties=True)
    qmodes = oracle.route_decisions(qml, np.zeros((nq, 4), np.float32), qt, w, Hq, d, Hkv)[0]
    q = wl.bf16_bits(rng.standard_normal((nq, Hq, d), dtype=np.float32))
    out = pair.gpu.decode_attn_routed(0, dev(qs, torch.int32), dev(qt, torch.int32), dev(q, torch.bfloat16),
                                      dev(qml, torch.float32), window_scalar=w)
    st_o, ref = pair.orc.decode_attn(0, qs, qt, q, qmodes, window_scalar=w)
    assert st_o == 0 and pair.gpu.status() == 0
    check_attention(out.float().cpu().numpy().astype(np.float64), ref, qmodes)

    gm = torch.zeros(nq, dtype=torch.uint8, device="cuda")
    trr.trr_route_decisions(dev(qml, torch.float32), dev(np.zeros((nq, 4), np.float32), torch.float32),
                            modes=gm)
    torch.cuda.synchronize()  # the plain call must not read the previous call's outputs early
    plain = pair.gpu.decode_attn(0, dev(qs, torch.int32), dev(qt, torch.int32), dev(q, torch.bfloat16), gm,
                                 window_scalar=w)
    torch.cuda.synchronize()
    assert torch.equal(plain.view(torch.int16), out.view(torch.int16))
