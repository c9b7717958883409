"""The bounded waits inside the attention and decode-step kernels: with a wait limit of
one nanosecond every wait that does not find its stage already in gives up, so the
call stops, lets its copies in flight land and records TRR_ERR_TIMEOUT (no fault, no
hang: the wait is a short limit that returns an error).  Reading the status resets the
per-call counters; the same cache then serves normal calls that match the oracle, and
a decode step that timed out stored nothing."""
import numpy as np
import pytest
import torch

from paper_2607_06601_gb300 import workloads as wl
from tests._parity import Pair, dev

pytestmark = pytest.mark.gpu

FULL = 2
TIMEOUT = 8


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)


def _pair(rng, d, G, P, Hq, Hkv, S=8, n=1500):
    maxctx = n + 16
    pair = Pair(1, S, Hq, Hkv, d, G, P, maxctx, [S * (maxctx // P + 2)] * 4)
    ent = [(s, p) for p in range(n) for s in range(S)]
    for i in range(0, len(ent), 1024):
        ch = ent[i:i + 1024]
        pair.append(0, [e[0] for e in ch], [e[1] for e in ch],
                    wl.bf16_bits(rng.standard_normal((len(ch), Hkv, d), dtype=np.float32)),
                    wl.bf16_bits(rng.standard_normal((len(ch), Hkv, d), dtype=np.float32)),
                    rng.choice((2, 4, 8, 16), size=len(ch)), rng.choice(3, size=len(ch), p=[0.1, 0.3, 0.6]))
    return pair


@pytest.mark.parametrize("d,G,P,Hq,Hkv", [(64, 32, 32, 8, 8), (128, 64, 16, 8, 2)])
def test_attention_wait_runs_out_then_cache_serves(d, G, P, Hq, Hkv):
    rng = np.random.default_rng(4)
    S, n = 8, 1500
    pair = _pair(rng, d, G, P, Hq, Hkv, S, n)
    q = wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32))
    seqs, ts = np.arange(S, dtype=np.int32), np.full(S, n - 1, np.int32)
    pair.gpu.set_wait_limit(1)
    pair.gpu.decode_attn(0, dev(seqs, torch.int32), dev(ts, torch.int32), dev(q, torch.bfloat16),
                         dev(np.full(S, FULL, np.uint8), torch.uint8))
    assert pair.gpu.status() == TIMEOUT
    pair.gpu.set_wait_limit(0)
    for _ in range(2):
        pair.attend(0, seqs, ts, q, [FULL] * S)


def test_decode_step_wait_runs_out_stores_nothing():
    rng = np.random.default_rng(5)
    d, G, P, Hq, Hkv, S, n = 64, 32, 32, 8, 8, 8, 1500
    pair = _pair(rng, d, G, P, Hq, Hkv, S, n)
    seqs, pos = np.arange(S, dtype=np.int32), np.full(S, n, np.int32)
    k = wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32))
    v = wl.bf16_bits(rng.standard_normal((S, Hkv, d), dtype=np.float32))
    q = wl.bf16_bits(rng.standard_normal((S, Hq, d), dtype=np.float32))
    bits = rng.choice((2, 4, 8, 16), size=S).astype(np.uint8)
    modes = np.full(S, FULL, np.uint8)
    before = {r: pair.gpu.region(r).cpu().numpy().copy() for r in ("last_pos", "ntok", "page_table", "next_page")}
    pair.gpu.set_wait_limit(1)
    pair.gpu.decode_step(0, dev(seqs, torch.int32), dev(pos, torch.int32), dev(k, torch.bfloat16),
                         dev(v, torch.bfloat16), dev(bits, torch.uint8), dev(modes, torch.uint8),
                         dev(q, torch.bfloat16))
    assert pair.gpu.status() == TIMEOUT
    for r, b in before.items():
        assert np.array_equal(pair.gpu.region(r).cpu().numpy(), b), f"{r} changed by a call that timed out"
    pair.gpu.set_wait_limit(0)
    pair.step(0, seqs, pos, k, v, bits, modes, q)
    pair.check_regions()
