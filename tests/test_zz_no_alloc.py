"""trr_decode_attn_static: decode attention whose per-call scratch lives in the
library's static device array, for callers that cannot allocate device memory where
they call it (for instance an engine inside a fixed, fully reserved memory budget).

Checked through the C ABI against the oracle on the same cache contents and queries (as
trr_decode_attn is, called in chunks of the cache's max_queries), on two calls in a row
(the second finds the array holding the first call's contents), with a query count
above the cache's max_queries, and a call too large for the array is refused before
anything runs."""
import numpy as np
import pytest
import torch

from paper_2607_06601_gb300 import trr, workloads as wl
from tests._parity import Pair, check_attention, dev

pytestmark = pytest.mark.gpu


def _cache_with_context(rng, S=6, n_ctx=400, Hq=8, Hkv=4, d=64):
    """A GPU cache and the oracle's, fed the same appends: n_ctx positions of S sequences,
    64 positions per call, random widths and modes."""
    pair = Pair(1, S, Hq, Hkv, d, 32, 16, 512, [S * 40] * 4, max_queries=16)
    for p0 in range(0, n_ctx, 64):
        ps = np.arange(p0, min(n_ctx, p0 + 64))
        seqs = np.repeat(np.arange(S), len(ps)).astype(np.int32)
        pos = np.tile(ps, S).astype(np.int32)
        k = wl.bf16_bits(rng.standard_normal((len(seqs), Hkv, d), dtype=np.float32))
        v = wl.bf16_bits(rng.standard_normal((len(seqs), Hkv, d), dtype=np.float32))
        order = np.lexsort((seqs, pos))  # position-major: each sequence in order
        pair.append(0, seqs[order], pos[order], k[order], v[order],
                    rng.choice([2, 4, 8, 16], size=len(seqs)).astype(np.uint8),
                    rng.choice(3, size=len(seqs)).astype(np.uint8))
    return pair


def _chunked_and_oracle(pair, seqs, ts, q, modes, wins):
    """The rows of trr_decode_attn called in chunks of max_queries (16), checked against
    the oracle, and the oracle's rows."""
    nq = seqs.shape[0]
    cache = pair.gpu
    st, ref = pair.orc.decode_attn(0, seqs.cpu().numpy(), ts.cpu().numpy(), q.view(torch.int16).cpu().numpy().view(np.uint16),
                                   modes.cpu().numpy(), wins.cpu().numpy())
    assert st == 0
    chunked = torch.empty((nq,) + tuple(q.shape[1:]), dtype=torch.bfloat16, device="cuda")
    for i0 in range(0, nq, 16):
        sl = slice(i0, min(nq, i0 + 16))
        trr.trr_decode_attn(cache.handle, 0, seqs[sl].contiguous(), ts[sl].contiguous(), q[sl].contiguous(),
                            modes[sl].contiguous(), wins[sl].contiguous(), 0, 0.0, chunked[sl])
    check_attention(chunked.float().cpu().numpy().astype(np.float64), ref, modes.cpu().numpy())
    return ref


def test_static_scratch_matches_the_oracle_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)
    rng = np.random.default_rng(77)
    S, Hq, d = 6, 8, 64
    pair = _cache_with_context(rng, S=S, Hq=Hq, d=d)
    cache = pair.gpu
    nq = 48  # more queries than the cache's max_queries (16)
    seqs = dev(rng.integers(0, S, nq).astype(np.int32), torch.int32)
    ts = dev(rng.integers(0, 400, nq).astype(np.int32), torch.int32)
    q = dev(wl.bf16_bits(rng.standard_normal((nq, Hq, d), dtype=np.float32)), torch.bfloat16)
    modes = dev(rng.choice(3, size=nq).astype(np.uint8), torch.uint8)
    wins = dev(rng.choice([1, 7, 64, 300], size=nq).astype(np.int32), torch.int32)
    ref = _chunked_and_oracle(pair, seqs, ts, q, modes, wins)
    assert np.abs(ref).max() > 0
    for _ in range(2):
        out = torch.full((nq, Hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        trr.trr_decode_attn_static(cache.handle, 0, seqs, ts, q, modes, wins, 0, 0.0, out)
        got = out.float().cpu().numpy().astype(np.float64)
        check_attention(got, ref, modes.cpu().numpy())
    assert cache.status() == 0


def test_static_scratch_refuses_calls_larger_than_the_array():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)
    rng = np.random.default_rng(78)
    cache = _cache_with_context(rng, n_ctx=64).gpu
    nq = 4000
    seqs = torch.zeros(nq, dtype=torch.int32, device="cuda")
    ts = torch.zeros(nq, dtype=torch.int32, device="cuda")
    q = torch.zeros((nq, 8, 64), dtype=torch.bfloat16, device="cuda")
    modes = torch.full((nq,), 2, dtype=torch.uint8, device="cuda")
    out = torch.zeros((nq, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(trr.TrrError) as err:
        trr.trr_decode_attn_static(cache.handle, 0, seqs, ts, q, modes, None, 0, 0.0, out)
    assert err.value.code == 2  # TRR_ERR_OUT_OF_MEMORY: nothing launched
    assert cache.launches() == 0
    assert cache.status() == 0


@pytest.mark.parametrize("Hkv", [4, 8])  # query groups of 2 (tensor cores), MHA (CUDA cores)
def test_static_scratch_above_one_launch_of_queries(Hkv):
    """About 1100 queries: the static entry point runs them as two launches, the second
    with its arrival counters offset into the array; every row matches the oracle (as do
    the rows of trr_decode_attn called in chunks of the cache's max_queries), on two
    calls in a row."""
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    torch.cuda.set_device(0)
    rng = np.random.default_rng(79 + Hkv)
    S, Hq, d = 6, 8, 64
    pair = _cache_with_context(rng, S=S, Hq=Hq, Hkv=Hkv, d=d)
    cache = pair.gpu
    nq = 1100
    seqs = dev(rng.integers(0, S, nq).astype(np.int32), torch.int32)
    ts = dev(rng.integers(0, 400, nq).astype(np.int32), torch.int32)
    q = dev(wl.bf16_bits(rng.standard_normal((nq, Hq, d), dtype=np.float32)), torch.bfloat16)
    modes = dev(rng.choice(3, size=nq).astype(np.uint8), torch.uint8)
    wins = dev(rng.choice([1, 7, 64, 300], size=nq).astype(np.int32), torch.int32)
    ref = _chunked_and_oracle(pair, seqs, ts, q, modes, wins)
    for _ in range(2):
        out = torch.full((nq, Hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        trr.trr_decode_attn_static(cache.handle, 0, seqs, ts, q, modes, wins, 0, 0.0, out)
        got = out.float().cpu().numpy().astype(np.float64)
        check_attention(got, ref, modes.cpu().numpy())
    assert cache.launches() >= 4  # clear kernel, two attention launches (and combines), status kernel
    assert cache.status() == 0
