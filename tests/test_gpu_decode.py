"""The decode kernel (sequences whose n_q x group query rows per kv-head fit in
16) against the oracle: head dims, group sizes, page sizes, ragged lengths,
every split regime (one split, forced counts, the last split holding fewer
keys than there are queries), mixed decode + prefill batches, peaked logits,
debug poison, and the split-merge counters staying consistent across calls."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, assert_within_rounding_bound, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _seq(pair, s, L, hkv, d, n, g, std=1.0):
    k = synth.normal_bf16(g, (L, n, hkv, d), std)
    v = synth.normal_bf16(g, (L, n, hkv, d), std)
    pair.append(s, k, v)
    return k, v


# (d, hq, hkv, ps, len, n_q): n_q x (hq/hkv) <= 16 in every case
CASES = [
    (128, 32, 8, 16, 1, 1),
    (128, 32, 8, 16, 63, 1),
    (128, 32, 8, 16, 64, 1),
    (128, 32, 8, 16, 65, 4),
    (128, 32, 8, 8, 4099, 1),
    (128, 32, 8, 128, 1000, 2),
    (128, 16, 16, 32, 777, 16),
    (128, 64, 4, 64, 2050, 1),
    (64, 8, 8, 16, 300, 8),
    (64, 16, 2, 8, 129, 2),
    (64, 16, 1, 128, 5000, 1),
    (64, 4, 2, 64, 70, 5),
]


@pytest.mark.parametrize("mode", [1, 2])
@pytest.mark.parametrize("d,hq,hkv,ps,n,nq", CASES)
def test_decode_matches_oracle(d, hq, hkv, ps, n, nq, mode):
    """mode 1: tcgen05 decode kernel (d = 64 and 128); mode 2: CUDA cores."""
    npg = -(-n // ps) + 2
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=n + nq)
    g = synth.rng(n, nq)
    pair.gpu.set_option("decode_kernel", mode)
    s = pair.seq()
    _seq(pair, s, 1, hkv, d, n, g)
    q = synth.normal_bf16(g, (nq, hq, d))
    ref = oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d))
    for split, ns in ((-1, 0), (0, 0), (1, 0), (1, 3), (1, 37)):
        pair.gpu.set_option("splitkv", split)
        pair.gpu.set_option("num_splits", ns)
        out = pair.gpu.replay_attn(s, 0, dev(q))
        torch.cuda.synchronize()
        assert_close(out, ref, f"splitkv={split} num_splits={ns}")
    assert pair.gpu.device_status() == 0


@pytest.mark.parametrize("mode,tile", [(1, 128), (2, 64)])
def test_last_split_shorter_than_the_queries(mode, tile):
    """n_q = 4 (16 rows) and one-tile splits of a (9 tiles + 2)-key sequence:
    the last split holds 2 keys, which the first two queries must not see."""
    d, hq, hkv, ps = 128, 16, 4, 16
    n = tile * 9 + 2
    npg = -(-n // ps) + 1
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=5)
    pair.gpu.set_option("decode_kernel", mode)
    g = synth.rng(5, 1)
    s = pair.seq()
    _seq(pair, s, 1, hkv, d, n, g)
    q = synth.normal_bf16(g, (4, hq, d))
    pair.gpu.set_option("splitkv", 1)
    pair.gpu.set_option("num_splits", 10)
    out = pair.gpu.replay_attn(s, 0, dev(q))
    torch.cuda.synchronize()
    assert pair.gpu.last_attn_plan()[1] == 10
    assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "short last split")


def test_both_kernels_in_one_batch_and_repeated_calls():
    """A batch mixing decode rows (n_q = 1) and prefill rows (n_q = 200): one
    call launches both kernels.  Repeating the call (split merge counters
    reused) gives bitwise the same output; switching the decode kernel off
    sends everything to the tensor-core kernel, still within tolerance."""
    d, hq, hkv, ps, L = 128, 32, 8, 16, 2
    lens = [3000, 200, 1, 4500, 777]
    nqs = [1, 200, 1, 1, 3]
    npg = sum(-(-n // ps) for n in lens) + 8
    pair = Pair(L, hkv, d, ps, npg, len(lens), max(-(-n // ps) for n in lens), seed=9)
    g = synth.rng(9, 2)
    seqs = [pair.seq() for _ in lens]
    for s, n in zip(seqs, lens):
        _seq(pair, s, L, hkv, d, n, g)
    cu = [0] + list(np.cumsum(nqs))
    q = synth.normal_bf16(g, (cu[-1], hq, d))
    refs = [oracle.replay_attention(pair.orc, s, 1, q[cu[i]:cu[i + 1]], 1 / math.sqrt(d)) for i, s in enumerate(seqs)]
    first = None
    for rep in range(3):
        out = pair.gpu.replay_attn_batch(seqs, 1, dev(q), cu)
        torch.cuda.synchronize()
        for i in range(len(seqs)):
            assert_close(out[cu[i]:cu[i + 1]], refs[i], f"rep {rep} seq {i}")
        if first is None:
            first = out.clone()
        else:
            assert torch.equal(first, out)
    for mode in (2, 0):
        pair.gpu.set_option("decode_kernel", mode)
        out = pair.gpu.replay_attn_batch(seqs, 1, dev(q), cu)
        torch.cuda.synchronize()
        for i in range(len(seqs)):
            assert_close(out[cu[i]:cu[i + 1]], refs[i], f"decode_kernel={mode}, seq {i}")
    assert pair.gpu.device_status() == 0


@pytest.mark.parametrize("mode,d", [(1, 128), (2, 128), (1, 64)])
@pytest.mark.parametrize("mult", [8.0, 64.0])
def test_peaked_logits(mult, mode, d):
    """Large logits move the tensor-core kernel's lazily kept row reference
    (O^T and the partial sums are rescaled in TMEM)."""
    hq, hkv, ps, n = 32, 8, 16, 2000
    npg = -(-n // ps) + 1
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=int(mult))
    pair.gpu.set_option("decode_kernel", mode)
    g = synth.rng(int(mult), 3)
    s = pair.seq()
    k, v = _seq(pair, s, 1, hkv, d, n, g)
    q = synth.normal_bf16(g, (1, hq, d), mult)
    pair.gpu.set_option("splitkv", 1)
    pair.gpu.set_option("num_splits", 4)
    out = pair.gpu.replay_attn(s, 0, dev(q))
    torch.cuda.synchronize()
    ref = oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d))
    vmax = float(np.abs(synth.bf16_bits_to_f32(v)).max())
    assert_within_rounding_bound(out, ref, vmax, f"peaked x{mult}")


@pytest.mark.parametrize("d", [64, 128])
def test_debug_poison_never_read(d):
    """Crop with debug poison (freed pages and the stale tail hold bf16 2^100),
    append one token, decode: the poisoned slots must stay masked."""
    hq, hkv, ps = 16, 4, 16
    n = 1000
    npg = -(-n // ps) + 2
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=17)
    pair.gpu.set_option("debug_poison", 1)
    g = synth.rng(17, 1)
    s = pair.seq()
    _seq(pair, s, 1, hkv, d, n, g)
    pair.crop(s, 523)                  # keeps 522 tokens: page 32 keeps 10 slots, 6 poisoned
    _seq(pair, s, 1, hkv, d, 1, g)
    q = synth.normal_bf16(g, (1, hq, d))
    for ns in (0, 3):
        pair.gpu.set_option("splitkv", 1 if ns else -1)
        pair.gpu.set_option("num_splits", ns)
        out = pair.gpu.replay_attn(s, 0, dev(q))
        torch.cuda.synchronize()
        assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), f"poison splits={ns}")


def test_decode_batch_beyond_one_launch():
    """70 sequences decoding one position each: two decode launches (64 + 6
    sequences) back to back reuse the merge tickets and the chunk counter."""
    d, hq, hkv, ps, n_seq = 128, 32, 8, 16, 70
    g = synth.rng(70, 7)
    lens = [int(x) for x in g.integers(1, 1500, size=n_seq)]
    npg = sum(-(-n // ps) for n in lens) + 8
    pair = Pair(1, hkv, d, ps, npg, n_seq, max(-(-n // ps) for n in lens), seed=70)
    seqs = [pair.seq() for _ in lens]
    for s, n in zip(seqs, lens):
        _seq(pair, s, 1, hkv, d, n, g)
    cu = list(range(n_seq + 1))
    q = synth.normal_bf16(g, (n_seq, hq, d))
    for rep in range(2):
        out = pair.gpu.replay_attn_batch(seqs, 0, dev(q), cu)
        torch.cuda.synchronize()
        for i, s in enumerate(seqs):
            assert_close(out[i:i + 1], oracle.replay_attention(pair.orc, s, 0, q[i:i + 1], 1 / math.sqrt(d)),
                         f"rep {rep} seq {i}")
    assert pair.gpu.device_status() == 0
