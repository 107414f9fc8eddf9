"""Limits and degenerate inputs on the GPU: batches larger than one launch
carries (attention groups of 64 sequences, append launches of 3072 new pages,
crop launches of 256 sequences), empty calls, and a sequence filled to its
page-table capacity, all against the oracle."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def test_batch_beyond_one_launch_group():
    """70 sequences: two attention launch groups and two append launches."""
    L, hq, hkv, d, ps = 1, 8, 2, 64, 16
    n = 70
    g = synth.rng(70, 1)
    lens = [int(x) for x in g.integers(1, 300, size=n)]
    keep = [int(g.integers(0, t)) for t in lens]          # P per sequence
    npg = sum(-(-t // ps) for t in lens) + 16
    pair = Pair(L, hkv, d, ps, npg, n, 32, seed=70)
    seqs = [pair.seq() for _ in range(n)]
    for s, t in zip(seqs, lens):
        pair.append(s, synth.normal_bf16(g, (L, t, hkv, d)), synth.normal_bf16(g, (L, t, hkv, d)))
    pair.gpu.crop_batch(seqs, [p + 1 for p in keep])
    for s, p in zip(seqs, keep):
        pair.orc.crop(s, p + 1)
    S = [t - p for t, p in zip(lens, keep)]
    cu = [0] + list(np.cumsum(S))
    kc = synth.normal_bf16(g, (L, cu[-1], hkv, d))
    vc = synth.normal_bf16(g, (L, cu[-1], hkv, d))
    pair.gpu.append_kv_batch(seqs, dev(kc), dev(vc), cu)
    for i, s in enumerate(seqs):
        pair.orc.append(s, kc[:, cu[i]:cu[i + 1]], vc[:, cu[i]:cu[i + 1]])
    pair.check_state(seqs)
    q = synth.normal_bf16(g, (cu[-1], hq, d))
    for split in (0, 1):
        pair.gpu.set_option("splitkv", split)
        out = pair.gpu.replay_attn_batch(seqs, 0, dev(q), cu)
        torch.cuda.synchronize()
        for i, s in enumerate(seqs):
            ref = oracle.replay_attention(pair.orc, s, 0, q[cu[i]:cu[i + 1]], 1 / math.sqrt(d))
            assert_close(out[cu[i]:cu[i + 1]], ref, f"split={split} seq {i}")
    assert pair.gpu.device_status() == 0


def test_append_beyond_one_launch_and_full_table():
    """One append of 3800 new pages (ps = 8) spans two append launches; the
    sequence ends exactly at its page-table capacity."""
    L, hq, hkv, d, ps = 1, 4, 1, 64, 8
    pages = 3800
    T = pages * ps
    pair = Pair(L, hkv, d, ps, pages + 4, 1, pages, seed=38)
    s = pair.seq()
    g = synth.rng(38, 1)
    k = synth.normal_bf16(g, (L, T, hkv, d))
    v = synth.normal_bf16(g, (L, T, hkv, d))
    pair.append(s, k, v)
    pair.check_state([s])
    q = synth.normal_bf16(g, (40, hq, d))
    out = pair.gpu.replay_attn(s, 0, dev(q))
    assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "30k-token sequence")
    from paper_2609_04875_gb300.binding import PEError
    with pytest.raises(PEError) as e:   # one more token exceeds max_pages_per_seq
        pair.gpu.append_kv(s, dev(k[:, :1]), dev(v[:, :1]))
    assert e.value.kind == "range"


def test_crop_batch_beyond_one_launch():
    """300 sequences cropped in one call: two crop launches."""
    L, hkv, d, ps, n = 1, 1, 64, 8, 300
    pair = Pair(L, hkv, d, ps, n * 3 + 8, n, 4, seed=300)
    g = synth.rng(300, 1)
    seqs = [pair.seq() for _ in range(n)]
    for s in seqs:
        t = int(g.integers(1, 24))
        pair.append(s, synth.normal_bf16(g, (L, t, hkv, d)), synth.normal_bf16(g, (L, t, hkv, d)))
    taus = [int(g.integers(1, pair.orc.length[s] + 2)) for s in seqs]
    pair.gpu.crop_batch(seqs, taus)
    for s, t in zip(seqs, taus):
        pair.orc.crop(s, t)
    pair.check_state(seqs)


def test_empty_and_degenerate_calls():
    L, hq, hkv, d, ps = 1, 8, 8, 64, 16
    pair = Pair(L, hkv, d, ps, 8, 2, 8, seed=1)
    s = pair.seq()
    empty_kv = torch.empty((L, 0, hkv, d), dtype=torch.bfloat16, device="cuda")
    pair.gpu.append_kv(s, empty_kv, empty_kv)                       # zero tokens
    assert pair.gpu.seq_info(s) == (0, 0)
    assert pair.gpu.crop(s, 1) == []                                 # crop of an empty sequence
    g = synth.rng(1, 1)
    k, v = synth.normal_bf16(g, (L, 20, hkv, d)), synth.normal_bf16(g, (L, 20, hkv, d))
    pair.append(s, k, v)
    q0 = torch.empty((0, hq, d), dtype=torch.bfloat16, device="cuda")
    out = pair.gpu.replay_attn(s, 0, q0)                             # no queries
    assert out.shape[0] == 0
    assert pair.gpu.crop(s, 21) == [] and pair.gpu.seq_info(s) == (20, 0)   # tau = len + 1 keeps all
    pair.orc.crop(s, 21)
    t = pair.seq()
    out = pair.gpu.replay_attn_batch([s, t], 0, dev(synth.normal_bf16(g, (3, hq, d))), [0, 3, 3])
    torch.cuda.synchronize()
    q = synth.normal_bf16(g, (3, hq, d))
    out = pair.gpu.replay_attn_batch([s, t], 0, dev(q), [0, 3, 3])   # second sequence has no queries
    assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "batch with an empty range")
    pair.check_state([s, t])
    assert pair.gpu.device_status() == 0
