"""The persistent stream-K attention kernel (option "attn_kernel" = 2 forces
it; by default it serves the launch groups whose one-item plan would leave
SMs idle): one CTA per SM, whole (sequence, kv-head, q-tile pair) units in
lockstep rounds, then balanced stretches of the remaining (unit, key tile)
work.  Units cut between CTAs are computed in pieces that write fp32
partials; the warp that finishes a unit's last part merges them in the kernel
(its own part straight from TMEM when the others are in already).

Checked against the oracle with forced CTA counts that cut units into up to
tens of parts (pieces where one q-tile of the pair has no key tile, odd q-tile
counts, d = 64 and 128, GQA groups 1 to 16, varlen batches, page sizes 16
and 64), and bit for bit against the one-work-item-per-CTA kernel when no
unit is cut (the same tile order and arithmetic per unit)."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _one(d, hq, hkv, ps, P, S, seed):
    T = P + S
    npg = -(-T // ps) + 3
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=seed)
    pair.gpu.set_option("attn_kernel", 2)
    g = synth.rng(seed, 61)
    s = pair.seq()
    pair.append(s, synth.normal_bf16(g, (1, T, hkv, d)), synth.normal_bf16(g, (1, T, hkv, d)))
    q = synth.normal_bf16(g, (S, hq, d))
    return pair, s, q


CASES = [  # d, hq, hkv, ps, P, S
    (128, 32, 8, 16, 3000, 700),    # 6 q-tiles (3 pairs) x 8 kv-heads, ~30 key tiles each
    (128, 8, 8, 64, 1500, 300),     # g = 1: 3 q-tiles, the last pair has one q-tile
    (64, 16, 1, 16, 5000, 100),     # g = 16: 13 q-tiles, one kv-head
    (128, 64, 8, 16, 200, 1000),    # g = 8: 63 q-tiles, short prefix (causal pieces)
    (64, 4, 2, 32, 9000, 40),       # long keys, 1 pair per kv-head: deep cuts
]


@pytest.mark.parametrize("case", CASES, ids=[f"d{c[0]}_h{c[1]}x{c[2]}_ps{c[3]}_P{c[4]}_S{c[5]}" for c in CASES])
@pytest.mark.parametrize("ctas", [0, 1, 7, 152])
def test_streamk_matches_oracle(case, ctas):
    d, hq, hkv, ps, P, S = case
    pair, s, q = _one(d, hq, hkv, ps, P, S, seed=P + S + d)
    pair.gpu.set_option("attn_ctas", ctas)
    pair.gpu.set_option("splitkv", 1 if ctas else -1)   # forced: cut units wherever a boundary falls
    scale = 1 / math.sqrt(d)
    ref = oracle.replay_attention(pair.orc, s, 0, q, scale)
    out = pair.gpu.replay_attn(s, 0, dev(q), softmax_scale=scale)
    torch.cuda.synchronize()
    split, parts, n_ctas = pair.gpu.last_attn_plan()
    if ctas:
        assert n_ctas <= ctas
    if ctas == 152:
        assert split == 1 and parts >= 2, (split, parts, n_ctas)
    assert_close(out, ref, f"{case} ctas={ctas} plan=({split},{parts},{n_ctas})")
    assert pair.gpu.device_status() == 0


def test_streamk_varlen_batch_with_cuts():
    """Twelve sequences of mixed lengths in one launch, cut at every CTA boundary."""
    d, hq, hkv, ps = 128, 32, 8, 16
    g = synth.rng(5, 62)
    lens = [int(x) for x in g.integers(100, 3000, size=12)]
    nq = [int(x) for x in g.integers(1, 400, size=12)]
    npg = sum(-(-n // ps) for n in lens) + 8
    pair = Pair(1, hkv, d, ps, npg, 12, 200, seed=5)
    pair.gpu.set_option("attn_kernel", 2)
    seqs = []
    for n in lens:
        s = pair.seq()
        pair.append(s, synth.normal_bf16(g, (1, n, hkv, d)), synth.normal_bf16(g, (1, n, hkv, d)))
        seqs.append(s)
    cu = [0]
    for k in nq:
        cu.append(cu[-1] + k)
    q = synth.normal_bf16(g, (cu[-1], hq, d))
    scale = 1 / math.sqrt(d)
    for ctas, split in [(0, -1), (152, 1), (33, 1)]:
        pair.gpu.set_option("attn_ctas", ctas)
        pair.gpu.set_option("splitkv", split)
        out = pair.gpu.replay_attn_batch(seqs, 0, dev(q), cu, softmax_scale=scale)
        torch.cuda.synchronize()
        for i, s in enumerate(seqs):
            ref = oracle.replay_attention(pair.orc, s, 0, q[cu[i]:cu[i + 1]], scale)
            assert_close(out[cu[i]:cu[i + 1]], ref, f"ctas={ctas} seq {i}")
    assert pair.gpu.device_status() == 0


@pytest.mark.parametrize("d,hq,hkv,ps,P,S", [(128, 32, 8, 16, 2000, 900), (64, 8, 8, 16, 512, 128)])
def test_whole_units_bitwise_equal_one_item_kernel(d, hq, hkv, ps, P, S):
    """With cuts off, every unit is computed whole, in the one-item kernel's
    tile order and arithmetic: the outputs are identical bit for bit."""
    pair, s, q = _one(d, hq, hkv, ps, P, S, seed=7 + d)
    pair.gpu.set_option("splitkv", 0)
    Q = dev(q)
    a = pair.gpu.replay_attn(s, 0, Q)
    pair.gpu.set_option("attn_kernel", 0)
    b = pair.gpu.replay_attn(s, 0, Q)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert_close(a, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "whole units")


@pytest.mark.parametrize("ctas", [152, 40, 7])
def test_cut_unit_merge_is_deterministic(ctas):
    """Whichever warp finishes a cut unit's last part merges the parts: from
    TMEM and L2 when the other parts are in before its epilogue, else all from
    L2 (or the many-part path).  Every path forms the same values in the same
    order, so repeated launches, whose timing differs, agree bit for bit."""
    d, hq, hkv, ps, P, S = 128, 32, 8, 16, 3000, 700
    pair, s, q = _one(d, hq, hkv, ps, P, S, seed=31)
    pair.gpu.set_option("attn_ctas", ctas)
    pair.gpu.set_option("splitkv", 1)
    Q = dev(q)
    outs = [pair.gpu.replay_attn(s, 0, Q) for _ in range(8)]
    torch.cuda.synchronize()
    split, parts, n_ctas = pair.gpu.last_attn_plan()
    assert split == 1 and parts >= 2, (split, parts, n_ctas)
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
    assert_close(outs[0], oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), f"ctas={ctas}")
    assert pair.gpu.device_status() == 0


def test_plan_with_empty_stretches():
    """Whole-unit rounds can leave a CTA at or above the mean load, so its tail
    stretch is empty and its two boundaries coincide inside a cut unit (this
    batch on 9 CTAs: twice, at key tile 4 of the last unit).  Each cut is
    counted once, so the unit's part count, and the count its merge waits
    for, stay right."""
    d, hq, hkv, ps = 128, 32, 8, 16
    lens = [3216, 684, 1623, 1045, 743]
    nq = [337, 85, 233, 411, 475]
    g = synth.rng(9, 63)
    npg = sum(-(-n // ps) for n in lens) + 8
    pair = Pair(1, hkv, d, ps, npg, 5, 256, seed=9)
    pair.gpu.set_option("attn_kernel", 2)
    pair.gpu.set_option("attn_ctas", 9)
    pair.gpu.set_option("splitkv", 1)
    seqs = []
    for n in lens:
        s = pair.seq()
        pair.append(s, synth.normal_bf16(g, (1, n, hkv, d)), synth.normal_bf16(g, (1, n, hkv, d)))
        seqs.append(s)
    cu = [0]
    for k in nq:
        cu.append(cu[-1] + k)
    q = synth.normal_bf16(g, (cu[-1], hq, d))
    scale = 1 / math.sqrt(d)
    out = pair.gpu.replay_attn_batch(seqs, 0, dev(q), cu, softmax_scale=scale)
    torch.cuda.synchronize()
    split, parts, n_ctas = pair.gpu.last_attn_plan()
    assert split == 1 and n_ctas == 9, (split, parts, n_ctas)
    for i, s in enumerate(seqs):
        ref = oracle.replay_attention(pair.orc, s, 0, q[cu[i]:cu[i + 1]], scale)
        assert_close(out[cu[i]:cu[i + 1]], ref, f"seq {i}")
    assert pair.gpu.device_status() == 0
