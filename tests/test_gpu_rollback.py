"""Rollback on a device cache: a call whose k-th device step fails (the
library's "fail_launch_after" test hook; the step is not launched, nothing
faults) leaves the host bookkeeping unchanged, rewrites the device page-table
mirror from it, and the cache then serves later calls exactly like the
oracle: page tables, free list, device mirror, and replay attention of every
sequence (which reads K/V through the device table)."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda
from paper_2609_04875_gb300 import binding

pytestmark = [pytest.mark.gpu, requires_cuda]


def _state(pair, seqs):
    g = pair.gpu
    return (g.free_list(), g.page_refs(), {q: (g.page_table(q), g.seq_info(q)) for q in seqs})


def _mirror_ok(pair, seqs):
    for q in seqs:
        tbl = pair.gpu.page_table(q)
        assert pair.gpu.device_page_table(q, len(tbl)) == tbl, f"device mirror of sequence {q}"


def _inject(pair, seqs, call, max_k=16):
    before = _state(pair, seqs)
    for k in range(max_k):
        pair.gpu.set_option("fail_launch_after", k)
        try:
            call()
        except binding.PEError as e:
            assert e.kind == "cuda" and "injected" in str(e), str(e)
            assert _state(pair, seqs) == before, f"failure at device step {k} changed the state"
            _mirror_ok(pair, seqs)
            continue
        pair.gpu.set_option("fail_launch_after", -1)
        return k
    raise AssertionError("the call never succeeded")


def test_failed_calls_leave_cache_and_mirror_unchanged():
    L, hq, hkv, d, ps = 2, 8, 2, 128, 16
    pair = Pair(L, hkv, d, ps, 120, 6, 40, seed=17)
    g = synth.rng(17, 3)
    a = pair.seq()
    pair.append(a, synth.normal_bf16(g, (L, 300, hkv, d)), synth.normal_bf16(g, (L, 300, hkv, d)))
    b = pair.gpu.seq_fork(a)
    assert b == pair.orc.seq_fork(a)
    seqs = [a, b]
    # crop of a to 99 tokens: its partial last page stays shared with b
    assert _inject(pair, seqs, lambda: pair.gpu.crop(a, 100)) == 1
    pair.orc.crop(a, 100)
    # batched append: copy-on-write of a's last page, then one append launch
    ka, va = synth.normal_bf16(g, (L, 40, hkv, d)), synth.normal_bf16(g, (L, 40, hkv, d))
    kb, vb = synth.normal_bf16(g, (L, 25, hkv, d)), synth.normal_bf16(g, (L, 25, hkv, d))
    K, V = dev(np.concatenate([ka, kb], 1)), dev(np.concatenate([va, vb], 1))
    n = _inject(pair, seqs, lambda: pair.gpu.append_kv_batch(seqs, K, V, [0, 40, 65]))
    assert n == 2
    pair.orc.append(a, ka, va)
    pair.orc.append(b, kb, vb)
    # fork and release roll back too
    assert _inject(pair, seqs, lambda: pair.gpu.seq_fork(b)) == 1
    c = pair.orc.seq_fork(b)
    assert _inject(pair, seqs + [c], lambda: pair.gpu.seq_release(c)) == 1
    pair.orc.seq_release(c)
    pair.check_state(seqs)
    # the cache serves attention like the oracle afterwards
    scale = 1.0 / math.sqrt(d)
    for s in seqs:
        q = synth.normal_bf16(g, (L, 30, hq, d))
        for layer in range(L):
            out = pair.gpu.replay_attn(s, layer, dev(q[layer]), softmax_scale=scale)
            ref = oracle.replay_attention(pair.orc, s, layer, q[layer], scale)
            assert_close(out, ref, f"after rollbacks, seq {s} layer {layer}")
    # an attention call that fails leaves nothing behind either
    pair.gpu.set_option("splitkv", 1)
    pair.gpu.set_option("num_splits", 2)          # two key splits: an attention launch, then a combine launch
    q = dev(synth.normal_bf16(g, (30, hq, d)))
    pair.gpu.set_option("fail_launch_after", 1)   # the combine launch
    with pytest.raises(binding.PEError):
        pair.gpu.replay_attn(a, 0, q, softmax_scale=scale)
    pair.gpu.set_option("fail_launch_after", -1)
    torch.cuda.synchronize()
    assert pair.gpu.device_status() == 0
    pair.check_state(seqs)
