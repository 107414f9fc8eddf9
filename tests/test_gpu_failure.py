"""Failure detection without a GPU fault: a kernel's bounded wait on a barrier
that nothing arrives at gives up after its limit, records status 1 in the
cache's device status word and returns; the context stays usable."""
import math

import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def test_bounded_wait_reports_and_context_survives():
    d, hq, hkv, ps, T = 128, 8, 2, 16, 300
    pair = Pair(1, hkv, d, ps, 32, 1, 32, seed=5)
    s = pair.seq()
    g = synth.rng(5, 1)
    pair.append(s, synth.normal_bf16(g, (1, T, hkv, d)), synth.normal_bf16(g, (1, T, hkv, d)))
    assert pair.gpu.device_status() == 0
    pair.gpu.selftest_bounded_wait(50_000_000)        # 50 ms, nothing ever arrives
    assert pair.gpu.device_status(clear=True) == 1
    assert pair.gpu.device_status() == 0               # cleared
    q = synth.normal_bf16(g, (40, hq, d))
    out = pair.gpu.replay_attn(s, 0, dev(q))
    torch.cuda.synchronize()
    assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "after timeout")
    assert pair.gpu.device_status() == 0
