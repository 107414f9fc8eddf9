"""The tail launch of the one-work-item-per-CTA attention kernel (option
"attn_kernel" = 0): one sequence whose q-tile pairs leave the last wave of
CTAs mostly empty runs its lightest pairs in a second, split-KV launch over
every SM.  Rows of both launches against the
oracle (every row of the tail pairs, a sample of the rest), and the same rows
with the tail launch off (uniform plan) for comparison."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _case(n_q, prefix, seed, d=128, hq=32, hkv=8, ps=16):
    n = prefix + n_q
    npg = -(-n // ps) + 4
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=seed)
    pair.gpu.set_option("attn_kernel", 0)
    g = synth.rng(seed, 41)
    s = pair.seq()
    pair.append(s, synth.normal_bf16(g, (1, n, hkv, d)), synth.normal_bf16(g, (1, n, hkv, d)))
    q = synth.normal_bf16(g, (n_q, hq, d))
    return pair, s, q


@pytest.mark.parametrize("n_q,prefix,d,hq", [(1280, 4096, 128, 32), (1344, 3000, 128, 32), (5120, 2048, 64, 8)])
def test_tail_launch_matches_oracle(n_q, prefix, d, hq):
    """20 (or 21) q-tile pairs x 8 kv-heads = 160 (168) CTAs on 152 SMs: the lightest pair(s) move
    to the split-KV tail launch (d = 128 with 4 q-heads per kv-head; d = 64 with one)."""
    pair, s, q = _case(n_q, prefix, seed=n_q, d=d, hq=hq)
    scale = 1 / math.sqrt(d)
    g4 = hq // 8                                # q-heads per kv-head
    bmq = 128 // g4                             # queries per 128-row q-tile
    tail_rows = np.arange(0, 4 * bmq)           # the two lightest pairs' queries: every row
    rest = np.unique(np.concatenate([np.arange(4 * bmq, n_q, 31), [n_q - 1]]))
    rows = np.concatenate([tail_rows, rest])
    ref = oracle.replay_attention(pair.orc, s, 0, q, scale, rows=rows)
    out = pair.gpu.replay_attn(s, 0, dev(q))
    torch.cuda.synchronize()
    split, n_splits, ctas = pair.gpu.last_attn_plan()
    n_pairs = -(-(-(-n_q * g4 // 128)) // 2)
    assert split == 1 and n_splits >= 2, (split, n_splits, ctas)
    assert ctas > 152 and (ctas - 152) % (8 * n_splits) == 0, (ctas, n_splits)  # 152 whole-pair CTAs + the tail
    assert_close(out[torch.from_numpy(rows).cuda()], ref, f"tail plan n_q={n_q}")
    assert pair.gpu.device_status() == 0
    # the uniform plan (tail launch off: splitkv forced on with a fixed count) computes the same rows
    pair.gpu.set_option("splitkv", 0)
    out0 = pair.gpu.replay_attn(s, 0, dev(q))
    torch.cuda.synchronize()
    assert pair.gpu.last_attn_plan()[2] == n_pairs * 8
    assert_close(out0[torch.from_numpy(rows).cuda()], ref, f"single pass n_q={n_q}")

