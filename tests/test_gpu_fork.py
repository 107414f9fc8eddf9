"""Branching from one contaminated base on the GPU (fork with copy-on-write,
metadata-only checkpoints, Restore(c*)) against the oracle: page tables,
reference counts, pool contents and replay attention of every branch."""
import ctypes
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _pool_bits(pair, L, hkv, ps, d):
    from paper_2609_04875_gb300 import binding
    kptr, vptr = ctypes.c_void_p(), ctypes.c_void_p()
    binding.lib().pe_cache_pools(pair.gpu.handle, ctypes.byref(kptr), ctypes.byref(vptr))
    n = L * pair.gpu.num_pages * hkv * ps * d

    class _Arr:
        def __init__(self, ptr):
            self.__cuda_array_interface__ = {"shape": (n,), "typestr": "<i2", "data": (ptr, False), "version": 3}

    shape = (L, pair.gpu.num_pages, hkv, ps, d)
    kb = synth.torch_to_bits(torch.as_tensor(_Arr(kptr.value), device="cuda").view(torch.bfloat16).view(shape))
    vb = synth.torch_to_bits(torch.as_tensor(_Arr(vptr.value), device="cuda").view(torch.bfloat16).view(shape))
    return kb, vb


def _check_seq(pair, s, hq, scale, g, L):
    n = pair.orc.length[s]
    nq = min(n, 70)
    q = synth.normal_bf16(g, (L, nq, hq, pair.orc.d))
    for layer in range(L):
        out = pair.gpu.replay_attn(s, layer, dev(q[layer]), softmax_scale=scale)
        assert_close(out, oracle.replay_attention(pair.orc, s, layer, q[layer], scale), f"seq {s} layer {layer}")


def _check_pools(pair, L, hkv, ps, d):
    torch.cuda.synchronize()
    kb, vb = _pool_bits(pair, L, hkv, ps, d)
    for s in pair.orc.table:
        tbl = pair.orc.page_table(s)
        for pos in range(pair.orc.length[s]):
            pg, slot = tbl[pos // ps], pos % ps
            assert np.array_equal(kb[:, pg, :, slot], pair.orc.k_pool[:, pg, :, slot]), (s, pos)
            assert np.array_equal(vb[:, pg, :, slot], pair.orc.v_pool[:, pg, :, slot]), (s, pos)


@pytest.mark.parametrize("poison", [0, 1])
def test_branches_with_copy_on_write(poison):
    L, hq, hkv, d, ps = 2, 8, 2, 128, 16
    T = 300
    npg = 80
    pair = Pair(L, hkv, d, ps, npg, 4, 40, seed=13)
    pair.gpu.set_option("debug_poison", poison)
    g = synth.rng(13, 4)
    scale = 1.0 / math.sqrt(d)
    a = pair.seq()
    pair.append(a, synth.normal_bf16(g, (L, T, hkv, d)), synth.normal_bf16(g, (L, T, hkv, d)))
    for b in (0, 96, 200, 288):
        pair.gpu.checkpoint_add(a, b)
        pair.orc.checkpoint_add(a, b)
    # branch B from the contaminated base; its partial last page (300 % 16 = 12) is shared
    b_ = pair.gpu.seq_fork(a)
    assert b_ == pair.orc.seq_fork(a)
    pair.check_state([a, b_])
    assert pair.gpu.page_refs() == list(pair.orc.refs)
    # B grows: copy-on-write of the shared partial page
    kb = synth.normal_bf16(g, (L, 50, hkv, d))
    vb = synth.normal_bf16(g, (L, 50, hkv, d))
    pair.append(b_, kb, vb)
    # A restores to the last checkpoint before tau = 250 (offset 200) and replays 100 tokens;
    # its page of tokens 192..207 is still shared with B: copy-on-write again
    off_g = pair.gpu.restore(a, 250)
    off_o = pair.orc.restore(a, 250)
    assert off_g == off_o and off_g[0] == 200
    pair.append(a, synth.normal_bf16(g, (L, 100, hkv, d)), synth.normal_bf16(g, (L, 100, hkv, d)))
    pair.check_state([a, b_])
    assert pair.gpu.page_refs() == list(pair.orc.refs)
    assert pair.gpu.checkpoints(a) == pair.orc.checkpoints[a]
    _check_pools(pair, L, hkv, ps, d)
    _check_seq(pair, a, hq, scale, g, L)
    _check_seq(pair, b_, hq, scale, g, L)
    # a third branch from B, then A is released: B and C keep their content
    c_ = pair.gpu.seq_fork(b_)
    assert c_ == pair.orc.seq_fork(b_)
    pair.gpu.crop(c_, 321)
    pair.orc.crop(c_, 321)
    pair.append(c_, synth.normal_bf16(g, (L, 7, hkv, d)), synth.normal_bf16(g, (L, 7, hkv, d)))
    pair.gpu.seq_release(a)
    pair.orc.seq_release(a)
    pair.check_state([b_, c_])
    assert pair.gpu.page_refs() == list(pair.orc.refs)
    _check_pools(pair, L, hkv, ps, d)
    _check_seq(pair, b_, hq, scale, g, L)
    _check_seq(pair, c_, hq, scale, g, L)
    assert pair.gpu.device_status() == 0
