"""pe_replay_attn_static_scratch: the replay-attention entry point for callers
that cannot allocate device memory when they run attention (stream host
callbacks, latency-critical loops where cudaMalloc may synchronise the device,
processes whose device memory belongs to their own allocator).  Its split-KV
partials live in a fixed device array inside the library instead of the
cache's workspace.

Checked through the C-ABI on two calls in a row with different queries, so
contents left in the shared array by the first call cannot leak into the
second: each call's output against the fp64 oracle (both parity gates) and
against the existing entry point (pe_replay_attn on its split-KV path).
Collected last on purpose: a run stopping at its first failure has already run
every other test.  Works alone in a fresh process (the first call performs the
per-device address lookup) and after the other tests."""
import ctypes
import math

import pytest
import torch

import oracle
import synth
from gpu_common import assert_close, dev, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _cache(P, S, hq=32, hkv=8, d=128, ps=16, seed=314):
    import paper_2609_04875_gb300 as pe
    T = P + S
    npg = -(-T // ps) + 2
    c = pe.PagedKVCache(1, hkv, d, ps, npg, 1, npg, init_free_order=synth.page_permutation(seed, npg))
    s = c.seq_create()
    g = synth.rng(seed, 1)
    k, v = synth.normal_bf16(g, (1, T, hkv, d)), synth.normal_bf16(g, (1, T, hkv, d))
    c.append_kv(s, dev(k), dev(v))
    return c, s, g, k[0], v[0]


def test_static_scratch_matches_oracle_and_existing_entry_point_twice():
    from paper_2609_04875_gb300 import binding
    lib = binding.lib()
    hq, hkv, d = 32, 8, 128
    c, s, g, k, v = _cache(P=6000, S=16, hq=hq, hkv=hkv, d=d)
    c.set_option("splitkv", 1)   # the existing entry point on its split-KV (scratch-using) path
    scale = 1.0 / math.sqrt(d)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        q_bits = synth.normal_bf16(g, (16, hq, d))
        q = dev(q_bits)
        got = torch.full_like(q, float("nan"))
        rc = lib.pe_replay_attn_static_scratch(c.handle, s, 0, ctypes.c_void_p(q.data_ptr()),
                                               ctypes.c_void_p(got.data_ptr()), q.shape[0], hq, scale, stream)
        assert rc == 0, lib.pe_last_error().decode()
        torch.cuda.synchronize()
        # the queries are the sequence's last 16 positions: the oracle's bottom-right causal attention
        ref = oracle.causal_attention(q_bits, k, v, scale)
        assert_close(got, ref, f"static scratch, call {call}, vs oracle")
        want = c.replay_attn(s, 0, q, softmax_scale=scale)
        torch.cuda.synchronize()
        assert_close(got, want.double().cpu().numpy(), f"static scratch, call {call}, vs pe_replay_attn")
    assert c.device_status() == 0


def test_static_scratch_rejects_oversized_call():
    from paper_2609_04875_gb300 import binding
    hq, hkv, d = 32, 8, 128
    c, s, g, _, _ = _cache(P=100, S=2000, hq=hq, hkv=hkv, d=d)
    q = dev(synth.normal_bf16(g, (2000, hq, d)))   # 63 q-tiles x 8 heads x 128 rows x 516 B > 16 MiB
    with pytest.raises(binding.PEError) as e:
        c.replay_attn_static_scratch(s, 0, q)
    assert e.value.kind == "range" and "static scratch" in str(e.value)
