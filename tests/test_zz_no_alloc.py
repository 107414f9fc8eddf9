"""pe_replay_attn_static_scratch: the replay-attention entry point for callers
that cannot allocate device memory when they run attention (stream host
callbacks, latency-critical loops where cudaMalloc may synchronise the device,
processes whose device memory belongs to their own allocator).  Its split-KV
partials live in a fixed device array inside the library instead of the
cache's workspace.

Checked through the C-ABI against the existing entry point (pe_replay_attn on
its split-KV path) on two calls in a row with different queries, so contents
left in the shared array by the first call cannot leak into the second.
Collected last on purpose: a run stopping at its first failure has already run
every other test.  Works alone in a fresh process (the first call performs the
per-device address lookup) and after the other tests."""
import ctypes
import math

import numpy as np
import pytest
import torch

import synth
from gpu_common import MAX_ABS, MEAN_ABS, dev, errors, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _cache(P, S, hq=32, hkv=8, d=128, ps=16, seed=314):
    import paper_2609_04875_gb300 as pe
    T = P + S
    npg = -(-T // ps) + 2
    c = pe.PagedKVCache(1, hkv, d, ps, npg, 1, npg, init_free_order=synth.page_permutation(seed, npg))
    s = c.seq_create()
    g = synth.rng(seed, 1)
    c.append_kv(s, dev(synth.normal_bf16(g, (1, T, hkv, d))), dev(synth.normal_bf16(g, (1, T, hkv, d))))
    return c, s, g


def test_static_scratch_matches_existing_entry_point_twice():
    from paper_2609_04875_gb300 import binding
    lib = binding.lib()
    hq, hkv, d = 32, 8, 128
    c, s, g = _cache(P=6000, S=16, hq=hq, hkv=hkv, d=d)
    c.set_option("splitkv", 1)   # the existing entry point on its split-KV (scratch-using) path
    scale = 1.0 / math.sqrt(d)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        q = dev(synth.normal_bf16(g, (16, hq, d)))
        want = c.replay_attn(s, 0, q, softmax_scale=scale)
        got = torch.full_like(q, float("nan"))
        rc = lib.pe_replay_attn_static_scratch(c.handle, s, 0, ctypes.c_void_p(q.data_ptr()),
                                               ctypes.c_void_p(got.data_ptr()), q.shape[0], hq, scale, stream)
        assert rc == 0, lib.pe_last_error().decode()
        torch.cuda.synchronize()
        mx, mean, arr = errors(got, want.float().cpu().numpy().astype(np.float64))
        assert np.all(np.isfinite(arr)), f"call {call}: non-finite output"
        assert mx <= MAX_ABS and mean <= MEAN_ABS, f"call {call}: max-abs {mx:.3e} mean-abs {mean:.3e}"
    assert c.device_status() == 0


def test_static_scratch_rejects_oversized_call():
    from paper_2609_04875_gb300 import binding
    hq, hkv, d = 32, 8, 128
    c, s, g = _cache(P=100, S=2000, hq=hq, hkv=hkv, d=d)
    q = dev(synth.normal_bf16(g, (2000, hq, d)))   # 63 q-tiles x 8 heads x 128 rows x 516 B > 16 MiB
    with pytest.raises(binding.PEError) as e:
        c.replay_attn_static_scratch(s, 0, q)
    assert e.value.kind == "range" and "static scratch" in str(e.value)
