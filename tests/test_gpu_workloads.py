"""The five workloads at full size, in the launch configuration bench.py times
(ReplayDriver.step: one batched crop, one batched append, one batched replay
launch per layer).  Bookkeeping is compared with the oracle in full; attention
on sampled query rows (first/last rows, tile boundaries, random rows), each
computed by the oracle from the counterfactual sequence's definition (retained
prefix of the original session followed by the sanitized suffix).

Every attention block passes the absolute gate and the gate normalised by the
oracle's size (tests/parity.py), so an output of the right magnitude but the
wrong values (zeros, another page table, a dropped key split) fails.  Each
shape also runs with std-1 draws (logits of standard deviation 1 instead of
the workloads' ~0.008), where a wrong key changes the output visibly."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import assert_close, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]


def _rows(w, a, n_random, edge_tiles=4):
    g = w.num_q_heads // w.num_kv_heads
    bmq = 128 // g
    n_tiles = -(-a.S // bmq)
    rows = {0, a.S - 1}
    for t in list(range(1, min(edge_tiles, n_tiles))) + list(range(max(1, n_tiles - edge_tiles), n_tiles)):
        rows.update({t * bmq - 1, t * bmq})
    r = synth.rng(w.seed, synth.STREAM_SAMPLE, a.index)
    rows.update(int(x) for x in r.integers(0, a.S, size=n_random))
    return np.array(sorted(x for x in rows if 0 <= x < a.S), dtype=np.int64)


def _draw(w):
    """Host bf16 draws of the workload, shared by the driver and the oracle."""
    out = {}
    for i, a in enumerate(w.agents):
        k0, v0 = w.kv_original(a)
        kc, vc = w.kv_counterfactual(a)
        out[i] = (k0, v0, kc, vc, w.q_counterfactual(a))
    return out


def _check_bookkeeping(drv, steps=1):
    w = drv.w
    orc = oracle.OracleKVCache(w.num_layers, w.num_kv_heads, w.head_dim, w.page_size, w.num_pages,
                               len(w.agents), w.max_pages_per_seq, init_free_order=w.init_free_order(),
                               store_values=False)
    for a in w.agents:
        s = orc.seq_create()
        orc.append(s, n_tokens=a.T)
    for _ in range(steps):
        for s, a in enumerate(w.agents):
            orc.crop(s, a.tau)
        for s, a in enumerate(w.agents):
            orc.append(s, n_tokens=a.S)
    assert drv.cache.free_list() == orc.free_list()
    for s, a in enumerate(w.agents):
        assert drv.cache.page_table(s) == orc.page_table(s)
        assert drv.cache.seq_info(s) == (a.T, a.S)          # Corollary 1: T - tau + 1 recomputed
        tbl = drv.cache.page_table(s)
        assert drv.cache.device_page_table(s, len(tbl)) == tbl


def _check_attention(drv, inputs, agents, layers, n_random):
    """Each (agent, layer) block of sampled rows through both gates."""
    w = drv.w
    worst = (0.0, 0.0)
    for i in agents:
        a = w.agents[i]
        k0, v0, kc, vc, qc = inputs[i]
        rows = _rows(w, a, n_random)
        for layer in layers:
            keys = np.concatenate([k0[layer, : a.P], kc[layer]], axis=0)
            vals = np.concatenate([v0[layer, : a.P], vc[layer]], axis=0)
            ref = oracle.causal_attention(qc[layer], keys, vals, w.softmax_scale, rows=rows)
            got = drv.out[layer, drv.cu[i] + torch.from_numpy(rows).cuda()]
            mx, mean = assert_close(got, ref, f"{w.name} agent {i} layer {layer}")
            worst = (max(worst[0], mx), max(worst[1], mean))
    return worst


def _run(w):
    from paper_2609_04875_gb300.driver import ReplayDriver
    inputs = _draw(w)
    drv = ReplayDriver(w, inputs=inputs)
    drv.step()
    torch.cuda.synchronize()
    assert drv.cache.device_status() == 0
    return drv, inputs


def test_tiny_full():
    """Config 1 draws N(0, 1) values already (logits of standard deviation 1)."""
    w = synth.tiny()
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    a = w.agents[0]
    k0, v0, kc, vc, qc = inputs[0]
    ref = oracle.causal_attention(qc[0], np.concatenate([k0[0, : a.P], kc[0]]),
                                  np.concatenate([v0[0, : a.P], vc[0]]), w.softmax_scale)
    assert_close(drv.out[0], ref, f"{w.name} (all rows)")


def test_agent_batch():
    w = synth.agent_batch()
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=24)
    # a second step (steady state of the benchmark) gives the same output
    first = drv.out.clone()
    drv.step()
    torch.cuda.synchronize()
    assert torch.equal(first, drv.out)
    _check_bookkeeping(drv, steps=2)


def test_agent_batch_std1():
    """The 5256-CTA launch of the agent batch with logits of standard deviation 1."""
    w = synth.with_std(synth.agent_batch(), 1.0)
    drv, inputs = _run(w)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=16)


def test_decode_batch():
    """Decode after replay: one new token per agent (n_q = 1) over the full cache."""
    w = synth.decode_batch()
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=0)
    first = drv.out.clone()
    drv.step()
    torch.cuda.synchronize()
    assert torch.equal(first, drv.out)


def test_decode_batch_d64():
    """The decode batch with head dim 64: the tensor-core decode kernel's d = 64 form (O^T GEMM
    over a zero upper half), split items merged by its combine launch."""
    import copy
    import math
    w = copy.deepcopy(synth.decode_batch())
    w.head_dim, w.softmax_scale, w.name = 64, 1.0 / math.sqrt(64), "decode_batch_d64"
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=0)


def test_decode_batch_std1():
    w = synth.with_std(synth.decode_batch(), 1.0)
    drv, inputs = _run(w)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=0)


@pytest.mark.parametrize("std", [None, 1.0])
def test_short_suffix_splitkv(std):
    """32k-token prefixes, 16 queries: the split-KV launch (7 key splits) and its combine."""
    w = synth.short_suffix() if std is None else synth.with_std(synth.short_suffix(), std)
    drv, inputs = _run(w)
    split, n_splits, _ = drv.cache.last_attn_plan()
    assert split and n_splits > 1
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, [0, 7], [0], n_random=16)
    _check_attention(drv, inputs, range(1, 7), [0], n_random=2)


@pytest.mark.parametrize("std", [None, 1.0])
def test_long_suffix(std):
    """ps = 64, 16k-query suffixes over 4k prefixes, 64 q-heads on 8 kv-heads."""
    w = synth.long_suffix() if std is None else synth.with_std(synth.long_suffix(), std)
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=32)


@pytest.mark.parametrize("ratio", [0.1, 0.3, 0.5, 0.7, 0.9, 0.0])
def test_tau_sweep(ratio):
    """Every tau/T of the sweep and the full-reset comparator (ratio 0: an empty
    prefix, the whole counterfactual sequence recomputed), 32 layers."""
    w = synth.tau_sweep(ratio)
    drv, inputs = _run(w)
    _check_bookkeeping(drv)
    _check_attention(drv, inputs, [0], [0, 17, w.num_layers - 1], n_random=24)


@pytest.mark.parametrize("ratio", [0.3, 0.9])
def test_tau_sweep_std1(ratio):
    w = synth.with_std(synth.tau_sweep(ratio), 1.0)
    drv, inputs = _run(w)
    _check_attention(drv, inputs, [0], [0, 13, w.num_layers - 1], n_random=16)
