"""Replay with the indep split on the GPU (pe_replay_rounds): known turns
re-prefilled, the others re-decoded one position per round, many agents per
round.  Outputs against the oracle element by element (small cases) or on
sampled rows (the full turn-structured workload), and the bookkeeping of
every round bit-exact against the oracle running the same rounds."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import Pair, assert_close, dev, requires_cuda
from test_gpu_workloads import _check_attention, _draw
from test_oracle_schedule import random_turns

pytestmark = [pytest.mark.gpu, requires_cuda]


def _small_case(seed, d, policy, split=None, n_agents=5):
    L, hq, hkv, ps = 2, 8, 2, 16
    g = synth.rng(seed, 31)
    agents = random_turns(seed, n_agents, max_turns=8, max_len=40)
    agents[0] = agents[0] + ((150, 1), (3, 2), (140, 0))   # a run longer than one 32-query tile, then decode
    prefixes = [int(g.integers(0, 300)) for _ in agents]
    S = [sum(n for n, _ in t) for t in agents]
    cu = [0] + list(np.cumsum(S).astype(int))
    N = cu[-1]
    npg = sum(-(-(p + 4 + s) // ps) for p, s in zip(prefixes, S)) + 8
    max_pages = max(-(-(p + 4 + s) // ps) for p, s in zip(prefixes, S)) + 1
    pair = Pair(L, hkv, d, ps, npg, n_agents, max_pages, seed=seed)
    if split is not None:
        pair.gpu.set_option("splitkv", split)
    seqs = []
    for p in prefixes:   # original session: clean prefix + 4 contaminated positions, then crop to tau = p + 1
        s = pair.seq()
        pair.append(s, synth.normal_bf16(g, (L, p + 4, hkv, d)), synth.normal_bf16(g, (L, p + 4, hkv, d)))
        pair.crop(s, p + 1)
        seqs.append(s)
    K = synth.normal_bf16(g, (L, N, hkv, d))
    V = synth.normal_bf16(g, (L, N, hkv, d))
    Q = synth.normal_bf16(g, (L, N, hq, d))
    import paper_2609_04875_gb300 as pe
    take, dec = pe.replay_schedule(agents, policy)
    assert np.array_equal(take, oracle.schedule.replay_rounds(agents, policy))
    scale = 1.0 / math.sqrt(d)
    out = pair.gpu.replay_rounds(seqs, take, cu, dev(K), dev(V), dev(Q), softmax_scale=scale)
    ref = oracle.execute_rounds(pair.orc, seqs, take, K, V, Q, np.array(cu), scale)
    torch.cuda.synchronize()
    return pair, seqs, out, ref, take


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("policy", [0, 1])
def test_rounds_match_oracle(d, policy):
    for seed in (1, 2):
        pair, seqs, out, ref, take = _small_case(seed, d, policy)
        pair.check_state(seqs)
        for layer in range(2):
            assert_close(out[layer], ref[layer], f"d={d} policy={policy} seed={seed} layer {layer}")
        assert pair.gpu.device_status() == 0


def test_rounds_split_kv_forced():
    pair, seqs, out, ref, _ = _small_case(3, 128, 1, split=1)
    pair.check_state(seqs)
    for layer in range(2):
        assert_close(out[layer], ref[layer], f"split layer {layer}")


@pytest.mark.parametrize("indep", [2 / 3, 1.0])
def test_turn_workload_full_size(indep):
    """The turn-structured workload (16 agents, GQA 32/8, d = 128) through
    RoundsDriver.step (crop + one pe_replay_rounds call), both policies."""
    from paper_2609_04875_gb300.driver import RoundsDriver
    w = synth.indep_split(indep)
    inputs = _draw(w)
    drv = RoundsDriver(w, 0, inputs=inputs)
    outs = {}
    for policy in (0, 1):
        drv.set_policy(policy)
        drv.step()
        torch.cuda.synchronize()
        assert drv.cache.device_status() == 0
        # bookkeeping: the oracle crops and runs the same rounds from the original session
        orc = oracle.OracleKVCache(1, w.num_kv_heads, w.head_dim, w.page_size, w.num_pages, 2 * len(w.agents),
                                   w.max_pages_per_seq, init_free_order=w.init_free_order(), store_values=False)
        for a in w.agents:
            orc.append(orc.seq_create(), n_tokens=a.T)
        for pol in ([0] if policy == 0 else [0, 1]):   # the driver's cache saw the selective step first
            for s, a in enumerate(w.agents):
                orc.crop(s, a.tau)
            t = oracle.schedule.replay_rounds([a.turns for a in w.agents], pol)
            for r in range(t.shape[0]):
                for s in range(len(w.agents)):
                    if t[r, s]:
                        orc.append(s, n_tokens=int(t[r, s]))
        assert drv.cache.free_list() == orc.free_list()
        for s, a in enumerate(w.agents):
            assert drv.cache.page_table(s) == orc.page_table(s)
            assert drv.cache.seq_info(s) == (a.T, a.S)   # Corollary 1: T - tau + 1 recomputed
        _check_attention(drv, inputs, range(len(w.agents)), [0], n_random=12)
        outs[policy] = drv.out.clone()
    # the per-round public calls (used to time attention alone) compute the same rows
    drv.set_policy(0)
    per_round = drv.round_buffers()
    drv.step_per_round(per_round)
    torch.cuda.synchronize()
    done = [0] * len(drv.seqs)
    for r, (seqs, cu, _, _, _, o) in enumerate(per_round):
        j = 0
        for i in range(len(drv.seqs)):
            t = int(drv.take[r, i])
            if t:
                lo = drv.cu[i] + done[i]
                assert torch.equal(o[:, cu[j]:cu[j + 1]], outs[0][:, lo:lo + t]), (r, i)
                done[i] += t
                j += 1
