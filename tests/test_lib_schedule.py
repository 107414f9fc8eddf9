"""libpe's replay schedule (pe_replay_schedule) and the bookkeeping of
pe_replay_rounds on host-only caches, bit-exact against the oracle; error
paths leave the state unchanged."""
import numpy as np
import pytest

import oracle
import synth
from oracle import schedule as sched
from paper_2609_04875_gb300 import PEError, PagedKVCache, replay_schedule
from test_oracle_schedule import load_example, random_turns


def test_schedule_matches_oracle_on_random_suffixes():
    for seed in range(40):
        agents = random_turns(seed, int(synth.rng(seed, 23).integers(1, 9)), max_turns=9, max_len=12)
        for pol in (0, 1):
            take, dec = replay_schedule(agents, pol)
            ref = sched.replay_rounds(agents, pol)
            assert take.shape == ref.shape and np.array_equal(take, ref), (seed, pol)
            assert dec == sum(sched.decode_tokens(t, pol) for t in agents)


def test_schedule_hand_derived_example():
    ex = load_example()
    agents = [[tuple(t) for t in turns] for turns in ex["agents_turns"]]
    for name, pol in (("selective", 0), ("prefix_cache", 1)):
        take, dec = replay_schedule(agents, pol)
        assert take.tolist() == ex[name]["take"]
        assert dec == sum(ex[name]["decode_tokens"])


@pytest.mark.parametrize("indep", [0.0, 1 / 3, 2 / 3, 1.0])
def test_schedule_on_the_turn_workload(indep):
    w = synth.indep_split(indep)
    for pol in (0, 1):
        take, dec = replay_schedule([a.turns for a in w.agents], pol)
        assert np.array_equal(take, sched.replay_rounds([a.turns for a in w.agents], pol))
        assert take.sum(axis=0).tolist() == [a.S for a in w.agents]


def test_schedule_errors():
    from paper_2609_04875_gb300 import binding
    import ctypes
    lib = binding.lib()
    n = ctypes.c_int32()
    cu = binding._i32_array([0, 2])
    for lens, kinds, pol in (([1, 2], [0, 3], 0), ([1, -1], [0, 2], 0), ([1, 2], [0, 2], 2)):
        rc = lib.pe_replay_schedule(1, cu, binding._i32_array(lens), binding._i32_array(kinds), pol, None, 0,
                                    ctypes.byref(n), None)
        assert rc == -1
    rc = lib.pe_replay_schedule(1, binding._i32_array([1, 2]), binding._i32_array([1, 2]),
                                binding._i32_array([0, 2]), 0, None, 0, ctypes.byref(n), None)
    assert rc == -1  # cu_turns[0] != 0
    take = binding._i32_array([0] * 2)
    rc = lib.pe_replay_schedule(1, cu, binding._i32_array([1, 3]), binding._i32_array([0, 2]), 0, take, 2,
                                ctypes.byref(n), None)
    assert rc == -2 and n.value == 4  # 1 prefill unit + 3 decode units need 4 entries
    assert replay_schedule([], 0)[0].shape == (0, 0)


def _pair(seed, n_agents, ps=8, forks=False):
    g = synth.rng(seed, 24)
    agents = random_turns(seed, n_agents, max_turns=8, max_len=20)
    prefixes = [int(g.integers(0, 40)) for _ in agents]
    S = [sum(n for n, _ in t) for t in agents]
    npg = sum(-(-(p + 5 + s) // ps) for p, s in zip(prefixes, S)) * 2 + 16
    order = g.permutation(npg).astype(np.int32)
    max_pages = max(-(-(p + 5 + s) // ps) for p, s in zip(prefixes, S)) + 1
    n_seqs = 2 * n_agents
    lib = PagedKVCache(2, 2, 64, ps, npg, n_seqs, max_pages, init_free_order=order, host_only=True)
    orc = oracle.OracleKVCache(2, 2, 64, ps, npg, n_seqs, max_pages, init_free_order=order, store_values=False)
    seqs = []
    for p in prefixes:
        s = lib.seq_create()
        assert s == orc.seq_create()
        lib.append_kv(s, n_tokens=p + 5)
        orc.append(s, n_tokens=p + 5)
        seqs.append(s)
    if forks:  # replay on branches of the contaminated base: the first append copies a shared partial page
        seqs = [lib.seq_fork(s) for s in seqs]
        assert seqs == [orc.seq_fork(s) for s in range(n_agents)]
    for s, p in zip(seqs, prefixes):
        lib.crop(s, p + 1)
        orc.crop(s, p + 1)
    cu = [0] + list(np.cumsum(S).astype(int))
    return lib, orc, seqs, agents, cu


def _same_state(lib, orc, seqs):
    assert lib.free_list() == orc.free_list()
    assert lib.page_refs() == list(orc.refs)
    for s in seqs:
        assert lib.page_table(s) == orc.page_table(s)
        assert lib.seq_info(s) == orc.seq_info(s)


def _oracle_rounds(orc, seqs, take):
    for r in range(take.shape[0]):
        for i, s in enumerate(seqs):
            if take[r, i]:
                orc.append(s, n_tokens=int(take[r, i]))


@pytest.mark.parametrize("forks", [False, True])
def test_rounds_bookkeeping_matches_oracle(forks):
    for seed in range(12):
        for pol in (0, 1):
            lib, orc, seqs, agents, cu = _pair(seed, 5, forks=forks)
            take, _ = replay_schedule(agents, pol)
            lib.replay_rounds(seqs, take, cu)
            _oracle_rounds(orc, seqs, take)
            _same_state(lib, orc, seqs)
            for s, a in zip(seqs, agents):
                assert lib.seq_info(s)[1] == sum(n for n, _ in a)  # Corollary 1: T - tau + 1 recomputed
            lib.close()


def test_rounds_errors_leave_state_unchanged():
    lib, orc, seqs, agents, cu = _pair(3, 4)
    take, _ = replay_schedule(agents, 0)
    snap = (lib.free_list(), [lib.page_table(s) for s in seqs], [lib.seq_info(s) for s in seqs])

    def unchanged():
        assert snap == (lib.free_list(), [lib.page_table(s) for s in seqs], [lib.seq_info(s) for s in seqs])

    if take.size:
        bad = take.copy()
        bad[0, 0] += 1  # covers one row too many
        with pytest.raises(PEError) as e:
            lib.replay_rounds(seqs, bad, cu)
        assert e.value.kind == "invalid"
        unchanged()
    with pytest.raises(PEError) as e:
        lib.replay_rounds([seqs[0], seqs[0]] + seqs[2:], take, cu)
    assert e.value.kind == "invalid"
    unchanged()
    # more rows than the pool holds (2 + 5 pages of 6): OOM before any round runs
    small = PagedKVCache(1, 1, 64, 8, 6, 2, 64, host_only=True)
    s0, s1 = small.seq_create(), small.seq_create()
    with pytest.raises(PEError) as e:
        small.replay_rounds([s0, s1], np.array([[16, 40]], dtype=np.int32), [0, 16, 56])
    assert e.value.kind == "oom"
    assert small.free_list() == list(range(6)) and small.seq_info(s0) == (0, 0)
