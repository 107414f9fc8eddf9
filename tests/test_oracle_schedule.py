"""The replay-schedule oracle (which suffix positions are re-prefilled and
which re-decoded; lockstep rounds over agents) against a hand-derived example,
a token-level brute force, Corollary 1's count, the indep = 0 degenerate case
of Sec. 4.5, the workload's monotone decode counts, and execution on the
oracle cache matching a one-shot replay bit for bit."""
import json
import math
import os
import re

import numpy as np
import pytest

import oracle
import synth
from oracle import schedule as sched

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
POLICIES = {"selective": 0, "prefix_cache": 1}


def load_example():
    with open(os.path.join(GOLDEN, "replay_rounds_example.json")) as f:
        return json.load(f)


def random_turns(seed, n_agents, max_turns=7, max_len=6):
    """Random suffixes: up to max_turns turns of 0..max_len tokens, random kinds."""
    g = synth.rng(seed, 21)
    out = []
    for _ in range(n_agents):
        k = int(g.integers(0, max_turns + 1))
        out.append(tuple((int(g.integers(0, max_len + 1)), int(g.integers(0, 3))) for _ in range(k)))
    return out


def brute_units(turns, known):
    """Token-level restatement: label every position 'k' (known) or 'd'
    (re-decoded) and read the units off the label string with a regex."""
    labels = "".join(("k" if kind in known else "d") * n for n, kind in turns)
    return [len(m.group(0)) if m.group(0)[0] == "k" else 1 for m in re.finditer(r"k+|d", labels)]


# ---- pins (take the schedule module, so planted mistakes can be run through them)
def pin_golden(sm):
    ex = load_example()
    for name, pol in POLICIES.items():
        exp = ex[name]
        got_units = [sm.replay_units([tuple(t) for t in turns], pol) for turns in ex["agents_turns"]]
        assert got_units == exp["units"], (name, got_units)
        take = sm.replay_rounds([[tuple(t) for t in turns] for turns in ex["agents_turns"]], pol)
        assert take.tolist() == exp["take"], (name, take.tolist())
        assert [sm.decode_tokens([tuple(t) for t in turns], pol) for turns in ex["agents_turns"]] == \
            exp["decode_tokens"]


def pin_bruteforce_and_count(sm, seeds=range(20)):
    known = {0: (0, 1), 1: (0,)}
    for seed in seeds:
        agents = random_turns(seed, 5)
        for pol in (0, 1):
            take = sm.replay_rounds(agents, pol)
            for i, turns in enumerate(agents):
                units = sm.replay_units(turns, pol)
                assert units == brute_units(turns, known[pol]), (seed, pol, turns)
                assert all(u > 0 for u in units)
                S = sum(n for n, _ in turns)
                assert int(take[:, i].sum()) == S            # Corollary 1: every suffix position once
                assert units.count(1) >= sm.decode_tokens(turns, pol)
                assert take[:len(units), i].tolist() == units and not take[len(units):, i].any()
            assert take.shape[0] == max([len(sm.replay_units(t, pol)) for t in agents], default=0)


def pin_degenerate(sm, seeds=range(20)):
    """With no independent model turn, selective replay and the prefix cache coincide (Sec. 4.5)."""
    for seed in seeds:
        agents = [tuple((n, 2 if k == 1 else k) for n, k in turns) for turns in random_turns(seed, 4)]
        assert np.array_equal(sm.replay_rounds(agents, 0), sm.replay_rounds(agents, 1))


def pin_workload_monotone(sm):
    """On the turn-structured workload: the selective decode count falls as
    independent turns are added; the prefix cache's stays flat (Sec. 4.5)."""
    prev = None
    flat = None
    for x in (0.0, 1 / 3, 2 / 3, 1.0):
        w = synth.indep_split(x)
        dec = [sm.decode_tokens(a.turns, 0) for a in w.agents]
        dec_pc = [sm.decode_tokens(a.turns, 1) for a in w.agents]
        model = [sum(n for n, k in a.turns if k != synth.TURN_INPUT) for a in w.agents]
        dep = [sum(n for n, k in a.turns if k == synth.TURN_MODEL_DEP) for a in w.agents]
        assert dec == dep and dec_pc == model
        if x == 0.0:
            assert dec == dec_pc
        if prev is not None:
            assert all(a <= b for a, b in zip(dec, prev)) and sum(dec) < sum(prev)
        flat = dec_pc if flat is None else flat
        assert dec_pc == flat
        prev = dec
        for pol in (0, 1):
            take = sm.replay_rounds([a.turns for a in w.agents], pol)
            assert take.sum(axis=0).tolist() == [a.S for a in w.agents]


def _tiny_batch(seed):
    L, hq, hkv, d, ps = 2, 4, 2, 8, 4
    g = synth.rng(seed, 22)
    agents = random_turns(seed, 3, max_turns=6, max_len=5)
    prefixes = [int(g.integers(0, 9)) for _ in agents]
    S = [sum(n for n, _ in t) for t in agents]
    cu = np.concatenate([[0], np.cumsum(S)]).astype(np.int64)
    N = int(cu[-1])
    K = synth.normal_bf16(g, (L, N, hkv, d))
    V = synth.normal_bf16(g, (L, N, hkv, d))
    Q = synth.normal_bf16(g, (L, N, hq, d))
    pre = [(synth.normal_bf16(g, (L, p + 3, hkv, d)), synth.normal_bf16(g, (L, p + 3, hkv, d))) for p in prefixes]
    return dict(L=L, hq=hq, hkv=hkv, d=d, ps=ps, agents=agents, prefixes=prefixes, cu=cu, K=K, V=V, Q=Q, pre=pre)


def _cropped_cache(pkg, b):
    """Each agent holds its prefix plus 3 stale (contaminated) positions, then crops to tau = P + 1."""
    npg = sum(-(-(p + 3 + s) // b["ps"]) for p, s in zip(b["prefixes"], np.diff(b["cu"]))) + 8
    c = pkg.OracleKVCache(b["L"], b["hkv"], b["d"], b["ps"], npg, len(b["agents"]), npg)
    seqs = [c.seq_create() for _ in b["agents"]]
    for s, (k, v), p in zip(seqs, b["pre"], b["prefixes"]):
        c.append(s, k, v)
        c.crop(s, p + 1)
    return c, seqs


def pin_execution(pkg, seeds=range(6)):
    """Rounds on the oracle cache give, bit for bit, the outputs of one-shot
    append + replay of every agent's whole suffix, and the same lengths and
    recomputation counters (the route through the rounds does not matter)."""
    for seed in seeds:
        b = _tiny_batch(seed)
        scale = 1.0 / math.sqrt(b["d"])
        one, seqs1 = _cropped_cache(pkg, b)
        ref = np.zeros((b["L"], int(b["cu"][-1]), b["hq"], b["d"]))
        for i, s in enumerate(seqs1):
            lo, hi = int(b["cu"][i]), int(b["cu"][i + 1])
            one.append(s, b["K"][:, lo:hi], b["V"][:, lo:hi])
            for layer in range(b["L"]):
                if hi > lo:
                    ref[layer, lo:hi] = pkg.replay_attention(one, s, layer, b["Q"][layer, lo:hi], scale)
        for pol in (0, 1):
            c, seqs = _cropped_cache(pkg, b)
            take = pkg.schedule.replay_rounds(b["agents"], pol)
            out = pkg.execute_rounds(c, seqs, take, b["K"], b["V"], b["Q"], b["cu"], scale)
            assert np.array_equal(out, ref), (seed, pol)
            for s, s1 in zip(seqs, seqs1):
                assert c.seq_info(s) == one.seq_info(s1)
                k1, v1 = one.gather(s1, 1)
                k2, v2 = c.gather(s, 1)
                assert np.array_equal(k1, k2) and np.array_equal(v1, v2)


# ---- tests
def test_hand_derived_example():
    pin_golden(sched)


def test_units_match_token_level_brute_force_and_cover_the_suffix():
    pin_bruteforce_and_count(sched)


def test_no_independent_turn_means_identical_schedules():
    pin_degenerate(sched)


def test_workload_decode_counts():
    pin_workload_monotone(sched)


def test_rounds_on_the_oracle_cache_match_one_shot_replay():
    pin_execution(oracle)


def test_errors():
    with pytest.raises(oracle.OracleError):
        sched.replay_units([(3, 5)], 0)
    with pytest.raises(oracle.OracleError):
        sched.replay_units([(-1, 0)], 0)
    with pytest.raises(oracle.OracleError):
        sched.replay_rounds([[(1, 0)]], 7)
    assert sched.replay_rounds([], 0).shape == (0, 0)
    assert sched.replay_rounds([(), ((0, 2),)], 1).shape == (0, 2)
