"""Oracle: which suffix tokens a replay re-prefills and which it re-decodes,
and the lockstep rounds that batch many agents' replays.

TEST INFRASTRUCTURE ONLY (see the package docstring).  Written from the paper;
shares no code with the C++ library.

Sec. 4.5 (the T - tau + 1 paragraph) splits the post-target suffix by
causal dependence on the target z.  Turns whose content is the same in the
counterfactual world can be written into the cache by prefill, many positions
in one parallel pass; turns that depend on z must be generated again, one
position per pass (decode).  The two methods compared there differ only in
which model turns count as known:

  selective (B7, Alg. 1 with the indep split)   known = inputs + model turns
                                                 independent of z
  prefix-cache (B5', Sec. 4.1)                   known = inputs; every model
                                                 turn of the suffix is decoded

Both reuse the clean prefix (tau - 1 positions) and recompute the same
T - tau + 1 positions (Corollary 1); only the number of sequential passes
changes.  With no independent model turn the two coincide (Sec. 4.5).

A replay is a list of units in session order: a maximal run of consecutive
known tokens is one prefill unit; every other token is a decode unit of size
one.  Agents replay side by side in rounds: round r runs every agent's r-th
unit (an agent with fewer units idles).  ``take[r][i]`` is the number of
positions agent i appends and attends in round r.

Turn kinds: 0 input, 1 model turn independent of z, 2 model turn dependent on z.
"""
from __future__ import annotations

import numpy as np

from .kvcache import OracleError

SELECTIVE = 0
PREFIX_CACHE = 1
_KNOWN = {SELECTIVE: (0, 1), PREFIX_CACHE: (0,)}


def _known_kinds(policy):
    if policy not in _KNOWN:
        raise OracleError("invalid", f"unknown policy {policy}")
    return _KNOWN[policy]


def replay_units(turns, policy):
    """The units of one agent's suffix (turns: ((n_tokens, kind), ...)), in order."""
    known = _known_kinds(policy)
    units, run = [], 0
    for n, kind in turns:
        if kind not in (0, 1, 2):
            raise OracleError("invalid", f"unknown turn kind {kind}")
        if n < 0:
            raise OracleError("invalid", "negative turn length")
        if n == 0:
            continue                      # units are read off positions: an empty turn has none
        if kind in known:
            run += n                      # known tokens extend the current prefill run
            continue
        if run > 0:
            units.append(run)
            run = 0
        units.extend([1] * n)             # generated again, one position per pass
    if run > 0:
        units.append(run)
    return units


def decode_tokens(turns, policy):
    """Positions that must be generated again (one pass each)."""
    known = _known_kinds(policy)
    return sum(n for n, kind in turns if kind not in known)


def replay_rounds(agents_turns, policy):
    """take: int32 [rounds][agents]; round r runs every agent's r-th unit."""
    units = [replay_units(t, policy) for t in agents_turns]
    n_rounds = max((len(u) for u in units), default=0)
    take = np.zeros((n_rounds, len(units)), dtype=np.int32)
    for i, u in enumerate(units):
        take[:len(u), i] = u
    return take


def execute_rounds(cache, seqs, take, k_bits, v_bits, q_bits, cu_tok, scale, attend):
    """Runs the rounds on an oracle cache: for each round, append each active
    agent's next ``take`` positions (all layers), then attend those queries.

    k_bits, v_bits: bf16 bits [L][N][Hkv][d]; q_bits [L][N][Hq][d]; agent i's
    positions are rows cu_tok[i]:cu_tok[i+1].  attend(cache, seq, layer, q) is
    the attention routine (the package's replay_attention).  Returns fp64
    [L][N][Hq][d]."""
    L = k_bits.shape[0]
    N = int(cu_tok[-1])
    out = np.zeros((L, N, q_bits.shape[2], q_bits.shape[3]), dtype=np.float64)
    done = [0] * len(seqs)
    for r in range(take.shape[0]):
        active = [i for i in range(len(seqs)) if take[r][i] > 0]
        for i in active:
            lo = int(cu_tok[i]) + done[i]
            hi = lo + int(take[r][i])
            cache.append(seqs[i], k_bits[:, lo:hi], v_bits[:, lo:hi])
        for layer in range(L):
            for i in active:
                lo = int(cu_tok[i]) + done[i]
                hi = lo + int(take[r][i])
                out[layer, lo:hi] = attend(cache, seqs[i], layer, q_bits[layer, lo:hi], scale)
        for i in active:
            done[i] += int(take[r][i])
    for i in range(len(seqs)):
        if done[i] != int(cu_tok[i + 1]) - int(cu_tok[i]):
            raise OracleError("invalid", f"agent {i}: rounds cover {done[i]} of its positions")
    return out
