"""The provenance oracle against a brute-force transitive closure (boolean
matrix powers), a hand-derived episode and Lemma 2(i) monotonicity."""
import json
import os

import numpy as np
import pytest

from oracle.provenance import OracleProvenance, ProvError
import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load_episode():
    with open(os.path.join(GOLDEN, "provenance_episode.json")) as f:
        return json.load(f)


def build(g, arts):
    for a in arts:
        g.add(a["id"], a["type"], a["parents"], a["sources"], a["begin"], a["end"], a["turn"], a["committed"])
    return g


def random_dag(seed, n, z=9):
    return synth.provenance_dag(seed, n, z)


def brute_closure(arts, s):
    n = len(arts)
    A = np.zeros((n, n), dtype=bool)
    for a in arts:
        for p in a["parents"]:
            A[p, a["id"]] = True
    R = np.eye(n, dtype=bool) | A
    while True:
        R2 = R | ((R.astype(np.int64) @ R.astype(np.int64)) > 0)
        if (R2 == R).all():
            break
        R = R2
    return sorted(int(j) for j in np.nonzero(R[s])[0])


def test_hand_derived_episode():
    ep = load_episode()
    g = build(OracleProvenance(), ep["artifacts"])
    q = ep["query"]
    s = g.locate_source(q["z"])
    assert s == q["source"]
    clo = g.taint_closure(s)
    assert clo == q["closure"]
    assert g.first_entry(s) == q["tau"]
    assert g.committed_in(clo) == q["committed"]


@pytest.mark.parametrize("seed", range(12))
def test_closure_equals_brute_force(seed):
    arts = random_dag(seed, 60)
    g = build(OracleProvenance(), arts)
    s = g.locate_source(9)
    assert 9 in g.art[s]["sources"]
    assert not any(9 in g.art[p]["sources"] for p in g.art[s]["parents"])
    clo = g.taint_closure(s)
    assert clo == brute_closure(arts, s)
    assert g.first_entry(s) == min(arts[a]["begin"] for a in clo) + 1
    # every carrier of z lies in the closure of its source (propagation only along edges)
    assert {a["id"] for a in arts if 9 in a["sources"]} <= set(clo)


def test_closure_is_monotone_in_the_graph():
    """Lemma 2(i): execution only adds nodes and edges, so I_t(z) only grows."""
    arts = random_dag(99, 80)
    g = OracleProvenance()
    prev = set()
    for a in arts:
        build(g, [a])
        try:
            s = g.locate_source(9)
        except ProvError:
            continue
        clo = set(g.taint_closure(s))
        assert prev <= clo
        prev = clo


def test_errors():
    g = OracleProvenance()
    g.add(1)
    with pytest.raises(ProvError):
        g.add(1)
    with pytest.raises(ProvError):
        g.add(2, parents=[5])
    with pytest.raises(ProvError) as e:
        g.locate_source(3)
    assert e.value.kind == "range"
