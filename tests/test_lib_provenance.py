"""libpe's provenance-graph queries (host only) against the oracle: the
hand-derived episode, random DAGs, a large graph, and error codes; then tau
feeds a crop on a host-only cache."""
import pytest

import oracle
from oracle.provenance import OracleProvenance, ProvError
import test_oracle_provenance as tp

pe = pytest.importorskip("paper_2609_04875_gb300")
from paper_2609_04875_gb300.binding import PEError  # noqa: E402


def _both(arts):
    g, o = pe.ProvenanceGraph(), OracleProvenance()
    for a in arts:
        g.add(a["id"], a["type"], a["parents"], a["sources"], a["begin"], a["end"], a["turn"], a["committed"])
        o.add(a["id"], a["type"], a["parents"], a["sources"], a["begin"], a["end"], a["turn"], a["committed"])
    return g, o


def test_episode_and_crop():
    ep = tp.load_episode()
    g, o = _both(ep["artifacts"])
    q = ep["query"]
    s = g.locate_source(q["z"])
    assert s == q["source"] == o.locate_source(q["z"])
    clo, nc = g.taint_closure(s)
    assert clo == q["closure"] and nc == q["committed"]
    tau = g.first_entry(s)
    assert tau == q["tau"]
    # the query's tau drives the crop: the clean prefix (80 tokens) survives
    c = pe.PagedKVCache(1, 1, 64, 16, 32, 1, 32, host_only=True)
    seq = c.seq_create()
    c.append_kv(seq, n_tokens=ep["artifacts"][-1]["end"])
    c.crop(seq, tau)
    assert c.seq_info(seq) == (tau - 1, 0)


@pytest.mark.parametrize("seed", range(10))
def test_random_dags_match_oracle(seed):
    arts = tp.random_dag(seed, 300)
    g, o = _both(arts)
    s = g.locate_source(9)
    assert s == o.locate_source(9)
    clo, nc = g.taint_closure(s)
    assert clo == o.taint_closure(s) and nc == o.committed_in(clo)
    assert g.first_entry(s) == o.first_entry(s)
    for other in (0, len(arts) // 2, len(arts) - 1):
        assert g.taint_closure(other)[0] == o.taint_closure(other)


def test_large_graph():
    arts = tp.random_dag(123, 5000)
    g, o = _both(arts)
    s = g.locate_source(9)
    assert g.taint_closure(s)[0] == o.taint_closure(s)


def test_errors():
    g = pe.ProvenanceGraph()
    g.add(1, token_begin=0, token_end=4)
    for fn in (lambda: g.add(1), lambda: g.add(2, parents=[9]), lambda: g.add(3, token_begin=5, token_end=2)):
        with pytest.raises(PEError) as e:
            fn()
        assert e.value.kind == "invalid"
    for fn in (lambda: g.locate_source(42), lambda: g.taint_closure(77), lambda: g.first_entry(77)):
        with pytest.raises(PEError) as e:
            fn()
        assert e.value.kind == "range"
