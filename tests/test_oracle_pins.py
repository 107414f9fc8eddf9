"""The oracle against what the paper and mathematics fix (CPU only)."""
import pytest

import oracle
import oracle_pins as pins


def test_bruteforce_dense_masked_softmax():
    pins.pin_bruteforce(oracle, full=True)


def test_library_sdpa_at_empty_prefix():
    pytest.importorskip("torch")
    pins.pin_library(oracle)


def test_closed_forms():
    pins.pin_closed_forms(oracle)


def test_splice_theorem_exact():
    pins.pin_splice(oracle)


def test_recompute_lower_bound():
    pins.pin_corollary(oracle)


def test_bookkeeping_trace_and_invariants():
    pins.pin_bookkeeping(oracle)


def test_error_rules():
    c = oracle.OracleKVCache(1, 1, 2, 4, 4, 2, 4)
    s = c.seq_create()
    c.append(s, n_tokens=5)
    for tau, kind in ((0, "invalid"), (-3, "invalid"), (7, "range")):
        with pytest.raises(oracle.OracleError) as e:
            c.crop(s, tau)
        assert e.value.kind == kind
    with pytest.raises(oracle.OracleError) as e:
        c.crop(9, 1)
    assert e.value.kind == "invalid"
    assert c.seq_info(s) == (5, 5)
    with pytest.raises(oracle.OracleError) as e:
        c.append(s, n_tokens=12)   # 17 tokens > 4 pages * 4
    assert e.value.kind == "range"
    s2 = c.seq_create()
    c.append(s2, n_tokens=8)
    with pytest.raises(oracle.OracleError) as e:
        c.append(s2, n_tokens=1)    # pool exhausted
    assert e.value.kind == "oom"
    assert c.seq_info(s2) == (8, 8) and len(c.free) == 0


def test_fork_copy_on_write_checkpoints():
    pins.pin_fork(oracle)
