"""The parity gate itself, on the CPU: at the workloads' own scale (GQA 32/8,
d = 128, Q/K/V ~ N(0, 1/128)) it must pass outputs that differ from the fp64
oracle only by the kernels' roundings, and fail outputs of the right size but
the wrong values.  Every wrong output here is built on the host with the
oracle (no kernel is broken): all zeros, one zeroed query row, keys and
values read through another sequence's page table or another layer, V read
through a page order other than K's, and a key split dropped from the merge.  The absolute gate alone passes
the all-zero output at this scale; the normalised gate is what catches it."""
import math

import numpy as np
import pytest

import oracle
import synth
from parity import REL_MAX, REL_MEAN, check_parity, parity_errors, parity_failures

HQ, HKV, D, PS = 32, 8, 128, 16
STD = 1.0 / math.sqrt(128)
SCALE = 1.0 / math.sqrt(D)


def _draw(seed, n_keys, n_q, layers=1):
    g = synth.rng(seed, 51)
    k = synth.normal_bf16(g, (layers, n_keys, HKV, D), STD)
    v = synth.normal_bf16(g, (layers, n_keys, HKV, D), STD)
    q = synth.normal_bf16(g, (n_q, HQ, D), STD)
    return k, v, q


def _bf16(x: np.ndarray) -> np.ndarray:
    """fp64 -> nearest bf16 value (through float32), as fp64."""
    return synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(x.astype(np.float32))).astype(np.float64)


def _kernel_like(q_bits, k_bits, v_bits, rows):
    """The exact result with the kernels' two roundings applied: every softmax
    weight exp(s - max) rounded to bf16 before the P V sum (the denominator
    keeps the unrounded weights), then the output rounded to bf16."""
    q = synth.bf16_bits_to_f32(q_bits).astype(np.float64)
    k = synth.bf16_bits_to_f32(k_bits).astype(np.float64)
    v = synth.bf16_bits_to_f32(v_bits).astype(np.float64)
    n_q, n_keys, g = q.shape[0], k.shape[0], HQ // HKV
    out = np.zeros((len(rows), HQ, D))
    for r, i in enumerate(rows):
        vis = n_keys - n_q + i + 1
        for h in range(HQ):
            s = SCALE * (k[:vis, h // g] @ q[i, h])
            p = np.exp(s - s.max())
            out[r, h] = (_bf16(p) @ v[:vis, h // g]) / p.sum()
    return _bf16(out)


@pytest.fixture(scope="module")
def case():
    P, S = 7 * 512, 16                      # a 7-split prefix, a short suffix
    k, v, q = _draw(3, P + S, S)
    rows = np.arange(S)
    ref = oracle.causal_attention(q, k[0], v[0], SCALE, rows=rows)
    return dict(P=P, S=S, k=k, v=v, q=q, rows=rows, ref=ref)


def test_passes_the_kernels_roundings(case):
    check_parity(_bf16(case["ref"]), case["ref"], "oracle rounded to bf16")
    got = _kernel_like(case["q"], case["k"][0], case["v"][0], case["rows"])
    e = check_parity(got, case["ref"], "weights and output rounded to bf16")
    # the derivation in tests/parity.py: ~2e-3 of the mean, a few 2^-9 of the largest |O|;
    # the gate leaves room above both
    assert e["rel_mean"] < 0.25 * REL_MEAN and e["rel_max"] < 0.25 * REL_MAX, e


def test_rejects_all_zero(case):
    e = parity_errors(np.zeros_like(case["ref"]), case["ref"])
    bad = parity_failures(e)
    assert bad
    # at the workloads' scale the absolute gate alone would have passed it
    assert all("/" in b for b in bad), bad


def test_rejects_one_wrong_row():
    """One query row (all heads) of 300 zeroed, as a mis-indexed tile row would
    leave it: the mean barely moves, the normalised max catches it."""
    k, v, q = _draw(6, 900, 300)
    ref = oracle.causal_attention(q, k[0], v[0], SCALE)
    got = _bf16(ref)
    got[137] = 0.0
    e = parity_errors(got, ref)
    assert e["rel_mean"] < REL_MEAN and e["rel_max"] > REL_MAX
    assert parity_failures(e)


def test_rejects_another_sequences_pages(case):
    k2, v2, _ = _draw(4, case["P"] + case["S"], case["S"])
    wrong = oracle.causal_attention(case["q"], k2[0], v2[0], SCALE, rows=case["rows"])
    assert parity_failures(parity_errors(wrong, case["ref"]))


def test_rejects_another_layer():
    k, v, q = _draw(5, 1500, 40, layers=2)
    rows = np.arange(40)
    ref = oracle.causal_attention(q, k[0], v[0], SCALE, rows=rows)
    wrong = oracle.causal_attention(q, k[1], v[1], SCALE, rows=rows)
    assert parity_failures(parity_errors(wrong, ref))


def test_rejects_v_read_in_another_page_order(case):
    """K through the right page table, V through a permuted one (pages of the
    prefix swapped in pairs): each query mixes the wrong values."""
    P, S = case["P"], case["S"]
    pages = np.arange(P // PS)
    perm = pages.reshape(-1, 2)[:, ::-1].reshape(-1)
    v = case["v"][0].copy()
    v[:P] = v[:P].reshape(P // PS, PS, HKV, D)[perm].reshape(P, HKV, D)
    wrong = oracle.causal_attention(case["q"], case["k"][0], v, SCALE, rows=case["rows"])
    assert parity_failures(parity_errors(wrong, case["ref"]))


@pytest.mark.parametrize("dropped", [0, 3, 6])
def test_rejects_a_dropped_split(case, dropped):
    """The merge of 7 key splits without split `dropped` (its 512 keys)."""
    P = case["P"]
    lo, hi = dropped * 512, (dropped + 1) * 512
    keep = np.r_[0:lo, hi:P + case["S"]]
    wrong = oracle.causal_attention(case["q"], case["k"][0][keep], case["v"][0][keep], SCALE, rows=case["rows"])
    assert parity_failures(parity_errors(wrong, case["ref"]))
