"""Shared helpers of the GPU parity tests: build the CUDA cache and the oracle
cache from the same seeded bf16 draws, run crop + append + replay on both, and
compare.  The gate (tests/parity.py): max-abs 2e-2 and mean-abs 2e-3 against
the fp64 oracle (bf16 inputs, fp32 accumulation), and the same errors
normalised by the oracle's own size (max-abs / max|ref| <= 2e-2, mean-abs /
mean|ref| <= 1e-2), which an output of the right size but wrong values cannot
pass.  Every checked block's errors are logged in PARITY_LOG."""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
import synth
from parity import MAX_ABS, MEAN_ABS, check_parity, parity_errors, parity_failures  # noqa: F401

requires_cuda = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")

# (what, errors) of every block a test checked; written out by conftest when
# PE_PARITY_REPORT names a file.
PARITY_LOG: list = []


def dev(bits):
    return synth.bits_to_torch(bits).cuda()


def to_f64(out_gpu) -> np.ndarray:
    return out_gpu.float().cpu().numpy().astype(np.float64)


def errors(out_gpu: torch.Tensor, ref: np.ndarray):
    got = to_f64(out_gpu)
    diff = np.abs(got - ref)
    return float(diff.max()) if diff.size else 0.0, float(diff.mean()) if diff.size else 0.0, got


def assert_close(out_gpu, ref, what=""):
    """Both gates of tests/parity.py; returns (max-abs, mean-abs)."""
    e = parity_errors(to_f64(out_gpu), ref)
    PARITY_LOG.append((what, e))
    bad = parity_failures(e)
    assert not bad, f"{what}: " + "; ".join(bad)
    return e["max_abs"], e["mean_abs"]


def assert_within_rounding_bound(out_gpu, ref, vmax, what=""):
    """Element-wise bound derived from the arithmetic, for inputs outside the
    configurations' scale (e.g. very peaked logits, |O| up to max|V|):
    bf16 rounding of the output (half ulp <= 2^-8 |O|) plus bf16 rounding of
    each softmax weight before the P V product (<= 2^-8 max|V|), plus 1e-3 for
    fp32 accumulation and the exp2 approximation.  Mean-abs 2e-3 and the
    normalised gates still apply."""
    got = to_f64(out_gpu)
    e = parity_errors(got, ref)
    PARITY_LOG.append((what, e))
    bound = 2.0 ** -8 * (np.abs(ref) + vmax) + 1e-3
    excess = np.abs(got - ref) - bound
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert excess.max() <= 0, f"{what}: exceeds the rounding bound by {excess.max():.3e}"
    bad = parity_failures(e, absolute=False)
    assert not bad, f"{what}: " + "; ".join(bad)


class Pair:
    """A CUDA cache and an oracle cache driven in lockstep."""

    def __init__(self, L, hkv, d, ps, num_pages, max_seqs, max_pages, seed=1, pe_kwargs=None):
        import paper_2609_04875_gb300 as pe
        order = synth.page_permutation(seed, num_pages)
        self.gpu = pe.PagedKVCache(L, hkv, d, ps, num_pages, max_seqs, max_pages, init_free_order=order,
                                   **(pe_kwargs or {}))
        self.orc = oracle.OracleKVCache(L, hkv, d, ps, num_pages, max_seqs, max_pages, init_free_order=order)

    def seq(self):
        a, b = self.gpu.seq_create(), self.orc.seq_create()
        assert a == b
        return a

    def append(self, s, k_bits, v_bits):
        self.gpu.append_kv(s, dev(k_bits), dev(v_bits))
        self.orc.append(s, k_bits, v_bits)

    def crop(self, s, tau):
        f1 = self.gpu.crop(s, tau)
        f2 = self.orc.crop(s, tau)
        assert f1 == f2
        return f1

    def check_state(self, seqs):
        assert self.gpu.free_list() == self.orc.free_list()
        for s in seqs:
            assert self.gpu.page_table(s) == self.orc.page_table(s)
            assert self.gpu.seq_info(s) == self.orc.seq_info(s)
            tbl = self.gpu.page_table(s)
            assert self.gpu.device_page_table(s, len(tbl)) == tbl


def replay_case(L, hq, hkv, d, ps, P, S, seed, scale=None, std=1.0, split=None, slack_pages=3, options=None):
    """Original session of T = P + S tokens, crop to tau = P + 1, append the
    counterfactual suffix, replay; returns (pair, seq, gpu out [L][S][Hq][d], oracle fp64).
    `options`: further cache options (pe_set_option) set before the replay."""
    T = P + S
    npg = -(-T // ps) + slack_pages
    pair = Pair(L, hkv, d, ps, npg, 2, npg, seed=seed)
    if split is not None:
        pair.gpu.set_option("splitkv", split)
    for key, value in (options or {}).items():
        pair.gpu.set_option(key, value)
    g = synth.rng(seed, 11)
    k0 = synth.normal_bf16(g, (L, T, hkv, d), std)
    v0 = synth.normal_bf16(g, (L, T, hkv, d), std)
    kc = synth.normal_bf16(g, (L, S, hkv, d), std)
    vc = synth.normal_bf16(g, (L, S, hkv, d), std)
    qc = synth.normal_bf16(g, (L, S, hq, d), std)
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    s = pair.seq()
    pair.append(s, k0, v0)
    pair.crop(s, P + 1)
    pair.append(s, kc, vc)
    outs, refs = [], []
    for layer in range(L):
        outs.append(pair.gpu.replay_attn(s, layer, dev(qc[layer]), softmax_scale=scale))
        refs.append(oracle.replay_attention(pair.orc, s, layer, qc[layer], scale))
    torch.cuda.synchronize()
    return pair, s, outs, refs, (k0, v0, kc, vc, qc, scale)
