"""Pins for the oracle: checks that tie it to what the paper and mathematics fix,
never to itself.  Each pin takes the oracle *module* so that the mutation tests
can run the same pins against copies of the oracle with a planted mistake.

  pin_bruteforce   - a separately written dense masked softmax (numpy einsum
                     over contiguous arrays) on tiny paged crop+replay cases,
                     for every query row and for a subset of rows in reverse
  pin_library      - P = 0 (plain causal self-attention) against torch's SDPA
                     in float64, a library routine
  pin_closed_forms - one key, constant V, Q = 0, one dominant logit, and a
                     two-key case whose weights are the logistic function
  pin_splice       - Theorem 1: crop to tau-1 + replay of the sanitized suffix
                     equals the counterfactual computed from scratch, exactly
  pin_corollary    - Corollary 1: the recomputation counter is T - tau + 1, and
                     recomputing one position fewer changes the result
  pin_bookkeeping  - the hand-derived trace in tests/golden and invariants of
                     the allocation policy under random operations
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def decode(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def dense_attention(q, k, v, scale):
    """Dense masked softmax on contiguous float64 arrays (q [n_q][Hq][d],
    k/v [n][Hkv][d]); queries are the last n_q positions."""
    n_q, hq, _ = q.shape
    n_keys, hkv, _ = k.shape
    g = hq // hkv
    kr = np.repeat(k, g, axis=1)
    vr = np.repeat(v, g, axis=1)
    logits = np.einsum("qhd,khd->hqk", q, kr) * scale
    qpos = np.arange(n_keys - n_q, n_keys)
    masked = np.arange(n_keys)[None, :] > qpos[:, None]
    logits = np.where(masked[None], -np.inf, logits)
    logits = logits - logits.max(axis=-1, keepdims=True)
    w = np.exp(logits)
    w = w / w.sum(axis=-1, keepdims=True)
    return np.einsum("hqk,khd->qhd", w, vr)


def _cache(orc, L, hkv, d, ps, num_pages, seed, max_pages=None):
    order = synth.page_permutation(seed, num_pages)
    return orc.OracleKVCache(L, hkv, d, ps, num_pages, max_seqs=4,
                             max_pages_per_seq=max_pages or num_pages, init_free_order=order)


def _draw(seed, stream, shape):
    return synth.normal_bf16(synth.rng(seed, stream), shape)


# ---------------------------------------------------------------------------
def pin_bruteforce(orc, full=True):
    """Paged crop + replay vs dense masked softmax, many tiny shapes."""
    ps_list = (1, 2, 3, 16)
    heads = ((1, 1), (2, 1), (4, 2), (4, 4), (4, 1))
    dims = (1, 4, 8)
    Ts = (1, 2, 7, 16, 17, 40) if full else (7, 17)
    case = 0
    for ps in ps_list:
        for hq, hkv in heads:
            for d in dims:
                for T in Ts:
                    seed = 1000 + case
                    case += 1
                    kv = _draw(seed, 1, (2, 1, T, hkv, d))
                    kvc = _draw(seed, 2, (2, 1, T, hkv, d))
                    qc = _draw(seed, 3, (T, hq, d))
                    scale = 1.0 / math.sqrt(d)
                    taus = range(1, T + 1) if full else sorted({1, T // 2 + 1, T})
                    for tau in taus:
                        P, S = tau - 1, T - tau + 1
                        c = _cache(orc, 1, hkv, d, ps, -(-T // ps) + 3, seed)
                        s = c.seq_create()
                        c.append(s, kv[0], kv[1])
                        c.crop(s, tau)
                        c.append(s, kvc[0][:, :S], kvc[1][:, :S])
                        got = orc.replay_attention(c, s, 0, qc[:S], scale)
                        kf = np.concatenate([decode(kv[0][0, :P]), decode(kvc[0][0, :S])])
                        vf = np.concatenate([decode(kv[1][0, :P]), decode(kvc[1][0, :S])])
                        want = dense_attention(decode(qc[:S]), kf, vf, scale)
                        assert got.shape == want.shape
                        assert np.allclose(got, want, rtol=1e-12, atol=1e-12), \
                            f"brute force mismatch ps={ps} hq={hq} hkv={hkv} d={d} T={T} tau={tau}: " \
                            f"{np.max(np.abs(got - want))}"
                        if S >= 2:  # a subset of query rows, last first, against the same dense rows
                            sub = np.arange(S - 1, -1, -2)
                            got_sub = orc.replay_attention(c, s, 0, qc[:S], scale, rows=sub)
                            assert np.allclose(got_sub, want[sub], rtol=1e-12, atol=1e-12), \
                                f"row-subset mismatch ps={ps} hq={hq} hkv={hkv} d={d} T={T} tau={tau}"


def pin_library(orc):
    """P = 0: plain causal self-attention == torch SDPA (float64, is_causal)."""
    import torch
    import torch.nn.functional as F
    for (hq, hkv, d, n) in ((4, 4, 8, 33), (8, 2, 16, 50), (4, 1, 4, 7)):
        q = _draw(7, 1, (n, hq, d))
        k = _draw(7, 2, (n, hkv, d))
        v = _draw(7, 3, (n, hkv, d))
        scale = 0.37
        got = orc.causal_attention(q, k, v, scale)
        tq = torch.from_numpy(decode(q)).permute(1, 0, 2)[None]
        tk = torch.from_numpy(decode(k)).permute(1, 0, 2).repeat_interleave(hq // hkv, dim=0)[None]
        tv = torch.from_numpy(decode(v)).permute(1, 0, 2).repeat_interleave(hq // hkv, dim=0)[None]
        want = F.scaled_dot_product_attention(tq, tk, tv, is_causal=True, scale=scale)[0].permute(1, 0, 2).numpy()
        assert np.allclose(got, want, rtol=1e-12, atol=1e-12), f"SDPA mismatch {np.max(np.abs(got - want))}"


def pin_closed_forms(orc):
    bf = synth.f32_to_bf16_bits
    # one key: the output is that key's value row, exactly
    q = _draw(11, 1, (1, 2, 8))
    k = _draw(11, 2, (1, 1, 8))
    v = _draw(11, 3, (1, 1, 8))
    out = orc.causal_attention(q, k, v, 0.5)
    assert np.array_equal(out, np.broadcast_to(decode(v)[0, 0], out.shape)), "one key != V"
    # constant V rows: output equals the constant
    n = 29
    q = _draw(12, 1, (n, 4, 8))
    k = _draw(12, 2, (n, 2, 8))
    row = _draw(12, 3, (1, 2, 8))
    v = np.repeat(row, n, axis=0)
    out = orc.causal_attention(q[5:], k, v, 0.3)
    g = 2
    for h in range(4):
        assert np.allclose(out[:, h], decode(row)[0, h // g][None], rtol=1e-14, atol=1e-15), "constant V"
    # Q = 0: uniform weights, output = mean of the visible value rows
    q0 = np.zeros((7, 2, 8), np.uint16)
    v = _draw(13, 3, (n, 1, 8))
    out = orc.causal_attention(q0, _draw(13, 2, (n, 1, 8)), v, 1.0)
    vf = decode(v)
    for i in range(7):
        a = n - 7 + i
        assert np.allclose(out[i, 0], vf[: a + 1, 0].mean(axis=0), rtol=1e-13, atol=1e-14), "Q=0 mean"
    # one dominant logit: K rows one-hot, q = 30 e_t, scale 1
    d = 16
    kk = np.zeros((d, 1, d), np.float32)
    for j in range(d):
        kk[j, 0, j] = 1.0
    t = 9
    qq = np.zeros((1, 1, d), np.float32)
    qq[0, 0, t] = 30.0
    v = _draw(14, 3, (d, 1, d))
    out = orc.causal_attention(bf(qq), bf(kk), v, 1.0)
    bound = (d - 1) * math.exp(-30.0) * np.max(np.abs(decode(v))) * 2
    assert np.max(np.abs(out[0, 0] - decode(v)[t, 0])) <= bound, "dominant logit"
    # two keys, logits 1 and 0: weights are logistic(1) and logistic(-1)
    qq = np.array([[[1.0, 0.0]]], np.float32)
    kk = np.array([[[1.0, 0.0]], [[0.0, 1.0]]], np.float32)
    vv = np.array([[[1.0, 2.0]], [[3.0, -1.0]]], np.float32)
    out = orc.causal_attention(bf(qq), bf(kk), bf(vv), 1.0)
    w0 = 1.0 / (1.0 + math.exp(-1.0))
    want = np.array([w0 * 1.0 + (1 - w0) * 3.0, w0 * 2.0 + (1 - w0) * -1.0])
    assert np.allclose(out[0, 0], want, rtol=1e-14, atol=1e-15), "two-key logistic"
    # decode (one query at the last position) sees every key
    k = _draw(15, 2, (23, 1, 4))
    v = _draw(15, 3, (23, 1, 4))
    q = _draw(15, 1, (1, 1, 4))
    out = orc.causal_attention(q, k, v, 0.5)
    s = decode(k)[:, 0] @ decode(q)[0, 0] * 0.5
    w = np.exp(s - s.max())
    assert np.allclose(out[0, 0], (w[:, None] * decode(v)[:, 0]).sum(0) / w.sum(), rtol=1e-12, atol=1e-13)


def _splice_case(orc, L, hq, hkv, d, ps, T, tau, seed):
    """Returns (replayed suffix output, from-scratch counterfactual suffix output, cache, seq)."""
    P, S = tau - 1, T - tau + 1
    kv = _draw(seed, 1, (2, L, T, hkv, d))          # original session (suffix contaminated)
    kvc = _draw(seed, 2, (2, L, S, hkv, d))         # sanitized suffix K', V'
    qp = _draw(seed, 3, (L, P, hq, d))              # prefix queries (from-scratch pass only)
    qc = _draw(seed, 4, (L, S, hq, d))              # suffix queries Q'
    scale = 1.0 / math.sqrt(d)
    npg = -(-T // ps) + 2
    a = _cache(orc, L, hkv, d, ps, npg, seed)
    sa = a.seq_create()
    a.append(sa, kv[0], kv[1])
    a.crop(sa, tau)
    a.append(sa, kvc[0], kvc[1])
    rep = np.stack([orc.replay_attention(a, sa, l, qc[l], scale) for l in range(L)])
    b = _cache(orc, L, hkv, d, ps, npg, seed + 1)
    sb = b.seq_create()
    b.append(sb, np.concatenate([kv[0][:, :P], kvc[0]], axis=1), np.concatenate([kv[1][:, :P], kvc[1]], axis=1))
    full = np.stack([orc.replay_attention(b, sb, l, np.concatenate([qp[l], qc[l]], axis=0), scale)
                     for l in range(L)])
    return rep, full[:, P:], a, sa, (kv, kvc, qc, scale)


def pin_splice(orc):
    """Theorem 1 (with Lemma 1 for the base case): exact equality in fp64."""
    for (L, hq, hkv, d, ps, T) in ((2, 4, 2, 8, 4, 37), (1, 2, 1, 4, 16, 50), (1, 8, 8, 16, 3, 20)):
        for tau in sorted({1, 2, T // 3, T // 2 + 1, T}):
            rep, cf, _, _, _ = _splice_case(orc, L, hq, hkv, d, ps, T, tau, seed=500 + T + tau)
            assert np.array_equal(rep, cf), f"splice mismatch T={T} tau={tau} max={np.max(np.abs(rep - cf))}"


def pin_corollary(orc):
    """Corollary 1: recomputation = T - tau + 1, and one position fewer is wrong."""
    L, hq, hkv, d, ps, T = 1, 4, 2, 8, 4, 31
    for tau in (1, 9, 16, 31):
        S = T - tau + 1
        rep, cf, a, sa, (kv, kvc, qc, scale) = _splice_case(orc, L, hq, hkv, d, ps, T, tau, seed=900 + tau)
        length, appended = a.seq_info(sa)
        assert length == T and appended == S, f"count {appended} != T - tau + 1 = {S}"
        last_cf = cf[0, -1]
        # (i) crop one position later (keep the tainted token), recompute S - 1 positions
        b = _cache(orc, L, hkv, d, ps, -(-T // ps) + 2, 77)
        sb = b.seq_create()
        b.append(sb, kv[0], kv[1])
        b.crop(sb, tau + 1)
        b.append(sb, kvc[0][:, 1:], kvc[1][:, 1:])
        assert b.seq_info(sb) == (T, S - 1)
        out = orc.replay_attention(b, sb, 0, qc[0][-1:], scale)[0]
        assert np.max(np.abs(out - last_cf)) > 1e-9, "keeping the tainted position went unnoticed"
        # (ii) reuse one original suffix token instead of recomputing it
        j = S // 2
        k2, v2 = kvc[0].copy(), kvc[1].copy()
        k2[:, j], v2[:, j] = kv[0][:, tau - 1 + j], kv[1][:, tau - 1 + j]
        c = _cache(orc, L, hkv, d, ps, -(-T // ps) + 2, 78)
        sc = c.seq_create()
        c.append(sc, kv[0], kv[1])
        c.crop(sc, tau)
        c.append(sc, k2, v2)
        out = orc.replay_attention(c, sc, 0, qc[0][-1:], scale)[0]
        assert np.max(np.abs(out - last_cf)) > 1e-9, "reusing an original suffix token went unnoticed"


# ---------------------------------------------------------------------------
def run_trace(orc, trace):
    """Replays the golden bookkeeping trace on an oracle cache."""
    cfg = trace["config"]
    c = orc.OracleKVCache(cfg["num_layers"], cfg["num_kv_heads"], cfg["head_dim"], cfg["page_size"],
                          cfg["num_pages"], cfg["max_seqs"], cfg["max_pages_per_seq"],
                          init_free_order=cfg["init_free_order"])
    hkv, d = cfg["num_kv_heads"], cfg["head_dim"]
    for idx, st in enumerate(trace["steps"]):
        op = st["op"]
        try:
            if op == "create":
                got = c.seq_create()
                assert got == st["expect_seq"], f"step {idx}: seq {got}"
                continue
            if op == "append":
                n = st["n"]
                base = c.length[st["seq"]]
                code = (1000 * idx + base + np.arange(n)).astype(np.uint16)
                kb = np.broadcast_to(code[None, :, None, None], (1, n, hkv, d)).copy()
                c.append(st["seq"], kb, kb ^ np.uint16(0x4000))
            elif op == "crop":
                freed = c.crop(st["seq"], st["tau"])
                assert freed == st["expect_freed"], f"step {idx}: freed {freed}"
            elif op == "release":
                freed = c.seq_release(st["seq"])
                assert freed == st["expect_freed"], f"step {idx}: freed {freed}"
                assert c.free_list() == st["expect_free"], f"step {idx}: free {c.free_list()}"
                continue
        except orc.OracleError as e:
            assert st.get("expect_error") == e.kind, f"step {idx}: unexpected {e.kind}"
            continue
        assert "expect_error" not in st, f"step {idx}: expected {st.get('expect_error')}"
        if "expect" in st:
            ex = st["expect"]
            s = st["seq"]
            assert c.page_table(s) == ex["table"], f"step {idx}: table {c.page_table(s)}"
            assert c.seq_info(s) == (ex["len"], ex["appended"]), f"step {idx}: info {c.seq_info(s)}"
            assert c.free_list() == ex["free"], f"step {idx}: free {c.free_list()}"
        for tok, page, slot in st.get("slots", []):
            assert np.all(c.k_pool[0, page, :, slot, :] == 1000 * idx + tok), f"step {idx}: slot of {tok}"
            assert np.all(c.v_pool[0, page, :, slot, :] == (1000 * idx + tok) ^ 0x4000)
    return c


def load_trace():
    with open(os.path.join(GOLDEN, "bookkeeping_trace.json")) as f:
        return json.load(f)


def check_invariants(c, num_pages):
    used = [p for s in c.table for p in c.table[s]]
    assert len(used) + len(c.free) == num_pages, "pages lost or duplicated"
    assert len(set(used) | set(c.free)) == num_pages, "a page is in two places"
    for s in c.table:
        assert len(c.table[s]) == c.pages_for(c.length[s]), "table size != ceil(len / ps)"


def pin_bookkeeping(orc, n_ops=400):
    run_trace(orc, load_trace())
    g = synth.rng(4242, 0)
    ps, num_pages = 4, 40
    c = orc.OracleKVCache(1, 1, 1, ps, num_pages, 4, 30, init_free_order=synth.page_permutation(4242, num_pages))
    seqs = [c.seq_create() for _ in range(3)]
    for _ in range(n_ops):
        s = seqs[int(g.integers(0, len(seqs)))]
        n = c.length[s]
        if g.random() < 0.5:
            tau = int(g.integers(1, n + 2))
            before = list(c.table[s])
            keep = -(-(tau - 1) // ps)
            freed = c.crop(s, tau)
            assert freed == before[keep:], "freed set != table[ceil(L'/ps):]"
            # re-append of the same count restores the identical page table
            try:
                c.append(s, n_tokens=n - (tau - 1))
                assert c.table[s] == before, "crop + re-append did not restore the table"
                c.crop(s, tau)
            except orc.OracleError:
                pass
        else:
            try:
                c.append(s, n_tokens=int(g.integers(0, 12)))
            except orc.OracleError:
                pass
        check_invariants(c, num_pages)


# ---------------------------------------------------------------------------
def load_fork_trace():
    with open(os.path.join(GOLDEN, "fork_trace.json")) as f:
        return json.load(f)


def run_fork_trace(orc, trace):
    """Replays the hand-derived fork / copy-on-write / checkpoint trace."""
    cfg = trace["config"]
    c = orc.OracleKVCache(cfg["num_layers"], cfg["num_kv_heads"], cfg["head_dim"], cfg["page_size"],
                          cfg["num_pages"], cfg["max_seqs"], cfg["max_pages_per_seq"],
                          init_free_order=cfg["init_free_order"])
    hkv, d = cfg["num_kv_heads"], cfg["head_dim"]
    codes = {}  # seq -> per-token value code currently expected at that position
    for idx, st in enumerate(trace["steps"]):
        op, seq = st["op"], st.get("seq")
        try:
            if op == "create":
                s = c.seq_create()
                assert s == st["expect_seq"], f"step {idx}"
                codes[s] = []
                continue
            if op == "append":
                n = st["n"]
                base = c.length[seq]
                code = (1000 * idx + base + np.arange(n)).astype(np.uint16)
                kb = np.broadcast_to(code[None, :, None, None], (1, n, hkv, d)).copy()
                c.append(seq, kb, kb ^ np.uint16(0x4000))
                codes[seq] = codes[seq][:base] + [int(x) for x in code]
            elif op == "checkpoint":
                for b in st["offsets"]:
                    c.checkpoint_add(seq, b)
                continue
            elif op == "fork":
                s = c.seq_fork(seq)
                assert s == st["expect_seq"], f"step {idx}"
                codes[s] = list(codes[seq])
            elif op == "crop":
                freed = c.crop(seq, st["tau"])
                assert freed == st["expect_freed"], f"step {idx}: freed {freed}"
                codes[seq] = codes[seq][: st["tau"] - 1]
            elif op == "restore":
                b, freed = c.restore(seq, st["tau"])
                assert b == st["expect_offset"], f"step {idx}: offset {b}"
                assert freed == st["expect_freed"], f"step {idx}: freed {freed}"
                codes[seq] = codes[seq][:b]
            elif op == "release":
                freed = c.seq_release(seq)
                assert freed == st["expect_freed"], f"step {idx}: freed {freed}"
                assert c.free_list() == st["expect_free"], f"step {idx}"
                del codes[seq]
                continue
        except orc.OracleError as e:
            assert st.get("expect_error") == e.kind, f"step {idx}: unexpected {e.kind}"
            continue
        assert "expect_error" not in st, f"step {idx}"
        ex = st.get("expect", {})
        s = ex.get("seq", seq)
        if "table" in ex:
            assert c.page_table(s) == ex["table"], f"step {idx}: table {c.page_table(s)}"
        if "len" in ex:
            assert c.length[s] == ex["len"], f"step {idx}"
        if "free" in ex:
            assert c.free_list() == ex["free"], f"step {idx}: free {c.free_list()}"
        for pg, r in ex.get("refs", {}).items():
            assert c.refs[int(pg)] == r, f"step {idx}: refs[{pg}] = {c.refs[int(pg)]}"
        if "checkpoints" in ex:
            assert c.checkpoints[s] == ex["checkpoints"], f"step {idx}"
        for tok, page, slot, _ in st.get("slots", []):
            assert c.page_table(seq)[tok // cfg["page_size"]] == page, f"step {idx}: token {tok}"
            assert np.all(c.k_pool[0, page, :, slot, :] == codes[seq][tok]), f"step {idx}: slot of {tok}"
        for q, cq in codes.items():   # every branch still reads its own tokens
            k, _ = c.gather(q, 0)
            assert np.array_equal(k[:, 0, 0], np.array(cq, dtype=np.uint16)), f"step {idx}: seq {q} content"
    return c


def check_ref_invariants(c, num_pages):
    counts = [0] * num_pages
    for s in c.table:
        for p in c.table[s]:
            counts[p] += 1
    assert counts == list(c.refs), "reference counts != table occurrences"
    assert sorted(c.free) == [p for p in range(num_pages) if counts[p] == 0], "free list != unreferenced pages"
    for s in c.table:
        assert len(c.table[s]) == c.pages_for(c.length[s]), "table size != ceil(len / ps)"


def pin_fork(orc, n_ops=400):
    run_fork_trace(orc, load_fork_trace())
    g = synth.rng(5151, 0)
    ps, num_pages, L, hkv, d = 4, 48, 1, 1, 1
    c = orc.OracleKVCache(L, hkv, d, ps, num_pages, 6, 40, init_free_order=synth.page_permutation(5151, num_pages))
    codes = {}
    s0 = c.seq_create()
    codes[s0] = []
    step = 0
    for _ in range(n_ops):
        step += 1
        live = list(c.table)
        s = live[int(g.integers(0, len(live)))]
        r = g.random()
        try:
            if r < 0.2 and len(live) < 6:
                t = c.seq_fork(s)
                codes[t] = list(codes[s])
            elif r < 0.45:
                tau = int(g.integers(1, c.length[s] + 2))
                c.crop(s, tau)
                codes[s] = codes[s][: tau - 1]
            elif r < 0.55:
                c.checkpoint_add(s, int(g.integers(0, c.length[s] + 1)))
            elif r < 0.62 and c.checkpoints[s]:
                b, _ = c.restore(s, int(g.integers(1, c.length[s] + 2)))
                codes[s] = codes[s][:b]
            elif r < 0.68 and len(live) > 1:
                c.seq_release(s)
                del codes[s]
            else:
                n = int(g.integers(0, 9))
                base = c.length[s]
                code = ((step * 37 + base + np.arange(n)) % 60000).astype(np.uint16)
                c.append(s, code[None, :, None, None].copy(), code[None, :, None, None].copy())
                codes[s] = codes[s][:base] + [int(x) for x in code]
        except orc.OracleError:
            pass
        check_ref_invariants(c, num_pages)
        for q in c.table:
            k, v = c.gather(q, 0)
            assert np.array_equal(k[:, 0, 0], np.array(codes[q], dtype=np.uint16)), "a branch lost its content"
