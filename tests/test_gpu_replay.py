"""CUDA path vs the fp64 oracle through the C-ABI: crop, append and replay
attention on small cases that span several tiles and ragged tails, plus the
paper's splice theorem and recomputation bound checked on the GPU output."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_common import MAX_ABS, Pair, assert_close, assert_within_rounding_bound, dev, replay_case, requires_cuda

pytestmark = [pytest.mark.gpu, requires_cuda]

# (d, Hq, Hkv, ps, P, S): multi-tile, ragged tails, len not a multiple of ps,
# P = 0 (plain causal), S = 1 (decode), g from 1 to 128, every page size.
CASES = [
    (64, 8, 8, 16, 512, 128),
    (128, 32, 8, 16, 300, 77),
    (128, 64, 8, 64, 200, 333),
    (128, 8, 8, 8, 0, 257),
    (64, 4, 1, 32, 1000, 1),
    (128, 16, 2, 128, 129, 130),
    (128, 2, 2, 16, 5, 3),
    (64, 128, 1, 16, 37, 9),
    (128, 32, 8, 16, 1, 1),
    (64, 16, 4, 8, 640, 250),
]


@pytest.mark.parametrize("case", CASES, ids=[f"d{c[0]}_h{c[1]}x{c[2]}_ps{c[3]}_P{c[4]}_S{c[5]}" for c in CASES])
def test_replay_matches_oracle(case):
    d, hq, hkv, ps, P, S = case
    pair, s, outs, refs, _ = replay_case(1, hq, hkv, d, ps, P, S, seed=hash(case) % 1000)
    assert_close(outs[0], refs[0], f"{case}")
    pair.check_state([s])
    assert pair.gpu.device_status() == 0


@pytest.mark.parametrize("scale_mult", [4.0, 8.0, 64.0])
def test_peaked_logits_exercise_rescaling(scale_mult):
    """Logit std 4 to 64: running maxima jump between key tiles; at 64 later
    tiles exceed the first tile's max by far more than 2^64 in weight, so the
    reference moves and O in TMEM is rescaled.  The output is then close to
    single value rows (|O| up to max|V|): at x4 the stated 2e-2 gate still
    holds and is applied; beyond it the check uses the derived rounding bound
    (both with the normalised gates)."""
    d = 128
    pair, s, outs, refs, inputs = replay_case(1, 32, 8, d, 16, 700, 300, seed=5, scale=scale_mult / math.sqrt(d),
                                              split=0)
    if scale_mult <= 4.0:
        assert_close(outs[0], refs[0], f"peaked x{scale_mult}")
        return
    vmax = float(np.abs(synth.bf16_bits_to_f32(np.concatenate([inputs[1], inputs[3]], 1))).max())
    assert_within_rounding_bound(outs[0], refs[0], vmax, f"peaked x{scale_mult}")


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("split", [0, 1])
@pytest.mark.parametrize("jump", [128, 192])
def test_reference_moves_on_large_jump(split, jump, d):
    """Keys from `jump` on are scaled by 16 (exact in bf16), so for nearly
    every row a later tile's logits exceed the first tile's max by far more
    than 64 in log2 units: the row's reference must move and O be rescaled.
    At 128 the jump starts a key tile; at 192 it falls in the middle of one,
    so that tile mixes weights near the old reference with weights far above
    it.  At d = 64 P has its own TMEM columns and the next tile's S GEMM runs
    during the softmax: the rescale must still see this tile's S intact."""
    hq, hkv, ps, P, S = 32, 8, 16, 600, 100
    T = P + S
    npg = -(-T // ps) + 3
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=61)
    if split:
        pair.gpu.set_option("splitkv", 1)
    g = synth.rng(61, 1)
    f = synth.bf16_bits_to_f32
    k0 = f(synth.normal_bf16(g, (1, T, hkv, d)))
    k0[:, jump:] *= 16.0
    k0 = synth.f32_to_bf16_bits(k0)
    v0 = synth.normal_bf16(g, (1, T, hkv, d))
    q = synth.normal_bf16(g, (S, hq, d))
    s = pair.seq()
    pair.append(s, k0, v0)
    scale = 4.0 / math.sqrt(d)
    out = pair.gpu.replay_attn(s, 0, dev(q), softmax_scale=scale)
    ref = oracle.replay_attention(pair.orc, s, 0, q, scale)
    vmax = float(np.abs(f(v0)).max())
    assert_within_rounding_bound(out, ref, vmax, f"large jump at {jump} split={split}")


def test_multilayer_and_pool_contents():
    L, hq, hkv, d, ps = 3, 8, 2, 128, 16
    pair, s, outs, refs, _ = replay_case(L, hq, hkv, d, ps, 100, 61, seed=3)
    for layer in range(L):
        assert_close(outs[layer], refs[layer], f"layer {layer}")
    # pool contents: every valid slot holds the oracle's bits
    import ctypes
    from paper_2609_04875_gb300 import binding
    kptr, vptr = ctypes.c_void_p(), ctypes.c_void_p()
    binding.lib().pe_cache_pools(pair.gpu.handle, ctypes.byref(kptr), ctypes.byref(vptr))
    n = L * pair.gpu.num_pages * hkv * ps * d
    kpool = _view_device(kptr.value, n).view(L, pair.gpu.num_pages, hkv, ps, d)
    vpool = _view_device(vptr.value, n).view(L, pair.gpu.num_pages, hkv, ps, d)
    length, _ = pair.orc.seq_info(s)
    tbl = pair.orc.page_table(s)
    kb = synth.torch_to_bits(kpool)
    vb = synth.torch_to_bits(vpool)
    for pos in range(length):
        pg, slot = tbl[pos // ps], pos % ps
        assert np.array_equal(kb[:, pg, :, slot], pair.orc.k_pool[:, pg, :, slot]), pos
        assert np.array_equal(vb[:, pg, :, slot], pair.orc.v_pool[:, pg, :, slot]), pos


def _view_device(ptr, n):
    """A bf16 CUDA tensor over n elements at a raw device pointer (read-only use)."""
    class _Arr:
        __cuda_array_interface__ = {"shape": (n,), "typestr": "<i2", "data": (ptr, False), "version": 3}
    return torch.as_tensor(_Arr(), device="cuda").view(torch.bfloat16)


@pytest.mark.parametrize("order", [-1, 1])
@pytest.mark.parametrize("split", [0, 1])
def test_splitkv_forced(split, order):
    """The split-KV kernel + LSE combine and the single-pass kernel, forced;
    CTAs numbered in the default order and pairs fastest ("attn_order" = 1)."""
    for case in [(128, 32, 8, 16, 4000, 16), (64, 8, 2, 64, 1500, 70), (128, 8, 8, 16, 130, 3),
                 (128, 32, 8, 16, 900, 700)]:
        d, hq, hkv, ps, P, S = case
        pair, s, outs, refs, _ = replay_case(1, hq, hkv, d, ps, P, S, seed=17, split=split,
                                             options={"attn_order": order, "attn_kernel": 0})
        assert_close(outs[0], refs[0], f"split={split} order={order} {case}")


def test_splitkv_many_splits():
    """A forced split count larger than needed: empty splits must contribute nothing."""
    d, hq, hkv, ps, P, S = 128, 32, 8, 16, 9000, 16
    T = P + S
    npg = -(-T // ps) + 2
    pair = Pair(1, hkv, d, ps, npg, 1, npg, seed=23)
    pair.gpu.set_option("splitkv", 1)
    pair.gpu.set_option("num_splits", 37)
    g = synth.rng(23, 2)
    s = pair.seq()
    pair.append(s, synth.normal_bf16(g, (1, T, hkv, d)), synth.normal_bf16(g, (1, T, hkv, d)))
    q = synth.normal_bf16(g, (S, hq, d))
    out = pair.gpu.replay_attn(s, 0, dev(q))
    assert_close(out, oracle.replay_attention(pair.orc, s, 0, q, 1 / math.sqrt(d)), "37 splits")


@pytest.mark.parametrize("decode_kernel", [0, 1])
def test_splice_theorem_bitwise(decode_kernel):
    """Theorem 1 on the GPU: crop to tau-1 + replay of the sanitized suffix equals
    a from-scratch pass over the counterfactual sequence, bit for bit (key tiles
    are keyed to logical positions, not to physical pages).  With the decode
    kernel on, a one-position suffix takes it on both sides (the from-scratch
    side attends that position alone); off, every call takes the tensor-core
    kernel and the from-scratch side attends every position."""
    L, hq, hkv, d, ps = 1, 32, 8, 128, 16
    for (T, tau) in [(700, 301), (1000, 1), (513, 513), (2049, 1000), (4100, 4100)]:
        P, S = tau - 1, T - tau + 1
        g = synth.rng(tau, 5)
        k0 = synth.normal_bf16(g, (L, T, hkv, d))
        v0 = synth.normal_bf16(g, (L, T, hkv, d))
        kc = synth.normal_bf16(g, (L, S, hkv, d))
        vc = synth.normal_bf16(g, (L, S, hkv, d))
        qp = synth.normal_bf16(g, (L, P, hq, d))
        qc = synth.normal_bf16(g, (L, S, hq, d))
        import paper_2609_04875_gb300 as pe
        npg = -(-T // ps) + 2
        a = pe.PagedKVCache(L, hkv, d, ps, npg, 1, npg, init_free_order=synth.page_permutation(1, npg))
        a.set_option("splitkv", 0)
        a.set_option("decode_kernel", decode_kernel)
        sa = a.seq_create()
        a.append_kv(sa, dev(k0), dev(v0))
        a.crop(sa, tau)
        a.append_kv(sa, dev(kc), dev(vc))
        rep = a.replay_attn(sa, 0, dev(qc[0]))
        b = pe.PagedKVCache(L, hkv, d, ps, npg, 1, npg, init_free_order=synth.page_permutation(2, npg))
        b.set_option("splitkv", 0)
        b.set_option("decode_kernel", decode_kernel)
        sb = b.seq_create()
        b.append_kv(sb, dev(np.concatenate([k0[:, :P], kc], 1)), dev(np.concatenate([v0[:, :P], vc], 1)))
        if decode_kernel and S * (hq // hkv) <= 16:
            full = b.replay_attn(sb, 0, dev(qc[0]))
            torch.cuda.synchronize()
            assert torch.equal(rep, full), f"T={T} tau={tau}: splice differs (decode kernel)"
        else:
            full = b.replay_attn(sb, 0, dev(np.concatenate([qp[0], qc[0]], 0)))
            torch.cuda.synchronize()
            assert torch.equal(rep, full[P:]), f"T={T} tau={tau}: splice differs"
        assert a.seq_info(sa) == (T, S)


def test_recompute_bound_on_gpu():
    """Corollary 1: after the replay the counter reads T - tau + 1, and reusing one
    original suffix token instead of recomputing it changes the last query's output."""
    L, hq, hkv, d, ps, T, tau = 1, 8, 2, 64, 16, 300, 121
    S = T - tau + 1
    pair, s, outs, refs, (k0, v0, kc, vc, qc, scale) = replay_case(L, hq, hkv, d, ps, tau - 1, S, seed=41)
    assert pair.gpu.seq_info(s) == (T, S)
    k2, v2 = kc.copy(), vc.copy()
    j = S // 2
    k2[:, j], v2[:, j] = k0[:, tau - 1 + j], v0[:, tau - 1 + j]
    pair.gpu.crop(s, tau)
    pair.gpu.append_kv(s, dev(k2), dev(v2))
    wrong = pair.gpu.replay_attn(s, 0, dev(qc[0]), softmax_scale=scale)
    diff = (wrong[-1].float() - outs[0][-1].float()).abs().max().item()
    assert diff > MAX_ABS / 4, f"reusing an original suffix token went unnoticed ({diff})"


def test_closed_forms_on_gpu():
    import paper_2609_04875_gb300 as pe
    # one key: the output is that value row exactly
    c = pe.PagedKVCache(1, 2, 128, 16, 4, 1, 4)
    s = c.seq_create()
    g = synth.rng(3, 3)
    k = synth.normal_bf16(g, (1, 1, 2, 128))
    v = synth.normal_bf16(g, (1, 1, 2, 128))
    c.append_kv(s, dev(k), dev(v))
    q = dev(synth.normal_bf16(g, (1, 8, 128)))
    out = c.replay_attn(s, 0, q)
    torch.cuda.synchronize()
    want = synth.bits_to_torch(v[0, 0]).cuda().repeat_interleave(4, dim=0)
    assert torch.equal(out[0], want)
    # Q = 0: uniform weights -> mean of the visible values
    c2 = pe.PagedKVCache(1, 1, 64, 16, 8, 1, 8)
    s2 = c2.seq_create()
    k = synth.normal_bf16(g, (1, 90, 1, 64))
    v = synth.normal_bf16(g, (1, 90, 1, 64))
    c2.append_kv(s2, dev(k), dev(v))
    out = c2.replay_attn(s2, 0, torch.zeros((7, 1, 64), dtype=torch.bfloat16, device="cuda"))
    vf = synth.bf16_bits_to_f32(v[0, :, 0]).astype(np.float64)
    want = np.stack([vf[: 90 - 7 + i + 1].mean(0) for i in range(7)])
    got = out[:, 0].float().cpu().numpy()
    assert np.max(np.abs(got - want)) < 1e-2


def test_batch_varlen_matches_oracle():
    L, hq, hkv, d, ps = 1, 32, 8, 128, 16
    specs = [(700, 50), (64, 300), (1500, 1), (0, 129), (333, 333)]  # (P, S) per agent
    npg = sum(-(-(P + S) // ps) for P, S in specs) + 8
    pair = Pair(L, hkv, d, ps, npg, len(specs), npg, seed=77)
    seqs = [pair.seq() for _ in specs]
    g = synth.rng(77, 1)
    kcs, vcs, qcs = [], [], []
    for s, (P, S) in zip(seqs, specs):
        pair.append(s, synth.normal_bf16(g, (L, P + S, hkv, d)), synth.normal_bf16(g, (L, P + S, hkv, d)))
        kcs.append(synth.normal_bf16(g, (L, S, hkv, d)))
        vcs.append(synth.normal_bf16(g, (L, S, hkv, d)))
        qcs.append(synth.normal_bf16(g, (S, hq, d)))
    taus = [P + 1 for P, _ in specs]
    pair.gpu.crop_batch(seqs, taus)
    for s, t in zip(seqs, taus):
        pair.orc.crop(s, t)
    cu = [0] + list(np.cumsum([S for _, S in specs]))
    pair.gpu.append_kv_batch(seqs, dev(np.concatenate(kcs, 1)), dev(np.concatenate(vcs, 1)), cu)
    for s, k, v in zip(seqs, kcs, vcs):
        pair.orc.append(s, k, v)
    pair.check_state(seqs)
    out = pair.gpu.replay_attn_batch(seqs, 0, dev(np.concatenate(qcs, 0)), cu)
    torch.cuda.synchronize()
    for i, s in enumerate(seqs):
        ref = oracle.replay_attention(pair.orc, s, 0, qcs[i], 1 / math.sqrt(d))
        assert_close(out[cu[i]:cu[i + 1]], ref, f"agent {i}")


def test_debug_poison_never_read():
    """Freed pages and stale tails are overwritten with a finite sentinel; a
    correct kernel never reads them unmasked, so results stay within tolerance."""
    L, hq, hkv, d, ps = 2, 8, 2, 128, 16
    T, tau = 900, 401
    npg = -(-T // ps) + 4
    pair = Pair(L, hkv, d, ps, npg, 2, npg, seed=9)
    pair.gpu.set_option("debug_poison", 1)
    s = pair.seq()
    g = synth.rng(9, 1)
    pair.append(s, synth.normal_bf16(g, (L, T, hkv, d)), synth.normal_bf16(g, (L, T, hkv, d)))
    pair.crop(s, tau)
    S = T - tau + 1
    kc, vc = synth.normal_bf16(g, (L, S, hkv, d)), synth.normal_bf16(g, (L, S, hkv, d))
    # a second sequence takes pages the crop poisoned, then the first re-appends
    s2 = pair.seq()
    pair.append(s2, synth.normal_bf16(g, (L, 40, hkv, d)), synth.normal_bf16(g, (L, 40, hkv, d)))
    pair.append(s, kc, vc)
    qc = synth.normal_bf16(g, (L, S, hq, d))
    for layer in range(L):
        out = pair.gpu.replay_attn(s, layer, dev(qc[layer]))
        assert_close(out, oracle.replay_attention(pair.orc, s, layer, qc[layer], 1 / math.sqrt(d)), "poison")
    out2 = pair.gpu.replay_attn(s2, 1, dev(synth.normal_bf16(g, (40, hq, d))))
    assert torch.isfinite(out2.float()).all()
    pair.check_state([s, s2])


def test_gpu_error_paths_leave_state_unchanged():
    import paper_2609_04875_gb300 as pe
    from paper_2609_04875_gb300.binding import PEError
    c = pe.PagedKVCache(2, 2, 128, 16, 6, 2, 6)
    s = c.seq_create()
    k = torch.zeros((2, 40, 2, 128), dtype=torch.bfloat16, device="cuda")
    c.append_kv(s, k, k)
    s2 = c.seq_create()
    c.append_kv(s2, k[:, :32].contiguous(), k[:, :32].contiguous())   # 3 + 2 pages used, 1 free
    before = (c.page_table(s), c.free_list(), c.seq_info(s))
    q = torch.zeros((41, 8, 128), dtype=torch.bfloat16, device="cuda")
    for fn, kind in [(lambda: c.replay_attn(s, 0, q), "range"),
                     (lambda: c.replay_attn(s, 2, q[:4]), "range"),
                     (lambda: c.replay_attn(s, 0, torch.zeros((4, 6, 128), dtype=torch.bfloat16, device="cuda")), "unsupported"),
                     (lambda: c.replay_attn(s, 0, q[:4], softmax_scale=-1.0), "invalid"),
                     (lambda: c.append_kv(s, torch.zeros((2, 60, 2, 128), dtype=torch.bfloat16, device="cuda"),
                                          torch.zeros((2, 60, 2, 128), dtype=torch.bfloat16, device="cuda")), "range"),
                     (lambda: c.append_kv(s, torch.zeros((2, 40, 2, 128), dtype=torch.bfloat16, device="cuda"),
                                          torch.zeros((2, 40, 2, 128), dtype=torch.bfloat16, device="cuda")), "oom"),
                     (lambda: c.crop(s, 0), "invalid"), (lambda: c.crop(s, 42), "range")]:
        with pytest.raises(PEError) as e:
            fn()
        assert e.value.kind == kind
    assert (c.page_table(s), c.free_list(), c.seq_info(s)) == before
    # misaligned pointer
    raw = torch.zeros(8 * 128 * 4 + 8, dtype=torch.bfloat16, device="cuda")
    qm = raw[1:1 + 4 * 8 * 128].view(4, 8, 128)
    with pytest.raises(PEError) as e:
        c.replay_attn(s, 0, qm)
    assert e.value.kind == "invalid"
    assert c.device_status() == 0


@pytest.mark.parametrize("order", [0, 1])
@pytest.mark.parametrize("split", [0, 1])
def test_batch_item_orders(order, split):
    """A launch of six sequences of mixed lengths (one-item kernel), with and
    without key splits, its CTAs numbered kv-heads fastest or pairs fastest:
    every sequence's rows against the oracle."""
    d, hq, hkv, ps = 128, 32, 8, 16
    g = synth.rng(71, 5)
    lens = [int(x) for x in g.integers(200, 2500, size=6)]
    nq = [int(x) for x in g.integers(1, 300, size=6)]
    npg = sum(-(-n // ps) for n in lens) + 8
    pair = Pair(1, hkv, d, ps, npg, 6, 200, seed=71)
    pair.gpu.set_option("attn_kernel", 0)
    pair.gpu.set_option("attn_order", order)
    pair.gpu.set_option("splitkv", split)
    seqs = []
    for n in lens:
        s = pair.seq()
        pair.append(s, synth.normal_bf16(g, (1, n, hkv, d)), synth.normal_bf16(g, (1, n, hkv, d)))
        seqs.append(s)
    cu = [0]
    for k in nq:
        cu.append(cu[-1] + k)
    q = synth.normal_bf16(g, (cu[-1], hq, d))
    scale = 1 / math.sqrt(d)
    out = pair.gpu.replay_attn_batch(seqs, 0, dev(q), cu, softmax_scale=scale)
    torch.cuda.synchronize()
    for i, s in enumerate(seqs):
        ref = oracle.replay_attention(pair.orc, s, 0, q[cu[i]:cu[i + 1]], scale)
        assert_close(out[cu[i]:cu[i + 1]], ref, f"order={order} split={split} seq {i}")
    assert pair.gpu.device_status() == 0
