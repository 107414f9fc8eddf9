"""The persistent prefill kernel's work plan, checked on the host.

pe_attn_plan_persistent returns the plan the attention call would launch: the
units (sequence, kv-head, pair of 128-row q-tiles), the lockstep rounds of
whole units and each CTA's tail stretch of (unit, key tile) work, and the cut
units whose pieces are merged in the kernel.  The kernel walks its pieces by
fixed rules (restated below from the header's description of the plan); this
test replays those rules for every CTA of thousands of random launch groups
and checks what the kernel needs of the plan:
  - each unit's key tiles are those its later q-tile sees under the causal
    mask (queries are a sequence's last positions);
  - every key tile of every unit is computed exactly once;
  - a whole piece writes the output directly, a cut unit's pieces are parts
    0 .. n_parts-1 of one slot, each once, in key order, so the count its
    merge waits for is reached exactly (a planner that counted a boundary
    twice left a unit unmerged on the GPU before);
  - the slots and parts fit the workspace and the kernel's limits.
No GPU is used: host-only caches plan without device memory."""
import math
import random

import pytest

pe = pytest.importorskip("paper_2609_04875_gb300")
from paper_2609_04875_gb300 import binding  # noqa: E402

BM = BN = 128          # query rows and keys per tile
MAX_CTAS = 160
MAX_PARTS = 32


def unit_key_tiles(lens_in_order, n_q_in_order, g, hkv):
    """Key tiles of every unit in the kernel's unit order: sequences in order,
    pairs from the latest queries down, kv-heads fastest.  A pair of q-tiles
    loads the key tiles its later q-tile sees: its last query row sits at
    position len - n_q + q_last and attends every key up to it."""
    rows_per_tile = BM // g
    tiles = []
    for n, nq in zip(lens_in_order, n_q_in_order):
        n_qtiles = -(-nq * g // BM)
        n_pairs = -(-n_qtiles // 2)
        for local in range(n_pairs * hkv):
            pair = n_pairs - 1 - local // hkv
            later = min(2 * pair + 1, n_qtiles - 1)
            q_last = min((later + 1) * rows_per_tile, nq) - 1
            tiles.append(-(-(n - nq + q_last + 1) // BN))
    return tiles


def pieces_of(plan, k):
    """The pieces CTA k computes, as the kernel walks them: (unit, first key
    tile, end key tile, slot, part); slot -1 is a whole unit."""
    nc, rounds, tiles = plan["n_ctas"], plan["rounds"], plan["unit_tiles"]
    out = []
    for r in range(rounds):
        u = r * nc + (nc - 1 - k if r % 2 else k)
        out.append((u, 0, tiles[u], -1, 0))
    u0, t0, u1, t1, s0, p0, s1, p1 = plan["ctas"][k]
    j = 0
    while True:
        u = u0 + j
        if u > u1 or (u == u1 and t1 == 0 and u != u0):
            break
        lo = t0 if j == 0 else 0
        hi = t1 if (u == u1 and t1 > 0) else tiles[u]
        slot, part = (s0, p0) if j == 0 else ((s1, p1) if u == u1 else (-1, 0))
        if hi <= lo:  # the kernel stops at an empty piece
            break
        out.append((u, lo, hi, slot, part))
        j += 1
    return out


def check_plan(plan, lens, nqs, seqs, g, hkv, d, num_sms, ws_bytes, attn_ctas):
    by_seq = dict(zip(seqs, zip(lens, nqs)))
    order = plan["order"]
    assert sorted(order) == sorted(seqs)
    # longest first, ties in the given order
    assert order == sorted(seqs, key=lambda s: (-by_seq[s][0], seqs.index(s)))
    want = unit_key_tiles([by_seq[s][0] for s in order], [by_seq[s][1] for s in order], g, hkv)
    tiles = plan["unit_tiles"]
    assert tiles == want
    U, nc = len(tiles), plan["n_ctas"]
    assert 1 <= nc <= (attn_ctas if attn_ctas else num_sms) and nc <= MAX_CTAS
    assert plan["rounds"] * nc <= U
    assert plan["n_slots"] == len(plan["slots"]) and 1 <= plan["max_parts"] <= MAX_PARTS
    if plan["n_slots"]:
        assert plan["n_slots"] * plan["max_parts"] * 2 * BM * (4 * d + 4) <= ws_bytes

    spans = [[] for _ in range(U)]  # (lo, hi, slot, part) of every piece of each unit
    for k in range(nc):
        for u, lo, hi, slot, part in pieces_of(plan, k):
            assert 0 <= u < U and 0 <= lo < hi <= tiles[u]
            spans[u].append((lo, hi, slot, part))
    slot_unit = {i: (unit, n) for i, (unit, n) in enumerate(plan["slots"])}
    assert len({unit for unit, _ in slot_unit.values()}) == len(slot_unit)  # one slot per cut unit
    for u in range(U):
        sp = sorted(spans[u])
        assert sp, f"unit {u} is never computed"
        # the pieces tile [0, key tiles) with no gap and no overlap
        assert sp[0][0] == 0 and sp[-1][1] == tiles[u], (u, sp)
        for a, b in zip(sp, sp[1:]):
            assert a[1] == b[0], (u, sp)
        if len(sp) == 1:
            assert sp[0][2] == -1, f"unit {u} is whole but written as a part"
            continue
        slots = {s for _, _, s, _ in sp}
        assert len(slots) == 1 and -1 not in slots, (u, sp)
        slot = slots.pop()
        assert 0 <= slot < plan["n_slots"]
        unit, n_parts = slot_unit[slot]
        assert unit == u and n_parts == len(sp) <= plan["max_parts"], (u, sp, slot_unit[slot])
        assert [p for _, _, _, p in sp] == list(range(n_parts)), (u, sp)


def _cache(hkv, d, max_seqs, ws_bytes):
    return pe.PagedKVCache(1, hkv, d, 16, 20000, max_seqs, 2100, host_only=True, workspace_bytes=ws_bytes)


def _plan(c, lens, nqs, hq, num_sms):
    seqs = []
    for n in lens:
        s = c.seq_create()
        c.append_kv(s, n_tokens=n)
        seqs.append(s)
    return seqs, c.plan_persistent(seqs, nqs, hq, num_sms=num_sms)


def test_plan_with_empty_stretches():
    """The batch whose empty tail stretches met inside a cut unit (9 CTAs):
    every boundary is counted once, so the unit's part count is reached."""
    lens, nqs = [3216, 684, 1623, 1045, 743], [337, 85, 233, 411, 475]
    c = _cache(8, 128, 8, 0)
    c.set_option("splitkv", 1)
    c.set_option("attn_ctas", 9)
    seqs, plan = _plan(c, lens, nqs, 32, 152)
    assert plan["n_ctas"] == 9 and plan["n_slots"] > 0
    # an empty stretch: two consecutive CTA boundaries coincide inside a unit
    bounds = [(r[0], r[1]) for r in plan["ctas"]]
    assert any(a == b for a, b in zip(bounds, bounds[1:])) or any(r[0] > r[2] for r in plan["ctas"])
    check_plan(plan, lens, nqs, seqs, 4, 8, 128, 152, 256 << 20, 9)


@pytest.mark.parametrize("case", [
    # (d, hq, hkv, lens, n_q, SMs): the persistent kernel's GPU parity cases and the sweep's tau/T 0.9
    (128, 32, 8, [3700], [700], 152),
    (128, 8, 8, [1800], [300], 152),
    (64, 16, 1, [5100], [100], 152),
    (128, 64, 8, [1200], [1000], 152),
    (64, 4, 2, [9040], [40], 152),
    (128, 32, 8, [16384], [1638], 152),
    (128, 32, 8, [32784] * 8, [16] * 8, 152),
])
def test_plans_of_the_gpu_cases(case):
    d, hq, hkv, lens, nqs, sms = case
    for splitkv in (-1, 1):
        for ctas in (0, 1, 7, 152):
            c = _cache(hkv, d, len(lens), 0)
            c.set_option("splitkv", splitkv)
            c.set_option("attn_ctas", ctas)
            seqs, plan = _plan(c, lens, nqs, hq, sms)
            check_plan(plan, lens, nqs, seqs, hq // hkv, hkv, d, sms, 256 << 20, ctas)
            c.close()


def test_random_plans_cover_every_key_tile_once():
    rng = random.Random(2609)
    cases = 0
    for _ in range(4000):
        d = rng.choice([64, 128])
        hkv = rng.choice([1, 2, 4, 8])
        g = rng.choice([1, 2, 4, 8, 16])
        n = rng.choice([1, 1, 2, 3, 5, 8, 12])
        lens, nqs = [], []
        for _ in range(n):
            length = rng.choice([rng.randint(1, 300), rng.randint(300, 4000), rng.randint(4000, 20000)])
            lens.append(length)
            nqs.append(rng.choice([1, rng.randint(1, min(length, 64)), rng.randint(1, length)]))
        sms = rng.choice([1, 2, 7, 9, 37, 148, 152, 160])
        ws = rng.choice([0, 1 << 20, 8 << 20])   # 0: the default 256 MiB; small ones force fewer cuts
        c = _cache(hkv, d, n, ws)
        splitkv = rng.choice([-1, 1, 1])
        ctas = rng.choice([0, 0, rng.randint(1, MAX_CTAS)])
        c.set_option("splitkv", splitkv)
        c.set_option("attn_ctas", ctas)
        seqs, plan = _plan(c, lens, nqs, g * hkv, sms)
        check_plan(plan, lens, nqs, seqs, g, hkv, d, sms, ws or (256 << 20), ctas)
        cases += plan["n_slots"] > 0
        c.close()
    assert cases > 1000  # a good share of the plans cut units


def test_plan_arguments_are_checked():
    c = _cache(8, 128, 4, 0)
    s = c.seq_create()
    c.append_kv(s, n_tokens=500)
    with pytest.raises(binding.PEError, match="num_sms"):
        c.plan_persistent([s], [10], 32, num_sms=0)   # a host-only cache has no SM count
    with pytest.raises(binding.PEError) as e:
        c.plan_persistent([s], [501], 32, num_sms=152)
    assert e.value.kind == "range"
    with pytest.raises(binding.PEError) as e:
        c.plan_persistent([s], [0], 32, num_sms=152)
    assert e.value.kind == "range"
    with pytest.raises(binding.PEError) as e:
        c.plan_persistent([s], [10], 24, num_sms=152)
    assert e.value.kind == "unsupported"
    with pytest.raises(binding.PEError) as e:
        c.plan_persistent([s, s], [10, 10], 32, num_sms=152)
    assert e.value.kind == "invalid"
    plan = c.plan_persistent([s], [10], 32, num_sms=152)
    assert plan["unit_tiles"] == [math.ceil(500 / 128)] * 8


def test_checker_rejects_broken_plans():
    """The checks above catch the plan mistakes that would go wrong on the GPU:
    a part count one too high (the merge never runs), a stretch starting one
    tile late (a tile skipped) or early (a tile computed twice), a part
    numbered twice, and a cut unit's piece written as a whole unit."""
    import copy
    lens, nqs = [3216, 684, 1623, 1045, 743], [337, 85, 233, 411, 475]
    c = _cache(8, 128, 8, 0)
    c.set_option("splitkv", 1)
    c.set_option("attn_ctas", 9)
    seqs, plan = _plan(c, lens, nqs, 32, 152)
    args = (lens, nqs, seqs, 4, 8, 128, 152, 256 << 20, 9)
    check_plan(plan, *args)
    k = next(i for i, r in enumerate(plan["ctas"]) if r[4] >= 0 and r[1] > 0)  # a stretch starting inside a cut unit

    def broken(edit):
        p = copy.deepcopy(plan)
        edit(p)
        with pytest.raises(AssertionError):
            check_plan(p, *args)

    broken(lambda p: p["slots"][0].__setitem__(1, p["slots"][0][1] + 1))
    broken(lambda p: p["ctas"][k].__setitem__(1, p["ctas"][k][1] + 1))
    broken(lambda p: p["ctas"][k].__setitem__(1, p["ctas"][k][1] - 1))
    broken(lambda p: p["ctas"][k].__setitem__(5, (p["ctas"][k][5] + 1) % p["slots"][p["ctas"][k][4]][1]))
    broken(lambda p: p["ctas"][k].__setitem__(4, -1))
    broken(lambda p: p["unit_tiles"].__setitem__(0, p["unit_tiles"][0] + 1))


# ---------------------------------------------------------------- every launch of an attention call
def q_tile_key_tiles(n, nq, g, qt):
    """128-key tiles q-tile qt of a sequence of n keys whose last nq positions
    are the queries sees: its last row sits at position n - nq + q_last."""
    q_last = min((qt + 1) * (BM // g), nq) - 1
    return -(-(n - nq + q_last + 1) // BN)


def one_item_ctas(launch, hkv):
    """(sequence index, kv-head, split, pair) of every CTA of a one-item launch,
    decoded by the kernel's rules (stated with pe_attn_plan_launches)."""
    seqs, ctas = launch["seqs"], launch["ctas"]
    out = []
    for b in range(ctas):
        i = max(k for k, q in enumerate(seqs) if q["item0"] <= b)
        q = seqs[i]
        end = seqs[i + 1]["item0"] if i + 1 < len(seqs) else ctas
        local, ns = b - q["item0"], q["n_splits"]
        assert (end - q["item0"]) % (hkv * ns) == 0
        if launch["pairs_fastest"]:
            pairs = (end - q["item0"]) // (hkv * ns)
            pair, split, kvh = q["pair_top"] - 1 - local % pairs, (local // pairs) % ns, local // pairs // ns
        else:
            kvh, split, pair = local % hkv, (local // hkv) % ns, q["pair_top"] - 1 - local // hkv // ns
        out.append((i, kvh, split, pair))
    return out


def check_launches(plan, lens, nqs, seqs, g, hkv, d, ws_bytes, decode_rows_max):
    by_seq = dict(zip(seqs, zip(lens, nqs)))
    done = {}          # (seq, kv-head, q-tile) -> how it was computed
    seen = {s: [] for s in seqs if by_seq[s][1] > 0}
    for li, launch in enumerate(plan):
        assert 1 <= len(launch["seqs"]) <= 64
        for q in launch["seqs"]:
            seen[q["seq"]].append(launch["kind"])
            assert (q["n_keys"], q["n_q"]) == by_seq[q["seq"]]
        if launch["kind"] == "decode":
            for q in launch["seqs"]:
                assert q["n_q"] * g <= decode_rows_max
            continue
        for q in launch["seqs"]:
            assert q["n_q"] * g > decode_rows_max
            assert q["n_qtiles"] == -(-q["n_q"] * g // BM)
        if launch["kind"] == "persistent":
            continue
        split, st = launch["split"], launch["split_tiles"]
        cover = {}
        for i, kvh, sp, pair in one_item_ctas(launch, hkv):
            q = launch["seqs"][i]
            assert 0 <= kvh < hkv and 0 <= sp < q["n_splits"] and 0 <= pair < q["pair_top"]
            assert 2 * pair < q["n_qtiles"]
            for qt in (2 * pair, 2 * pair + 1):
                if qt >= q["n_qtiles"]:
                    continue
                key = (q["seq"], kvh, qt)
                cover.setdefault(key, []).append(sp)
                if split:
                    # every key tile the q-tile sees lies in one of the splits
                    assert q["n_splits"] * st >= q_tile_key_tiles(q["n_keys"], q["n_q"], g, qt)
        for key, sps in cover.items():
            ns = launch["seqs"][[q["seq"] for q in launch["seqs"]].index(key[0])]["n_splits"]
            assert sorted(sps) == list(range(ns)), (key, sps)     # each split once
            assert key not in done, f"{key} computed twice"
            done[key] = (li, split)
        if not split:
            assert launch["combine_rows"] == 0 and all(q["n_splits"] == 1 for q in launch["seqs"])
            continue
        # partial rows: each sequence's block in the workspace, disjoint; the combine reads what was written
        blocks, comb = [], 0
        for i, q in enumerate(launch["seqs"]):
            n_qt = q["n_qtiles"] if launch["kind"] == "one_item" else min(q["n_qtiles"], 2 * q["pair_top"])
            blocks.append((q["part_row0"], q["part_row0"] + n_qt * hkv * q["n_splits"] * BM))
            assert q["comb0"] == comb
            comb += n_qt * hkv * BM
            for qt in range(n_qt):
                for kvh in range(hkv):
                    assert sorted(cover[(q["seq"], kvh, qt)]) == list(range(q["n_splits"]))
        assert launch["combine_rows"] == comb
        blocks.sort()
        for a, b in zip(blocks, blocks[1:]):
            assert a[1] <= b[0], blocks
        assert blocks[-1][1] * (4 * d + 4) <= ws_bytes
    for s, kinds in seen.items():
        assert kinds in (["decode"], ["persistent"], ["one_item"], ["one_item", "one_item_tail"]), (s, kinds)
        if kinds[0] in ("one_item",):
            n, nq = by_seq[s]
            for kvh in range(hkv):
                for qt in range(-(-nq * g // BM)):
                    assert (s, kvh, qt) in done, f"sequence {s} q-tile {qt} kv-head {kvh} never computed"


def test_random_launch_plans():
    rng = random.Random(4875)
    kinds = {}
    for _ in range(1200):
        d = rng.choice([64, 128])
        hkv = rng.choice([1, 2, 4, 8])
        g = rng.choice([1, 2, 4, 8, 16])
        n = rng.choice([1, 1, 1, 2, 3, 5, 16, 70])
        lens, nqs = [], []
        for _ in range(n):
            length = rng.choice([rng.randint(1, 300), rng.randint(300, 4000), rng.randint(4000, 16384)])
            if n > 16:
                length = min(length, 3000)
            lens.append(length)
            nqs.append(rng.choice([0, 1, rng.randint(1, min(length, 64)), rng.randint(1, length)]))
        sms = rng.choice([7, 37, 148, 152, 160])
        ws = rng.choice([0, 1 << 20, 8 << 20])
        c = pe.PagedKVCache(1, hkv, d, 16, 40000, max(n, 1), 1100, host_only=True, workspace_bytes=ws)
        opts = {"splitkv": rng.choice([-1, -1, 0, 1]), "num_splits": rng.choice([0, 0, 0, rng.randint(1, 9)]),
                "attn_kernel": rng.choice([1, 1, 0, 2]), "attn_order": rng.choice([-1, -1, 0, 1]),
                "decode_kernel": rng.choice([1, 1, 0, 2])}
        for k, v in opts.items():
            c.set_option(k, v)
        seqs = []
        for length in lens:
            s = c.seq_create()
            c.append_kv(s, n_tokens=length)
            seqs.append(s)
        plan = c.plan_launches(seqs, nqs, g * hkv, num_sms=sms)
        decodes = opts["decode_kernel"] and not (opts["decode_kernel"] == 1 and opts["splitkv"] == 0)
        check_launches(plan, lens, nqs, seqs, g, hkv, d, ws or (256 << 20), 16 if decodes else 0)
        for launch in plan:
            k = (launch["kind"], launch["split"], launch["pairs_fastest"])
            kinds[k] = kinds.get(k, 0) + 1
        c.close()
    # the plans span every launch kind, split and unsplit, in both CTA orders
    for k in [("decode", False, False), ("persistent", False, False), ("persistent", True, False),
              ("one_item", False, False), ("one_item", False, True), ("one_item", True, False),
              ("one_item", True, True), ("one_item_tail", True, False)]:
        assert kinds.get(k, 0) > 0, (k, kinds)


def test_launch_plans_of_the_workloads():
    """The configurations' own launch groups plan as measured: tau/T 0.7 with a
    tail launch of 19 splits over 8 units, tau/T 0.9 and the short suffix on the
    persistent kernel, the tiny launch in one pass of 8 CTAs, tau/T 0.5 in four
    waves, the long suffix's 16384 CTAs pairs fastest."""
    def plan_of(hkv, d, lens, nqs, hq, ps=16):
        c = pe.PagedKVCache(1, hkv, d, ps, 40000, len(lens), 4100, host_only=True)
        seqs = []
        for n in lens:
            s = c.seq_create()
            c.append_kv(s, n_tokens=n)
            seqs.append(s)
        p = c.plan_launches(seqs, nqs, hq, num_sms=152)
        check_launches(p, lens, nqs, seqs, hq // hkv, hkv, d, 256 << 20, 16)
        return [(x["kind"], x["split"], x["ctas"], x["pairs_fastest"]) for x in p]

    assert plan_of(8, 128, [16384], [4915], 32) == [("one_item", False, 608, False), ("one_item_tail", True, 152, False)]
    assert plan_of(8, 128, [16384], [1638], 32)[0][0] == "persistent"
    assert plan_of(8, 128, [32784] * 8, [16] * 8, 32)[0][0] == "persistent"
    assert plan_of(8, 64, [640], [128], 8) == [("one_item", False, 8, False)]
    assert plan_of(8, 128, [16384], [8192], 32) == [("one_item", False, 1024, False)]
    lens = [20480] * 4
    assert plan_of(8, 128, lens, [16384] * 4, 64, ps=64) == [("one_item", False, 16384, True)]


def test_launch_checker_rejects_broken_plans():
    """check_launches catches a lost split, a sequence boundary between CTAs
    moved by one (kv-head x split) group, overlapping partial blocks, a combine
    that misses rows, a sequence left out of every launch and splits too short
    for the keys.  (The two CTA orders are both valid numberings of the same
    work, so swapping them is not a mistake.)"""
    import copy
    c = pe.PagedKVCache(1, 8, 128, 16, 40000, 4, 4100, host_only=True)
    c.set_option("splitkv", 1)
    c.set_option("attn_kernel", 0)   # the one-item kernel with key splits
    lens, nqs = [9000, 5000, 3000], [700, 300, 129]
    seqs = []
    for n in lens:
        s = c.seq_create()
        c.append_kv(s, n_tokens=n)
        seqs.append(s)
    plan = c.plan_launches(seqs, nqs, 32, num_sms=152)
    args = (lens, nqs, seqs, 4, 8, 128, 256 << 20, 16)
    check_launches(plan, *args)
    assert [x["kind"] for x in plan] == ["one_item"] and plan[0]["split"] and len(plan[0]["seqs"]) == 3

    def broken(edit):
        p = copy.deepcopy(plan)
        edit(p[0])
        with pytest.raises(AssertionError):
            check_launches(p, *args)

    broken(lambda x: x["seqs"][0].__setitem__("n_splits", x["seqs"][0]["n_splits"] - 1))
    broken(lambda x: x["seqs"][1].__setitem__("item0", x["seqs"][1]["item0"] + 16))
    broken(lambda x: x["seqs"][1].__setitem__("part_row0", x["seqs"][1]["part_row0"] - BM))
    broken(lambda x: x.__setitem__("combine_rows", x["combine_rows"] - BM))
    broken(lambda x: x["seqs"].pop())
    broken(lambda x: x.__setitem__("split_tiles", x["split_tiles"] - 1))


def test_persistent_launches_agree_with_the_persistent_plan():
    """Where an attention call takes the persistent kernel, its launch record
    and pe_attn_plan_persistent describe the same plan: the same sequences in
    the same order and the same CTA count and cut units."""
    rng = random.Random(99)
    for _ in range(300):
        hkv, g = rng.choice([1, 2, 8]), rng.choice([2, 4, 8])
        n = rng.choice([1, 2, 4, 9])
        lens = [rng.randint(200, 12000) for _ in range(n)]
        nqs = [rng.randint(max(1, 17 // g + 1), min(x, 3000)) for x in lens]
        c = pe.PagedKVCache(1, hkv, 128, 16, 40000, n, 1100, host_only=True)
        c.set_option("attn_kernel", 2)
        c.set_option("splitkv", rng.choice([-1, 1]))
        seqs = []
        for length in lens:
            s = c.seq_create()
            c.append_kv(s, n_tokens=length)
            seqs.append(s)
        sms = rng.choice([9, 152])
        launches = c.plan_launches(seqs, nqs, g * hkv, num_sms=sms)
        plan = c.plan_persistent(seqs, nqs, g * hkv, num_sms=sms)
        assert [x["kind"] for x in launches] == ["persistent"]
        rec = launches[0]
        assert [q["seq"] for q in rec["seqs"]] == plan["order"]
        assert rec["ctas"] == plan["n_ctas"] and rec["split"] == (plan["n_slots"] > 0)
        c.close()
