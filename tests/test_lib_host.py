"""libpe on the CPU: it loads, exports every entry point of include/pe.h, and its
host bookkeeping (free list, page tables, lengths, counters, error codes)
matches the oracle bit for bit.  Host-only caches run no device work."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import oracle_pins as pins
import synth

pe = pytest.importorskip("paper_2609_04875_gb300")
from paper_2609_04875_gb300 import binding  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "pe.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pe_[a-z_0-9]+)\s*\(", src)))


def test_exports_every_declared_symbol():
    names = declared_symbols()
    assert "pe_crop" in names and "pe_replay_attn" in names and "pe_cache_create" in names
    lib = ctypes.CDLL(binding.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in pe.h but not exported"
    assert set(names) <= set(binding.EXPORTED)


def test_version_and_error_string():
    assert "sm_103a" in pe.version()
    with pytest.raises(binding.PEError) as e:
        pe.PagedKVCache(1, 1, 96, 16, 8, 1, 8, host_only=True)
    assert e.value.kind == "unsupported" and "head_dim" in str(e.value)


def _mk(cfg, **kw):
    return pe.PagedKVCache(cfg["num_layers"], cfg["num_kv_heads"], 64, 8, cfg["num_pages"], cfg["max_seqs"],
                           cfg["max_pages_per_seq"], init_free_order=cfg.get("init_free_order"), host_only=True, **kw)


def test_golden_trace_page_granular():
    """The hand-derived trace, replayed on libpe (ps = 4 in the trace; libpe needs
    ps >= 8, so every token count and tau is scaled by 2: same pages, same order)."""
    trace = pins.load_trace()
    cfg = trace["config"]
    c = _mk(cfg)
    f = 8 // cfg["page_size"]
    for idx, st in enumerate(trace["steps"]):
        op = st["op"]
        try:
            if op == "create":
                assert c.seq_create() == st["expect_seq"]
                continue
            if op == "append":
                c.append_kv(st["seq"], n_tokens=st["n"] * f)
            elif op == "crop":
                freed = c.crop(st["seq"], (st["tau"] - 1) * f + 1)
                assert freed == st["expect_freed"], f"step {idx}"
            elif op == "release":
                c.seq_release(st["seq"])
                assert c.free_list() == st["expect_free"], f"step {idx}"
                continue
        except binding.PEError as e:
            assert st.get("expect_error") == e.kind, f"step {idx}: {e}"
            continue
        assert "expect_error" not in st, f"step {idx}"
        if "expect" in st:
            ex = st["expect"]
            assert c.page_table(st["seq"]) == ex["table"], f"step {idx}"
            assert c.seq_info(st["seq"]) == (ex["len"] * f, ex["appended"] * f), f"step {idx}"
            assert c.free_list() == ex["free"], f"step {idx}"


@pytest.mark.parametrize("ps", [8, 16, 64])
def test_random_ops_match_oracle(ps):
    num_pages, max_pages = 96, 40
    order = synth.page_permutation(99 + ps, num_pages)
    lib = pe.PagedKVCache(2, 2, 64, ps, num_pages, 5, max_pages, init_free_order=order, host_only=True)
    orc = oracle.OracleKVCache(2, 2, 64, ps, num_pages, 5, max_pages, init_free_order=order, store_values=False)
    g = synth.rng(7, ps)
    live = []
    for step in range(1500):
        r = g.random()
        if r < 0.08 or not live:
            try:
                s1 = orc.seq_create()
            except oracle.OracleError as e:
                with pytest.raises(binding.PEError) as pe_err:
                    lib.seq_create()
                assert pe_err.value.kind == e.kind
                continue
            assert lib.seq_create() == s1
            live.append(s1)
            continue
        s = live[int(g.integers(0, len(live)))]
        n = orc.length[s]
        try:
            if r < 0.12:
                orc.seq_release(s)
                lib.seq_release(s)
                live.remove(s)
            elif r < 0.55:
                tau = int(g.integers(-1, n + 3))
                try:
                    want = orc.crop(s, tau)
                except oracle.OracleError as e:
                    with pytest.raises(binding.PEError) as pe_err:
                        lib.crop(s, tau)
                    assert pe_err.value.kind == e.kind
                    continue
                assert lib.crop(s, tau) == want
            else:
                k = int(g.integers(0, 5 * ps))
                try:
                    orc.append(s, n_tokens=k)
                except oracle.OracleError as e:
                    with pytest.raises(binding.PEError) as pe_err:
                        lib.append_kv(s, n_tokens=k)
                    assert pe_err.value.kind == e.kind
                    continue
                lib.append_kv(s, n_tokens=k)
        finally:
            pass
        assert lib.free_list() == orc.free_list(), f"step {step}"
        for q in live:
            assert lib.page_table(q) == orc.page_table(q), f"step {step}"
            assert lib.seq_info(q) == orc.seq_info(q), f"step {step}"


def test_batch_ops_all_or_nothing():
    c = pe.PagedKVCache(1, 1, 64, 16, 20, 4, 10, host_only=True)
    a, b = c.seq_create(), c.seq_create()
    c.append_kv_batch([a, b], cu_tokens=[0, 40, 70])
    assert c.seq_info(a) == (40, 40) and c.seq_info(b) == (30, 30)
    state = (c.page_table(a), c.page_table(b), c.free_list())
    with pytest.raises(binding.PEError) as e:
        c.crop_batch([a, b], [10, 99])        # second tau out of range
    assert e.value.kind == "range"
    with pytest.raises(binding.PEError) as e:
        c.crop_batch([a, a], [10, 5])         # duplicate sequence
    assert e.value.kind == "invalid"
    with pytest.raises(binding.PEError) as e:
        c.append_kv_batch([a, b], cu_tokens=[0, 16, 16 + 16 * 20])   # OOM on the total
    assert e.value.kind in ("oom", "range")
    assert (c.page_table(a), c.page_table(b), c.free_list()) == state
    c.crop_batch([a, b], [17, 1])
    assert c.seq_info(a) == (16, 0) and c.seq_info(b) == (0, 0)
    assert c.page_table(a) == state[0][:1] and c.page_table(b) == []


def test_error_codes():
    c = pe.PagedKVCache(1, 1, 64, 16, 4, 2, 4, host_only=True)
    s = c.seq_create()
    c.append_kv(s, n_tokens=20)
    for tau, kind in ((0, "invalid"), (22, "range")):
        with pytest.raises(binding.PEError) as e:
            c.crop(s, tau)
        assert e.value.kind == kind
    with pytest.raises(binding.PEError) as e:
        c.crop(3, 1)
    assert e.value.kind == "invalid"
    with pytest.raises(binding.PEError) as e:
        c.append_kv(s, n_tokens=16 * 4)      # 84 tokens > 4 pages
    assert e.value.kind == "range"
    t = c.seq_create()
    c.append_kv(t, n_tokens=30)
    with pytest.raises(binding.PEError) as e:
        c.append_kv(t, n_tokens=3)           # pool exhausted (2 + 2 pages used)
    assert e.value.kind == "oom"
    assert c.seq_info(t) == (30, 30)
    with pytest.raises(binding.PEError) as e:
        c.set_option("nonsense", 1)
    assert e.value.kind == "invalid"
    for key, good, bad in (("attn_order", 1, 2), ("attn_kernel", 2, 3), ("splitkv", -1, 2)):
        c.set_option(key, good)
        with pytest.raises(binding.PEError) as e:
            c.set_option(key, bad)
        assert e.value.kind == "invalid", key
    with pytest.raises(binding.PEError) as e:
        pe.PagedKVCache(1, 1, 64, 16, 4, 2, 4, init_free_order=[0, 1, 1, 2], host_only=True)
    assert e.value.kind == "invalid"


def test_golden_fork_trace():
    """The hand-derived fork / copy-on-write / checkpoint trace on libpe
    (ps = 4 in the trace, 8 here: token counts, taus and offsets doubled)."""
    trace = pins.load_fork_trace()
    cfg = trace["config"]
    c = _mk(cfg)
    f = 8 // cfg["page_size"]
    for idx, st in enumerate(trace["steps"]):
        op, seq = st["op"], st.get("seq")
        try:
            if op == "create":
                assert c.seq_create() == st["expect_seq"]
                continue
            if op == "append":
                c.append_kv(seq, n_tokens=st["n"] * f)
            elif op == "checkpoint":
                for b in st["offsets"]:
                    c.checkpoint_add(seq, b * f)
                continue
            elif op == "fork":
                assert c.seq_fork(seq) == st["expect_seq"], f"step {idx}"
            elif op == "crop":
                assert c.crop(seq, (st["tau"] - 1) * f + 1) == st["expect_freed"], f"step {idx}"
            elif op == "restore":
                b, freed = c.restore(seq, (st["tau"] - 1) * f + 1)
                assert (b, freed) == (st["expect_offset"] * f, st["expect_freed"]), f"step {idx}"
            elif op == "release":
                c.seq_release(seq)
                assert c.free_list() == st["expect_free"], f"step {idx}"
                continue
        except binding.PEError as e:
            assert st.get("expect_error") == e.kind, f"step {idx}: {e}"
            continue
        assert "expect_error" not in st, f"step {idx}"
        ex = st.get("expect", {})
        s = ex.get("seq", seq)
        if "table" in ex:
            assert c.page_table(s) == ex["table"], f"step {idx}: {c.page_table(s)}"
        if "len" in ex:
            assert c.seq_info(s)[0] == ex["len"] * f, f"step {idx}"
        if "free" in ex:
            assert c.free_list() == ex["free"], f"step {idx}"
        refs = c.page_refs()
        for pg, r in ex.get("refs", {}).items():
            assert refs[int(pg)] == r, f"step {idx}: refs[{pg}]"
        if "checkpoints" in ex:
            assert c.checkpoints(s) == [b * f for b in ex["checkpoints"]], f"step {idx}"


@pytest.mark.parametrize("ps", [8, 16])
def test_random_fork_ops_match_oracle(ps):
    num_pages, max_pages, max_seqs = 64, 30, 6
    order = synth.page_permutation(77 + ps, num_pages)
    lib = pe.PagedKVCache(1, 1, 64, ps, num_pages, max_seqs, max_pages, init_free_order=order, host_only=True)
    orc = oracle.OracleKVCache(1, 1, 64, ps, num_pages, max_seqs, max_pages, init_free_order=order,
                               store_values=False)
    assert lib.seq_create() == orc.seq_create()
    g = synth.rng(31, ps)
    for step in range(1500):
        live = sorted(orc.table)
        s = live[int(g.integers(0, len(live)))]
        r = g.random()

        def both(f_orc, f_lib):
            try:
                want = f_orc()
            except oracle.OracleError as e:
                with pytest.raises(binding.PEError) as pe_err:
                    f_lib()
                assert pe_err.value.kind == e.kind, f"step {step}"
                return
            got = f_lib()
            if got is not None:
                assert got == want, f"step {step}"

        n = orc.length[s]
        if r < 0.15:
            both(lambda: orc.seq_fork(s), lambda: lib.seq_fork(s))
        elif r < 0.35:
            tau = int(g.integers(0, n + 3))
            both(lambda: orc.crop(s, tau), lambda: lib.crop(s, tau))
        elif r < 0.45:
            b = int(g.integers(-1, n + 2))
            both(lambda: orc.checkpoint_add(s, b), lambda: lib.checkpoint_add(s, b))
        elif r < 0.55:
            tau = int(g.integers(0, n + 3))
            both(lambda: orc.restore(s, tau), lambda: lib.restore(s, tau))
        elif r < 0.62 and len(live) > 1:
            both(lambda: orc.seq_release(s), lambda: lib.seq_release(s))
        else:
            k = int(g.integers(0, 3 * ps))
            both(lambda: orc.append(s, n_tokens=k), lambda: lib.append_kv(s, n_tokens=k))
        assert lib.free_list() == orc.free_list(), f"step {step}"
        assert lib.page_refs() == list(orc.refs), f"step {step}"
        for q in orc.table:
            assert lib.page_table(q) == orc.page_table(q), f"step {step}"
            assert lib.seq_info(q) == orc.seq_info(q), f"step {step}"
            assert lib.checkpoints(q) == orc.checkpoints[q], f"step {step}"


def test_binding_rejects_mismatched_out_before_any_device_call():
    """An `out` of another shape than Q would let the kernels write past its
    end; the binding refuses it before reaching the library (checked here on a
    host-only cache with CPU tensors, so nothing is launched)."""
    import torch
    c = pe.PagedKVCache(1, 2, 64, 8, 16, 2, 16, host_only=True)
    s = c.seq_create()
    c.append_kv(s, n_tokens=20)
    q = torch.zeros(4, 4, 64, dtype=torch.bfloat16)
    short = torch.zeros(3, 4, 64, dtype=torch.bfloat16)
    for call in (lambda: c.replay_attn(s, 0, q, out=short),
                 lambda: c.replay_attn_static_scratch(s, 0, q, out=short),
                 lambda: c.replay_attn_batch([s], 0, q, [0, 4], out=short)):
        with pytest.raises(ValueError, match="must match"):
            call()
    c.close()


def test_binding_rejects_tensors_off_the_cache_device():
    """Tensors must live on the cache's device; the check runs before the
    pointer is handed to the library."""
    class FakeCuda:
        dtype = __import__("torch").bfloat16
        is_cuda = True

        class device:
            index = 1

        def is_contiguous(self):
            return True

        def data_ptr(self):
            return 0

    with pytest.raises(ValueError, match="cuda:1, the cache on cuda:0"):
        binding._dev_ptr(FakeCuda(), "Q", 0)
    assert binding._dev_ptr(FakeCuda(), "Q", 1).value is None  # same device: accepted


def test_header_is_plain_c():
    """include/pe.h is a C ABI: it compiles as strict C99 with no warnings,
    so a C caller (no C++ compiler, no CUDA headers) can use it."""
    import shutil
    import subprocess
    import tempfile
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    with tempfile.TemporaryDirectory() as tmp:
        src = os.path.join(tmp, "use_pe.c")
        with open(src, "w") as f:
            f.write('#include "pe.h"\nint main(void) { pe_cache *c = 0; (void)c; return PE_OK; }\n')
        r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-fsyntax-only",
                            "-I", os.path.join(ROOT, "include"), src], capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
