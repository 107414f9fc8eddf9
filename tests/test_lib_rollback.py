"""Every call that changes the cache leaves it unchanged when it fails (pe.h:
"On any error the cache state is unchanged"), including a failure of a device
step after the bookkeeping was applied: an append whose kernel launch fails
has already popped its pages and grown the table, a crop has already pushed
its freed pages.  The library's "fail_launch_after" test hook makes the
(k+1)-th device step of a call fail without running; on a host-only cache the
steps a device cache would launch are counted the same way, so the rollback
is checked here on the CPU against the oracle's bookkeeping (the GPU test
tests/test_gpu_rollback.py checks the device mirror and the pool as well)."""
import pytest

import oracle
import synth

pe = pytest.importorskip("paper_2609_04875_gb300")
from paper_2609_04875_gb300 import binding  # noqa: E402


def state(lib, seqs):
    return (lib.free_list(), lib.page_refs(),
            {q: (lib.page_table(q), lib.seq_info(q), lib.checkpoints(q)) for q in seqs})


def oracle_state(orc):
    return (orc.free_list(), list(orc.refs),
            {q: (orc.page_table(q), orc.seq_info(q), list(orc.checkpoints[q])) for q in orc.table})


def with_injected_failures(lib, call, live, max_k=8):
    """Runs `call` with the hook armed at k = 0, 1, ... until it succeeds; after
    every injected failure the state must equal the state before the call.
    Returns (result, number of injected failures)."""
    before = state(lib, live)
    for k in range(max_k):
        lib.set_option("fail_launch_after", k)
        try:
            out = call()
        except binding.PEError as e:
            if "injected" not in str(e):
                lib.set_option("fail_launch_after", -1)
                raise
            assert e.kind == "cuda"
            assert state(lib, live) == before, f"state changed by a call that failed at device step {k}"
            continue
        lib.set_option("fail_launch_after", -1)
        return out, k
    raise AssertionError("the call never succeeded")


@pytest.mark.parametrize("ps", [8, 16])
def test_random_ops_roll_back_injected_failures(ps):
    num_pages, max_pages, max_seqs = 96, 30, 6
    order = synth.page_permutation(91 + ps, num_pages)
    lib = pe.PagedKVCache(1, 1, 64, ps, num_pages, max_seqs, max_pages, init_free_order=order, host_only=True)
    orc = oracle.OracleKVCache(1, 1, 64, ps, num_pages, max_seqs, max_pages, init_free_order=order,
                               store_values=False)
    assert lib.seq_create() == orc.seq_create()
    g = synth.rng(53, ps)
    injected = 0
    for step in range(600):
        live = sorted(orc.table)
        s = live[int(g.integers(0, len(live)))]
        n = orc.length[s]
        r = g.random()

        def both(f_orc, f_lib):
            nonlocal injected
            try:
                want = f_orc()
            except oracle.OracleError as e:
                with pytest.raises(binding.PEError) as pe_err:
                    f_lib()
                assert pe_err.value.kind == e.kind, f"step {step}"
                return
            got, k = with_injected_failures(lib, f_lib, live)
            injected += k
            if got is not None:
                assert got == want, f"step {step}"

        if r < 0.12:
            both(lambda: orc.seq_fork(s), lambda: lib.seq_fork(s))
        elif r < 0.27:
            tau = int(g.integers(1, n + 2))
            both(lambda: orc.crop(s, tau), lambda: lib.crop(s, tau))
        elif r < 0.37:
            taus = [int(g.integers(1, orc.length[q] + 2)) for q in live]
            both(lambda: [orc.crop(q, t) for q, t in zip(live, taus)] and None,
                 lambda: lib.crop_batch(live, taus))
        elif r < 0.45:
            b = int(g.integers(0, n + 1))
            both(lambda: orc.checkpoint_add(s, b), lambda: lib.checkpoint_add(s, b))
        elif r < 0.52:
            tau = int(g.integers(1, n + 3))
            both(lambda: orc.restore(s, tau), lambda: lib.restore(s, tau))
        elif r < 0.58 and len(live) > 1:
            both(lambda: orc.seq_release(s), lambda: lib.seq_release(s))
        elif r < 0.75:
            ks = [int(g.integers(0, 2 * ps)) for _ in live]
            cu = [0]
            for k in ks:
                cu.append(cu[-1] + k)

            def orc_batch():
                need = sum(orc.pages_for(orc.length[q] + k) - len(orc.table[q]) for q, k in zip(live, ks))
                if need > len(orc.free):
                    raise oracle.OracleError("oom", "batch")
                for q, k in zip(live, ks):
                    orc.append(q, n_tokens=k)
            both(orc_batch, lambda: lib.append_kv_batch(live, cu_tokens=cu))
        else:
            k = int(g.integers(0, 3 * ps))
            both(lambda: orc.append(s, n_tokens=k), lambda: lib.append_kv(s, n_tokens=k))
        assert state(lib, sorted(orc.table)) == oracle_state(orc), f"step {step}"
    assert injected > 100, injected


def test_every_device_step_of_a_multi_launch_call_rolls_back():
    """65 sequences: a batched append needs two append launches (64 segments
    each at most) and copy-on-write launches for the shared last pages of the
    forks; a batched crop of all of them is one launch.  A failure injected at
    each of those steps leaves the state unchanged; the call then succeeds and
    matches the oracle."""
    ps, num_pages, n = 8, 400, 65
    order = synth.page_permutation(5, num_pages)
    lib = pe.PagedKVCache(1, 1, 64, ps, num_pages, 2 * n, 16, init_free_order=order, host_only=True)
    orc = oracle.OracleKVCache(1, 1, 64, ps, num_pages, 2 * n, 16, init_free_order=order, store_values=False)
    base = lib.seq_create()
    orc.seq_create()
    lib.append_kv(base, n_tokens=13)
    orc.append(base, n_tokens=13)
    seqs = [base]
    for _ in range(n - 1):           # forks share the partially filled last page
        seqs.append(lib.seq_fork(base))
        orc.seq_fork(base)
    ks = [3 + (i % 5) for i in range(n)]
    cu = [0]
    for k in ks:
        cu.append(cu[-1] + k)
    _, failures = with_injected_failures(lib, lambda: lib.append_kv_batch(seqs, cu_tokens=cu), seqs, max_k=200)
    for q, k in zip(seqs, ks):
        orc.append(q, n_tokens=k)
    assert failures >= 2 + (n - 1)     # two append launches and the copy-on-write steps
    assert state(lib, seqs) == oracle_state(orc)
    taus = [1 + (i % 7) for i in range(n)]
    _, failures = with_injected_failures(lib, lambda: lib.crop_batch(seqs, taus), seqs)
    for q, t in zip(seqs, taus):
        orc.crop(q, t)
    assert failures == 1
    assert state(lib, seqs) == oracle_state(orc)


def test_rounds_roll_back_as_a_whole():
    """pe_replay_rounds appends round by round; a failure in a later round also
    undoes the rounds already applied."""
    ps = 8
    order = synth.page_permutation(9, 64)
    lib = pe.PagedKVCache(1, 1, 64, ps, 64, 3, 20, init_free_order=order, host_only=True)
    a, b = lib.seq_create(), lib.seq_create()
    lib.append_kv(a, n_tokens=10)
    lib.append_kv(b, n_tokens=21)
    take = [[5, 3], [1, 0], [0, 4], [6, 1]]
    cu = [0, 12, 20]
    _, failures = with_injected_failures(lib, lambda: lib.replay_rounds([a, b], take, cu), [a, b])
    assert failures == 4               # every round has work: one append launch each
    assert lib.seq_info(a) == (22, 22) and lib.seq_info(b) == (29, 29)  # no crop yet: every append counts


def test_hook_option_is_checked():
    lib = pe.PagedKVCache(1, 1, 64, 8, 8, 1, 8, host_only=True)
    with pytest.raises(binding.PEError) as e:
        lib.set_option("fail_launch_after", -2)
    assert e.value.kind == "invalid"
