"""Host-side pieces of bench.py that need no GPU: the workload table, the
algorithmic units, and the kernel-source hashes that keep recorded ncu
traffic valid only for the kernel version it was captured on."""
import bench
import synth


def test_every_named_workload_builds():
    for name in ["tiny", "agent_batch", "decode_batch", "short_suffix", "long_suffix", "tau_sweep_r0.7",
                 "tau_sweep_r0", "indep_split_1", "indep_split_0.5"]:
        w = bench.make_workload(name)
        assert w.agents and w.num_layers >= 1, name


def test_algorithmic_units_match_closed_forms():
    w = synth.tiny()
    a = w.agents[0]
    # 4 d Hq [S P + S (S + 1) / 2] FLOP per layer
    assert bench.workload_flops(w) == 4.0 * w.head_dim * w.num_q_heads * w.num_layers * (
        a.S * a.P + a.S * (a.S + 1) / 2)
    assert bench.attn_bytes(w) > 0


def test_kernel_source_spans_are_found():
    # the hashed spans must exist, or recorded traffic would silently lapse for every kernel
    for kernel in bench.KERNEL_SRC:
        h = bench._src_sha(kernel)
        assert h is not None and len(h) == 64, kernel
    for wl, t in bench.NCU_TRAFFIC.items():
        assert t.get("kernel", "prefill") in bench.KERNEL_SRC, wl
        assert t["bytes"] > 0 and t["profile"].startswith("profiles/"), wl
