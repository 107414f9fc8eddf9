"""Host-side pieces of bench.py that need no GPU: the workload table, the
algorithmic units, and the kernel-source hashes that keep recorded ncu
traffic valid only for the kernel version it was captured on."""
import os

import bench
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


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
        assert t["kernels"] and all(k in bench.KERNEL_SRC for k in t["kernels"]), wl
        assert set(t["src_sha256"]) == set(t["kernels"]), wl
        assert t["bytes"] > 0 and t["profile"].startswith("profiles/"), wl
        assert os.path.exists(os.path.join(ROOT, t["profile"])), wl


def test_reference_arm_prints_one_contract_line():
    """`bench.py --impl reference` times the fp64 oracle on the host cores and prints one JSON line
    with the contract's keys; it needs no GPU."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1", "--ref-step-budget", "0.3"],
                       capture_output=True, text=True, timeout=300, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["higher_is_better"] is True and d["config"]["workload"] == "tiny"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["cpu_baseline"]["value"] == d["value"] and d["e2e"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["unit"] == d["e2e"]["unit"] == d["cpu_baseline"]["unit"]
    assert "N(0,1^2)" in d["data"]  # the tiny workload draws unscaled N(0, 1) values
    # ms_per_step is the measured wall time of a step's bounded sample, not an extrapolation
    assert d["ms_per_step"] < 5000 and d["full_step_ms_extrapolated"] > 0


def test_option_flag_parses_key_value_pairs():
    import argparse

    import pytest
    assert bench._option("attn_kernel=2") == ("attn_kernel", 2)
    assert bench._option("splitkv=-1") == ("splitkv", -1)
    for bad in ("attn_kernel", "=2", "attn_kernel=x"):
        with pytest.raises((argparse.ArgumentTypeError, ValueError)):
            bench._option(bad)
