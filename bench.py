"""Benchmark of the crop + suffix replay path on GB300.

One step = one forget request for every agent of a workload: batched crop to
tau, batched append of the sanitized suffix K'/V', and batched causal replay
attention of the suffix queries per layer, all through the C-ABI library.

Default (`--workload suite`): the five workload configurations, each measured
on its own, in the `configs` block of one JSON line; the headline is the
largest of them, the tau sweep (1 agent, 32 layers of GQA 32/8, d = 128,
T = 16384, tau/T in {0.1, 0.3, 0.5, 0.7, 0.9}): one step replays the five
forget requests back to back, and the full-reset comparator (the whole
counterfactual sequence recomputed from an empty cache) is timed beside it.
`--workload <name>` measures one workload alone.

`value` = suffix tokens replayed per second over the whole job, inputs
resident in HBM; `e2e` = the same with the step's inputs copied from pinned
host memory and the outputs read back inside the timed region; `roofline` =
the replay-attention kernel's algorithmic FLOP (or byte) rate over the
measured peak; `cpu_baseline` = the fp64 CPU oracle timed on a bounded sample
of the same workload.

`--impl reference` times the oracle alone (the reference arm).
Multi-GPU (torchrun): every rank runs its own replica of the workload
(agents are independent; no collective on the data path), weak scaling.
"""
from __future__ import annotations

import argparse
import contextlib
import gc
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "suffix replay tokens/sec & % of roofline (BF16 peak / HBM BW); crop latency µs"
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# The five workload configurations, in the order they are measured; the last is the headline.
SUITE = [
    ("tiny", "config 1: 1 agent, 1 layer, 8/8 heads, d 64, ps 16, prefix 512, suffix 128, N(0,1)"),
    ("agent_batch", "config 2: 16 agents, 1 layer, GQA 32/8, d 128, ps 16, T ~ U{2048..8192}, tau/T ~ U[0.2,0.9]"),
    ("short_suffix", "config 3: 8 agents, GQA 32/8, d 128, ps 16, prefix 32768, suffix 16 (split-KV)"),
    ("long_suffix", "config 4: 4 agents, GQA 64/8, d 128, ps 64, prefix 4096, suffix 16384"),
    ("tau_sweep", "config 5: 1 agent, 32 layers of GQA 32/8, d 128, ps 16, T 16384, tau/T in "
                  "{0.1,0.3,0.5,0.7,0.9}, one step = the five forget requests; full reset beside it"),
]


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def make_workload(name, replica=0):
    """agent_batch | tiny | decode_batch | short_suffix | long_suffix | tau_sweep_r<ratio> (ratio 0 =
    full reset) | indep_split[_<indep>] (turn-structured suffixes; indep defaults to 1).
    replica r > 0 (the rank under torchrun) draws the same shapes from its own seeds."""
    if name.startswith("tau_sweep_r"):
        w = synth.tau_sweep(float(name[len("tau_sweep_r"):]))
    elif name.startswith("indep_split_"):
        w = synth.indep_split(float(name[len("indep_split_"):]))
    else:
        w = synth.WORKLOADS[name]()
    if replica:
        w = synth.replica(w, replica)
    return w


def reduce_max(x, dist):
    """Max over ranks (gloo, on the host) of a float; identity without a process group."""
    if not dist:
        return x
    import torch
    import torch.distributed as tdist
    t = torch.tensor([x], dtype=torch.float64)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist:
        import torch.distributed as tdist
        tdist.barrier()


def workload_flops(w):
    """4 d Hq L sum_agents [S P + S (S + 1) / 2]: unmasked (query, key) pairs x 2d
    for Q K^T and 2d for P V, all layers."""
    pairs = sum(a.S * a.P + a.S * (a.S + 1) / 2 for a in w.agents)
    return 4.0 * w.head_dim * w.num_q_heads * w.num_layers * pairs


def attn_bytes(w):
    """Algorithmic bytes of one attention launch (one layer): every cached K/V
    row of each kv-head read once, Q read, O written (bf16)."""
    keys = sum(a.T for a in w.agents)
    q = sum(a.S for a in w.agents)
    return 2.0 * (2 * keys * w.num_kv_heads * w.head_dim + 2 * q * w.num_q_heads * w.head_dim)


def step_bytes(w):
    """Algorithmic bytes of one step, all layers (append + attention): prefix K/V
    read once per kv-head, new K/V read and written, Q read, O written."""
    P = sum(a.P for a in w.agents)
    S = sum(a.S for a in w.agents)
    per_layer = 2.0 * (2 * P * w.num_kv_heads * w.head_dim + 4 * S * w.num_kv_heads * w.head_dim
                       + 2 * S * w.num_q_heads * w.head_dim)
    return per_layer * w.num_layers


def median(x):
    return statistics.median(x) if x else None


# ------------------------------------------------------------------ clocks
@contextlib.contextmanager
def no_gc():
    """A timed region without Python's cyclic garbage collector (a collection pass would land
    inside the region).  No collection is forced before it either: after one, the host loop of
    a small step ran markedly slower."""
    gc.disable()
    try:
        yield
    finally:
        gc.enable()


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------ workloads as units
class OracleSource:
    """Host arrays of one agent's counterfactual sequence for the oracle:
    per layer the retained prefix of the original session followed by the
    sanitized suffix, and the suffix queries."""

    def __init__(self, w, agent, arrays):
        self.w, self.agent, self._arrays = w, agent, arrays

    def layer(self, layer):
        k0, v0, kc, vc, qc = self._arrays()
        P = self.agent.P
        return (np.concatenate([k0[layer, :P], kc[layer]], 0), np.concatenate([v0[layer, :P], vc[layer]], 0),
                qc[layer])


def oracle_sources(w, shared=None):
    """One OracleSource per agent.  shared = (k0, v0, ks, vs, qs): the agent's
    original and sanitized sessions over all T positions (one agent), so the
    suffix arrays are slices and nothing is redrawn."""
    if shared is not None:
        k0, v0, ks, vs, qs = shared
        a = w.agents[0]
        return [OracleSource(w, a, lambda a=a: (k0, v0, ks[:, a.P:], vs[:, a.P:], qs[:, a.P:]))]
    cache = {}

    def arrays(i):
        if i not in cache:
            a = w.agents[i]
            cache.clear()
            cache[i] = (*w.kv_original(a), *w.kv_counterfactual(a), w.q_counterfactual(a))
        return cache[i]
    return [OracleSource(w, a, lambda i=i: arrays(i)) for i, a in enumerate(w.agents)]


def sweep_sessions(replica=0):
    """The tau sweep's forget requests share one session: the original K/V
    (positions [0, T)) and the sanitized K'/V'/Q' of every position; the
    request at tau/T = r keeps the original's first round(r T) positions and
    replays the sanitized rest.  Returns ({ratio: workload}, full-reset
    workload, (k0, v0, ks, vs, qs))."""
    ws = {r: synth.tau_sweep(r) for r in synth.TAU_SWEEP_RATIOS}
    w_full = synth.tau_sweep(0.0)
    if replica:
        ws = {r: synth.replica(w, replica) for r, w in ws.items()}
        w_full = synth.replica(w_full, replica)
    a = w_full.agents[0]
    k0, v0 = w_full.kv_original(a)
    ks, vs = w_full.kv_counterfactual(a)   # P = 0: the sanitized session, every position
    qs = w_full.q_counterfactual(a)
    return ws, w_full, (k0, v0, ks, vs, qs)


class Unit:
    """One workload on its own ReplayDriver (cache, device inputs, output)."""

    def __init__(self, label, w, drv, oracle_src):
        self.label, self.w, self.drv, self.oracle_src = label, w, drv, oracle_src
        self.L = w.num_layers
        self.S = w.total_suffix
        self.flops_step = workload_flops(w)
        self.flops_launch = self.flops_step / self.L
        self.bytes_launch = attn_bytes(w)
        self.bytes_step = step_bytes(w)


def build_units(name, replica, device):
    """(units, comparator unit or None, shared host sessions or None)."""
    from paper_2609_04875_gb300.driver import ReplayDriver
    if name == "tau_sweep":
        ws, w_full, shared = sweep_sessions(replica)
        k0, v0, ks, vs, qs = shared
        units = []
        for r, w in ws.items():
            P = w.agents[0].P
            drv = ReplayDriver(w, device=device, inputs={0: (k0, v0, ks[:, P:], vs[:, P:], qs[:, P:])})
            units.append(Unit(f"tau/T={r:g}", w, drv, oracle_sources(w, shared)))
        drv = ReplayDriver(w_full, device=device, inputs={0: (k0, v0, ks, vs, qs)})
        comp = Unit("full reset", w_full, drv, oracle_sources(w_full, shared))
        return units, comp, shared
    w = make_workload(name, replica)
    return [Unit(name, w, ReplayDriver(w, device=device), oracle_sources(w))], None, None


# ------------------------------------------------------------------ CPU oracle
def oracle_tokens_per_s(units, budget_s, seed=7):
    """fp64 oracle on a bounded, uniformly random sample of the units' suffix
    tokens (all heads, all layers): returns (tokens/s, cores, sample text,
    wall seconds of oracle work).  Only the oracle calls are timed; building
    a layer's key array (a concatenation) is not."""
    import oracle
    cores = oracle.num_cpus()
    g = synth.rng(seed, synth.STREAM_SAMPLE, 999)
    srcs = [s for u in units for s in u.oracle_src]
    weights = np.array([s.agent.S for s in srcs], dtype=np.float64)
    weights /= weights.sum()
    done, spent = 0, 0.0
    batch = 2
    while spent < budget_s:
        src = srcs[int(g.choice(len(srcs), p=weights))]
        w, a = src.w, src.agent
        rows = np.sort(g.integers(0, a.S, size=batch))
        for layer in range(w.num_layers):
            keys, vals, q = src.layer(layer)
            t0 = time.perf_counter()
            oracle.causal_attention(q, keys, vals, w.softmax_scale, rows=rows)
            spent += time.perf_counter() - t0
        done += batch
        batch = max(1, min(256, int(batch * 1.5)))
    names = sorted({s.w.name for s in srcs})
    sample = (f"{done} suffix tokens drawn uniformly over the suffixes of {len(srcs)} sequence(s) "
              f"({', '.join(names)}), all heads x layers, fp64 oracle, {spent:.1f} s")
    return done / spent, cores, sample, spent


# ------------------------------------------------------------------ recorded ncu traffic
# DRAM traffic per attention launch from one ncu capture (profiles/), valid only
# while the kernel source is the one that was captured.
NCU_TRAFFIC = {
    "tiny": {"bytes": 1.5081e6, "profile": "profiles/traffic_attention_configs.md", "kernels": ["prefill"],
             "src_sha256": {"prefill": "91bcdf4963eaa5385a46b5fc32b465f5b50af0d236a020b33013751418d6a9b6"}},
    "agent_batch": {"bytes": 684.646e6 + 315.236e6, "profile": "profiles/traffic_attention_configs.md",
                    "kernels": ["prefill"], "src_sha256": {"prefill": "91bcdf4963eaa5385a46b5fc32b465f5b50af0d236a020b33013751418d6a9b6"}},
    "short_suffix": {"bytes": 1.0883e9 + 5.88058e6, "profile": "profiles/traffic_attention_configs.md",
                     "kernels": ["prefill_sk"], "src_sha256": {"prefill_sk": "b25d958540e6002039fda210f04a46af7fb34514ee9402af13b2c16be2709172"}},
    "long_suffix": {"bytes": 1.41056e9 + 1.0372e9, "profile": "profiles/traffic_attention_configs.md",
                    "kernels": ["prefill"], "src_sha256": {"prefill": "91bcdf4963eaa5385a46b5fc32b465f5b50af0d236a020b33013751418d6a9b6"}},
    # one sweep step's 224 attention launches (5 forget requests x 32 layers, two launches per layer where a
    # tail launch runs), per layer: bytes / 160
    "tau_sweep": {"bytes": (48092.5e6 + 8159.95e6) / 160, "profile": "profiles/traffic_attention_configs.md",
                  "kernels": ["prefill", "prefill_sk"], "src_sha256": {"prefill": "91bcdf4963eaa5385a46b5fc32b465f5b50af0d236a020b33013751418d6a9b6", "prefill_sk": "b25d958540e6002039fda210f04a46af7fb34514ee9402af13b2c16be2709172"}},
    "decode_batch": {"bytes": 341.569792e6 + 3.933952e6, "profile": "profiles/decode_tc_decode_batch.md",
                     "kernels": ["decode"],
                     "src_sha256": {"decode": "a29203afa92b6d3d8108227a2ee31a613331b3c42dd2904b8ef84b5de69006ab"}},
}
CSRC = os.path.join(ROOT, "paper_2609_04875_gb300", "csrc")
# (file, first line of the kernel's source, the text that follows it): the span that is hashed
KERNEL_SRC = {
    "prefill": ("pe_attn.cu", "template <int HD, bool SPLIT>\n__global__", "// Exercises the bounded wait on its own"),
    "prefill_sk": ("pe_attn_sk.cu", "// Merge of one row of a cut unit's q-tile", "template <int HD>\ncudaError_t launch_sk_t("),
    "decode": ("pe_decode.cu", "template <int HD, int RB>\n__global__ void __launch_bounds__(kTcThreads, 1)",
               "template <int HD, int RB>\ncudaError_t launch_tc("),
}


def _src_sha(kernel="prefill"):
    """sha256 of a kernel function's source, so that recorded counters lapse
    when the kernel changes."""
    import hashlib
    name, start, end = KERNEL_SRC[kernel]
    with open(os.path.join(CSRC, name)) as f:
        txt = f.read()
    try:
        a = txt.index(start)
        b = txt.index(end, a)
    except ValueError:
        return None
    return hashlib.sha256(txt[a:b].encode()).hexdigest()


def traffic_for(workload):
    """Recorded DRAM bytes per attention launch of `workload`, or None when any
    kernel it launches has changed since the capture."""
    t = NCU_TRAFFIC.get(workload)
    if not t or any(t["src_sha256"][k] != _src_sha(k) for k in t["kernels"]):
        return None, None
    return t["bytes"], t["profile"]


# ------------------------------------------------------------------ roofline
def peaks_of(peaks):
    return (float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])),
            float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])),
            float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])))


def roofline(flops, nbytes, seconds, peaks, peak_src):
    """Roofline of `flops` FLOP and `nbytes` algorithmic bytes done in `seconds`:
    the slower of the two at the measured peaks decides the bound."""
    tflops, gbs, sus = peaks_of(peaks)
    t_flop = flops / (tflops * 1e12)
    t_hbm = nbytes / (gbs * 1e9)
    if t_flop >= t_hbm:
        r = {"bound": "tensor", "achieved": flops / seconds / 1e12, "peak": tflops, "unit": "TFLOP/s",
             "peak_source": f"bf16_tflops (burst) of {peak_src}"}
        r["frac"] = r["achieved"] / r["peak"]
        r["frac_of_sustained"] = r["achieved"] / sus
    else:
        r = {"bound": "hbm", "achieved": nbytes / seconds / 1e9, "peak": gbs, "unit": "GB/s",
             "peak_source": f"hbm_gbs of {peak_src}"}
        r["frac"] = r["achieved"] / r["peak"]
    r["roofline_s"] = max(t_flop, t_hbm)
    return r


def kernel_name(w, plan):
    rows = max(a.S for a in w.agents) * (w.num_q_heads // w.num_kv_heads)
    if rows <= 16:  # every sequence's query rows fit the decode kernel
        rb = 4 if rows <= 4 else (8 if rows <= 8 else 16)
        return f"decode_tc_kernel<{w.head_dim},{rb}> (+ decode_tc_combine_kernel<{w.head_dim},{rb}> for split items)"
    return f"replay_attn_kernel<{w.head_dim},{'split' if plan[0] else 'single'}> (+ splitkv_combine when split)"


# ------------------------------------------------------------------ GPU timing passes
def timed_pass(units, steps, stream, dist):
    """`steps` steps of every unit back to back, inputs resident in HBM.  Events
    on the launching stream bracket each attention launch, and each unit's step
    when there are several units (the sweep's requests); a lone unit's step time
    is the region's.  Few events per step, so that a host-bound step (the tiny
    configuration) is not slowed by them.  Returns the elapsed ms (max over
    ranks), the per-unit event times and the library's launch count."""
    import torch
    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    many = len(units) > 1
    ev = [[((E(), E()) if many else None, [(E(), E()) for _ in range(u.L)]) for _ in range(steps)] for u in units]
    calls = [u.drv._calls(None, None) for u in units]  # the step's prepared C-ABI calls
    launches0 = sum(u.drv.cache.kernel_launches() for u in units)
    barrier(dist)
    torch.cuda.synchronize()
    t0, t1 = E(), E()
    with no_gc():
        t0.record(stream)
        for k in range(steps):
            for (crop, append, attend), e in zip(calls, ev):
                se, attn = e[k]
                if many:
                    se[0].record(stream)
                crop()
                append()
                for layer, call in enumerate(attend):
                    attn[layer][0].record(stream)
                    call()
                    attn[layer][1].record(stream)
                if many:
                    se[1].record(stream)
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(dist)
    launches = sum(u.drv.cache.kernel_launches() for u in units) - launches0
    elapsed = t0.elapsed_time(t1)
    per_unit = []
    for u, e in zip(units, ev):
        per_unit.append({
            "step_ms": [se[0].elapsed_time(se[1]) for se, _ in e] if many else [elapsed / steps],
            "attn_ms": [b.elapsed_time(c) for _, at in e for b, c in at],
        })
    return reduce_max(elapsed, dist), per_unit, launches


def gated_pass(units, reps, stream):
    """Kernel times without host gaps: before each timed section a busy kernel
    (torch.cuda._sleep) holds the stream while the host enqueues the section's
    launches, so the events bracket device work only.  Also the host time of
    the crop call (GPU idle, synchronised before the call).  Each rep is one
    full step per unit (crop and append restore the same state)."""
    import torch
    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    cyc_us = 2000  # busy-kernel cycles per microsecond (SM clock about 2 GHz)
    out = []
    for u in units:
        drv = u.drv
        host_crop, crop, app, attn = [], [], [], []
        for _ in range(reps):
            torch.cuda.synchronize()
            h0 = time.perf_counter()
            drv.crop()
            h1 = time.perf_counter()
            drv.append()
            for layer in range(u.L):
                drv.attend(layer)
            torch.cuda.synchronize()
            host_crop.append((h1 - h0) * 1e6)
            e = [E() for _ in range(6)]
            torch.cuda._sleep(150 * cyc_us)
            e[0].record(stream)
            drv.crop()
            e[1].record(stream)
            torch.cuda._sleep(150 * cyc_us)
            e[2].record(stream)
            drv.append()
            e[3].record(stream)
            torch.cuda._sleep((100 + 40 * u.L) * cyc_us)
            e[4].record(stream)
            for layer in range(u.L):
                drv.attend(layer)
            e[5].record(stream)
            torch.cuda.synchronize()
            crop.append(e[0].elapsed_time(e[1]) * 1e3)
            app.append(e[2].elapsed_time(e[3]))
            attn.append(e[4].elapsed_time(e[5]))
        out.append({"crop_host_us": median(host_crop), "crop_kernel_us": median(crop), "append_ms": median(app),
                    "attn_ms_all_layers": median(attn)})
    return out


def unit_report(u, t, gated, peaks, peak_src, steps):
    """Numbers of one unit from its timed-pass events `t` and gated times (the
    append's device time comes from the gated pass)."""
    ms_step = statistics.mean(t["step_ms"])
    attn_launch_s = statistics.mean(t["attn_ms"]) / 1e3
    app_ms = gated["append_ms"]
    kern = roofline(u.flops_launch, u.bytes_launch, attn_launch_s, peaks, peak_src)
    attn_step_ms = attn_launch_s * 1e3 * u.L
    step = roofline(u.flops_step, u.bytes_step, (app_ms + attn_step_ms) / 1e3, peaks, peak_src)
    gk = roofline(u.flops_launch, u.bytes_launch, gated["attn_ms_all_layers"] / 1e3 / u.L, peaks, peak_src)
    plan = u.drv.cache.last_attn_plan()
    return {
        "value": u.S / (ms_step / 1e3), "unit": UNIT, "steps": steps, "ms_per_step": ms_step,
        "suffix_tokens": u.S, "prefix_tokens": sum(a.P for a in u.w.agents), "layers": u.L,
        "kernel": kernel_name(u.w, plan),
        "plan": {"split_kv": bool(plan[0]), "key_splits": plan[1], "ctas": plan[2]},
        "attn_ms_per_launch": attn_launch_s * 1e3,
        "algorithmic_flop_per_launch": u.flops_launch,
        "algorithmic_bytes_per_launch": u.bytes_launch,
        "units_per_launch": {"agents": len(u.w.agents), "suffix_tokens": u.S,
                             "keys": sum(a.T for a in u.w.agents)},
        "roofline_ms_per_launch": kern["roofline_s"] * 1e3,
        "kernel_frac": kern["frac"], "kernel_frac_of_sustained": kern.get("frac_of_sustained"),
        "kernel_bound": kern["bound"],
        "kernel_achieved": kern["achieved"], "kernel_unit": kern["unit"],
        # the step fraction: roofline time of append + attention over their measured device time
        "step_frac": step["frac"], "step_bound": step["bound"], "step_roofline_ms": step["roofline_s"] * 1e3,
        "append_ms": app_ms, "attention_ms_all_layers": attn_step_ms,
        "gated": {**gated, "attn_ms_per_launch": gated["attn_ms_all_layers"] / u.L, "kernel_frac": gk["frac"]},
    }


# ------------------------------------------------------------------ end to end with host buffers
PINNED_COPY_GBS = 330.0  # pinned host<->device copy rate, both directions at once, measured on a GB300


def _copy_rows(dst, src):
    """dst <- src (same shape, non-blocking): one copy when both are contiguous,
    else one per leading index (each leading slice is contiguous)."""
    if dst.is_contiguous() and src.is_contiguous():
        dst.copy_(src, non_blocking=True)
    else:
        for i in range(dst.shape[0]):
            dst[i].copy_(src[i], non_blocking=True)


def run_e2e(units, dev, steps, world, dist, step_ms, host=None):
    """The same step through the public API with the step's inputs (K', V', Q')
    in pinned host memory: every step copies each unit's inputs host->device,
    runs its crop + append + replay and copies its output device->host.
    Copies run on their own streams and overlap other units' and steps'
    compute.  host: per unit (K, V, Q, O) pinned host tensors shaped like the
    unit's device buffers (a tau-sweep unit's are views of the shared pinned
    session); default: pinned copies of the device inputs.  Buffer sets: a
    second device set per unit lets one unit's copies run while another set
    computes; a lone unit whose copies take at least half its step gets four,
    so its input copy waits only for the output copy four steps back.  The
    timed region spans the first input copy to the last output copy."""
    import torch
    if host is None:
        host = []
        for u in units:
            K, V, Q, O = u.drv.buffers()
            host.append((K.cpu().pin_memory(), V.cpu().pin_memory(), Q.cpu().pin_memory(),
                         torch.empty(O.shape, dtype=O.dtype).pin_memory()))
    h2d = sum(h[0].numel() + h[1].numel() + h[2].numel() for h in host) * 2
    d2h = sum(h[3].numel() for h in host) * 2
    copy_ms = (h2d + d2h) / (PINNED_COPY_GBS * 1e9) * 1e3
    nb = 4 if len(units) == 1 and copy_ms >= 0.5 * step_ms else 2
    sets = []
    for u in units:
        own = u.drv.buffers()
        sets.append([own] + [tuple(torch.empty_like(x) for x in own) for _ in range(nb - 1)])
    comp = torch.cuda.current_stream(dev)
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    free = [[torch.cuda.Event() for _ in range(nb)] for _ in units]
    ready = [[torch.cuda.Event() for _ in range(nb)] for _ in units]
    done = [[torch.cuda.Event() for _ in range(nb)] for _ in units]
    for f in free:
        for e in f:
            e.record(comp)

    def one(i, k):
        b = k % nb
        bufs = sets[i][b]
        hK, hV, hQ, hO = host[i]
        s_in.wait_event(free[i][b])
        with torch.cuda.stream(s_in):
            for dst, src in zip(bufs[:3], (hK, hV, hQ)):
                _copy_rows(dst, src)
            ready[i][b].record(s_in)
        comp.wait_event(ready[i][b])
        units[i].drv.step(bufs=bufs)
        done[i][b].record(comp)
        s_out.wait_event(done[i][b])
        with torch.cuda.stream(s_out):
            _copy_rows(hO, bufs[3])
            free[i][b].record(s_out)

    for k in range(nb + 1):
        for i in range(len(units)):
            one(i, k)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with no_gc():
        e0.record(comp)
        s_in.wait_stream(comp)
        for k in range(steps):
            for i in range(len(units)):
                one(i, k)
        comp.wait_stream(s_out)
        e1.record(comp)
        torch.cuda.synchronize(dev)
    ms = reduce_max(e0.elapsed_time(e1), dist)
    tokens = world * sum(u.S for u in units) * steps
    return {"value": tokens / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps, "ms_per_step": ms / steps,
            "overlap": f"{nb} device buffer sets per sequence group: copies of other groups and steps overlap "
                       "the compute"}


# ------------------------------------------------------------------ one workload / the suite
def measure(name, args, rank, world, local_rank, dev, peaks, peak_src, headline):
    """Builds the workload's units, warms up, runs the timed pass (args.steps for
    the headline; enough steps for at least args.min_timed_s otherwise), the
    gated pass, and for the headline the end-to-end pass and host-side
    latencies.  Returns (report, units, comparator, shared sessions)."""
    import torch
    stream = torch.cuda.current_stream(dev)
    dist = world > 1
    units, comp, shared = build_units(name, rank, dev)
    for u in units + ([comp] if comp else []):
        for key, val in args.set:
            u.drv.cache.set_option(key, val)
    for _ in range(args.warmup):
        for u in units:
            u.drv.step()
    torch.cuda.synchronize(dev)
    steps = args.steps
    if not headline:
        t0 = time.perf_counter()
        for u in units:
            u.drv.step()
        torch.cuda.synchronize(dev)
        est = max(time.perf_counter() - t0, 1e-6)
        steps = max(args.steps, min(20000, int(math.ceil(args.min_timed_s / est))))
        steps = int(reduce_max(steps, dist))
    clocks = ClockSampler(local_rank) if rank == 0 else None
    if clocks:
        clocks.start()
    elapsed_ms, per_unit, launches = timed_pass(units, steps, stream, dist)
    clk = clocks.stop() if clocks else None
    gated = gated_pass(units, args.gated_reps, stream)
    reports = [unit_report(u, t, g, peaks, peak_src, steps) for u, t, g in zip(units, per_unit, gated)]
    S_step = sum(u.S for u in units)
    ms_per_step = elapsed_ms / steps
    rep = {
        "value": world * S_step * steps / (elapsed_ms / 1e3), "unit": UNIT, "steps": steps,
        "ms_per_step": ms_per_step, "suffix_tokens_per_step": S_step, "gpu_launches": launches, "clocks": clk,
    }
    # the attention kernel over every launch of the step, and the step fraction (append + attention)
    attn_s = sum(statistics.mean(t["attn_ms"]) / 1e3 * u.L for u, t in zip(units, per_unit))
    flops = sum(u.flops_step for u in units)
    n_launch = sum(u.L for u in units)
    kern = roofline(flops, sum(u.bytes_launch * u.L for u in units), attn_s, peaks, peak_src)
    step_meas = sum(r["append_ms"] + r["attention_ms_all_layers"] for r in reports)
    step_roof = sum(r["step_roofline_ms"] for r in reports)
    gated_attn = sum(g["attn_ms_all_layers"] for g in gated)
    kern_g = roofline(flops, sum(u.bytes_launch * u.L for u in units), gated_attn / 1e3, peaks, peak_src)
    rep["roofline"] = {
        "bound": kern["bound"], "achieved": kern["achieved"], "peak": kern["peak"], "unit": kern["unit"],
        "frac": kern["frac"], "peak_source": kern["peak_source"],
        "frac_of_sustained": kern.get("frac_of_sustained"),
        "kernel": reports[0]["kernel"] if len(reports) == 1 else
        "replay_attn_kernel<128,*> (+ splitkv_combine when split); one launch per layer and forget request",
        "attn_ms_per_launch": attn_s * 1e3 / n_launch,
        "algorithmic_flop_per_launch": flops / n_launch,
        "algorithmic_bytes_per_launch": sum(u.bytes_launch * u.L for u in units) / n_launch,
        "launches_per_step": n_launch,
        "roofline_ms_per_launch": kern["roofline_s"] * 1e3 / n_launch,
        "step_frac": step_roof / step_meas,
        "step_frac_definition": "roofline time of append + attention (max of FLOP at bf16 peak, step bytes at "
                                "HBM peak) over their measured device time (attention: the timed region's "
                                "events; append: the busy-gated pass)",
        "gated_frac": kern_g["frac"],
        "gated_definition": "the same attention launches timed behind a busy kernel, so no host gap is inside "
                            "the events",
    }
    tr, prof = traffic_for(name)
    rep["roofline"]["traffic"], rep["roofline"]["traffic_profile"] = tr, prof
    if len(units) == 1:
        rep["roofline"]["plan"] = reports[0]["plan"]
        rep["roofline"]["units_per_launch"] = reports[0]["units_per_launch"]
        rep.update({k: reports[0][k] for k in ("append_ms", "attention_ms_all_layers")})
    else:
        rep["roofline"]["units_per_launch"] = {
            "requests": len(units), "suffix_tokens": sum(u.S for u in units),
            "keys": sum(a.T for u in units for a in u.w.agents), "layers": units[0].L,
            "note": "per-launch figures are means over the step's launches (one per layer and request)"}
        rep["per_request"] = {u.label: r for u, r in zip(units, reports)}
    rep["crop_us"] = {"kernel_median": median([g["crop_kernel_us"] for g in gated]),
                      "host_call_median": median([g["crop_host_us"] for g in gated]),
                      "agents_per_call": len(units[0].w.agents),
                      "how": "kernel: CUDA events behind a busy kernel (device time only); host: the C-ABI call "
                             "with the GPU idle"}
    if comp is not None:
        rep["comparator"] = measure_comparator(comp, units, reports, args, rank, local_rank, stream, dist,
                                               peaks, peak_src)
    return rep, units, comp, shared


def measure_comparator(comp, units, reports, args, rank, local_rank, stream, dist, peaks, peak_src):
    """Full reset: the whole counterfactual sequence (T positions) recomputed
    from an empty cache, on the same session, timed like the sweep's requests."""
    import torch
    for _ in range(args.warmup):
        comp.drv.step()
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank) if rank == 0 else None
    if clocks:
        clocks.start()
    _, per_unit, _ = timed_pass([comp], args.steps, stream, dist)
    clk = clocks.stop() if clocks else None
    g = gated_pass([comp], args.gated_reps, stream)[0]
    r = unit_report(comp, per_unit[0], g, peaks, peak_src, args.steps)
    T = comp.w.agents[0].T
    r["clocks"] = clk
    r["vs_selective_replay"] = {
        u.label: {"recomputed_token_ratio": T / u.S, "wall_time_speedup": r["ms_per_step"] / ur["ms_per_step"],
                  "attention_flop_ratio": comp.flops_step / u.flops_step}
        for u, ur in zip(units, reports)}
    return r


def run_pe(args, rank, world, local_rank):
    import torch

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_src = load_peaks()
    names = [n for n, _ in SUITE] if args.workload == "suite" else [args.workload]
    head_name = names[-1]
    configs = {}
    head = None
    for name in names:
        headline = name == head_name
        rep, units, comp, shared = measure(name, args, rank, world, local_rank, dev, peaks, peak_src, headline)
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            budget = args.cpu_budget if headline else args.cpu_budget_other
            tps, cores, sample, _ = oracle_tokens_per_s(units, budget)
            rep["cpu_baseline"] = {"value": tps, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample}
        elif rank == 0:
            rep["cpu_baseline"] = None
        if headline:
            if not args.no_e2e:
                host = None
                if shared is not None:  # the sweep: one pinned copy of the shared sessions serves every request
                    _, _, ks, vs, qs = shared
                    hK, hV, hQ = (synth.bits_to_torch(x).pin_memory() for x in (ks, vs, qs))
                    hO = torch.empty(hQ.shape, dtype=torch.bfloat16).pin_memory()
                    host = [(hK[:, u.w.agents[0].P:], hV[:, u.w.agents[0].P:], hQ[:, u.w.agents[0].P:],
                             hO[:, u.w.agents[0].P:]) for u in units]
                rep["e2e"] = run_e2e(units, dev, min(args.steps, args.e2e_steps), world, world > 1,
                                     rep["ms_per_step"], host)
            else:
                rep["e2e"] = None
            rep.update(host_latencies(units, dev))
            head = (name, rep, units)
        else:
            del units, comp, shared
            gc.collect()
            torch.cuda.empty_cache()
        desc = dict(SUITE).get(name, name)
        configs[name] = {"description": desc, **rep}
    name, rep, units = head
    w = units[0].w
    cfg = {**w.describe(), "workload": name if name != "tau_sweep" else "tau_sweep",
           "description": dict(SUITE).get(name, name),
           "parallelism": f"replicas x{world} (independent agents, no collective)",
           "l2": "inputs larger than L2 (KV cache %.0f MB per GPU, L2 129 MB)" % (
               sum(sum(a.T for a in u.w.agents) * u.w.num_kv_heads * u.w.head_dim * 4 * u.w.num_layers
                   for u in units) / 1e6)}
    if len(units) > 1:
        cfg["requests"] = {u.label: {"prefix_tokens": u.w.agents[0].P, "suffix_tokens": u.S} for u in units}
        cfg["suffix_tokens"] = sum(u.S for u in units)
        cfg.pop("prefix_tokens", None)
        cfg.pop("seed", None)
        cfg["seed"] = w.seed
    result = {
        "metric": METRIC,
        "value": rep["value"],
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": rep["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": f"synthetic (seeded N(0,{w.std:.4g}^2) bf16 Q/K/V; no dataset)",
        "config": dict(cfg, **({"options": dict(args.set)} if args.set else {})),
        "roofline": rep["roofline"],
        "cpu_baseline": rep.get("cpu_baseline"),
        "clocks": rep["clocks"],
        "e2e": rep["e2e"],
        "gpu_launches": rep["gpu_launches"],
        "crop_us": rep["crop_us"],
        "recomputed_tokens": rep["suffix_tokens_per_step"],
        "session_tokens": sum(a.T for u in units for a in u.w.agents),
    }
    for k in ("comparator", "per_request", "append_ms", "attention_ms_all_layers", "fork_us",
              "provenance_query_us"):
        if k in rep:
            result[k] = rep[k]
    if len(configs) > 1:
        result["configs"] = {k: {kk: vv for kk, vv in v.items() if kk not in ("fork_us", "provenance_query_us")}
                             for k, v in configs.items()}
    if rank == 0:
        print(json.dumps(result), flush=True)


def host_latencies(units, dev):
    """Host-side calls of the path around the replay: fork + release of every
    agent of the first unit, and provenance queries on a 100k-artifact graph."""
    import torch
    drv = units[0].drv
    fork_us, rel_us = [], []
    for _ in range(10):
        torch.cuda.synchronize(dev)
        h0 = time.perf_counter()
        forks = [drv.cache.seq_fork(s) for s in drv.seqs]
        h1 = time.perf_counter()
        for f in forks:
            drv.cache.seq_release(f)
        h2 = time.perf_counter()
        fork_us.append((h1 - h0) * 1e6 / len(forks))
        rel_us.append((h2 - h1) * 1e6 / len(forks))
    torch.cuda.synchronize(dev)
    from paper_2609_04875_gb300 import ProvenanceGraph
    arts = synth.provenance_dag(units[0].w.seed, 100000)
    pg = ProvenanceGraph()
    for a in arts:
        pg.add(a["id"], a["type"], a["parents"], a["sources"], a["begin"], a["end"], a["turn"], a["committed"])
    h0 = time.perf_counter()
    src = pg.locate_source(9)
    closure, _ = pg.taint_closure(src)
    tau_q = pg.first_entry(src)
    prov_us = (time.perf_counter() - h0) * 1e6
    pg.close()
    return {"fork_us": {"host_per_fork_median": median(fork_us), "host_per_release_median": median(rel_us)},
            "provenance_query_us": {"artifacts": len(arts), "closure": len(closure), "tau": tau_q,
                                    "locate_closure_first_entry": prov_us}}


def run_rounds(args, rank, world, local_rank):
    """Turn-structured workload: one step = crop every agent to tau, then the
    lockstep rounds of selective replay (known turns re-prefilled, dependent
    model turns re-decoded one position per round) in one pe_replay_rounds
    call.  The prefix-cache comparator (every model turn re-decoded) runs on
    the same cache and inputs and is reported beside it."""
    import torch

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2609_04875_gb300.binding import POLICY_PREFIX_CACHE, POLICY_SELECTIVE
    from paper_2609_04875_gb300.driver import RoundsDriver

    w = make_workload(args.workload, replica=rank)
    drv = RoundsDriver(w, POLICY_SELECTIVE, device=dev)
    stream = torch.cuda.current_stream(dev)
    dist = world > 1
    tokens_per_step = w.total_suffix

    def barrier():
        if dist:
            import torch.distributed as tdist
            tdist.barrier()

    def timed(policy, steps, clocks=None):
        drv.set_policy(policy)
        for _ in range(args.warmup):
            drv.step()
        torch.cuda.synchronize(dev)
        if clocks:
            clocks.start()
        l0 = drv.cache.kernel_launches()
        barrier()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with no_gc():
            e0.record(stream)
            for _ in range(steps):
                drv.step()
            e1.record(stream)
            torch.cuda.synchronize(dev)
        barrier()
        clk = clocks.stop() if clocks else None
        return reduce_max(e0.elapsed_time(e1), dist) / steps, drv.cache.kernel_launches() - l0, clk

    clocks = ClockSampler(local_rank) if rank == 0 else None
    ms_sel, launches, clk = timed(POLICY_SELECTIVE, args.steps, clocks)
    sel = {"rounds": drv.rounds, "decode_tokens": drv.decode_tokens, "ms_per_step": ms_sel}
    comp_steps = max(3, min(args.steps, 50))
    ms_pc, _, _ = timed(POLICY_PREFIX_CACHE, comp_steps)
    comp = {"policy": "prefix_cache (full reset + prefix cache: every model turn of the suffix re-decoded)",
            "rounds": drv.rounds, "decode_tokens": drv.decode_tokens, "ms_per_step": ms_pc,
            "steps": comp_steps, "value": world * tokens_per_step / (ms_pc / 1e3)}

    # attention alone, per round (same kernels and plans through the per-round calls)
    drv.set_policy(POLICY_SELECTIVE)
    per_round = drv.round_buffers()
    work = drv.round_work()
    for _ in range(3):
        drv.step_per_round(per_round)
    n_inst = 3
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in per_round] for _ in range(n_inst)]
    for k in range(n_inst):  # ~200 us gate per round: the events time kernels, not host calls
        drv.step_per_round(per_round, attn_events=ev[k], gate_cycles=400_000)
    torch.cuda.synchronize(dev)
    t_round = [statistics.median(ev[k][r][0].elapsed_time(ev[k][r][1]) for k in range(n_inst)) / 1e3
               for r in range(len(per_round))]
    peaks, peak_src = load_peaks()
    tflops = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    gbs = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    roof_t = [max(f / (tflops * 1e12), b / (gbs * 1e9)) for f, b in work]
    hbm_rounds = [r for r, (f, b) in enumerate(work) if b / (gbs * 1e9) >= f / (tflops * 1e12)]
    ten_rounds = [r for r in range(len(work)) if r not in set(hbm_rounds)]
    t_hbm_total = sum(roof_t[r] for r in hbm_rounds)
    t_ten_total = sum(roof_t[r] for r in ten_rounds)
    if t_hbm_total >= t_ten_total:
        rs = hbm_rounds
        achieved = sum(work[r][1] for r in rs) / sum(t_round[r] for r in rs) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": gbs, "unit": "GB/s",
                "peak_source": f"hbm_gbs of {peak_src}"}
    else:
        rs = ten_rounds
        achieved = sum(work[r][0] for r in rs) / sum(t_round[r] for r in rs) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": tflops, "unit": "TFLOP/s",
                "peak_source": f"bf16_tflops (burst) of {peak_src}"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = None
    roof["kernel"] = (f"replay_attn_kernel<{w.head_dim},*> (+ splitkv_combine) for prefill rounds, "
                      "decode_tc_kernel for decode rounds; one launch group per round")
    roof["rounds_counted"] = len(rs)
    roof["frac_all_rounds"] = sum(roof_t) / sum(t_round)
    roof["attn_ms_all_rounds"] = sum(t_round) * 1e3
    roof["roofline_ms_all_rounds"] = sum(roof_t) * 1e3

    e2e = None
    if not args.no_e2e:
        drv.set_policy(POLICY_SELECTIVE)
        e2e = run_e2e([Unit(w.name, w, drv, oracle_sources(w))], dev, min(args.steps, args.e2e_steps), world,
                      dist, ms_sel)
    value = world * tokens_per_step / (ms_sel / 1e3)
    result = {
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_sel,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": f"synthetic (seeded N(0,{w.std:.4g}^2) bf16 Q/K/V, seeded turn lengths and labels; no dataset)",
        "config": {
            **w.describe(),
            "policy": "selective (known turns re-prefilled, target-dependent model turns re-decoded)",
            "parallelism": f"replicas x{world} (independent agents, no collective)",
            "l2": "KV cache %.0f MB per GPU (L2 129 MB); each round re-reads its agents' keys" % (
                sum(a.T for a in w.agents) * w.num_kv_heads * w.head_dim * 4 * w.num_layers / 1e6),
        },
        "selective": sel,
        "comparator": comp,
        "speedup_vs_prefix_cache": ms_pc / ms_sel,
        "roofline": roof,
        "recomputed_tokens": tokens_per_step,
        "gpu_launches": launches,
        "clocks": clk,
        "e2e": e2e,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        tps, cores, sample, _ = oracle_tokens_per_s([Unit(w.name, w, drv, oracle_sources(w))], args.cpu_budget)
        result["cpu_baseline"] = {"value": tps, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample}
    elif rank == 0:
        result["cpu_baseline"] = None
    if rank == 0:
        print(json.dumps(result), flush=True)


# ------------------------------------------------------------------ reference arm
def reference_units(name):
    """The workload's oracle sources without any GPU state (the reference arm)."""
    class _U:
        pass
    units = []
    if name == "tau_sweep":
        ws, _, shared = sweep_sessions()
        for r, w in ws.items():
            u = _U()
            u.w, u.S, u.oracle_src = w, w.total_suffix, oracle_sources(w, shared)
            units.append(u)
        return units
    w = make_workload(name)
    u = _U()
    u.w, u.S, u.oracle_src = w, w.total_suffix, oracle_sources(w)
    return [u]


def run_reference(args, rank, world):
    """The fp64 CPU oracle, timed as it stands on the host cores, on the same
    workload as the GPU arm's headline; each step is a bounded sample of it
    (about --ref-step-budget seconds of oracle work), and ms_per_step is that
    sample's measured wall time.  The time a whole step of the workload would
    take at the sampled rate is reported separately, labelled as an
    extrapolation."""
    if rank != 0:
        return
    name = SUITE[-1][0] if args.workload == "suite" else args.workload
    units = reference_units(name)
    S_step = sum(u.S for u in units)
    for _ in range(args.warmup):
        oracle_tokens_per_s(units, 0.2, seed=11)
    tokens, spent, walls, samples, cores = 0.0, 0.0, [], [], None
    for k in range(args.steps):
        w0 = time.perf_counter()
        tps, cores, sample, sec = oracle_tokens_per_s(units, args.ref_step_budget, seed=100 + k)
        walls.append((time.perf_counter() - w0) * 1e3)
        tokens += tps * sec
        spent += sec
        samples.append(sample)
    value = tokens / spent
    w = units[0].w
    cfg = {**w.describe(), "workload": name, "description": dict(SUITE).get(name, name),
           "parallelism": "host cores (oracle)"}
    if len(units) > 1:
        cfg["requests"] = {f"tau/T={r:g}": {"prefix_tokens": u.w.agents[0].P, "suffix_tokens": u.S}
                           for r, u in zip(synth.TAU_SWEEP_RATIOS, units)}
        cfg["suffix_tokens"] = S_step
        cfg.pop("prefix_tokens", None)
    result = {
        "impl": "reference",
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": statistics.mean(walls),
        "ms_per_step_meaning": "measured wall time of one step's bounded sample of the workload",
        "full_step_ms_extrapolated": 1e3 * S_step / value,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": f"synthetic (seeded N(0,{w.std:.4g}^2) bf16 Q/K/V; no dataset)",
        "config": cfg,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"per step: {samples[-1]}"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(result), flush=True)


def _option(text):
    key, sep, val = text.partition("=")
    if not sep or not key:
        raise argparse.ArgumentTypeError(f"expected KEY=VALUE, got {text!r}")
    return key, int(val)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["pe", "reference"], default="pe")
    ap.add_argument("--workload", default="suite",
                    help="suite (the five configurations; headline: the tau sweep) | tau_sweep | agent_batch | "
                         "tiny | decode_batch | short_suffix | long_suffix | tau_sweep_r<ratio> | "
                         "indep_split[_<indep>]")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=100)
    ap.add_argument("--gated-reps", type=int, default=5, help="repetitions of the busy-gated kernel timing")
    ap.add_argument("--min-timed-s", type=float, default=0.3,
                    help="minimum timed region of a non-headline configuration (more steps when short)")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--cpu-budget-other", type=float, default=3.0,
                    help="seconds of oracle work for each non-headline configuration's cpu_baseline")
    ap.add_argument("--ref-step-budget", type=float, default=2.0, help="seconds of oracle work per reference step")
    ap.add_argument("--set", action="append", default=[], type=_option, metavar="KEY=VALUE",
                    help="a cache option (pe_cache_set_option) applied to every workload cache, e.g. attn_kernel=2; "
                         "named in config.options")
    args = ap.parse_args()

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch.distributed as tdist
        tdist.init_process_group("gloo")
    try:
        if args.workload.startswith("indep_split"):
            run_rounds(args, rank, world, local_rank)
        else:
            run_pe(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as tdist
            tdist.destroy_process_group()


if __name__ == "__main__":
    main()
