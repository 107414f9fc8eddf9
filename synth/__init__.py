"""Seeded synthetic inputs for the crop + replay path.

This module only draws random numbers and lays out the five workload shapes;
it holds none of the method's arithmetic (no attention, no paging policy).
Tests, the benchmark and the smoke check import it to feed the CUDA library and
the fp64 oracle the very same bf16 bit patterns.

Values are drawn with numpy's PCG64 generator as float32 standard normals,
multiplied by the workload's standard deviation in float32 and rounded once to
bf16 (round-to-nearest-even).  Every independent quantity has its own stream so
that, e.g., the counterfactual suffix of an agent never shares draws with its
original ("contaminated") suffix.

A workload's per-position tensors (K, V, Q of a session) are drawn in blocks
of ``SESSION_BLOCK`` positions of one layer, each block from its own generator
``SeedSequence([base, stream, agent, tensor, layer, block])``.  The value at a
position therefore does not depend on which range of positions is asked for
(the sanitized suffix of any tau is a slice of one sanitized session), and the
blocks are drawn on all host cores at once.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

BASE_SEED = 2609_04875

# Stream identifiers: one independent generator per quantity.
STREAM_PERM = 1          # physical page pop order of the pool
STREAM_KV_ORIG = 2       # K/V of the original session, positions [0, T)
STREAM_KV_CF = 3         # K'/V' of the counterfactual (sanitized) suffix
STREAM_Q_CF = 4          # Q' of the counterfactual suffix
STREAM_LENGTHS = 6       # per-agent T and tau/T (agent batch)
STREAM_SAMPLE = 7        # query rows sampled for large-size checks
STREAM_TURNS = 8         # per-agent turn lengths of the suffix (turn-structured workload)
STREAM_LABELS = 9        # which model turns are independent of the target

# Turn kinds of a turn-structured suffix (labels of the synthetic session; the
# replay policy that reads them lives in the library and in the oracle).
TURN_INPUT = 0           # user message, tool observation or loaded document
TURN_MODEL_INDEP = 1     # model turn causally independent of the target
TURN_MODEL_DEP = 2       # model turn that depends on the target


def rng(seed: int, stream: int, index: int = 0) -> np.random.Generator:
    """Independent generator for (seed, stream, index)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream, index])))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if not np.all(np.isfinite(x)):
        raise ValueError("non-finite value in synthetic draw")
    u = x.view(np.uint32)
    # finite inputs: u + 0x8000 stays below 2^32, so uint32 arithmetic is exact
    r = u >> np.uint32(16)
    r &= np.uint32(1)
    r += np.uint32(0x7FFF)
    r += u
    r >>= np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32 (for host-side inspection)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def normal_bf16(g: np.random.Generator, shape, std: float = 1.0, chunk: int = 1 << 24) -> np.ndarray:
    """i.i.d. N(0, std^2) draws rounded to bf16, as uint16 bits of the given shape."""
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape)) if shape else 1
    out = np.empty(n, dtype=np.uint16)
    s32 = np.float32(std)
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        x = g.standard_normal(hi - lo, dtype=np.float32)
        if std != 1.0:
            x = x * s32
        out[lo:hi] = f32_to_bf16_bits(x)
    return out.reshape(shape)


SESSION_BLOCK = 256      # positions of one layer drawn from one generator


def host_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except (AttributeError, OSError):
        return max(1, os.cpu_count() or 1)


def session_bf16(seed: int, stream: int, index: int, tensor: int, num_layers: int, lo: int, hi: int,
                 width: int, std: float) -> np.ndarray:
    """Positions [lo, hi) of a per-position session tensor, all layers: bf16 bits
    [num_layers][hi - lo][width] of i.i.d. N(0, std^2).  Block b of layer l
    (positions [b B, (b + 1) B), B = SESSION_BLOCK) is drawn whole from
    SeedSequence([seed, stream, index, tensor, l, b]), so a position's value is
    the same whatever range contains it."""
    if not 0 <= lo <= hi:
        raise ValueError("bad position range")
    out = np.empty((num_layers, hi - lo, width), dtype=np.uint16)
    if hi == lo or num_layers == 0 or width == 0:
        return out
    B = SESSION_BLOCK
    s32 = np.float32(std)
    tasks = [(l, b) for l in range(num_layers) for b in range(lo // B, -(-hi // B))]

    def draw(task):
        l, b = task
        g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream, index, tensor, l, b])))
        x = g.standard_normal(B * width, dtype=np.float32)
        if std != 1.0:
            x *= s32
        a, z = max(lo, b * B), min(hi, (b + 1) * B)
        out[l, a - lo:z - lo] = f32_to_bf16_bits(x[(a - b * B) * width:(z - b * B) * width]).reshape(z - a, width)

    n = min(host_threads(), len(tasks))
    if n <= 1:
        for t in tasks:
            draw(t)
    else:
        with ThreadPoolExecutor(max_workers=n) as ex:
            list(ex.map(draw, tasks))
    return out


def page_permutation(seed: int, num_pages: int) -> np.ndarray:
    """A seeded permutation of [0, num_pages): the pool's initial pop order."""
    return rng(seed, STREAM_PERM).permutation(num_pages).astype(np.int32)


def bits_to_torch(bits: np.ndarray):
    """View uint16 bf16 bits as a torch.bfloat16 CPU tensor (no copy)."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def torch_to_bits(t) -> np.ndarray:
    """bf16 torch tensor (any device) -> uint16 numpy bits."""
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


# --------------------------------------------------------------------------
# Workloads.  Notation: page size ps, prefix P = tau-1 kept tokens,
# suffix S = T - tau + 1 recomputed tokens, Hq/Hkv heads, head dim d, L layers.
# --------------------------------------------------------------------------

@dataclass
class Agent:
    T: int            # session length (tokens) before the forget request
    tau: int          # 1-based position of the first tainted token
    index: int        # agent index inside the workload (stream index)
    turns: tuple = ()  # optional suffix turns ((n_tokens, kind), ...) summing to S

    @property
    def P(self) -> int:
        return self.tau - 1

    @property
    def S(self) -> int:
        return self.T - self.tau + 1


@dataclass
class Workload:
    name: str
    seed: int
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    std: float
    agents: list = field(default_factory=list)
    num_pages: int = 0
    softmax_scale: float = 0.0

    def pages_for(self, n_tokens: int) -> int:
        return -(-n_tokens // self.page_size)

    @property
    def total_suffix(self) -> int:
        return sum(a.S for a in self.agents)

    @property
    def max_pages_per_seq(self) -> int:
        return max(self.pages_for(a.T) for a in self.agents)

    def describe(self) -> dict:
        return {
            "workload": self.name,
            "agents": len(self.agents),
            "layers": self.num_layers,
            "q_heads": self.num_q_heads,
            "kv_heads": self.num_kv_heads,
            "head_dim": self.head_dim,
            "page_size": self.page_size,
            "num_pages": self.num_pages,
            "suffix_tokens": self.total_suffix,
            "prefix_tokens": sum(a.P for a in self.agents),
            "seed": self.seed,
        }

    # -- draws ---------------------------------------------------------------
    def _session(self, stream, agent, tensor, lo, hi, heads):
        x = session_bf16(self.seed, stream, agent.index, tensor, self.num_layers, lo, hi, heads * self.head_dim,
                         self.std)
        return x.reshape(self.num_layers, hi - lo, heads, self.head_dim)

    def kv_original(self, agent: Agent):
        """K, V of the original session, positions [0, T): bf16 bits [L][T][Hkv][d] each."""
        return (self._session(STREAM_KV_ORIG, agent, 0, 0, agent.T, self.num_kv_heads),
                self._session(STREAM_KV_ORIG, agent, 1, 0, agent.T, self.num_kv_heads))

    def kv_counterfactual(self, agent: Agent):
        """K', V' of the sanitized suffix, positions [P, T) of the agent's sanitized
        session: bf16 bits [L][S][Hkv][d] each."""
        return (self._session(STREAM_KV_CF, agent, 0, agent.P, agent.T, self.num_kv_heads),
                self._session(STREAM_KV_CF, agent, 1, agent.P, agent.T, self.num_kv_heads))

    def q_counterfactual(self, agent: Agent):
        """Q' of the sanitized suffix, positions [P, T): bf16 bits [L][S][Hq][d]."""
        return self._session(STREAM_Q_CF, agent, 0, agent.P, agent.T, self.num_q_heads)

    def init_free_order(self) -> np.ndarray:
        return page_permutation(self.seed, self.num_pages)


def _finish(w: Workload, slack_pages: int = 64) -> Workload:
    if w.num_pages == 0:
        w.num_pages = sum(w.pages_for(a.T) for a in w.agents) + slack_pages
    if w.softmax_scale == 0.0:
        w.softmax_scale = 1.0 / math.sqrt(w.head_dim)
    return w


def tiny() -> Workload:
    """1 agent, 1 layer, 8/8 heads, d=64, ps=16, 64-page pool; T=640, prefix 512, suffix 128; N(0,1)."""
    w = Workload("tiny", BASE_SEED + 1, 1, 8, 8, 64, 16, 1.0, num_pages=64)
    w.agents = [Agent(T=640, tau=513, index=0)]
    return _finish(w)


def agent_batch(n_agents: int = 16, seed: int = BASE_SEED + 2) -> Workload:
    """16 agents, 1 layer, GQA 32/8, d=128, ps=16; T ~ U{2048..8192}, tau/T ~ U[0.2, 0.9]; N(0,1)/sqrt(128)."""
    w = Workload("agent_batch", seed, 1, 32, 8, 128, 16, 1.0 / math.sqrt(128))
    g = rng(w.seed, STREAM_LENGTHS)
    for i in range(n_agents):
        T = int(g.integers(2048, 8192, endpoint=True))
        r = float(g.uniform(0.2, 0.9))
        P = int(round(r * T))
        w.agents.append(Agent(T=T, tau=P + 1, index=i))
    return _finish(w)


def decode_batch(n_agents: int = 16, seed: int = BASE_SEED + 6) -> Workload:
    """Decode after replay: the 16 agents of the agent batch each generate one
    token (S = 1, P = T - 1): the last position is cropped and recomputed, so
    steps repeat without growing the caches."""
    base = agent_batch(n_agents, seed=seed - 4)  # the agent batch's lengths (seed + 2 <-> + 6)
    w = Workload("decode_batch", seed, 1, 32, 8, 128, 16, 1.0 / math.sqrt(128))
    w.agents = [Agent(T=a.T, tau=a.T, index=i) for i, a in enumerate(base.agents)]
    return _finish(w)


def short_suffix(n_agents: int = 8, prefix: int = 32768, suffix: int = 16) -> Workload:
    """8 agents, GQA 32/8, d=128, ps=16; prefix 32k, suffix 16; N(0,1)/sqrt(128)."""
    w = Workload("short_suffix", BASE_SEED + 3, 1, 32, 8, 128, 16, 1.0 / math.sqrt(128))
    w.agents = [Agent(T=prefix + suffix, tau=prefix + 1, index=i) for i in range(n_agents)]
    return _finish(w)


def long_suffix(n_agents: int = 4, prefix: int = 4096, suffix: int = 16384) -> Workload:
    """4 agents, GQA 64/8, d=128, ps=64; prefix 4k, suffix 16k; N(0,1)/sqrt(128)."""
    w = Workload("long_suffix", BASE_SEED + 4, 1, 64, 8, 128, 64, 1.0 / math.sqrt(128))
    w.agents = [Agent(T=prefix + suffix, tau=prefix + 1, index=i) for i in range(n_agents)]
    return _finish(w)


INDEP_MODEL_TURNS = 4    # model turns in the suffix; the last (the answer) always depends on z


def indep_split(indep: float = 1.0, n_agents: int = 16, seed: int = BASE_SEED + 7) -> Workload:
    """16 agents, 1 layer, GQA 32/8, d=128, ps=16, N(0,1)/sqrt(128); turn-structured suffixes.

    Each agent keeps a clean prefix P ~ U{1024..4096}.  Its suffix starts with
    the (sanitized) acquisition input and alternates model and input turns:
    input, model, input, model, input, model, input, model (the final answer).
    Inputs are U{32..256} tokens, model turns U{64..192}.  Of the three model
    turns before the answer, round(3 * indep) are independent of the target,
    chosen by a seeded per-agent order, so the independent sets grow with
    indep and the lengths do not change."""
    w = Workload(f"indep_split_{indep:g}", seed, 1, 32, 8, 128, 16, 1.0 / math.sqrt(128))
    g = rng(seed, STREAM_LENGTHS)
    n_indep = int(round((INDEP_MODEL_TURNS - 1) * float(indep)))
    if not 0 <= n_indep <= INDEP_MODEL_TURNS - 1:
        raise ValueError("indep must lie in [0, 1]")
    for i in range(n_agents):
        P = int(g.integers(1024, 4096, endpoint=True))
        gt = rng(seed, STREAM_TURNS, i)
        order = rng(seed, STREAM_LABELS, i).permutation(INDEP_MODEL_TURNS - 1)
        indep_turns = set(int(x) for x in order[:n_indep])
        turns = []
        for m in range(INDEP_MODEL_TURNS):
            turns.append((int(gt.integers(32, 256, endpoint=True)), TURN_INPUT))
            kind = TURN_MODEL_INDEP if m in indep_turns else TURN_MODEL_DEP
            turns.append((int(gt.integers(64, 192, endpoint=True)), kind))
        S = sum(n for n, _ in turns)
        w.agents.append(Agent(T=P + S, tau=P + 1, index=i, turns=tuple(turns)))
    return _finish(w)


def replica(w: Workload, r: int) -> Workload:
    """The same workload shape drawn from replica r's own seeds (one replica per
    GPU under weak scaling): the base seed moves by 1000 * r.  The agent batch
    redraws its agents' lengths and injection steps too."""
    seed = w.seed + 1000 * r
    if w.name == "agent_batch":
        return agent_batch(len(w.agents), seed=seed)
    if w.name == "decode_batch":
        return decode_batch(len(w.agents), seed=seed)
    if w.name.startswith("indep_split_"):
        return indep_split(float(w.name[len("indep_split_"):]), len(w.agents), seed=seed)
    import copy
    w2 = copy.deepcopy(w)
    w2.seed = seed
    return w2


def with_std(w: Workload, std: float) -> Workload:
    """The same shapes, lengths and page order with Q/K/V drawn at another
    standard deviation (std 1: logits q.k / sqrt(d) of standard deviation 1,
    a sharper softmax than the workloads' own N(0, 1/128) draws)."""
    import copy
    w2 = copy.deepcopy(w)
    w2.std = float(std)
    w2.name = f"{w.name}_std{std:g}"
    return w2


TAU_SWEEP_RATIOS = (0.1, 0.3, 0.5, 0.7, 0.9)


def tau_sweep(ratio: float, T: int = 16384, num_layers: int = 32) -> Workload:
    """1 agent, 32 layers of GQA 32/8, d=128, ps=16, T=16k; prefix = round(ratio*T).

    ratio = 0 is the full-reset comparator (empty prefix, whole sequence replayed).
    """
    w = Workload(f"tau_sweep_r{ratio:g}", BASE_SEED + 5, num_layers, 32, 8, 128, 16, 1.0 / math.sqrt(128))
    P = int(round(ratio * T))
    w.agents = [Agent(T=T, tau=P + 1, index=0)]
    return _finish(w)


WORKLOADS = {
    "tiny": tiny,
    "agent_batch": agent_batch,
    "decode_batch": decode_batch,
    "short_suffix": short_suffix,
    "long_suffix": long_suffix,
    "indep_split": indep_split,
}


def sample_rows(seed: int, n_q: int, n_random: int, tile_rows: int = 128, index: int = 0) -> np.ndarray:
    """Query rows to check at full size: first/last row, both rows around every
    tile boundary, plus ``n_random`` uniform rows (sorted, unique)."""
    rows = {0, n_q - 1}
    for b in range(tile_rows, n_q, tile_rows):
        rows.add(b - 1)
        rows.add(b)
    g = rng(seed, STREAM_SAMPLE, index)
    if n_q > 0 and n_random > 0:
        rows.update(int(x) for x in g.integers(0, n_q, size=n_random))
    return np.array(sorted(r for r in rows if 0 <= r < n_q), dtype=np.int64)


def provenance_dag(seed: int, n: int, z: int = 9):
    """A session's artifacts in execution order: random parents (up to 3 earlier
    artifacts), token spans of 1-39 tokens laid end to end, one artifact where
    the target z enters, and z inherited by each descendant of a carrier with
    probability 0.7; about 10% of artifacts committed a side effect."""
    g = rng(seed, 0)
    arts, begin, carriers = [], 0, set()
    entry = int(g.integers(0, n))
    for i in range(n):
        k = int(g.integers(0, min(i, 3) + 1))
        parents = sorted({int(x) for x in g.integers(0, i, size=k)}) if i > 0 and k > 0 else []
        length = int(g.integers(1, 40))
        src = []
        if i == entry or (any(p in carriers for p in parents) and g.random() < 0.7):
            src = [z]
            carriers.add(i)
        arts.append(dict(id=i, type=0, parents=parents, sources=src, begin=begin, end=begin + length, turn=i,
                         committed=int(g.random() < 0.1)))
        begin += length
    return arts
