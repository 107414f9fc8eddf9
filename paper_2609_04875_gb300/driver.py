"""Forget-request driver over the C-ABI: turns a workload of agents, each with
its injection step tau, into the calls of the replay path.

For every agent the original session (T positions, suffix contaminated) is
first written into one shared paged cache.  One `step()` then performs, for
all agents at once:
  1. crop to tau (Alg. 1 Restore; keeps tau-1 tokens)       -> pe_crop_batch
  2. append the sanitized suffix K'/V' (T-tau+1 positions)   -> pe_append_kv_batch
  3. replay attention of the suffix queries Q', per layer    -> pe_replay_attn_batch
After a step every agent again holds T tokens, so steps repeat without reset.
All inputs are device-resident bf16 tensors; the driver only orders the calls.
"""
from __future__ import annotations

import numpy as np
import torch

from .binding import PagedKVCache


def _dev(bits: np.ndarray, device) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(device)


class ReplayDriver:
    """Device-resident crop + replay of a synthetic workload (``synth.Workload``)."""

    def __init__(self, w, device="cuda", fill=True, cache_kwargs=None, inputs=None):
        """inputs: optional {agent index: (k0, v0, kc, vc, qc)} host bf16 bits, as
        drawn by the workload; drawn here when absent."""
        self.w = w
        self.device = torch.device(device)
        L, hq, hkv, d = w.num_layers, w.num_q_heads, w.num_kv_heads, w.head_dim
        # twice the agents' sequence slots: room for one branch (fork) of every agent
        self.cache = PagedKVCache(L, hkv, d, w.page_size, w.num_pages, max_seqs=2 * len(w.agents),
                                  max_pages_per_seq=w.max_pages_per_seq, init_free_order=w.init_free_order(),
                                  **(cache_kwargs or {}))
        self.seqs = [self.cache.seq_create() for _ in w.agents]
        self.taus = [a.tau for a in w.agents]
        S = [a.S for a in w.agents]
        self.cu = [0] + list(np.cumsum(S).astype(int))
        n = self.cu[-1]
        # (twice the agents' sequence slots: room for a branch of every agent)
        # sanitized suffix inputs, packed over agents: K'/V' [L][sum S][Hkv][d], Q' [L][sum S][Hq][d]
        self.Kc = torch.empty((L, n, hkv, d), dtype=torch.bfloat16, device=self.device)
        self.Vc = torch.empty_like(self.Kc)
        self.Qc = torch.empty((L, n, hq, d), dtype=torch.bfloat16, device=self.device)
        self._inputs = inputs
        for i, a in enumerate(w.agents):
            if inputs is not None:
                _, _, k, v, q = inputs[i]
            else:
                (k, v), q = w.kv_counterfactual(a), w.q_counterfactual(a)
            lo, hi = self.cu[i], self.cu[i + 1]
            self.Kc[:, lo:hi] = _dev(k, self.device)
            self.Vc[:, lo:hi] = _dev(v, self.device)
            self.Qc[:, lo:hi] = _dev(q, self.device)
            del k, v, q
        self.out = torch.empty_like(self.Qc)
        if fill:
            self.fill_original()

    def fill_original(self):
        """Writes every agent's original session (T positions) in agent order."""
        for i, (s, a) in enumerate(zip(self.seqs, self.w.agents)):
            k, v = self._inputs[i][:2] if self._inputs is not None else self.w.kv_original(a)
            self.cache.append_kv(s, _dev(k, self.device), _dev(v, self.device))
            del k, v
        torch.cuda.synchronize(self.device)

    # -- the hot path ------------------------------------------------------------
    def buffers(self):
        """The step's device buffers (K', V', Q', out)."""
        return self.Kc, self.Vc, self.Qc, self.out

    def crop(self, stream=None):
        self.cache.crop_batch(self.seqs, self.taus, stream=stream)

    def append(self, stream=None, bufs=None):
        K, V = (bufs or self.buffers())[:2]
        self.cache.append_kv_batch(self.seqs, K, V, self.cu, stream=stream)

    def attend(self, layer, stream=None, bufs=None):
        Q, out = (bufs or self.buffers())[2:]
        self.cache.replay_attn_batch(self.seqs, layer, Q[layer], self.cu, out=out[layer],
                                     softmax_scale=self.w.softmax_scale, stream=stream)

    def step(self, stream=None, attn_events=None, bufs=None):
        """One forget request for every agent.  attn_events: optional list of
        (start, end) CUDA event pairs, one per layer, recorded around attention.
        bufs: optional (K', V', Q', out) device tensors shaped like buffers()."""
        self.crop(stream)
        self.append(stream, bufs)
        for layer in range(self.w.num_layers):
            if attn_events is not None:
                attn_events[layer][0].record(stream)
            self.attend(layer, stream, bufs)
            if attn_events is not None:
                attn_events[layer][1].record(stream)
        return (bufs or self.buffers())[3]

    # -- bookkeeping -------------------------------------------------------------
    def algorithmic_flops(self) -> float:
        """4 d Hq sum_agents L [S P + S (S + 1) / 2]: unmasked (query, key) pairs x 2d for
        QK^T and 2d for PV."""
        w = self.w
        pairs = sum(a.S * a.P + a.S * (a.S + 1) / 2 for a in w.agents)
        return 4.0 * w.head_dim * w.num_q_heads * w.num_layers * pairs

    def algorithmic_attn_bytes(self) -> float:
        """Bytes one attention launch per layer must move: every cached K/V row of
        each kv-head read once (prefix + suffix), Q read, O written."""
        w = self.w
        keys = sum(a.T for a in w.agents)
        q = sum(a.S for a in w.agents)
        return 2.0 * (2 * keys * w.num_kv_heads * w.head_dim + 2 * q * w.num_q_heads * w.head_dim)

    def algorithmic_step_bytes(self) -> float:
        """Per step, all layers: prefix K/V read + new K/V read and written + Q read + O written."""
        w = self.w
        P = sum(a.P for a in w.agents)
        S = sum(a.S for a in w.agents)
        per_layer = 2.0 * (2 * P * w.num_kv_heads * w.head_dim + 4 * S * w.num_kv_heads * w.head_dim
                           + 2 * S * w.num_q_heads * w.head_dim)
        return per_layer * w.num_layers
