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

`RoundsDriver` replays turn-structured suffixes instead: after the crop, one
pe_replay_rounds call runs the lockstep rounds of a replay policy (known turns
re-prefilled, the others re-decoded one position per round; Sec. 4.5).
"""
from __future__ import annotations

import numpy as np
import torch

from .binding import PagedKVCache, i32_array, i64_array


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
        # the ids of every step's calls, converted once
        self._seqs_c, self._taus_c, self._cu_c = i32_array(self.seqs), i64_array(self.taus), i32_array(self.cu)
        n = self.cu[-1]
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
        self._prepared = {}
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

    def _calls(self, stream, bufs):
        """The step's C-ABI calls for (stream, buffer set), validated and marshalled
        once (binding.prepare_*): crop, append, one attention call per layer."""
        from .binding import _stream
        key = (_stream(stream).value,  # the stream the calls will use (the current one when None)
               None if bufs is None else tuple(t.data_ptr() for t in bufs))
        calls = self._prepared.get(key)
        if calls is None:
            K, V, Q, out = bufs or self.buffers()
            c = self.cache
            st = key[0]
            calls = (c.prepare_crop_batch(self._seqs_c, self._taus_c, stream=st),
                     c.prepare_append_kv_batch(self._seqs_c, K, V, self._cu_c, stream=st),
                     [c.prepare_replay_attn_batch(self._seqs_c, layer, Q[layer], self._cu_c, out[layer],
                                                  softmax_scale=self.w.softmax_scale, stream=st)
                      for layer in range(self.w.num_layers)])
            self._prepared[key] = calls
        return calls

    def crop(self, stream=None):
        self._calls(stream, None)[0]()

    def append(self, stream=None, bufs=None):
        self._calls(stream, bufs)[1]()

    def attend(self, layer, stream=None, bufs=None):
        self._calls(stream, bufs)[2][layer]()

    def step(self, stream=None, attn_events=None, bufs=None):
        """One forget request for every agent.  attn_events: optional list of
        (start, end) CUDA event pairs, one per layer, recorded around attention.
        bufs: optional (K', V', Q', out) device tensors shaped like buffers()."""
        crop, append, attend = self._calls(stream, bufs)
        crop()
        append()
        if attn_events is None:
            for call in attend:
                call()
        else:
            for layer, call in enumerate(attend):
                attn_events[layer][0].record(stream)
                call()
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


class RoundsDriver(ReplayDriver):
    """Replay of a turn-structured workload (agents carry ``turns``) with the
    indep split (Sec. 4.5): one step crops every agent to tau and then runs
    the rounds of ``policy`` (selective replay or the prefix-cache comparator)
    through pe_replay_rounds, all layers, in one library call."""

    def __init__(self, w, policy, device="cuda", **kw):
        super().__init__(w, device, **kw)
        self.set_policy(policy)

    def set_policy(self, policy):
        from .binding import replay_schedule
        self.policy = policy
        self.take, self.decode_tokens = replay_schedule([a.turns for a in self.w.agents], policy)

    @property
    def rounds(self) -> int:
        return int(self.take.shape[0])

    def step(self, stream=None, attn_events=None, bufs=None):
        K, V, Q, out = bufs or self.buffers()
        self.crop(stream)
        self.cache.replay_rounds(self._seqs_c, self.take, self._cu_c, K, V, Q, out, softmax_scale=self.w.softmax_scale,
                                 stream=stream)
        return out

    # -- the same rounds through the per-round public calls, for timing attention alone
    def round_buffers(self):
        """Per round: (seqs, cu, K, V, Q, out) with the round's rows gathered and packed."""
        done = [0] * len(self.seqs)
        per_round = []
        for r in range(self.rounds):
            seqs, cu, idx = [], [0], []
            for i, s in enumerate(self.seqs):
                t = int(self.take[r, i])
                if t == 0:
                    continue
                lo = self.cu[i] + done[i]
                idx.extend(range(lo, lo + t))
                seqs.append(s)
                cu.append(cu[-1] + t)
                done[i] += t
            ix = torch.tensor(idx, dtype=torch.long, device=self.device)
            per_round.append((seqs, cu, self.Kc.index_select(1, ix).contiguous(),
                              self.Vc.index_select(1, ix).contiguous(), self.Qc.index_select(1, ix).contiguous(),
                              torch.empty((self.w.num_layers, len(idx), self.w.num_q_heads, self.w.head_dim),
                                          dtype=torch.bfloat16, device=self.device)))
        return per_round

    def step_per_round(self, per_round, stream=None, attn_events=None, gate_cycles=0):
        """crop, then per round: pe_append_kv_batch and one pe_replay_attn_batch per
        layer; attn_events[r] = (start, end) recorded around round r's attention.
        gate_cycles > 0 enqueues a fixed-length busy kernel (torch.cuda._sleep)
        before each start event, so that the host has queued the round's
        launches before the GPU reaches them and the events time the kernels,
        not the host."""
        self.crop(stream)
        for r, (seqs, cu, K, V, Q, out) in enumerate(per_round):
            self.cache.append_kv_batch(seqs, K, V, cu, stream=stream)
            if attn_events is not None:
                if gate_cycles > 0:
                    with torch.cuda.stream(stream or torch.cuda.current_stream(self.device)):
                        torch.cuda._sleep(int(gate_cycles))
                attn_events[r][0].record(stream)
            for layer in range(self.w.num_layers):
                self.cache.replay_attn_batch(seqs, layer, Q[layer], cu, out=out[layer],
                                             softmax_scale=self.w.softmax_scale, stream=stream)
            if attn_events is not None:
                attn_events[r][1].record(stream)

    def round_work(self):
        """Per round: (algorithmic FLOPs, algorithmic bytes) of its attention,
        all layers: unmasked (query, key) pairs x 4d x Hq; every key of the
        round's agents read once per kv-head, their Q read and O written."""
        w = self.w
        lens = [a.P for a in w.agents]
        work = []
        for r in range(self.rounds):
            fl = by = 0.0
            for i in range(len(self.seqs)):
                t = int(self.take[r, i])
                if t == 0:
                    continue
                lens[i] += t
                n = lens[i]
                fl += 4.0 * w.head_dim * w.num_q_heads * (t * (n - t) + t * (t + 1) / 2)
                by += 2.0 * (2 * n * w.num_kv_heads * w.head_dim + 2 * t * w.num_q_heads * w.head_dim)
            work.append((fl * w.num_layers, by * w.num_layers))
        return work
