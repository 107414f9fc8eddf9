"""Oracle: the paged KV cache's state (exact integers and bf16 bit patterns).

TEST INFRASTRUCTURE ONLY: imported by the tests, the smoke check and the
benchmark's CPU-baseline leg, never by the product path.  Written from the
paper and the stated allocation policy; it shares no code with the CUDA
library.

Paper objects followed:
  * crop = restore (Sec. 3.4(b): a checkpoint holds a token offset, and
    cropping the cache is restoring it; Alg. 1, Restore: "crop KV to c*");
  * with every token position a crop point, c* = tau - 1: crop keeps the
    tau - 1 tokens before the first tainted one (Lemma 1: those states are the
    counterfactual's own; Lemma 2: nothing at or after tau may be kept);
  * replay re-materialises the sanitized suffix by prefill on the cropped cache
    (Sec. 3.2), one appended token position per transition, so the number of
    tokens appended since the crop is the recomputation count T - tau + 1 of
    Corollary 1.

Allocation policy (the paper is silent; this is the reading both sides follow):
  * the free list is a LIFO stack; its initial pop order is ``init_free_order``
    (first element popped first), default 0..num_pages-1;
  * append pops one page per new logical page, in logical order;
  * crop / release push the removed pages in DESCENDING logical order, so the
    lowest removed logical page ends on top and is the next one popped;
  * a partially kept page stays in the table; its slots past the new length are
    stale and are overwritten by the next append;
  * sequence ids: the lowest id not in use.

Branching from one base ("cache cloned", Sec. 4.1) and checkpoints (Sec. 3.4(b)):
  * fork(seq) gives a new sequence sharing every page (reference counts);
  * crop / release drop one reference per removed page; a page returns to the
    free list (same descending push order) only when its last reference goes;
  * an append into a partially filled page that another sequence also holds
    first copies that page's valid slots into a freshly popped page
    (copy-on-write), then pops the new logical pages;
  * checkpoints are token offsets b (the state after the first b tokens,
    metadata only); Restore(c*) takes c* = the largest offset b < tau (Alg. 1:
    argmax over boundaries before tau) and crops to keep b tokens.  A crop
    drops the checkpoints past the new length; a fork copies them.
Pool layout: per layer [num_pages][Hkv][page_size][d] bf16 for K and for V.
"""
from __future__ import annotations

import numpy as np


class OracleError(Exception):
    """Raised for the error cases of the crop / append / query rules."""

    def __init__(self, kind: str, msg: str):
        super().__init__(f"{kind}: {msg}")
        self.kind = kind  # "invalid" | "range" | "oom"


class OracleKVCache:
    def __init__(self, num_layers, num_kv_heads, head_dim, page_size, num_pages,
                 max_seqs, max_pages_per_seq, init_free_order=None, store_values=True):
        self.L = int(num_layers)
        self.Hkv = int(num_kv_heads)
        self.d = int(head_dim)
        self.ps = int(page_size)
        self.num_pages = int(num_pages)
        self.max_seqs = int(max_seqs)
        self.max_pages_per_seq = int(max_pages_per_seq)
        order = list(range(self.num_pages)) if init_free_order is None else [int(p) for p in init_free_order]
        if sorted(order) != list(range(self.num_pages)):
            raise OracleError("invalid", "init_free_order is not a permutation of the pool")
        # stack: top is the END of the python list; first popped = order[0]
        self.free = list(reversed(order))
        self.refs = [0] * self.num_pages        # sequences holding each page
        self.table: dict[int, list[int]] = {}
        self.length: dict[int, int] = {}
        self.appended: dict[int, int] = {}
        self.checkpoints: dict[int, list[int]] = {}
        self.store_values = store_values
        if store_values:
            shape = (self.L, self.num_pages, self.Hkv, self.ps, self.d)
            self.k_pool = np.zeros(shape, dtype=np.uint16)
            self.v_pool = np.zeros(shape, dtype=np.uint16)

    # -- helpers -----------------------------------------------------------
    def pages_for(self, n_tokens: int) -> int:
        return -(-n_tokens // self.ps)

    def _check_seq(self, seq):
        if seq not in self.table:
            raise OracleError("invalid", f"unknown sequence {seq}")

    # -- sequences -----------------------------------------------------------
    def _free_slot(self) -> int:
        for s in range(self.max_seqs):
            if s not in self.table:
                return s
        raise OracleError("oom", "no free sequence slot")

    def seq_create(self) -> int:
        s = self._free_slot()
        self.table[s] = []
        self.length[s] = 0
        self.appended[s] = 0
        self.checkpoints[s] = []
        return s

    def _drop(self, pages) -> list[int]:
        """Drop one reference per page, visiting them in descending logical order;
        returns the pages that reached zero (ascending logical order) after
        pushing them onto the free list."""
        freed = []
        for p in reversed(pages):
            self.refs[p] -= 1
            if self.refs[p] == 0:
                self.free.append(p)
                freed.append(p)
        return list(reversed(freed))

    def seq_release(self, seq) -> list[int]:
        """Drop every page of ``seq`` (like a crop to tau = 1) and the slot."""
        self._check_seq(seq)
        freed = self._drop(self.table[seq])
        del self.table[seq], self.length[seq], self.appended[seq], self.checkpoints[seq]
        return freed

    def seq_fork(self, seq) -> int:
        """A new sequence sharing all of ``seq``'s pages, length and checkpoints."""
        self._check_seq(seq)
        s = self._free_slot()
        self.table[s] = list(self.table[seq])
        for p in self.table[s]:
            self.refs[p] += 1
        self.length[s] = self.length[seq]
        self.appended[s] = self.appended[seq]
        self.checkpoints[s] = list(self.checkpoints[seq])
        return s

    # -- checkpoints (metadata only) -------------------------------------------
    def checkpoint_add(self, seq, offset):
        self._check_seq(seq)
        if not 0 <= offset <= self.length[seq]:
            raise OracleError("range", f"checkpoint offset {offset} outside [0, {self.length[seq]}]")
        if offset not in self.checkpoints[seq]:
            self.checkpoints[seq] = sorted(self.checkpoints[seq] + [offset])

    def checkpoint_select(self, seq, tau) -> int:
        """c* = the largest checkpoint offset b < tau."""
        self._check_seq(seq)
        if tau < 1:
            raise OracleError("invalid", f"tau = {tau} < 1")
        cands = [b for b in self.checkpoints[seq] if b < tau]
        if not cands:
            raise OracleError("range", f"no checkpoint before tau = {tau}")
        return max(cands)

    def restore(self, seq, tau):
        """Restore(c*): crop to the selected checkpoint; returns (offset, freed)."""
        b = self.checkpoint_select(seq, tau)
        if tau - 1 > self.length[seq]:
            raise OracleError("range", f"tau - 1 = {tau - 1} exceeds length {self.length[seq]}")
        return b, self.crop(seq, b + 1)

    # -- crop (Alg. 1, Restore) ----------------------------------------------
    def crop(self, seq, tau) -> list[int]:
        """Keep the first tau-1 tokens; return the freed pages in ascending logical order."""
        self._check_seq(seq)
        if tau < 1:
            raise OracleError("invalid", f"tau = {tau} < 1")
        n = self.length[seq]
        if tau - 1 > n:
            raise OracleError("range", f"tau - 1 = {tau - 1} exceeds length {n}")
        new_len = tau - 1
        keep = self.pages_for(new_len)
        removed = self.table[seq][keep:]
        freed = self._drop(removed)   # descending logical order onto the stack
        self.table[seq] = self.table[seq][:keep]
        self.length[seq] = new_len
        self.appended[seq] = 0
        self.checkpoints[seq] = [b for b in self.checkpoints[seq] if b <= new_len]
        return freed

    # -- append (prefill write of the replayed suffix) -------------------------
    def append(self, seq, k_bits=None, v_bits=None, n_tokens=None):
        """Append n tokens. k_bits / v_bits: bf16 bits [L][n][Hkv][d] (or None when
        values are not stored)."""
        self._check_seq(seq)
        if k_bits is not None:
            n = int(k_bits.shape[1])
        else:
            n = int(n_tokens)
        if n < 0:
            raise OracleError("invalid", "negative token count")
        old = self.length[seq]
        new_len = old + n
        if self.pages_for(new_len) > self.max_pages_per_seq:
            raise OracleError("range", "sequence would exceed max_pages_per_seq")
        need = self.pages_for(new_len) - len(self.table[seq])
        tbl = self.table[seq]
        cow = n > 0 and old % self.ps != 0 and self.refs[tbl[-1]] > 1
        if need + (1 if cow else 0) > len(self.free):
            raise OracleError("oom", f"need {need + (1 if cow else 0)} pages, {len(self.free)} free")
        if cow:  # the partial last page is shared: copy its valid slots first
            src, dst = tbl[-1], self.free.pop()
            self.refs[src] -= 1
            self.refs[dst] = 1
            if self.store_values:
                used = old % self.ps
                self.k_pool[:, dst, :, :used] = self.k_pool[:, src, :, :used]
                self.v_pool[:, dst, :, :used] = self.v_pool[:, src, :, :used]
            tbl[-1] = dst
        for _ in range(need):
            p = self.free.pop()
            self.refs[p] = 1
            tbl.append(p)
        if self.store_values and k_bits is not None:
            for t in range(n):
                pos = old + t
                page, slot = tbl[pos // self.ps], pos % self.ps
                self.k_pool[:, page, :, slot, :] = k_bits[:, t]
                self.v_pool[:, page, :, slot, :] = v_bits[:, t]
        self.length[seq] = new_len
        self.appended[seq] += n

    # -- queries ---------------------------------------------------------------
    def free_list(self) -> list[int]:
        """Free pages, top of the stack (next popped) first."""
        return list(reversed(self.free))

    def page_table(self, seq) -> list[int]:
        self._check_seq(seq)
        return list(self.table[seq])

    def seq_info(self, seq):
        self._check_seq(seq)
        return self.length[seq], self.appended[seq]

    def gather(self, seq, layer):
        """The sequence's K and V in logical order: bf16 bits [len][Hkv][d] each."""
        self._check_seq(seq)
        if not 0 <= layer < self.L:
            raise OracleError("range", f"layer {layer} out of range")
        n = self.length[seq]
        pos = np.arange(n)
        pages = np.asarray(self.table[seq], dtype=np.int64)[pos // self.ps] if n else np.zeros(0, np.int64)
        slots = pos % self.ps
        k = self.k_pool[layer][pages, :, slots, :]
        v = self.v_pool[layer][pages, :, slots, :]
        return np.ascontiguousarray(k), np.ascontiguousarray(v)
