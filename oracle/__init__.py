"""fp64 CPU oracle for crop + replay attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package.  The
product library never loads it, and it shares no code, header, table or helper
with the CUDA path; the two meet only in the seeded inputs of ``synth``.

Contents
  * ``kvcache.OracleKVCache`` -- paged cache state: allocator, page tables,
    lengths, recomputation counter, pool contents (exact bits).
  * ``causal_attention`` -- attention by its definition in fp64 (C, threaded
    over rows; see attention.c).
  * ``replay_attention`` -- gathers a sequence through the oracle cache's page
    table and runs ``causal_attention`` on its last n_q positions.
  * ``schedule`` -- which suffix positions a replay re-prefills and which it
    re-decodes (selective replay vs full reset with a prefix cache), the
    lockstep rounds over many agents, and ``execute_rounds`` on the oracle cache.
  * ``provenance.OracleProvenance`` -- the artifact graph queries.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .kvcache import OracleError, OracleKVCache  # noqa: F401
from . import schedule  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attention.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile attention.c with gcc (IEEE order kept: no fast-math, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-ffp-contract=off",
               "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            lib.oracle_causal_attention.restype = ctypes.c_int
            lib.oracle_causal_attention.argtypes = [
                ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_double,
                ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int32]
            lib.oracle_num_cpus.restype = ctypes.c_int
            _lib = lib
    return _lib


def num_cpus() -> int:
    return int(_load().oracle_num_cpus())


def causal_attention(q_bits, k_bits, v_bits, scale, rows=None, nthreads=0):
    """Bottom-right causal attention in fp64.

    q_bits: bf16 bits [n_q][Hq][d]; k_bits, v_bits: bf16 bits [n_keys][Hkv][d].
    Query i is at position n_keys - n_q + i and sees keys 0..that position.
    rows: optional query indices; returns fp64 [len(rows) or n_q][Hq][d].
    """
    lib = _load()
    q = np.ascontiguousarray(q_bits, dtype=np.uint16)
    k = np.ascontiguousarray(k_bits, dtype=np.uint16)
    v = np.ascontiguousarray(v_bits, dtype=np.uint16)
    n_q, hq, d = q.shape
    n_keys, hkv, dk = k.shape
    if dk != d or v.shape != k.shape:
        raise ValueError("shape mismatch")
    if rows is not None:
        rows = np.ascontiguousarray(rows, dtype=np.int64)
        n_rows = int(rows.shape[0])
        rows_ptr = rows.ctypes.data
    else:
        n_rows, rows_ptr = n_q, None
    out = np.zeros((n_rows, hq, d), dtype=np.float64)
    rc = lib.oracle_causal_attention(q.ctypes.data, n_q, k.ctypes.data, v.ctypes.data, n_keys,
                                     hq, hkv, d, float(scale), rows_ptr, n_rows, out.ctypes.data,
                                     int(nthreads))
    if rc != 0:
        raise ValueError("oracle_causal_attention: invalid arguments")
    return out


def replay_attention(cache: OracleKVCache, seq: int, layer: int, q_bits, scale, rows=None, nthreads=0):
    """Attention of the last n_q positions of ``seq`` (queries q_bits [n_q][Hq][d])
    over the cache's keys, read through the oracle's own page table."""
    k, v = cache.gather(seq, layer)
    n_keys = k.shape[0]
    if q_bits.shape[0] > n_keys:
        raise OracleError("range", "more queries than cached tokens")
    return causal_attention(q_bits, k, v, scale, rows=rows, nthreads=nthreads)


def execute_rounds(cache: OracleKVCache, seqs, take, k_bits, v_bits, q_bits, cu_tok, scale, nthreads=0):
    """``schedule.execute_rounds`` with this package's replay attention."""
    def attend(c, seq, layer, q, sc):
        return replay_attention(c, seq, layer, q, sc, nthreads=nthreads)
    return schedule.execute_rounds(cache, seqs, take, k_bits, v_bits, q_bits, cu_tok, scale, attend)
