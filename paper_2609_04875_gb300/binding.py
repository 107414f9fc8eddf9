"""ctypes binding of libpe (include/pe.h): argument marshalling only.

Every step of the path -- crop, append, replay attention, split-KV combine --
runs in the library's CUDA kernels; this module passes tensor pointers, sizes
and the current CUDA stream, and turns status codes into exceptions.  There is
no other implementation behind it: if libpe.so is missing, importing this
module fails.
"""
from __future__ import annotations

import ctypes
import math
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpe.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")

_lib = ctypes.CDLL(LIB_PATH)

PE_OK = 0
ERROR_KINDS = {-1: "invalid", -2: "range", -3: "oom", -4: "cuda", -5: "unsupported", -6: "device_timeout"}

EXPORTED = [
    "pe_cache_create", "pe_cache_destroy", "pe_seq_create", "pe_seq_release", "pe_crop", "pe_crop_batch",
    "pe_append_kv", "pe_append_kv_batch", "pe_replay_attn", "pe_replay_attn_batch", "pe_seq_info",
    "pe_seq_page_table", "pe_free_list", "pe_seq_device_page_table", "pe_cache_pools", "pe_set_option",
    "pe_device_status", "pe_kernel_launches", "pe_replay_attn_static_scratch", "pe_selftest_bounded_wait",
    "pe_last_attn_plan", "pe_seq_fork", "pe_checkpoint_add", "pe_checkpoint_select", "pe_restore",
    "pe_seq_checkpoints", "pe_page_refs", "pe_prov_create", "pe_prov_destroy", "pe_prov_add",
    "pe_prov_locate_source", "pe_prov_taint_closure", "pe_prov_first_entry", "pe_replay_schedule",
    "pe_replay_rounds", "pe_attn_plan_persistent", "pe_attn_plan_launches", "pe_last_error", "pe_version",
]

# Turn kinds and replay policies of pe_replay_schedule (pe.h).
TURN_INPUT, TURN_MODEL_INDEP, TURN_MODEL_DEP = 0, 1, 2
POLICY_SELECTIVE, POLICY_PREFIX_CACHE = 0, 1


class PEError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERROR_KINDS.get(code, code)}: {msg}")
        self.code = code
        self.kind = ERROR_KINDS.get(code, str(code))


class _Config(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32), ("num_pages", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32), ("host_only", ctypes.c_int32),
        ("init_free_order", ctypes.POINTER(ctypes.c_int32)), ("k_pool", ctypes.c_void_p),
        ("v_pool", ctypes.c_void_p), ("workspace_bytes", ctypes.c_int64),
    ]


_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_I32P = ctypes.POINTER(ctypes.c_int32)
_I64P = ctypes.POINTER(ctypes.c_int64)

_sigs = {
    "pe_cache_create": [ctypes.POINTER(_Config), ctypes.POINTER(_P)],
    "pe_cache_destroy": [_P],
    "pe_seq_create": [_P, _I32P],
    "pe_seq_release": [_P, _I32, _P],
    "pe_crop": [_P, _I32, _I64, _I32P, _I32, _I32P, _P],
    "pe_crop_batch": [_P, _I32, _I32P, _I64P, _P],
    "pe_append_kv": [_P, _I32, _P, _P, _I32, _P],
    "pe_append_kv_batch": [_P, _I32, _I32P, _P, _P, _I32P, _P],
    "pe_replay_attn": [_P, _I32, _I32, _P, _P, _I32, _I32, ctypes.c_float, _P],
    "pe_replay_attn_batch": [_P, _I32, _I32P, _I32, _P, _I32P, _P, _I32, ctypes.c_float, _P],
    "pe_seq_info": [_P, _I32, _I64P, _I64P],
    "pe_seq_page_table": [_P, _I32, _I32P, _I32, _I32P],
    "pe_free_list": [_P, _I32P, _I32, _I32P],
    "pe_seq_device_page_table": [_P, _I32, _I32P, _I32, _P],
    "pe_cache_pools": [_P, ctypes.POINTER(_P), ctypes.POINTER(_P)],
    "pe_set_option": [_P, ctypes.c_char_p, _I64],
    "pe_device_status": [_P, _I32P, _I32, _P],
    "pe_kernel_launches": [_P, _I64P],
    "pe_selftest_bounded_wait": [_P, _I64, _P],
    "pe_last_attn_plan": [_P, _I32P, _I32P, _I32P],
    "pe_seq_fork": [_P, _I32, _I32P, _P],
    "pe_checkpoint_add": [_P, _I32, _I64],
    "pe_checkpoint_select": [_P, _I32, _I64, _I64P],
    "pe_restore": [_P, _I32, _I64, _I64P, _I32P, _I32, _I32P, _P],
    "pe_seq_checkpoints": [_P, _I32, _I64P, _I32, _I32P],
    "pe_page_refs": [_P, _I32P, _I32],
    "pe_prov_create": [ctypes.POINTER(_P)],
    "pe_prov_destroy": [_P],
    "pe_prov_add": [_P, _I64, _I32, _I64P, _I32, _I64P, _I32, _I64, _I64, _I32, _I32],
    "pe_prov_locate_source": [_P, _I64, _I64P],
    "pe_prov_taint_closure": [_P, _I64, _I64P, _I32, _I32P, _I32P],
    "pe_prov_first_entry": [_P, _I64, _I64P],
    "pe_replay_attn_static_scratch": [_P, _I32, _I32, _P, _P, _I32, _I32, ctypes.c_float, _P],
    "pe_replay_schedule": [_I32, _I32P, _I32P, _I32P, _I32, _I32P, _I64, _I32P, _I64P],
    "pe_replay_rounds": [_P, _I32, _I32P, _I32, _I32P, _I32P, _P, _P, _P, _P, _I32, ctypes.c_float, _P],
    "pe_attn_plan_persistent": [_P, _I32, _I32P, _I32P, _I32, _I32, _I32P, _I32P, _I32P, _I32, _I32P, _I32,
                                _I32P, _I32],
    "pe_attn_plan_launches": [_P, _I32, _I32P, _I32P, _I32, _I32, _I64P, _I64, _I64P],
}
for _name, _args in _sigs.items():
    _fn = getattr(_lib, _name)
    _fn.argtypes = _args
    _fn.restype = ctypes.c_int32
_lib.pe_last_error.restype = ctypes.c_char_p
_lib.pe_last_error.argtypes = []
_lib.pe_version.restype = ctypes.c_char_p
_lib.pe_version.argtypes = []


def lib():
    return _lib


def version() -> str:
    return _lib.pe_version().decode()


def _check(rc: int):
    if rc != PE_OK:
        raise PEError(rc, _lib.pe_last_error().decode())


def i32_array(vals):
    """A ctypes int32 array of ``vals``; the batch calls take it as is, so a
    caller repeating a call with the same ids can convert them once."""
    if isinstance(vals, ctypes.Array) and vals._type_ is ctypes.c_int32:
        return vals
    vals = [int(v) for v in vals]
    return (ctypes.c_int32 * max(1, len(vals)))(*vals)


def i64_array(vals):
    """A ctypes int64 array of ``vals`` (taken as is by the batch calls)."""
    if isinstance(vals, ctypes.Array) and vals._type_ is ctypes.c_int64:
        return vals
    vals = [int(v) for v in vals]
    return (ctypes.c_int64 * max(1, len(vals)))(*vals)


_i32_array, _i64_array = i32_array, i64_array


def replay_schedule(agents_turns, policy):
    """pe_replay_schedule: agents_turns[i] = ((n_tokens, kind), ...).  Returns
    (take, decode_tokens): take is int32 numpy [rounds][agents] (positions each
    agent appends and attends per round); decode_tokens the positions decoded."""
    import numpy as np
    cu, lens, kinds = [0], [], []
    for turns in agents_turns:
        for n, k in turns:
            lens.append(int(n))
            kinds.append(int(k))
        cu.append(len(lens))
    n = len(agents_turns)
    rounds, dec = ctypes.c_int32(), ctypes.c_int64()
    cu_a, len_a, kind_a = _i32_array(cu), _i32_array(lens), _i32_array(kinds)
    _check(_lib.pe_replay_schedule(n, cu_a, len_a, kind_a, int(policy), None, 0, ctypes.byref(rounds),
                                   ctypes.byref(dec)))
    take = np.zeros((rounds.value, n), dtype=np.int32)
    if take.size:
        _check(_lib.pe_replay_schedule(n, cu_a, len_a, kind_a, int(policy), take.ctypes.data_as(_I32P), take.size,
                                       ctypes.byref(rounds), ctypes.byref(dec)))
    return take, dec.value


def _stream(stream):
    import torch
    if stream is None:
        raw = getattr(torch._C, "_cuda_getCurrentRawStream", None)
        dev = getattr(torch._C, "_cuda_getDevice", None)
        if raw is not None and dev is not None and torch.cuda.is_initialized():
            return ctypes.c_void_p(raw(dev()))  # the current stream's handle, without a Stream object
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream))


def _dev_ptr(t, name, device=None):
    """Device pointer of a contiguous bf16 CUDA tensor; with ``device`` given,
    the tensor must live on that CUDA device (the cache's)."""
    import torch
    if t.dtype != torch.bfloat16:
        raise TypeError(f"{name} must be bfloat16")
    if not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if device is not None and t.device.index != device:
        raise ValueError(f"{name} is on cuda:{t.device.index}, the cache on cuda:{device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _same_shape(out, Q):
    if out is not None and tuple(out.shape) != tuple(Q.shape):
        raise ValueError(f"out has shape {tuple(out.shape)}, Q {tuple(Q.shape)}: they must match")


class PagedKVCache:
    """Paged KV cache with crop and replay attention (one GPU).

    Pool layout per layer: [num_pages][Hkv][page_size][d] bf16 for K and V.
    ``k_pool`` / ``v_pool``: optional caller-owned CUDA tensors of shape
    [L][num_pages][Hkv][page_size][d] (bf16); otherwise the library allocates.
    ``host_only=True`` keeps only the host bookkeeping (no device memory).
    A device cache lives on the CUDA device current at construction; its calls
    must be made with that device current, on tensors that live there.
    """

    def __init__(self, num_layers, num_kv_heads, head_dim, page_size, num_pages, max_seqs, max_pages_per_seq,
                 init_free_order=None, k_pool=None, v_pool=None, host_only=False, workspace_bytes=0):
        cfg = _Config()
        cfg.num_layers, cfg.num_kv_heads, cfg.head_dim = num_layers, num_kv_heads, head_dim
        cfg.page_size, cfg.num_pages, cfg.max_seqs = page_size, num_pages, max_seqs
        cfg.max_pages_per_seq, cfg.host_only = max_pages_per_seq, 1 if host_only else 0
        self._order = None
        if init_free_order is not None:
            self._order = _i32_array(init_free_order)
            if len(init_free_order) != num_pages:
                raise ValueError("init_free_order must list every page")
            cfg.init_free_order = ctypes.cast(self._order, _I32P)
        self._device = None
        if not host_only:
            import torch
            self._device = torch.cuda.current_device()
        self._pools = (k_pool, v_pool)  # keep caller tensors alive
        if k_pool is not None:
            cfg.k_pool = self._ptr(k_pool, "k_pool").value
            cfg.v_pool = self._ptr(v_pool, "v_pool").value
        cfg.workspace_bytes = int(workspace_bytes)
        self.num_layers, self.num_kv_heads, self.head_dim = num_layers, num_kv_heads, head_dim
        self.page_size, self.num_pages, self.max_seqs = page_size, num_pages, max_seqs
        self.max_pages_per_seq = max_pages_per_seq
        self.host_only = host_only
        h = ctypes.c_void_p()
        _check(_lib.pe_cache_create(ctypes.byref(cfg), ctypes.byref(h)))
        self._h = h

    # -- lifetime ------------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(_lib.pe_cache_destroy(self._h))
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    @property
    def handle(self):
        return self._h

    def _s(self, stream):
        return ctypes.c_void_p(None) if self.host_only else _stream(stream)

    def _ptr(self, t, name):
        return _dev_ptr(t, name, self._device)

    # -- sequences -----------------------------------------------------------
    def seq_create(self) -> int:
        s = ctypes.c_int32()
        _check(_lib.pe_seq_create(self._h, ctypes.byref(s)))
        return s.value

    def seq_release(self, seq, stream=None):
        _check(_lib.pe_seq_release(self._h, seq, self._s(stream)))

    def seq_fork(self, seq, stream=None) -> int:
        """New sequence sharing all of ``seq``'s pages (copy-on-write on append)."""
        out = ctypes.c_int32()
        _check(_lib.pe_seq_fork(self._h, seq, ctypes.byref(out), self._s(stream)))
        return out.value

    # -- checkpoints (metadata only) --------------------------------------------
    def checkpoint_add(self, seq, offset):
        _check(_lib.pe_checkpoint_add(self._h, seq, int(offset)))

    def checkpoint_select(self, seq, tau) -> int:
        out = ctypes.c_int64()
        _check(_lib.pe_checkpoint_select(self._h, seq, int(tau), ctypes.byref(out)))
        return out.value

    def checkpoints(self, seq):
        n = ctypes.c_int32()
        _check(_lib.pe_seq_checkpoints(self._h, seq, None, 0, ctypes.byref(n)))
        buf = (ctypes.c_int64 * max(1, n.value))()
        _check(_lib.pe_seq_checkpoints(self._h, seq, buf, n.value, ctypes.byref(n)))
        return list(buf[: n.value])

    def restore(self, seq, tau, stream=None):
        """Restore(c*): crop to the last checkpoint before tau; returns (offset, freed pages)."""
        cap = self.max_pages_per_seq
        buf = (ctypes.c_int32 * cap)()
        n = ctypes.c_int32()
        off = ctypes.c_int64()
        _check(_lib.pe_restore(self._h, seq, int(tau), ctypes.byref(off), buf, cap, ctypes.byref(n), self._s(stream)))
        return off.value, list(buf[: n.value])

    def page_refs(self):
        buf = (ctypes.c_int32 * self.num_pages)()
        _check(_lib.pe_page_refs(self._h, buf, self.num_pages))
        return list(buf)

    # -- crop (restore) --------------------------------------------------------
    def crop(self, seq, tau, stream=None):
        """Keep the first tau-1 tokens; returns the freed page ids (ascending logical)."""
        cap = self.max_pages_per_seq
        buf = (ctypes.c_int32 * cap)()
        n = ctypes.c_int32()
        _check(_lib.pe_crop(self._h, seq, int(tau), buf, cap, ctypes.byref(n), self._s(stream)))
        return list(buf[: n.value])

    def crop_batch(self, seqs, taus, stream=None):
        _check(_lib.pe_crop_batch(self._h, len(seqs), _i32_array(seqs), _i64_array(taus), self._s(stream)))

    # -- append (prefill write) ------------------------------------------------
    def append_kv(self, seq, K=None, V=None, n_tokens=None, stream=None):
        """K, V: CUDA bf16 [L][n][Hkv][d].  Host-only caches take n_tokens instead."""
        if K is None:
            if not self.host_only:
                raise ValueError("K and V are required")
            _check(_lib.pe_append_kv(self._h, seq, None, None, int(n_tokens), self._s(stream)))
            return
        self._check_kv(K, V)
        _check(_lib.pe_append_kv(self._h, seq, self._ptr(K, "K"), self._ptr(V, "V"), K.shape[1], self._s(stream)))

    def append_kv_batch(self, seqs, K=None, V=None, cu_tokens=None, stream=None):
        """K, V: CUDA bf16 [L][cu_tokens[-1]][Hkv][d]; sequence i gets tokens cu_tokens[i]:cu_tokens[i+1]."""
        cu = _i32_array(cu_tokens)
        if K is None:
            if not self.host_only:
                raise ValueError("K and V are required")
            _check(_lib.pe_append_kv_batch(self._h, len(seqs), _i32_array(seqs), None, None, cu, self._s(stream)))
            return
        self._check_kv(K, V)
        if K.shape[1] != cu_tokens[-1]:
            raise ValueError("K token count does not match cu_tokens")
        _check(_lib.pe_append_kv_batch(self._h, len(seqs), _i32_array(seqs), self._ptr(K, "K"), self._ptr(V, "V"),
                                       cu, self._s(stream)))

    def _check_kv(self, K, V):
        if K.shape != V.shape or K.dim() != 4:
            raise ValueError("K and V must both be [L][n][Hkv][d]")
        if K.shape[0] != self.num_layers or K.shape[2] != self.num_kv_heads or K.shape[3] != self.head_dim:
            raise ValueError(f"K shape {tuple(K.shape)} does not match the cache")

    # -- replay attention ------------------------------------------------------
    def replay_attn(self, seq, layer, Q, out=None, softmax_scale=None, stream=None):
        """Attention of the last Q.shape[0] positions of ``seq``; Q, out: CUDA bf16 [n_q][Hq][d]."""
        import torch
        if Q.dim() != 3 or Q.shape[2] != self.head_dim:
            raise ValueError("Q must be [n_q][Hq][d]")
        _same_shape(out, Q)
        if out is None:
            out = torch.empty_like(Q)
        scale = 1.0 / math.sqrt(self.head_dim) if softmax_scale is None else float(softmax_scale)
        _check(_lib.pe_replay_attn(self._h, seq, layer, self._ptr(Q, "Q"), self._ptr(out, "out"), Q.shape[0],
                                   Q.shape[1], scale, self._s(stream)))
        return out

    def replay_attn_batch(self, seqs, layer, Q, cu_q, out=None, softmax_scale=None, stream=None):
        """Q, out: CUDA bf16 [cu_q[-1]][Hq][d]; rows cu_q[i]:cu_q[i+1] are the last positions of seqs[i]."""
        import torch
        if Q.dim() != 3 or Q.shape[2] != self.head_dim or Q.shape[0] != cu_q[-1]:
            raise ValueError("Q must be [cu_q[-1]][Hq][d]")
        _same_shape(out, Q)
        if out is None:
            out = torch.empty_like(Q)
        scale = 1.0 / math.sqrt(self.head_dim) if softmax_scale is None else float(softmax_scale)
        _check(_lib.pe_replay_attn_batch(self._h, len(seqs), _i32_array(seqs), layer, self._ptr(Q, "Q"),
                                         _i32_array(cu_q), self._ptr(out, "out"), Q.shape[1], scale,
                                         self._s(stream)))
        return out

    def replay_rounds(self, seqs, take, cu_tok, K=None, V=None, Q=None, out=None, softmax_scale=None,
                      num_q_heads=None, stream=None):
        """pe_replay_rounds: round r appends take[r][i] positions of agent i and
        attends them, all layers.  K, V: CUDA bf16 [L][N][Hkv][d]; Q, out:
        [L][N][Hq][d]; agent i owns rows cu_tok[i]:cu_tok[i+1].  Host-only
        caches take no tensors (bookkeeping only)."""
        import numpy as np
        import torch
        take = np.ascontiguousarray(take, dtype=np.int32)
        n_rounds = int(take.shape[0]) if take.ndim == 2 else 0
        if take.size and take.shape[1] != len(seqs):
            raise ValueError("take must be [rounds][len(seqs)]")
        take_p = take.ctypes.data_as(_I32P) if take.size else None
        scale = 1.0 / math.sqrt(self.head_dim) if softmax_scale is None else float(softmax_scale)
        if self.host_only:
            hq = num_q_heads or self.num_kv_heads
            _check(_lib.pe_replay_rounds(self._h, len(seqs), _i32_array(seqs), n_rounds, take_p, _i32_array(cu_tok),
                                         None, None, None, None, hq, scale, self._s(stream)))
            return None
        self._check_kv(K, V)
        if Q.dim() != 4 or Q.shape[0] != self.num_layers or Q.shape[1] != K.shape[1] or Q.shape[3] != self.head_dim:
            raise ValueError("Q must be [L][N][Hq][d] with the rows of K")
        if K.shape[1] != cu_tok[-1]:
            raise ValueError("K row count does not match cu_tok")
        _same_shape(out, Q)
        if out is None:
            out = torch.empty_like(Q)
        _check(_lib.pe_replay_rounds(self._h, len(seqs), _i32_array(seqs), n_rounds, take_p, _i32_array(cu_tok),
                                     self._ptr(K, "K"), self._ptr(V, "V"), self._ptr(Q, "Q"), self._ptr(out, "out"),
                                     Q.shape[2], scale, self._s(stream)))
        return out

    # -- prepared calls ----------------------------------------------------------
    # A caller repeating the same call (the same sequences, buffers and stream,
    # e.g. one step of a benchmark loop) can validate and marshal its arguments
    # once: each prepare_* checks them like the plain method and returns a
    # function of no arguments that only calls the library.  The tensors are
    # kept alive by the returned function; their contents may change between
    # calls, their storage may not.
    def prepare_crop_batch(self, seqs, taus, stream=None):
        args = (self._h, len(seqs), _i32_array(seqs), _i64_array(taus), self._s(stream))
        fn = _lib.pe_crop_batch

        def call():
            rc = fn(*args)
            if rc:
                _check(rc)
        return call

    def prepare_append_kv_batch(self, seqs, K, V, cu_tokens, stream=None):
        self._check_kv(K, V)
        if K.shape[1] != cu_tokens[-1]:
            raise ValueError("K token count does not match cu_tokens")
        keep = (K, V)
        args = (self._h, len(seqs), _i32_array(seqs), self._ptr(K, "K"), self._ptr(V, "V"), _i32_array(cu_tokens),
                self._s(stream))
        fn = _lib.pe_append_kv_batch

        def call():
            rc = fn(*args)
            if rc:
                _check(rc)
            return keep
        return call

    def prepare_replay_attn_batch(self, seqs, layer, Q, cu_q, out, softmax_scale=None, stream=None):
        if Q.dim() != 3 or Q.shape[2] != self.head_dim or Q.shape[0] != cu_q[-1] or out.shape != Q.shape:
            raise ValueError("Q and out must be [cu_q[-1]][Hq][d]")
        scale = 1.0 / math.sqrt(self.head_dim) if softmax_scale is None else float(softmax_scale)
        keep = (Q, out)
        args = (self._h, len(seqs), _i32_array(seqs), int(layer), self._ptr(Q, "Q"), _i32_array(cu_q),
                self._ptr(out, "out"), Q.shape[1], ctypes.c_float(scale), self._s(stream))
        fn = _lib.pe_replay_attn_batch

        def call():
            rc = fn(*args)
            if rc:
                _check(rc)
            return keep
        return call

    def replay_attn_static_scratch(self, seq, layer, Q, out=None, softmax_scale=None, stream=None):
        """pe_replay_attn_static_scratch: split-KV replay attention whose partials
        live in the library's fixed device array (the call allocates nothing)."""
        import torch
        if Q.dim() != 3 or Q.shape[2] != self.head_dim:
            raise ValueError("Q must be [n_q][Hq][d]")
        _same_shape(out, Q)
        if out is None:
            out = torch.empty_like(Q)
        scale = 1.0 / math.sqrt(self.head_dim) if softmax_scale is None else float(softmax_scale)
        _check(_lib.pe_replay_attn_static_scratch(self._h, seq, layer, self._ptr(Q, "Q"), self._ptr(out, "out"),
                                                  Q.shape[0], Q.shape[1], scale, self._s(stream)))
        return out

    # -- state -----------------------------------------------------------------
    def seq_info(self, seq):
        n, a = ctypes.c_int64(), ctypes.c_int64()
        _check(_lib.pe_seq_info(self._h, seq, ctypes.byref(n), ctypes.byref(a)))
        return n.value, a.value

    def page_table(self, seq):
        n = ctypes.c_int32()
        _check(_lib.pe_seq_page_table(self._h, seq, None, 0, ctypes.byref(n)))
        buf = (ctypes.c_int32 * max(1, n.value))()
        _check(_lib.pe_seq_page_table(self._h, seq, buf, n.value, ctypes.byref(n)))
        return list(buf[: n.value])

    def free_list(self):
        n = ctypes.c_int32()
        _check(_lib.pe_free_list(self._h, None, 0, ctypes.byref(n)))
        buf = (ctypes.c_int32 * max(1, n.value))()
        _check(_lib.pe_free_list(self._h, buf, n.value, ctypes.byref(n)))
        return list(buf[: n.value])

    def device_page_table(self, seq, n=None, stream=None):
        n = self.max_pages_per_seq if n is None else n
        buf = (ctypes.c_int32 * max(1, n))()
        _check(_lib.pe_seq_device_page_table(self._h, seq, buf, n, self._s(stream)))
        return list(buf[:n])

    def set_option(self, key: str, value: int):
        _check(_lib.pe_set_option(self._h, key.encode(), int(value)))

    def selftest_bounded_wait(self, limit_ns: int, stream=None):
        """Launches a kernel whose bounded wait runs out (nothing arrives); the
        device status word then reads 1.  Tests failure detection without a fault."""
        _check(_lib.pe_selftest_bounded_wait(self._h, int(limit_ns), self._s(stream)))

    def last_attn_plan(self):
        """(split path used, key splits, attention CTAs) of the last attention launch."""
        a, b, c = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        _check(_lib.pe_last_attn_plan(self._h, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)))
        return bool(a.value), b.value, c.value

    def plan_persistent(self, seqs, n_q, num_q_heads, num_sms=0):
        """pe_attn_plan_persistent: the persistent kernel's plan for the group
        (sequence i attends its last n_q[i] positions), made on the host.
        Returns a dict: n_ctas, rounds, n_slots, max_parts, order (sequences in
        planning order), unit_tiles, ctas (rows u0, t0, u1, t1, slot0, part0,
        slot1, part1) and slots (rows unit, n_parts)."""
        cu = [0]
        for q in n_q:
            cu.append(cu[-1] + int(q))
        info = (ctypes.c_int32 * 5)()
        order = (ctypes.c_int32 * max(1, len(seqs)))()
        args = (self._h, len(seqs), _i32_array(seqs), _i32_array(cu), int(num_q_heads), int(num_sms), info, order)
        _check(_lib.pe_attn_plan_persistent(*args, None, 0, None, 0, None, 0))
        n_ctas, rounds, n_slots, max_parts, n_units = list(info)
        tiles = (ctypes.c_int32 * max(1, n_units))()
        ctas = (ctypes.c_int32 * max(1, 8 * n_ctas))()
        slots = (ctypes.c_int32 * max(1, 2 * n_slots))()
        _check(_lib.pe_attn_plan_persistent(*args, tiles, n_units, ctas, n_ctas, slots, n_slots))
        return {"n_ctas": n_ctas, "rounds": rounds, "n_slots": n_slots, "max_parts": max_parts,
                "order": list(order[: len(seqs)]), "unit_tiles": list(tiles[:n_units]),
                "ctas": [list(ctas[8 * k: 8 * k + 8]) for k in range(n_ctas)],
                "slots": [list(slots[2 * k: 2 * k + 2]) for k in range(n_slots)]}

    LAUNCH_KINDS = {0: "one_item", 1: "one_item_tail", 2: "persistent", 3: "decode"}
    _SEQ_FIELDS = ("seq", "item0", "n_q", "n_keys", "n_qtiles", "n_splits", "pair_top", "part_row0", "comb0",
                   "q_row0")

    def plan_launches(self, seqs, n_q, num_q_heads, num_sms=0):
        """pe_attn_plan_launches: the launches an attention call over these
        sequences (each attending its last n_q[i] positions) would make, planned
        on the host.  A list of dicts: kind, split, ctas, combine_rows,
        split_tiles, pairs_fastest and seqs (one dict per sequence)."""
        cu = [0]
        for q in n_q:
            cu.append(cu[-1] + int(q))
        n_words = ctypes.c_int64()
        args = (self._h, len(seqs), _i32_array(seqs), _i32_array(cu), int(num_q_heads), int(num_sms))
        _check(_lib.pe_attn_plan_launches(*args, None, 0, ctypes.byref(n_words)))
        buf = (ctypes.c_int64 * max(1, n_words.value))()
        _check(_lib.pe_attn_plan_launches(*args, buf, n_words.value, ctypes.byref(n_words)))
        words, out, i = list(buf[: n_words.value]), [], 0
        while i < len(words):
            kind, split, ctas, comb, split_tiles, pairs_fastest, n = words[i: i + 7]
            i += 7
            rows = [dict(zip(self._SEQ_FIELDS, words[i + 10 * k: i + 10 * k + 10])) for k in range(n)]
            i += 10 * n
            out.append({"kind": self.LAUNCH_KINDS[kind], "split": bool(split), "ctas": ctas,
                        "combine_rows": comb, "split_tiles": split_tiles, "pairs_fastest": bool(pairs_fastest),
                        "seqs": rows})
        return out

    def kernel_launches(self) -> int:
        n = ctypes.c_int64()
        _check(_lib.pe_kernel_launches(self._h, ctypes.byref(n)))
        return n.value

    def device_status(self, clear=True, stream=None):
        code = ctypes.c_int32()
        rc = _lib.pe_device_status(self._h, ctypes.byref(code), 1 if clear else 0, self._s(stream))
        if rc not in (PE_OK, -6):
            _check(rc)
        return code.value


class ProvenanceGraph:
    """Artifact DAG of one session (Sec. 3.4(a)) and the queries of Alg. 1,
    lines 1-3: locate_source(z), taint_closure(s), first_entry(s) -> tau."""

    def __init__(self):
        h = ctypes.c_void_p()
        _check(_lib.pe_prov_create(ctypes.byref(h)))
        self._h = h

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            _check(_lib.pe_prov_destroy(self._h))
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def add(self, aid, type_=0, parents=(), source_ids=(), token_begin=0, token_end=0, turn=0, committed=False):
        par = _i64_array(parents)
        src = _i64_array(source_ids)
        _check(_lib.pe_prov_add(self._h, int(aid), int(type_), par, len(parents), src, len(source_ids),
                                int(token_begin), int(token_end), int(turn), 1 if committed else 0))

    def locate_source(self, z) -> int:
        out = ctypes.c_int64()
        _check(_lib.pe_prov_locate_source(self._h, int(z), ctypes.byref(out)))
        return out.value

    def taint_closure(self, s):
        """(ids ascending, number that committed a side effect)"""
        n, nc = ctypes.c_int32(), ctypes.c_int32()
        _check(_lib.pe_prov_taint_closure(self._h, int(s), None, 0, ctypes.byref(n), ctypes.byref(nc)))
        buf = (ctypes.c_int64 * max(1, n.value))()
        _check(_lib.pe_prov_taint_closure(self._h, int(s), buf, n.value, ctypes.byref(n), ctypes.byref(nc)))
        return list(buf[: n.value]), nc.value

    def first_entry(self, s) -> int:
        out = ctypes.c_int64()
        _check(_lib.pe_prov_first_entry(self._h, int(s), ctypes.byref(out)))
        return out.value
