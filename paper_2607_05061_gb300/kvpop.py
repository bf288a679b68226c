"""ctypes binding of the KVpop C ABI (include/kvpop.h).

Argument marshalling only: every step of the decode path runs in the CUDA
library ``libkvpop.so``.  Tensors are passed by ``data_ptr()`` and the current
torch stream by its ``cuda_stream`` handle; torch is used only for device
memory and streams.  Importing this module fails loudly when the library has
not been built -- there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int32, c_size_t, c_void_p
from typing import Optional, Sequence

import torch  # loads the CUDA runtime the library links against

_HERE = os.path.dirname(os.path.abspath(__file__))
# KVPOP_DEVICE_CHECKS=1 selects the device-check build (index checks that record an
# error instead of trapping), built by ``build.build(checked=True)``
CHECKED = os.environ.get("KVPOP_DEVICE_CHECKS", "0") == "1"
LIB_PATH = os.path.join(_HERE, "libkvpop_checked.so" if CHECKED else "libkvpop.so")

KVPOP_F32, KVPOP_BF16 = 0, 1
STATUS = {0: "KVPOP_OK", 1: "KVPOP_ERR_INVALID_ARG", 2: "KVPOP_ERR_ALIGN", 3: "KVPOP_ERR_OOM",
          4: "KVPOP_ERR_CUDA", 5: "KVPOP_ERR_STATE", 6: "KVPOP_ERR_DEVICE_CHECK"}

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -m paper_2607_05061_gb300.build`"
                      + (" -c" if CHECKED else "") +
                      " (or __graft_entry__.build()); the decode path has no non-CUDA fallback")
_lib = ctypes.CDLL(LIB_PATH)


class kvpop_config(ctypes.Structure):
    _fields_ = [("batch", c_int32), ("n_kv_heads", c_int32), ("q_per_kv", c_int32),
                ("head_dim", c_int32), ("budget_B", c_int32), ("delay_D", c_int32),
                ("n_sink", c_int32), ("scorer_hidden", c_int32), ("kv_dtype", ctypes.c_int)]


class kvpop_scorer(ctypes.Structure):
    _fields_ = [("W1", c_void_p), ("b1", c_void_p), ("w2", c_void_p), ("b2", c_void_p),
                ("log_gamma", c_void_p), ("input_kind", c_int32), ("activation", c_int32)]


ACTIVATIONS = {"gelu": 0, "silu": 1, "identity": 2}


class kvpop_mlstm_scorer(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in ("Wq", "Wk", "Wv", "wi", "wf", "bi", "bf", "a", "b",
                                        "log_gamma")]


_P = c_void_p
_SIGS = {
    "kvpop_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "kvpop_init_cache": (ctypes.c_int, [POINTER(kvpop_config), POINTER(kvpop_scorer), _P, POINTER(_P)]),
    "kvpop_init_cache_mlstm": (ctypes.c_int, [POINTER(kvpop_config), POINTER(kvpop_mlstm_scorer), _P,
                                              POINTER(_P)]),
    "kvpop_free": (ctypes.c_int, [_P]),
    "kvpop_prefill_compress": (ctypes.c_int, [_P, _P, _P, _P, POINTER(c_int32), c_int32, c_int32,
                                              c_int32, _P, _P]),
    "kvpop_decode_ingest": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P]),
    "kvpop_decode_attend": (ctypes.c_int, [_P, _P, _P, _P]),
    "kvpop_decode_step": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "kvpop_decode_step_host": (ctypes.c_int, [_P, _P, _P, _P, _P, _P]),
    "kvpop_step_is_fused": (c_int32, [_P]),
    "kvpop_check": (ctypes.c_int, [_P, _P]),
    "kvpop_export_state": (ctypes.c_int, [_P, _P, POINTER(c_size_t), _P]),
    "kvpop_import_state": (ctypes.c_int, [_P, _P, c_size_t, _P]),
    "kvpop_get_lengths": (ctypes.c_int, [_P, POINTER(c_int32), _P]),
    "kvpop_get_pair_state": (ctypes.c_int, [_P, c_int32, c_int32, POINTER(c_int32), POINTER(c_float),
                                            POINTER(c_int32), _P]),
    "kvpop_attend_noalloc": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, c_int32, c_int32, c_int32,
                                            c_int32, c_int32, c_int32, ctypes.c_int, _P]),
    "kvpop_prefill_attend": (ctypes.c_int, [_P, _P, _P, _P, POINTER(c_int32), c_int32, c_int32,
                                            c_int32, _P, _P, _P, _P, _P, _P, _P]),
    "kvpop_topk_workspace_bytes": (c_size_t, [c_int32, c_int32]),
    "kvpop_topk_cutoff": (ctypes.c_int, [_P, _P, c_int32, c_int32, c_int32, c_int32, c_int32, _P, _P,
                                         _P, _P, c_size_t, _P]),
    "kvpop_prompt_attention": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, c_int32, c_int32, c_int32,
                                              c_int32, c_int32, c_int32, c_int32, c_int32,
                                              ctypes.c_int, _P, _P, _P]),
    "kvpop_causal_lse": (ctypes.c_int, [_P, _P, _P, c_int32, c_int32, c_int32, c_int32, c_int32,
                                        ctypes.c_int, _P, _P]),
    "kvpop_future_target": (ctypes.c_int, [_P, _P, _P, _P, c_int32, c_int32, c_int32, c_int32, c_int32,
                                           c_int32, c_int32, ctypes.c_int, _P, _P, c_int32, c_int32,
                                           c_float, _P]),
    "kvpop_standalone_status": (ctypes.c_int, [_P]),
    "kvpop_last_error": (ctypes.c_char_p, []),
    "kvpop_debug_fail_alloc_after": (None, [c_int32]),
    "kvpop_debug_skip_attention_copies": (None, [c_int32]),
}
for _name, (_res, _args) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args
    globals()[_name] = _fn

EXPORTED = tuple(_SIGS)


class KVpopError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        msg = kvpop_status_string(status).decode()
        last = kvpop_last_error().decode()
        super().__init__(f"{what}: {STATUS.get(status, status)} ({msg})" + (f" [{last}]" if last else ""))


def _ck(status: int, what: str):
    if status != 0:
        raise KVpopError(status, what)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream=None) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def dtype_code(dtype) -> int:
    return KVPOP_F32 if dtype in ("f32", torch.float32) else KVPOP_BF16


class KVpopCache:
    """One attention layer's compressed KV cache (library-owned device state)."""

    def __init__(self, batch: int, n_kv_heads: int, q_per_kv: int, head_dim: int, budget_B: int,
                 delay_D: int, scorer_hidden: int, kv_dtype, W1=None, b1=None, w2=None, b2=None,
                 log_gamma=None, n_sink: int = 0, stream=None, mlstm: Optional[dict] = None,
                 activation: str = "gelu", kv_only: bool = False):
        """MLP scorer from ``W1, b1, w2, b2`` (``W1 [H][3d][F]`` on [k; v; qbar], or
        ``[H][2d][F]`` on [k; v] with ``kv_only``; hidden ``activation`` gelu / silu /
        identity); or, with ``mlstm`` (a dict of ``Wq, Wk, Wv, wi, wf, bi, bf, a, b`` and
        optionally ``log_gamma``), the stateful mLSTM scorer."""
        self.cfg = kvpop_config(batch, n_kv_heads, q_per_kv, head_dim, budget_B, delay_D, n_sink,
                                scorer_hidden, dtype_code(kv_dtype))
        h = _P()
        if mlstm is not None:
            names = ("Wq", "Wk", "Wv", "wi", "wf", "bi", "bf", "a", "b")
            keep = {n: mlstm[n].contiguous().float() for n in names}
            lg = mlstm.get("log_gamma")
            lg = None if lg is None else lg.contiguous().float()
            ms = kvpop_mlstm_scorer(*[keep[n].data_ptr() for n in names],
                                    None if lg is None else lg.data_ptr())
            _ck(kvpop_init_cache_mlstm(ctypes.byref(self.cfg), ctypes.byref(ms), _stream(stream),
                                       ctypes.byref(h)), "kvpop_init_cache_mlstm")
        else:
            keep = [t.contiguous().float() for t in (W1, b1, w2, b2)]
            lg = None if log_gamma is None else log_gamma.contiguous().float()
            sc = kvpop_scorer(*[t.data_ptr() for t in keep], None if lg is None else lg.data_ptr(),
                              1 if kv_only else 0, ACTIVATIONS[activation])
            _ck(kvpop_init_cache(ctypes.byref(self.cfg), ctypes.byref(sc), _stream(stream),
                                 ctypes.byref(h)), "kvpop_init_cache")
        self.handle = h.value
        self.mlstm = mlstm is not None
        self.batch, self.H, self.G, self.d = batch, n_kv_heads, q_per_kv, head_dim

    def prefill(self, Q, K, V, prompt_lens: Sequence[int], first_seq: int = 0, override=None,
                stream=None):
        n_seq = len(prompt_lens)
        arr = (c_int32 * n_seq)(*[int(x) for x in prompt_lens])
        Pmax = K.shape[2] if K is not None else 0
        _ck(kvpop_prefill_compress(self.handle, _ptr(Q), _ptr(K), _ptr(V), arr, first_seq, n_seq, Pmax,
                                   _ptr(override), _stream(stream)), "kvpop_prefill_compress")

    def prefill_attend(self, Q, K, V, prompt_lens: Sequence[int], Y, lse=None, first_seq: int = 0,
                       override=None, rank=None, tau=None, order=None, stream=None):
        """``prefill`` plus the prompt's outputs ``Y [n][H*G][Pmax][d]`` (fp32) under the
        running top-k mask; optionally the LSE, ranks and cutoffs."""
        n_seq = len(prompt_lens)
        arr = (c_int32 * n_seq)(*[int(x) for x in prompt_lens])
        Pmax = K.shape[2]
        _ck(kvpop_prefill_attend(self.handle, _ptr(Q), _ptr(K), _ptr(V), arr, first_seq, n_seq, Pmax,
                                 _ptr(override), _ptr(Y), _ptr(lse), _ptr(rank), _ptr(tau),
                                 _ptr(order), _stream(stream)), "kvpop_prefill_attend")

    def ingest(self, q, k, v, override=None, evict_info=None, score_out=None, stream=None):
        _ck(kvpop_decode_ingest(self.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(override),
                                _ptr(evict_info), _ptr(score_out), _stream(stream)), "kvpop_decode_ingest")

    def attend(self, q, out, stream=None):
        _ck(kvpop_decode_attend(self.handle, _ptr(q), _ptr(out), _stream(stream)), "kvpop_decode_attend")

    def step(self, q, k, v, out, override=None, evict_info=None, score_out=None, stream=None):
        _ck(kvpop_decode_step(self.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(override),
                              _ptr(evict_info), _ptr(score_out), _stream(stream)), "kvpop_decode_step")

    @property
    def fused_step(self) -> bool:
        """True when step() runs the whole decode step as one kernel."""
        return kvpop_step_is_fused(self.handle) == 1

    def step_host(self, q, k, v, out, stream=None):
        _ck(kvpop_decode_step_host(self.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(out), _stream(stream)),
            "kvpop_decode_step_host")

    def check(self, stream=None):
        _ck(kvpop_check(self.handle, _stream(stream)), "kvpop_check")

    def lengths(self, stream=None):
        arr = (c_int32 * self.batch)()
        _ck(kvpop_get_lengths(self.handle, arr, _stream(stream)), "kvpop_get_lengths")
        return list(arr)

    def pair_state(self, seq: int, head: int, stream=None):
        """(positions of the used slots in slot order, their priorities) of one KV head."""
        B = self.cfg.budget_B
        pos = (c_int32 * B)()
        sc = (c_float * B)()
        nv = c_int32(0)
        _ck(kvpop_get_pair_state(self.handle, seq, head, pos, sc, ctypes.byref(nv), _stream(stream)),
            "kvpop_get_pair_state")
        n = nv.value
        return list(pos)[:n], list(sc)[:n]

    def export_state(self, stream=None) -> bytes:
        n = c_size_t(0)
        _ck(kvpop_export_state(self.handle, None, ctypes.byref(n), _stream(stream)), "kvpop_export_state")
        buf = ctypes.create_string_buffer(n.value)
        _ck(kvpop_export_state(self.handle, buf, ctypes.byref(n), _stream(stream)), "kvpop_export_state")
        return buf.raw

    def import_state(self, blob: bytes, stream=None):
        _ck(kvpop_import_state(self.handle, blob, len(blob), _stream(stream)), "kvpop_import_state")

    def free(self):
        if getattr(self, "handle", None):
            _ck(kvpop_free(self.handle), "kvpop_free")
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def topk_cutoff(prio, n_sink: int, window: int, k: int, lengths=None, rank=None, tau=None,
                order=None, stream=None):
    """Static ranks and running top-k cutoffs of each row of ``prio [n_rows][S]`` (fp32, CUDA)."""
    n_rows, S = prio.shape
    dev = prio.device
    rank = torch.empty((n_rows, S), dtype=torch.int32, device=dev) if rank is None else rank
    tau = torch.empty((n_rows, S), dtype=torch.int32, device=dev) if tau is None else tau
    nb = int(kvpop_topk_workspace_bytes(n_rows, S))
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device=dev)
    _ck(kvpop_topk_cutoff(_ptr(prio), _ptr(lengths), n_rows, S, n_sink, window, k, _ptr(rank),
                          _ptr(tau), _ptr(order), _ptr(ws), nb, _stream(stream)), "kvpop_topk_cutoff")
    return rank, tau


def prompt_attention(Q, K, V, rank, tau, n_sink: int, window: int, k: int, lengths=None, Y=None,
                     lse=None, want_lse: bool = True, order=None, stream=None):
    """Masked causal attention under the running top-k mask.  ``Q [n][H*G][S][d]``,
    ``K, V [n][H][S][d]``, ``rank, tau [n][H][S]``; returns (Y fp32, LSE fp32 or None)."""
    n_seq, H, S, d = K.shape
    G = Q.shape[1] // H
    dev = K.device
    Y = torch.empty((n_seq, H * G, S, d), dtype=torch.float32, device=dev) if Y is None else Y
    if lse is None and want_lse:
        lse = torch.empty((n_seq, H * G, S), dtype=torch.float32, device=dev)
    _ck(kvpop_prompt_attention(_ptr(Q), _ptr(K), _ptr(V), _ptr(rank), _ptr(tau), _ptr(order),
                               _ptr(lengths), n_seq,
                               H, G, d, S, n_sink, window, k, dtype_code(K.dtype), _ptr(Y), _ptr(lse),
                               _stream(stream)), "kvpop_prompt_attention")
    return Y, lse


def causal_lse(Q, K, lengths=None, lse=None, stream=None):
    """Dense causal log-normalisers ``[n][H*G][S]`` (fp32) of ``Q [n][H*G][S][d]`` against
    ``K [n][H][S][d]``."""
    n_seq, H, S, d = K.shape
    G = Q.shape[1] // H
    lse = torch.empty((n_seq, H * G, S), dtype=torch.float32, device=K.device) if lse is None else lse
    _ck(kvpop_causal_lse(_ptr(Q), _ptr(K), _ptr(lengths), n_seq, H, G, d, S, dtype_code(K.dtype),
                         _ptr(lse), _stream(stream)), "kvpop_causal_lse")
    return lse


def future_target(Q, K, lse, window: int, lookahead: int = 0, agg: str = "max",
                  count_norm: bool = True, eps: float = 1e-6, lengths=None, want_target: bool = True,
                  logm=None, target=None, stream=None):
    """Per-head future log masses ``[n][H*G][S]`` and, optionally, the per-KV-head target
    ``[n][H][S]`` (both fp32)."""
    n_seq, H, S, d = K.shape
    G = Q.shape[1] // H
    dev = K.device
    logm = torch.empty((n_seq, H * G, S), dtype=torch.float32, device=dev) if logm is None else logm
    if target is None and want_target:
        target = torch.empty((n_seq, H, S), dtype=torch.float32, device=dev)
    _ck(kvpop_future_target(_ptr(Q), _ptr(K), _ptr(lse), _ptr(lengths), n_seq, H, G, d, S, window,
                            lookahead, dtype_code(K.dtype), _ptr(logm), _ptr(target),
                            0 if agg == "max" else 1, int(bool(count_norm)), float(eps),
                            _stream(stream)), "kvpop_future_target")
    return logm, target


def parse_state(blob: bytes, cfg: kvpop_config) -> dict:
    """Split a ``kvpop_export_state`` blob into named numpy arrays (checkpoint inspection)."""
    import numpy as np
    pairs = cfg.batch * cfg.n_kv_heads
    B, D, d = cfg.budget_B, cfg.delay_D, cfg.head_dim
    kv_np = np.float32 if cfg.kv_dtype == KVPOP_F32 else np.uint16   # bf16 kept as raw bits
    esz = 4 if cfg.kv_dtype == KVPOP_F32 else 2
    layout = [("slotK", kv_np, (pairs, B, d), esz), ("slotV", kv_np, (pairs, B, d), esz),
              ("ringK", kv_np, (pairs, D, d), esz), ("ringV", kv_np, (pairs, D, d), esz),
              ("ringQm", np.float32, (pairs, D, d), 4), ("score", np.float32, (pairs, B), 4),
              ("pos", np.int32, (pairs, B), 4), ("nvalid", np.int32, (pairs,), 4),
              ("len", np.int32, (pairs,), 4), ("min_score", np.float32, (pairs,), 4),
              ("min_slot", np.int32, (pairs,), 4),
              ("blk_score", np.float32, (pairs, (B + 63) // 64), 4),
              ("blk_slot", np.int32, (pairs, (B + 63) // 64), 4),
              ("mlstm_C", np.float32, (pairs, d, d // 2), 4), ("mlstm_z", np.float32, (pairs, d), 4),
              ("mlstm_m", np.float32, (pairs,), 4)]
    off = 4 * 8 + ctypes.sizeof(kvpop_config)
    out = {}
    for name, dt, shape, sz in layout:
        n = int(np.prod(shape)) * sz
        if name.startswith("mlstm_") and off + n > len(blob):
            break                                   # MLP-scorer caches have no recurrent state
        out[name] = np.frombuffer(blob, dtype=dt, count=int(np.prod(shape)), offset=off).reshape(shape)
        off += n
    return out
