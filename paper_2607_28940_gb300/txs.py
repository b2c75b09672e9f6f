"""Thin ctypes binding of libtxs (include/txs.h): argument marshalling only.

Every step of the serving path runs in the library's CUDA kernels; this module
converts Python/NumPy/torch arguments to the C ABI and raises ``TxsError`` on a
non-zero status.  PyTorch provides device memory and streams.  If libtxs.so is
missing the binding raises: there is no other implementation to fall back on.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence, Tuple

import numpy as np
import torch

from . import workload as W

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libtxs.so")

TXS_OK = 0
TXS_ERR_INVALID_ARG = 1
TXS_ERR_COLD_START = 2
TXS_ERR_CAPACITY = 3
TXS_ERR_STALE_CACHE = 4
TXS_ERR_CUDA = 5
TXS_ERR_DEVICE_TIMEOUT = 6
TXS_ERR_BOUNDS = 7
TXS_ERR_UNSUPPORTED = 8

TXS_FP32, TXS_BF16 = 0, 1
LOCAL_GLOBAL, FULL = 0, 1
N_KERNEL_CLASSES = 24


class TxsError(RuntimeError):
    def __init__(self, status: int, what: str, detail: str = ""):
        self.status = status
        msg = f"{what}: {status_string(status)} ({status})"
        if detail:
            msg += f" [{detail}]"
        super().__init__(msg)


class txs_config(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("n_actions", ctypes.c_int32), ("n_ctx", ctypes.c_int32),
                ("l_local", ctypes.c_int32), ("attn_mode", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("ln_eps", ctypes.c_float), ("n_kv_heads", ctypes.c_int32), ("cand_mlp_hidden", ctypes.c_int32),
                ("head_dw_hidden", ctypes.c_int32), ("head_dw_in", ctypes.c_int32), ("head_dw_out", ctypes.c_int32)]


class txs_enc_config(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("type_dim", ctypes.c_int32), ("n_types", ctypes.c_int32),
                ("n_rel", ctypes.c_int32), ("window", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("ln_eps", ctypes.c_float)]


_lib: Optional[ctypes.CDLL] = None

_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I32P = ctypes.POINTER(ctypes.c_int32)

_SIGS = {
    "txs_model_create": (_I32, [ctypes.POINTER(txs_config), ctypes.POINTER(_P), ctypes.POINTER(_P)]),
    "txs_model_destroy": (None, [_P]),
    "txs_model_hash": (ctypes.c_uint64, [_P]),
    "txs_build_kv_cache": (_I32, [_P, _I32, _I32P, _P, _I32, _P, ctypes.POINTER(_P)]),
    "txs_cache_destroy": (None, [_P]),
    "txs_rebuild_kv_cache": (_I32, [_P, _P, _I32, _I32P, _P, _P]),
    "txs_append_behavior": (_I32, [_P, _P, _I32, _I32P, _P, _P]),
    "txs_rebuild_append_kv_cache": (_I32, [_P, _P, _I32, _I32P, _P, _I32P, _P, _P]),
    "txs_cache_read_rows": (_I32, [_P, _I32, _I32, _I32, _I32, _I32, _P, _P]),
    "txs_cache_read_anchor": (_I32, [_P, _I32, _I32, _P, _P]),
    "txs_cache_lengths": (_I32, [_P, _I32P]),
    "txs_cache_export_size": (_I32, [_P, ctypes.POINTER(ctypes.c_size_t)]),
    "txs_cache_export": (_I32, [_P, ctypes.c_uint32, _P, ctypes.c_size_t, _P]),
    "txs_cache_import": (_I32, [_P, ctypes.c_uint32, _P, ctypes.c_size_t, _I32, _P, ctypes.POINTER(_P)]),
    "txs_cache_n_req": (_I32, [_P]),
    "txs_score_workspace_size": (_I32, [_P, _I32, ctypes.c_int64, ctypes.POINTER(ctypes.c_size_t)]),
    "txs_score_candidates": (_I32, [_P, _P, _I32, _I32P, _P, _P, _P, ctypes.c_size_t, _P, _P, _P]),
    "txs_score_candidates_after": (_I32, [_P, _P, _I32, _I32P, _P, _P, _P, ctypes.c_size_t, _P, _P, _P, _P]),
    "txs_rank_candidates": (_I32, [_I32, _I32P, _P, _I32, _I32, _I32, _P, _P]),
    "txs_events_workspace_size": (_I32, [_P, _I32, ctypes.c_int64, _I32, ctypes.POINTER(ctypes.c_size_t)]),
    "txs_score_events": (_I32, [_P, _P, _I32, _P, _I32, _I32P, _I32P, _P, _P, _P, ctypes.c_size_t, _P, _P, _P]),
    "txs_device_status": (_I32, [_P]),
    "txs_encoder_create": (_I32, [ctypes.POINTER(txs_enc_config), ctypes.POINTER(_P), ctypes.POINTER(_P)]),
    "txs_encoder_destroy": (None, [_P]),
    "txs_encoder_hash": (ctypes.c_uint64, [_P]),
    "txs_encoder_workspace_size": (_I32, [_P, ctypes.c_int64, ctypes.POINTER(ctypes.c_size_t)]),
    "txs_encode_build": (_I32, [_P, _I32, _I32P, _P, _P, _I32, _P, ctypes.c_size_t, _P, _P, ctypes.POINTER(_P)]),
    "txs_encode_append": (_I32, [_P, _P, _I32, _I32P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "txs_enc_state_lengths": (_I32, [_P, _I32P]),
    "txs_enc_state_n_req": (_I32, [_P]),
    "txs_enc_state_read_rows": (_I32, [_P, _I32, _I32, _I32, _I32, _I32, _P, _P]),
    "txs_enc_state_destroy": (None, [_P]),
    "txs_encoder_device_status": (_I32, [_P]),
    "txs_pool_anchor_static": (_I32, [_P, _I32, _I32P, _P, _P, _P]),
    "txs_gelu_eval": (_I32, [_P, _P, ctypes.c_int64, _I32, _P]),
    "txs_selftest_wait_timeout": (_I32, [_P, _P]),
    "txs_profile_enable": (_I32, [_I32]),
    "txs_profile_collect": (_I32, [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64), _I32]),
    "txs_kernel_class_name": (ctypes.c_char_p, [_I32]),
    "txs_status_string": (ctypes.c_char_p, [_I32]),
    "txs_last_error": (ctypes.c_char_p, []),
    "txs_version": (ctypes.c_char_p, []),
}


def lib() -> ctypes.CDLL:
    """The loaded libtxs.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run paper_2607_28940_gb300.build.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(s: int) -> str:
    return lib().txs_status_string(s).decode()


def last_error() -> str:
    return lib().txs_last_error().decode()


def _check(st: int, what: str):
    if st != TXS_OK:
        raise TxsError(st, what, last_error() if st == TXS_ERR_CUDA or st == TXS_ERR_UNSUPPORTED else "")


def _offsets(off) -> Tuple[np.ndarray, ctypes.Array]:
    a = np.ascontiguousarray(np.asarray(off, dtype=np.int32))
    return a, a.ctypes.data_as(_I32P)


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CUDA tensor")
    return t.data_ptr()


def torch_dtype(dtype: str) -> torch.dtype:
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def kv_width(wl: W.Workload) -> int:
    """Width of a cached K or V row: n_kv_heads * d_head."""
    return (wl.n_kv_heads or wl.n_heads) * (wl.d_model // wl.n_heads)


def make_config(wl: W.Workload, mode: int = LOCAL_GLOBAL) -> txs_config:
    return txs_config(wl.d_model, wl.n_heads, wl.d_ff, wl.n_layers, wl.n_actions, wl.n_ctx, wl.l_local, mode,
                      TXS_BF16 if wl.dtype == "bf16" else TXS_FP32, wl.ln_eps, wl.n_kv_heads, wl.cand_mlp,
                      wl.dw_hidden, wl.dw_in, wl.dw_out)


def weight_order(n_layers: int, cand_mlp: int = 0, dw_hidden: int = 0) -> Sequence[str]:
    """Names of the weight tensors in the order of txs_model_create."""
    names = [f"{n}.{l}" for l in range(n_layers) for n, _ in W.LAYER_WEIGHTS]
    names += [n for n, _ in W.HEAD_WEIGHTS]
    names += [n for n, _ in W.CAND_WEIGHTS] if cand_mlp else []
    return names + ([n for n, _ in W.DW_WEIGHTS] if dw_hidden else [])


class Model:
    """A decoder model on the GPU (txs_model)."""

    def __init__(self, wl: W.Workload, weights: Dict[str, np.ndarray], mode: int = LOCAL_GLOBAL,
                 device: str = "cuda"):
        self.wl = wl
        self.mode = mode
        self.dtype = torch_dtype(wl.dtype)
        self.cfg = make_config(wl, mode)
        names = weight_order(wl.n_layers, wl.cand_mlp, wl.dw_hidden)
        dev = [torch.as_tensor(np.asarray(weights[n]), dtype=torch.float32).to(device).to(self.dtype).contiguous()
               if n in weights and np.asarray(weights[n]).size else None for n in names]
        ptrs = (_P * len(dev))(*[t.data_ptr() if t is not None else None for t in dev])
        h = _P()
        _check(lib().txs_model_create(ctypes.byref(self.cfg), ptrs, ctypes.byref(h)), "txs_model_create")
        self.handle = h
        del dev  # the library keeps its own copy

    @property
    def hash(self) -> int:
        return int(lib().txs_model_hash(self.handle))

    def device_status(self) -> int:
        return int(lib().txs_device_status(self.handle))

    def selftest_wait_timeout(self) -> None:
        """Enqueue the bounded-wait self-test; device_status() then reports the timeout."""
        _check(lib().txs_selftest_wait_timeout(self.handle, _stream(None)), "txs_selftest_wait_timeout")

    def close(self):
        if getattr(self, "handle", None):
            lib().txs_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class KVCache:
    """Per-request behavior K/V cache (txs_kv_cache)."""

    def __init__(self, model: Model, beh_offsets, beh_enc: torch.Tensor, capacity_extra: int = 0, stream=None):
        off, p = _offsets(beh_offsets)
        self.n_req = len(off) - 1
        self.model = model
        h = _P()
        _check(lib().txs_build_kv_cache(model.handle, self.n_req, p, _ptr(beh_enc), int(capacity_extra),
                                        _stream(stream), ctypes.byref(h)), "txs_build_kv_cache")
        self.handle = h

    def rebuild(self, beh_offsets, beh_enc: torch.Tensor, stream=None):
        off, p = _offsets(beh_offsets)
        _check(lib().txs_rebuild_kv_cache(self.model.handle, self.handle, len(off) - 1, p, _ptr(beh_enc),
                                          _stream(stream)), "txs_rebuild_kv_cache")

    def rebuild_append(self, beh_offsets, beh_enc: torch.Tensor, new_offsets, new_enc: Optional[torch.Tensor],
                       stream=None):
        """rebuild(beh_offsets, beh_enc) then append(new_offsets, new_enc) in one
        call (txs_rebuild_append_kv_cache)."""
        off, p = _offsets(beh_offsets)
        noff, np_ = _offsets(new_offsets)
        _check(lib().txs_rebuild_append_kv_cache(self.model.handle, self.handle, len(off) - 1, p, _ptr(beh_enc), np_,
                                                 _ptr(new_enc) if new_enc is not None and new_enc.numel() else None,
                                                 _stream(stream)), "txs_rebuild_append_kv_cache")

    def append(self, new_offsets, new_enc: Optional[torch.Tensor], stream=None, model: Optional[Model] = None):
        off, p = _offsets(new_offsets)
        m = model or self.model
        _check(lib().txs_append_behavior(m.handle, self.handle, len(off) - 1, p, _ptr(new_enc), _stream(stream)),
               "txs_append_behavior")

    def lengths(self) -> np.ndarray:
        out = np.zeros(self.n_req, dtype=np.int32)
        _check(lib().txs_cache_lengths(self.handle, out.ctypes.data_as(_I32P)), "txs_cache_lengths")
        return out

    def read_rows(self, layer: int, which: int, req: int, row0: int, n_rows: int, stream=None) -> torch.Tensor:
        out = torch.empty((n_rows, kv_width(self.model.wl)), dtype=self.model.dtype, device="cuda")
        _check(lib().txs_cache_read_rows(self.handle, layer, which, req, row0, n_rows, _ptr(out), _stream(stream)),
               "txs_cache_read_rows")
        return out

    def read_anchor(self, layer: int, which: int, stream=None) -> torch.Tensor:
        width = self.model.wl.d_model if which == 2 else kv_width(self.model.wl)
        out = torch.empty((self.n_req, width), dtype=torch.float32, device="cuda")
        _check(lib().txs_cache_read_anchor(self.handle, layer, which, _ptr(out), _stream(stream)),
               "txs_cache_read_anchor")
        return out

    def export(self, schema_version: int = 0, stream=None) -> np.ndarray:
        """The cache serialised into a host byte array (txs_cache_export)."""
        n = ctypes.c_size_t()
        _check(lib().txs_cache_export_size(self.handle, ctypes.byref(n)), "txs_cache_export_size")
        buf = np.empty(int(n.value), dtype=np.uint8)
        _check(lib().txs_cache_export(self.handle, int(schema_version), buf.ctypes.data, buf.size, _stream(stream)),
               "txs_cache_export")
        return buf

    @classmethod
    def import_blob(cls, model: Model, blob: np.ndarray, schema_version: int = 0, capacity_extra: int = 0,
                    stream=None) -> "KVCache":
        """A cache rebuilt from an exported blob (txs_cache_import)."""
        blob = np.ascontiguousarray(blob, dtype=np.uint8)
        h = _P()
        _check(lib().txs_cache_import(model.handle, int(schema_version), blob.ctypes.data, blob.size,
                                      int(capacity_extra), _stream(stream), ctypes.byref(h)), "txs_cache_import")
        self = cls.__new__(cls)
        self.model = model
        self.handle = h
        self.n_req = int(lib().txs_cache_n_req(h))
        return self

    def close(self):
        if getattr(self, "handle", None):
            lib().txs_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def workspace_bytes(model: Model, n_req: int, total_cand: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().txs_score_workspace_size(model.handle, n_req, total_cand, ctypes.byref(n)), "workspace_size")
    return int(n.value)


def score(model: Model, cache: KVCache, cand_offsets, cand_tok: torch.Tensor, ctx_tok: Optional[torch.Tensor],
          workspace: Optional[torch.Tensor] = None, out_logits: Optional[torch.Tensor] = None,
          out_probs: Optional[torch.Tensor] = None, want_probs: bool = True, stream=None,
          cache_ready: Optional[torch.cuda.Event] = None):
    """Scores of all candidates: (logits, probs) as [sum M, k] float32 CUDA tensors.
    With ``cache_ready`` (an event recorded after the cache's last write on
    another stream), the work that does not read the cache starts at once
    (txs_score_candidates_after)."""
    off, p = _offsets(cand_offsets)
    n_req = len(off) - 1
    n_cand = int(off[-1])
    k = model.wl.n_actions
    if workspace is None:
        workspace = torch.empty(max(workspace_bytes(model, n_req, n_cand), 256), dtype=torch.uint8, device="cuda")
    if out_logits is None:
        out_logits = torch.empty((n_cand, k), dtype=torch.float32, device="cuda")
    if out_probs is None and want_probs:
        out_probs = torch.empty((n_cand, k), dtype=torch.float32, device="cuda")
    if cache_ready is not None:
        _check(lib().txs_score_candidates_after(model.handle, cache.handle, n_req, p, _ptr(cand_tok), _ptr(ctx_tok),
                                                _ptr(workspace), workspace.numel(), _ptr(out_logits),
                                                _ptr(out_probs), cache_ready.cuda_event, _stream(stream)),
               "txs_score_candidates_after")
    else:
        _check(lib().txs_score_candidates(model.handle, cache.handle, n_req, p, _ptr(cand_tok), _ptr(ctx_tok),
                                          _ptr(workspace), workspace.numel(), _ptr(out_logits), _ptr(out_probs),
                                          _stream(stream)), "txs_score_candidates")
    return out_logits, out_probs


def events_workspace_bytes(model: Model, n_events: int, total_cand: int, max_event_end: int) -> int:
    n = ctypes.c_size_t()
    _check(lib().txs_events_workspace_size(model.handle, n_events, total_cand, max_event_end, ctypes.byref(n)),
           "events_workspace_size")
    return int(n.value)


def score_events(model: Model, cache: KVCache, user: int, beh_enc: torch.Tensor, event_ends, cand_offsets,
                 cand_tok: torch.Tensor, ctx_tok: Optional[torch.Tensor], workspace: Optional[torch.Tensor] = None,
                 out_logits: Optional[torch.Tensor] = None, out_probs: Optional[torch.Tensor] = None,
                 want_probs: bool = True, stream=None):
    """Streaming multi-event scores of request ``user`` of ``cache`` (txs_score_events):
    event t sees the first event_ends[t] rows of the user's stream ``beh_enc``."""
    ends = np.ascontiguousarray(np.asarray(event_ends, dtype=np.int32))
    off, p = _offsets(cand_offsets)
    n_ev = len(off) - 1
    if len(ends) != n_ev:
        raise ValueError("one event end per slate")
    n_cand = int(off[-1])
    k = model.wl.n_actions
    if workspace is None:
        max_end = int(ends.max()) if len(ends) else 0
        workspace = torch.empty(max(events_workspace_bytes(model, n_ev, n_cand, max_end), 256), dtype=torch.uint8,
                                device="cuda")
    if out_logits is None:
        out_logits = torch.empty((n_cand, k), dtype=torch.float32, device="cuda")
    if out_probs is None and want_probs:
        out_probs = torch.empty((n_cand, k), dtype=torch.float32, device="cuda")
    _check(lib().txs_score_events(model.handle, cache.handle, int(user), _ptr(beh_enc), n_ev,
                                  ends.ctypes.data_as(_I32P), p, _ptr(cand_tok), _ptr(ctx_tok), _ptr(workspace),
                                  workspace.numel(), _ptr(out_logits), _ptr(out_probs), _stream(stream)),
           "txs_score_events")
    return out_logits, out_probs


def rank(cand_offsets, probs: torch.Tensor, n_actions: int, action: int = 0, top_k: int = 0,
         out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    off, p = _offsets(cand_offsets)
    n_req = len(off) - 1
    if out is None:
        n = int(off[-1]) if top_k == 0 else n_req * top_k
        out = torch.empty(max(n, 1), dtype=torch.int32, device="cuda")
    _check(lib().txs_rank_candidates(n_req, p, _ptr(probs) if probs is not None and probs.numel() else None,
                                     n_actions, action, top_k, _ptr(out), _stream(stream)), "txs_rank_candidates")
    return out


def pool_anchor_static(model: Model, beh_offsets, beh_enc: torch.Tensor, out: Optional[torch.Tensor] = None,
                       stream=None) -> torch.Tensor:
    """Pooled anchor g [n_req, d] without any device allocation inside the
    library (for callers that cannot allocate while serving; `out` may be
    preallocated by the caller)."""
    off, p = _offsets(beh_offsets)
    n_req = len(off) - 1
    if out is None:
        out = torch.empty((n_req, model.wl.d_model), dtype=torch.float32, device="cuda")
    _check(lib().txs_pool_anchor_static(model.handle, n_req, p, _ptr(beh_enc), _ptr(out), _stream(stream)),
           "txs_pool_anchor_static")
    return out


# ---------------------------------------------------------------- behavior encoder

def make_enc_config(ew: W.EncWorkload) -> txs_enc_config:
    return txs_enc_config(ew.d_model, ew.n_heads, ew.d_ff, ew.n_layers, ew.type_dim, ew.n_types, ew.n_rel,
                          ew.window, TXS_BF16 if ew.dtype == "bf16" else TXS_FP32, ew.ln_eps)


def enc_weight_order(ew: W.EncWorkload) -> Sequence[str]:
    """Names of the encoder weight tensors in the order of txs_encoder_create."""
    names = [f"{n}.{l}" for l in range(ew.n_layers) for n, _ in W.ENC_LAYER_WEIGHTS]
    return names + ([n for n, _ in W.ENC_TYPE_WEIGHTS] if ew.type_dim else [])


class Encoder:
    """The behavior-stream encoder on the GPU (txs_encoder)."""

    def __init__(self, ew: W.EncWorkload, weights: Dict[str, np.ndarray], device: str = "cuda"):
        self.ew = ew
        self.dtype = torch_dtype(ew.dtype)
        self.cfg = make_enc_config(ew)
        dev = [torch.as_tensor(np.asarray(weights[n]), dtype=torch.float32).to(device).to(self.dtype).contiguous()
               for n in enc_weight_order(ew)]
        ptrs = (_P * len(dev))(*[t.data_ptr() for t in dev])
        h = _P()
        _check(lib().txs_encoder_create(ctypes.byref(self.cfg), ptrs, ctypes.byref(h)), "txs_encoder_create")
        self.handle = h
        del dev

    @property
    def hash(self) -> int:
        return int(lib().txs_encoder_hash(self.handle))

    def workspace_bytes(self, n_rows: int) -> int:
        n = ctypes.c_size_t()
        _check(lib().txs_encoder_workspace_size(self.handle, int(n_rows), ctypes.byref(n)), "workspace_size")
        return int(n.value)

    def device_status(self) -> int:
        return int(lib().txs_encoder_device_status(self.handle))

    def close(self):
        if getattr(self, "handle", None):
            lib().txs_encoder_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _enc_io(enc: Encoder, off: np.ndarray, workspace, phi_out):
    n = int(off[-1])
    if workspace is None:
        workspace = torch.empty(max(enc.workspace_bytes(n), 256), dtype=torch.uint8, device="cuda")
    if phi_out is None:
        phi_out = torch.empty((n, enc.ew.d_model), dtype=enc.dtype, device="cuda")
    return workspace, phi_out


class EncState:
    """Per-user encoder state: every layer's K/V rows (txs_enc_state)."""

    def __init__(self, enc: Encoder, offsets, subj: torch.Tensor, types: Optional[torch.Tensor],
                 capacity_extra: int = 0, workspace: Optional[torch.Tensor] = None,
                 phi_out: Optional[torch.Tensor] = None, stream=None):
        """Encode each user's stream from its first token (txs_encode_build);
        the encoded rows are in ``self.phi``."""
        off, p = _offsets(offsets)
        self.enc = enc
        self.n_req = len(off) - 1
        workspace, phi_out = _enc_io(enc, off, workspace, phi_out)
        h = _P()
        _check(lib().txs_encode_build(enc.handle, self.n_req, p, _ptr(subj) if subj.numel() else None,
                                      _ptr(types) if types is not None and types.numel() else None,
                                      int(capacity_extra), _ptr(workspace), workspace.numel(),
                                      _ptr(phi_out) if phi_out.numel() else None, _stream(stream), ctypes.byref(h)),
               "txs_encode_build")
        self.handle = h
        self.phi = phi_out

    def append(self, new_offsets, subj: torch.Tensor, types: Optional[torch.Tensor],
               workspace: Optional[torch.Tensor] = None, phi_out: Optional[torch.Tensor] = None,
               stream=None, enc: Optional[Encoder] = None) -> torch.Tensor:
        """Encode new tokens after each user's current ones (txs_encode_append);
        returns their encoded rows."""
        off, p = _offsets(new_offsets)
        e = enc or self.enc
        workspace, phi_out = _enc_io(e, off, workspace, phi_out)
        _check(lib().txs_encode_append(e.handle, self.handle, len(off) - 1, p, _ptr(subj) if subj.numel() else None,
                                       _ptr(types) if types is not None and types.numel() else None,
                                       _ptr(workspace), workspace.numel(),
                                       _ptr(phi_out) if phi_out.numel() else None, _stream(stream)),
               "txs_encode_append")
        return phi_out

    def lengths(self) -> np.ndarray:
        out = np.zeros(self.n_req, dtype=np.int32)
        _check(lib().txs_enc_state_lengths(self.handle, out.ctypes.data_as(_I32P)), "txs_enc_state_lengths")
        return out

    def read_rows(self, layer: int, which: int, req: int, row0: int, n_rows: int, stream=None) -> torch.Tensor:
        out = torch.empty((n_rows, self.enc.ew.d_model), dtype=self.enc.dtype, device="cuda")
        _check(lib().txs_enc_state_read_rows(self.handle, layer, which, req, row0, n_rows,
                                             _ptr(out) if n_rows else None, _stream(stream)),
               "txs_enc_state_read_rows")
        return out

    def close(self):
        if getattr(self, "handle", None):
            lib().txs_enc_state_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def gelu_eval(x: torch.Tensor, variant: int = 0) -> torch.Tensor:
    """The FFN epilogues' GELU on a device float32 tensor (variant 0: bf16
    tensor-core epilogue, 1: fp32 path)."""
    assert x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()
    y = torch.empty_like(x)
    _check(lib().txs_gelu_eval(ctypes.c_void_p(x.data_ptr()), ctypes.c_void_p(y.data_ptr()), x.numel(), variant,
                               _stream(None)), "txs_gelu_eval")
    return y


def profile_enable(on: bool = True):
    _check(lib().txs_profile_enable(1 if on else 0), "txs_profile_enable")


def profile_collect() -> Dict[str, Tuple[float, int]]:
    ms = (ctypes.c_double * N_KERNEL_CLASSES)()
    cnt = (ctypes.c_int64 * N_KERNEL_CLASSES)()
    _check(lib().txs_profile_collect(ms, cnt, N_KERNEL_CLASSES), "txs_profile_collect")
    out = {}
    for i in range(N_KERNEL_CLASSES):
        name = lib().txs_kernel_class_name(i).decode()
        if name and cnt[i]:
            out[name] = (float(ms[i]), int(cnt[i]))
    return out


def to_device(a: np.ndarray, dtype: torch.dtype) -> torch.Tensor:
    """Host array (already rounded to the storage type) -> contiguous CUDA tensor."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to("cuda").to(dtype).contiguous()
