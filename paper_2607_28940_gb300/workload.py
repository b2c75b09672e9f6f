"""Seeded synthetic workloads for the TransX serving path.

This module only draws numbers: model weights, behavior encodings, serving
context tokens, candidate tokens and appended behavior rows.  It contains none
of the method's arithmetic, so both the fp64 oracle (via the tests) and the
CUDA path consume exactly the same arrays.

Shapes follow the workloads the paper serves (Sec. 4.3: ~500 candidates per
request on average, long behavior histories, L_local = 10 from Sec. 5.1), with
distributions stated for the synthetic stand-ins: inputs ~ N(0, 1), weights and
biases ~ N(0, 0.02), LayerNorm gain 1 + N(0, 0.02) and bias N(0, 0.02).

Random streams.  ``np.random.SeedSequence(seed)`` is split into three
independent PCG64 streams: one for per-request sizes, one for weights, and one
parent from which request ``r`` gets its own child stream.  Request ``r``'s data
therefore depends only on (seed, r, its sizes), which lets a test regenerate a
subset of requests of a large workload.

Storage rounding.  For bf16 workloads every drawn value is rounded to the
nearest bf16 (ties to even) and kept as float32, so the oracle sees exactly the
values the GPU receives.

Weight names follow the paper's notation (Sec. 4.1.2, Sec. 4.1.3, App. B):
per decoder layer ``l`` the serving-stream attention (``W_qkv``, ``b_qkv``,
``W_os``, ``b_os``, ``ln1_g``, ``ln1_b``), the cross-attention (``W_Q``,
``b_Q``, ``W_K``, ``b_K``, ``W_V``, ``b_V``, ``W_oc``, ``b_oc``, ``ln2_g``,
``ln2_b``) and the FFN (``W_1``, ``b_1``, ``W_2``, ``b_2``, ``ln3_g``,
``ln3_b``); then the head: ``w_pool``, ``W_dec``, ``b_dec``, ``Q_dec``.
Matrices are stored in the row-vector convention ``y = x W + b`` with ``W`` of
shape ``[d_in, d_out]``.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional, Sequence, Tuple, Union

import numpy as np

LAYER_WEIGHTS: Tuple[Tuple[str, str], ...] = (
    # (name, shape code) in draw order; shape codes resolved by _shape()
    ("W_qkv", "d,3d"), ("b_qkv", "3d"), ("W_os", "d,d"), ("b_os", "d"),
    ("ln1_g", "d"), ("ln1_b", "d"),
    ("W_Q", "d,d"), ("b_Q", "d"), ("W_K", "d,dkv"), ("b_K", "dkv"),
    ("W_V", "d,dkv"), ("b_V", "dkv"), ("W_oc", "d,d"), ("b_oc", "d"),
    ("ln2_g", "d"), ("ln2_b", "d"),
    ("W_1", "d,F"), ("b_1", "F"), ("W_2", "F,d"), ("b_2", "d"),
    ("ln3_g", "d"), ("ln3_b", "d"),
)
HEAD_WEIGHTS: Tuple[Tuple[str, str], ...] = (
    ("w_pool", "d"), ("W_dec", "2d,d"), ("b_dec", "d"), ("Q_dec", "k,d"),
)
# candidate-to-query MLP (drawn after the head, only when cand_mlp > 0)
CAND_WEIGHTS: Tuple[Tuple[str, str], ...] = (
    ("W_c1", "d,Fc"), ("b_c1", "Fc"), ("W_c2", "Fc,d"), ("b_c2", "d"),
)

# Deep & Wide head (App. B; drawn last, only when dw_hidden > 0): the wide
# linear map of x[:, :dw_in] and the deep FFN of [z, x[:, dw_in:]]
DW_WEIGHTS: Tuple[Tuple[str, str], ...] = (
    ("W_w", "dwi,dwo"), ("b_w", "dwo"), ("W_d1", "dd,Fh"), ("b_d1", "Fh"), ("W_d2", "Fh,ddo"), ("b_d2", "ddo"),
)

SizeSpec = Union[int, Tuple[str, int, int], Sequence[int]]


@dataclass(frozen=True)
class Workload:
    name: str
    dtype: str              # "fp32" or "bf16": storage and transfer type
    n_req: int              # R
    n_layers: int           # nL decoder layers
    d_model: int            # d
    n_heads: int            # H (d_h = d / H)
    d_ff: int               # F
    L: SizeSpec             # behavior length per request
    M: SizeSpec             # candidates per request
    seed: int
    n_ctx: int = 2          # S shared serving-context tokens per request
    n_actions: int = 4      # k action tokens
    l_local: int = 10       # L_local (Sec. 5.1)
    ln_eps: float = 1e-5
    dL: SizeSpec = 0        # appended behavior rows per request
    capacity_extra: int = 64
    n_kv_heads: int = 0     # K/V heads of the cache (0: one per query head)
    cand_mlp: int = 0       # hidden width of the candidate-to-query MLP (0: none)
    dw_hidden: int = 0      # Deep & Wide head: deep FFN hidden width (0: linear head)
    dw_in: int = 0          # Deep & Wide head: width of the wide features x[:, :dw_in]
    dw_out: int = 0         # Deep & Wide head: width of the wide part of k_dec

    @property
    def d_head(self) -> int:
        return self.d_model // self.n_heads


# The five workloads: shapes of the paper's serving setting at growing scale.
WORKLOADS: Dict[str, Workload] = {
    "tiny_fp32": Workload("tiny_fp32", "fp32", 1, 1, 64, 2, 256, 64, 16, 20261, dL=4),
    "small_bf16": Workload("small_bf16", "bf16", 32, 2, 256, 8, 1024, 1024, 256, 20262, dL=8),
    "mid_bf16": Workload("mid_bf16", "bf16", 64, 4, 512, 8, 2048, 4096, 512, 20263, dL=8),
    "ragged_bf16": Workload("ragged_bf16", "bf16", 64, 4, 512, 8, 2048,
                            ("uniform", 1024, 16384), 1000, 20264, dL=8),
    "sweep_bf16": Workload("sweep_bf16", "bf16", 16, 4, 512, 8, 2048, 8192, 1024, 20265,
                           dL=("uniform", 1, 64)),
}


def _streams(seed: int):
    ss = np.random.SeedSequence(seed)
    s_sizes, s_weights, s_data = ss.spawn(3)
    return s_sizes, s_weights, s_data


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even), as float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = (r & 0xFFFFFFFF).astype(np.uint32).view(np.float32)
    nan = np.isnan(x)
    if nan.any():
        out = out.copy()
        out[nan] = np.float32("nan")
    return out


def _store(wl: Workload, x: np.ndarray) -> np.ndarray:
    x = np.asarray(x, dtype=np.float32)
    return round_bf16(x) if wl.dtype == "bf16" else x


def _draw_sizes(spec: SizeSpec, n: int, rng: np.random.Generator) -> np.ndarray:
    if isinstance(spec, (int, np.integer)):
        return np.full(n, int(spec), dtype=np.int64)
    if isinstance(spec, tuple) and len(spec) == 3 and spec[0] == "uniform":
        lo, hi = int(spec[1]), int(spec[2])
        return rng.integers(lo, hi + 1, size=n).astype(np.int64)  # inclusive bounds
    arr = np.asarray(spec, dtype=np.int64)
    if arr.shape != (n,):
        raise ValueError(f"size list has shape {arr.shape}, expected ({n},)")
    return arr


def sizes(wl: Workload) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Per-request (L_r, M_r, dL_r), drawn from the size stream in that order."""
    s_sizes, _, _ = _streams(wl.seed)
    rng = np.random.default_rng(s_sizes)
    L = _draw_sizes(wl.L, wl.n_req, rng)
    M = _draw_sizes(wl.M, wl.n_req, rng)
    dL = _draw_sizes(wl.dL, wl.n_req, rng)
    return L, M, dL


def _shape(code: str, wl: Workload) -> Tuple[int, ...]:
    dkv = (wl.n_kv_heads or wl.n_heads) * (wl.d_model // wl.n_heads)
    env = {"d": wl.d_model, "3d": 3 * wl.d_model, "2d": 2 * wl.d_model,
           "F": wl.d_ff, "k": wl.n_actions, "dkv": dkv, "Fc": wl.cand_mlp,
           "dwi": wl.dw_in, "dwo": wl.dw_out, "dd": 2 * wl.d_model - wl.dw_in, "Fh": wl.dw_hidden,
           "ddo": wl.d_model - wl.dw_out}
    return tuple(env[c] for c in code.split(","))


def weights(wl: Workload) -> Dict[str, np.ndarray]:
    """All model weights.  Per-layer names get the suffix ``.<l>``."""
    _, s_weights, _ = _streams(wl.seed)
    rng = np.random.default_rng(s_weights)
    out: Dict[str, np.ndarray] = {}
    for l in range(wl.n_layers):
        for name, code in LAYER_WEIGHTS:
            shp = _shape(code, wl)
            x = rng.standard_normal(shp) * 0.02
            if name.endswith("_g"):
                x = 1.0 + x
            out[f"{name}.{l}"] = _store(wl, x)
    for name, code in HEAD_WEIGHTS:
        out[name] = _store(wl, rng.standard_normal(_shape(code, wl)) * 0.02)
    if wl.cand_mlp:
        for name, code in CAND_WEIGHTS:
            out[name] = _store(wl, rng.standard_normal(_shape(code, wl)) * 0.02)
    if wl.dw_hidden:
        for name, code in DW_WEIGHTS:
            out[name] = _store(wl, rng.standard_normal(_shape(code, wl)) * 0.02)
    return out


def sharp_gains(wl: Workload) -> Dict[str, float]:
    """Power-of-two gains of ``sharp_weights`` for this workload's width.

    ``att``  on the query and key projections of both attentions (scores of
             standard deviation ~1.6 at d = 256, ~3.3 at d = 512, so the
             softmax over the keys is far from uniform);
    ``oc``   on the cross-attention output projection (the attended values
             move the residual stream);
    ``head`` on W_dec (logits of standard deviation ~0.3; with N(0, 0.02)
             weights it is about 0.0004 * sqrt(2) * d; larger logits make
             the bf16 rounding of the activations through four decoder
             layers exceed the mean tolerance of 2e-3 on their own);
    ``pool`` on w_pool (pooling logits of standard deviation ~2.6, so the
             anchor is a weighted mix of a few rows, not the mean).
    """
    d = wl.d_model
    head = 2.0 ** max(0, int(round(np.log2(0.3 / (0.0004 * np.sqrt(2.0) * d)))))
    return {"att": 4.0, "oc": 4.0, "head": head, "pool": 128.0}


def sharp_weights(wl: Workload, base: Optional[Dict[str, np.ndarray]] = None) -> Dict[str, np.ndarray]:
    """The workload's weights with the gains of ``sharp_gains`` applied.

    The gains are powers of two, so bf16-stored weights stay exactly
    representable and both sides of a parity test still see identical
    values.  With the plain N(0, 0.02) draws every attention softmax is
    nearly uniform and logits have a standard deviation of ~0.14, which hides
    errors in which keys an attention reads; these weights make such errors
    move the scores by far more than the bf16 tolerances.
    """
    w = dict(weights(wl) if base is None else base)
    gn = sharp_gains(wl)
    d = wl.d_model
    for l in range(wl.n_layers):
        qkv = np.array(w[f"W_qkv.{l}"], dtype=np.float32, copy=True)
        qkv[:, :2 * d] *= gn["att"]
        w[f"W_qkv.{l}"] = qkv
        w[f"W_Q.{l}"] = np.asarray(w[f"W_Q.{l}"], np.float32) * np.float32(gn["att"])
        w[f"W_K.{l}"] = np.asarray(w[f"W_K.{l}"], np.float32) * np.float32(gn["att"])
        w[f"W_oc.{l}"] = np.asarray(w[f"W_oc.{l}"], np.float32) * np.float32(gn["oc"])
    w["W_dec"] = np.asarray(w["W_dec"], np.float32) * np.float32(gn["head"])
    w["w_pool"] = np.asarray(w["w_pool"], np.float32) * np.float32(gn["pool"])
    return w


@dataclass
class Batch:
    """One synthetic serving batch, packed request after request.

    ``beh``  [sum L_r, d]  encoded behavior rows Phi_b (Sec. 4.1.2)
    ``ctx``  [R, S, d]     serving-context tokens (App. B)
    ``cand`` [sum M_r, d]  candidate tokens Phi_c rows (Sec. 4.1.2)
    ``app``  [sum dL_r, d] behavior rows appended after the cache build (App. D)
    Offsets are exclusive prefix sums with a leading 0.
    """
    beh: np.ndarray
    beh_off: np.ndarray
    ctx: np.ndarray
    cand: np.ndarray
    cand_off: np.ndarray
    app: np.ndarray
    app_off: np.ndarray
    L: np.ndarray
    M: np.ndarray
    dL: np.ndarray
    requests: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int64))


def _offsets(n: np.ndarray) -> np.ndarray:
    off = np.zeros(len(n) + 1, dtype=np.int32)
    off[1:] = np.cumsum(n)
    return off


def batch(wl: Workload, requests: Optional[Sequence[int]] = None,
          M_override: Optional[int] = None) -> Batch:
    """Draw the batch, or only the listed ``requests`` (same values as in the full batch).

    Per request ``r`` the draw order is: Phi_b rows, context rows, candidate
    rows, appended rows.  ``M_override`` replaces every M_r (used by the
    candidate-count sweep; the drawn values then differ from the default M).
    """
    Ls, Ms, dLs = sizes(wl)
    if M_override is not None:
        Ms = np.full_like(Ms, int(M_override))
    reqs = np.arange(wl.n_req) if requests is None else np.asarray(requests, dtype=np.int64)
    _, _, s_data = _streams(wl.seed)
    children = s_data.spawn(wl.n_req)
    d, S = wl.d_model, wl.n_ctx
    beh, ctx, cand, app = [], [], [], []
    for r in reqs:
        rng = np.random.default_rng(children[int(r)])
        beh.append(rng.standard_normal((int(Ls[r]), d), dtype=np.float32))
        ctx.append(rng.standard_normal((S, d), dtype=np.float32))
        cand.append(rng.standard_normal((int(Ms[r]), d), dtype=np.float32))
        app.append(rng.standard_normal((int(dLs[r]), d), dtype=np.float32))
    L, M, dL = Ls[reqs], Ms[reqs], dLs[reqs]
    cat = lambda xs: _store(wl, np.concatenate(xs, axis=0)) if xs else np.zeros((0, d), np.float32)
    return Batch(
        beh=cat(beh), beh_off=_offsets(L),
        ctx=_store(wl, np.stack(ctx, 0)) if ctx else np.zeros((0, S, d), np.float32),
        cand=cat(cand), cand_off=_offsets(M),
        app=cat(app), app_off=_offsets(dL),
        L=L, M=M, dL=dL, requests=reqs,
    )


@dataclass
class Events:
    """One user's behavior stream and T serving events (streaming form).

    ``beh``  [L, d]        encoded behavior rows Phi_b of the whole stream
    ``ends`` [T]           rows of the stream before each event (1 <= end <= L)
    ``ctx``  [T, S, d]     each event's context tokens
    ``cand`` [sum m_t, d]  each event's candidate tokens, packed by ``cand_off``
    """
    beh: np.ndarray
    ends: np.ndarray
    ctx: np.ndarray
    cand: np.ndarray
    cand_off: np.ndarray


def events(wl: Workload, L: int, T: int, m: Union[int, Sequence[int]], seed: int) -> Events:
    """Draw a stream of L rows and T events; event ends are uniform in
    [1, L] (sorted, the last one L), slates of m_t candidates."""
    rng = np.random.default_rng(seed)
    d, S = wl.d_model, wl.n_ctx
    beh = rng.standard_normal((L, d), dtype=np.float32)
    ends = np.sort(rng.integers(1, L + 1, size=T)).astype(np.int32)
    ends[-1] = L
    ms = np.full(T, int(m), dtype=np.int64) if np.isscalar(m) else np.asarray(m, dtype=np.int64)
    ctx = rng.standard_normal((T, S, d), dtype=np.float32)
    cand = rng.standard_normal((int(ms.sum()), d), dtype=np.float32)
    return Events(_store(wl, beh), ends, _store(wl, ctx), _store(wl, cand), _offsets(ms))


def with_sizes(wl: Workload, **kw) -> Workload:
    """A copy of ``wl`` with some fields replaced (e.g. a smaller L or M)."""
    return replace(wl, **kw)


# ---------------------------------------------------------------- behavior encoder

# Behavior-stream encoder Phi_behavior (Sec. 4.1.1; two causal layers with a
# relative position bias in Sec. 5.1).  Per encoder layer ``l``, in draw order:
ENC_LAYER_WEIGHTS: Tuple[Tuple[str, str], ...] = (
    ("W_qkv", "d,3d"), ("b_qkv", "3d"), ("rel_bias", "H,R"), ("W_o", "d,d"), ("b_o", "d"),
    ("ln1_g", "d"), ("ln1_b", "d"), ("W_1", "d,F"), ("b_1", "F"), ("W_2", "F,d"), ("b_2", "d"),
    ("ln2_g", "d"), ("ln2_b", "d"),
)
# then, when type_dim > 0, the behavior-type embedding table
ENC_TYPE_WEIGHTS: Tuple[Tuple[str, str], ...] = (("E_type", "T,dt"),)


@dataclass(frozen=True)
class EncWorkload:
    """Sizes of an encoder workload.  Each user has L_r earlier behavior tokens
    and dL_r new ones; a token is a subject row (width d - type_dim) and a
    behavior-type id in [0, n_types)."""
    name: str
    dtype: str
    n_req: int
    n_layers: int
    d_model: int
    n_heads: int
    d_ff: int
    L: SizeSpec
    dL: SizeSpec
    type_dim: int
    n_types: int
    n_rel: int              # R relative-bias entries per head
    window: int             # 0: full causal
    seed: int
    ln_eps: float = 1e-5
    capacity_extra: int = 64

    @property
    def subj_dim(self) -> int:
        return self.d_model - self.type_dim


ENC_WORKLOADS: Dict[str, EncWorkload] = {
    "enc_tiny_fp32": EncWorkload("enc_tiny_fp32", "fp32", 3, 2, 64, 2, 128, ("uniform", 20, 60),
                                 ("uniform", 0, 6), 16, 7, 16, 0, 30261),
    "enc_small_bf16": EncWorkload("enc_small_bf16", "bf16", 32, 2, 256, 8, 1024, 1024, 8, 32, 16, 256, 0, 30262),
    "enc_mid_bf16": EncWorkload("enc_mid_bf16", "bf16", 64, 2, 512, 8, 2048, 4096, 8, 64, 32, 512, 0, 30263),
}


def enc_weights(ew: EncWorkload) -> Dict[str, np.ndarray]:
    """Encoder weights: matrices ~ N(0, 1/d_in), biases ~ N(0, 0.02), LN gains
    1 + N(0, 0.02), relative-bias tables ~ N(0, 1), type table ~ N(0, 1)."""
    _, s_weights, _ = _streams(ew.seed)
    rng = np.random.default_rng(s_weights)
    env = {"d": ew.d_model, "3d": 3 * ew.d_model, "F": ew.d_ff, "H": ew.n_heads, "R": ew.n_rel,
           "T": ew.n_types, "dt": ew.type_dim}
    out: Dict[str, np.ndarray] = {}
    for l in range(ew.n_layers):
        for name, code in ENC_LAYER_WEIGHTS:
            shp = tuple(env[c] for c in code.split(","))
            x = rng.standard_normal(shp)
            if name.startswith("W_"):
                x = x / np.sqrt(shp[0])
            elif name == "rel_bias":
                pass
            else:
                x = x * 0.02
                if name.endswith("_g"):
                    x = 1.0 + x
            out[f"{name}.{l}"] = _store(ew, x)
    if ew.type_dim:
        out["E_type"] = _store(ew, rng.standard_normal((ew.n_types, ew.type_dim)))
    return out


@dataclass
class EncBatch:
    """Behavior tokens of all users, packed user after user.

    ``subj`` [sum L_r, d - d_t] subject embeddings, ``types`` [sum L_r] int32
    type ids; ``subj_app``/``types_app`` the dL_r new tokens of each user.
    """
    subj: np.ndarray
    types: np.ndarray
    off: np.ndarray
    subj_app: np.ndarray
    types_app: np.ndarray
    app_off: np.ndarray
    L: np.ndarray
    dL: np.ndarray


def enc_batch(ew: EncWorkload) -> EncBatch:
    """Per user r (own child stream): L_r subject rows ~ N(0, 1), L_r type ids
    uniform in [0, n_types), then the dL_r new tokens drawn the same way."""
    s_sizes, _, s_data = _streams(ew.seed)
    rng = np.random.default_rng(s_sizes)
    L = _draw_sizes(ew.L, ew.n_req, rng)
    dL = _draw_sizes(ew.dL, ew.n_req, rng)
    children = s_data.spawn(ew.n_req)
    ds, T = ew.subj_dim, max(ew.n_types, 1)
    subj, types, subj_a, types_a = [], [], [], []
    for r in range(ew.n_req):
        g = np.random.default_rng(children[r])
        subj.append(g.standard_normal((int(L[r]), ds), dtype=np.float32))
        types.append(g.integers(0, T, size=int(L[r])).astype(np.int32))
        subj_a.append(g.standard_normal((int(dL[r]), ds), dtype=np.float32))
        types_a.append(g.integers(0, T, size=int(dL[r])).astype(np.int32))
    cat = lambda xs: _store(ew, np.concatenate(xs, axis=0))
    return EncBatch(cat(subj), np.concatenate(types), _offsets(L), cat(subj_a), np.concatenate(types_a),
                    _offsets(dL), L, dL)
