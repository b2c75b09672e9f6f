"""fp64 CPU oracle for the TransX serving path.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  It shares no code with
the CUDA library: it is the paper's definitions written out plainly, in float64,
one request at a time, with NumPy matmuls as the only library primitive.

What it computes (row-vector convention ``y = x W + b``):

* Cache build (Sec. 4.1.2, the Q/K/V projection equation; Sec. 4.3 "KV
  caching"): for every layer l, ``K_l = Phi_b W_K^l + b_K^l`` and
  ``V_l = Phi_b W_V^l + b_V^l`` over all behavior rows of the request.
* Global anchor token (Sec. 4.1.2, local-global sparse set; Sec. 5.1 "attention
  pooling ... global token"): ``alpha = softmax(Phi_b w_pool / sqrt(d))``,
  ``g = alpha^T Phi_b``, projected by each layer's ``W_K``/``W_V``.  The pooling
  state (running max m, running sum s, weighted sum acc) is kept so that an
  incremental append (App. D, incremental-encoding remark) can merge new rows.
* Grouped K/V heads (the MQA/GQA variants Sec. 4.1.2 cites): the cache may
  hold n_kv_heads < n_heads key/value heads (W_K, W_V of width n_kv_heads *
  d_h); query head h attends with key/value head h // (n_heads / n_kv_heads).
* Key set I_t (Sec. 4.1.2): LOCAL_GLOBAL uses the most recent L_local rows plus
  the global token; FULL ("-sparseAttn", Sec. 5.2) uses all rows and no global
  token.
* Decoder layer (Sec. 4.1.2 crossAttend equation, App. B serving-stream mask):
  rows X = [context tokens; candidate tokens];
  X1 = LN(X + MHA_serving(X)), each context row attending to the context rows
  and each candidate row attending to the context rows and itself;
  X2 = LN(X1 + MHA(X1 W_Q + b_Q, K_I, V_I)) (the sparse cross-attention
  equation, scale 1/sqrt(d_h));
  X3 = LN(X2 + GELU(X2 W_1 + b_1) W_2 + b_2).
* Candidate encoder (Sec. 4.1.2, Phi_candidate "a multi-layer perceptron"):
  optional, GELU(x W_c1 + b_c1) W_c2 + b_c2 on each candidate token before
  the decoder; the head still takes the raw token x.
* Head (Sec. 4.1.3, the action-decoding equation): for candidate rows,
  ``k_dec = [z, x] W_dec + b_dec`` (linear f_dec, Sec. 4.4), logits
  ``= Q_dec k_dec`` (no scale), probabilities ``= softmax(logits)``.
  Optionally the Deep & Wide f_dec (App. B): with x = [x_wide, x_deep],
  ``k_dec = [x_wide W_w + b_w, GELU([z, x_deep] W_d1 + b_d1) W_d2 + b_d2]``.
* Ranking: per request, candidates by descending probability of one action,
  ties to the lower candidate index.
* Streaming multi-event scoring (Sec. 4.2 prefix reuse, Sec. 5.1 per-event
  global token): event t of a user is scored against the behavior prefix
  before it, exactly as a request whose history is that prefix.

Readings where the paper is silent (LN eps 1e-5 with biased variance, exact erf
GELU, k = 4 actions, S = 2 context tokens, the serving-stream mask) are listed
in the design notes and fixed by the workload fields passed in.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from math import sqrt
from typing import Dict, List, Optional, Sequence

import numpy as np
from scipy.special import erf

LOCAL_GLOBAL = 0
FULL = 1


# ---------------------------------------------------------------- primitives

def layer_norm(y: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float) -> np.ndarray:
    """LN over the last axis: gamma * (y - mean) / sqrt(biased var + eps) + beta."""
    mu = y.mean(axis=-1, keepdims=True)
    var = ((y - mu) ** 2).mean(axis=-1, keepdims=True)
    return gamma * (y - mu) / np.sqrt(var + eps) + beta


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact GELU, 0.5 x (1 + erf(x / sqrt(2)))."""
    return 0.5 * x * (1.0 + erf(x / sqrt(2.0)))


def softmax(z: np.ndarray, axis: int = -1) -> np.ndarray:
    z = z - z.max(axis=axis, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=axis, keepdims=True)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, n_heads: int,
              allowed: Optional[np.ndarray] = None, n_kv_heads: Optional[int] = None) -> np.ndarray:
    """Multi-head scaled dot-product attention, heads concatenated.

    q [n, d], k/v [m, n_kv_heads * d_h]; query head h uses columns
    h*d_h ... (h+1)*d_h - 1 of q and key/value head h // (n_heads / n_kv_heads)
    (grouped-query sharing of K/V heads, the MQA/GQA variants Sec. 4.1.2
    cites; n_kv_heads = n_heads is plain multi-head attention).
    ``allowed`` [n, m] bool restricts the keys of each query row
    (Sec. 4.1.2 sparse cross-attention equation; App. B mask).
    """
    n, d = q.shape
    dh = d // n_heads
    n_kv = n_heads if n_kv_heads is None else n_kv_heads
    group = n_heads // n_kv
    out = np.empty((n, d), dtype=np.float64)
    for h in range(n_heads):
        c = slice(h * dh, (h + 1) * dh)
        g = h // group
        ck = slice(g * dh, (g + 1) * dh)
        s = (q[:, c] @ k[:, ck].T) / sqrt(dh)
        if allowed is not None:
            s = np.where(allowed, s, -np.inf)
        out[:, c] = softmax(s, axis=-1) @ v[:, ck]
    return out


# ---------------------------------------------------------------- model

@dataclass
class Model:
    """Weights as float64 arrays plus the hyper-parameters the path needs."""
    w: Dict[str, np.ndarray]
    n_layers: int
    d_model: int
    n_heads: int
    n_ctx: int
    n_actions: int
    l_local: int
    ln_eps: float
    n_kv_heads: int = 0   # K/V heads of the cache; 0 or n_heads: one per query head
    cand_mlp: int = 0     # hidden width of the candidate-to-query MLP; 0: none
    dw_hidden: int = 0    # Deep & Wide head: hidden width of the deep FFN; 0: linear head
    dw_in: int = 0        # width of x_wide (the first dw_in features of x)
    dw_out: int = 0       # width of the wide part of k_dec

    @property
    def kv_heads(self) -> int:
        return self.n_kv_heads or self.n_heads

    @staticmethod
    def from_arrays(weights: Dict[str, np.ndarray], wl) -> "Model":
        return Model({k: np.asarray(v, dtype=np.float64) for k, v in weights.items()},
                     wl.n_layers, wl.d_model, wl.n_heads, wl.n_ctx, wl.n_actions,
                     wl.l_local, wl.ln_eps, getattr(wl, "n_kv_heads", 0), getattr(wl, "cand_mlp", 0),
                     getattr(wl, "dw_hidden", 0), getattr(wl, "dw_in", 0), getattr(wl, "dw_out", 0))


@dataclass
class PoolState:
    """Online-softmax attention-pooling state over behavior rows seen so far."""
    m: float          # max pooling logit
    s: float          # sum of exp(logit - m)
    acc: np.ndarray   # sum of exp(logit - m) * phi, [d]

    @property
    def g(self) -> np.ndarray:
        return self.acc / self.s


@dataclass
class RequestCache:
    """Per-request cache: per-layer K/V of every behavior row and the global token."""
    K: List[np.ndarray]
    V: List[np.ndarray]
    pool: PoolState
    Kg: List[np.ndarray]
    Vg: List[np.ndarray]

    @property
    def length(self) -> int:
        return self.K[0].shape[0]


def pool_logits(model: Model, phi: np.ndarray) -> np.ndarray:
    """Pooling logits phi_i . w_pool / sqrt(d) (attention pooling, Sec. 5.1)."""
    return phi @ model.w["w_pool"] / sqrt(model.d_model)


def pool_direct(model: Model, phi: np.ndarray) -> PoolState:
    """Attention pooling over all rows at once: alpha = softmax(logits), g = alpha^T phi."""
    z = pool_logits(model, phi)
    m = float(z.max())
    e = np.exp(z - m)
    return PoolState(m, float(e.sum()), e @ phi)


def pool_merge(a: PoolState, b: PoolState) -> PoolState:
    """Merge two pooling states over disjoint row sets (incremental update, App. D)."""
    m = max(a.m, b.m)
    ea, eb = np.exp(a.m - m), np.exp(b.m - m)
    return PoolState(m, a.s * ea + b.s * eb, a.acc * ea + b.acc * eb)


def project_kv(model: Model, phi: np.ndarray, l: int):
    """K = phi W_K + b_K, V = phi W_V + b_V for layer l (Sec. 4.1.2)."""
    w = model.w
    return phi @ w[f"W_K.{l}"] + w[f"b_K.{l}"], phi @ w[f"W_V.{l}"] + w[f"b_V.{l}"]


def _global_kv(model: Model, pool: PoolState):
    Kg, Vg = [], []
    for l in range(model.n_layers):
        k, v = project_kv(model, pool.g[None, :], l)
        Kg.append(k[0])
        Vg.append(v[0])
    return Kg, Vg


def build_cache(model: Model, phi: np.ndarray) -> RequestCache:
    """Nearline cache build for one request (Sec. 4.3 amortised encoding + KV caching)."""
    phi = np.asarray(phi, dtype=np.float64)
    if phi.shape[0] == 0:
        raise ValueError("cold start: no behavior rows (App. D falls back to another model)")
    K, V = zip(*(project_kv(model, phi, l) for l in range(model.n_layers)))
    pool = pool_direct(model, phi)
    Kg, Vg = _global_kv(model, pool)
    return RequestCache(list(K), list(V), pool, Kg, Vg)


def append_cache(model: Model, cache: RequestCache, phi_new: np.ndarray) -> RequestCache:
    """Incremental update (App. D remark): project only the new rows, merge the pool.

    Old rows' K/V are left as they are; the global token is re-projected from the
    merged pooling state.
    """
    phi_new = np.asarray(phi_new, dtype=np.float64)
    if phi_new.shape[0] == 0:
        return cache
    K, V = [], []
    for l in range(model.n_layers):
        k, v = project_kv(model, phi_new, l)
        K.append(np.concatenate([cache.K[l], k], axis=0))
        V.append(np.concatenate([cache.V[l], v], axis=0))
    pool = pool_merge(cache.pool, pool_direct(model, phi_new))
    Kg, Vg = _global_kv(model, pool)
    return RequestCache(K, V, pool, Kg, Vg)


def key_set(model: Model, cache: RequestCache, l: int, mode: int, use_global: bool = True):
    """Keys/values of I_t for layer l (Sec. 4.1.2 local-global sparse set)."""
    if mode == FULL:
        return cache.K[l], cache.V[l]
    L = cache.length
    lo = max(0, L - model.l_local)
    K, V = cache.K[l][lo:], cache.V[l][lo:]
    if use_global:
        K = np.concatenate([K, cache.Kg[l][None, :]], axis=0)
        V = np.concatenate([V, cache.Vg[l][None, :]], axis=0)
    return K, V


def serving_mask(n_ctx: int, n_cand: int) -> np.ndarray:
    """App. B mask over rows [ctx; cand]: context rows see context rows; a candidate
    sees the context rows and itself, never another candidate."""
    n = n_ctx + n_cand
    allowed = np.zeros((n, n), dtype=bool)
    allowed[:, :n_ctx] = True
    allowed[np.arange(n_ctx, n), np.arange(n_ctx, n)] = True
    return allowed


def decoder_layer(model: Model, X: np.ndarray, Kc: np.ndarray, Vc: np.ndarray, l: int,
                  n_ctx: int) -> np.ndarray:
    """One decoder block: serving attention, cross-attention, FFN, each post-LN
    with a residual (Sec. 4.1.2 crossAttend equation; App. B mask)."""
    w, H, eps = model.w, model.n_heads, model.ln_eps
    d = model.d_model
    # serving-stream attention
    qkv = X @ w[f"W_qkv.{l}"] + w[f"b_qkv.{l}"]
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    a = attention(q, k, v, H, serving_mask(n_ctx, X.shape[0] - n_ctx))
    X1 = layer_norm(X + a @ w[f"W_os.{l}"] + w[f"b_os.{l}"], w[f"ln1_g.{l}"], w[f"ln1_b.{l}"], eps)
    # multi-query cross-attention against the shared K/V of this request
    qc = X1 @ w[f"W_Q.{l}"] + w[f"b_Q.{l}"]
    c = attention(qc, Kc, Vc, H, n_kv_heads=model.kv_heads)
    X2 = layer_norm(X1 + c @ w[f"W_oc.{l}"] + w[f"b_oc.{l}"], w[f"ln2_g.{l}"], w[f"ln2_b.{l}"], eps)
    # FFN
    f = gelu(X2 @ w[f"W_1.{l}"] + w[f"b_1.{l}"]) @ w[f"W_2.{l}"] + w[f"b_2.{l}"]
    return layer_norm(X2 + f, w[f"ln3_g.{l}"], w[f"ln3_b.{l}"], eps)


def f_dec_deep_wide(model: Model, z: np.ndarray, x: np.ndarray) -> np.ndarray:
    """Deep & Wide f_dec (App. B): the concatenation of a linear map of the
    wide features x[:, :dw_in] and an FFN of the cross-attention output z with
    the deep features x[:, dw_in:]."""
    w, a = model.w, model.dw_in
    wide = x[:, :a] @ w["W_w"] + w["b_w"]
    deep = gelu(np.concatenate([z, x[:, a:]], axis=1) @ w["W_d1"] + w["b_d1"]) @ w["W_d2"] + w["b_d2"]
    return np.concatenate([wide, deep], axis=1)


def head(model: Model, z: np.ndarray, x: np.ndarray):
    """Query-key softmax action decoder (Sec. 4.1.3): logits = Q_dec k_dec, with
    k_dec = f_dec(z, x) linear in [z, x], or the Deep & Wide f_dec."""
    w = model.w
    if model.dw_hidden:
        kdec = f_dec_deep_wide(model, z, x)
    else:
        kdec = np.concatenate([z, x], axis=1) @ w["W_dec"] + w["b_dec"]
    logits = kdec @ w["Q_dec"].T
    return logits, softmax(logits, axis=-1)


def candidate_encoder(model: Model, cand: np.ndarray) -> np.ndarray:
    """Phi_candidate (Sec. 4.1.2): with a candidate MLP, GELU(x W_c1 + b_c1) W_c2
    + b_c2 per candidate; without one the tokens are already its outputs."""
    if not model.cand_mlp:
        return cand
    w = model.w
    return gelu(cand @ w["W_c1"] + w["b_c1"]) @ w["W_c2"] + w["b_c2"]


def score_request(model: Model, cache: RequestCache, ctx: np.ndarray, cand: np.ndarray,
                  mode: int = LOCAL_GLOBAL, use_global: bool = True):
    """Scores of one request's candidates: (logits [M, k], probs [M, k]).  The
    decoder sees Phi_candidate(x); the head f_dec(z, x) the raw token x."""
    ctx = np.asarray(ctx, dtype=np.float64).reshape(-1, model.d_model)
    cand = np.asarray(cand, dtype=np.float64)
    S = ctx.shape[0]
    X = np.concatenate([ctx, candidate_encoder(model, cand)], axis=0)
    for l in range(model.n_layers):
        Kc, Vc = key_set(model, cache, l, mode, use_global)
        X = decoder_layer(model, X, Kc, Vc, l, S)
    return head(model, X[S:], cand)


# ---------------------------------------------------------------- batches

def build_caches(model: Model, beh: np.ndarray, beh_off: Sequence[int]) -> List[RequestCache]:
    return [build_cache(model, beh[beh_off[r]:beh_off[r + 1]]) for r in range(len(beh_off) - 1)]


def append_caches(model: Model, caches: List[RequestCache], app: np.ndarray,
                  app_off: Sequence[int]) -> List[RequestCache]:
    return [append_cache(model, c, app[app_off[r]:app_off[r + 1]]) for r, c in enumerate(caches)]


def score_batch(model: Model, caches: List[RequestCache], ctx: np.ndarray, cand: np.ndarray,
                cand_off: Sequence[int], mode: int = LOCAL_GLOBAL, use_global: bool = True):
    """Concatenated (logits, probs) over the packed candidates of all requests."""
    lg, pr = [], []
    for r, c in enumerate(caches):
        a, b = score_request(model, c, ctx[r], cand[cand_off[r]:cand_off[r + 1]], mode, use_global)
        lg.append(a)
        pr.append(b)
    return np.concatenate(lg, axis=0), np.concatenate(pr, axis=0)


# ---------------------------------------------------------------- streaming events

def score_events(model: Model, phi: np.ndarray, ends: Sequence[int], ctx: np.ndarray, cand: np.ndarray,
                 cand_off: Sequence[int], mode: int = LOCAL_GLOBAL, use_global: bool = True):
    """Multi-event scoring of one user in the streaming form (Sec. 4.2, causal
    attention and prefix reuse; Sec. 5.1, a global token for each event
    timestamp).  Event t sees only the behavior prefix ``phi[:ends[t]]``: its
    key set is the most recent L_local rows of that prefix plus the anchor
    pooled over that prefix (LOCAL_GLOBAL), or the whole prefix (FULL).  Its
    slate is ``cand[cand_off[t]:cand_off[t + 1]]`` with context rows
    ``ctx[t]``.  Written as the definition: one cache per event, built from
    the prefix alone.  Returns concatenated (logits, probs) over all events."""
    phi = np.asarray(phi, dtype=np.float64)
    lg, pr = [], []
    for t, e in enumerate(ends):
        e = int(e)
        if e <= 0:
            raise ValueError("cold start: an event with no behavior rows before it")
        if e > phi.shape[0]:
            raise ValueError("event end beyond the behavior stream")
        cache = build_cache(model, phi[:e])
        a, b = score_request(model, cache, ctx[t], cand[cand_off[t]:cand_off[t + 1]], mode, use_global)
        lg.append(a)
        pr.append(b)
    return np.concatenate(lg, axis=0), np.concatenate(pr, axis=0)


def rank(scores: np.ndarray, cand_off: Sequence[int], top_k: int = 0) -> List[np.ndarray]:
    """Per request: candidate indices (local to the request) by descending score,
    ties to the lower index, NaN scores after all numbers.  ``top_k > 0`` keeps
    the first top_k."""
    out = []
    for r in range(len(cand_off) - 1):
        s = np.asarray(scores[cand_off[r]:cand_off[r + 1]], dtype=np.float64)
        key = lambda i: (1, 0.0, i) if np.isnan(s[i]) else (0, -s[i], i)
        order = sorted(range(len(s)), key=key)
        order = np.asarray(order, dtype=np.int32)
        out.append(order[:top_k] if top_k > 0 else order)
    return out
