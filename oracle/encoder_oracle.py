"""fp64 CPU oracle for the behavior-stream encoder Phi_behavior.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  It shares no code
with the CUDA library: the definitions below are written out plainly, in
float64, one user at a time, with NumPy matmuls as the only library primitive.

What it computes (row-vector convention ``y = x W + b``):

* Behavior token (Sec. 4.1.1): the concatenation of the subject embedding
  (given as input rows of width d - d_t) and the behavior-type embedding
  ``E_type[type]`` (width d_t).  Position does not enter the token; it enters
  the attention as a relative position bias (Sec. 4.1.1 item (iii) with the
  relative scheme of Dai et al.; Table "encoder ablation", rel pos bias).
* Encoder layer (Sec. 4.1.1: standard dot-product self-attention with a causal
  mask, FFN, residual connections and layer normalization), post-LN:
  ``H = LN1(X + MHA(X) W_o + b_o)``, ``Y = LN2(H + GELU(H W_1 + b_1) W_2 + b_2)``
  with ``[q | k | v] = X W_qkv + b_qkv``.  Query i attends to key j iff
  j <= i (causal) and, with a window w > 0, i - j < w.  Head h's logit is
  ``q_i . k_j / sqrt(d_h) + beta_h[min(i - j, R - 1)]``: a learned scalar per
  head and relative distance, distances of R - 1 and more sharing the last
  entry.
* Incremental encoding (App. D, incremental-encoding remark): because the
  mask is causal and the bias depends only on i - j, appending tokens leaves
  every earlier token's output unchanged, and a new token's layer-l output
  needs only the layer-l keys and values of the tokens before it.  The state
  kept per user is therefore each layer's K and V rows, as in the key-value
  caching of autoregressive Transformers.

Readings where the paper is silent (post-LN, exact-erf GELU as in the decoder,
the clipped scalar bias table, the optional window, d_t) are fixed by the
fields of ``EncModel``.
"""
from __future__ import annotations

from dataclasses import dataclass
from math import sqrt
from typing import Dict, List, Sequence, Tuple

import numpy as np
from scipy.special import erf


def layer_norm(y: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float) -> np.ndarray:
    """LN over the last axis with the biased variance."""
    mu = y.mean(axis=-1, keepdims=True)
    var = ((y - mu) ** 2).mean(axis=-1, keepdims=True)
    return gamma * (y - mu) / np.sqrt(var + eps) + beta


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact GELU, 0.5 x (1 + erf(x / sqrt(2)))."""
    return 0.5 * x * (1.0 + erf(x / sqrt(2.0)))


@dataclass
class EncModel:
    """Encoder weights as float64 arrays plus its hyper-parameters."""
    w: Dict[str, np.ndarray]
    n_layers: int
    d_model: int
    n_heads: int
    type_dim: int     # d_t, width of the behavior-type embedding
    n_rel: int        # R, entries of each head's relative-bias table
    window: int       # 0: every earlier token; w > 0: the w most recent (self included)
    ln_eps: float

    @staticmethod
    def from_arrays(weights: Dict[str, np.ndarray], ew) -> "EncModel":
        return EncModel({k: np.asarray(v, dtype=np.float64) for k, v in weights.items()},
                        ew.n_layers, ew.d_model, ew.n_heads, ew.type_dim, ew.n_rel, ew.window, ew.ln_eps)


def embed(model: EncModel, subj: np.ndarray, types: np.ndarray) -> np.ndarray:
    """Behavior tokens: [subject embedding, E_type[type]] (Sec. 4.1.1)."""
    subj = np.asarray(subj, dtype=np.float64)
    if model.type_dim == 0:
        return subj
    t = np.asarray(types, dtype=np.int64)
    if t.size and (t.min() < 0 or t.max() >= model.w["E_type"].shape[0]):
        raise IndexError("behavior type outside the type table")
    return np.concatenate([subj, model.w["E_type"][t]], axis=1)


def visible(pos_q: np.ndarray, pos_k: np.ndarray, window: int) -> np.ndarray:
    """[n_q, n_k] bool: key position j is visible to query position i."""
    diff = pos_q[:, None] - pos_k[None, :]
    ok = diff >= 0
    if window > 0:
        ok &= diff < window
    return ok


def rel_bias(beta: np.ndarray, pos_q: np.ndarray, pos_k: np.ndarray) -> np.ndarray:
    """[H, n_q, n_k]: beta[h, min(i - j, R - 1)] for i - j >= 0 (0 elsewhere;
    those pairs are masked anyway)."""
    R = beta.shape[1]
    diff = pos_q[:, None] - pos_k[None, :]
    idx = np.clip(diff, 0, R - 1)
    return beta[:, idx]


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, n_heads: int, beta: np.ndarray,
                     pos_q: np.ndarray, pos_k: np.ndarray, window: int) -> np.ndarray:
    """Multi-head attention with the causal (and window) mask and the relative
    position bias, heads concatenated.  q [n, d] at positions pos_q, k/v [m, d]
    at positions pos_k."""
    n, d = q.shape
    dh = d // n_heads
    allowed = visible(pos_q, pos_k, window)
    bias = rel_bias(beta, pos_q, pos_k)
    out = np.empty((n, d), dtype=np.float64)
    for h in range(n_heads):
        c = slice(h * dh, (h + 1) * dh)
        s = (q[:, c] @ k[:, c].T) / sqrt(dh) + bias[h]
        s = np.where(allowed, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        e = np.exp(s)
        out[:, c] = (e / e.sum(axis=1, keepdims=True)) @ v[:, c]
    return out


@dataclass
class EncState:
    """Per-user encoder state: each layer's K and V rows of all tokens so far."""
    K: List[np.ndarray]
    V: List[np.ndarray]

    @property
    def length(self) -> int:
        return self.K[0].shape[0]


def encoder_layer(model: EncModel, X: np.ndarray, l: int, K_prev: np.ndarray, V_prev: np.ndarray
                  ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Layer l for the tokens X (positions len(K_prev) ...), attending to the
    earlier tokens' keys/values K_prev/V_prev and to each other causally.
    Returns (layer output, K rows of X, V rows of X)."""
    w, d = model.w, model.d_model
    n0 = K_prev.shape[0]
    qkv = X @ w[f"W_qkv.{l}"] + w[f"b_qkv.{l}"]
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    K = np.concatenate([K_prev, k], axis=0)
    V = np.concatenate([V_prev, v], axis=0)
    pos_q = np.arange(n0, n0 + X.shape[0])
    pos_k = np.arange(K.shape[0])
    a = causal_attention(q, K, V, model.n_heads, w[f"rel_bias.{l}"], pos_q, pos_k, model.window)
    Hh = layer_norm(X + a @ w[f"W_o.{l}"] + w[f"b_o.{l}"], w[f"ln1_g.{l}"], w[f"ln1_b.{l}"], model.ln_eps)
    f = gelu(Hh @ w[f"W_1.{l}"] + w[f"b_1.{l}"]) @ w[f"W_2.{l}"] + w[f"b_2.{l}"]
    Y = layer_norm(Hh + f, w[f"ln2_g.{l}"], w[f"ln2_b.{l}"], model.ln_eps)
    return Y, k, v


def empty_state(model: EncModel) -> EncState:
    z = np.zeros((0, model.d_model))
    return EncState([z] * model.n_layers, [z] * model.n_layers)


def encode_append(model: EncModel, state: EncState, subj: np.ndarray, types: np.ndarray
                  ) -> Tuple[np.ndarray, EncState]:
    """Encode new tokens of one user after the ones in ``state`` (App. D
    incremental encoding): returns (Phi_b rows of the new tokens, new state).
    No new tokens leave the state as it is."""
    X = embed(model, subj, types)
    if X.shape[0] == 0:
        return np.zeros((0, model.d_model)), state
    K, V = [], []
    for l in range(model.n_layers):
        X, k, v = encoder_layer(model, X, l, state.K[l], state.V[l])
        K.append(np.concatenate([state.K[l], k], axis=0))
        V.append(np.concatenate([state.V[l], v], axis=0))
    return X, EncState(K, V)


def encode(model: EncModel, subj: np.ndarray, types: np.ndarray) -> Tuple[np.ndarray, EncState]:
    """Encode a user's whole behavior stream at once: (Phi_b [L, d], state)."""
    return encode_append(model, empty_state(model), subj, types)


def encode_batch(model: EncModel, subj: np.ndarray, types: np.ndarray, off: Sequence[int]):
    """Per-user encode of packed streams: (concatenated Phi_b, list of states)."""
    outs, states = [], []
    for r in range(len(off) - 1):
        y, st = encode(model, subj[off[r]:off[r + 1]], types[off[r]:off[r + 1]])
        outs.append(y)
        states.append(st)
    return np.concatenate(outs, axis=0), states


def append_batch(model: EncModel, states: List[EncState], subj: np.ndarray, types: np.ndarray,
                 off: Sequence[int]):
    """Per-user incremental encode of packed new tokens."""
    outs, new = [], []
    for r, st in enumerate(states):
        y, s2 = encode_append(model, st, subj[off[r]:off[r + 1]], types[off[r]:off[r + 1]])
        outs.append(y)
        new.append(s2)
    return np.concatenate(outs, axis=0), new
