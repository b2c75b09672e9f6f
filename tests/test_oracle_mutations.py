"""Planted mistakes in the oracle must be caught by the independent pins.

Each case patches one plausible slip into the oracle on the CPU (a dropped term,
a wrong scale, a wrong index set, a transposed or permuted operand, pre-LN for
post-LN) and checks that the PyTorch recompute of ``tests/test_oracle_pins.py``
then disagrees.  This shows the pins are sharp enough to see such errors.
"""
import math

import numpy as np
import pytest

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W
from tests.test_oracle_pins import torch_score


def _setup():
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_layers=2)
    model = O.Model.from_arrays(W.weights(wl), wl)
    model.w["w_pool"] = model.w["w_pool"] * 25.0   # make pooling non-uniform
    rng = np.random.default_rng(11)
    phi = rng.standard_normal((30, wl.d_model))
    ctx = rng.standard_normal((wl.n_ctx, wl.d_model))
    cand = rng.standard_normal((6, wl.d_model))
    return wl, model, phi, ctx, cand


def _gap(model, phi, ctx, cand, mode):
    cache = O.build_cache(model, phi)
    lg, pr = O.score_request(model, cache, ctx, cand, mode)
    rl, rp = torch_score(model, phi, ctx, cand, mode)
    return max(np.abs(lg - rl).max(), np.abs(pr - rp).max())


_orig_ln = O.layer_norm
_orig_attn = O.attention
_orig_gelu = O.gelu
_orig_key_set = O.key_set
_orig_head = O.head
_orig_pool_logits = O.pool_logits
_orig_project = O.project_kv


def _ln_no_eps(y, g, b, eps):
    return _orig_ln(y, g, b, 0.0)


def _ln_unbiased(y, g, b, eps):
    mu = y.mean(-1, keepdims=True)
    var = ((y - mu) ** 2).sum(-1, keepdims=True) / (y.shape[-1] - 1)
    return g * (y - mu) / np.sqrt(var + eps) + b


def _gelu_tanh(x):
    return 0.5 * x * (1 + np.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))


def _attn_scale_dh(q, k, v, n_heads, allowed=None, n_kv_heads=None):
    dh = q.shape[1] // n_heads
    return _orig_attn(q / math.sqrt(dh), k, v, n_heads, allowed, n_kv_heads)   # scale 1/d_h overall


def _attn_no_mask(q, k, v, n_heads, allowed=None, n_kv_heads=None):
    return _orig_attn(q, k, v, n_heads, None, n_kv_heads)


def _attn_heads_interleaved(q, k, v, n_heads, allowed=None, n_kv_heads=None):
    n, d = q.shape
    perm = np.arange(d).reshape(d // n_heads, n_heads).T.reshape(-1)
    out = _orig_attn(q[:, perm], k[:, perm], v[:, perm], n_heads, allowed, n_kv_heads)
    inv = np.argsort(perm)
    return out[:, inv]


def _key_set_short_window(model, cache, l, mode, use_global=True):
    K, V = _orig_key_set(model, cache, l, mode, use_global)
    return (K[1:], V[1:]) if mode == O.LOCAL_GLOBAL else (K, V)


def _key_set_no_anchor(model, cache, l, mode, use_global=True):
    return _orig_key_set(model, cache, l, mode, False)


def _key_set_kv_swapped(model, cache, l, mode, use_global=True):
    K, V = _orig_key_set(model, cache, l, mode, use_global)
    return V, K


def _head_q_permuted(model, z, x):
    w = dict(model.w)
    saved = model.w
    model.w = w
    w["Q_dec"] = saved["Q_dec"][::-1]
    try:
        return _orig_head(model, z, x)
    finally:
        model.w = saved


def _head_drop_x(model, z, x):
    return _orig_head(model, z, np.zeros_like(x))


def _pool_no_scale(model, phi):
    return phi @ model.w["w_pool"]


def _project_no_v_bias(model, phi, l):
    # (dropping b_K instead would be invisible: it adds q . b_K to every score of
    # a query row, and softmax is shift invariant; the cached K rows themselves
    # are compared element by element in the GPU parity tests)
    k, v = _orig_project(model, phi, l)
    return k, v - model.w[f"b_V.{l}"]


def _decoder_pre_ln(model, X, Kc, Vc, l, n_ctx):
    w, H, eps, d = model.w, model.n_heads, model.ln_eps, model.d_model
    ln = lambda y, i: _orig_ln(y, w[f"ln{i}_g.{l}"], w[f"ln{i}_b.{l}"], eps)
    h = ln(X, 1)
    qkv = h @ w[f"W_qkv.{l}"] + w[f"b_qkv.{l}"]
    a = _orig_attn(qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:], H, O.serving_mask(n_ctx, X.shape[0] - n_ctx))
    X = X + a @ w[f"W_os.{l}"] + w[f"b_os.{l}"]
    c = _orig_attn(ln(X, 2) @ w[f"W_Q.{l}"] + w[f"b_Q.{l}"], Kc, Vc, H)
    X = X + c @ w[f"W_oc.{l}"] + w[f"b_oc.{l}"]
    return X + _orig_gelu(ln(X, 3) @ w[f"W_1.{l}"] + w[f"b_1.{l}"]) @ w[f"W_2.{l}"] + w[f"b_2.{l}"]


MUTATIONS = {
    "pre_ln_block": ("decoder_layer", _decoder_pre_ln),
    "ln_no_eps": ("layer_norm", _ln_no_eps),
    "ln_unbiased_var": ("layer_norm", _ln_unbiased),
    "gelu_tanh": ("gelu", _gelu_tanh),
    "attn_scale_1_over_dh": ("attention", _attn_scale_dh),
    "serving_mask_dropped": ("attention", _attn_no_mask),
    "heads_interleaved": ("attention", _attn_heads_interleaved),
    "window_one_short": ("key_set", _key_set_short_window),
    "anchor_dropped": ("key_set", _key_set_no_anchor),
    "k_v_swapped": ("key_set", _key_set_kv_swapped),
    "q_dec_rows_permuted": ("head", _head_q_permuted),
    "head_drops_x": ("head", _head_drop_x),
    "pool_logit_unscaled": ("pool_logits", _pool_no_scale),
    "v_bias_dropped": ("project_kv", _project_no_v_bias),
}


def test_unmutated_oracle_agrees():
    wl, model, phi, ctx, cand = _setup()
    for mode in (O.LOCAL_GLOBAL, O.FULL):
        assert _gap(model, phi, ctx, cand, mode) < 1e-11


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, monkeypatch):
    attr, fn = MUTATIONS[name]
    wl, model, phi, ctx, cand = _setup()
    monkeypatch.setattr(O, attr, fn)
    gaps = [_gap(model, phi, ctx, cand, mode) for mode in (O.LOCAL_GLOBAL, O.FULL)]
    assert max(gaps) > 1e-9, f"mutation {name} went unnoticed (gaps {gaps})"


# ---------------------------------------------------------------- streaming events

def _events_gap(model, ev, mode=O.LOCAL_GLOBAL):
    lg, _ = O.score_events(model, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, mode)
    gap = 0.0
    for t, e in enumerate(ev.ends):
        sl = slice(ev.cand_off[t], ev.cand_off[t + 1])
        rl, _ = torch_score(model, np.asarray(ev.beh[:e], np.float64), np.asarray(ev.ctx[t], np.float64),
                            np.asarray(ev.cand[sl], np.float64), mode)
        gap = max(gap, float(np.abs(lg[sl] - rl).max()))
    return gap


def test_event_mistakes_are_caught(monkeypatch):
    wl, model, _, _, _ = _setup()
    ev = W.events(wl, 30, 4, 3, 21)
    ev.ends[:3] = [4, 12, 19]
    assert _events_gap(model, ev) < 1e-10
    orig_build = O.build_cache

    # anchor pooled over the whole stream instead of the event's prefix
    def build_with_stream_anchor(m, phi):
        c = orig_build(m, phi)
        full = orig_build(m, ev.beh)
        return O.RequestCache(c.K, c.V, full.pool, full.Kg, full.Vg)
    monkeypatch.setattr(O, "build_cache", build_with_stream_anchor)
    assert _events_gap(model, ev) > 1e-4
    monkeypatch.setattr(O, "build_cache", orig_build)

    # window taken from the end of the stream instead of the event's prefix
    def build_with_stream_rows(m, phi):
        c = orig_build(m, ev.beh)
        return O.RequestCache(c.K, c.V, orig_build(m, phi).pool, orig_build(m, phi).Kg, orig_build(m, phi).Vg)
    monkeypatch.setattr(O, "build_cache", build_with_stream_rows)
    assert _events_gap(model, ev) > 1e-4
