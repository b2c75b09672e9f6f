"""Planted mistakes in the encoder oracle must be caught by its pins.

Each case patches one plausible slip into ``oracle.encoder_oracle`` on the CPU
(the bias indexed by the wrong distance, an unclipped or absolute index, an
off-by-one in the causal or window mask, pre-LN for post-LN, the wrong score
scale, the token halves swapped) and checks that the PyTorch recompute of
``tests/test_oracle_encoder.py`` or the closed form there then disagrees.
"""
import numpy as np
import pytest

from oracle import encoder_oracle as E
from tests.test_oracle_encoder import _bias_only, _model, _tokens, torch_encode

_orig_rel = E.rel_bias
_orig_vis = E.visible
_orig_attn = E.causal_attention
_orig_layer = E.encoder_layer
_orig_embed = E.embed


def _rel_reversed(beta, pos_q, pos_k):
    R = beta.shape[1]
    return beta[:, np.clip(pos_k[None, :] - pos_q[:, None], 0, R - 1)]


def _rel_absolute(beta, pos_q, pos_k):
    R = beta.shape[1]
    return beta[:, np.clip(np.broadcast_to(pos_k[None, :], (len(pos_q), len(pos_k))), 0, R - 1)]


def _rel_wrap(beta, pos_q, pos_k):
    R = beta.shape[1]
    return beta[:, (pos_q[:, None] - pos_k[None, :]) % R]


def _rel_off_by_one(beta, pos_q, pos_k):
    R = beta.shape[1]
    return beta[:, np.clip(pos_q[:, None] - pos_k[None, :] - 1, 0, R - 1)]


def _vis_strict(pos_q, pos_k, window):
    ok = _orig_vis(pos_q, pos_k, window)
    return ok & (pos_q[:, None] != pos_k[None, :])


def _vis_window_wide(pos_q, pos_k, window):
    return _orig_vis(pos_q, pos_k, window + 1 if window > 0 else 0)


def _attn_scale_dh(q, k, v, n_heads, beta, pos_q, pos_k, window):
    dh = q.shape[1] // n_heads
    return _orig_attn(q / np.sqrt(dh), k, v, n_heads, beta, pos_q, pos_k, window)


def _layer_pre_ln(model, X, l, K_prev, V_prev):
    w, d = model.w, model.d_model
    n0 = K_prev.shape[0]
    Xn = E.layer_norm(X, w[f"ln1_g.{l}"], w[f"ln1_b.{l}"], model.ln_eps)
    qkv = Xn @ w[f"W_qkv.{l}"] + w[f"b_qkv.{l}"]
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    K = np.concatenate([K_prev, k])
    V = np.concatenate([V_prev, v])
    a = E.causal_attention(q, K, V, model.n_heads, w[f"rel_bias.{l}"], np.arange(n0, n0 + len(X)),
                           np.arange(len(K)), model.window)
    Hh = X + a @ w[f"W_o.{l}"] + w[f"b_o.{l}"]
    Hn = E.layer_norm(Hh, w[f"ln2_g.{l}"], w[f"ln2_b.{l}"], model.ln_eps)
    return Hh + E.gelu(Hn @ w[f"W_1.{l}"] + w[f"b_1.{l}"]) @ w[f"W_2.{l}"] + w[f"b_2.{l}"], k, v


def _embed_swapped(model, subj, types):
    X = _orig_embed(model, subj, types)
    ds = X.shape[1] - model.type_dim
    return np.concatenate([X[:, ds:], X[:, :ds]], axis=1)


MUTANTS = {
    "rel_reversed": ("rel_bias", _rel_reversed),
    "rel_absolute": ("rel_bias", _rel_absolute),
    "rel_wrap": ("rel_bias", _rel_wrap),
    "rel_off_by_one": ("rel_bias", _rel_off_by_one),
    "mask_strict": ("visible", _vis_strict),
    "window_wide": ("visible", _vis_window_wide),
    "scale_dh": ("causal_attention", _attn_scale_dh),
    "pre_ln": ("encoder_layer", _layer_pre_ln),
    "embed_swapped": ("embed", _embed_swapped),
}


def _caught(window, n_rel):
    """Largest gap between the (patched) oracle and the torch recompute, plus
    whether the closed-form bias weights still hold."""
    ew, model = _model(window=window, n_rel=n_rel)
    subj, types = _tokens(ew, 21, 9)
    phi, _ = E.encode(model, subj, types)
    # the torch pin builds its tokens by plain concatenation, not via the oracle
    X = np.concatenate([subj, model.w["E_type"][types]], axis=1)
    gap = np.abs(phi - torch_encode(model, X)).max()
    beta = np.log(np.array([[1.0, 2.0, 4.0]]))
    try:
        A = _bias_only(beta, 4)
        closed = np.allclose(A[3], [4 / 11, 4 / 11, 2 / 11, 1 / 11], atol=1e-12) and \
            np.allclose(A[2], [4 / 7, 2 / 7, 1 / 7, 0], atol=1e-12)
    except Exception:
        closed = False
    return gap, closed


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_caught(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(E, attr, fn)
    caught = False
    for window, n_rel in [(0, 16), (5, 4)]:
        gap, closed = _caught(window, n_rel)
        caught |= gap > 1e-6 or not closed
    assert caught, name


def test_unpatched_passes():
    for window, n_rel in [(0, 16), (5, 4)]:
        gap, closed = _caught(window, n_rel)
        assert gap < 1e-10 and closed
