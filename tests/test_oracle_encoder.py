"""Pins of the behavior-encoder oracle (Sec. 4.1.1; App. D incremental encoding).

The oracle is checked against things fixed outside it:
* PyTorch's own post-LN ``TransformerEncoderLayer`` (exact GELU, no dropout),
  fed the causal mask and the relative bias as an additive float mask, in
  float64 (a library routine for the whole layer stack);
* closed forms of the attention weights when q . k = 0, where the weights are
  the softmax of the bias table alone;
* the incremental-encoding property the paper states (App. D remark): earlier
  outputs do not change when tokens are appended, and encoding new tokens
  against the cached K/V equals encoding the whole stream;
* invariants of a relative bias: a constant shift of a head's table changes
  nothing; with a window w a token's output depends only on the last
  n_layers * (w - 1) + 1 tokens, wherever they sit in the stream.
"""
import math

import numpy as np
import pytest

from oracle import encoder_oracle as E
from paper_2607_28940_gb300 import workload as W

torch = pytest.importorskip("torch")


def _model(window=0, n_rel=16, **kw):
    ew = W.with_sizes(W.ENC_WORKLOADS["enc_tiny_fp32"], window=window, n_rel=n_rel, **kw)
    return ew, E.EncModel.from_arrays(W.enc_weights(ew), ew)


def _tokens(ew, n, seed):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n, ew.subj_dim)), rng.integers(0, ew.n_types, size=n)


def torch_encode(model: E.EncModel, X: np.ndarray) -> np.ndarray:
    """The encoder stack recomputed by torch.nn.TransformerEncoderLayer."""
    n, d = X.shape
    H = model.n_heads
    w = model.w
    x = torch.tensor(X[None], dtype=torch.float64)
    for l in range(model.n_layers):
        F = w[f"W_1.{l}"].shape[1]
        layer = torch.nn.TransformerEncoderLayer(d, H, F, dropout=0.0, activation="gelu", batch_first=True,
                                                 norm_first=False, layer_norm_eps=model.ln_eps,
                                                 dtype=torch.float64)
        layer.train()  # keeps the generic (mask-honouring) path; dropout is 0
        t = lambda a: torch.tensor(a, dtype=torch.float64)
        with torch.no_grad():
            layer.self_attn.in_proj_weight.copy_(t(w[f"W_qkv.{l}"].T))
            layer.self_attn.in_proj_bias.copy_(t(w[f"b_qkv.{l}"]))
            layer.self_attn.out_proj.weight.copy_(t(w[f"W_o.{l}"].T))
            layer.self_attn.out_proj.bias.copy_(t(w[f"b_o.{l}"]))
            layer.linear1.weight.copy_(t(w[f"W_1.{l}"].T))
            layer.linear1.bias.copy_(t(w[f"b_1.{l}"]))
            layer.linear2.weight.copy_(t(w[f"W_2.{l}"].T))
            layer.linear2.bias.copy_(t(w[f"b_2.{l}"]))
            layer.norm1.weight.copy_(t(w[f"ln1_g.{l}"]))
            layer.norm1.bias.copy_(t(w[f"ln1_b.{l}"]))
            layer.norm2.weight.copy_(t(w[f"ln2_g.{l}"]))
            layer.norm2.bias.copy_(t(w[f"ln2_b.{l}"]))
        # additive mask [H, n, n]: beta_h[min(i - j, R - 1)] where visible, -inf elsewhere
        beta = w[f"rel_bias.{l}"]
        R = beta.shape[1]
        mask = np.full((H, n, n), -np.inf)
        for i in range(n):
            for j in range(n):
                if j <= i and (model.window == 0 or i - j < model.window):
                    mask[:, i, j] = beta[:, min(i - j, R - 1)]
        with torch.no_grad():
            x = layer(x, src_mask=torch.tensor(mask))
    return x[0].numpy()


@pytest.mark.parametrize("window,n_rel", [(0, 16), (0, 4), (5, 16), (1, 8)])
def test_matches_torch_encoder_layer(window, n_rel):
    ew, model = _model(window=window, n_rel=n_rel)
    subj, types = _tokens(ew, 23, 1)
    phi, _ = E.encode(model, subj, types)
    ref = torch_encode(model, E.embed(model, subj, types))
    assert np.abs(phi - ref).max() < 1e-10


def test_embed_is_concatenation():
    ew, model = _model()
    subj, types = _tokens(ew, 9, 2)
    X = E.embed(model, subj, types)
    assert X.shape == (9, ew.d_model)
    assert np.array_equal(X[:, :ew.subj_dim], subj)
    for i in range(9):
        assert np.array_equal(X[i, ew.subj_dim:], model.w["E_type"][types[i]])
    with pytest.raises(IndexError):
        E.embed(model, subj[:1], np.array([ew.n_types]))


def _bias_only(beta, n, window=0):
    """q = k = 0, v = one-hot of the position: row i of the output is row i of
    the attention-weight matrix."""
    H = beta.shape[0]
    dh = n
    q = np.zeros((n, H * dh))
    v = np.zeros((n, H * dh))
    for h in range(H):
        v[:, h * dh:(h + 1) * dh] = np.eye(n)
    pos = np.arange(n)
    return E.causal_attention(q, q, v, H, beta, pos, pos, window)


def test_bias_closed_form():
    beta = np.log(np.array([[1.0, 2.0, 4.0]]))        # distance 0, 1, >= 2
    A = _bias_only(beta, 4)
    assert np.allclose(A[0], [1, 0, 0, 0], atol=1e-15)
    assert np.allclose(A[1], [2 / 3, 1 / 3, 0, 0], atol=1e-15)       # distances 1, 0
    assert np.allclose(A[2], [4 / 7, 2 / 7, 1 / 7, 0], atol=1e-15)   # distances 2, 1, 0
    assert np.allclose(A[3], [4 / 11, 4 / 11, 2 / 11, 1 / 11], atol=1e-15)  # 3 clipped to 2
    Aw = _bias_only(beta, 4, window=2)
    assert np.allclose(Aw[3], [0, 0, 2 / 3, 1 / 3], atol=1e-15)
    # two heads with their own tables
    beta2 = np.log(np.array([[1.0, 2.0, 4.0], [1.0, 1.0, 1.0]]))
    A2 = _bias_only(beta2, 3)
    assert np.allclose(A2[2, 3:], [1 / 3, 1 / 3, 1 / 3], atol=1e-15)


def test_score_scale():
    # one key equal to the query: weight e^{|q|^2/sqrt(dh)} against a zero key
    dh = 4
    q = np.zeros((2, dh))
    q[1, 0] = 2.0
    k = np.zeros((2, dh))
    k[1, 0] = 2.0                                  # q1 . k1 = 4, scale 1/2 -> logit 2
    v = np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0]])
    out = E.causal_attention(q, k, v, 1, np.zeros((1, 1)), np.arange(2), np.arange(2), 0)
    p = math.exp(2.0) / (1 + math.exp(2.0))
    assert np.allclose(out[1, :2], [1 - p, p], atol=1e-15)


@pytest.mark.parametrize("cuts", [[23], [1, 22], [10, 13], [5, 1, 1, 16], [22, 1]])
def test_incremental_equals_full(cuts):
    ew, model = _model()
    subj, types = _tokens(ew, 23, 3)
    full, st_full = E.encode(model, subj, types)
    st = E.empty_state(model)
    outs = []
    at = 0
    for c in cuts:
        y, st = E.encode_append(model, st, subj[at:at + c], types[at:at + c])
        outs.append(y)
        at += c
    inc = np.concatenate(outs, axis=0)
    assert np.abs(inc - full).max() < 1e-12
    for l in range(model.n_layers):
        assert np.abs(st.K[l] - st_full.K[l]).max() < 1e-12
        assert np.abs(st.V[l] - st_full.V[l]).max() < 1e-12


def test_causal():
    ew, model = _model()
    subj, types = _tokens(ew, 20, 4)
    a, _ = E.encode(model, subj, types)
    subj2 = subj.copy()
    subj2[12:] += 1.0
    b, _ = E.encode(model, subj2, types)
    assert np.array_equal(a[:12], b[:12])
    assert np.abs(a[12:] - b[12:]).max() > 1e-3


def test_bias_shift_invariance():
    ew, model = _model()
    subj, types = _tokens(ew, 17, 5)
    a, _ = E.encode(model, subj, types)
    for l in range(model.n_layers):
        model.w[f"rel_bias.{l}"] = model.w[f"rel_bias.{l}"] + np.array([[3.0], [-2.0]])
    b, _ = E.encode(model, subj, types)
    assert np.abs(a - b).max() < 1e-12


def test_bias_matters():
    ew, model = _model()
    subj, types = _tokens(ew, 17, 5)
    a, _ = E.encode(model, subj, types)
    model.w["rel_bias.0"] = model.w["rel_bias.0"][:, ::-1].copy()
    b, _ = E.encode(model, subj, types)
    assert np.abs(a - b).max() > 1e-3


def test_window_relative_only():
    # with window w, token i depends only on tokens i - nL (w - 1) .. i, and
    # only through their relative positions
    w = 4
    ew, model = _model(window=w)
    subj, types = _tokens(ew, 30, 6)
    full, _ = E.encode(model, subj, types)
    span = model.n_layers * (w - 1) + 1
    for i in (span - 1, 17, 29):
        part, _ = E.encode(model, subj[i - span + 1:i + 1], types[i - span + 1:i + 1])
        assert np.abs(part[-1] - full[i]).max() < 1e-12


def test_window_reductions():
    ew, model = _model(window=0)
    subj, types = _tokens(ew, 15, 7)
    a, _ = E.encode(model, subj, types)
    model.window = 15
    b, _ = E.encode(model, subj, types)
    assert np.abs(a - b).max() < 1e-13
    # window 1: every token attends to itself only, so attention returns v
    model.window = 1
    X = E.embed(model, subj, types)
    qkv = X @ model.w["W_qkv.0"] + model.w["b_qkv.0"]
    pos = np.arange(15)
    d = ew.d_model
    att = E.causal_attention(qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:], model.n_heads, model.w["rel_bias.0"],
                             pos, pos, 1)
    assert np.abs(att - qkv[:, 2 * d:]).max() < 1e-13


def test_batch_is_per_user():
    ew, model = _model()
    b = W.enc_batch(ew)
    phi, states = E.encode_batch(model, b.subj, b.types, b.off)
    r = 1
    own, _ = E.encode(model, b.subj[b.off[r]:b.off[r + 1]], b.types[b.off[r]:b.off[r + 1]])
    assert np.array_equal(phi[b.off[r]:b.off[r + 1]], own)
    new, _ = E.append_batch(model, states, b.subj_app, b.types_app, b.app_off)
    assert new.shape == (int(b.dL.sum()), ew.d_model)


def test_empty_streams():
    ew, model = _model()
    subj, types = _tokens(ew, 0, 8)
    y, st = E.encode(model, subj, types)
    assert y.shape == (0, ew.d_model) and st.length == 0
    s2, t2 = _tokens(ew, 6, 8)
    a, sa = E.encode_append(model, st, s2, t2)
    b, _ = E.encode(model, s2, t2)
    assert np.array_equal(a, b)
    y, sb = E.encode_append(model, sa, subj, types)
    assert y.shape == (0, ew.d_model) and sb.length == 6
