"""Pins of the Deep & Wide action head in the oracle (App. B).

f_dec(z, x) = [x_wide W_w + b_w, GELU([z, x_deep] W_d1 + b_d1) W_d2 + b_d2],
logits = Q_dec f_dec, probabilities = softmax(logits).  Checked against:
* torch modules (nn.Linear, nn.GELU, nn.Sequential, torch.softmax) in float64,
  on the z the oracle's (separately pinned) decoder stack produces;
* reductions: all features wide and no deep output -> the linear head with
  W_dec = [0; W_w], b_dec = b_w; no wide part -> a pure FFN of [z, x];
* exact linearity of the logits in the wide features;
* planted slips (wrong feature slice, concatenation orders, a dropped bias, a
  non-linearity on the wide part), each caught.
"""
import numpy as np
import pytest

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W

torch = pytest.importorskip("torch")


def _setup(dw_in=64, dw_out=32, dw_hidden=128, n_layers=2):
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_layers=n_layers, dw_in=dw_in, dw_out=dw_out,
                      dw_hidden=dw_hidden, d_model=128, n_heads=4)
    w = W.weights(wl)
    # larger deep weights so that GELU is not in its linear range
    for k in ("W_d1", "W_d2", "W_w"):
        w[k] = w[k] * 30.0
    model = O.Model.from_arrays(w, wl)
    rng = np.random.default_rng(5)
    return wl, model, rng.standard_normal((40, wl.d_model)), rng.standard_normal((wl.n_ctx, wl.d_model)), \
        rng.standard_normal((9, wl.d_model))


def torch_head(model, z, x):
    """The Deep & Wide head from torch modules."""
    w = model.w
    t = lambda a: torch.tensor(a, dtype=torch.float64)
    d, a = model.d_model, model.dw_in
    wide = torch.nn.Linear(a, model.dw_out, dtype=torch.float64)
    l1 = torch.nn.Linear(2 * d - a, model.dw_hidden, dtype=torch.float64)
    l2 = torch.nn.Linear(model.dw_hidden, d - model.dw_out, dtype=torch.float64)
    with torch.no_grad():
        wide.weight.copy_(t(w["W_w"].T))
        wide.bias.copy_(t(w["b_w"]))
        l1.weight.copy_(t(w["W_d1"].T))
        l1.bias.copy_(t(w["b_d1"]))
        l2.weight.copy_(t(w["W_d2"].T))
        l2.bias.copy_(t(w["b_d2"]))
        deep = torch.nn.Sequential(l1, torch.nn.GELU(), l2)
        zt, xt = t(z), t(x)
        kdec = torch.cat([wide(xt[:, :a]), deep(torch.cat([zt, xt[:, a:]], dim=1))], dim=1)
        logits = kdec @ t(w["Q_dec"]).T
        return logits.numpy(), torch.softmax(logits, dim=1).numpy()


def _z(model, cache, ctx, cand):
    """Decoder output z of the candidate rows (the oracle's pinned decoder stack)."""
    S = ctx.shape[0]
    X = np.concatenate([ctx, O.candidate_encoder(model, cand)], axis=0)
    for l in range(model.n_layers):
        Kc, Vc = O.key_set(model, cache, l, O.LOCAL_GLOBAL)
        X = O.decoder_layer(model, X, Kc, Vc, l, S)
    return X[S:]


@pytest.mark.parametrize("dw", [(64, 32, 128), (0, 0, 64), (128, 64, 192), (64, 127, 64)])
def test_matches_torch_modules(dw):
    wl, model, phi, ctx, cand = _setup(*dw)
    cache = O.build_cache(model, phi)
    lg, pr = O.score_request(model, cache, ctx, cand)
    z = _z(model, cache, ctx, cand)
    rl, rp = torch_head(model, z, cand)
    assert np.abs(lg - rl).max() < 1e-10
    assert np.abs(pr - rp).max() < 1e-12


def test_all_wide_reduces_to_linear_head():
    wl, model, phi, ctx, cand = _setup(64, 32, 64)
    d = model.d_model
    model.dw_in, model.dw_out = d, d
    rng = np.random.default_rng(6)
    model.w["W_w"] = rng.standard_normal((d, d)) * 0.1
    model.w["b_w"] = rng.standard_normal(d) * 0.1
    model.w["W_d1"] = rng.standard_normal((d, 64)) * 0.1      # [z, x_deep] has d columns
    model.w["W_d2"] = np.zeros((64, 0))
    model.w["b_d2"] = np.zeros(0)
    z = rng.standard_normal((9, d))
    lg, pr = O.head(model, z, cand)
    lin = O.Model(dict(model.w), model.n_layers, d, model.n_heads, model.n_ctx, model.n_actions, model.l_local,
                  model.ln_eps)
    lin.w["W_dec"] = np.concatenate([np.zeros((d, d)), model.w["W_w"]], axis=0)
    lin.w["b_dec"] = model.w["b_w"]
    rl, rp = O.head(lin, z, cand)
    assert np.abs(lg - rl).max() < 1e-12 and np.abs(pr - rp).max() < 1e-12


def test_no_wide_is_pure_ffn():
    wl, model, phi, ctx, cand = _setup(0, 0, 64)
    rng = np.random.default_rng(7)
    z = rng.standard_normal((9, model.d_model))
    lg, _ = O.head(model, z, cand)
    w = model.w
    h = np.concatenate([z, cand], axis=1) @ w["W_d1"] + w["b_d1"]
    h = h * 0.5 * (1.0 + np.vectorize(__import__("math").erf)(h / np.sqrt(2.0)))
    ref = (h @ w["W_d2"] + w["b_d2"]) @ w["Q_dec"].T
    assert np.abs(lg - ref).max() < 1e-10


def test_linear_in_wide_features():
    wl, model, phi, ctx, cand = _setup(64, 32, 128)
    rng = np.random.default_rng(8)
    z = rng.standard_normal((9, model.d_model))
    base, _ = O.head(model, z, cand)
    w = model.w
    for j in (0, 17, 63):
        x2 = cand.copy()
        x2[:, j] += 2.5
        moved, _ = O.head(model, z, x2)
        expect = 2.5 * (w["W_w"][j] @ w["Q_dec"][:, :model.dw_out].T)
        assert np.abs((moved - base) - expect[None, :]).max() < 1e-10
    # a deep feature moves the logits non-linearly
    x3 = cand.copy()
    x3[:, 70] += 2.5
    x4 = cand.copy()
    x4[:, 70] += 5.0
    d1 = O.head(model, z, x3)[0] - base
    d2 = O.head(model, z, x4)[0] - base
    assert np.abs(d2 - 2 * d1).max() > 1e-6


_orig = O.f_dec_deep_wide


def _wrong_slice(model, z, x):
    a = model.dw_in
    return _orig(model, z, np.concatenate([x[:, -a:], x[:, :-a]], axis=1) if a else x)


def _deep_order(model, z, x):
    w, a = model.w, model.dw_in
    wide = x[:, :a] @ w["W_w"] + w["b_w"]
    deep = O.gelu(np.concatenate([x[:, a:], z], axis=1) @ w["W_d1"] + w["b_d1"]) @ w["W_d2"] + w["b_d2"]
    return np.concatenate([wide, deep], axis=1)


def _kdec_order(model, z, x):
    k = _orig(model, z, x)
    b = model.dw_out
    return np.concatenate([k[:, b:], k[:, :b]], axis=1)


def _no_wide_bias(model, z, x):
    k = _orig(model, z, x).copy()
    k[:, :model.dw_out] -= model.w["b_w"]
    return k


def _gelu_wide(model, z, x):
    k = _orig(model, z, x).copy()
    k[:, :model.dw_out] = O.gelu(k[:, :model.dw_out])
    return k


@pytest.mark.parametrize("fn", [_wrong_slice, _deep_order, _kdec_order, _no_wide_bias, _gelu_wide])
def test_mutants_caught(fn, monkeypatch):
    wl, model, phi, ctx, cand = _setup(64, 32, 128)
    cache = O.build_cache(model, phi)
    z = _z(model, cache, ctx, cand)
    monkeypatch.setattr(O, "f_dec_deep_wide", fn)
    lg, _ = O.score_request(model, cache, ctx, cand)
    rl, _ = torch_head(model, z, cand)
    assert np.abs(lg - rl).max() > 1e-6
