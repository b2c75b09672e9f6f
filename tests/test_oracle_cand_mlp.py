"""Pins for the optional candidate-to-query encoder Phi_candidate of the
oracle (Sec. 4.1.2: "a simple instantiation ... is a multi-layer perceptron"):
the decoder sees GELU(x W_c1 + b_c1) W_c2 + b_c2, the head f_dec(z, x) the
raw candidate token x.

* an MLP that is the identity (W_c1 = W_c2 = I, b_c1 = +60, b_c2 = -60, so
  GELU acts as the identity on the shifted inputs) scores exactly like the
  model without one;
* against PyTorch: torch.nn.Sequential(Linear, GELU, Linear) feeding the
  PyTorch decoder stack, the raw token feeding the head;
* the slip of giving the head Phi_candidate(x) instead of x is caught.
"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W
from tests.test_oracle_pins import torch_score

RNG = np.random.default_rng(23)


def _models(hidden):
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_layers=2, cand_mlp=hidden)
    model = O.Model.from_arrays(W.weights(wl), wl)
    return wl, model


def test_identity_mlp_equals_no_mlp():
    wl, model = _models(64)
    d = wl.d_model
    model.w["W_c1"] = np.eye(d)
    model.w["b_c1"] = np.full(d, 60.0)
    model.w["W_c2"] = np.eye(d)
    model.w["b_c2"] = np.full(d, -60.0)
    plain = O.Model(model.w, model.n_layers, d, model.n_heads, model.n_ctx, model.n_actions, model.l_local,
                    model.ln_eps, 0, 0)
    phi = RNG.standard_normal((20, d))
    ctx = RNG.standard_normal((wl.n_ctx, d))
    cand = RNG.standard_normal((6, d))
    a = O.score_request(model, O.build_cache(model, phi), ctx, cand)
    b = O.score_request(plain, O.build_cache(plain, phi), ctx, cand)
    np.testing.assert_allclose(a[0], b[0], atol=1e-12)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("hidden", [64, 192])
def test_candidate_mlp_matches_torch(mode, hidden):
    wl, model = _models(hidden)
    w = model.w
    phi = RNG.standard_normal((30, wl.d_model))
    ctx = RNG.standard_normal((wl.n_ctx, wl.d_model))
    cand = RNG.standard_normal((7, wl.d_model))
    mlp = torch.nn.Sequential(torch.nn.Linear(wl.d_model, hidden, dtype=torch.float64), torch.nn.GELU(),
                              torch.nn.Linear(hidden, wl.d_model, dtype=torch.float64))
    with torch.no_grad():
        mlp[0].weight.copy_(torch.from_numpy(w["W_c1"].T.copy()))
        mlp[0].bias.copy_(torch.from_numpy(w["b_c1"]))
        mlp[2].weight.copy_(torch.from_numpy(w["W_c2"].T.copy()))
        mlp[2].bias.copy_(torch.from_numpy(w["b_c2"]))
        enc = mlp(torch.from_numpy(cand)).numpy()
    rl, rp = torch_score(model, phi, ctx, enc, mode, head_x=cand)
    lg, pr = O.score_request(model, O.build_cache(model, phi), ctx, cand, mode)
    np.testing.assert_allclose(lg, rl, atol=1e-11)
    np.testing.assert_allclose(pr, rp, atol=1e-12)


def test_head_on_encoded_token_is_caught(monkeypatch):
    wl, model = _models(64)
    phi = RNG.standard_normal((12, wl.d_model))
    ctx = RNG.standard_normal((wl.n_ctx, wl.d_model))
    cand = RNG.standard_normal((5, wl.d_model))
    ref, _ = O.score_request(model, O.build_cache(model, phi), ctx, cand)
    orig_head = O.head
    monkeypatch.setattr(O, "head", lambda m, z, x: orig_head(m, z, O.candidate_encoder(m, x)))
    bad, _ = O.score_request(model, O.build_cache(model, phi), ctx, cand)
    assert np.abs(bad - ref).max() > 1e-4
