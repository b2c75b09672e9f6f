"""Pins for grouped K/V heads in the oracle (the MQA/GQA variants Sec. 4.1.2
cites to shrink the cache): query head h attends with key/value head
h // (n_heads / n_kv_heads).

* a model with n_kv_heads K/V heads scores exactly like the multi-head model
  whose W_K, W_V (and biases) repeat each K/V head's columns for every query
  head of its group (the multi-head path is itself pinned to PyTorch);
* the attention function matches PyTorch's scaled_dot_product_attention with
  enable_gqa;
* a plausible slip (head h using K/V head h mod n_kv_heads) is caught.
"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W

RNG = np.random.default_rng(17)


def _expanded(model_g):
    """The multi-head model equivalent to a grouped one."""
    H, n_kv, d = model_g.n_heads, model_g.kv_heads, model_g.d_model
    dh, group = d // H, H // n_kv
    cols = np.concatenate([np.arange((h // group) * dh, (h // group + 1) * dh) for h in range(H)])
    w = dict(model_g.w)
    for l in range(model_g.n_layers):
        for name in ("W_K", "W_V"):
            w[f"{name}.{l}"] = model_g.w[f"{name}.{l}"][:, cols]
        for name in ("b_K", "b_V"):
            w[f"{name}.{l}"] = model_g.w[f"{name}.{l}"][cols]
    return O.Model(w, model_g.n_layers, d, H, model_g.n_ctx, model_g.n_actions, model_g.l_local,
                   model_g.ln_eps, 0)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("n_kv", [1, 2, 4])
def test_grouped_heads_equal_expanded_multi_head(mode, n_kv):
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_layers=2, n_heads=8, n_kv_heads=n_kv)
    model = O.Model.from_arrays(W.weights(wl), wl)
    assert model.w["W_K.0"].shape == (wl.d_model, n_kv * wl.d_model // 8)
    mha = _expanded(model)
    phi = RNG.standard_normal((23, wl.d_model))
    ctx = RNG.standard_normal((wl.n_ctx, wl.d_model))
    cand = RNG.standard_normal((7, wl.d_model))
    a = O.score_request(model, O.build_cache(model, phi), ctx, cand, mode)
    b = O.score_request(mha, O.build_cache(mha, phi), ctx, cand, mode)
    np.testing.assert_allclose(a[0], b[0], atol=1e-12)
    np.testing.assert_allclose(a[1], b[1], atol=1e-13)
    assert O.build_cache(model, phi).K[0].shape[1] == n_kv * wl.d_model // 8   # the cache shrinks


@pytest.mark.parametrize("n_kv", [1, 2, 4, 8])
def test_attention_matches_torch_sdpa_gqa(n_kv):
    H, dh, n, m = 8, 8, 5, 9
    q = RNG.standard_normal((n, H * dh))
    k = RNG.standard_normal((m, n_kv * dh))
    v = RNG.standard_normal((m, n_kv * dh))
    out = O.attention(q, k, v, H, n_kv_heads=n_kv)
    t = lambda a, h: torch.from_numpy(a).reshape(a.shape[0], h, dh).transpose(0, 1)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(t(q, H), t(k, n_kv), t(v, n_kv), enable_gqa=True)
    ref = ref[0].transpose(0, 1).reshape(n, H * dh).numpy()
    np.testing.assert_allclose(out, ref, atol=1e-13)


def test_wrong_head_grouping_is_caught(monkeypatch):
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], n_layers=1, n_heads=8, n_kv_heads=2)
    model = O.Model.from_arrays(W.weights(wl), wl)
    mha = _expanded(model)
    phi = RNG.standard_normal((15, wl.d_model))
    ctx = RNG.standard_normal((wl.n_ctx, wl.d_model))
    cand = RNG.standard_normal((4, wl.d_model))
    ref = O.score_request(mha, O.build_cache(mha, phi), ctx, cand, O.FULL)[0]
    orig = O.attention

    def modulo_grouping(q, k, v, n_heads, allowed=None, n_kv_heads=None):
        if n_kv_heads is None or n_kv_heads == n_heads:
            return orig(q, k, v, n_heads, allowed, n_kv_heads)
        dh = q.shape[1] // n_heads
        cols = np.concatenate([np.arange((h % n_kv_heads) * dh, (h % n_kv_heads + 1) * dh) for h in range(n_heads)])
        return orig(q, k[:, cols], v[:, cols], n_heads, allowed, None)
    monkeypatch.setattr(O, "attention", modulo_grouping)
    bad = O.score_request(model, O.build_cache(model, phi), ctx, cand, O.FULL)[0]
    assert np.abs(bad - ref).max() > 1e-4
