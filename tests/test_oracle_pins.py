"""Pins for the fp64 oracle, each against something other than the oracle itself.

* closed forms of softmax attention, LayerNorm, GELU and the k = 2 head;
* PyTorch's own ``TransformerDecoderLayer`` / ``scaled_dot_product_attention``
  / ``layer_norm`` in float64 (library routines for the textbook definitions the
  paper cites: post-LN blocks with a residual, Sec. 4.1.2 crossAttend equation);
* the invariants the paper asserts: shared K/V equals per-candidate recompute
  (Sec. 4.1.2 multi-query formulation, Sec. 4.3 KV caching), per-candidate
  factorisation (Sec. 4.1.3), append equals rebuild (App. D remark), and
  LOCAL_GLOBAL with a window covering everything and no anchor equals FULL
  (Sec. 5.2, -sparseAttn).
"""
import math

import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W

RNG = np.random.default_rng(7)


def _tiny(**kw):
    wl = W.with_sizes(W.WORKLOADS["tiny_fp32"], **kw)
    model = O.Model.from_arrays(W.weights(wl), wl)
    return wl, model


# ---------------------------------------------------------------- attention closed forms

def test_attention_single_key_returns_value():
    q = RNG.standard_normal((5, 8))
    k = RNG.standard_normal((1, 8))
    v = RNG.standard_normal((1, 8))
    out = O.attention(q, k, v, n_heads=2)
    np.testing.assert_allclose(out, np.repeat(v, 5, axis=0), rtol=0, atol=1e-15)


def test_attention_identical_keys_average_values():
    q = RNG.standard_normal((3, 8))
    k = np.repeat(RNG.standard_normal((1, 8)), 4, axis=0)
    v = RNG.standard_normal((4, 8))
    out = O.attention(q, k, v, n_heads=2)
    np.testing.assert_allclose(out, np.repeat(v.mean(0, keepdims=True), 3, axis=0), atol=1e-14)


def test_attention_zero_query_is_mean_of_values():
    k = RNG.standard_normal((6, 8))
    v = RNG.standard_normal((6, 8))
    out = O.attention(np.zeros((2, 8)), k, v, n_heads=4)
    np.testing.assert_allclose(out, np.repeat(v.mean(0, keepdims=True), 2, axis=0), atol=1e-14)


def test_attention_two_keys_closed_form():
    # one head of width 4: weights are sigmoid(+-(s1 - s2)) with s = q.k / 2
    q = np.array([[1.0, 2.0, 0.0, -1.0]])
    k = np.array([[0.5, 0.0, 1.0, 0.0], [0.0, 1.0, 0.0, 1.0]])
    v = np.array([[1.0, 0.0, 3.0, 0.0], [0.0, 2.0, 0.0, -4.0]])
    s1, s2 = 0.5 / 2.0, 1.0 / 2.0
    a = 1.0 / (1.0 + math.exp(-(s1 - s2)))
    want = a * v[0] + (1 - a) * v[1]
    np.testing.assert_allclose(O.attention(q, k, v, n_heads=1)[0], want, atol=1e-15)


def test_attention_dominant_key_selects_its_value():
    k = np.zeros((5, 4))
    k[3] = [200.0, 0, 0, 0]
    v = RNG.standard_normal((5, 4))
    out = O.attention(np.array([[10.0, 0, 0, 0]]), k, v, n_heads=1)
    np.testing.assert_allclose(out[0], v[3], atol=1e-12)


@pytest.mark.parametrize("heads", [1, 2, 4])
def test_attention_matches_torch_sdpa_with_mask(heads):
    n, m, d = 7, 9, 16
    q, k, v = (RNG.standard_normal((x, d)) for x in (n, m, m))
    allowed = RNG.random((n, m)) < 0.6
    allowed[:, 0] = True
    out = O.attention(q, k, v, heads, allowed)
    dh = d // heads
    tq = torch.from_numpy(q).reshape(n, heads, dh).transpose(0, 1)
    tk = torch.from_numpy(k).reshape(m, heads, dh).transpose(0, 1)
    tv = torch.from_numpy(v).reshape(m, heads, dh).transpose(0, 1)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, attn_mask=torch.from_numpy(allowed))
    ref = ref.transpose(0, 1).reshape(n, d).numpy()
    np.testing.assert_allclose(out, ref, atol=1e-13)


# ---------------------------------------------------------------- LN, GELU

def test_layer_norm_constant_row_gives_beta():
    g, b = RNG.standard_normal(8), RNG.standard_normal(8)
    y = np.full((3, 8), 2.5)
    np.testing.assert_allclose(O.layer_norm(y, g, b, 1e-5), np.repeat(b[None], 3, 0), atol=1e-15)


def test_layer_norm_moments_and_torch():
    y = RNG.standard_normal((4, 32)) * 3 + 1
    out = O.layer_norm(y, np.ones(32), np.zeros(32), 0.0)
    np.testing.assert_allclose(out.mean(-1), 0, atol=1e-13)
    np.testing.assert_allclose((out ** 2).mean(-1), 1, atol=1e-12)  # biased variance
    g, b = RNG.standard_normal(32), RNG.standard_normal(32)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(y), (32,), torch.from_numpy(g),
                                         torch.from_numpy(b), eps=1e-5).numpy()
    np.testing.assert_allclose(O.layer_norm(y, g, b, 1e-5), ref, atol=1e-13)


def test_gelu_closed_forms():
    assert O.gelu(np.array([0.0]))[0] == 0.0
    x = RNG.standard_normal(50) * 3
    np.testing.assert_allclose(O.gelu(x) - O.gelu(-x), x, atol=1e-14)
    # GELU(1) = Phi(1), the standard normal CDF at 1 (textbook value)
    assert abs(O.gelu(np.array([1.0]))[0] - 0.8413447460685429) < 1e-15
    ref = torch.nn.functional.gelu(torch.from_numpy(x), approximate="none").numpy()
    np.testing.assert_allclose(O.gelu(x), ref, atol=1e-14)


# ---------------------------------------------------------------- head

def test_head_two_actions_is_sigmoid():
    wl, model = _tiny(n_actions=2)
    z = RNG.standard_normal((5, wl.d_model))
    x = RNG.standard_normal((5, wl.d_model))
    logits, p = O.head(model, z, x)
    sig = 1.0 / (1.0 + np.exp(-(logits[:, 0] - logits[:, 1])))
    np.testing.assert_allclose(p[:, 0], sig, atol=1e-15)
    np.testing.assert_allclose(p.sum(1), 1.0, atol=1e-15)


def test_head_uniform_action_tokens_give_uniform_probs():
    wl, model = _tiny()
    model.w["Q_dec"] = np.repeat(model.w["Q_dec"][:1], wl.n_actions, axis=0)
    _, p = O.head(model, RNG.standard_normal((3, wl.d_model)), RNG.standard_normal((3, wl.d_model)))
    np.testing.assert_allclose(p, 1.0 / wl.n_actions, atol=1e-15)


def test_head_logits_are_bilinear_in_k_dec():
    # logits_a = q_a . k_dec with k_dec = z W_dec[:d] + x W_dec[d:] + b_dec (Sec. 4.1.3)
    wl, model = _tiny()
    d = wl.d_model
    z = np.zeros((1, d))
    x = np.zeros((1, d))
    logits, _ = O.head(model, z, x)
    np.testing.assert_allclose(logits[0], model.w["Q_dec"] @ model.w["b_dec"], atol=1e-15)
    e = np.zeros((1, d)); e[0, 3] = 1.0
    logits_z, _ = O.head(model, e, x)
    want = model.w["Q_dec"] @ (model.w["W_dec"][3] + model.w["b_dec"])
    np.testing.assert_allclose(logits_z[0], want, atol=1e-15)
    logits_x, _ = O.head(model, z, e)
    want = model.w["Q_dec"] @ (model.w["W_dec"][d + 3] + model.w["b_dec"])
    np.testing.assert_allclose(logits_x[0], want, atol=1e-15)


# ---------------------------------------------------------------- pooling

def test_pool_zero_weight_gives_mean():
    wl, model = _tiny()
    model.w["w_pool"] = np.zeros(wl.d_model)
    phi = RNG.standard_normal((11, wl.d_model))
    np.testing.assert_allclose(O.pool_direct(model, phi).g, phi.mean(0), atol=1e-15)


def test_pool_dominant_row():
    wl, model = _tiny()
    d = wl.d_model
    model.w["w_pool"] = np.zeros(d); model.w["w_pool"][0] = 1.0
    phi = RNG.standard_normal((6, d))
    phi[2, 0] = 1e4
    np.testing.assert_allclose(O.pool_direct(model, phi).g, phi[2], atol=1e-12)


def test_pool_merge_equals_direct():
    wl, model = _tiny()
    model.w["w_pool"] = RNG.standard_normal(wl.d_model)  # large weights: non-uniform alpha
    phi = RNG.standard_normal((40, wl.d_model))
    whole = O.pool_direct(model, phi)
    for cut in (1, 17, 39):
        merged = O.pool_merge(O.pool_direct(model, phi[:cut]), O.pool_direct(model, phi[cut:]))
        np.testing.assert_allclose(merged.g, whole.g, atol=1e-13)
    alpha = np.exp(phi @ model.w["w_pool"] / math.sqrt(wl.d_model))
    alpha /= alpha.sum()
    np.testing.assert_allclose(whole.g, alpha @ phi, atol=1e-13)


def test_single_row_history():
    # L = 1: g is that row, the key set is {row, g}; both keys are equal, so the
    # cross-attention output of every query is that row's V.
    wl, model = _tiny()
    phi = RNG.standard_normal((1, wl.d_model))
    c = O.build_cache(model, phi)
    np.testing.assert_allclose(c.pool.g, phi[0], atol=1e-15)
    K, V = O.key_set(model, c, 0, O.LOCAL_GLOBAL)
    assert K.shape[0] == 2
    out = O.attention(RNG.standard_normal((4, wl.d_model)), K, V, wl.n_heads)
    np.testing.assert_allclose(out, np.repeat(V[:1], 4, 0), atol=1e-14)


def test_cold_start_rejected():
    wl, model = _tiny()
    with pytest.raises(ValueError):
        O.build_cache(model, np.zeros((0, wl.d_model)))


# ---------------------------------------------------------------- decoder vs PyTorch

def _torch_layer(model, l):
    w, d, H = model.w, model.d_model, model.n_heads
    F = w[f"W_1.{l}"].shape[1]
    layer = torch.nn.TransformerDecoderLayer(d, H, F, dropout=0.0, activation="gelu",
                                             batch_first=True, norm_first=False,
                                             layer_norm_eps=model.ln_eps, dtype=torch.float64)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))
    sd = {
        "self_attn.in_proj_weight": t(w[f"W_qkv.{l}"].T), "self_attn.in_proj_bias": t(w[f"b_qkv.{l}"]),
        "self_attn.out_proj.weight": t(w[f"W_os.{l}"].T), "self_attn.out_proj.bias": t(w[f"b_os.{l}"]),
        "multihead_attn.in_proj_weight": t(np.concatenate([w[f"W_Q.{l}"].T, w[f"W_K.{l}"].T, w[f"W_V.{l}"].T])),
        "multihead_attn.in_proj_bias": t(np.concatenate([w[f"b_Q.{l}"], w[f"b_K.{l}"], w[f"b_V.{l}"]])),
        "multihead_attn.out_proj.weight": t(w[f"W_oc.{l}"].T), "multihead_attn.out_proj.bias": t(w[f"b_oc.{l}"]),
        "linear1.weight": t(w[f"W_1.{l}"].T), "linear1.bias": t(w[f"b_1.{l}"]),
        "linear2.weight": t(w[f"W_2.{l}"].T), "linear2.bias": t(w[f"b_2.{l}"]),
        "norm1.weight": t(w[f"ln1_g.{l}"]), "norm1.bias": t(w[f"ln1_b.{l}"]),
        "norm2.weight": t(w[f"ln2_g.{l}"]), "norm2.bias": t(w[f"ln2_b.{l}"]),
        "norm3.weight": t(w[f"ln3_g.{l}"]), "norm3.bias": t(w[f"ln3_b.{l}"]),
    }
    layer.load_state_dict(sd)
    layer.eval()
    return layer


def torch_score(model, phi, ctx, cand, mode, use_global=True, head_x=None):
    """Independent recompute with PyTorch modules: K/V are projected from Phi_b
    (and from the pooled g) inside torch's cross-attention, per call.  ``cand``
    enters the decoder; the head takes ``head_x`` (default: ``cand``)."""
    head_x = cand if head_x is None else head_x
    S = ctx.shape[0]
    if mode == O.FULL:
        memory = phi
    else:
        lo = max(0, phi.shape[0] - model.l_local)
        memory = phi[lo:]
        if use_global:
            a = torch.softmax(torch.from_numpy(phi @ model.w["w_pool"]) / math.sqrt(model.d_model), 0)
            g = (a[:, None] * torch.from_numpy(phi)).sum(0).numpy()
            memory = np.concatenate([memory, g[None]], 0)
    X = torch.from_numpy(np.concatenate([ctx, cand], 0))[None]
    mem = torch.from_numpy(memory)[None]
    n = X.shape[1]
    blocked = torch.ones(n, n, dtype=torch.bool)
    blocked[:, :S] = False
    blocked[torch.arange(S, n), torch.arange(S, n)] = False
    with torch.no_grad():
        for l in range(model.n_layers):
            X = _torch_layer(model, l)(X, mem, tgt_mask=blocked)
    z = X[0, S:].numpy()
    kdec = torch.nn.functional.linear(torch.from_numpy(np.concatenate([z, head_x], 1)),
                                      torch.from_numpy(model.w["W_dec"].T.copy()),
                                      torch.from_numpy(model.w["b_dec"]))
    logits = kdec @ torch.from_numpy(model.w["Q_dec"]).T
    return logits.numpy(), torch.softmax(logits, -1).numpy()


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("n_layers,L,S", [(1, 64, 2), (2, 7, 2), (2, 23, 0), (1, 3, 1)])
def test_decoder_matches_torch_transformer_decoder(mode, n_layers, L, S):
    wl, model = _tiny(n_layers=n_layers, n_ctx=S)
    phi = RNG.standard_normal((L, wl.d_model))
    ctx = RNG.standard_normal((S, wl.d_model))
    cand = RNG.standard_normal((9, wl.d_model))
    cache = O.build_cache(model, phi)
    lg, pr = O.score_request(model, cache, ctx, cand, mode)
    rl, rp = torch_score(model, phi, ctx, cand, mode)
    np.testing.assert_allclose(lg, rl, atol=1e-11)
    np.testing.assert_allclose(pr, rp, atol=1e-12)


def test_serving_attention_without_context_is_value_projection():
    # S = 0: a candidate attends only to itself, so the block's attention output
    # is (x W_v + b_v) W_os + b_os, head by head (App. B mask).
    wl, model = _tiny(n_ctx=0)
    w, d = model.w, wl.d_model
    x = RNG.standard_normal((5, d))
    qkv = x @ w["W_qkv.0"] + w["b_qkv.0"]
    a = O.attention(qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:], wl.n_heads, O.serving_mask(0, 5))
    np.testing.assert_allclose(a, qkv[:, 2 * d:], atol=1e-14)


# ---------------------------------------------------------------- invariants

def _request(wl, model, L, M, seed):
    rng = np.random.default_rng(seed)
    phi = rng.standard_normal((L, wl.d_model))
    ctx = rng.standard_normal((wl.n_ctx, wl.d_model))
    cand = rng.standard_normal((M, wl.d_model))
    return phi, ctx, cand


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_candidates_are_independent_of_order_and_batching(mode):
    wl, model = _tiny(n_layers=2)
    phi, ctx, cand = _request(wl, model, 50, 12, 1)
    cache = O.build_cache(model, phi)
    lg, _ = O.score_request(model, cache, ctx, cand, mode)
    perm = np.random.default_rng(2).permutation(12)
    lg_p, _ = O.score_request(model, cache, ctx, cand[perm], mode)
    np.testing.assert_allclose(lg_p, lg[perm], atol=1e-12)
    parts = [O.score_request(model, cache, ctx, cand[a:b], mode)[0] for a, b in ((0, 1), (1, 5), (5, 12))]
    np.testing.assert_allclose(np.concatenate(parts), lg, atol=1e-12)


def test_cached_kv_equals_recompute_per_candidate():
    # the shared cache serves every candidate; recomputing projections from Phi_b
    # for each candidate alone (torch, above) gives the same scores
    wl, model = _tiny(n_layers=2)
    phi, ctx, cand = _request(wl, model, 30, 6, 3)
    cache = O.build_cache(model, phi)
    lg, _ = O.score_request(model, cache, ctx, cand)
    for j in range(6):
        rl, _ = torch_score(model, phi, ctx, cand[j:j + 1], O.LOCAL_GLOBAL)
        np.testing.assert_allclose(lg[j], rl[0], atol=1e-11)


@pytest.mark.parametrize("L,dL", [(1, 1), (5, 7), (40, 1), (64, 30)])
def test_append_equals_rebuild(L, dL):
    wl, model = _tiny(n_layers=2)
    model.w["w_pool"] = RNG.standard_normal(wl.d_model) * 0.5
    phi = RNG.standard_normal((L + dL, wl.d_model))
    full = O.build_cache(model, phi)
    inc = O.append_cache(model, O.build_cache(model, phi[:L]), phi[L:])
    for l in range(2):
        np.testing.assert_allclose(inc.K[l], full.K[l], atol=1e-13)
        np.testing.assert_allclose(inc.V[l], full.V[l], atol=1e-13)
        np.testing.assert_allclose(inc.Kg[l], full.Kg[l], atol=1e-13)
        np.testing.assert_allclose(inc.Vg[l], full.Vg[l], atol=1e-13)
    _, ctx, cand = _request(wl, model, 1, 8, 4)
    for mode in (O.LOCAL_GLOBAL, O.FULL):
        np.testing.assert_allclose(O.score_request(model, inc, ctx, cand, mode)[0],
                                   O.score_request(model, full, ctx, cand, mode)[0], atol=1e-12)


def test_local_window_covering_history_without_anchor_equals_full():
    wl, model = _tiny(n_layers=2, l_local=100)
    phi, ctx, cand = _request(wl, model, 37, 5, 5)
    cache = O.build_cache(model, phi)
    a = O.score_request(model, cache, ctx, cand, O.LOCAL_GLOBAL, use_global=False)[0]
    b = O.score_request(model, cache, ctx, cand, O.FULL)[0]
    np.testing.assert_allclose(a, b, atol=1e-13)


def test_local_window_uses_most_recent_rows():
    wl, model = _tiny(l_local=10)
    phi, ctx, cand = _request(wl, model, 25, 3, 6)
    cache = O.build_cache(model, phi)
    K, V = O.key_set(model, cache, 0, O.LOCAL_GLOBAL)
    np.testing.assert_array_equal(K[:10], cache.K[0][15:])
    np.testing.assert_array_equal(K[10], cache.Kg[0])
    # changing a row outside the window changes nothing but the anchor; with the
    # anchor off the scores are unchanged
    phi2 = phi.copy(); phi2[3] += 5.0
    c2 = O.build_cache(model, phi2)
    np.testing.assert_allclose(O.score_request(model, c2, ctx, cand, use_global=False)[0],
                               O.score_request(model, cache, ctx, cand, use_global=False)[0], atol=1e-13)
    # a short history (L < L_local) attends to all of its rows
    c3 = O.build_cache(model, phi[:4])
    assert O.key_set(model, c3, 0, O.LOCAL_GLOBAL)[0].shape[0] == 5


def test_rank_ties_and_nan():
    s = np.array([0.2, 0.5, 0.2, np.nan, 0.9, 0.5, 0.1])
    (order,) = O.rank(s, [0, 7])
    np.testing.assert_array_equal(order, [4, 1, 5, 0, 2, 6, 3])
    (top,) = O.rank(s, [0, 7], top_k=3)
    np.testing.assert_array_equal(top, [4, 1, 5])
    o = O.rank(np.array([3.0, 1.0, 2.0, 5.0]), [0, 1, 4])
    np.testing.assert_array_equal(o[0], [0])
    np.testing.assert_array_equal(o[1], [2, 1, 0])
