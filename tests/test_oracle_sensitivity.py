"""The sharp test weights make key-set errors visible at the bf16 tolerances.

With the plain N(0, 0.02) weights every attention softmax over the cached
keys is nearly uniform, so the cross-attention output is about b_V plus a
term of order 1/sqrt(L), and logits have a standard deviation of ~0.14:
reading the wrong keys moves the scores by less than the bf16 tolerances
(max|d| 2e-2, mean|d| 2e-3).  ``workload.sharp_weights`` applies
power-of-two gains (exact in bf16) to the attention projections, the
cross-attention output, the head and the pooling vector.

Each case below plants one error of the kind a cross-attention or serving-
stream attention kernel can make into a copy of the oracle (a patched function, on the CPU; no kernel is
touched) and checks that, at the sharp weights and the shapes of the small
(d = 256, d_h = 32) and mid (d = 512, d_h = 64) workloads, the scores move by
more than the bf16 tolerances.  A GPU parity test at these weights therefore
fails if the kernel makes that error.  The key sets are the ones of the
sparse cross-attention equation of Sec. 4.1.2 (the last L_local rows plus the
global token) and of -sparseAttn in Sec. 5.2 (all rows).
"""
import numpy as np
import pytest

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W

BF16_MAX, BF16_MEAN = 2e-2, 2e-3
TILE = 128        # key rows per staged K/V tile of the tensor-core attention

_key_set = O.key_set
_attention = O.attention


def _full_last_tile_dropped(model, cache, l, mode, use_global=True):
    K, V = _key_set(model, cache, l, mode, use_global)
    if mode == O.FULL:
        n = K.shape[0] - ((K.shape[0] - 1) % TILE + 1)
        return K[:max(n, 1)], V[:max(n, 1)]
    return K, V


def _full_second_half_dropped(model, cache, l, mode, use_global=True):
    K, V = _key_set(model, cache, l, mode, use_global)
    if mode == O.FULL:
        return K[:K.shape[0] // 2], V[:V.shape[0] // 2]
    return K, V


def _window_one_short(model, cache, l, mode, use_global=True):
    K, V = _key_set(model, cache, l, mode, use_global)
    return (K[1:], V[1:]) if mode == O.LOCAL_GLOBAL else (K, V)


def _window_shifted_back(model, cache, l, mode, use_global=True):
    # the window ends one row early: rows [L - L_local - 1, L - 1) + anchor
    if mode != O.LOCAL_GLOBAL:
        return _key_set(model, cache, l, mode, use_global)
    L = cache.length
    lo, hi = max(0, L - model.l_local - 1), L - 1
    K = np.concatenate([cache.K[l][lo:hi], cache.Kg[l][None, :]], axis=0)
    V = np.concatenate([cache.V[l][lo:hi], cache.Vg[l][None, :]], axis=0)
    return K, V


def _anchor_dropped(model, cache, l, mode, use_global=True):
    return _key_set(model, cache, l, mode, False)


def _next_kv_head(q, k, v, n_heads, allowed=None, n_kv_heads=None):
    if allowed is not None:          # the serving-stream attention is left alone
        return _attention(q, k, v, n_heads, allowed, n_kv_heads)
    dh = q.shape[1] // n_heads
    return _attention(q, np.roll(k, -dh, axis=1), np.roll(v, -dh, axis=1), n_heads, allowed, n_kv_heads)


_serving_mask = O.serving_mask


def _serving_self_dropped(n_ctx, n_cand):
    # a candidate sees the context rows but not itself
    m = _serving_mask(n_ctx, n_cand)
    m[np.arange(n_ctx, n_ctx + n_cand), np.arange(n_ctx, n_ctx + n_cand)] = False
    return m


def _serving_last_context_row_dropped(n_ctx, n_cand):
    m = _serving_mask(n_ctx, n_cand)
    if n_ctx > 1:
        m[n_ctx:, n_ctx - 1] = False
    return m


def _serving_context_rows_of_other_request(n_ctx, n_cand):
    # a candidate reads the context keys at the wrong rows: its own row and
    # the next candidate instead of the context rows
    m = _serving_mask(n_ctx, n_cand)
    rows = np.arange(n_ctx, n_ctx + n_cand)
    m[rows, :n_ctx] = False
    m[rows, n_ctx + (rows - n_ctx + 1) % n_cand] = True
    return m


SLIPS = {
    "serving_self_key_dropped": ("serving_mask", _serving_self_dropped, O.LOCAL_GLOBAL),
    "serving_last_context_row_dropped": ("serving_mask", _serving_last_context_row_dropped, O.LOCAL_GLOBAL),
    "serving_wrong_context_keys": ("serving_mask", _serving_context_rows_of_other_request, O.LOCAL_GLOBAL),
    "full_last_key_tile_dropped": ("key_set", _full_last_tile_dropped, O.FULL),
    "full_half_of_keys_dropped": ("key_set", _full_second_half_dropped, O.FULL),
    "full_query_head_reads_next_kv_head": ("attention", _next_kv_head, O.FULL),
    "lg_query_head_reads_next_kv_head": ("attention", _next_kv_head, O.LOCAL_GLOBAL),
    "lg_window_one_short": ("key_set", _window_one_short, O.LOCAL_GLOBAL),
    "lg_window_shifted_back": ("key_set", _window_shifted_back, O.LOCAL_GLOBAL),
    "lg_anchor_dropped": ("key_set", _anchor_dropped, O.LOCAL_GLOBAL),
}

_CACHE = {}


def _setup(name):
    if name not in _CACHE:
        wl = W.WORKLOADS[name]
        model = O.Model.from_arrays(W.sharp_weights(wl), wl)
        b = W.batch(wl, requests=[0, wl.n_req - 1], M_override=64)
        caches = O.build_caches(model, b.beh, b.beh_off)
        base = {m: O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, m) for m in (O.LOCAL_GLOBAL, O.FULL)}
        _CACHE[name] = (model, b, caches, base)
    return _CACHE[name]


@pytest.mark.parametrize("name", ["small_bf16", "mid_bf16"])
def test_sharp_weights_are_exact_in_bf16_and_sharpen_the_scores(name):
    wl = W.WORKLOADS[name]
    sw = W.sharp_weights(wl)
    for k, v in sw.items():
        np.testing.assert_array_equal(W.round_bf16(v), v, err_msg=k)
    model, b, caches, base = _setup(name)
    for mode in (O.LOCAL_GLOBAL, O.FULL):
        assert 0.2 < base[mode][0].std() < 0.6          # logits: ~0.3 (d = 256: ~0.14 with the plain weights)
    # pooling puts far more than uniform weight on its largest row
    phi = b.beh[b.beh_off[0]:b.beh_off[1]].astype(np.float64)
    z = O.pool_logits(model, phi)
    assert np.exp(z.max() - caches[0].pool.m) / caches[0].pool.s > 8.0 / phi.shape[0]


@pytest.mark.parametrize("slip", sorted(SLIPS))
@pytest.mark.parametrize("name", ["small_bf16", "mid_bf16"])
def test_key_set_slip_exceeds_bf16_tolerance(name, slip, monkeypatch):
    model, b, caches, base = _setup(name)
    attr, fn, mode = SLIPS[slip]
    monkeypatch.setattr(O, attr, fn)
    lg, pr = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, mode)
    monkeypatch.undo()
    dl, dp = np.abs(lg - base[mode][0]), np.abs(pr - base[mode][1])
    seen = max(dl.max(), dp.max()) > BF16_MAX or max(dl.mean(), dp.mean()) > BF16_MEAN
    assert seen, (f"{slip} at {name}: logits max {dl.max():.2e} mean {dl.mean():.2e}, "
                  f"probs max {dp.max():.2e} mean {dp.mean():.2e}")


def test_plain_weights_hide_the_slips():
    # the reason for the sharp weights: at the plain ones a dropped key tile
    # stays inside the bf16 tolerances
    wl = W.WORKLOADS["small_bf16"]
    model = O.Model.from_arrays(W.weights(wl), wl)
    b = W.batch(wl, requests=[0, wl.n_req - 1], M_override=64)
    caches = O.build_caches(model, b.beh, b.beh_off)
    lg0, _ = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, O.FULL)
    O_key_set = O.key_set
    try:
        O.key_set = _full_last_tile_dropped
        lg1, _ = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, O.FULL)
    finally:
        O.key_set = O_key_set
    d = np.abs(lg1 - lg0)
    assert d.max() < BF16_MAX and d.mean() < BF16_MEAN
