"""Deep & Wide action head on the GPU (App. B): k_dec = [x_wide W_w + b_w,
GELU([z, x_deep] W_d1 + b_d1) W_d2 + b_d2], logits = Q_dec k_dec, against the
fp64 oracle through the C ABI, both key-set modes, fp32 and bf16, with appends,
the candidate MLP, grouped K/V heads and multi-event scoring.  The head's
weights are scaled by powers of two (exact in bf16): W_w x8, W_d1 x4, W_d2 x4
and Q_dec by a per-case factor, so that the logits have a standard deviation
of 0.3 to 0.6 and the head, not the biases, decides the scores.  (The main
workloads' linear-head logits have a standard deviation near 0.14; the logit
tolerance is absolute.  At a standard deviation near 1 the bf16 path is off
by 0.26 % of it in mean: the deep FFN runs on the tensor cores, so z and
x_deep enter it rounded to bf16.)"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import assert_scores_close, oracle_scores, run_gpu

pytestmark = pytest.mark.gpu


def _weights(wl, q=4.0):
    w = W.weights(wl)
    for k, f in (("W_w", 8.0), ("W_d1", 4.0), ("W_d2", 4.0), ("Q_dec", q)):
        w[k] = w[k] * f
    return w


def _wl(base, dw_in, dw_out, dw_hidden, **kw):
    spec = dict(n_req=4, L=[3, 11, 200, 700], M=[5, 129, 1, 40], dL=[2, 0, 9, 64])
    spec.update(kw)
    return W.with_sizes(W.WORKLOADS[base], dw_in=dw_in, dw_out=dw_out, dw_hidden=dw_hidden, **spec)


CASES = [  # (workload, dw_in, dw_out, dw_hidden, Q_dec factor, other fields)
    ("tiny_fp32", 64, 16, 128, 8.0, {}),
    ("tiny_fp32", 0, 0, 64, 16.0, {}),
    ("small_bf16", 64, 32, 256, 1.0, dict(n_layers=2)),
    ("small_bf16", 256, 128, 64, 1.0, dict(n_layers=2)),
    ("small_bf16", 128, 0, 192, 1.0, dict(n_layers=2, cand_mlp=128, n_kv_heads=2)),
    ("mid_bf16", 128, 64, 512, 0.5, dict(n_layers=2)),
]


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("base,a,o,fh,q,kw", CASES)
def test_deep_wide_scores_match_oracle(mode, base, a, o, fh, q, kw):
    wl = _wl(base, a, o, fh, **kw)
    w = _weights(wl, q)
    g = run_gpu(wl, mode, append=True, weights=w)
    lg, pr, _, _ = oracle_scores(wl, mode, append=True, weights=w)
    assert 0.25 < lg.std() < 1.5, "the head must decide the scores"
    assert_scores_close(g.logits, lg, wl.dtype, "logits")
    assert_scores_close(g.probs, pr, wl.dtype, "probs")


def test_unused_linear_head_weights_may_be_null():
    wl = _wl("small_bf16", 64, 32, 128, n_layers=2)
    w = _weights(wl, 1.0)
    g = run_gpu(wl, O.LOCAL_GLOBAL, weights=w)
    w2 = {k: v for k, v in w.items() if k not in ("W_dec", "b_dec")}
    g2 = run_gpu(wl, O.LOCAL_GLOBAL, weights=w2)
    assert np.array_equal(g.logits, g2.logits)
    assert g.model.hash == g2.model.hash
    w3 = dict(w)
    w3["b_d1"] = w3["b_d1"] + 1.0
    assert txs.Model(wl, w3).hash != g.model.hash


def test_deep_wide_events():
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_layers=2, dw_in=64, dw_out=32, dw_hidden=128)
    w = _weights(wl, 1.0)
    model = txs.Model(wl, w, O.FULL)
    ev = W.events(wl, 200, 3, [20, 1, 64], 73)
    dt = txs.torch_dtype(wl.dtype)
    beh = txs.to_device(ev.beh, dt)
    cache = txs.KVCache(model, np.array([0, 200], np.int32), beh)
    lg, pr = txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, txs.to_device(ev.cand, dt),
                              txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt))
    torch.cuda.synchronize()
    rl, rp = O.score_events(O.Model.from_arrays(w, wl), ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, O.FULL)
    assert_scores_close(lg.cpu().numpy(), rl, "bf16", "event logits")
    assert_scores_close(pr.cpu().numpy(), rp, "bf16", "event probs")


def test_full_size_sampled_requests():
    """The benchmark's Deep & Wide configuration: the whole small_bf16 batch
    (32 requests x 256 candidates) scored on the GPU; requests 0 and 31
    against the oracle."""
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], dw_in=64, dw_out=32, dw_hidden=256)
    w = _weights(wl, 1.0)
    g = run_gpu(wl, O.LOCAL_GLOBAL, append=True, weights=w)
    assert np.isfinite(g.logits).all()
    for r in (0, wl.n_req - 1):
        lg, pr, _, _ = oracle_scores(wl, O.LOCAL_GLOBAL, requests=[r], append=True, weights=w)
        sl = slice(g.batch.cand_off[r], g.batch.cand_off[r + 1])
        assert_scores_close(g.logits[sl], lg, "bf16", f"logits request {r}")
        assert_scores_close(g.probs[sl], pr, "bf16", f"probs request {r}")
