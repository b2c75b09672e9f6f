"""Grouped K/V heads on the GPU (the MQA/GQA variants Sec. 4.1.2 cites to
shrink the behavior cache): the cache holds n_kv_heads * d_h-wide rows and
query head h attends with K/V head h // (n_heads / n_kv_heads).  Scores,
cached rows and anchors against the fp64 oracle in both key-set modes (the
FULL tensor-core kernel for bf16), through append, multi-event scoring and a
cache export/import round trip."""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import assert_scores_close, oracle_scores, rows_of, run_gpu

pytestmark = pytest.mark.gpu


def _wl(base, n_kv, **kw):
    spec = dict(n_req=4, L=[3, 11, 200, 700], M=[5, 129, 1, 40], dL=[2, 0, 9, 64])
    spec.update(kw)
    return W.with_sizes(W.WORKLOADS[base], n_kv_heads=n_kv, **spec)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("base,n_kv", [("tiny_fp32", 1), ("small_bf16", 1), ("small_bf16", 2),
                                       ("small_bf16", 4), ("mid_bf16", 2)])
def test_grouped_heads_scores_match_oracle(mode, base, n_kv):
    wl = _wl(base, n_kv, n_layers=2) if base != "tiny_fp32" else _wl(base, n_kv)
    g = run_gpu(wl, mode, append=True)
    lg, pr, caches, b = oracle_scores(wl, mode, append=True)
    assert_scores_close(g.logits, lg, wl.dtype, "logits")
    assert_scores_close(g.probs, pr, wl.dtype, "probs")
    dkv = txs.kv_width(wl)
    assert dkv == n_kv * wl.d_model // wl.n_heads
    tol = dict(atol=3e-2, rtol=1e-2) if wl.dtype == "bf16" else dict(atol=1e-5, rtol=1e-5)
    r = 3
    L = int(g.cache.lengths()[r])
    for which, ref in ((0, caches[r].K[1 if wl.n_layers > 1 else 0]), (1, caches[r].V[1 if wl.n_layers > 1 else 0])):
        rows = g.cache.read_rows(1 if wl.n_layers > 1 else 0, which, r, 0, L).float().cpu().numpy()
        assert rows.shape == (L, dkv)
        np.testing.assert_allclose(rows, ref, **tol)
    np.testing.assert_allclose(g.cache.read_anchor(0, 0).cpu().numpy(), np.stack([c.Kg[0] for c in caches]), **tol)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_grouped_heads_events_and_export(mode):
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_layers=2, n_kv_heads=2)
    weights = W.weights(wl)
    model = txs.Model(wl, weights, mode)
    ev = W.events(wl, 300, 4, [20, 1, 64, 9], 71)
    ev.ends[:] = [1, 10, 150, 300]
    dt = txs.torch_dtype(wl.dtype)
    beh = txs.to_device(ev.beh, dt)
    cache = txs.KVCache(model, np.array([0, 300], np.int32), beh, capacity_extra=4)
    cand = txs.to_device(ev.cand, dt)
    ctx = txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt)
    lg, _ = txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, cand, ctx)
    om = O.Model.from_arrays(weights, wl)
    rl, _ = O.score_events(om, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, mode)
    assert_scores_close(lg.cpu().numpy(), rl, "bf16", "event logits")
    other = txs.KVCache.import_blob(model, cache.export(1), 1, capacity_extra=4)
    lg2, _ = txs.score_events(model, other, 0, beh, ev.ends, ev.cand_off, cand, ctx)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lg.cpu().numpy(), lg2.cpu().numpy())
    assert model.device_status() == txs.TXS_OK
