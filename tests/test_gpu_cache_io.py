"""Cache export / import (App. D cache management: warm start from a persisted
cache, entries versioned by the model identifier and the feature schema).

An imported cache must behave exactly as the exported one: identical scores
(bit for bit, both key-set modes), identical K/V rows and anchors, and the
same result after a further append.  Blobs of another model or schema are
rejected as stale, damaged blobs as invalid."""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import upload_batch

pytestmark = pytest.mark.gpu


def _setup(base, mode, seed_shift=0):
    wl = W.with_sizes(W.WORKLOADS[base], n_req=5, L=[1, 9, 130, 700, 64], M=[3, 40, 0, 129, 7], dL=[2, 0, 5, 64, 1],
                      seed=W.WORKLOADS[base].seed + seed_shift)
    b = W.batch(wl)
    model = txs.Model(wl, W.weights(wl), mode)
    beh, cand, ctx, app = upload_batch(wl, b)
    cache = txs.KVCache(model, b.beh_off, beh, capacity_extra=64)
    return wl, b, model, cache, cand, ctx, app


@pytest.mark.parametrize("base", ["tiny_fp32", "small_bf16"])
@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_import_scores_and_appends_exactly_like_the_export(base, mode):
    wl, b, model, cache, cand, ctx, app = _setup(base, mode)
    blob = cache.export(schema_version=7)
    other = txs.KVCache.import_blob(model, blob, schema_version=7, capacity_extra=64)
    assert other.n_req == cache.n_req
    np.testing.assert_array_equal(other.lengths(), cache.lengths())
    l1, p1 = txs.score(model, cache, b.cand_off, cand, ctx)
    l2, p2 = txs.score(model, other, b.cand_off, cand, ctx)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
    np.testing.assert_array_equal(p1.cpu().numpy(), p2.cpu().numpy())
    for which in (0, 1, 2):
        np.testing.assert_array_equal(cache.read_anchor(wl.n_layers - 1, which).cpu().numpy(),
                                      other.read_anchor(wl.n_layers - 1, which).cpu().numpy())
    # the same append on both caches gives the same state and scores
    cache.append(b.app_off, app)
    other.append(b.app_off, app)
    np.testing.assert_array_equal(other.lengths(), cache.lengths())
    for r in range(cache.n_req):
        L = int(cache.lengths()[r])
        for which in (0, 1):
            np.testing.assert_array_equal(cache.read_rows(0, which, r, 0, L).cpu().float().numpy(),
                                          other.read_rows(0, which, r, 0, L).cpu().float().numpy())
    l1, _ = txs.score(model, cache, b.cand_off, cand, ctx)
    l2, _ = txs.score(model, other, b.cand_off, cand, ctx)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
    assert model.device_status() == txs.TXS_OK


def test_stale_and_damaged_blobs_are_rejected():
    wl, b, model, cache, cand, ctx, app = _setup("tiny_fp32", O.LOCAL_GLOBAL)
    blob = cache.export(schema_version=3)
    with pytest.raises(txs.TxsError) as e:                       # another feature schema
        txs.KVCache.import_blob(model, blob, schema_version=4)
    assert e.value.status == txs.TXS_ERR_STALE_CACHE
    w2 = W.weights(wl)
    w2["b_2.0"] = w2["b_2.0"] + 1.0
    model2 = txs.Model(wl, w2, O.LOCAL_GLOBAL)                   # another model (hash)
    with pytest.raises(txs.TxsError) as e:
        txs.KVCache.import_blob(model2, blob, schema_version=3)
    assert e.value.status == txs.TXS_ERR_STALE_CACHE
    with pytest.raises(txs.TxsError) as e:                       # truncated
        txs.KVCache.import_blob(model, blob[:-4], schema_version=3)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    bad = blob.copy()
    bad[0] ^= 0xFF                                               # not a cache blob
    with pytest.raises(txs.TxsError) as e:
        txs.KVCache.import_blob(model, bad, schema_version=3)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    assert model.device_status() == txs.TXS_OK
