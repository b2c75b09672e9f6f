"""The allocation-free anchor pooling entry point (txs_pool_anchor_static).

It exists for callers that cannot allocate device memory while they serve:
a process that reserves its GPU memory up front and forbids driver
allocations later, a plugin inside another runtime without an allocator of its
own, or a path that cannot take the device synchronisation cudaMalloc and
cudaFree imply.  Its scratch is a fixed array inside the library, shared by
every call, so the test checks two calls in a row: the second must not see
anything the first left behind.  Both are compared with the pooled anchor
that the cache build (txs_build_kv_cache, read back with
txs_cache_read_anchor) computes for the same rows, and with the fp64
oracle's attention pooling of each request's rows (alpha = softmax(phi .
w_pool / sqrt(d)), g = alpha^T phi; Sec. 4.1.2 global token, Sec. 5.1).

The file name makes pytest collect it last, so a run that stops at the first
failure has run every other test before this one.
"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W

pytestmark = pytest.mark.gpu

# same tolerance as the anchor check of the cache build in test_gpu_parity.py
ATOL, RTOL = 1e-4, 1e-4


def _anchor_from_cache_build(model, b, beh):
    cache = txs.KVCache(model, b.beh_off, beh)
    g = cache.read_anchor(0, 2)
    torch.cuda.synchronize()
    out = g.cpu().numpy()
    cache.close()
    return out


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_static_pooling_matches_cache_build_on_two_calls_in_a_row(dtype):
    if dtype == "bf16":
        base = W.with_sizes(W.WORKLOADS["mid_bf16"], n_layers=1)
    else:
        base = W.WORKLOADS["tiny_fp32"]
    weights = W.weights(base)
    weights["w_pool"] = weights["w_pool"] * 32.0    # uneven pooling weights (a power of two: still exact in bf16)
    model = txs.Model(base, weights)
    dt = txs.torch_dtype(base.dtype)
    first = W.with_sizes(base, n_req=6, L=[1, 127, 128, 129, 2000, 5000], M=1, seed=101)
    second = W.with_sizes(base, n_req=4, L=[3, 16, 17, 700], M=1, seed=202)
    results = []
    for wl in (first, second):
        b = W.batch(wl)
        beh = txs.to_device(b.beh, dt)
        got = txs.pool_anchor_static(model, b.beh_off, beh)
        torch.cuda.synchronize()
        got = got.cpu().numpy()
        ref = _anchor_from_cache_build(model, b, beh)
        np.testing.assert_allclose(got, ref, atol=ATOL, rtol=RTOL)
        om = O.Model.from_arrays(weights, wl)
        g64 = np.stack([O.pool_direct(om, b.beh[b.beh_off[r]:b.beh_off[r + 1]]).g for r in range(wl.n_req)])
        np.testing.assert_allclose(got, g64, atol=ATOL, rtol=RTOL)
        results.append(got)
    assert model.device_status() == txs.TXS_OK
    # the first batch again gives the same values as its first call
    b = W.batch(first)
    again = txs.pool_anchor_static(model, b.beh_off, txs.to_device(b.beh, dt)).cpu().numpy()
    np.testing.assert_array_equal(again, results[0])


def test_static_pooling_rejects_calls_beyond_its_scratch():
    base = W.with_sizes(W.WORKLOADS["mid_bf16"], n_layers=1)
    model = txs.Model(base, W.weights(base))
    n_req = 128                                     # 128 * 16 * 514 floats > 1,048,576
    off = np.arange(n_req + 1, dtype=np.int32)
    beh = torch.zeros((n_req, base.d_model), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(txs.TxsError) as e:
        txs.pool_anchor_static(model, off, beh)
    assert e.value.status == txs.TXS_ERR_UNSUPPORTED
    assert "static scratch" in str(e.value)
    with pytest.raises(txs.TxsError) as e:
        txs.pool_anchor_static(model, [0, 1, 1], beh)
    assert e.value.status == txs.TXS_ERR_COLD_START
