"""GPU parity at the sharp test weights (``workload.sharp_weights``).

With the plain N(0, 0.02) weights the cross-attention softmax is nearly
uniform and a kernel that reads the wrong keys stays inside the bf16
tolerances.  At the sharp weights (power-of-two gains on the attention
projections, the cross-attention output, the head and the pooling vector;
exact in bf16) the CPU test ``test_oracle_sensitivity.py`` shows that a
dropped key tile, half of the keys dropped, a query head reading another
K/V head, a window off by one or a dropped anchor each move the scores by
more than max|d| 2e-2 or mean|d| 2e-3.  The cases below run the kernels of
both key sets of Sec. 4.1.2 (the local window plus the global token) and
Sec. 5.2 (-sparseAttn, every row) at those weights, on the shapes that take
each path of the tensor-core FULL attention: lone query tiles that split
their keys, pairs of query tiles, many query tiles per request (4096
candidates), one long request (the latency shape), grouped K/V heads,
appended rows and streaming events.
"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import (assert_scores_close, oracle_candidate_subset, oracle_scores, rows_of, run_gpu,
                              upload_batch)

pytestmark = pytest.mark.gpu

MODES = [txs.LOCAL_GLOBAL, txs.FULL]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need CUDA")
    txs.lib()


def _check(g_lg, g_pr, lg, pr, dtype, what):
    assert_scores_close(g_lg, lg, dtype, f"{what} logits")
    assert_scores_close(g_pr, pr, dtype, f"{what} probs")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_sharp_full_batch(name, mode):
    wl = W.WORKLOADS[name]
    w = W.sharp_weights(wl)
    g = run_gpu(wl, mode, weights=w, append=True)
    lg, pr, _, _ = oracle_scores(wl, mode, weights=w, append=True)
    _check(g.logits, g.probs, lg, pr, wl.dtype, name)


@pytest.mark.parametrize("name", ["small_bf16", "mid_bf16"])
def test_sharp_lone_query_tiles(name):
    # slates of 252..259 candidates + 2 context rows: the last query tile of
    # most requests is alone in its CTA and splits the request's key tiles
    # over two softmax groups; histories of one, two, an odd number of key
    # tiles and ragged last tiles
    L = [100, 129, 300, 1000, 257, 128, 640, 385] * 3
    M = [252 + (r % 8) for r in range(24)]
    wl = W.with_sizes(W.WORKLOADS[name], n_req=24, n_layers=1, L=L, M=M)
    w = W.sharp_weights(wl)
    g = run_gpu(wl, txs.FULL, weights=w)
    lg, pr, _, _ = oracle_scores(wl, txs.FULL, weights=w)
    _check(g.logits, g.probs, lg, pr, wl.dtype, name)


def _sample_requests(wl, b):
    reqs = {int(np.argmin(b.L)), int(np.argmax(b.L))}
    rng = np.random.default_rng(wl.seed + 1)
    while len(reqs) < 3:
        reqs.add(int(rng.integers(wl.n_req)))
    return sorted(reqs)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("name", ["mid_bf16", "ragged_bf16"])
def test_sharp_full_size_sampled_requests(name, mode):
    # the whole workload on the GPU (the launch configuration the benchmark
    # times), three requests through the oracle: the shortest and longest
    # histories and one more
    wl = W.WORKLOADS[name]
    w = W.sharp_weights(wl)
    g = run_gpu(wl, mode, weights=w, append=True)
    reqs = _sample_requests(wl, g.batch)
    lg, pr, _, _ = oracle_scores(wl, mode, requests=reqs, weights=w, append=True)
    _check(rows_of(g.batch, reqs, g.logits), rows_of(g.batch, reqs, g.probs), lg, pr, wl.dtype, f"{name} {reqs}")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("M", [64, 1024, 4096])
def test_sharp_sweep_candidate_counts(M, mode):
    # 16 requests x 8192 cached rows; at M = 4096 every request has 33 query
    # tiles.  Request 5's candidates are checked on every 7th candidate (all
    # query tiles), plus the last few
    wl = W.WORKLOADS["sweep_bf16"]
    w = W.sharp_weights(wl)
    b = W.batch(wl, M_override=M)
    g = run_gpu(wl, mode, b=b, weights=w)
    r = 5
    idx = np.unique(np.concatenate([np.arange(0, M, 7), np.arange(max(0, M - 3), M)]))
    lg, pr = oracle_candidate_subset(wl, mode, r, idx, w, M_override=M)
    rows = b.cand_off[r] + idx
    _check(g.logits[rows], g.probs[rows], lg, pr, "bf16", f"M={M}")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("L", [1024, 16384])
def test_sharp_single_long_request(L, mode):
    # the latency shape: one request, M = 1000 candidates, L cached rows
    # (one query tile per CTA, key tiles split over two softmax groups)
    base = W.WORKLOADS["ragged_bf16"]
    wl = W.with_sizes(base, n_req=1, L=L, M=1000, dL=0)
    w = W.sharp_weights(wl)
    g = run_gpu(wl, mode, weights=w)
    idx = np.unique(np.concatenate([np.arange(0, 1000, 5), [998, 999]]))
    lg, pr = oracle_candidate_subset(wl, mode, 0, idx, w)
    _check(g.logits[idx], g.probs[idx], lg, pr, "bf16", f"L={L}")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("base,n_kv", [("small_bf16", 1), ("small_bf16", 2), ("mid_bf16", 1), ("mid_bf16", 2)])
def test_sharp_grouped_kv_heads(base, n_kv, mode):
    wl = W.with_sizes(W.WORKLOADS[base], n_req=4, n_layers=2, n_kv_heads=n_kv, L=[3, 11, 300, 700],
                      M=[5, 129, 1, 300], dL=[2, 0, 9, 64])
    w = W.sharp_weights(wl)
    g = run_gpu(wl, mode, weights=w, append=True)
    lg, pr, _, _ = oracle_scores(wl, mode, weights=w, append=True)
    _check(g.logits, g.probs, lg, pr, "bf16", f"{base} n_kv={n_kv}")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("base", ["small_bf16", "mid_bf16"])
def test_sharp_events(base, mode):
    wl = W.with_sizes(W.WORKLOADS[base], n_layers=2)
    w = W.sharp_weights(wl)
    model = txs.Model(wl, w, mode)
    L = 1500
    ev = W.events(wl, L, 8, [40, 130, 1, 7, 300, 90, 2, 129], 43)
    ev.ends[:] = [1, 10, 11, 127, 129, 700, 1499, L]
    dt = txs.torch_dtype(wl.dtype)
    beh = txs.to_device(ev.beh, dt)
    cache = txs.KVCache(model, np.array([0, L], np.int32), beh)
    cand = txs.to_device(ev.cand, dt)
    ctx = txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt)
    lg, pr = txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, cand, ctx)
    torch.cuda.synchronize()
    assert model.device_status() == txs.TXS_OK
    om = O.Model.from_arrays(w, wl)
    rl, rp = O.score_events(om, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, mode)
    _check(lg.cpu().numpy(), pr.cpu().numpy(), rl, rp, "bf16", f"{base} events")


@pytest.mark.parametrize("name", ["small_bf16", "mid_bf16"])
def test_sharp_cache_rows_and_anchor(name):
    # with the sharp pooling vector the anchor is a weighted mix of a few
    # rows, so the pooled g and its projections test the softmax weights
    wl = W.with_sizes(W.WORKLOADS[name], n_req=4, n_layers=2, L=[1, 64, 65, 3000], M=2, dL=[0, 1, 63, 8])
    w = W.sharp_weights(wl)
    g = run_gpu(wl, txs.LOCAL_GLOBAL, weights=w, append=True)
    _, _, caches, b = oracle_scores(wl, txs.LOCAL_GLOBAL, weights=w, append=True)
    np.testing.assert_allclose(g.cache.read_anchor(0, 2).cpu().numpy(), np.stack([c.pool.g for c in caches]),
                               atol=1e-4, rtol=1e-4)
    for l in range(wl.n_layers):
        for which, key in ((0, "Kg"), (1, "Vg")):
            ref = np.stack([getattr(c, key)[l] for c in caches])
            got = g.cache.read_anchor(l, which).cpu().numpy()
            scale = np.sqrt((ref ** 2).mean())
            np.testing.assert_allclose(got / scale, ref / scale, atol=2e-2)


@pytest.mark.parametrize("S", [0, 1, 2, 8])
def test_sharp_fused_serving_attention(S):
    # batches large enough for the serving-stream attention fused into the
    # candidate rows' QKV projection (bf16, d_h = 64, a 256-row x one-head
    # tile per SM): 0, 1, 2 and 8 context rows per request (the fused path
    # takes up to 8), ragged slates incl. a single candidate, every candidate
    # compared; the attention gain makes the serving softmax decide the scores
    wl = W.Workload(f"serve{S}", seed=880 + S, dtype="bf16", n_req=6, n_layers=1, d_model=512, n_heads=8,
                    d_ff=512, L=[40, 3, 12, 90, 1, 25], M=[1100, 900, 1000, 1300, 1, 1000], n_ctx=S)
    w = W.sharp_weights(wl)
    g = run_gpu(wl, txs.LOCAL_GLOBAL, weights=w)
    lg, pr, _, _ = oracle_scores(wl, txs.LOCAL_GLOBAL, weights=w)
    _check(g.logits, g.probs, lg, pr, wl.dtype, f"fused serving S={S}")
