"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Small workloads are compared on every candidate; the full-size workloads are
run whole on the GPU (the launch configuration the benchmark times) and
compared on sampled requests, which the oracle computes one by one (requests
are independent, Sec. 4.1.3 factorisation).  Tolerances: max|d| <= 2e-2 and
mean|d| <= 2e-3 on logits and probabilities for bf16 storage, max|d| <= 1e-4
for the fp32 workload.  Integer outputs (lengths, rankings) are bit-exact.
"""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import (assert_scores_close, oracle_scores, rows_of, run_gpu, upload_batch)

pytestmark = pytest.mark.gpu

MODES = [txs.LOCAL_GLOBAL, txs.FULL]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need CUDA")
    txs.lib()


# ---------------------------------------------------------------- whole workloads, every candidate

@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_full_batch_matches_oracle(name, mode):
    wl = W.WORKLOADS[name]
    g = run_gpu(wl, mode)
    lg, pr, _, _ = oracle_scores(wl, mode)
    assert_scores_close(g.logits, lg, wl.dtype, f"{name} logits")
    assert_scores_close(g.probs, pr, wl.dtype, f"{name} probs")


@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_cache_rows_and_anchor_match_oracle(name):
    wl = W.WORKLOADS[name]
    g = run_gpu(wl, txs.LOCAL_GLOBAL)
    reqs = [0, wl.n_req - 1]
    _, _, caches, b = oracle_scores(wl, txs.LOCAL_GLOBAL, requests=reqs)
    tol = dict(atol=3e-2, rtol=1e-2) if wl.dtype == "bf16" else dict(atol=1e-5, rtol=1e-5)
    for j, r in enumerate(reqs):
        L = int(g.batch.L[r])
        for l in range(wl.n_layers):
            for which, ref in ((0, caches[j].K[l]), (1, caches[j].V[l])):
                rows = g.cache.read_rows(l, which, r, 0, L).float().cpu().numpy()
                np.testing.assert_allclose(rows, ref, **tol)
    gref = np.stack([c.pool.g for c in caches])
    got = g.cache.read_anchor(0, 2).cpu().numpy()[reqs]
    np.testing.assert_allclose(got, gref, atol=1e-4, rtol=1e-4)
    for l in range(wl.n_layers):
        np.testing.assert_allclose(g.cache.read_anchor(l, 0).cpu().numpy()[reqs],
                                   np.stack([c.Kg[l] for c in caches]), **tol)
        np.testing.assert_allclose(g.cache.read_anchor(l, 1).cpu().numpy()[reqs],
                                   np.stack([c.Vg[l] for c in caches]), **tol)


# ---------------------------------------------------------------- full-size workloads, sampled requests

def _sample_requests(wl, b, n_extra=1):
    L = b.L
    reqs = {int(np.argmin(L)), int(np.argmax(L))}
    rng = np.random.default_rng(wl.seed)
    while len(reqs) < 2 + n_extra and len(reqs) < wl.n_req:
        reqs.add(int(rng.integers(wl.n_req)))
    return sorted(reqs)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("name", ["mid_bf16", "ragged_bf16"])
def test_full_size_sampled_requests(name, mode):
    wl = W.WORKLOADS[name]
    g = run_gpu(wl, mode)
    reqs = _sample_requests(wl, g.batch)
    lg, pr, _, _ = oracle_scores(wl, mode, requests=reqs)
    assert_scores_close(rows_of(g.batch, reqs, g.logits), lg, wl.dtype, f"{name} logits {reqs}")
    assert_scores_close(rows_of(g.batch, reqs, g.probs), pr, wl.dtype, f"{name} probs {reqs}")
    assert np.isfinite(g.probs).all()
    np.testing.assert_allclose(g.probs.sum(1), 1.0, atol=1e-5)


@pytest.mark.parametrize("name", ["small_bf16", "mid_bf16"])
def test_full_attention_lone_query_tiles(name):
    # FULL mode with enough requests for two query tiles per CTA: slates of
    # 252..259 candidates (+ 2 context rows) leave the last query tile of
    # most requests alone in its CTA, which then splits the request's key
    # tiles over its two softmax groups and merges them; histories of one key
    # tile (no split), two, an odd number and ragged last tiles
    L = [100, 129, 300, 1000, 257, 128, 640, 385] * 3
    M = [252 + (r % 8) for r in range(24)]
    wl = W.with_sizes(W.WORKLOADS[name], n_req=24, n_layers=1, L=L, M=M)
    g = run_gpu(wl, txs.FULL)
    lg, pr, _, _ = oracle_scores(wl, txs.FULL)
    assert_scores_close(g.logits, lg, wl.dtype, f"{name} logits")
    assert_scores_close(g.probs, pr, wl.dtype, f"{name} probs")


@pytest.mark.parametrize("M", [64, 256, 1024, 4096])
def test_sweep_candidate_counts(M):
    wl = W.WORKLOADS["sweep_bf16"]
    b = W.batch(wl, M_override=M)
    g = run_gpu(wl, txs.LOCAL_GLOBAL, b=b)
    reqs = [3]
    lg, pr, _, _ = oracle_scores(wl, txs.LOCAL_GLOBAL, requests=reqs, M_override=M)
    assert_scores_close(rows_of(b, reqs, g.logits), lg, "bf16", f"M={M}")
    assert_scores_close(rows_of(b, reqs, g.probs), pr, "bf16", f"M={M}")


# ---------------------------------------------------------------- incremental append

@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16", "sweep_bf16"])
def test_append_matches_oracle_and_rebuild(name):
    wl = W.WORKLOADS[name]
    b = W.batch(wl)
    g = run_gpu(wl, txs.LOCAL_GLOBAL, b=b, append=True)
    np.testing.assert_array_equal(g.cache.lengths(), b.L + b.dL)
    reqs = [0] if wl.n_req == 1 else [0, wl.n_req - 1]
    lg, pr, _, _ = oracle_scores(wl, txs.LOCAL_GLOBAL, requests=reqs, append=True)
    assert_scores_close(rows_of(b, reqs, g.logits), lg, wl.dtype, "appended logits")
    # rebuild from the concatenated rows: every K/V row bit-identical
    full_off = np.zeros(wl.n_req + 1, np.int32)
    full_off[1:] = np.cumsum(b.L + b.dL)
    rows = np.concatenate([np.concatenate([b.beh[b.beh_off[r]:b.beh_off[r + 1]],
                                           b.app[b.app_off[r]:b.app_off[r + 1]]]) for r in range(wl.n_req)])
    dt = txs.torch_dtype(wl.dtype)
    rebuilt = txs.KVCache(g.model, full_off, txs.to_device(rows, dt), capacity_extra=0)
    for r in reqs:
        n = int(b.L[r] + b.dL[r])
        for l in range(wl.n_layers):
            for which in (0, 1):
                a = g.cache.read_rows(l, which, r, 0, n)
                c = rebuilt.read_rows(l, which, r, 0, n)
                assert torch.equal(a, c), f"request {r} layer {l} {'KV'[which]} rows differ"
    ga = g.cache.read_anchor(0, 2).cpu().numpy()
    gr = rebuilt.read_anchor(0, 2).cpu().numpy()
    np.testing.assert_allclose(ga, gr, atol=1e-5, rtol=1e-4)


def test_capacity_exceeded_leaves_cache_unchanged():
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=2, L=16, M=4)
    b = W.batch(wl)
    g = run_gpu(wl, txs.LOCAL_GLOBAL, b=b)
    big = np.array([0, wl.capacity_extra + 1, wl.capacity_extra + 1], np.int32)
    rows = txs.to_device(np.zeros((int(big[-1]), wl.d_model), np.float32), torch.bfloat16)
    with pytest.raises(txs.TxsError) as e:
        g.cache.append(big, rows)
    assert e.value.status == txs.TXS_ERR_CAPACITY
    np.testing.assert_array_equal(g.cache.lengths(), b.L)


# ---------------------------------------------------------------- ranking (integer output, bit-exact)

@pytest.mark.parametrize("top_k", [0, 5, 300])
def test_rank_is_exact(top_k):
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=5, M=[0, 1, 7, 256, 299], L=20)
    g = run_gpu(wl, txs.LOCAL_GLOBAL)
    off = g.batch.cand_off
    for action in (0, 3):
        idx = txs.rank(off, torch.from_numpy(g.probs).cuda(), wl.n_actions, action, top_k).cpu().numpy()
        want = O.rank(g.probs[:, action], off, top_k)
        for r in range(wl.n_req):
            if top_k == 0:
                got = idx[off[r]:off[r + 1]]
                np.testing.assert_array_equal(got, want[r])
            else:
                got = idx[r * top_k:(r + 1) * top_k]
                m = len(want[r])
                np.testing.assert_array_equal(got[:m], want[r])
                assert (got[m:] == -1).all()


def test_rank_ties_and_nan():
    probs = np.array([[0.2], [0.5], [0.2], [np.nan], [0.9], [0.5], [0.1], [-0.0], [0.0]], np.float32)
    off = np.array([0, 9], np.int32)
    idx = txs.rank(off, torch.from_numpy(probs).cuda(), 1, 0, 0).cpu().numpy()
    np.testing.assert_array_equal(idx, [4, 1, 5, 0, 2, 6, 7, 8, 3])


def test_ranking_agrees_with_oracle_where_scores_are_separated():
    wl = W.WORKLOADS["small_bf16"]
    g = run_gpu(wl, txs.LOCAL_GLOBAL)
    _, pr, _, _ = oracle_scores(wl, txs.LOCAL_GLOBAL, requests=[0])
    idx = txs.rank(g.batch.cand_off, torch.from_numpy(g.probs).cuda(), wl.n_actions, 0, 0).cpu().numpy()
    got = idx[:wl.M] if isinstance(wl.M, int) else idx
    ref = np.asarray(O.rank(pr[:, 0], [0, pr.shape[0]])[0])
    s = pr[ref, 0]
    # compare the order of candidate pairs whose oracle scores differ by more than the tolerance
    pos = np.empty_like(got)
    pos[got] = np.arange(len(got))
    for i in range(len(ref) - 1):
        for j in range(i + 1, len(ref)):
            if s[i] - s[j] > 4e-2:
                assert pos[ref[i]] < pos[ref[j]]


# ---------------------------------------------------------------- edge cases

EDGE = [
    # ragged: empty slate, L below and at L_local, single rows, tails of 128-row tiles
    dict(dtype="bf16", n_req=5, n_layers=2, d_model=128, n_heads=4, d_ff=256, L=[1, 3, 10, 11, 300],
         M=[0, 1, 7, 130, 129]),
    dict(dtype="fp32", n_req=4, n_layers=2, d_model=64, n_heads=2, d_ff=128, L=[1, 9, 10, 70], M=[3, 0, 1, 40]),
    dict(dtype="bf16", n_req=3, n_layers=1, d_model=64, n_heads=1, d_ff=64, L=[5, 1, 40], M=[2, 3, 200],
         n_ctx=0, n_actions=2),
    dict(dtype="bf16", n_req=2, n_layers=1, d_model=512, n_heads=16, d_ff=512, L=[33, 2], M=[1, 5], n_ctx=8,
         n_actions=16, l_local=3),
]


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("i", range(len(EDGE)))
def test_edge_shapes(i, mode):
    wl = W.Workload(f"edge{i}", seed=777 + i, **EDGE[i])
    g = run_gpu(wl, mode)
    lg, pr, _, _ = oracle_scores(wl, mode)
    assert_scores_close(g.logits, lg, wl.dtype, f"edge{i} logits")
    assert_scores_close(g.probs, pr, wl.dtype, f"edge{i} probs")


def test_no_candidates_is_a_no_op():
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=2, L=4, M=0)
    g = run_gpu(wl, txs.LOCAL_GLOBAL)
    assert g.logits.shape == (0, wl.n_actions)


def test_errors_are_reported_before_launch():
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=2, L=8, M=4)
    b = W.batch(wl)
    weights = W.weights(wl)
    m = txs.Model(wl, weights)
    beh, cand, ctx, _ = upload_batch(wl, b)
    with pytest.raises(txs.TxsError) as e:
        txs.KVCache(m, [0, 8, 8], beh)
    assert e.value.status == txs.TXS_ERR_COLD_START
    with pytest.raises(txs.TxsError) as e:
        txs.KVCache(m, [0, 9, 8], beh)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    cache = txs.KVCache(m, b.beh_off, beh)
    other = dict(weights)
    other["W_1.0"] = weights["W_1.0"] * 2
    m2 = txs.Model(wl, other)
    assert m2.hash != m.hash
    assert txs.Model(wl, weights).hash == m.hash
    with pytest.raises(txs.TxsError) as e:
        txs.score(m2, cache, b.cand_off, cand, ctx)
    assert e.value.status == txs.TXS_ERR_STALE_CACHE
    with pytest.raises(txs.TxsError) as e:
        txs.score(m, cache, [0, 4], cand, ctx)   # request count differs from the cache
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(txs.TxsError) as e:
        txs.score(m, cache, b.cand_off, cand, ctx, workspace=ws)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    assert m.device_status() == txs.TXS_OK


def test_window_covering_history_both_modes():
    # LOCAL_GLOBAL with L_local >= L and FULL differ only by the anchor; with a
    # dominant pooling weight the anchor is one row, so the two stay close
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=3, L=12, M=16, l_local=64)
    lg_l = run_gpu(wl, txs.LOCAL_GLOBAL).logits
    lg_f = run_gpu(wl, txs.FULL).logits
    ref_l, _, _, _ = oracle_scores(wl, txs.LOCAL_GLOBAL)
    ref_f, _, _, _ = oracle_scores(wl, txs.FULL)
    assert_scores_close(lg_l, ref_l, "bf16")
    assert_scores_close(lg_f, ref_f, "bf16")


@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_rebuild_append_equals_the_two_calls(name):
    """txs_rebuild_append_kv_cache gives the bytes of txs_rebuild_kv_cache
    followed by txs_append_behavior: cached rows, anchor and scores."""
    wl = W.with_sizes(W.WORKLOADS[name], n_req=3, L=[20, 300, 7], M=[5, 40, 1], dL=[4, 0, 9])
    b = W.batch(wl)
    dt = txs.torch_dtype(wl.dtype)
    model = txs.Model(wl, W.weights(wl), O.LOCAL_GLOBAL)
    beh, app = txs.to_device(b.beh, dt), txs.to_device(b.app, dt)
    cand, ctx = txs.to_device(b.cand, dt), txs.to_device(b.ctx.reshape(-1, wl.d_model), dt)
    c1 = txs.KVCache(model, b.beh_off, beh, capacity_extra=16)
    c2 = txs.KVCache(model, b.beh_off, beh, capacity_extra=16)
    c1.rebuild(b.beh_off, beh)
    c1.append(b.app_off, app)
    c2.rebuild_append(b.beh_off, beh, b.app_off, app)
    torch.cuda.synchronize()
    assert np.array_equal(c1.lengths(), c2.lengths())
    for r in range(wl.n_req):
        n = int(c1.lengths()[r])
        for l in range(wl.n_layers):
            for which in (0, 1):
                assert torch.equal(c1.read_rows(l, which, r, 0, n), c2.read_rows(l, which, r, 0, n))
    for which in (0, 1, 2):
        assert torch.equal(c1.read_anchor(0, which), c2.read_anchor(0, which))
    s1 = txs.score(model, c1, b.cand_off, cand, ctx)
    s2 = txs.score(model, c2, b.cand_off, cand, ctx)
    assert torch.equal(s1[0], s2[0]) and torch.equal(s1[1], s2[1])
    # capacity is checked for the sum, before anything runs
    big = np.array([0, 20, 20, 20], np.int32)
    with pytest.raises(txs.TxsError) as e:
        c2.rebuild_append(b.beh_off, beh, big, txs.to_device(np.zeros((20, wl.d_model), np.float32), dt))
    assert e.value.status == txs.TXS_ERR_CAPACITY
    assert np.array_equal(c2.lengths(), c1.lengths())
