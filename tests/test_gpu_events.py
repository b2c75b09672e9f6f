"""Streaming multi-event scoring on the GPU (txs_score_events) against the
fp64 oracle (Sec. 4.2 prefix reuse; Sec. 5.1 a global token per event
timestamp): event t of a user is scored against the first ends[t] rows of the
user's stream, reusing the cached K/V rows and pooling a per-event anchor.

The user is request 1 of a three-request cache, so the cache rows of the user
do not start at row 0; event ends cover a window shorter than, equal to and
longer than L_local, single-row prefixes and the whole stream."""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import assert_scores_close

pytestmark = pytest.mark.gpu


def _setup(wl, mode, L, T, m, seed, ends=None):
    weights = W.weights(wl)
    model = txs.Model(wl, weights, mode)
    ev = W.events(wl, L, T, m, seed)
    if ends is not None:
        ev.ends[:] = np.sort(np.asarray(ends, dtype=np.int32))
    dt = txs.torch_dtype(wl.dtype)
    rng = np.random.default_rng(seed + 1)
    other = [W.round_bf16(rng.standard_normal((n, wl.d_model)).astype(np.float32)) if wl.dtype == "bf16"
             else rng.standard_normal((n, wl.d_model)).astype(np.float32) for n in (37, 11)]
    rows = np.concatenate([other[0], ev.beh, other[1]], 0)
    off = np.array([0, 37, 37 + L, 37 + L + 11], dtype=np.int32)
    cache = txs.KVCache(model, off, txs.to_device(rows, dt), capacity_extra=8)
    beh = txs.to_device(ev.beh, dt)
    cand = txs.to_device(ev.cand, dt)
    ctx = txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt) if wl.n_ctx else None
    return weights, model, ev, cache, beh, cand, ctx


def _oracle(wl, weights, ev, mode, events=None):
    model = O.Model.from_arrays(weights, wl)
    idx = range(len(ev.ends)) if events is None else events
    lg, pr = [], []
    for t in idx:
        sl = slice(ev.cand_off[t], ev.cand_off[t + 1])
        a, b = O.score_events(model, ev.beh, ev.ends[t:t + 1], ev.ctx[t:t + 1], ev.cand[sl],
                              [0, ev.cand_off[t + 1] - ev.cand_off[t]], mode)
        lg.append(a)
        pr.append(b)
    return np.concatenate(lg, 0), np.concatenate(pr, 0)


def _rows(ev, events):
    return np.concatenate([np.arange(ev.cand_off[t], ev.cand_off[t + 1]) for t in events])


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_events_tiny_fp32(mode):
    wl = W.WORKLOADS["tiny_fp32"]
    weights, model, ev, cache, beh, cand, ctx = _setup(wl, mode, 64, 7, 5, 31, ends=[1, 2, 9, 10, 11, 40, 64])
    lg, pr = txs.score_events(model, cache, 1, beh, ev.ends, ev.cand_off, cand, ctx)
    torch.cuda.synchronize()
    assert model.device_status() == txs.TXS_OK
    rl, rp = _oracle(wl, weights, ev, mode)
    assert_scores_close(lg.cpu().numpy(), rl, "fp32", "logits")
    assert_scores_close(pr.cpu().numpy(), rp, "fp32", "probs")


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("base", ["small_bf16", "mid_bf16"])
def test_events_bf16(mode, base):
    wl = W.with_sizes(W.WORKLOADS[base], n_layers=2)
    L = 1500
    weights, model, ev, cache, beh, cand, ctx = _setup(wl, mode, L, 12, [40, 130, 1, 7, 64, 90, 2, 128, 129, 33, 5, 17],
                                                       41, ends=[1, 3, 10, 11, 100, 127, 128, 129, 700, 1024, 1499, L])
    lg, pr = txs.score_events(model, cache, 1, beh, ev.ends, ev.cand_off, cand, ctx)
    torch.cuda.synchronize()
    assert model.device_status() == txs.TXS_OK
    events = [0, 1, 3, 6, 7, 10, 11]
    rl, rp = _oracle(wl, weights, ev, mode, events)
    rows = _rows(ev, events)
    assert_scores_close(lg.cpu().numpy()[rows], rl, "bf16", "logits")
    assert_scores_close(pr.cpu().numpy()[rows], rp, "bf16", "probs")


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_event_at_stream_end_matches_request_scoring(mode):
    # the last event sees the whole stream: the same key set as scoring the
    # user's request of the cache; FULL has no anchor, so the same kernels see
    # identical inputs and the scores are bit-identical
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_layers=2)
    L = 300
    weights, model, ev, cache, beh, cand, ctx = _setup(wl, mode, L, 3, 50, 51, ends=[20, 150, L])
    lg, _ = txs.score_events(model, cache, 1, beh, ev.ends, ev.cand_off, cand, ctx)
    sl = slice(int(ev.cand_off[2]), int(ev.cand_off[3]))
    # score the same slate through txs_score_candidates: the user is request 1,
    # the other two requests get an empty slate
    cand_off = np.array([0, 0, 50, 50], dtype=np.int32)
    dt = txs.torch_dtype(wl.dtype)
    ctx3 = torch.zeros((3 * wl.n_ctx, wl.d_model), dtype=dt, device="cuda")
    ctx3[wl.n_ctx:2 * wl.n_ctx] = ctx[2 * wl.n_ctx:3 * wl.n_ctx]
    rl, _ = txs.score(model, cache, cand_off, cand[sl].contiguous(), ctx3)
    torch.cuda.synchronize()
    a, b = lg.cpu().numpy()[sl], rl.cpu().numpy()
    if mode == O.FULL:
        np.testing.assert_array_equal(a, b)
    else:
        np.testing.assert_allclose(a, b, atol=2e-3)


def test_event_errors():
    wl = W.WORKLOADS["tiny_fp32"]
    weights, model, ev, cache, beh, cand, ctx = _setup(wl, O.LOCAL_GLOBAL, 64, 3, 2, 61, ends=[5, 6, 64])
    with pytest.raises(txs.TxsError) as e:
        txs.score_events(model, cache, 1, beh, [0, 6, 64], ev.cand_off, cand, ctx)
    assert e.value.status == txs.TXS_ERR_COLD_START
    with pytest.raises(txs.TxsError) as e:
        txs.score_events(model, cache, 1, beh, [5, 6, 65], ev.cand_off, cand, ctx)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    with pytest.raises(txs.TxsError) as e:
        txs.score_events(model, cache, 3, beh, ev.ends, ev.cand_off, cand, ctx)
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    big = np.zeros(4098, dtype=np.int32)
    with pytest.raises(txs.TxsError) as e:
        txs.score_events(model, cache, 1, beh, np.ones(4097, np.int32), big, cand, ctx)
    assert e.value.status == txs.TXS_ERR_UNSUPPORTED
    assert model.device_status() == txs.TXS_OK


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_benchmark_configuration_sampled_events(mode):
    """The benchmark's streaming configuration: one 8192-row stream of the
    mid_bf16 model, 64 events at sorted prefix ends with 256 candidates each,
    scored in one call; the first, a middle and the last event against the
    oracle."""
    wl = W.with_sizes(W.WORKLOADS["mid_bf16"], n_req=1, L=8192, M=1, dL=0)
    weights = W.weights(wl)
    model = txs.Model(wl, weights, mode)
    ev = W.events(wl, 8192, 64, 256, 20267)
    dt = txs.torch_dtype(wl.dtype)
    beh = txs.to_device(ev.beh, dt)
    cache = txs.KVCache(model, np.array([0, 8192], np.int32), beh)
    lg, pr = txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, txs.to_device(ev.cand, dt),
                              txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt))
    torch.cuda.synchronize()
    assert model.device_status() == txs.TXS_OK
    lg, pr = lg.cpu().numpy(), pr.cpu().numpy()
    assert np.isfinite(lg).all()
    om = O.Model.from_arrays(weights, wl)
    for t in (0, 31, 63):
        sl = slice(ev.cand_off[t], ev.cand_off[t + 1])
        rl, rp = O.score_events(om, ev.beh, ev.ends[t:t + 1], ev.ctx[t:t + 1], ev.cand[sl],
                                np.array([0, sl.stop - sl.start]), mode)
        assert_scores_close(lg[sl], rl, "bf16", f"event {t} logits")
        assert_scores_close(pr[sl], rp, "bf16", f"event {t} probs")
