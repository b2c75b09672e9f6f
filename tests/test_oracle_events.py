"""Pins for the oracle's streaming multi-event scoring (Sec. 4.2, causal
attention and prefix reuse; Sec. 5.1, a global token for each event
timestamp), each against something other than the oracle's own event code:

* every event equals PyTorch's ``TransformerDecoderLayer`` stack fed that
  event's prefix (window of the prefix + anchor pooled over the prefix);
* the cache of a prefix is the prefix of the full stream's cache (the K/V
  projection of a row does not depend on later rows), and a prefix cache
  appended with the rest of the stream is the full cache;
* an event whose prefix is the whole stream scores exactly as a request with
  that history;
* events are independent: their order and grouping do not change any score;
* an event end of 0 (no history) or beyond the stream is rejected.
"""
import numpy as np
import pytest

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import workload as W
from tests.test_oracle_pins import _tiny, torch_score


def _events(wl, L, T, m, seed):
    return W.events(wl, L, T, m, seed)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_each_event_matches_torch_on_its_prefix(mode):
    wl, model = _tiny(n_layers=2)
    ev = _events(wl, 40, 6, 5, 11)
    ev.ends[:3] = [1, 9, 10]                    # window shorter than, equal to, longer than L_local
    ev.ends.sort()
    lg, pr = O.score_events(model, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, mode)
    for t, e in enumerate(ev.ends):
        sl = slice(ev.cand_off[t], ev.cand_off[t + 1])
        rl, rp = torch_score(model, np.asarray(ev.beh[:e], np.float64), np.asarray(ev.ctx[t], np.float64),
                             np.asarray(ev.cand[sl], np.float64), mode)
        np.testing.assert_allclose(lg[sl], rl, atol=1e-11)
        np.testing.assert_allclose(pr[sl], rp, atol=1e-12)


def test_prefix_cache_is_prefix_of_full_cache_and_appends_to_it():
    wl, model = _tiny(n_layers=2)
    phi = np.random.default_rng(3).standard_normal((30, wl.d_model))
    full = O.build_cache(model, phi)
    pre = O.build_cache(model, phi[:17])
    for l in range(model.n_layers):
        np.testing.assert_allclose(pre.K[l], full.K[l][:17], atol=1e-13)
        np.testing.assert_allclose(pre.V[l], full.V[l][:17], atol=1e-13)
    grown = O.append_cache(model, pre, phi[17:])
    for l in range(model.n_layers):
        np.testing.assert_allclose(grown.Kg[l], full.Kg[l], atol=1e-12)
        np.testing.assert_allclose(grown.Vg[l], full.Vg[l], atol=1e-12)


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_event_at_stream_end_equals_request_with_that_history(mode):
    wl, model = _tiny(n_layers=1)
    ev = _events(wl, 25, 3, 4, 5)
    lg, pr = O.score_events(model, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off, mode)
    t = len(ev.ends) - 1                         # its end is the stream length
    sl = slice(ev.cand_off[t], ev.cand_off[t + 1])
    rl, rp = O.score_request(model, O.build_cache(model, ev.beh), ev.ctx[t], ev.cand[sl], mode)
    np.testing.assert_array_equal(lg[sl], rl)
    np.testing.assert_array_equal(pr[sl], rp)


def test_events_are_independent_of_order_and_grouping():
    wl, model = _tiny(n_layers=2)
    ev = _events(wl, 33, 5, [3, 1, 4, 2, 6], 8)
    lg, _ = O.score_events(model, ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off)
    perm = [3, 0, 4, 2, 1]
    sizes = np.diff(ev.cand_off)[perm]
    off = np.concatenate([[0], np.cumsum(sizes)])
    cand = np.concatenate([ev.cand[ev.cand_off[t]:ev.cand_off[t + 1]] for t in perm], 0)
    lg2, _ = O.score_events(model, ev.beh, ev.ends[perm], ev.ctx[perm], cand, off)
    for i, t in enumerate(perm):
        np.testing.assert_allclose(lg2[off[i]:off[i + 1]], lg[ev.cand_off[t]:ev.cand_off[t + 1]], atol=1e-14)
    # one event at a time gives the same scores as all at once
    for t in range(len(ev.ends)):
        one, _ = O.score_events(model, ev.beh, ev.ends[t:t + 1], ev.ctx[t:t + 1],
                                ev.cand[ev.cand_off[t]:ev.cand_off[t + 1]], [0, ev.cand_off[t + 1] - ev.cand_off[t]])
        np.testing.assert_array_equal(one, lg[ev.cand_off[t]:ev.cand_off[t + 1]])


def test_event_end_out_of_range_rejected():
    wl, model = _tiny()
    ev = _events(wl, 10, 2, 2, 1)
    with pytest.raises(ValueError):
        O.score_events(model, ev.beh, [0, 10], ev.ctx, ev.cand, ev.cand_off)
    with pytest.raises(ValueError):
        O.score_events(model, ev.beh, [3, 11], ev.ctx, ev.cand, ev.cand_off)
