"""The candidate-to-query MLP Phi_candidate on the GPU (Sec. 4.1.2): the
decoder sees GELU(x W_c1 + b_c1) W_c2 + b_c2 for each candidate token x, the
head f_dec(z, x) the raw x.  Scores against the fp64 oracle in both key-set
modes, fp32 and bf16, with and without grouped K/V heads, and for streaming
events."""
import numpy as np
import pytest
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import assert_scores_close, oracle_scores, run_gpu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
@pytest.mark.parametrize("base,hidden,n_kv", [("tiny_fp32", 128, 0), ("small_bf16", 256, 0),
                                              ("small_bf16", 1024, 2), ("mid_bf16", 512, 0)])
def test_candidate_mlp_scores_match_oracle(mode, base, hidden, n_kv):
    wl = W.with_sizes(W.WORKLOADS[base], n_req=3, L=[5, 130, 600], M=[1, 64, 257], dL=0,
                      n_layers=min(2, W.WORKLOADS[base].n_layers), cand_mlp=hidden, n_kv_heads=n_kv)
    g = run_gpu(wl, mode)
    lg, pr, _, _ = oracle_scores(wl, mode)
    assert_scores_close(g.logits, lg, wl.dtype, "logits")
    assert_scores_close(g.probs, pr, wl.dtype, "probs")


def test_candidate_mlp_events():
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_layers=2, cand_mlp=256)
    weights = W.weights(wl)
    model = txs.Model(wl, weights, O.LOCAL_GLOBAL)
    ev = W.events(wl, 200, 3, [30, 2, 65], 81)
    dt = txs.torch_dtype(wl.dtype)
    beh = txs.to_device(ev.beh, dt)
    cache = txs.KVCache(model, np.array([0, 200], np.int32), beh)
    lg, _ = txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, txs.to_device(ev.cand, dt),
                             txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt))
    rl, _ = O.score_events(O.Model.from_arrays(weights, wl), ev.beh, ev.ends, ev.ctx, ev.cand, ev.cand_off)
    assert_scores_close(lg.cpu().numpy(), rl, "bf16", "event logits")
    assert model.device_status() == txs.TXS_OK
