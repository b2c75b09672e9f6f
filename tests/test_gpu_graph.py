"""The serving calls can be captured into a CUDA graph: a step of cache
rebuild + append + scoring + ranking (and an encoder append) captured once
and replayed gives the same bytes as the calls issued directly.  Offsets
reach the device as kernel parameters, so replays do not depend on host
memory the library reuses."""
import numpy as np
import pytest
import torch

from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,mode", [("small_bf16", txs.LOCAL_GLOBAL), ("small_bf16", txs.FULL),
                                       ("tiny_fp32", txs.LOCAL_GLOBAL)])
def test_step_replays_from_a_graph(name, mode):
    wl = W.with_sizes(W.WORKLOADS[name], n_req=4, L=[30, 300, 5, 77], M=[9, 1, 40, 0], dL=[3, 0, 8, 1])
    b = W.batch(wl)
    dt = txs.torch_dtype(wl.dtype)
    model = txs.Model(wl, W.weights(wl), mode)
    beh, cand, app = txs.to_device(b.beh, dt), txs.to_device(b.cand, dt), txs.to_device(b.app, dt)
    ctx = txs.to_device(b.ctx.reshape(-1, wl.d_model), dt)
    cache = txs.KVCache(model, b.beh_off, beh, capacity_extra=wl.capacity_extra)
    n = int(b.cand_off[-1])
    ws = torch.empty(txs.workspace_bytes(model, wl.n_req, n), dtype=torch.uint8, device="cuda")
    lg = torch.empty((n, wl.n_actions), dtype=torch.float32, device="cuda")
    pr = torch.empty_like(lg)
    rk = torch.empty(n, dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()

    def step():
        cache.rebuild(b.beh_off, beh)
        cache.append(b.app_off, app)
        txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr)
        txs.rank(b.cand_off, pr, wl.n_actions, 0, 0, out=rk)

    with torch.cuda.stream(s):
        step()
    torch.cuda.synchronize()
    ref = (lg.clone(), pr.clone(), rk.clone())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        step()
    for _ in range(3):
        lg.zero_(); pr.zero_(); rk.zero_()
        cache.rebuild(b.beh_off, beh)     # other work between replays reuses the library's host staging
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(lg, ref[0]) and torch.equal(pr, ref[1]) and torch.equal(rk, ref[2])
    assert model.device_status() == txs.TXS_OK
    # a replay repeats device work only: the host-side lengths are those of
    # the last direct call (the rebuild)
    assert np.array_equal(cache.lengths(), b.L)


def test_encoder_append_replays_from_a_graph():
    ew = W.with_sizes(W.ENC_WORKLOADS["enc_small_bf16"], n_req=3, L=[100, 7, 260], dL=[8, 1, 20])
    b = W.enc_batch(ew)
    enc = txs.Encoder(ew, W.enc_weights(ew))
    dt = txs.torch_dtype(ew.dtype)
    subj, types = txs.to_device(b.subj, dt), torch.from_numpy(b.types).cuda()
    sa, ta = txs.to_device(b.subj_app, dt), torch.from_numpy(b.types_app).cuda()
    na = int(b.app_off[-1])
    ws = torch.empty(enc.workspace_bytes(max(na, int(b.off[-1]))), dtype=torch.uint8, device="cuda")
    out = torch.empty((na, ew.d_model), dtype=dt, device="cuda")
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=64)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        st.append(b.app_off, sa, ta, workspace=ws, phi_out=out)
    torch.cuda.synchronize()
    ref = out.clone()
    # a fresh state at the same point, the append captured and replayed once
    st2 = txs.EncState(enc, b.off, subj, types, capacity_extra=64)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        st2.append(b.app_off, sa, ta, workspace=ws, phi_out=out)
    out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out, ref)
    assert enc.device_status() == txs.TXS_OK


@pytest.mark.parametrize("mode", [txs.LOCAL_GLOBAL, txs.FULL])
def test_score_after_cache_event_matches_sequential(mode):
    """txs_score_candidates_after: the cache refreshed on a side stream while
    the part of scoring that does not read it runs on the main stream gives
    the same bytes as the calls issued one after the other."""
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=4, L=[30, 300, 5, 77], M=[9, 1, 40, 0], dL=[3, 0, 8, 1])
    b = W.batch(wl)
    dt = txs.torch_dtype(wl.dtype)
    model = txs.Model(wl, W.weights(wl), mode)
    beh, cand, app = txs.to_device(b.beh, dt), txs.to_device(b.cand, dt), txs.to_device(b.app, dt)
    ctx = txs.to_device(b.ctx.reshape(-1, wl.d_model), dt)
    cache = txs.KVCache(model, b.beh_off, beh, capacity_extra=wl.capacity_extra)
    n = int(b.cand_off[-1])
    ws = torch.empty(txs.workspace_bytes(model, wl.n_req, n), dtype=torch.uint8, device="cuda")
    lg = torch.empty((n, wl.n_actions), dtype=torch.float32, device="cuda")
    pr = torch.empty_like(lg)
    cache.rebuild(b.beh_off, beh)
    cache.append(b.app_off, app)
    txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr)
    torch.cuda.synchronize()
    ref = (lg.clone(), pr.clone())
    main, side, ready = torch.cuda.current_stream(), torch.cuda.Stream(), torch.cuda.Event()
    for _ in range(3):
        lg.zero_(); pr.zero_()
        side.wait_stream(main)
        with torch.cuda.stream(side):
            cache.rebuild(b.beh_off, beh)
            cache.append(b.app_off, app)
            ready.record(side)
        txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr, cache_ready=ready)
        torch.cuda.synchronize()
        assert torch.equal(lg, ref[0]) and torch.equal(pr, ref[1])
    assert model.device_status() == txs.TXS_OK
