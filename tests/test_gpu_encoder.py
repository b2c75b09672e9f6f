"""Behavior-stream encoder on the GPU (Sec. 4.1.1; App. D incremental
encoding) against the fp64 oracle, through the C ABI.

* Encoded rows Phi_b and every layer's cached K/V rows match the oracle after
  a build and after appends (fp32 1e-4; bf16 max 5e-2, mean 5e-3 on these
  unit-variance rows, bounds derived below), with and without an attention
  window, ragged users and users with no tokens.
* Incremental encoding is exact: building from a prefix and appending the rest
  gives the same bytes as building from the whole stream (the property the
  paper's remark states, here bit for bit).
* At the full encoder workload (64 users x 4096 tokens, d = 512, in the launch
  configuration the benchmark times) sampled users match the oracle.
* The encoded rows feed the decoder's cache build, append and scoring.
* Errors: capacity, stale state, bad type ids, bad arguments.
"""
import numpy as np
import pytest
import torch

from oracle import encoder_oracle as E
from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import assert_scores_close

pytestmark = pytest.mark.gpu


# Encoder rows are unit-variance LN outputs.  With bf16 storage, rounding the
# fp64 result alone is off by up to 1.6e-2 (mean 1.1e-3); the path stores
# seven intermediates per layer in bf16 (q, k, v, attention, H, GELU hidden,
# Y), which over two layers gives about 2.6x that in mean and 2x in max,
# independent of the stream length.  Bounds: max 5e-2, mean 5e-3 (bf16);
# 1e-4 (fp32).  Cached K/V rows are compared after dividing by their rms.
ENC_BF16_MAX, ENC_BF16_MEAN, ENC_FP32_MAX = 5e-2, 5e-3, 1e-4


def _close(gpu, ref, dtype, what=""):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    assert np.isfinite(gpu).all(), what
    if gpu.size == 0:
        return
    err = np.abs(gpu - ref)
    if dtype == "bf16":
        assert err.max() <= ENC_BF16_MAX and err.mean() <= ENC_BF16_MEAN, \
            f"{what}: max {err.max():.3g} mean {err.mean():.3g}"
    else:
        assert err.max() <= ENC_FP32_MAX, f"{what}: max {err.max():.3g}"


def _up(ew, b):
    dt = txs.torch_dtype(ew.dtype)
    return (txs.to_device(b.subj, dt), torch.from_numpy(b.types).to("cuda"),
            txs.to_device(b.subj_app, dt), torch.from_numpy(b.types_app).to("cuda"))


def _ew(base, **kw):
    return W.with_sizes(W.ENC_WORKLOADS[base], **kw)


CASES = [
    ("enc_tiny_fp32", {}),
    ("enc_tiny_fp32", dict(window=7, n_rel=4)),
    ("enc_tiny_fp32", dict(type_dim=0, n_rel=1, n_req=4, L=[0, 33, 1, 70], dL=[5, 0, 40, 1])),
    ("enc_small_bf16", dict(n_req=4, L=[100, 0, 37, 300], dL=[8, 3, 0, 40])),
    ("enc_small_bf16", dict(n_req=3, L=[90, 200, 64], dL=[1, 33, 8], window=50)),
    ("enc_mid_bf16", dict(n_req=2, L=[129, 260], dL=[8, 31])),
]


@pytest.mark.parametrize("base,kw", CASES)
def test_build_and_append_match_oracle(base, kw):
    ew = _ew(base, **kw)
    w = W.enc_weights(ew)
    b = W.enc_batch(ew)
    enc = txs.Encoder(ew, w)
    subj, types, subj_a, types_a = _up(ew, b)
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=ew.capacity_extra)
    phi_new = st.append(b.app_off, subj_a, types_a)
    torch.cuda.synchronize()
    assert enc.device_status() == txs.TXS_OK
    assert np.array_equal(st.lengths(), b.L + b.dL)
    om = E.EncModel.from_arrays(w, ew)
    phi_ref, states = E.encode_batch(om, b.subj, b.types, b.off)
    _close(st.phi.float().cpu().numpy(), phi_ref, ew.dtype, "build Phi_b")
    new_ref, states = E.append_batch(om, states, b.subj_app, b.types_app, b.app_off)
    _close(phi_new.float().cpu().numpy(), new_ref, ew.dtype, "append Phi_b")
    for r in range(ew.n_req):
        n = int(b.L[r] + b.dL[r])
        for l in range(ew.n_layers):
            for which, ref in ((0, states[r].K[l]), (1, states[r].V[l])):
                if n == 0:
                    continue
                rows = st.read_rows(l, which, r, 0, n).float().cpu().numpy()
                rms = float(np.sqrt((ref ** 2).mean()))
                _close(rows / rms, ref / rms, ew.dtype, f"K/V layer {l} user {r}")


@pytest.mark.parametrize("base,kw", [("enc_tiny_fp32", dict(n_req=2, L=[50, 61], dL=[0, 0])),
                                     ("enc_small_bf16", dict(n_req=3, L=[300, 77, 1], dL=[0, 0, 0])),
                                     ("enc_small_bf16", dict(n_req=2, L=[200, 150], dL=[0, 0], window=40))])
@pytest.mark.parametrize("cuts", [[1], [17, 1, 5], [64]])
def test_incremental_is_bit_identical(base, kw, cuts):
    ew = _ew(base, **kw)
    w = W.enc_weights(ew)
    b = W.enc_batch(ew)
    enc = txs.Encoder(ew, w)
    subj, types, _, _ = _up(ew, b)
    full = txs.EncState(enc, b.off, subj, types)
    ref = full.phi.clone()
    # the same stream: a prefix at build, then the rest in len(cuts)+1 appends
    L = b.L.astype(np.int64)
    pre = np.maximum(L - sum(cuts), 0)
    parts = [pre] + [np.minimum(np.maximum(L - pre - sum(cuts[:i]), 0), c) for i, c in enumerate(cuts)]
    parts[-1] = parts[-1] + (L - sum(parts))
    assert (sum(parts) == L).all()
    starts = np.concatenate([[0], np.cumsum(L)[:-1]])
    got = torch.empty_like(ref)
    done = np.zeros_like(L)
    st = None
    for k, part in enumerate(parts):
        rows = np.concatenate([np.arange(starts[r] + done[r], starts[r] + done[r] + part[r]) for r in range(len(L))])
        rows = rows.astype(np.int64)
        off = np.zeros(len(L) + 1, np.int32)
        off[1:] = np.cumsum(part)
        ridx = torch.from_numpy(rows).to("cuda")
        s_sub, t_sub = subj[ridx].contiguous(), types[ridx].contiguous()
        if st is None:
            st = txs.EncState(enc, off, s_sub, t_sub, capacity_extra=int(L.max()))
            out = st.phi
        else:
            out = st.append(off, s_sub, t_sub)
        if rows.size:
            got[ridx] = out
        done += part
    torch.cuda.synchronize()
    assert enc.device_status() == txs.TXS_OK
    assert torch.equal(got, ref)
    for r in range(ew.n_req):
        for l in range(ew.n_layers):
            for which in (0, 1):
                if L[r]:
                    assert torch.equal(st.read_rows(l, which, r, 0, int(L[r])),
                                       full.read_rows(l, which, r, 0, int(L[r])))


def test_full_size_sampled_users():
    """64 users x 4096 earlier tokens, 8 new tokens each, d = 512, 2 layers:
    the launch configuration of the benchmark; users 0 and 63 against the
    oracle, all users' outputs finite."""
    ew = W.ENC_WORKLOADS["enc_mid_bf16"]
    w = W.enc_weights(ew)
    b = W.enc_batch(ew)
    enc = txs.Encoder(ew, w)
    subj, types, subj_a, types_a = _up(ew, b)
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=ew.capacity_extra)
    new = st.append(b.app_off, subj_a, types_a)
    torch.cuda.synchronize()
    assert enc.device_status() == txs.TXS_OK
    phi = st.phi.float().cpu().numpy()
    newh = new.float().cpu().numpy()
    assert np.isfinite(phi).all() and np.isfinite(newh).all()
    om = E.EncModel.from_arrays(w, ew)
    for r in (0, ew.n_req - 1):
        sl = slice(b.off[r], b.off[r + 1])
        ref, state = E.encode(om, b.subj[sl], b.types[sl])
        # the last 512 rows of the build (the oracle's are all computed)
        _close(phi[sl][-512:], ref[-512:], "bf16", f"user {r} build")
        sa = slice(b.app_off[r], b.app_off[r + 1])
        nref, _ = E.encode_append(om, state, b.subj_app[sa], b.types_app[sa])
        _close(newh[sa], nref, "bf16", f"user {r} append")


@pytest.mark.parametrize("mode", [O.LOCAL_GLOBAL, O.FULL])
def test_encoder_feeds_decoder(mode):
    """Phi_b from the encoder builds the decoder's cache; the appended tokens'
    rows extend it; scores match the oracle chain (encoder then decoder)."""
    ew = _ew("enc_small_bf16", n_req=3, L=[40, 300, 9], dL=[4, 1, 20])
    wl = W.with_sizes(W.WORKLOADS["small_bf16"], n_req=3, n_layers=2, L=[40, 300, 9], M=[7, 50, 1], dL=[4, 1, 20])
    ewt, wt = W.enc_weights(ew), W.weights(wl)
    b = W.enc_batch(ew)
    db = W.batch(wl)
    enc = txs.Encoder(ew, ewt)
    model = txs.Model(wl, wt, mode)
    subj, types, subj_a, types_a = _up(ew, b)
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=32)
    cache = txs.KVCache(model, b.off, st.phi, capacity_extra=32)
    new = st.append(b.app_off, subj_a, types_a)
    cache.append(b.app_off, new)
    dt = txs.torch_dtype(wl.dtype)
    lg, pr = txs.score(model, cache, db.cand_off, txs.to_device(db.cand, dt),
                       txs.to_device(db.ctx.reshape(-1, wl.d_model), dt))
    torch.cuda.synchronize()
    om, dm = E.EncModel.from_arrays(ewt, ew), O.Model.from_arrays(wt, wl)
    phi, states = E.encode_batch(om, b.subj, b.types, b.off)
    # the decoder consumes Phi_b in storage precision, as the GPU does
    phi = W.round_bf16(phi.astype(np.float32)).astype(np.float64)
    newr, _ = E.append_batch(om, states, b.subj_app, b.types_app, b.app_off)
    newr = W.round_bf16(newr.astype(np.float32)).astype(np.float64)
    caches = O.append_caches(dm, O.build_caches(dm, phi, b.off), newr, b.app_off)
    rl, rp = O.score_batch(dm, caches, db.ctx, db.cand, db.cand_off, mode)
    assert_scores_close(lg.cpu().numpy(), rl, "bf16", "logits")
    assert_scores_close(pr.cpu().numpy(), rp, "bf16", "probs")


def test_errors():
    ew = _ew("enc_tiny_fp32", n_req=2, L=[5, 6], dL=[1, 1])
    w = W.enc_weights(ew)
    b = W.enc_batch(ew)
    enc = txs.Encoder(ew, w)
    subj, types, subj_a, types_a = _up(ew, b)
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=2)
    # capacity: 3 more tokens for user 0 exceed its 2 spare rows
    off = np.array([0, 3, 3], np.int32)
    s3 = torch.zeros((3, ew.subj_dim), device="cuda")
    t3 = torch.zeros(3, dtype=torch.int32, device="cuda")
    with pytest.raises(txs.TxsError) as e:
        st.append(off, s3, t3)
    assert e.value.status == txs.TXS_ERR_CAPACITY
    assert np.array_equal(st.lengths(), b.L)
    # a state of another encoder is stale
    w2 = dict(w)
    w2["b_o.0"] = w2["b_o.0"] + 1.0
    enc2 = txs.Encoder(ew, w2)
    assert enc2.hash != enc.hash
    with pytest.raises(txs.TxsError) as e:
        st.append(b.app_off, subj_a, types_a, enc=enc2)
    assert e.value.status == txs.TXS_ERR_STALE_CACHE
    # wrong user count
    with pytest.raises(txs.TxsError) as e:
        st.append(np.array([0, 1], np.int32), subj_a[:1], types_a[:1])
    assert e.value.status == txs.TXS_ERR_INVALID_ARG
    # a type id outside the table latches a bounds error (the row's type part is zero)
    bad = types_a.clone()
    bad[0] = ew.n_types
    st.append(b.app_off, subj_a, bad)
    assert enc.device_status() == txs.TXS_ERR_BOUNDS
    assert enc.device_status() == txs.TXS_OK
    # an empty call is a no-op
    z = torch.zeros((0, ew.subj_dim), device="cuda")
    out = st.append(np.zeros(3, np.int32), z, torch.zeros(0, dtype=torch.int32, device="cuda"))
    assert out.shape == (0, ew.d_model)
