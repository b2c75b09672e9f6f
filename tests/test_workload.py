"""The seeded generator: determinism, request-subset consistency, bf16 rounding."""
import numpy as np

from paper_2607_28940_gb300 import workload as W


def test_deterministic_and_subset_consistent():
    wl = W.with_sizes(W.WORKLOADS["ragged_bf16"], n_req=6, L=("uniform", 20, 40), M=5, d_model=64,
                      n_heads=2, d_ff=128, n_layers=1)
    a, b = W.batch(wl), W.batch(wl)
    np.testing.assert_array_equal(a.beh, b.beh)
    np.testing.assert_array_equal(a.cand, b.cand)
    sub = W.batch(wl, requests=[4, 1])
    for j, r in enumerate([4, 1]):
        np.testing.assert_array_equal(sub.beh[sub.beh_off[j]:sub.beh_off[j + 1]],
                                      a.beh[a.beh_off[r]:a.beh_off[r + 1]])
        np.testing.assert_array_equal(sub.cand[sub.cand_off[j]:sub.cand_off[j + 1]],
                                      a.cand[a.cand_off[r]:a.cand_off[r + 1]])
        np.testing.assert_array_equal(sub.ctx[j], a.ctx[r])
    L, M, dL = W.sizes(wl)
    assert ((L >= 20) & (L <= 40)).all() and (M == 5).all()
    assert a.beh_off[-1] == L.sum() and a.beh.shape == (L.sum(), 64)


def test_round_bf16_is_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -9, -2.5, 0.0, np.inf], np.float32)
    r = W.round_bf16(x)
    # 1+2^-8 is halfway between 1 and 1+2^-7: ties to even -> 1; 1+3*2^-8 -> 1+2^-6
    np.testing.assert_array_equal(r, np.array([1.0, 1.0, 1.0 + 2 ** -6, 1.0, -2.5, 0.0, np.inf], np.float32))
    y = np.random.default_rng(0).standard_normal(1000).astype(np.float32)
    ry = W.round_bf16(y)
    assert (ry.view(np.uint32) & 0xFFFF == 0).all()
    assert np.abs(ry - y).max() <= np.abs(y).max() * 2 ** -8
    assert np.isnan(W.round_bf16(np.array([np.nan], np.float32)))[0]


def test_weights_shapes_and_names():
    wl = W.WORKLOADS["small_bf16"]
    w = W.weights(wl)
    assert w["W_qkv.1"].shape == (256, 768) and w["W_1.0"].shape == (256, 1024)
    assert w["W_dec"].shape == (512, 256) and w["Q_dec"].shape == (4, 256)
    assert abs(float(w["ln1_g.0"].mean()) - 1.0) < 0.01
    assert len(w) == 22 * wl.n_layers + 4
