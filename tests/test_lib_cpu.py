"""CPU-side checks of the C ABI library: it builds, loads without a GPU, exports
every entry point that include/txs.h declares, and rejects bad arguments on the
host before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2607_28940_gb300 import build
from paper_2607_28940_gb300 import txs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return txs.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "txs.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(txs_[a-z_0-9]+)\s*\(", text)))


def test_exports_every_declared_function(lib):
    names = declared_functions()
    assert len(names) >= 18
    for n in names:
        assert hasattr(lib, n), n
    out = os.popen(f"nm -D --defined-only {txs.LIB_PATH}").read()
    exported = set(re.findall(r" T (txs_\w+)", out))
    assert exported == set(names), (exported ^ set(names))


def test_status_strings_and_version(lib):
    assert txs.status_string(0) == "ok"
    assert "capacity" in txs.status_string(txs.TXS_ERR_CAPACITY)
    assert lib.txs_version().decode().startswith("txs")


def _cfg(**kw):
    base = dict(d_model=256, n_heads=8, d_ff=1024, n_layers=2, n_actions=4, n_ctx=2, l_local=10,
                attn_mode=0, dtype=txs.TXS_BF16, ln_eps=1e-5)
    base.update(kw)
    return txs.txs_config(**base)


@pytest.mark.parametrize("bad", [
    dict(d_model=96), dict(n_heads=3), dict(n_heads=2), dict(d_ff=100), dict(n_actions=0),
    dict(n_actions=17), dict(n_ctx=9), dict(l_local=0), dict(attn_mode=2), dict(dtype=5),
    dict(ln_eps=0.0), dict(n_layers=0), dict(n_kv_heads=3), dict(n_kv_heads=-1),
])
def test_model_create_rejects_bad_config_on_host(lib, bad):
    cfg = _cfg(**bad)
    n = max(cfg.n_layers, 1) * 22 + 4
    ptrs = (ctypes.c_void_p * n)(*([16] * n))
    h = ctypes.c_void_p()
    st = lib.txs_model_create(ctypes.byref(cfg), ptrs, ctypes.byref(h))
    assert st == txs.TXS_ERR_UNSUPPORTED
    assert not h.value


def test_null_arguments_rejected(lib):
    h = ctypes.c_void_p()
    assert lib.txs_model_create(None, None, ctypes.byref(h)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_build_kv_cache(None, 1, None, None, 0, None, ctypes.byref(h)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_score_candidates(None, None, 1, None, None, None, None, 0, None, None, None) == \
        txs.TXS_ERR_INVALID_ARG
    assert lib.txs_device_status(None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_score_events(None, None, 0, None, 1, None, None, None, None, None, 0, None, None, None) == \
        txs.TXS_ERR_INVALID_ARG
    n = ctypes.c_size_t()
    assert lib.txs_events_workspace_size(None, 1, 1, 1, ctypes.byref(n)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_cache_export_size(None, ctypes.byref(n)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_cache_export(None, 0, None, 0, None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_cache_import(None, 0, None, 0, 0, None, ctypes.byref(h)) == txs.TXS_ERR_INVALID_ARG


def test_rank_rejects_bad_arguments_on_host(lib):
    import numpy as np
    off = np.array([0, 3, 5], np.int32)
    p = off.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
    assert lib.txs_rank_candidates(2, p, None, 4, 4, 0, None, None) == txs.TXS_ERR_INVALID_ARG   # action >= k
    assert lib.txs_rank_candidates(2, p, None, 4, 0, -1, None, None) == txs.TXS_ERR_INVALID_ARG  # top_k < 0
    bad = np.array([0, 3, 2], np.int32)
    assert lib.txs_rank_candidates(2, bad.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), None, 4, 0, 0, None,
                                   None) == txs.TXS_ERR_INVALID_ARG
    big = np.array([0, 40000], np.int32)
    assert lib.txs_rank_candidates(1, big.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), None, 4, 0, 0, None,
                                   None) == txs.TXS_ERR_UNSUPPORTED
    assert lib.txs_rank_candidates(0, p, None, 4, 0, 0, None, None) == txs.TXS_OK


def test_gelu_eval_rejects_bad_arguments_on_host(lib):
    assert lib.txs_gelu_eval(None, None, 4, 0, None) == txs.TXS_ERR_INVALID_ARG       # null arrays
    assert lib.txs_gelu_eval(16, 16, -1, 0, None) == txs.TXS_ERR_INVALID_ARG          # negative size
    assert lib.txs_gelu_eval(16, 16, 4, 2, None) == txs.TXS_ERR_INVALID_ARG           # unknown variant
    assert lib.txs_gelu_eval(None, None, 0, 1, None) == txs.TXS_OK                    # nothing to do


def test_profiler_collect_without_launches(lib):
    assert txs.profile_collect() == {}


def _enc_cfg(**kw):
    base = dict(d_model=256, n_heads=8, d_ff=1024, n_layers=2, type_dim=32, n_types=16, n_rel=128, window=0,
                dtype=txs.TXS_BF16, ln_eps=1e-5)
    base.update(kw)
    return txs.txs_enc_config(**base)


@pytest.mark.parametrize("bad", [
    dict(d_model=96), dict(n_heads=3), dict(n_heads=2), dict(d_ff=100), dict(n_layers=0), dict(n_layers=17),
    dict(type_dim=256), dict(type_dim=-1), dict(n_types=0), dict(n_rel=0), dict(n_rel=70000), dict(window=-1),
    dict(ln_eps=0.0),
])
def test_encoder_create_rejects_bad_config_on_host(lib, bad):
    cfg = _enc_cfg(**bad)
    n = max(cfg.n_layers, 1) * 13 + 1
    ptrs = (ctypes.c_void_p * n)(*([16] * n))
    h = ctypes.c_void_p()
    assert lib.txs_encoder_create(ctypes.byref(cfg), ptrs, ctypes.byref(h)) == txs.TXS_ERR_UNSUPPORTED
    assert not h.value
    cfg = _enc_cfg(dtype=7)
    assert lib.txs_encoder_create(ctypes.byref(cfg), ptrs, ctypes.byref(h)) == txs.TXS_ERR_INVALID_ARG


def test_encoder_null_arguments_rejected(lib):
    h = ctypes.c_void_p()
    n = ctypes.c_size_t()
    assert lib.txs_encoder_create(None, None, ctypes.byref(h)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_encoder_workspace_size(None, 1, ctypes.byref(n)) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_encode_build(None, 1, None, None, None, 0, None, 0, None, None, ctypes.byref(h)) == \
        txs.TXS_ERR_INVALID_ARG
    assert lib.txs_encode_append(None, None, 1, None, None, None, None, 0, None, None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_enc_state_lengths(None, None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_enc_state_read_rows(None, 0, 0, 0, 0, 1, None, None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_encoder_device_status(None) == txs.TXS_ERR_INVALID_ARG
    assert lib.txs_enc_state_n_req(None) == 0
    assert lib.txs_encoder_hash(None) == 0
    lib.txs_encoder_destroy(None)
    lib.txs_enc_state_destroy(None)
