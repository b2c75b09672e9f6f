"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
and the fp64 oracle on the same seeded inputs, and compare."""
from __future__ import annotations

import os
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

from oracle import txs_oracle as O
from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W

# Tolerances on logits and probabilities (bf16 storage / fp32 end to end).
BF16_MAX, BF16_MEAN = 2e-2, 2e-3
FP32_MAX = 1e-4


def assert_scores_close(gpu: np.ndarray, ref: np.ndarray, dtype: str, what: str = ""):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    assert np.isfinite(gpu).all(), f"{what}: non-finite GPU output"
    err = np.abs(gpu - ref)
    if err.size == 0:
        return
    if os.environ.get("TXS_PRINT_ERRORS"):
        print(f"[scores] {what}: max|d| {err.max():.3e} mean|d| {err.mean():.3e}")
    if dtype == "bf16":
        assert err.max() <= BF16_MAX and err.mean() <= BF16_MEAN, \
            f"{what}: max|d| {err.max():.3g} mean|d| {err.mean():.3g}"
    else:
        assert err.max() <= FP32_MAX, f"{what}: max|d| {err.max():.3g}"


@dataclass
class GpuRun:
    model: txs.Model
    cache: txs.KVCache
    batch: W.Batch
    logits: np.ndarray
    probs: np.ndarray


def upload_batch(wl: W.Workload, b: W.Batch):
    dt = txs.torch_dtype(wl.dtype)
    return (txs.to_device(b.beh, dt), txs.to_device(b.cand, dt),
            txs.to_device(b.ctx.reshape(-1, wl.d_model), dt) if wl.n_ctx else None,
            txs.to_device(b.app, dt) if b.app.shape[0] else None)


def run_gpu(wl: W.Workload, mode: int, b: Optional[W.Batch] = None, append: bool = False,
            weights: Optional[Dict[str, np.ndarray]] = None) -> GpuRun:
    weights = weights if weights is not None else W.weights(wl)
    b = b if b is not None else W.batch(wl)
    model = txs.Model(wl, weights, mode)
    beh, cand, ctx, app = upload_batch(wl, b)
    cache = txs.KVCache(model, b.beh_off, beh, capacity_extra=wl.capacity_extra)
    if append:
        cache.append(b.app_off, app)
    lg, pr = txs.score(model, cache, b.cand_off, cand, ctx)
    torch.cuda.synchronize()
    assert model.device_status() == txs.TXS_OK
    return GpuRun(model, cache, b, lg.cpu().numpy(), pr.cpu().numpy())


def oracle_scores(wl: W.Workload, mode: int, requests: Optional[Sequence[int]] = None, append: bool = False,
                  weights: Optional[Dict[str, np.ndarray]] = None, M_override: Optional[int] = None):
    """Oracle logits/probs of the listed requests (all if None), concatenated,
    plus their caches."""
    weights = weights if weights is not None else W.weights(wl)
    model = O.Model.from_arrays(weights, wl)
    b = W.batch(wl, requests=requests, M_override=M_override)
    caches = O.build_caches(model, b.beh, b.beh_off)
    if append:
        caches = O.append_caches(model, caches, b.app, b.app_off)
    lg, pr = O.score_batch(model, caches, b.ctx, b.cand, b.cand_off, mode)
    return lg, pr, caches, b


def rows_of(b: W.Batch, requests: Sequence[int], arr: np.ndarray) -> np.ndarray:
    """Concatenate the candidate rows of `requests` from a full-batch output."""
    return np.concatenate([arr[b.cand_off[r]:b.cand_off[r + 1]] for r in requests], axis=0)


def score_errors(gpu: np.ndarray, ref: np.ndarray):
    """(max|d|, mean|d|) of two score arrays, for reports."""
    e = np.abs(np.asarray(gpu, np.float64) - np.asarray(ref, np.float64))
    return (float(e.max()), float(e.mean())) if e.size else (0.0, 0.0)


def oracle_candidate_subset(wl: W.Workload, mode: int, r: int, cand_idx: Sequence[int],
                            weights: Dict[str, np.ndarray], M_override: Optional[int] = None, append: bool = False):
    """Oracle logits/probs of some candidates of request r.  Candidates are
    scored independently of each other (a candidate row attends to the context
    rows and itself only, App. B mask), so a subset of the slate gives the same
    values as the whole slate; the oracle pins this invariance."""
    model = O.Model.from_arrays(weights, wl)
    b = W.batch(wl, requests=[r], M_override=M_override)
    cache = O.build_cache(model, b.beh)
    if append:
        cache = O.append_cache(model, cache, b.app)
    cand = b.cand[np.asarray(cand_idx, dtype=np.int64)]
    return O.score_request(model, cache, b.ctx[0], cand, mode)
