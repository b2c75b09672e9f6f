"""Accuracy of the FFN epilogues' GELU (exact erf form, 0.5 x (1 + erf(x / sqrt 2)),
the activation read for the FFN of Sec. 4.1.2).  The bf16 tensor-core
epilogues evaluate erf with the rational approximation 7.1.26 of Abramowitz &
Stegun (absolute error <= 1.5e-7); the fp32 path calls erff.  Both are
checked against float64 on the CPU, and against each other."""
import math

import numpy as np
import pytest
import torch

from paper_2607_28940_gb300 import txs

pytestmark = pytest.mark.gpu


def _exact(x: np.ndarray) -> np.ndarray:
    erf = np.vectorize(math.erf)
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def test_epilogue_gelu_matches_exact_erf_gelu():
    rng = np.random.default_rng(7)
    half = np.concatenate([np.linspace(0.0, 12.0, 100001), np.abs(rng.standard_normal(100000)) * 3.0,
                           np.array([1e-30, 1e-8, 40.0])]).astype(np.float32)
    x = np.concatenate([half, -half])                       # exact negatives
    ref = _exact(x.astype(np.float64))
    xd = torch.from_numpy(x).cuda()
    fast = txs.gelu_eval(xd, 0).cpu().numpy().astype(np.float64)
    libm = txs.gelu_eval(xd, 1).cpu().numpy().astype(np.float64)
    assert np.isfinite(fast).all() and np.isfinite(libm).all()
    # the approximation's 1.5e-7 on erf plus its fp32 evaluation (worst near
    # erf(z) ~ 0.05, where 1 - poly * exp(-z^2) cancels: ~5e-7; 8e-7 allowed),
    # scaled by 0.5 |x|, plus the rounding of the product
    bound = 0.5 * np.abs(x) * 8e-7 + 2.0 * np.finfo(np.float32).eps * np.abs(ref) + 1e-30
    assert (np.abs(fast - ref) <= bound).all(), float(np.max(np.abs(fast - ref) - bound))
    # both evaluations round to the same bf16 value almost everywhere the value
    # is not tiny (where 1 + erf cancels in fp32 for both)
    bf = lambda a: torch.from_numpy(a.astype(np.float32)).to(torch.bfloat16).float().numpy()
    big = np.abs(ref) >= 1e-3
    agree = (bf(fast)[big] == bf(libm)[big]).mean()
    assert agree > 0.999, agree
    # odd part: gelu(x) - gelu(-x) = x
    n = half.size
    np.testing.assert_allclose(fast[:n] - fast[n:], half.astype(np.float64), atol=4e-6, rtol=0)
