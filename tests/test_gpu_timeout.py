"""Failure detection on the device without a GPU fault.

Every pipeline of the library waits with a bounded wait; when one runs out
the kernel latches TXS_ERR_DEVICE_TIMEOUT into the model's status word and
returns.  txs_selftest_wait_timeout runs that wait on a barrier nothing
arrives at (about a second); the host reads the code, the word is cleared,
and the context stays usable for the next calls."""
import numpy as np
import pytest
import torch

from paper_2607_28940_gb300 import txs
from paper_2607_28940_gb300 import workload as W
from tests.gpu_common import run_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need CUDA")
    txs.lib()


def test_bounded_wait_runs_out_and_is_reported():
    wl = W.WORKLOADS["tiny_fp32"]
    model = txs.Model(wl, W.weights(wl), txs.LOCAL_GLOBAL)
    assert model.device_status() == txs.TXS_OK
    model.selftest_wait_timeout()
    assert model.device_status() == txs.TXS_ERR_DEVICE_TIMEOUT
    assert model.device_status() == txs.TXS_OK          # read and cleared
    # the context is still usable: a whole build + score runs and reports OK
    g = run_gpu(wl, txs.LOCAL_GLOBAL)
    assert np.isfinite(g.logits).all() and np.isfinite(g.probs).all()
