"""Failure detection on the GPU without a fault.

Every device-side wait of the library is bounded (%globaltimer): when it gives
up, the kernel latches QE_ERR_TIMEOUT in the per-device error word and returns,
and qe_sync_status reports and clears it.  The test hook qe_opts.wait_test makes
one such wait run out for real: the first in-block kernel of a call waits for a
copy of its packed Sigma_bar block that is never issued (so nothing is in flight
when it gives up), with a 5 ms limit.  The context stays usable: the next call
runs normally and reproduces a clean run bit for bit.
"""
import numpy as np
import pytest
import torch

from paper_2309_01885_gb300 import inputs, qe

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qe.load()


def test_bounded_wait_gives_up_and_reports_timeout():
    q, p, bits, iters = 96, 320, 3, 3
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=71, device="cuda")
    X = inputs.calib_inputs(p, 2048, dtype=torch.bfloat16, seed=71, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    clean = qe.qe_quantize_layer(W, Sg, bits, iters)
    assert qe.qe_sync_status() == qe.QE_OK
    qe.qe_quantize_layer(W, Sg, bits, iters, wait_test=1)      # returns; the device latches the timeout
    assert qe.qe_sync_status() == qe.QE_ERR_TIMEOUT
    assert qe.qe_sync_status() == qe.QE_OK                      # read and cleared
    again = qe.qe_quantize_layer(W, Sg, bits, iters)
    assert qe.qe_sync_status() == qe.QE_OK
    assert torch.equal(again["codes"], clean["codes"])
    assert np.array_equal(again["obj"].cpu().numpy(), clean["obj"].cpu().numpy())


def test_wait_test_hook_rejects_unknown_values():
    W = torch.zeros(4, 64, dtype=torch.bfloat16, device="cuda")
    S = torch.eye(64, device="cuda")
    with pytest.raises(qe.QEError) as e:
        qe.qe_quantize_layer(W, S, 3, 1, wait_test=2)
    assert e.value.status == qe.QE_ERR_INVALID_ARG
