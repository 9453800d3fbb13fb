"""qe_build_sigma_static: Sigma = X X^T from a call that allocates nothing.

Some callers cannot let a library allocate device memory during a call: a
process whose device memory is handed out entirely by its own allocator, a
latency-critical loop that must stay off the allocator, or a platform without
stream-ordered allocation.  For them the library stages inputs through a fixed
scratch array that is part of its device image.  This test calls that entry
point through the C ABI twice in a row, on inputs that need staging
(token-major bf16, and an unaligned feature-major view), and checks each result
against qe_build_sigma, the allocating entry point, within the Sigma tolerance
used by the parity tests.  The second input is smaller than the first, so
stale contents of the shared array would show.

The file is named to be collected last: pytest -x stops at the first failure,
so every other test has run before this one.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2309_01885_gb300 import build, inputs, qe

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_lib()
    return qe.load()


def _close(a, b):
    """|a - b| <= 1e-5 sqrt(b_jj b_kk) entrywise, and a exactly symmetric."""
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    assert np.array_equal(a, a.T)
    d = np.sqrt(np.outer(np.abs(np.diag(b)), np.abs(np.diag(b))))
    assert np.all(np.abs(a - b) <= 1e-5 * np.maximum(d, 1e-30))


def _call(lib, X, layout, p, n, ld, out):
    st = lib.qe_build_sigma_static(ctypes.c_void_p(X.data_ptr()), qe.QE_BF16, layout, p, n, ld,
                                   ctypes.c_void_p(out.data_ptr()), 0,
                                   ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == qe.QE_OK, qe.qe_status_string(st)


def test_static_scratch_sigma_matches_allocating_call(lib):
    # call 1: token-major bf16, several staged chunks
    p1, n1 = 320, 20000
    X1 = inputs.calib_inputs(p1, n1, dtype=torch.bfloat16, seed=61, device="cuda", heavy_frac=0.02,
                             heavy_mult=30.0)
    X1t = X1.t().contiguous()
    ref1 = qe.qe_build_sigma(X1t, layout=qe.QE_TOKEN_MAJOR)
    out1 = torch.empty(p1, p1, dtype=torch.float32, device="cuda")
    _call(lib, X1t, qe.QE_TOKEN_MAJOR, p1, n1, p1, out1)
    assert qe.qe_sync_status() == qe.QE_OK
    _close(out1, ref1)

    # call 2, right after: a smaller feature-major view with an odd leading dimension
    p2, n2 = 130, 1001
    base = inputs.calib_inputs(p2, n2 + 3, dtype=torch.bfloat16, seed=62, device="cuda")
    X2 = base[:, :n2]                                  # leading dimension n2 + 3, not a multiple of 8
    ref2 = qe.qe_build_sigma(X2)
    out2 = torch.empty(p2, p2, dtype=torch.float32, device="cuda")
    _call(lib, X2, qe.QE_FEATURE_MAJOR, p2, n2, base.stride(0), out2)
    assert qe.qe_sync_status() == qe.QE_OK
    _close(out2, ref2)


def test_static_scratch_rejects_oversized_rows(lib):
    limit = lib.qe_build_sigma_static  # p beyond QE_STATIC_SCRATCH_BYTES / 128 is refused up front
    fake = ctypes.c_void_p(0x1000)
    st = limit(fake, qe.QE_BF16, qe.QE_TOKEN_MAJOR, 70000, 64, 70000, fake, 0, None)
    assert st == qe.QE_ERR_INVALID_ARG
