"""qe_build_sigma_static: Sigma = X X^T from a call that allocates nothing.

Some callers cannot let a library allocate device memory during a call: a
process whose device memory is handed out entirely by its own allocator, a
latency-critical loop that must stay off the allocator, or a platform without
stream-ordered allocation.  For them the library stages inputs through a fixed
scratch array that is part of its device image.  These tests call that entry
point through the C ABI several times in a row, on inputs that need staging
(token-major bf16, an unaligned feature-major view, and a width whose chunks
are limited by the array's size, with a ragged last chunk), and check each
result against binary64 Sigma = X X^T from the oracle (Lemma 1), within the
Sigma tolerance of the parity tests, and against qe_build_sigma, the allocating
entry point.  Each input after the first is smaller than the one before, so
stale contents of the shared array would show.

The file is named to be collected last: pytest -x stops at the first failure,
so every other test has run before this one.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2309_01885_gb300 import build, inputs, qe

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_lib()
    return qe.load()


def _close(a, b):
    """|a - b| <= 1e-5 sqrt(b_jj b_kk) entrywise (b binary64 or a torch tensor), and a
    exactly symmetric."""
    a = a.double().cpu().numpy()
    b = b if isinstance(b, np.ndarray) else b.double().cpu().numpy()
    assert np.array_equal(a, a.T)
    d = np.sqrt(np.outer(np.abs(np.diag(b)), np.abs(np.diag(b))))
    assert np.all(np.abs(a - b) <= 1e-5 * np.maximum(d, 1e-30))


def _oracle_sigma(X):
    """binary64 X X^T of the same bf16 values (the oracle's Sigma, Lemma 1)."""
    return oracle.get().sigma(X.double().cpu().numpy())


def _call(lib, X, layout, p, n, ld, out):
    st = lib.qe_build_sigma_static(ctypes.c_void_p(X.data_ptr()), qe.QE_BF16, layout, p, n, ld,
                                   ctypes.c_void_p(out.data_ptr()), 0,
                                   ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == qe.QE_OK, qe.qe_status_string(st)


def test_static_scratch_sigma_matches_oracle(lib):
    # call 1: token-major bf16, 8192-token chunks (the array holds 13107 tokens of p = 320)
    p1, n1 = 320, 20000
    X1 = inputs.calib_inputs(p1, n1, dtype=torch.bfloat16, seed=61, device="cuda", heavy_frac=0.02,
                             heavy_mult=30.0)
    X1t = X1.t().contiguous()
    out1 = torch.empty(p1, p1, dtype=torch.float32, device="cuda")
    _call(lib, X1t, qe.QE_TOKEN_MAJOR, p1, n1, p1, out1)
    assert qe.qe_sync_status() == qe.QE_OK
    _close(out1, _oracle_sigma(X1))
    _close(out1, qe.qe_build_sigma(X1t, layout=qe.QE_TOKEN_MAJOR))

    # call 2: p = 1024, where the array's size limits a chunk to 4096 tokens (the
    # allocating call stages 8192), over two full chunks and a ragged 777-token tail
    p2, n2 = 1024, 2 * 4096 + 777
    X2 = inputs.calib_inputs(p2, n2, dtype=torch.bfloat16, seed=63, device="cuda", heavy_frac=0.02,
                             heavy_mult=30.0)
    X2t = X2.t().contiguous()
    out2 = torch.empty(p2, p2, dtype=torch.float32, device="cuda")
    _call(lib, X2t, qe.QE_TOKEN_MAJOR, p2, n2, p2, out2)
    assert qe.qe_sync_status() == qe.QE_OK
    _close(out2, _oracle_sigma(X2))
    _close(out2, qe.qe_build_sigma(X2t, layout=qe.QE_TOKEN_MAJOR))

    # call 3, right after: a smaller feature-major view with an odd leading dimension
    p3, n3 = 130, 1001
    base = inputs.calib_inputs(p3, n3 + 3, dtype=torch.bfloat16, seed=62, device="cuda")
    X3 = base[:, :n3]                                  # leading dimension n3 + 3, not a multiple of 8
    out3 = torch.empty(p3, p3, dtype=torch.float32, device="cuda")
    _call(lib, X3, qe.QE_FEATURE_MAJOR, p3, n3, base.stride(0), out3)
    assert qe.qe_sync_status() == qe.QE_OK
    _close(out3, _oracle_sigma(X3))
    _close(out3, qe.qe_build_sigma(X3))


def test_static_scratch_width_limit(lib):
    """A staged X needs a chunk of at least 64 tokens in the array: p = 65536 fits
    (8 MiB / (2 * 65536) = 64 tokens), p = 65537 is refused before anything is
    enqueued.  Both calls pass pointers the library never dereferences: the first
    has n = 0 with accumulate = 1 (nothing to do), the second is refused up front."""
    fake = ctypes.c_void_p(0x1000)
    f = lib.qe_build_sigma_static
    assert f(fake, qe.QE_BF16, qe.QE_TOKEN_MAJOR, 65536, 0, 65536, fake, 1, None) == qe.QE_OK
    assert f(fake, qe.QE_BF16, qe.QE_TOKEN_MAJOR, 65537, 64, 65537, fake, 0, None) == qe.QE_ERR_INVALID_ARG
    assert f(fake, qe.QE_BF16, qe.QE_TOKEN_MAJOR, 70000, 64, 70000, fake, 0, None) == qe.QE_ERR_INVALID_ARG
