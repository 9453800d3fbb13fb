"""The C ABI: libqe.so builds, loads without a GPU, exports every function that
include/qe.h declares, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2309_01885_gb300 import build, qe

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build_lib()
    return qe.load()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "qe.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(qe_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert set(qe.EXPORTED) == set(names)
    for name in names:
        assert hasattr(lib, name), name


def test_status_strings_and_version(lib):
    assert qe.qe_version() >= 10000
    for s in range(7):
        assert qe.qe_status_string(s)
    assert qe.qe_status_string(99) == "unknown status"


def test_opts_struct_matches_header(tmp_path):
    """The ctypes mirror of qe_opts has the size and field offsets the C compiler
    gives the header's struct."""
    import subprocess
    fields = [f[0] for f in qe.QEOpts._fields_]
    src = tmp_path / "opts.c"
    src.write_text('#include "qe.h"\n#include <stdio.h>\n#include <stddef.h>\nint main(void) {\n'
                   '    printf("%zu\\n", sizeof(qe_opts));\n'
                   + "".join(f'    printf("%zu\\n", offsetof(qe_opts, {f}));\n' for f in fields)
                   + "    return 0;\n}\n")
    exe = tmp_path / "opts"
    subprocess.check_call(["gcc", "-std=c11", f"-I{os.path.join(ROOT, 'include')}", "-o", str(exe), str(src)])
    out = [int(x) for x in subprocess.check_output([str(exe)], text=True).split()]
    assert out[0] == ctypes.sizeof(qe.QEOpts)
    assert out[1:] == [getattr(qe.QEOpts, f).offset for f in fields]


def _fake(n=1):
    return ctypes.c_void_p(0x1000 * n)   # never dereferenced: rejected before any launch


def test_invalid_arguments_rejected_synchronously(lib):
    L = lib
    opts = None
    # p = 0
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 0, 4, _fake(2), 4, 1, opts, _fake(3), _fake(4),
                               _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    # bits out of range
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 9, 1, opts, _fake(3), _fake(4),
                               _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    # short leading dimension
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 8, 4, _fake(2), 3, 1, opts, _fake(3), _fake(4),
                               _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    # null output
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, opts, None, _fake(4),
                               _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    # iters = 0
    assert L.qe_quantize_layer(_fake(), qe.QE_BF16, 4, 4, 4, _fake(2), 3, 0, opts, _fake(3), _fake(4),
                               _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    # unsupported / invalid options
    o = qe.QEOpts()
    o.relax_period = -1
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    o = qe.QEOpts()
    o.relax_period = 3            # the outlier variant has no relax heuristic
    assert L.qe_quantize_layer_outlier(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, 4, ctypes.byref(o),
                                       _fake(3), _fake(4), _fake(5), _fake(7), _fake(8), _fake(9), _fake(6),
                                       None, None) == qe.QE_ERR_UNSUPPORTED
    o = qe.QEOpts()
    o.structured_outliers = 1     # only the outlier variant takes it
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_UNSUPPORTED
    o.structured_outliers = 2
    assert L.qe_quantize_layer_outlier(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, 4, ctypes.byref(o),
                                       _fake(3), _fake(4), _fake(5), _fake(7), _fake(8), _fake(9), _fake(6),
                                       None, None) == qe.QE_ERR_UNSUPPORTED
    o = qe.QEOpts()
    o.dense_sweeps = -1
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    o = qe.QEOpts()
    o.free_changes = -2
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    o = qe.QEOpts()
    o.group_size = 100            # not a multiple of the block width (256)
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_INVALID_ARG
    o.group_size = 256
    o.relax_period = 3            # groups and the relax heuristic do not combine
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_UNSUPPORTED
    o.relax_period = 0            # nor groups and the outlier variant
    assert L.qe_quantize_layer_outlier(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, 4, ctypes.byref(o),
                                       _fake(3), _fake(4), _fake(5), _fake(7), _fake(8), _fake(9), _fake(6),
                                       None, None) == qe.QE_ERR_UNSUPPORTED
    o = qe.QEOpts()
    o.block_width = 48
    assert L.qe_quantize_layer(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, ctypes.byref(o), _fake(3),
                               _fake(4), _fake(5), _fake(6), None) == qe.QE_ERR_UNSUPPORTED
    # outlier budget larger than the layer / missing outputs
    assert L.qe_quantize_layer_outlier(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, 17, None, _fake(3),
                                       _fake(4), _fake(5), _fake(7), _fake(8), _fake(9), _fake(6),
                                       None, None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_quantize_layer_outlier(_fake(), qe.QE_F32, 4, 4, 4, _fake(2), 3, 1, 2, None, _fake(3),
                                       _fake(4), _fake(5), None, None, _fake(9), _fake(6),
                                       None, None) == qe.QE_ERR_INVALID_ARG
    # Sigma: bad sizes / layouts
    assert L.qe_build_sigma(_fake(), qe.QE_BF16, qe.QE_FEATURE_MAJOR, 0, 10, 10, _fake(2), 0,
                            None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma(_fake(), qe.QE_BF16, qe.QE_FEATURE_MAJOR, 8, 10, 9, _fake(2), 0,
                            None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma(_fake(), qe.QE_BF16, qe.QE_TOKEN_MAJOR, 8, 10, 7, _fake(2), 0,
                            None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma(_fake(), 7, qe.QE_TOKEN_MAJOR, 8, 10, 8, _fake(2), 0,
                            None) == qe.QE_ERR_INVALID_ARG


def test_sigma_host_rejects_bad_arguments(lib):
    L = lib
    # chunk not a multiple of 64, staging too small, misaligned staging, NULL X, ldx < n
    assert L.qe_build_sigma_host(_fake(), 8, 100, 100, _fake(2), 0, _fake(3), 1 << 20, 100,
                                 None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma_host(_fake(), 8, 100, 100, _fake(2), 0, _fake(3), 2 * 8 * 64 * 2 - 2, 64,
                                 None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma_host(_fake(), 8, 100, 100, _fake(2), 0, ctypes.c_void_p(0x1008), 1 << 20, 64,
                                 None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma_host(None, 8, 100, 100, _fake(2), 0, _fake(3), 1 << 20, 64,
                                 None) == qe.QE_ERR_INVALID_ARG
    assert L.qe_build_sigma_host(_fake(), 8, 100, 99, _fake(2), 0, _fake(3), 1 << 20, 64,
                                 None) == qe.QE_ERR_INVALID_ARG


def test_pack_codes_rejects_bad_arguments(lib):
    L = lib
    for fn in (L.qe_pack_codes, L.qe_unpack_codes):
        # bits outside 1 .. 8, a stream row shorter than ceil(p bits / 8), ldc < p, NULL, p < 1
        assert fn(_fake(), 4, 10, 10, 0, _fake(2), 10, None) == qe.QE_ERR_INVALID_ARG
        assert fn(_fake(), 4, 10, 10, 9, _fake(2), 10, None) == qe.QE_ERR_INVALID_ARG
        assert fn(_fake(), 4, 10, 10, 3, _fake(2), 3, None) == qe.QE_ERR_INVALID_ARG
        assert fn(_fake(), 4, 10, 9, 3, _fake(2), 4, None) == qe.QE_ERR_INVALID_ARG
        assert fn(None, 4, 10, 10, 3, _fake(2), 4, None) == qe.QE_ERR_INVALID_ARG
        assert fn(_fake(), 4, 0, 10, 3, _fake(2), 4, None) == qe.QE_ERR_INVALID_ARG


def test_hard_threshold_rejects_bad_arguments(lib):
    L = lib
    ws = qe.qe_hard_threshold_workspace(1000)
    assert ws >= 3 * 2048 * 4    # the three digit histograms at least
    ok = dict(T=_fake(), N=1000, s=10, idx=_fake(2), val=_fake(3), nnz=_fake(4), w=ctypes.c_void_p(0x100000), wb=ws)

    def call(**kw):
        a = {**ok, **kw}
        return L.qe_hard_threshold(a["T"], a["N"], a["s"], a["idx"], a["val"], a["nnz"], a["w"], a["wb"], None)
    # NULL T / nnz / workspace, N < 1, s outside 0 .. N, NULL outputs with s > 0,
    # a short or misaligned workspace
    for bad in (dict(T=None), dict(nnz=None), dict(w=None), dict(N=0), dict(s=-1), dict(s=1001),
                dict(idx=None), dict(val=None), dict(wb=ws - 1), dict(w=ctypes.c_void_p(0x100010)),
                dict(N=1 << 32, s=0)):
        assert call(**bad) == qe.QE_ERR_INVALID_ARG, bad
    n = ctypes.c_size_t(0)
    assert L.qe_hard_threshold_workspace(0, ctypes.byref(n)) == qe.QE_ERR_INVALID_ARG
    assert L.qe_hard_threshold_workspace(10, None) == qe.QE_ERR_INVALID_ARG
    assert qe.qe_hard_threshold_workspace(1 << 24) > qe.qe_hard_threshold_workspace(1 << 12)


def test_workspace_size_grows_with_shape(lib):
    a = qe.qe_workspace_size(256, 256)
    b = qe.qe_workspace_size(512, 1024)
    c = qe.qe_workspace_size(256, 256, outlier=True)
    d = qe.qe_workspace_size(512, 1024, outlier=True)
    assert 0 < a < b and 0 < c < d
    # the plain layer holds at least Sigma_bar as 3 bf16 planes and in fp32, P and R
    assert b >= 1024 * 1024 * (3 * 2 + 4) + 2 * 512 * 1024 * 4
