"""Python binding of libqe.so (the C ABI declared in include/qe.h).

Argument marshalling only: torch tensors are passed as raw device pointers and
the current torch CUDA stream as the cudaStream_t; every step of the method runs
in the library's CUDA kernels.  There is no fallback: if libqe.so is missing the
calls raise.  The function names are those of the C ABI.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libqe.so")

QE_OK, QE_ERR_INVALID_ARG, QE_ERR_CUDA, QE_ERR_OOM, QE_ERR_NUMERIC, QE_ERR_TIMEOUT, \
    QE_ERR_UNSUPPORTED = range(7)
QE_F32, QE_BF16 = 0, 1
QE_FEATURE_MAJOR, QE_TOKEN_MAJOR = 0, 1

EXPORTED = ("qe_build_sigma", "qe_quantize_layer", "qe_quantize_layer_outlier",
            "qe_workspace_size", "qe_sync_status", "qe_status_string", "qe_version",
            "qe_build_sigma_static", "qe_timer_create", "qe_timer_read", "qe_timer_reset",
            "qe_timer_destroy", "qe_build_sigma_host", "qe_pack_codes", "qe_unpack_codes",
            "qe_hard_threshold", "qe_hard_threshold_workspace")
QE_KERNEL_PINIT_GEMM, QE_KERNEL_RESIDUAL_GEMM, QE_KERNEL_TRAIL_GEMM, QE_KERNEL_CD_BLOCK, \
    QE_KERNEL_CD_LISTS, QE_KERNEL_COUNT = range(6)


class QEError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: status {status} ({qe_status_string(status)})")
        self.status = status


class QEOpts(ctypes.Structure):
    """Mirror of ``qe_opts``."""
    _fields_ = [("block_width", ctypes.c_int), ("relax_period", ctypes.c_int),
                ("structured_outliers", ctypes.c_int), ("power_iters", ctypes.c_int),
                ("dense_sweeps", ctypes.c_int), ("free_changes", ctypes.c_int), ("group_size", ctypes.c_int),
                ("init_codes", ctypes.c_void_p), ("sweep_codes", ctypes.c_void_p),
                ("wx_norm2", ctypes.c_void_p), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_size_t), ("timer", ctypes.c_void_p),
                ("switch_below", ctypes.c_int64), ("sweep_forms", ctypes.c_void_p),
                ("wait_test", ctypes.c_int), ("tie_eps", ctypes.c_float)]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libqe.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libqe.so not found at {path}: build it with "
                           "paper_2309_01885_gb300.build.build_lib()")
    L = ctypes.CDLL(path)
    vp, i64, i32, st = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_int
    L.qe_build_sigma.argtypes = [vp, i32, i32, i64, i64, i64, vp, i32, vp]
    L.qe_build_sigma.restype = st
    L.qe_quantize_layer.argtypes = [vp, i32, i64, i64, i64, vp, i32, i32, ctypes.POINTER(QEOpts),
                                    vp, vp, vp, vp, vp]
    L.qe_quantize_layer.restype = st
    L.qe_quantize_layer_outlier.argtypes = [vp, i32, i64, i64, i64, vp, i32, i32, i64,
                                            ctypes.POINTER(QEOpts), vp, vp, vp, vp, vp, vp, vp, vp,
                                            vp]
    L.qe_quantize_layer_outlier.restype = st
    L.qe_workspace_size.argtypes = [i64, i64, i32, ctypes.POINTER(QEOpts),
                                    ctypes.POINTER(ctypes.c_size_t)]
    L.qe_workspace_size.restype = st
    L.qe_sync_status.argtypes = [vp]
    L.qe_sync_status.restype = st
    L.qe_status_string.argtypes = [st]
    L.qe_status_string.restype = ctypes.c_char_p
    L.qe_version.argtypes = []
    L.qe_version.restype = ctypes.c_int
    L.qe_build_sigma_static.argtypes = [vp, i32, i32, i64, i64, i64, vp, i32, vp]
    L.qe_build_sigma_static.restype = st
    L.qe_build_sigma_host.argtypes = [vp, i64, i64, i64, vp, i32, vp, ctypes.c_size_t, i64, vp]
    L.qe_build_sigma_host.restype = st
    L.qe_pack_codes.argtypes = [vp, i64, i64, i64, i32, vp, i64, vp]
    L.qe_pack_codes.restype = st
    L.qe_unpack_codes.argtypes = [vp, i64, i64, i64, i32, vp, i64, vp]
    L.qe_unpack_codes.restype = st
    L.qe_hard_threshold_workspace.argtypes = [i64, ctypes.POINTER(ctypes.c_size_t)]
    L.qe_hard_threshold_workspace.restype = st
    L.qe_hard_threshold.argtypes = [vp, i64, i64, vp, vp, vp, vp, ctypes.c_size_t, vp]
    L.qe_hard_threshold.restype = st
    L.qe_timer_create.argtypes = [ctypes.c_uint, i32, ctypes.POINTER(vp)]
    L.qe_timer_create.restype = st
    L.qe_timer_read.argtypes = [vp, i32, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_double)]
    L.qe_timer_read.restype = st
    L.qe_timer_reset.argtypes = [vp]
    L.qe_timer_reset.restype = st
    L.qe_timer_destroy.argtypes = [vp]
    L.qe_timer_destroy.restype = st
    _lib = L
    return L


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return QE_F32
    if t.dtype == torch.bfloat16:
        return QE_BF16
    raise TypeError(f"unsupported dtype {t.dtype}: bf16 or fp32")


def _check(status: int, what: str):
    if status != QE_OK:
        raise QEError(status, what)


def _rowmajor_ld(t: torch.Tensor) -> int:
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a 2-D tensor with unit column stride")
    return t.stride(0)


def qe_status_string(status: int) -> str:
    return load().qe_status_string(status).decode()


def qe_version() -> int:
    return load().qe_version()


def qe_sync_status(stream=None) -> int:
    """Wait for the stream; return the device-latched status (0 = ok)."""
    return load().qe_sync_status(_stream(stream))


def qe_workspace_size(q: int, p: int, outlier: bool = False, group_size: int = 0,
                      block_width: int = 0) -> int:
    out = ctypes.c_size_t(0)
    o = _opts(block_width, group_size=group_size)
    _check(load().qe_workspace_size(q, p, int(outlier), ctypes.byref(o), ctypes.byref(out)), "qe_workspace_size")
    return out.value


def qe_build_sigma(X: torch.Tensor, layout: int = QE_FEATURE_MAJOR, Sigma: torch.Tensor | None = None,
                   accumulate: bool = False, stream=None) -> torch.Tensor:
    """Sigma = X X^T (fp32, p x p) from X (bf16 / fp32, p x n feature-major or n x p token-major)."""
    ld = _rowmajor_ld(X)
    p, n = (X.shape[0], X.shape[1]) if layout == QE_FEATURE_MAJOR else (X.shape[1], X.shape[0])
    if Sigma is None:
        Sigma = torch.empty(p, p, dtype=torch.float32, device=X.device)
    _check(load().qe_build_sigma(_ptr(X), _dtype(X), layout, p, n, ld, _ptr(Sigma), int(accumulate),
                                 _stream(stream)), "qe_build_sigma")
    return Sigma


def sigma_host_staging(p: int, chunk: int, nbuf: int = 2, device="cuda") -> torch.Tensor:
    """A device staging area for qe_build_sigma_host (nbuf >= 2 chunk buffers)."""
    return torch.empty(nbuf * p * chunk * 2, dtype=torch.uint8, device=device)


def qe_build_sigma_host(X: torch.Tensor, Sigma: torch.Tensor, staging: torch.Tensor, chunk: int,
                        accumulate: bool = False, stream=None) -> torch.Tensor:
    """Sigma = X X^T for bf16 X (p x n feature-major) in host memory (pin it for the
    copies to overlap), streamed through `staging` in chunks of `chunk` tokens."""
    if X.device.type != "cpu" or X.dtype != torch.bfloat16:
        raise ValueError("qe_build_sigma_host takes a bf16 tensor in host memory")
    p, n = X.shape
    _check(load().qe_build_sigma_host(X.data_ptr(), p, n, _rowmajor_ld(X), _ptr(Sigma), int(accumulate),
                                      _ptr(staging), staging.numel() * staging.element_size(), int(chunk),
                                      _stream(stream)), "qe_build_sigma_host")
    return Sigma


def qe_build_sigma_static(X: torch.Tensor, layout: int = QE_FEATURE_MAJOR, Sigma: torch.Tensor | None = None,
                          accumulate: bool = False, stream=None) -> torch.Tensor:
    """As qe_build_sigma, but the library call allocates no device memory: staged
    inputs go through the library's fixed scratch array (see include/qe.h).  The
    output tensor, when not given, is still allocated here by torch."""
    ld = _rowmajor_ld(X)
    p, n = (X.shape[0], X.shape[1]) if layout == QE_FEATURE_MAJOR else (X.shape[1], X.shape[0])
    if Sigma is None:
        Sigma = torch.empty(p, p, dtype=torch.float32, device=X.device)
    _check(load().qe_build_sigma_static(_ptr(X), _dtype(X), layout, p, n, ld, _ptr(Sigma), int(accumulate),
                                        _stream(stream)), "qe_build_sigma_static")
    return Sigma


class Timer:
    """CUDA-event timing of selected kernel classes inside the library's calls."""

    def __init__(self, kernels, capacity: int = 4096):
        mask = 0
        for k in kernels:
            mask |= 1 << k
        h = ctypes.c_void_p()
        _check(load().qe_timer_create(mask, capacity, ctypes.byref(h)), "qe_timer_create")
        self.handle = h

    def read(self, kernel: int):
        """(launches, total milliseconds) of the timed launches of `kernel`."""
        n = ctypes.c_int(0)
        ms = ctypes.c_double(0.0)
        _check(load().qe_timer_read(self.handle, kernel, ctypes.byref(n), ctypes.byref(ms)), "qe_timer_read")
        return n.value, ms.value

    def reset(self):
        _check(load().qe_timer_reset(self.handle), "qe_timer_reset")

    def close(self):
        if self.handle:
            load().qe_timer_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _opts(block_width=0, power_iters=0, init_codes=None, sweep_codes=None, wx_norm2=None,
          workspace=None, timer=None, dense_sweeps=0, free_changes=0, relax_period=0,
          group_size=0, switch_below=0) -> QEOpts:
    o = QEOpts()
    o.switch_below = switch_below
    o.group_size = group_size
    o.relax_period = relax_period
    o.timer = None if timer is None else timer.handle.value
    o.block_width = block_width
    o.power_iters = power_iters
    o.dense_sweeps = dense_sweeps
    o.free_changes = free_changes
    o.init_codes = None if init_codes is None else init_codes.data_ptr()
    o.sweep_codes = None if sweep_codes is None else sweep_codes.data_ptr()
    o.wx_norm2 = None if wx_norm2 is None else wx_norm2.data_ptr()
    if workspace is not None:
        o.workspace = workspace.data_ptr()
        o.workspace_bytes = workspace.numel() * workspace.element_size()
    return o


def qe_pack_codes(codes: torch.Tensor, bits: int, stream=None) -> torch.Tensor:
    """q x p uint8 codes -> q x ceil(p bits / 8) bytes, each row a little-endian bit stream."""
    q, p = codes.shape
    out = torch.empty(q, (p * bits + 7) // 8, dtype=torch.uint8, device=codes.device)
    _check(load().qe_pack_codes(_ptr(codes), q, p, _rowmajor_ld(codes), bits, _ptr(out), out.shape[1],
                                _stream(stream)), "qe_pack_codes")
    return out


def qe_unpack_codes(packed: torch.Tensor, p: int, bits: int, stream=None) -> torch.Tensor:
    """The inverse of qe_pack_codes: q x p uint8 codes."""
    q = packed.shape[0]
    codes = torch.empty(q, p, dtype=torch.uint8, device=packed.device)
    _check(load().qe_unpack_codes(_ptr(packed), q, p, _rowmajor_ld(packed), bits, _ptr(codes), p,
                                  _stream(stream)), "qe_unpack_codes")
    return codes


def qe_hard_threshold_workspace(N: int) -> int:
    n = ctypes.c_size_t(0)
    _check(load().qe_hard_threshold_workspace(N, ctypes.byref(n)), "qe_hard_threshold_workspace")
    return n.value


def qe_hard_threshold(T: torch.Tensor, s: int, stream=None) -> tuple:
    """P_s of the IHT step on the flat fp32 tensor T: (indices ascending, values), the s entries
    of largest magnitude (zeros never kept; ties to the smaller index)."""
    if T.dtype != torch.float32 or not T.is_contiguous():
        raise ValueError("expected a contiguous fp32 tensor")
    N = T.numel()
    dev = T.device
    idx = torch.empty(max(s, 1), dtype=torch.int64, device=dev)
    val = torch.empty(max(s, 1), dtype=torch.float32, device=dev)
    nnz = torch.empty(1, dtype=torch.int64, device=dev)
    ws = torch.empty(qe_hard_threshold_workspace(N), dtype=torch.uint8, device=dev)
    _check(load().qe_hard_threshold(_ptr(T), N, s, _ptr(idx), _ptr(val), _ptr(nnz), _ptr(ws),
                                    ws.numel(), _stream(stream)), "qe_hard_threshold")
    k = int(nnz.item())
    return idx[:k], val[:k]


def qe_quantize_layer(W: torch.Tensor, Sigma: torch.Tensor, bits: int, iters: int, *,
                      init_codes: torch.Tensor | None = None, record_sweeps: bool = False,
                      want_norm: bool = False, block_width: int = 0,
                      workspace: torch.Tensor | None = None, timer: Timer | None = None,
                      dense_sweeps: int = 0, free_changes: int = 0, relax_period: int = 0,
                      group_size: int = 0, switch_below: int = 0, record_forms: bool = False,
                      wait_test: int = 0, tie_eps: float = 0.0, stream=None) -> dict:
    """QuantEase on one layer; returns codes (u8 q x p), scales, zeros, obj (fp64 per sweep),
    and optionally sweep_codes (iters x q x p) and wx_norm2.  dense_sweeps: sweeps whose
    cross-block term uses the tensor-core GEMM before the change lists take over (0 = the
    adaptive schedule: dense until a sweep changes fewer than switch_below codes, 0 = automatic);
    free_changes: changes per row below which list sweeps run row by row (0 = default, -1 = never);
    relax_period: the relax heuristic of Sec. 3.2 (sweep t from 1 with t mod R = 0 and t < iters
    keeps beta~ unquantized; 0 = off); group_size: grouped grids (scales / zeros q x groups);
    record_forms: also return sweep_forms (uint8 per sweep: 0 sequential, 1 dense, 2 lists);
    wait_test: the failure-path test hook of qe_opts (a bounded device wait made to give up);
    tie_eps: near-tie refinement threshold in grid steps (0 = default 1e-5, negative = off)."""
    q, p = W.shape
    dev = W.device
    codes = torch.empty(q, p, dtype=torch.uint8, device=dev)
    grid_shape = (q, -(-p // group_size)) if 0 < group_size < p else (q,)
    scales = torch.empty(grid_shape, dtype=torch.float32, device=dev)
    zeros = torch.empty(grid_shape, dtype=torch.float32, device=dev)
    obj = torch.empty(iters, dtype=torch.float64, device=dev)
    sweep = torch.empty(iters, q, p, dtype=torch.uint8, device=dev) if record_sweeps else None
    norm = torch.empty(1, dtype=torch.float64, device=dev) if want_norm else None
    o = _opts(block_width, 0, init_codes, sweep, norm, workspace, timer, dense_sweeps, free_changes,
              relax_period, group_size, switch_below)
    o.wait_test = wait_test
    o.tie_eps = tie_eps
    forms = torch.full((iters,), 255, dtype=torch.uint8, device=dev) if record_forms else None
    o.sweep_forms = None if forms is None else forms.data_ptr()
    _check(load().qe_quantize_layer(_ptr(W), _dtype(W), q, p, _rowmajor_ld(W), _ptr(Sigma), bits, iters,
                                    ctypes.byref(o), _ptr(codes), _ptr(scales), _ptr(zeros), _ptr(obj),
                                    _stream(stream)), "qe_quantize_layer")
    out = dict(codes=codes, scales=scales, zeros=zeros, obj=obj)
    if record_sweeps:
        out["sweep_codes"] = sweep
    if want_norm:
        out["wx_norm2"] = norm
    if record_forms:
        out["sweep_forms"] = forms
    return out


def qe_quantize_layer_outlier(W: torch.Tensor, Sigma: torch.Tensor, bits: int, iters: int,
                              s_budget: int, *, power_iters: int = 0, init_codes=None,
                              record_sweeps: bool = False, want_norm: bool = False,
                              workspace: torch.Tensor | None = None, structured: bool = False,
                              free_changes: int = 0, tie_eps: float = 0.0,
                              timer: Timer | None = None, stream=None) -> dict:
    """Outlier-aware QuantEase; adds H_val, H_idx (sorted linear indices), H_nnz, obj_cd.
    structured: H keeps whole columns (floor(s_budget / q) of them); free_changes: as for
    qe_quantize_layer, for the per-iteration sweeps after the first."""
    q, p = W.shape
    dev = W.device
    codes = torch.empty(q, p, dtype=torch.uint8, device=dev)
    scales = torch.empty(q, dtype=torch.float32, device=dev)
    zeros = torch.empty(q, dtype=torch.float32, device=dev)
    obj = torch.empty(iters, dtype=torch.float64, device=dev)
    obj_cd = torch.empty(iters, dtype=torch.float64, device=dev)
    cap = max(int(s_budget), 1)
    H_val = torch.empty(cap, dtype=torch.float32, device=dev)
    H_idx = torch.empty(cap, dtype=torch.int64, device=dev)
    H_nnz = torch.zeros(1, dtype=torch.int64, device=dev)
    sweep = torch.empty(iters, q, p, dtype=torch.uint8, device=dev) if record_sweeps else None
    norm = torch.empty(1, dtype=torch.float64, device=dev) if want_norm else None
    o = _opts(0, power_iters, init_codes, sweep, norm, workspace, timer, free_changes=free_changes)
    o.structured_outliers = int(structured)
    o.tie_eps = tie_eps
    _check(load().qe_quantize_layer_outlier(
        _ptr(W), _dtype(W), q, p, _rowmajor_ld(W), _ptr(Sigma), bits, iters, int(s_budget),
        ctypes.byref(o), _ptr(codes), _ptr(scales), _ptr(zeros), _ptr(H_val), _ptr(H_idx),
        _ptr(H_nnz), _ptr(obj), _ptr(obj_cd), _stream(stream)), "qe_quantize_layer_outlier")
    out = dict(codes=codes, scales=scales, zeros=zeros, obj=obj, obj_cd=obj_cd, H_val=H_val,
               H_idx=H_idx, H_nnz=H_nnz)
    if record_sweeps:
        out["sweep_codes"] = sweep
    if want_norm:
        out["wx_norm2"] = norm
    return out
