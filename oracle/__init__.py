"""QuantEase fp64 CPU oracle (Behdin et al., arXiv 2309.01885).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` import this package.  It shares no code with the
CUDA library (``paper_2309_01885_gb300``) and never imports it.

The arithmetic lives in ``qe_oracle.c`` (plain C, binary64, OpenMP over the
independent rows of Sec. 3.2); this module compiles it with gcc and marshals
numpy arrays through ctypes.  Parity pins: ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(_HERE, "qe_oracle.c")
LIB = os.path.join(_HERE, "_build", "libqe_oracle.so")
CFLAGS = ["-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared", "-std=c11"]


def build(src: str = SRC, out: str = LIB, force: bool = False) -> str:
    """Compile the oracle shared library with gcc; returns its path."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, src, "-lm"])
    os.replace(tmp, out)
    return out


_u8p = ctypes.POINTER(ctypes.c_uint8)
_f32p = ctypes.POINTER(ctypes.c_float)
_f64p = ctypes.POINTER(ctypes.c_double)
_i64p = ctypes.POINTER(ctypes.c_int64)
_i64 = ctypes.c_int64
_int = ctypes.c_int


def _ptr(a, typ):
    if a is None:
        return None
    return a.ctypes.data_as(typ)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


class Oracle:
    """ctypes front end over one build of ``qe_oracle.c``."""

    def __init__(self, path: str | None = None):
        self.path = path or build()
        lib = ctypes.CDLL(self.path)
        lib.qo_grid.argtypes = [_f64p, _i64, _i64, _int, _u8p, _f32p, _f32p]
        lib.qo_grid.restype = None
        lib.qo_grid_groups.argtypes = [_f64p, _i64, _i64, _i64, _int, _u8p, _f32p, _f32p]
        lib.qo_grid_groups.restype = None
        lib.qo_rtn_groups.argtypes = [_f64p, _i64, _i64, _i64, _f32p, _f32p, _int, _u8p]
        lib.qo_rtn_groups.restype = None
        lib.qo_objective_rows_groups.argtypes = [_f64p, _f64p, _u8p, _f32p, _f32p, _i64, _i64, _i64, _f64p,
                                                 _f64p]
        lib.qo_objective_rows_groups.restype = None
        lib.qo_quantease_alg1_groups.argtypes = [_f64p, _i64, _i64, _f64p, _i64, _f32p, _f32p, _int, _int,
                                                 _u8p, _u8p, _u8p, _f64p, _u8p, _f64p, _int]
        lib.qo_quantease_alg1_groups.restype = _int
        lib.qo_rtn.argtypes = [_f64p, _i64, _i64, _f32p, _f32p, _int, _u8p]
        lib.qo_rtn.restype = None
        lib.qo_sigma.argtypes = [_f64p, _i64, _i64, _f64p]
        lib.qo_sigma.restype = None
        lib.qo_objective_rows.argtypes = [_f64p, _f64p, _u8p, _f32p, _f32p, _i64, _i64, _f64p, _f64p]
        lib.qo_objective_rows.restype = None
        lib.qo_quantease_alg1.argtypes = [_f64p, _i64, _i64, _f64p, _f32p, _f32p, _int, _int,
                                          _u8p, _u8p, _u8p, _f64p, _u8p, _f64p, _int]
        lib.qo_quantease_alg1.restype = _int
        lib.qo_iht_step.argtypes = [_f64p, _i64, _i64, _f64p, _u8p, _f32p, _f32p, _f64p, ctypes.c_double,
                                    _i64, _int, _f64p, _i64p]
        lib.qo_iht_step.restype = _i64
        lib.qo_quantease_alg1_f32.argtypes = [_f64p, _i64, _i64, _f32p, _f32p, _f32p, _int, _int,
                                              _u8p, _u8p, _u8p, _f64p, _u8p, _f64p, _int]
        lib.qo_quantease_alg1_f32.restype = _int
        lib.qo_sigma_pairs_bf16.argtypes = [ctypes.POINTER(ctypes.c_uint16), _i64, _i64, _i64p, _i64p,
                                            _i64, _f64p]
        lib.qo_sigma_pairs_bf16.restype = None
        lib.qo_quantease_alg3.argtypes = [_f64p, _i64, _i64, _f64p, _f32p, _f32p, _int, _int,
                                          _u8p, _f64p, _int]
        lib.qo_quantease_alg3.restype = _int
        lib.qo_threads.argtypes = [_int]
        lib.qo_threads.restype = _int
        lib.qo_power_lambda.argtypes = [_f64p, _i64, _int]
        lib.qo_power_lambda.restype = ctypes.c_double
        lib.qo_topk.argtypes = [_f64p, _i64, _i64, _i64p]
        lib.qo_topk.restype = _i64
        lib.qo_quantease_outlier.argtypes = [_f64p, _i64, _i64, _f64p, _int, _int, _i64, _int,
                                             _u8p, _f32p, _f32p, _f64p, _f64p, _f64p, _f64p, _i64p, _int]
        lib.qo_topk_columns.argtypes = [_f64p, _i64, _i64, _i64, _i64p]
        lib.qo_topk_columns.restype = _i64
        lib.qo_quantease_outlier.restype = _int
        self.lib = lib

    # -- grid ---------------------------------------------------------------
    def grid(self, W, bits, excl=None, group_size=0):
        """(scale, zero) of the asymmetric min/max grid (binary32): per row, or with
        group_size > 0 per row and group of group_size columns (arrays q x groups)."""
        W = _f64(W)
        q, p = W.shape
        ex = None if excl is None else np.ascontiguousarray(excl, dtype=np.uint8)
        if group_size:
            ng = -(-p // group_size)
            scale = np.empty((q, ng), np.float32)
            zero = np.empty((q, ng), np.float32)
            self.lib.qo_grid_groups(_ptr(W, _f64p), q, p, group_size, bits, _ptr(ex, _u8p),
                                    _ptr(scale, _f32p), _ptr(zero, _f32p))
            return scale, zero
        scale = np.empty(q, np.float32)
        zero = np.empty(q, np.float32)
        self.lib.qo_grid(_ptr(W, _f64p), q, p, bits, _ptr(ex, _u8p),
                         _ptr(scale, _f32p), _ptr(zero, _f32p))
        return scale, zero

    def rtn(self, W, scale, zero, bits, group_size=0):
        W = _f64(W)
        q, p = W.shape
        codes = np.empty((q, p), np.uint8)
        self.lib.qo_rtn_groups(_ptr(W, _f64p), q, p, group_size or p,
                               _ptr(np.ascontiguousarray(scale, np.float32), _f32p),
                               _ptr(np.ascontiguousarray(zero, np.float32), _f32p), bits, _ptr(codes, _u8p))
        return codes

    # -- Sigma / objective --------------------------------------------------
    def sigma(self, X):
        X = _f64(X)
        p, n = X.shape
        S = np.empty((p, p), np.float64)
        self.lib.qo_sigma(_ptr(X, _f64p), p, n, _ptr(S, _f64p))
        return S

    def sigma_pairs_bf16(self, Xbits, a, b):
        """Sigma_ab = sum_k X_ak X_bk in binary64 for index arrays a, b; Xbits is the
        p x n matrix of bfloat16 bit patterns (uint16)."""
        X = np.ascontiguousarray(Xbits, np.uint16)
        a = np.ascontiguousarray(a, np.int64)
        b = np.ascontiguousarray(b, np.int64)
        out = np.empty(a.size, np.float64)
        self.lib.qo_sigma_pairs_bf16(X.ctypes.data_as(ctypes.POINTER(ctypes.c_uint16)), X.shape[1],
                                     X.shape[1], _ptr(a, _i64p), _ptr(b, _i64p), a.size,
                                     _ptr(out, _f64p))
        return out

    def objective_rows(self, W, codes, scale, zero, S, H=None, group_size=0):
        W = _f64(W)
        q, p = W.shape
        out = np.empty(q, np.float64)
        Hc = None if H is None else _f64(H)
        self.lib.qo_objective_rows_groups(_ptr(W, _f64p), _ptr(Hc, _f64p),
                                          _ptr(np.ascontiguousarray(codes, np.uint8), _u8p),
                                          _ptr(np.ascontiguousarray(scale, np.float32), _f32p),
                                          _ptr(np.ascontiguousarray(zero, np.float32), _f32p),
                                          q, p, group_size or p, _ptr(_f64(S), _f64p), _ptr(out, _f64p))
        return out

    def threads(self, n: int = 0) -> int:
        """Host threads of the row loops (timing only): n > 0 sets them; returns the
        count in effect before the call."""
        return int(self.lib.qo_threads(n))

    # -- Algorithm 1 / 3 ----------------------------------------------------
    def alg1(self, W, S, scale, zero, bits, iters, init_codes=None, forced=None,
             record=False, want_beta=False, relax_period=0, group_size=0):
        """Algorithm 1.  Returns dict(codes, obj_rows[iters, q], obj[iters],
        sweep_codes[iters, q, p] if record, beta[iters, q, p] if want_beta).
        relax_period > 0: sweeps t (from 1) with t mod relax_period = 0 and t < iters
        keep beta~ unquantized (the relax heuristic of Sec. 3.2).  group_size > 0: grouped
        grids, scale / zero q x groups (from grid(..., group_size)); binary64 S only.
        A float32 S is read as is and promoted exactly row by row (same binary64
        arithmetic, half the host memory); anything else is converted to float64."""
        W = _f64(W)
        f32 = isinstance(S, np.ndarray) and S.dtype == np.float32
        S = np.ascontiguousarray(S) if f32 else _f64(S)
        q, p = W.shape
        codes = np.empty((q, p), np.uint8)
        obj_rows = np.empty((iters, q), np.float64)
        sweep = np.empty((iters, q, p), np.uint8) if record else None
        beta = np.empty((iters, q, p), np.float64) if want_beta else None
        ic = None if init_codes is None else np.ascontiguousarray(init_codes, np.uint8)
        fc = None if forced is None else np.ascontiguousarray(forced, np.uint8)
        sc = _ptr(np.ascontiguousarray(scale, np.float32), _f32p)
        zc = _ptr(np.ascontiguousarray(zero, np.float32), _f32p)
        if group_size:
            if f32:
                S = S.astype(np.float64)
            rc = self.lib.qo_quantease_alg1_groups(
                _ptr(W, _f64p), q, p, _ptr(S, _f64p), group_size, sc, zc, bits, iters,
                _ptr(ic, _u8p), _ptr(fc, _u8p), _ptr(codes, _u8p), _ptr(obj_rows, _f64p),
                _ptr(sweep, _u8p), _ptr(beta, _f64p), relax_period)
        else:
            fn = self.lib.qo_quantease_alg1_f32 if f32 else self.lib.qo_quantease_alg1
            rc = fn(
                _ptr(W, _f64p), q, p, _ptr(S, _f32p if f32 else _f64p), sc, zc, bits, iters,
                _ptr(ic, _u8p), _ptr(fc, _u8p), _ptr(codes, _u8p), _ptr(obj_rows, _f64p),
                _ptr(sweep, _u8p), _ptr(beta, _f64p), relax_period)
        if rc:
            raise MemoryError("oracle alg1 allocation failed")
        out = dict(codes=codes, obj_rows=obj_rows, obj=obj_rows.sum(axis=1))
        if record:
            out["sweep_codes"] = sweep
        if want_beta:
            out["beta"] = beta
        return out

    def alg3(self, W, S, scale, zero, bits, iters, relax_period=0):
        W = _f64(W)
        S = _f64(S)
        q, p = W.shape
        codes = np.empty((q, p), np.uint8)
        obj_rows = np.empty((iters, q), np.float64)
        rc = self.lib.qo_quantease_alg3(
            _ptr(W, _f64p), q, p, _ptr(S, _f64p),
            _ptr(np.ascontiguousarray(scale, np.float32), _f32p),
            _ptr(np.ascontiguousarray(zero, np.float32), _f32p), bits, iters,
            _ptr(codes, _u8p), _ptr(obj_rows, _f64p), relax_period)
        if rc:
            raise MemoryError("oracle alg3 allocation failed")
        return dict(codes=codes, obj_rows=obj_rows, obj=obj_rows.sum(axis=1))

    # -- outlier-aware (Algorithm 4) ----------------------------------------
    def power_lambda(self, S, iters):
        S = _f64(S)
        return float(self.lib.qo_power_lambda(_ptr(S, _f64p), S.shape[0], iters))

    def topk(self, T, s):
        T = _f64(T).ravel()
        idx = np.empty(max(int(s), 1), np.int64)
        cnt = self.lib.qo_topk(_ptr(T, _f64p), T.size, int(s), _ptr(idx, _i64p))
        return idx[:cnt].copy()

    def topk_columns(self, T, k):
        """Indices (ascending) of the k columns of T with the largest l2 norms."""
        T = _f64(T)
        idx = np.empty(max(T.shape[1], 1), np.int64)
        cnt = self.lib.qo_topk_columns(_ptr(T, _f64p), T.shape[0], T.shape[1], int(k), _ptr(idx, _i64p))
        return idx[:cnt].copy()

    def iht_step(self, W, S, codes, scale, zero, H, eta, s_budget, structured=False):
        """One IHT half-step of Algorithm 4 from the state (codes on the grid, H):
        returns (T, support) with T = H - 2 eta (H + What - W) Sigma and the support of
        P_s(T) (ascending linear indices; the column selection with structured)."""
        W = _f64(W)
        S = _f64(S)
        q, p = W.shape
        H = _f64(H)
        T = np.empty((q, p), np.float64)
        idx = np.empty(max(int(s_budget), 1), np.int64)
        cnt = self.lib.qo_iht_step(_ptr(W, _f64p), q, p, _ptr(S, _f64p),
                                   _ptr(np.ascontiguousarray(codes, np.uint8), _u8p),
                                   _ptr(np.ascontiguousarray(scale, np.float32), _f32p),
                                   _ptr(np.ascontiguousarray(zero, np.float32), _f32p),
                                   _ptr(H, _f64p), float(eta), int(s_budget), int(structured),
                                   _ptr(T, _f64p), _ptr(idx, _i64p))
        if cnt < 0:
            raise MemoryError("oracle iht_step allocation failed")
        return T, idx[:cnt].copy()

    def outlier(self, W, S, bits, iters, s_budget, power_iters, structured=False):
        W = _f64(W)
        S = _f64(S)
        q, p = W.shape
        codes = np.empty((q, p), np.uint8)
        scale = np.empty(q, np.float32)
        zero = np.empty(q, np.float32)
        H = np.empty((q, p), np.float64)
        obj = np.empty(iters, np.float64)
        obj_cd = np.empty(iters, np.float64)
        eta = np.zeros(1, np.float64)
        nnz = np.zeros(1, np.int64)
        rc = self.lib.qo_quantease_outlier(
            _ptr(W, _f64p), q, p, _ptr(S, _f64p), bits, iters, int(s_budget), power_iters,
            _ptr(codes, _u8p), _ptr(scale, _f32p), _ptr(zero, _f32p), _ptr(H, _f64p),
            _ptr(obj, _f64p), _ptr(obj_cd, _f64p), _ptr(eta, _f64p), _ptr(nnz, _i64p), int(structured))
        if rc:
            raise MemoryError("oracle outlier allocation failed")
        return dict(codes=codes, scale=scale, zero=zero, H=H, obj=obj, obj_cd=obj_cd,
                    eta=float(eta[0]), nnz=int(nnz[0]))


_default: Oracle | None = None


def get() -> Oracle:
    """The oracle built from ``qe_oracle.c`` (compiled on first use)."""
    global _default
    if _default is None:
        _default = Oracle()
    return _default


def levels(codes, scale, zero):
    """Dequantised values s_i (c - z_i) in binary64."""
    return np.asarray(scale, np.float64)[:, None] * (np.asarray(codes, np.float64)
                                                     - np.asarray(zero, np.float64)[:, None])


# -- storage of the codes (Sec. 2.1 fixes them as integers 0 .. 2^b - 1) ------
def pack_codes(codes, bits: int) -> np.ndarray:
    """Each row as a little-endian bit stream, written out from its definition: bit
    k of code j is bit j * bits + k of the row; byte m holds bits 8m .. 8m + 7 (bit 8m
    the least significant); the padding bits of the last byte are zero."""
    codes = np.ascontiguousarray(codes, np.uint8)
    q, p = codes.shape
    bitv = (codes[:, :, None] >> np.arange(bits, dtype=np.uint8)[None, None, :]) & 1
    nbytes = (p * bits + 7) // 8
    stream = np.zeros((q, nbytes * 8), np.uint16)
    stream[:, :p * bits] = bitv.reshape(q, p * bits)
    weight = (1 << np.arange(8)).astype(np.uint16)
    return (stream.reshape(q, nbytes, 8) * weight).sum(axis=2).astype(np.uint8)

