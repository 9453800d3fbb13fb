"""Parity checks between the CUDA path and the fp64 oracle.

Tolerances (the layer-quantization parity bar):
  * objective per sweep: relative error <= 1e-4;
  * codes: >= 99.9% identical free-running; teacher-forced, every code equals
    the oracle's nearest level of beta~ (computed in fp64 from the GPU's own
    state) unless beta~/s + z lies within 1e-4 of a rounding midpoint;
  * scales / zero-points: bit-identical (both sides evaluate the grid in binary32).
"""
import numpy as np
import torch

import oracle

OBJ_RTOL = 1e-4
CODE_MATCH = 0.999
MIDPOINT_TOL = 1e-4


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float64).numpy()


def check_grid(scales, zeros, W64, bits, excl=None):
    O = oracle.get()
    s_o, z_o = O.grid(W64, bits, excl)
    s_g = scales.cpu().numpy()
    z_g = zeros.cpu().numpy()
    assert np.array_equal(s_g, s_o), f"scales differ in {np.sum(s_g != s_o)} rows"
    assert np.array_equal(z_g, z_o), f"zero-points differ in {np.sum(z_g != z_o)} rows"
    return s_o, z_o


def check_obj(obj_gpu, obj_oracle, rtol=OBJ_RTOL, what="objective", atol=0.0):
    """|gpu - oracle| <= rtol |oracle| + atol.  atol (a small multiple of
    ||W X||^2, i.e. of the relative calibration error's denominator) only matters
    for degenerate layers whose objective is a rounding residue near zero."""
    g = np.asarray(obj_gpu, np.float64)
    o = np.asarray(obj_oracle, np.float64)
    err = np.abs(g - o)
    ok = err <= rtol * np.abs(o) + atol
    rel = err / np.maximum(np.abs(o), 1e-300)
    assert np.all(ok), f"{what}: max rel err {rel.max():.3e} (gpu {g}, oracle {o})"
    return float(rel.max())


def teacher_forced(W64, S64, scale, zero, bits, sweep_codes_gpu, init_codes=None, want_run=False,
                   group_size=0):
    """Replay the GPU trajectory through Algorithm 1 with its own codes forced:
    every GPU code must be the nearest level of the fp64 beta~ unless beta~
    sits within MIDPOINT_TOL (in grid steps) of a rounding midpoint.
    Returns (number of near-midpoint disagreements, number of checks), plus the
    oracle's replay (objective of the GPU's codes after each sweep) with want_run.
    group_size > 0: grouped grids (scale / zero q x groups)."""
    O = oracle.get()
    iters = sweep_codes_gpu.shape[0]
    r = O.alg1(W64, S64, scale, zero, bits, iters, init_codes=init_codes,
               forced=sweep_codes_gpu, want_beta=True, group_size=group_size)
    maxq = 2 ** bits - 1
    p = W64.shape[1]
    if group_size:
        g = np.arange(p) // group_size
        sc, zc = scale.astype(np.float64)[:, g], zero.astype(np.float64)[:, g]
    else:
        sc, zc = scale.astype(np.float64)[:, None], zero.astype(np.float64)[:, None]
    t = r["beta"] / sc[None] + zc[None]
    ideal = np.clip(np.rint(t), 0, maxq)
    got = sweep_codes_gpu.astype(np.float64)
    bad = got != ideal
    if np.any(bad):
        frac = t[bad] - np.floor(t[bad])
        near = np.abs(frac - 0.5) <= MIDPOINT_TOL
        lo = np.clip(np.floor(t[bad]), 0, maxq)
        hi = np.clip(np.floor(t[bad]) + 1, 0, maxq)
        neighbour = (got[bad] == lo) | (got[bad] == hi)
        ok = near & neighbour
        assert np.all(ok), (f"{np.sum(~ok)} GPU codes are not the nearest level and not near a "
                            f"midpoint; worst |frac-0.5| = {np.min(np.abs(frac[~ok] - 0.5)):.3e}")
    if want_run:
        del r["beta"]
        return int(bad.sum()), int(bad.size), r
    return int(bad.sum()), int(bad.size)


def code_match(codes_gpu, codes_oracle):
    return float(np.mean(np.asarray(codes_gpu) == np.asarray(codes_oracle)))
