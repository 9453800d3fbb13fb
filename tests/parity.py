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


def first_divergence(sweep_gpu, ref, scale, zero, bits, group_size=0):
    """Compare the GPU's per-sweep codes with the oracle's free-running trajectory
    (ref: alg1 with record=True, want_beta=True) row by row.  Up to a row's first
    differing decision both sides hold the same state, so the oracle's fp64 beta~
    there is the teacher-forced one: that decision must lie within MIDPOINT_TOL
    (grid steps) of a rounding midpoint, which is what starts a legitimate cascade.
    Returns the rows that diverge, each as (row, sweep, column, |frac - 0.5|, codes
    that differ after the last sweep)."""
    sweep_gpu = np.asarray(sweep_gpu)
    oc = ref["sweep_codes"]
    iters, q, p = sweep_gpu.shape
    if group_size:
        g = np.arange(p) // group_size
        sc, zc = scale.astype(np.float64)[:, g], zero.astype(np.float64)[:, g]
    else:
        sc = np.repeat(scale.astype(np.float64)[:, None], p, axis=1)
        zc = np.repeat(zero.astype(np.float64)[:, None], p, axis=1)
    out = []
    for r in range(q):
        diff = sweep_gpu[:, r, :] != oc[:, r, :]
        if not diff.any():
            continue
        t = int(np.argmax(diff.any(axis=1)))
        j = int(np.argmax(diff[t]))
        x = ref["beta"][t, r, j] / sc[r, j] + zc[r, j]
        dist = abs(x - np.floor(x) - 0.5)
        assert dist <= MIDPOINT_TOL, (f"row {r}: first divergence at sweep {t + 1}, column {j} is not "
                                      f"near a midpoint (beta~/s + z = {x:.9f})")
        out.append((r, t, j, float(dist), int(diff[-1].sum())))
    return out


def outlier_replay(W64, S64, scale, zero, bits, sweep_gpu, H_idx_gpu, H_val_gpu, H0, eta, s_budget,
                   structured=False, h_rtol=1e-5):
    """Teacher-forced replay of Algorithm 4, iteration by iteration from the GPU's own
    state.  sweep_gpu[t]: the GPU's codes after iteration t; H_idx_gpu[t] /
    H_val_gpu[t]: its H after iteration t (support, ascending, and values); H0: the
    start H = P_s(W).  Iteration t:
      * CD half: Algorithm 1 for one sweep on the target W - H_{t-1}, from the GPU's
        codes after iteration t - 1 (iteration 0 starts at the target itself), with
        the GPU's decisions forced: each must be the nearest level of the fp64 beta~
        unless within MIDPOINT_TOL of a midpoint;
      * IHT half: the oracle's step from (codes_t, H_{t-1}) must keep the GPU's
        support, except entries (columns) whose |T| (column norm) ties the threshold
        within h_rtol, and the GPU's values must equal T there within h_rtol of max |T|.
    Returns the number of support entries that differed at ties."""
    q, p = W64.shape
    iters = sweep_gpu.shape[0]
    ties = 0
    for t in range(iters):
        Hprev = H0 if t == 0 else _dense(H_idx_gpu[t - 1], H_val_gpu[t - 1], q, p)
        init = None if t == 0 else sweep_gpu[t - 1]
        teacher_forced(W64 - Hprev, S64, scale, zero, bits, sweep_gpu[t][None], init_codes=init)
        T, sup = oracle.get().iht_step(W64, S64, sweep_gpu[t], scale, zero, Hprev, eta, s_budget, structured)
        gsup = np.asarray(H_idx_gpu[t])
        Tf = T.ravel()
        if structured:
            norms = np.sum(T * T, axis=0)
            oc, gc = np.unique(sup % p), np.unique(gsup % p)
            thr = norms[oc].min() if oc.size else 0.0
            for c in np.setxor1d(oc, gc):
                assert abs(norms[c] - thr) <= h_rtol * thr, f"iteration {t + 1}: column {c} kept by one side only"
                ties += 1
        else:
            thr = np.abs(Tf[sup]).min() if sup.size else 0.0
            for k in np.setxor1d(sup, gsup):
                assert abs(abs(Tf[k]) - thr) <= h_rtol * thr, f"iteration {t + 1}: entry {k} kept by one side only"
                ties += 1
        scale_t = np.abs(Tf).max() if Tf.size else 1.0
        err = np.abs(np.asarray(H_val_gpu[t], np.float64) - Tf[gsup])
        assert np.all(err <= h_rtol * scale_t), (f"iteration {t + 1}: H values off by {err.max():.3e} "
                                                 f"(max |T| {scale_t:.3e})")
    return ties


def _dense(idx, val, q, p):
    H = np.zeros(q * p)
    H[np.asarray(idx)] = np.asarray(val, np.float64)
    return H.reshape(q, p)
