"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these compares the oracle with itself: each one checks it against a
brute force, an exhaustive search, a closed form, an invariant, an algebraic
identity between two independently written forms, or a textbook special case.
"""
import itertools

import numpy as np
import pytest

import oracle
from oracle import levels

O = oracle.get()


def _rand_layer(rng, q, p, n, heavy=(), heavy_mult=8.0, zero_rows=(), corr=False):
    W = rng.normal(0.0, 0.02, size=(q, p))
    X = rng.normal(0.0, 1.0, size=(p, n))
    if corr:
        U = rng.normal(size=(p, 2)) / np.sqrt(p)
        V = rng.normal(size=(p, 2)) * 2.0
        X = X + U @ (V.T @ X)
    for r in heavy:
        X[r] *= heavy_mult
    for r in zero_rows:
        X[r] = 0.0
    # exact binary32 values, as the layers fed to the GPU path
    return W.astype(np.float32).astype(np.float64), X.astype(np.float32).astype(np.float64)


def _f_direct(W, What, X):
    """||W X - What X||_F^2 of Eq. (layerwise-main), from X itself."""
    R = (W - What) @ X
    return float(np.sum(R * R))


# --------------------------------------------------------------------------
# grid and quantization operator (Sec. 2.1, Eq. eq:quant)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_quantizer_returns_nearest_level(bits):
    rng = np.random.default_rng(bits)
    W = rng.normal(0, 0.05, size=(6, 300)).astype(np.float32).astype(np.float64)
    W[1] = np.abs(W[1])          # all non-negative row
    W[2] = -np.abs(W[2])         # all non-positive row
    W[3] = 0.0                   # all-zero row -> range [-1, 1]
    W[4, :3] = [4.0, -0.5, 0.25]  # one dominant entry
    s, z = O.grid(W, bits)
    maxq = 2 ** bits - 1
    assert np.all(s > 0) and np.all(z == np.round(z)) and np.all((z >= 0) & (z <= maxq))
    codes = O.rtn(W, s, z, bits)
    lev = s.astype(np.float64)[:, None] * (np.arange(maxq + 1)[None, :] - z.astype(np.float64)[:, None])
    dist = (W[:, :, None] - lev[:, None, :]) ** 2
    chosen = np.take_along_axis(dist, codes[:, :, None].astype(np.int64), axis=2)[..., 0]
    assert np.all(chosen <= dist.min(axis=2) * (1 + 1e-12) + 1e-300)


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_grid_covers_row_range_and_zero(bits):
    rng = np.random.default_rng(10 + bits)
    W = rng.normal(0, 0.02, size=(20, 64)).astype(np.float32).astype(np.float64)
    W[5] = np.abs(W[5])
    W[6] = 0.0
    s, z = O.grid(W, bits)
    maxq = 2 ** bits - 1
    lo = np.minimum(W.min(axis=1), 0.0)
    hi = np.maximum(W.max(axis=1), 0.0)
    lo[6], hi[6] = -1.0, 1.0
    s64, z64 = s.astype(np.float64), z.astype(np.float64)
    # 2^b distinct levels, zero is one of them exactly, the extremes are within half a step
    assert np.all(s64 * (0 - z64) <= lo + 0.5 * s64 * (1 + 1e-6))
    assert np.all(s64 * (maxq - z64) >= hi - 0.5 * s64 * (1 + 1e-6))
    assert np.all(s64 * (z64 - z64) == 0.0)
    assert np.allclose(s64 * maxq, hi - lo, rtol=1e-6)


def test_grid_excluded_entries_leave_the_pool():
    rng = np.random.default_rng(3)
    W = rng.normal(0, 0.02, size=(4, 50))
    W[0, 7] = 1.5
    W[2, 3] = -2.0
    excl = np.zeros(W.shape, np.uint8)
    excl[0, 7] = excl[2, 3] = 1
    s1, z1 = O.grid(W, 3, excl)
    W2 = W.copy()
    W2[0, 7] = W2[2, 3] = 0.0
    s2, z2 = O.grid(W2, 3)
    assert np.array_equal(s1, s2) and np.array_equal(z1, z2)


# --------------------------------------------------------------------------
# Lemma 1: every CD update is the exact 1-D minimiser over the grid
# --------------------------------------------------------------------------
@pytest.mark.parametrize("bits", [2, 3, 4])
def test_every_update_is_bruteforce_argmin(bits):
    rng = np.random.default_rng(100 + bits)
    q, p, n, iters = 3, 7, 40, 3
    W, X = _rand_layer(rng, q, p, n, heavy=(2,), zero_rows=(5,), corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, bits)
    r = O.alg1(W, S, s, z, bits, iters, record=True)
    sc = r["sweep_codes"]
    maxq = 2 ** bits - 1
    cand = np.arange(maxq + 1)
    for t in range(iters):
        before = W.copy() if t == 0 else levels(sc[t - 1], s, z)
        after = levels(sc[t], s, z)
        for i in range(q):
            for j in range(p):
                state = np.concatenate([after[i, :j], before[i, j:]])
                if j == 5:  # dead column: nearest level of W, fixed
                    assert sc[t, i, j] == O.rtn(W[i:i + 1, j:j + 1], s[i:i + 1], z[i:i + 1], bits)[0, 0]
                    continue
                f = []
                for c in cand:
                    row = state.copy()
                    row[j] = float(s[i]) * (c - float(z[i]))
                    f.append(_f_direct(W[i:i + 1], row[None, :], X))
                f = np.array(f)
                assert f[sc[t, i, j]] <= f.min() + 1e-12 * max(1.0, abs(f.min())), (t, i, j)


# --------------------------------------------------------------------------
# exhaustive search on tiny layers: CD ends at a coordinate-wise minimum
# --------------------------------------------------------------------------
@pytest.mark.parametrize("p", [2, 3, 4])
def test_exhaustive_tiny_layer_cw_minimum(p):
    bits = 2
    rng = np.random.default_rng(200 + p)
    for trial in range(5):
        W, X = _rand_layer(rng, 1, p, 12, corr=True)
        S = O.sigma(X)
        s, z = O.grid(W, bits)
        r = O.alg1(W, S, s, z, bits, iters=40)
        lev = lambda c: float(s[0]) * (np.asarray(c, np.float64) - float(z[0]))
        allf = {c: _f_direct(W, lev(c)[None, :], X)
                for c in itertools.product(range(4), repeat=p)}
        fstar = min(allf.values())
        c_cd = tuple(int(v) for v in r["codes"][0])
        f_cd = allf[c_cd]
        # the reported objective is f of the returned codes, and no code vector beats f*
        assert np.isclose(r["obj"][-1], f_cd, rtol=1e-10, atol=1e-300)
        assert f_cd >= fstar - 1e-15
        # coordinate-wise minimum (Sec. 3.3, Definition): no single coordinate change improves f
        for j in range(p):
            for c in range(4):
                alt = list(c_cd)
                alt[j] = c
                assert allf[tuple(alt)] >= f_cd - 1e-12 * max(1.0, f_cd)


# --------------------------------------------------------------------------
# monotone objective after the first (feasible) sweep (Sec. 3.1, Lemma 2)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed,corr", [(0, False), (1, True), (2, True)])
def test_objective_non_increasing(seed, corr):
    rng = np.random.default_rng(300 + seed)
    W, X = _rand_layer(rng, 16, 48, 200, heavy=(3, 11), heavy_mult=20.0, corr=corr)
    S = O.sigma(X)
    for bits in (3, 4):
        s, z = O.grid(W, bits)
        obj = O.alg1(W, S, s, z, bits, iters=8)["obj"]
        assert np.all(np.diff(obj) <= 1e-12 * obj[:-1])


# --------------------------------------------------------------------------
# Algorithm 1 == Algorithm 3 (Sec. 3.2: an exact reassociation)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("bits,relax", [(3, 0), (4, 0), (3, 2), (4, 3)])
def test_algorithm1_equals_algorithm3(bits, relax):
    rng = np.random.default_rng(400 + bits)
    W, X = _rand_layer(rng, 24, 40, 160, heavy=(1,), heavy_mult=30.0, zero_rows=(7,), corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, bits)
    a1 = O.alg1(W, S, s, z, bits, iters=5, relax_period=relax)
    a3 = O.alg3(W, S, s, z, bits, iters=5, relax_period=relax)
    assert np.array_equal(a1["codes"], a3["codes"])
    assert np.allclose(a1["obj_rows"], a3["obj_rows"], rtol=1e-10, atol=0)


# --------------------------------------------------------------------------
# relax heuristic (Sec. 3.2): a relaxed sweep takes beta~ itself, i.e. exact
# coordinate minimization of the convex quadratic f over all reals.  One such
# sweep over j = 1..p is one Gauss-Seidel step for the normal equations
# What Sigma = W Sigma (Lemma 1), so it is pinned by the textbook splitting
# Sigma = L + D + U:  (D + L) x_new = Sigma w - U x_old  (rows of W are
# independent, Sec. 3.2).
# --------------------------------------------------------------------------
def _gauss_seidel_step(S, w, x_old):
    from scipy.linalg import solve_triangular
    return solve_triangular(np.tril(S), S @ w - np.triu(S, 1) @ x_old, lower=True)


@pytest.mark.parametrize("bits", [2, 3])
def test_relaxed_sweep_is_one_gauss_seidel_step(bits):
    rng = np.random.default_rng(700 + bits)
    W, X = _rand_layer(rng, 8, 28, 120, heavy=(2, 9), heavy_mult=12.0, corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, bits)
    r = O.alg1(W, S, s, z, bits, iters=3, record=True, want_beta=True, relax_period=2)
    x_old = levels(r["sweep_codes"][0], s, z)          # state after sweep 1 (quantized)
    for i in range(W.shape[0]):
        x_new = _gauss_seidel_step(S, W[i], x_old[i])
        assert np.allclose(r["beta"][1][i], x_new, rtol=1e-9, atol=1e-12)
        f_new = float((W[i] - x_new) @ S @ (W[i] - x_new))
        assert np.isclose(r["obj_rows"][1][i], f_new, rtol=1e-9, atol=1e-18)
    # exact minimization along every coordinate: the relaxed sweep never increases f
    assert np.all(r["obj_rows"][1] <= r["obj_rows"][0] * (1 + 1e-12))
    # its code record is the nearest level of the relaxed values; sweep 3 quantizes again
    s32, z32 = s.astype(np.float64), z.astype(np.float64)
    near = np.clip(np.rint(r["beta"][1] / s32[:, None] + z32[:, None]), 0, 2 ** bits - 1)
    assert np.array_equal(r["sweep_codes"][1], near.astype(np.uint8))


def test_relaxed_sweep_with_diagonal_sigma_reaches_w():
    """Orthogonal input channels: beta~ = W_ij whatever the state (up to the rounding
    of (W_ij Sigma_jj) / Sigma_jj), so a relaxed sweep gives f = 0 and the following
    quantized sweep is round-to-nearest."""
    rng = np.random.default_rng(8)
    q, p, n = 6, 20, 48
    Qm, _ = np.linalg.qr(rng.normal(size=(n, p)))
    X = Qm.T * rng.uniform(0.5, 3.0, size=(p, 1))
    W = rng.normal(0, 0.02, size=(q, p))
    S = np.diag(np.diag(X @ X.T))
    s, z = O.grid(W, 3)
    rtn = O.rtn(W, s, z, 3)
    r = O.alg1(W, S, s, z, 3, iters=3, record=True, init_codes=np.zeros((q, p), np.uint8),
               relax_period=1)
    scale = (W * W) @ np.diag(S)                      # f of What = 0, per row
    assert np.all(r["obj_rows"][:2] <= 1e-24 * scale)
    assert np.array_equal(r["codes"], rtn)


def test_relaxed_sweeps_converge_to_w():
    """Gauss-Seidel on a positive definite Sigma converges: from round-to-nearest
    codes, relaxed sweeps (period 1: all but the last) drive What to W and f to 0
    (down to rounding), never increasing f on the way."""
    rng = np.random.default_rng(9)
    W, X = _rand_layer(rng, 5, 16, 400, heavy=(3,), heavy_mult=4.0)
    S = O.sigma(X)
    s, z = O.grid(W, 3)
    rtn = O.rtn(W, s, z, 3)
    f0 = O.alg1(W, S, s, z, 3, iters=1, init_codes=rtn, forced=rtn[None])["obj"][0]
    r = O.alg1(W, S, s, z, 3, iters=40, init_codes=rtn, want_beta=True, relax_period=1)
    obj = r["obj"][:-1]
    big = obj > 1e-20 * f0
    assert np.all(np.diff(obj)[big[:-1]] <= 1e-12 * obj[:-1][big[:-1]])
    assert obj[-1] <= 1e-20 * f0
    assert np.allclose(r["beta"][-2], W, rtol=0, atol=1e-12 * np.abs(W).max())


def test_relax_period_not_below_iters_is_plain_algorithm1():
    rng = np.random.default_rng(10)
    W, X = _rand_layer(rng, 6, 24, 100, corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, 4)
    a = O.alg1(W, S, s, z, 4, iters=4, record=True)
    b = O.alg1(W, S, s, z, 4, iters=4, record=True, relax_period=4)
    assert np.array_equal(a["sweep_codes"], b["sweep_codes"])
    assert np.array_equal(a["obj_rows"], b["obj_rows"])
    c = O.alg1(W, S, s, z, 4, iters=4, record=True, relax_period=3)
    assert not np.array_equal(a["obj_rows"][2], c["obj_rows"][2])


# --------------------------------------------------------------------------
# textbook special case: orthogonal input channels -> round-to-nearest
# --------------------------------------------------------------------------
def test_diagonal_sigma_gives_round_to_nearest():
    rng = np.random.default_rng(5)
    q, p, n = 10, 32, 64
    Qm, _ = np.linalg.qr(rng.normal(size=(n, p)))
    X = (Qm.T * rng.uniform(0.5, 3.0, size=(p, 1)))        # rows orthogonal
    W = rng.normal(0, 0.02, size=(q, p))
    S = X @ X.T
    S = np.diag(np.diag(S))                                  # exactly diagonal
    for bits in (2, 4):
        s, z = O.grid(W, bits)
        r = O.alg1(W, S, s, z, bits, iters=3, record=True)
        rtn = O.rtn(W, s, z, bits)
        for t in range(3):
            assert np.array_equal(r["sweep_codes"][t], rtn)


# --------------------------------------------------------------------------
# objective identity: tr(D Sigma D^T) == ||W X - What X||^2 (proof of Lemma 1)
# --------------------------------------------------------------------------
def test_objective_matches_direct_residual():
    rng = np.random.default_rng(6)
    W, X = _rand_layer(rng, 12, 30, 90, heavy=(4,), corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, 3)
    r = O.alg1(W, S, s, z, 3, iters=2)
    What = levels(r["codes"], s, z)
    direct = np.sum(((W - What) @ X) ** 2, axis=1)
    assert np.allclose(r["obj_rows"][-1], direct, rtol=1e-10)


# --------------------------------------------------------------------------
# Sigma: symmetric PSD, diagonal = squared row norms, X (X^T v) association
# --------------------------------------------------------------------------
def test_sigma_properties():
    rng = np.random.default_rng(7)
    X = rng.normal(size=(37, 111))
    X[3] *= 25.0
    X[9] = 0.0
    S = O.sigma(X)
    assert np.array_equal(S, S.T)
    assert np.allclose(np.diag(S), np.einsum("ij,ij->i", X, X), rtol=1e-13)
    assert S[9, 9] == 0.0 and np.all(S[9] == 0.0)
    ev = np.linalg.eigvalsh(S)
    assert ev.min() >= -1e-10 * ev.max()
    v = rng.normal(size=37)
    assert np.allclose(S @ v, X @ (X.T @ v), rtol=1e-10)


def test_sigma_pairs_from_bf16_bits():
    """Selected Sigma entries from bfloat16 bit patterns: the bit decoding on
    hand-picked patterns, then every entry against a numpy binary64 X X^T."""
    pat = np.array([[0x3F80, 0xC000, 0x3E80, 0x0000, 0x8000, 0x4049]], np.uint16)
    vals = np.array([1.0, -2.0, 0.25, 0.0, -0.0, 3.140625])
    got = O.sigma_pairs_bf16(pat, np.zeros(1, np.int64), np.zeros(1, np.int64))
    assert got[0] == float(np.sum(vals * vals))
    rng = np.random.default_rng(8)
    X = rng.normal(size=(40, 300)).astype(np.float32)
    X[5] *= 30.0
    bits = (X.view(np.uint32) >> 16).astype(np.uint16)          # truncate to bfloat16
    Xb = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    a = rng.integers(0, 40, size=500)
    b = rng.integers(0, 40, size=500)
    a[:40] = np.arange(40)
    b[:40] = np.arange(40)                                       # the diagonal
    ref = np.einsum("ij,ij->i", Xb[a], Xb[b])
    out = O.sigma_pairs_bf16(bits, a, b)
    assert np.allclose(out, ref, rtol=1e-13, atol=1e-13 * np.abs(ref).max())
    assert np.array_equal(out[:40], np.diag(O.sigma(Xb)))       # same sums, same order


def test_alg1_reads_binary32_sigma_exactly():
    """A binary32 Sigma is promoted exactly: the same run as with its binary64 copy."""
    rng = np.random.default_rng(9)
    W, X = _rand_layer(rng, 9, 40, 200, heavy=(3,), corr=True)
    S32 = O.sigma(X).astype(np.float32)
    s, z = O.grid(W, 3)
    a = O.alg1(W, S32, s, z, 3, 3, want_beta=True)
    b = O.alg1(W, S32.astype(np.float64), s, z, 3, 3, want_beta=True)
    assert np.array_equal(a["codes"], b["codes"])
    assert np.array_equal(a["obj_rows"], b["obj_rows"])
    assert np.array_equal(a["beta"], b["beta"])


# --------------------------------------------------------------------------
# invariances: scaling X, permuting / sub-setting rows (Sec. 3.2, rows independent)
# --------------------------------------------------------------------------
def test_invariances():
    rng = np.random.default_rng(8)
    W, X = _rand_layer(rng, 9, 20, 70, heavy=(2,), corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, 3)
    base = O.alg1(W, S, s, z, 3, iters=4)
    S2 = O.sigma(2.0 * X)            # power-of-two scale: bit-identical trajectory
    assert np.array_equal(O.alg1(W, S2, s, z, 3, iters=4)["codes"], base["codes"])
    S3 = O.sigma(3.0 * X)
    assert np.mean(O.alg1(W, S3, s, z, 3, iters=4)["codes"] == base["codes"]) > 0.99
    perm = rng.permutation(9)
    rp = O.alg1(W[perm], S, s[perm], z[perm], 3, iters=4)
    assert np.array_equal(rp["codes"], base["codes"][perm])
    assert np.allclose(rp["obj_rows"], base["obj_rows"][:, perm], rtol=1e-13)
    sub = [1, 4, 7]
    rs = O.alg1(W[sub], S, s[sub], z[sub], 3, iters=4)
    assert np.array_equal(rs["codes"], base["codes"][sub])


def test_warm_start_from_fixed_point_is_stationary():
    """Sec. 3.1: CD can refine any feasible What; a converged state stays put."""
    rng = np.random.default_rng(9)
    W, X = _rand_layer(rng, 6, 16, 60, corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, 3)
    conv = O.alg1(W, S, s, z, 3, iters=60)["codes"]
    again = O.alg1(W, S, s, z, 3, iters=2, init_codes=conv)
    assert np.array_equal(again["codes"], conv)


# --------------------------------------------------------------------------
# outlier-aware pieces (Sec. 4.3): lambda_max, P_s, Lemma 3, s = 0 reduction
# --------------------------------------------------------------------------
def test_power_lambda_matches_eigvalsh():
    rng = np.random.default_rng(11)
    A = rng.normal(size=(40, 80))
    A[0] *= 6.0
    S = A @ A.T
    lam = O.power_lambda(S, 800)
    ev = np.linalg.eigvalsh(S)
    assert abs(lam - ev[-1]) <= 1e-10 * ev[-1]
    for it in (0, 1, 3):                 # a Rayleigh quotient never exceeds lambda_max
        assert O.power_lambda(S, it) <= ev[-1] * (1 + 1e-12)


def test_topk_matches_full_sort_with_ties():
    rng = np.random.default_rng(12)
    T = rng.integers(-5, 6, size=(7, 31)).astype(np.float64) * 0.25   # many ties and zeros
    for s in (0, 1, 5, 40, 150, 217, 400):
        got = O.topk(T, s)
        flat = T.ravel()
        nz = np.nonzero(flat)[0]
        order = nz[np.lexsort((nz, -np.abs(flat[nz])))]
        want = np.sort(order[:s])
        assert np.array_equal(got, want), s


def test_outlier_iht_descent_and_budget():
    rng = np.random.default_rng(13)
    q, p, n, s_budget = 12, 24, 80, 20
    W, X = _rand_layer(rng, q, p, n, heavy=(5,), heavy_mult=10.0, corr=True)
    W[rng.integers(0, q, 8), rng.integers(0, p, 8)] += rng.normal(0, 0.3, 8)
    S = O.sigma(X)
    r = O.outlier(W, S, 3, 8, s_budget, 600)
    assert r["nnz"] <= s_budget and np.count_nonzero(r["H"]) <= s_budget
    # Lemma 3: each IHT step does not increase g; CD halves do not either once feasible
    assert np.all(r["obj"] <= r["obj_cd"] * (1 + 1e-10))
    assert np.all(r["obj_cd"][1:] <= r["obj"][:-1] * (1 + 1e-10))
    # the grid ignores the s largest |W| (Sec. 4.3)
    excl = np.zeros(q * p, np.uint8)
    excl[O.topk(W, s_budget)] = 1
    s_, z_ = O.grid(W, 3, excl.reshape(q, p))
    assert np.array_equal(s_, r["scale"]) and np.array_equal(z_, r["zero"])
    # eta = 1 / (2 lambda_max)
    assert np.isclose(r["eta"], 1.0 / (2.0 * np.linalg.eigvalsh(S)[-1]), rtol=1e-8)
    # reported g equals ||W X - (What + H) X||^2 from X
    What = levels(r["codes"], r["scale"], r["zero"])
    assert np.isclose(r["obj"][-1], _f_direct(W, What + r["H"], X), rtol=1e-10)


@pytest.mark.parametrize("structured", [False, True])
def test_iht_step_gradient_and_projection(structured):
    """The IHT half-step entered from outside state (used to replay the GPU's
    iterations): with a budget that keeps everything, (H - T) / eta is the gradient
    of g(H) = ||(W - What - H) X||^2 (Eq. main-outlier), checked by central
    differences of g computed from X itself; with a small budget the support is the
    s largest |T| (a full sort) or the columns of largest norm (brute force over
    column subsets), and the step never increases g (Lemma 3)."""
    rng = np.random.default_rng(31)
    q, p, n, bits = 4, 6, 30, 3
    W, X = _rand_layer(rng, q, p, n, heavy=(2,), heavy_mult=6.0)
    S = O.sigma(X)
    s_, z_ = O.grid(W, bits)
    codes = O.rtn(W, s_, z_, bits)
    What = levels(codes, s_, z_)
    H = np.zeros((q, p))
    H[rng.integers(0, q, 5), rng.integers(0, p, 5)] = rng.normal(0, 0.1, 5)
    eta = 1.0 / (2.0 * np.linalg.eigvalsh(S)[-1])
    T, sup = O.iht_step(W, S, codes, s_, z_, H, eta, q * p, structured)
    grad = (H - T) / eta
    eps = 1e-6
    for i in range(q):
        for j in range(p):
            E = np.zeros((q, p))
            E[i, j] = eps
            fd = (_f_direct(W - H - E, What, X) - _f_direct(W - H + E, What, X)) / (2 * eps)
            assert abs(fd - grad[i, j]) <= 1e-5 * max(1.0, abs(fd)), (i, j, fd, grad[i, j])
    # projection and descent with a small budget
    s_budget = 8 if not structured else 2 * q
    T, sup = O.iht_step(W, S, codes, s_, z_, H, eta, s_budget, structured)
    if structured:
        norms = np.sum(T * T, axis=0)
        best = max(itertools.combinations(range(p), s_budget // q), key=lambda c: norms[list(c)].sum())
        assert sorted({int(k) % p for k in sup}) == sorted(best)
        assert sup.size == s_budget
    else:
        order = np.argsort(-np.abs(T).ravel(), kind="stable")
        assert np.array_equal(np.sort(order[:s_budget]), sup)
    Hn = np.zeros(q * p)
    Hn[sup] = T.ravel()[sup]
    Hn = Hn.reshape(q, p)
    assert _f_direct(W - Hn, What, X) <= _f_direct(W - H, What, X) * (1 + 1e-12)


def test_iht_step_replays_algorithm4():
    """From the state one oracle iteration of Algorithm 4 leaves behind (the start
    H = P_s(W) and the codes of the first sweep), the IHT step gives that
    iteration's H bit for bit."""
    rng = np.random.default_rng(32)
    q, p, n, s_budget = 10, 20, 60, 15
    W, X = _rand_layer(rng, q, p, n, heavy=(3,), heavy_mult=10.0)
    W[rng.integers(0, q, 6), rng.integers(0, p, 6)] += rng.normal(0, 0.3, 6)
    S = O.sigma(X)
    r = O.outlier(W, S, 3, 1, s_budget, 200)
    H0 = np.zeros(q * p)
    k0 = O.topk(W, s_budget)
    H0[k0] = W.ravel()[k0]
    T, sup = O.iht_step(W, S, r["codes"], r["scale"], r["zero"], H0.reshape(q, p), r["eta"], s_budget)
    Hn = np.zeros(q * p)
    Hn[sup] = T.ravel()[sup]
    assert np.array_equal(Hn.reshape(q, p), r["H"])


def test_outlier_with_zero_budget_reduces_to_algorithm1():
    rng = np.random.default_rng(14)
    W, X = _rand_layer(rng, 8, 20, 50, corr=True)
    S = O.sigma(X)
    r = O.outlier(W, S, 3, 4, 0, 50)
    s, z = O.grid(W, 3)
    a1 = O.alg1(W, S, s, z, 3, iters=4)
    assert np.array_equal(r["codes"], a1["codes"])
    assert np.allclose(r["obj"], a1["obj"], rtol=1e-12) and np.allclose(r["obj_cd"], a1["obj"], rtol=1e-12)
    assert not np.any(r["H"])


# --------------------------------------------------------------------------
# structured outliers (Sec. 4.3, "Structured Outliers"): whole columns
# --------------------------------------------------------------------------
def test_column_selection_is_the_projection():
    """Keeping the k columns of largest l2 norm is the Euclidean projection onto
    matrices with at most k nonzero columns: brute force over every subset of k
    columns, with planted ties (smaller index wins) and a zero column (never kept)."""
    rng = np.random.default_rng(15)
    q, p = 5, 7
    for trial in range(30):
        T = rng.normal(size=(q, p))
        T[:, 2] = T[:, 4]                  # equal norms: column 2 ranks first
        T[:, 6] = 0.0
        for k in (1, 2, 3):
            sel = O.topk_columns(T, k)
            assert np.all(np.diff(sel) > 0) and 6 not in sel and sel.size == k
            # the kept columns leave the least residual ||T - H||_F^2 (up to rounding:
            # the planted tie makes two subsets equal in exact arithmetic)
            res = lambda c: np.sum(np.delete(T, list(c), axis=1) ** 2)
            best = min(res(c) for c in itertools.combinations(range(p), k))
            assert res(sel) <= best * (1 + 1e-12)
            if (2 in sel) != (4 in sel):
                assert 2 in sel                      # the tie goes to the smaller index
        norms = np.sum(T * T, axis=0)
        order = np.lexsort((np.arange(p), -norms))
        assert np.array_equal(O.topk_columns(T, 4), np.sort(order[:4]))
    # fewer nonzero columns than k: only those are kept
    T = np.zeros((q, p))
    T[:, 3] = 1.0
    assert np.array_equal(O.topk_columns(T, 3), [3])


def test_structured_outlier_descent_budget_and_columns():
    rng = np.random.default_rng(16)
    q, p, n = 10, 24, 90
    W, X = _rand_layer(rng, q, p, n, heavy=(5,), heavy_mult=10.0, corr=True)
    W[:, [3, 17]] += rng.normal(0, 0.3, size=(q, 2))        # two outlier columns
    S = O.sigma(X)
    s_budget = 3 * q + 4                                     # floor(s / q) = 3 columns
    r = O.outlier(W, S, 3, 8, s_budget, 600, structured=True)
    cols = np.nonzero(np.any(r["H"] != 0, axis=0))[0]
    assert cols.size <= 3 and r["nnz"] == q * 3
    # Lemma 3 carries over (the column selection is a projection): IHT halves never increase g
    assert np.all(r["obj"] <= r["obj_cd"] * (1 + 1e-10))
    assert np.all(r["obj_cd"][1:] <= r["obj"][:-1] * (1 + 1e-10))
    # the grid leaves out the starting columns, those of W with the largest norms
    start = O.topk_columns(W, 3)
    assert set(start) >= {3, 17}
    excl = np.zeros((q, p), np.uint8)
    excl[:, start] = 1
    s_, z_ = O.grid(W, 3, excl)
    assert np.array_equal(s_, r["scale"]) and np.array_equal(z_, r["zero"])
    What = levels(r["codes"], r["scale"], r["zero"])
    assert np.isclose(r["obj"][-1], _f_direct(W, What + r["H"], X), rtol=1e-10)


def test_structured_outlier_below_one_column_reduces_to_algorithm1():
    rng = np.random.default_rng(17)
    W, X = _rand_layer(rng, 8, 20, 50, corr=True)
    S = O.sigma(X)
    r = O.outlier(W, S, 3, 4, 7, 50, structured=True)        # s < q: no column fits
    s, z = O.grid(W, 3)
    a1 = O.alg1(W, S, s, z, 3, iters=4)
    assert np.array_equal(r["codes"], a1["codes"]) and not np.any(r["H"])
    assert np.allclose(r["obj"], a1["obj"], rtol=1e-12)


# --------------------------------------------------------------------------
# bit-packed storage of the codes (integers 0 .. 2^b - 1, Sec. 2.1)
# --------------------------------------------------------------------------
def test_pack_codes_hand_example():
    """3-bit codes 5, 3, 7, 1 -> bit stream 101 110 111 100 (each code least significant
    bit first) = bytes 0b11011101 = 221 and 0b0011 = 3 (zero padding)."""
    assert oracle.pack_codes(np.array([[5, 3, 7, 1]]), 3).tolist() == [[221, 3]]
    # 8 bits: the codes themselves; 1 bit: eight codes per byte
    c = np.array([[0, 255, 17, 128]], np.uint8)
    assert np.array_equal(oracle.pack_codes(c, 8), c)
    assert oracle.pack_codes(np.array([[1, 0, 1, 1, 0, 0, 0, 1, 1]]), 1).tolist() == [[0b10001101, 1]]


@pytest.mark.parametrize("bits", [1, 2, 3, 4, 5, 7, 8])
def test_pack_codes_matches_packbits_and_unpacks(bits):
    rng = np.random.default_rng(bits)
    codes = rng.integers(0, 2 ** bits, size=(7, 101), dtype=np.uint8)
    packed = oracle.pack_codes(codes, bits)
    assert packed.shape == (7, (101 * bits + 7) // 8)
    # numpy's own little-endian bit packing of the same stream
    stream = np.unpackbits(codes[:, :, None], axis=2, bitorder="little")[:, :, :bits].reshape(7, -1)
    assert np.array_equal(packed, np.packbits(stream, axis=1, bitorder="little"))
    # read back code j from bits j * bits .. j * bits + bits - 1
    bitsarr = np.unpackbits(packed, axis=1, bitorder="little")
    back = sum(bitsarr[:, k::bits][:, :101].astype(np.int64) << k for k in range(bits))
    assert np.array_equal(back, codes)


# --------------------------------------------------------------------------
# grouped grids: a grid per row and group of gsize consecutive columns (the
# grouping the paper notes can be incorporated into the per-channel grid)
# --------------------------------------------------------------------------
def _levels_grouped(codes, s, z, gsize):
    g = np.arange(codes.shape[1]) // gsize
    return s.astype(np.float64)[:, g] * (codes.astype(np.float64) - z.astype(np.float64)[:, g])


@pytest.mark.parametrize("bits,gsize", [(2, 8), (3, 16), (4, 24)])
def test_grouped_grid_is_the_row_rule_per_group(bits, gsize):
    """Each group gets the row rule over its own columns, in binary32: range with 0,
    s = (hi - lo) / (2^b - 1), z = round(-lo / s); an all-zero group gets [-1, 1]."""
    rng = np.random.default_rng(20 + bits)
    W = rng.normal(0, 0.02, size=(5, 70)).astype(np.float32).astype(np.float64)
    W[1, gsize:2 * gsize] = 0.0
    W[2, :gsize] = np.abs(W[2, :gsize])
    s, z = O.grid(W, bits, group_size=gsize)
    ng = -(-70 // gsize)
    assert s.shape == (5, ng) and z.shape == (5, ng)
    maxq = np.float32(2 ** bits - 1)
    for i in range(5):
        for g in range(ng):
            w = W[i, g * gsize:(g + 1) * gsize].astype(np.float32)
            lo, hi = min(np.float32(0), w.min()), max(np.float32(0), w.max())
            if lo == 0 and hi == 0:
                lo, hi = np.float32(-1), np.float32(1)
            sg = np.float32(hi - lo) / maxq
            assert s[i, g] == sg
            assert z[i, g] == np.rint(np.float32(-lo) / sg)
    # one group of p columns is the per-row grid
    s1, z1 = O.grid(W, bits, group_size=70)
    s0, z0 = O.grid(W, bits)
    assert np.array_equal(s1[:, 0], s0) and np.array_equal(z1[:, 0], z0)


def test_grouped_algorithm1_with_one_group_is_per_row_algorithm1():
    rng = np.random.default_rng(21)
    W, X = _rand_layer(rng, 6, 30, 120, heavy=(3,), corr=True)
    S = O.sigma(X)
    s, z = O.grid(W, 3)
    a = O.alg1(W, S, s, z, 3, iters=3, record=True)
    sg, zg = O.grid(W, 3, group_size=30)
    b = O.alg1(W, S, sg, zg, 3, iters=3, record=True, group_size=30)
    assert np.array_equal(a["sweep_codes"], b["sweep_codes"])
    assert np.array_equal(a["obj_rows"], b["obj_rows"])


def test_grouped_diagonal_sigma_gives_per_group_round_to_nearest():
    rng = np.random.default_rng(22)
    q, p, n, gsize = 6, 32, 64, 8
    Qm, _ = np.linalg.qr(rng.normal(size=(n, p)))
    X = Qm.T * rng.uniform(0.5, 3.0, size=(p, 1))
    W = rng.normal(0, 0.02, size=(q, p))
    W[:, 8:16] *= 5.0                       # groups of very different ranges
    S = np.diag(np.diag(X @ X.T))
    s, z = O.grid(W, 3, group_size=gsize)
    r = O.alg1(W, S, s, z, 3, iters=2, record=True, group_size=gsize)
    g = np.arange(p) // gsize
    sf, zf = s.astype(np.float64)[:, g], z.astype(np.float64)[:, g]
    rtn = np.clip(np.rint(W / sf + zf), 0, 7).astype(np.uint8)
    for t in range(2):
        assert np.array_equal(r["sweep_codes"][t], rtn)
    assert np.array_equal(O.rtn(W, s, z, 3, group_size=gsize), rtn)


@pytest.mark.parametrize("bits", [2, 3])
def test_grouped_update_is_bruteforce_argmin_on_its_group(bits):
    """Every update is the brute-force minimiser of ||W X - What X||^2 (from X itself,
    Lemma 1) over the 2^b levels of its own column's group; the objective never
    increases (Lemma 2) and equals the direct residual."""
    rng = np.random.default_rng(110 + bits)
    q, p, n, iters, gsize = 3, 9, 40, 3, 3
    W, X = _rand_layer(rng, q, p, n, heavy=(2,), corr=True)
    W[:, 3:6] *= 4.0
    S = O.sigma(X)
    s, z = O.grid(W, bits, group_size=gsize)
    r = O.alg1(W, S, s, z, bits, iters, record=True, group_size=gsize)
    sc = r["sweep_codes"]
    cand = np.arange(2 ** bits)
    for t in range(iters):
        before = W.copy() if t == 0 else _levels_grouped(sc[t - 1], s, z, gsize)
        after = _levels_grouped(sc[t], s, z, gsize)
        for i in range(q):
            for j in range(p):
                state = np.concatenate([after[i, :j], before[i, j:]])
                sg, zg = float(s[i, j // gsize]), float(z[i, j // gsize])
                f = []
                for c in cand:
                    row = state.copy()
                    row[j] = sg * (c - zg)
                    f.append(_f_direct(W[i:i + 1], row[None, :], X))
                f = np.array(f)
                assert f[sc[t, i, j]] <= f.min() + 1e-12 * max(1.0, abs(f.min())), (t, i, j)
    obj = r["obj"]
    assert np.all(np.diff(obj) <= 1e-12 * obj[:-1])
    direct = np.sum(((W - _levels_grouped(r["codes"], s, z, gsize)) @ X) ** 2, axis=1)
    assert np.allclose(r["obj_rows"][-1], direct, rtol=1e-10)
    assert np.allclose(O.objective_rows(W, r["codes"], s, z, S, group_size=gsize), direct, rtol=1e-10)
