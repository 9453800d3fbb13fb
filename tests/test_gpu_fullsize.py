"""GPU parity at the full workload sizes, in the launch configuration bench.py times.

The CUDA path runs exactly as in the benchmark: caller workspace, default
options, bf16 W and X of the synthetic workload.  Rows of W are independent
problems given Sigma (Sec. 3.2), so the fp64 oracle runs on a seeded sample
of rows (plus the row holding max |W|), fed the GPU's own Sigma (binary32,
promoted exactly).  Sigma itself is checked on sampled feature pairs against
binary64 dot products of the same bfloat16 X (Lemma 1).  What the sample
cannot show is checked through properties that hold at any size: exact
symmetry of Sigma, the non-increasing objective (Lemma 2), and the objective
of the GPU's final codes recomputed in fp64 where that is affordable.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2309_01885_gb300 import inputs
from paper_2309_01885_gb300 import qe
from tests import parity

pytestmark = pytest.mark.gpu
O = oracle.get()

# (workload, sampled rows).  The oracle runs Algorithm 1 free-running on the sample
# (about p^2 column updates per row and sweep on the host cores); the sizes keep
# each case within a few minutes on 16 host cores.
CASES = [
    ("llama7b_proj_4096x4096", 512),
    ("llama7b_up_11008x4096", 256),
    ("llama7b_down_4096x11008", 128),
    ("falcon180b_qkv_15360x14848", 64),
    ("falcon180b_down_14848x59392", 16),
]


def _log(rec: dict):
    """Append a parity record (what the sample reached) to $QE_PARITY_LOG, if set."""
    import json
    import os
    path = os.environ.get("QE_PARITY_LOG")
    if path:
        with open(path, "a") as fh:
            fh.write(json.dumps(rec) + "\n")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qe.load()
    yield
    torch.cuda.empty_cache()


def _bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _check_sigma_sampled(X, Sg, rng, nfeat=192, npairs=1536):
    """Exact symmetry everywhere; sampled entries within 1e-5 sqrt(S_aa S_bb) (binary64 oracle)."""
    p = X.shape[0]
    assert torch.equal(Sg, Sg.t()), "Sigma is not exactly symmetric"
    F = np.unique(np.concatenate([rng.choice(p, size=min(nfeat, p), replace=False), [0, p - 1]]))
    a = np.concatenate([np.arange(F.size), rng.integers(0, F.size, npairs)])
    b = np.concatenate([np.arange(F.size), rng.integers(0, F.size, npairs)])
    bits = _bf16_bits(X[torch.from_numpy(F).to(X.device)])
    ref = O.sigma_pairs_bf16(bits, a, b)
    Fa, Fb = torch.from_numpy(F[a]).cuda(), torch.from_numpy(F[b]).cuda()
    got = Sg[Fa, Fb].double().cpu().numpy()
    dref = O.sigma_pairs_bf16(bits, np.arange(F.size), np.arange(F.size))
    tol = 1e-5 * np.sqrt(dref[a] * dref[b])
    err = np.abs(got - ref)
    assert np.all(err <= tol), f"Sigma: max err/tol = {np.max(err / np.maximum(tol, 1e-300)):.3f}"


def _objective_full(W, codes, scales, zeros, Sg, H=None):
    """f = sum_i d_i Sigma d_i^T with D = W - What (- H) (proof of Lemma 1), from the
    final codes: binary64 products up to p = 16384; beyond that binary32 products
    (no TF32) summed in binary64, where GB300's low fp64 rate would take minutes
    (a relative error of about 1e-6 for these sums, far inside the 1e-4 bar)."""
    wide = Sg.shape[0] > 16384
    dt = torch.float32 if wide else torch.float64
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        S = Sg.to(dt)
        f = 0.0
        for r0 in range(0, W.shape[0], 1024):
            sl = slice(r0, r0 + 1024)
            What = scales[sl].double()[:, None] * (codes[sl].double() - zeros[sl].double()[:, None])
            D = W[sl].double() - What
            if H is not None:
                D -= H[sl]
            Dd = D.to(dt)
            f += float(torch.sum((Dd @ S).double() * D).item())
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    return f


@pytest.mark.parametrize("name,nrows", CASES, ids=[c[0] for c in CASES])
def test_fullsize_layer_sampled_rows(name, nrows):
    """Every benchmark layer in the bench configuration, against the free-running
    oracle on a row sample (plus the row of max |W|), fed the GPU's Sigma:
      * grids bit for bit;
      * each row's trajectory (codes after every sweep) against the oracle's; where a
        row diverges, its first differing decision lies within 1e-4 grid steps of a
        rounding midpoint (the state is shared up to there, so that is the
        teacher-forced check), and every later decision of that row passes the
        teacher-forced check on the GPU's own trajectory;
      * the sampled rows' objective after every sweep within 1e-4 relative;
      * codes >= 99.9% equal over the sample;
      * the reported objective against the objective of the final codes recomputed
        over the whole layer."""
    cfg = inputs.CONFIGS[name]
    q, p = cfg.q, cfg.p
    rng = np.random.default_rng(2309)
    W = inputs.layer_weights(q, p, dtype=cfg.w_dtype, seed=cfg.seed, device="cuda")
    X = inputs.calib_inputs(p, cfg.n, dtype=cfg.x_dtype, seed=cfg.seed, device="cuda",
                            heavy_frac=cfg.heavy_frac, heavy_mult=cfg.heavy_mult)
    Sg = qe.qe_build_sigma(X)
    torch.cuda.synchronize()
    _check_sigma_sampled(X, Sg, rng)
    del X
    ws = torch.empty(qe.qe_workspace_size(q, p), dtype=torch.uint8, device="cuda")
    wmax = int(torch.argmax(W.abs().amax(dim=1)).item())
    rows = np.unique(np.concatenate([rng.choice(q, size=nrows - 1, replace=False), [wmax]]))
    rows_t = torch.from_numpy(rows).cuda()
    W64 = W[rows_t].double().cpu().numpy()
    S32 = Sg.cpu().numpy()                                  # the GPU's Sigma, binary32
    for bits in cfg.bits:
        out = qe.qe_quantize_layer(W, Sg, bits, cfg.iters, workspace=ws, record_sweeps=True, record_forms=True)
        assert qe.qe_sync_status() == qe.QE_OK
        obj = out["obj"].cpu().numpy()
        assert np.all(obj > 0) and np.all(np.diff(obj) <= 1e-6 * obj[:-1]), "objective not monotone"
        s, z = O.grid(W64, bits)
        assert np.array_equal(out["scales"][rows_t].cpu().numpy(), s)
        assert np.array_equal(out["zeros"][rows_t].cpu().numpy(), z)
        sweep = out["sweep_codes"][:, rows_t, :].cpu().numpy()
        forms = out["sweep_forms"].tolist()
        del out["sweep_codes"]
        # free-running oracle with its trajectory and beta~ at every decision
        ref = O.alg1(W64, S32, s, z, bits, cfg.iters, record=True, want_beta=True)
        div = parity.first_divergence(sweep, ref, s, z, bits)
        obj_rows = ref["obj_rows"].copy()           # the GPU rows' objective, sweep by sweep
        if div:
            d = np.array([r for r, *_ in div])
            _, _, forced = parity.teacher_forced(W64[d], S32, s[d], z[d], bits, sweep[:, d], want_run=True)
            obj_rows[:, d] = forced["obj_rows"]
        del ref["beta"]
        parity.check_obj(obj_rows.sum(axis=1), ref["obj"], what="sampled-row objective per sweep")
        m = parity.code_match(sweep[-1], ref["codes"])
        cascades = [dict(row=int(rows[r]), sweep=t + 1, column=j, midpoint_dist=dist, codes_differing=nd)
                    for r, t, j, dist, nd in div]
        f = _objective_full(W, out["codes"], out["scales"], out["zeros"], Sg)
        # fraction of the sampled codes that changed in each sweep after the first
        chg = [float(np.mean(sweep[t] != sweep[t - 1])) for t in range(1, sweep.shape[0])]
        _log(dict(test="fullsize", workload=name, bits=bits, rows=int(rows.size), code_match=m, changed=chg,
                  obj_rel_err=float(np.max(np.abs(obj_rows.sum(axis=1) - ref["obj"]) / ref["obj"])),
                  full_obj_rel_err=abs(obj[-1] - f) / f, sweep_forms=forms, cascades=cascades))
        assert m >= parity.CODE_MATCH, f"codes match {m:.5f} on {rows.size} rows; cascades {cascades}"
        parity.check_obj(obj[-1], f, what="objective of the final codes over the whole layer")
        del out
        torch.cuda.empty_cache()


def test_fullsize_grouped_grids():
    """Grouped grids (groups of 256 columns) on the 4096 x 4096 projection in the bench
    configuration: per-group grids bit for bit on sampled rows, teacher-forced
    decisions and the sampled rows' objective against the oracle's grouped
    Algorithm 1 (fed the GPU's Sigma), a non-increasing objective, and the objective
    of the final codes recomputed in fp64."""
    cfg = inputs.CONFIGS["llama7b_proj_4096x4096"]
    q, p, G, bits = cfg.q, cfg.p, 256, 3
    rng = np.random.default_rng(2310)
    W = inputs.layer_weights(q, p, dtype=cfg.w_dtype, seed=cfg.seed, device="cuda")
    X = inputs.calib_inputs(p, cfg.n, dtype=cfg.x_dtype, seed=cfg.seed, device="cuda",
                            heavy_frac=cfg.heavy_frac, heavy_mult=cfg.heavy_mult)
    Sg = qe.qe_build_sigma(X)
    del X
    out = qe.qe_quantize_layer(W, Sg, bits, cfg.iters, record_sweeps=True, group_size=G)
    assert qe.qe_sync_status() == qe.QE_OK
    obj = out["obj"].cpu().numpy()
    assert np.all(np.diff(obj) <= 1e-6 * obj[:-1]), "objective not monotone"
    rows = np.sort(rng.choice(q, size=24, replace=False))
    rows_t = torch.from_numpy(rows).cuda()
    W64 = W[rows_t].double().cpu().numpy()
    S64 = Sg.double().cpu().numpy()
    s, z = O.grid(W64, bits, group_size=G)
    assert np.array_equal(out["scales"][rows_t].cpu().numpy(), s)
    assert np.array_equal(out["zeros"][rows_t].cpu().numpy(), z)
    sweep = out["sweep_codes"][:, rows_t, :].cpu().numpy()
    _, _, forced = parity.teacher_forced(W64, S64, s, z, bits, sweep, want_run=True, group_size=G)
    ref = O.alg1(W64, S64, s, z, bits, cfg.iters, group_size=G)
    parity.check_obj(forced["obj"], ref["obj"], what="sampled-row objective (groups)")
    # the whole objective of the final codes in fp64
    g = torch.arange(p, device="cuda") // G
    sc, zc = out["scales"].double()[:, g], out["zeros"].double()[:, g]
    D = W.double() - sc * (out["codes"].double() - zc)
    f = sum(float(torch.sum((D[r0:r0 + 2048] @ Sg.double()) * D[r0:r0 + 2048]).item()) for r0 in range(0, q, 2048))
    parity.check_obj(obj[-1], f, what="objective of the final codes (fp64, groups)")


@pytest.mark.parametrize("rows,structured", [(256, False), (128, True)], ids=["entries", "columns"])
def test_fullsize_outlier_oracle(rows, structured):
    """The outlier-aware variant (Algorithm 4) through its full-size paths against the
    oracle: the first `rows` rows of the 4096 x 4096 outlier workload (its planted
    entries, Sigma from its 262144 tokens), 3 bits, s = 1% of the slice's entries
    (structured: floor(s / q) whole columns), 20 iterations, the library's default
    64 power steps on both sides; the oracle is fed the GPU's Sigma.
      * teacher-forced, iteration by iteration from the GPU's own state (its codes and
        H after the previous iteration, taken from runs stopped there): every CD
        decision is the nearest level of the fp64 beta~ unless within 1e-4 of a
        midpoint, and the oracle's IHT step keeps the GPU's support with the GPU's
        values within 1e-5 of max |T| (one fp32 step from a shared state);
      * free-running (entries): g after every CD half and after every IHT step within
        1e-4, the support, H on the common support, codes >= 99.9%."""
    cfg = inputs.CONFIGS["llama7b_proj_outlier_4096x4096"]
    p, bits, iters = cfg.p, cfg.bits[0], cfg.iters
    W = cfg.weights("cuda")[:rows].contiguous()
    X = cfg.inputs("cuda")
    Sg = qe.qe_build_sigma(X)
    del X
    s_budget = int(round(cfg.outlier_budget_frac * rows * p))
    runs = []
    for k in range(1, iters + 1):       # H after every iteration: runs stopped there
        runs.append(qe.qe_quantize_layer_outlier(W, Sg, bits, k, s_budget, structured=structured,
                                                 record_sweeps=(k == iters)))
    assert qe.qe_sync_status() == qe.QE_OK
    out = runs[-1]
    for o in runs[:-1]:                 # a run stopped early is a prefix of the full run
        k = o["obj"].numel()
        assert torch.equal(o["obj"], out["obj"][:k]) and torch.equal(o["obj_cd"], out["obj_cd"][:k])
    W64, S64 = parity.f64(W), parity.f64(Sg)
    if structured:
        cols = O.topk_columns(W64, s_budget // rows)
        H0 = np.zeros_like(W64)
        H0[:, cols] = W64[:, cols]
        excl = (H0 != 0).astype(np.uint8)
        excl[:, cols] = 1
    else:
        k0 = O.topk(W64, s_budget)
        H0 = np.zeros(W64.size)
        H0[k0] = W64.ravel()[k0]
        H0 = H0.reshape(W64.shape)
        excl = np.zeros(W64.size, np.uint8)
        excl[k0] = 1
        excl = excl.reshape(W64.shape)
    s, z = O.grid(W64, bits, excl)
    assert np.array_equal(out["scales"].cpu().numpy(), s)
    assert np.array_equal(out["zeros"].cpu().numpy(), z)
    eta = 1.0 / (2.0 * O.power_lambda(S64, 64))
    sweep = out["sweep_codes"].cpu().numpy()
    nnz = [int(o["H_nnz"].item()) for o in runs]
    hidx = [o["H_idx"][:m].cpu().numpy() for o, m in zip(runs, nnz)]
    hval = [o["H_val"][:m].cpu().numpy() for o, m in zip(runs, nnz)]
    ties = parity.outlier_replay(W64, S64, s, z, bits, sweep, hidx, hval, H0, eta, s_budget, structured)
    rec = dict(test="fullsize_outlier", rows=rows, structured=structured, support_ties=ties)
    if not structured:
        ref = O.outlier(W64, S64, bits, iters, s_budget, 64)
        parity.check_obj(out["obj_cd"].cpu().numpy(), ref["obj_cd"], what="g after CD")
        parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="g after IHT")
        m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
        ref_idx = np.flatnonzero(ref["H"].ravel())
        common = np.intersect1d(hidx[-1], ref_idx)
        Hd = np.zeros(W64.size)
        Hd[hidx[-1]] = hval[-1]
        herr = float(np.max(np.abs(Hd[common] - ref["H"].ravel()[common])) / np.abs(ref["H"]).max())
        rec.update(code_match=m, support_common=int(common.size), nnz=nnz[-1], nnz_oracle=int(ref["nnz"]),
                   h_err_rel_max=herr,
                   obj_rel_err=float(np.max(np.abs(out["obj"].cpu().numpy() - ref["obj"]) / ref["obj"])))
        _log(rec)
        assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"
        assert nnz[-1] == ref["nnz"] and common.size >= 0.999 * nnz[-1]
        assert herr <= 1e-4, f"H on the common support off by {herr:.3e} of max |H|"
    else:
        _log(rec)


@pytest.mark.parametrize("name,structured", [("llama7b_proj_outlier_4096x4096", False),
                                             ("llama7b_proj_outlier_4096x4096", True),
                                             ("llama7b_proj_outlier2b_4096x4096", False)],
                         ids=["3bit-entries", "3bit-columns", "2bit-entries"])
def test_fullsize_outlier_properties(name, structured):
    """The outlier-aware workload at full size.  The IHT support is a global
    top-s (Eq. iht-update), so rows are not independent here: the sampled-row
    check covers the grid (W without the initial support P_s(W), Sec. 4.3);
    the rest are properties: the budget, sorted unique indices, Lemma 3 (the
    IHT half never increases g), a non-increasing g, and g of the final state
    recomputed in fp64."""
    cfg = inputs.CONFIGS[name]
    q, p = cfg.q, cfg.p
    W = cfg.weights("cuda")
    X = cfg.inputs("cuda")
    Sg = qe.qe_build_sigma(X)
    del X
    bits = cfg.bits[0]
    out = qe.qe_quantize_layer_outlier(W, Sg, bits, cfg.iters, cfg.s_budget, structured=structured)
    assert qe.qe_sync_status() == qe.QE_OK
    nnz = int(out["H_nnz"].item())
    assert 0 < nnz <= cfg.s_budget
    if structured:   # whole columns, floor(s / q) of them
        assert nnz == q * (cfg.s_budget // q)
        assert np.unique(out["H_idx"][:nnz].cpu().numpy() % p).size == cfg.s_budget // q
    idx = out["H_idx"][:nnz].cpu().numpy()
    assert np.all(np.diff(idx) > 0) and idx[0] >= 0 and idx[-1] < q * p
    obj, obj_cd = out["obj"].cpu().numpy(), out["obj_cd"].cpu().numpy()
    assert np.all(obj <= obj_cd * (1 + 1e-6)), "IHT step increased g (Lemma 3)"
    assert np.all(np.diff(obj[1:]) <= 1e-6 * obj[1:-1])
    # grid on sampled rows, from W without P_s(W)
    W64 = W.double().cpu().numpy()
    excl = np.zeros(q * p, np.uint8)
    if structured:
        excl.reshape(q, p)[:, O.topk_columns(W64, cfg.s_budget // q)] = 1
    else:
        excl[O.topk(W64, cfg.s_budget)] = 1
    rows = np.random.default_rng(5).choice(q, size=64, replace=False)
    s, z = O.grid(W64[rows], bits, excl.reshape(q, p)[rows])
    rows_t = torch.from_numpy(rows).cuda()
    assert np.array_equal(out["scales"][rows_t].cpu().numpy(), s)
    assert np.array_equal(out["zeros"][rows_t].cpu().numpy(), z)
    # g of the final state
    H = torch.zeros(q * p, dtype=torch.float64, device="cuda")
    H[out["H_idx"][:nnz]] = out["H_val"][:nnz].double()
    f = _objective_full(W, out["codes"], out["scales"], out["zeros"], Sg, H.view(q, p))
    parity.check_obj(obj[-1], f, what="g of the final state (fp64)")
