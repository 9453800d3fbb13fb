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

SAMPLE_CODE_MATCH = 0.995

# (workload, sampled rows, free-running oracle run, fp64 recomputation of the whole
# objective).  For the 59392-wide layer one oracle run over the sampled rows takes
# minutes on the host, so there the teacher-forced replay alone carries the parity.
CASES = [
    ("llama7b_proj_4096x4096", 48, True, True),
    ("llama7b_up_11008x4096", 48, True, True),
    ("llama7b_down_4096x11008", 24, True, True),
    ("falcon180b_qkv_15360x14848", 15, True, True),
    ("falcon180b_down_14848x59392", 15, False, False),
]


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


def _objective_fp64(W, codes, scales, zeros, Sg, H=None):
    """f = sum_i d_i Sigma d_i^T with D = W - What (- H), in fp64 (proof of Lemma 1)."""
    What = scales.double()[:, None] * (codes.double() - zeros.double()[:, None])
    D = W.double() - What
    if H is not None:
        D -= H
    S = Sg.double()
    f = 0.0
    for r0 in range(0, D.shape[0], 2048):
        Dr = D[r0:r0 + 2048]
        f += float(torch.sum((Dr @ S) * Dr).item())
    return f


@pytest.mark.parametrize("name,nrows,free_run,full_obj", CASES, ids=[c[0] for c in CASES])
def test_fullsize_layer_sampled_rows(name, nrows, free_run, full_obj):
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
    rows = np.unique(np.concatenate([rng.choice(q, size=nrows, replace=False),
                                     [int(torch.argmax(W.abs().amax(dim=1)).item())]]))
    rows_t = torch.from_numpy(rows).cuda()
    W64 = W[rows_t].double().cpu().numpy()
    S32 = Sg.cpu().numpy()                                  # the GPU's Sigma, binary32
    for bits in cfg.bits:
        out = qe.qe_quantize_layer(W, Sg, bits, cfg.iters, workspace=ws, record_sweeps=True)
        assert qe.qe_sync_status() == qe.QE_OK
        obj = out["obj"].cpu().numpy()
        assert np.all(obj > 0) and np.all(np.diff(obj) <= 1e-6 * obj[:-1]), "objective not monotone"
        # grid: bit-identical on the sampled rows
        s, z = O.grid(W64, bits)
        assert np.array_equal(out["scales"][rows_t].cpu().numpy(), s)
        assert np.array_equal(out["zeros"][rows_t].cpu().numpy(), z)
        # teacher-forced decisions on the sampled rows
        sweep = out["sweep_codes"][:, rows_t, :].cpu().numpy()
        del out["sweep_codes"]
        _, _, forced = parity.teacher_forced(W64, S32, s, z, bits, sweep, want_run=True)
        # free-running oracle on the same rows.  The objective of the rows meets the
        # parity bar.  Codes: a decision within ~1e-7 grid steps of a midpoint (which
        # the teacher-forced check above accepts) can round either way and then
        # cascades along its row (tens of codes in a row of 11008); over a sample of
        # a few rows one such row weighs a lot, so the code match is a sanity bound
        # here (the whole-layer 99.9% bar is held by the oracle-sized tests).
        if free_run:
            ref = O.alg1(W64, S32, s, z, bits, cfg.iters)
            parity.check_obj(forced["obj"], ref["obj"], what="sampled-row objective (GPU codes vs oracle run)")
            m = parity.code_match(out["codes"][rows_t].cpu().numpy(), ref["codes"])
            assert m >= SAMPLE_CODE_MATCH, f"codes match {m:.5f} on the sampled rows"
        # the whole objective, recomputed in fp64 from the GPU's final codes
        if full_obj:
            f = _objective_fp64(W, out["codes"], out["scales"], out["zeros"], Sg)
            parity.check_obj(obj[-1], f, what="objective of the final codes (fp64)")
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
    f = _objective_fp64(W, out["codes"], out["scales"], out["zeros"], Sg, H.view(q, p))
    parity.check_obj(obj[-1], f, what="g of the final state (fp64)")
