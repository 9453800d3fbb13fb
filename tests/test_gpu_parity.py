"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Sizes here run in seconds on the oracle and span several GEMM tiles, several
64-column CD blocks and ragged tails.  Full-size workloads are in
test_gpu_fullsize.py.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2309_01885_gb300 import inputs
from paper_2309_01885_gb300 import qe
from tests import parity

pytestmark = pytest.mark.gpu
O = oracle.get()


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qe.load()


def _sigma_check(Sg, X64):
    S64 = O.sigma(X64)
    Sg64 = parity.f64(Sg)
    assert np.array_equal(Sg64, Sg64.T), "Sigma is not exactly symmetric"
    dg = np.sqrt(np.outer(np.diag(S64), np.diag(S64)))
    err = np.abs(Sg64 - S64)
    tol = 1e-5 * np.maximum(dg, 1e-30)
    assert np.all(err <= tol), f"Sigma: max err/tol = {np.max(err / tol):.3f}"
    return S64


# ---------------------------------------------------------------------------
# Sigma = X X^T
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("p,n", [(200, 1000), (384, 4096), (130, 70), (640, 3000)])
def test_sigma_bf16_feature_major(p, n):
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=1, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    torch.cuda.synchronize()
    _sigma_check(Sg, parity.f64(X))


def test_sigma_bf16_token_major_and_accumulate():
    p, n = 272, 5000
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=2, device="cuda", heavy_frac=0.02,
                            heavy_mult=20.0)
    Xt = X.t().contiguous()                      # n x p, token-major
    Sg = qe.qe_build_sigma(Xt, layout=qe.QE_TOKEN_MAJOR)
    torch.cuda.synchronize()
    _sigma_check(Sg, parity.f64(X))
    # Sigma over the token stream in two chunks equals Sigma of the whole
    S2 = qe.qe_build_sigma(X[:, :3000].contiguous())
    qe.qe_build_sigma(X[:, 3000:].contiguous(), Sigma=S2, accumulate=True)
    torch.cuda.synchronize()
    _sigma_check(S2, parity.f64(X))


@pytest.mark.parametrize("accumulate", [False, True])
def test_sigma_two_waves(accumulate):
    """p = 3584 has 210 tiles on or above the diagonal, more than one wave on 152 SMs,
    with heavy features; direct and accumulated over two token halves.  Sampled
    entries against binary64 dot products of the same bf16 X (Lemma 1), exact
    symmetry, every diagonal entry."""
    p, n = 3584, 1536
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=5, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    if accumulate:
        Sg = qe.qe_build_sigma(X[:, :768].contiguous())
        qe.qe_build_sigma(X[:, 768:].contiguous(), Sigma=Sg, accumulate=True)
    else:
        Sg = qe.qe_build_sigma(X)
    torch.cuda.synchronize()
    assert qe.qe_sync_status() == qe.QE_OK
    assert torch.equal(Sg, Sg.t())
    rng = np.random.default_rng(6)
    bits = X.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    a = np.concatenate([np.arange(p), rng.integers(0, p, 6000), np.arange(p - 300, p)])
    b = np.concatenate([np.arange(p), rng.integers(0, p, 6000), rng.integers(0, p, 300)])
    ref = O.sigma_pairs_bf16(bits, a, b)
    got = Sg[torch.from_numpy(a).cuda(), torch.from_numpy(b).cuda()].double().cpu().numpy()
    d = ref[:p]
    tol = 1e-5 * np.sqrt(d[a] * d[b])
    assert np.all(np.abs(got - ref) <= tol), f"max err/tol {np.max(np.abs(got - ref) / tol):.3f}"


def test_sigma_host_streamed():
    """Sigma from pinned host X streamed in token chunks (ragged last chunk), the
    staging area reused by the next calls, and accumulation over two token ranges
    given as strided views of the host array."""
    p, n, chunk = 384, 5000, 1024
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=4, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Xh = X.cpu().pin_memory()
    staging = qe.sigma_host_staging(p, chunk)
    S = torch.empty(p, p, dtype=torch.float32, device="cuda")
    qe.qe_build_sigma_host(Xh, S, staging, chunk)
    S2 = torch.empty_like(S)
    qe.qe_build_sigma_host(Xh[:, :2000], S2, staging, chunk)
    qe.qe_build_sigma_host(Xh[:, 2000:], S2, staging, chunk, accumulate=True)
    torch.cuda.synchronize()
    assert qe.qe_sync_status() == qe.QE_OK
    X64 = parity.f64(X)
    _sigma_check(S, X64)
    _sigma_check(S2, X64)
    Sd = qe.qe_build_sigma(X)
    torch.cuda.synchronize()
    rel = (S.double() - Sd.double()).abs().max() / Sd.double().abs().max()
    assert rel.item() < 1e-6


def test_sigma_host_buffers_rotate_across_calls():
    """One chunk per call and two buffers: consecutive calls copy into the buffers in
    turn (the next call's copy overlaps this call's GEMM), with no synchronization in
    between; each Sigma is that of its own X."""
    p, n = 256, 4096
    Xs = [inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=40 + k, device="cuda", heavy_frac=0.02,
                              heavy_mult=30.0) for k in range(3)]
    hosts = [X.cpu().pin_memory() for X in Xs]
    staging = qe.sigma_host_staging(p, n, nbuf=2)
    outs = [torch.empty(p, p, dtype=torch.float32, device="cuda") for _ in Xs]
    for Xh, S in zip(hosts, outs):
        qe.qe_build_sigma_host(Xh, S, staging, n)
    torch.cuda.synchronize()
    assert qe.qe_sync_status() == qe.QE_OK
    for X, S in zip(Xs, outs):
        assert torch.equal(S, qe.qe_build_sigma(X))


@pytest.mark.parametrize("layout", [qe.QE_FEATURE_MAJOR, qe.QE_TOKEN_MAJOR])
def test_sigma_fp32(layout):
    p, n = 150, 777
    X = inputs.calib_inputs(p, n, dtype=torch.float32, seed=3, device="cuda", heavy_frac=0.02,
                            heavy_mult=20.0)
    src = X if layout == qe.QE_FEATURE_MAJOR else X.t().contiguous()
    Sg = qe.qe_build_sigma(src, layout=layout)
    torch.cuda.synchronize()
    _sigma_check(Sg, parity.f64(X))


# ---------------------------------------------------------------------------
# qe_quantize_layer
# ---------------------------------------------------------------------------
def _layer_case(q, p, n, w_dtype, bits, iters, seed, corr_rank=0, zero_rows=(), w_outlier=0.0):
    W = inputs.layer_weights(q, p, dtype=w_dtype, seed=seed, device="cuda",
                             w_outlier_frac=w_outlier, w_outlier_mult=10.0)
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=seed, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0, corr_rank=corr_rank,
                            zero_rows=zero_rows)
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, bits, iters, record_sweeps=True, want_norm=True)
    assert qe.qe_sync_status() == qe.QE_OK
    return W, X, Sg, out


def _check_layer(W, Sg, out, bits, iters, init_codes=None, free_running=True):
    """Teacher-forced decisions and the objective of the GPU's own state always
    meet the parity bar.  The free-running oracle trajectory meets it on
    uncorrelated inputs; on strongly correlated inputs one legitimate
    near-midpoint flip cascades through the row, so there it is only held to
    a sanity bound (free_running=False)."""
    W64 = parity.f64(W)
    S64 = parity.f64(Sg)                      # the same Sigma on both sides
    wx = float(np.einsum("ij,jk,ik->", W64, S64, W64))   # ||W X||^2
    atol = 1e-7 * wx
    s, z = parity.check_grid(out["scales"], out["zeros"], W64, bits)
    sweep = out["sweep_codes"].cpu().numpy()
    # teacher-forced: every decision is the nearest level of the fp64 beta~
    nbad, ntot = parity.teacher_forced(W64, S64, s, z, bits, sweep, init_codes=init_codes)
    # objective of the GPU's own state, fp64
    forced = O.alg1(W64, S64, s, z, bits, iters, init_codes=init_codes, forced=sweep)
    parity.check_obj(out["obj"].cpu().numpy(), forced["obj"], what="objective (GPU state)", atol=atol)
    # free-running oracle
    ref = O.alg1(W64, S64, s, z, bits, iters, init_codes=init_codes)
    m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
    if free_running:
        parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="objective (free-running)", atol=atol)
        assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"
    else:
        parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], rtol=2e-2, atol=atol,
                         what="objective (free-running, correlated input)")
        assert m >= 0.9, f"codes match {m:.5f}"
    assert abs(out["wx_norm2"].item() - wx) <= 1e-4 * wx
    return nbad, ntot


@pytest.mark.parametrize("corr_rank", [0, 4])
@pytest.mark.parametrize("w_dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("bits", [3, 4])
def test_layer_parity_small(w_dtype, bits, corr_rank):
    W, X, Sg, out = _layer_case(200, 300, 2048, w_dtype, bits, 4, seed=bits, corr_rank=corr_rank)
    _check_layer(W, Sg, out, bits, 4, free_running=corr_rank == 0)
    # objective non-increasing after the first sweep (Lemma 2)
    obj = out["obj"].cpu().numpy()
    assert np.all(np.diff(obj) <= 1e-6 * obj[:-1])


@pytest.mark.parametrize("block_width", [64, 128, 256])
def test_layer_parity_multi_tile_ragged(block_width):
    W = inputs.layer_weights(300, 520, dtype=torch.bfloat16, seed=11, device="cuda")
    X = inputs.calib_inputs(520, 4096, dtype=torch.bfloat16, seed=11, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0, corr_rank=8)
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, 3, 3, record_sweeps=True, want_norm=True,
                               block_width=block_width)
    assert qe.qe_sync_status() == qe.QE_OK
    _check_layer(W, Sg, out, 3, 3, free_running=False)


@pytest.mark.parametrize("dense_sweeps", [1, 2, 100])
@pytest.mark.parametrize("block_width,corr_rank", [(64, 8), (256, 0)])
def test_layer_correction_forms(dense_sweeps, block_width, corr_rank):
    """The cross-block term from the dense tensor-core GEMM (sweeps <= dense_sweeps)
    and from the per-row change lists (later sweeps) both meet the parity bar:
    lists from sweep 2, from sweep 3, and never.  p = 520 leaves a ragged last
    block (8 columns at B = 64, 8 at B = 256)."""
    iters = 6
    W = inputs.layer_weights(260, 520, dtype=torch.bfloat16, seed=61, device="cuda")
    X = inputs.calib_inputs(520, 4096, dtype=torch.bfloat16, seed=61, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0, corr_rank=corr_rank)
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, 3, iters, record_sweeps=True, want_norm=True,
                               block_width=block_width, dense_sweeps=dense_sweeps)
    assert qe.qe_sync_status() == qe.QE_OK
    _check_layer(W, Sg, out, 3, iters, free_running=corr_rank == 0)
    obj = out["obj"].cpu().numpy()
    assert np.all(np.diff(obj) <= 1e-6 * obj[:-1])


def test_layer_lists_agree_with_dense():
    """Both forms of the cross-block term reach the same codes and objective
    (uncorrelated inputs, where no near-midpoint cascade is expected)."""
    W = inputs.layer_weights(384, 640, dtype=torch.bfloat16, seed=62, device="cuda")
    X = inputs.calib_inputs(640, 8192, dtype=torch.bfloat16, seed=62, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    a = qe.qe_quantize_layer(W, Sg, 4, 8, dense_sweeps=100)
    b = qe.qe_quantize_layer(W, Sg, 4, 8, dense_sweeps=1)
    assert qe.qe_sync_status() == qe.QE_OK
    parity.check_obj(b["obj"].cpu().numpy(), a["obj"].cpu().numpy(), what="lists vs dense")
    m = parity.code_match(a["codes"].cpu().numpy(), b["codes"].cpu().numpy())
    assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"


@pytest.mark.parametrize("corr_rank,group_size,dense", [(0, 0, 0), (4, 0, 0), (0, 256, 0), (4, 0, 100)],
                         ids=["plain", "correlated", "groups", "dense-window"])
def test_near_tie_refinement(corr_rank, group_size, dense):
    """With the near-tie refinement (the default), every GPU decision is the nearest
    level of the binary64 beta~ of the GPU's own state: the teacher-forced replay
    finds no disagreement at all, not even within the 1e-4 midpoint tolerance, and
    the trajectory matches the free-running oracle code for code.  With it off the
    same run stays within the tolerance.  Sweep 1 (sequential kernel), the change
    lists, the dense window and grouped grids all decide near-ties this way."""
    q, p, bits, iters = 160, 520, 4, 6
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=81, device="cuda")
    X = inputs.calib_inputs(p, 4096, dtype=torch.bfloat16, seed=81, device="cuda", heavy_frac=0.01,
                            heavy_mult=30.0, corr_rank=corr_rank)
    Sg = qe.qe_build_sigma(X)
    kw = dict(record_sweeps=True, group_size=group_size, dense_sweeps=dense)
    out = qe.qe_quantize_layer(W, Sg, bits, iters, **kw)
    off = qe.qe_quantize_layer(W, Sg, bits, iters, tie_eps=-1.0, **kw)
    assert qe.qe_sync_status() == qe.QE_OK
    W64, S64 = parity.f64(W), parity.f64(Sg)
    s, z = O.grid(W64, bits, group_size=group_size)
    assert np.array_equal(out["scales"].cpu().numpy(), s)
    sweep = out["sweep_codes"].cpu().numpy()
    nbad, ntot = parity.teacher_forced(W64, S64, s, z, bits, sweep, group_size=group_size)
    assert nbad == 0, f"{nbad} of {ntot} decisions off the binary64 nearest level"
    ref = O.alg1(W64, S64, s, z, bits, iters, group_size=group_size, record=True)
    assert np.array_equal(sweep, ref["sweep_codes"])
    parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="objective with refinement")
    parity.teacher_forced(W64, S64, s, z, bits, off["sweep_codes"].cpu().numpy(), group_size=group_size)


@pytest.mark.parametrize("group_size", [0, 256])
def test_layer_adaptive_schedule(group_size):
    """The adaptive sweep schedule (dense form until a sweep changes fewer than
    switch_below codes, then the change lists, chosen on the device): with a
    threshold no sweep reaches it is the all-dense schedule bit for bit; with one
    every sweep reaches it switches after sweep 2 and is the dense_sweeps = 2
    schedule bit for bit (one list launch per sweep against one for all); with a
    threshold between the two it switches mid-way and meets the parity bar
    against the oracle (teacher-forced decisions, objectives, codes).  p = 1000
    leaves a ragged last block."""
    q, p, iters, bits = 200, 1000, 8, 3
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=63, device="cuda")
    X = inputs.calib_inputs(p, 8192, dtype=torch.bfloat16, seed=63, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    kw = dict(record_sweeps=True, group_size=group_size, record_forms=True)
    dense_all = qe.qe_quantize_layer(W, Sg, bits, iters, dense_sweeps=100, **kw)
    never = qe.qe_quantize_layer(W, Sg, bits, iters, switch_below=1, **kw)
    dense2 = qe.qe_quantize_layer(W, Sg, bits, iters, dense_sweeps=2, **kw)
    always = qe.qe_quantize_layer(W, Sg, bits, iters, switch_below=q * p, **kw)
    assert qe.qe_sync_status() == qe.QE_OK
    changes = [int((dense_all["sweep_codes"][t] != dense_all["sweep_codes"][t - 1]).sum().item())
               for t in range(1, iters)]
    assert all(c > 0 for c in changes), changes      # switch_below = 1 never switches
    for x, y in ((never, dense_all), (always, dense2)):
        for key in ("codes", "obj", "sweep_codes", "sweep_forms"):
            assert torch.equal(x[key], y[key]), key
    assert dense_all["sweep_forms"].tolist() == [0] + [1] * (iters - 1)
    assert dense2["sweep_forms"].tolist() == [0, 1] + [2] * (iters - 2)
    # the fourth sweep's count as the threshold: dense at least through sweep 5, lists
    # from the sweep after the first one that changes fewer codes
    mid = changes[2]
    out = qe.qe_quantize_layer(W, Sg, bits, iters, switch_below=mid, want_norm=True, **kw)
    assert qe.qe_sync_status() == qe.QE_OK
    forms = out["sweep_forms"].tolist()
    assert forms[:5] == [0, 1, 1, 1, 1] and forms == sorted(forms), forms
    if group_size:
        W64 = parity.f64(W)
        S64 = parity.f64(Sg)
        s, z = O.grid(W64, bits, group_size=group_size)
        assert np.array_equal(out["scales"].cpu().numpy(), s)
        sweep = out["sweep_codes"].cpu().numpy()
        parity.teacher_forced(W64, S64, s, z, bits, sweep, group_size=group_size)
        ref = O.alg1(W64, S64, s, z, bits, iters, group_size=group_size)
        parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="adaptive, groups")
    else:
        _check_layer(W, Sg, out, bits, iters, free_running=True)
    obj = out["obj"].cpu().numpy()
    assert np.all(np.diff(obj) <= 1e-6 * obj[:-1])


@pytest.mark.parametrize("p,group_size", [(640, 0), (1000, 0), (1000, 256)])
def test_layer_list_modes_identical(p, group_size):
    """The list sweeps in lockstep (shared packed Sigma_bar block, lists read from
    global memory) and row by row (coupling rows from global Sigma_bar, the window
    held in registers while it fits one entry per lane) take the same decisions in
    the same order: codes, every sweep's codes and the objective are identical.
    p = 1000 ends on a ragged block; with grouped grids every change is scaled into
    the block's group the same way in both modes."""
    q = 512
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=63, device="cuda")
    X = inputs.calib_inputs(p, 8192, dtype=torch.bfloat16, seed=63, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    runs = [qe.qe_quantize_layer(W, Sg, 3, 12, record_sweeps=True, free_changes=f, group_size=group_size)
            for f in (-1, 0, 100000)]
    assert qe.qe_sync_status() == qe.QE_OK
    ref = runs[0]
    for r in runs[1:]:
        assert torch.equal(r["codes"], ref["codes"])
        assert torch.equal(r["sweep_codes"], ref["sweep_codes"])
        assert torch.equal(r["obj"], ref["obj"])
    # the late sweeps change few codes per row, so the register window is in use
    sc = ref["sweep_codes"]
    late = (sc[-1] != sc[-2]).sum(dim=1)
    assert int(late.max()) <= 32


@pytest.mark.parametrize("relax,w_dtype,zero_rows", [(3, torch.bfloat16, ()), (2, torch.float32, (5,)),
                                                     (1, torch.bfloat16, ())])
def test_layer_relax_heuristic(relax, w_dtype, zero_rows):
    """The relax heuristic of Sec. 3.2 against the oracle's Algorithm 1 with the same
    period: the objective after every sweep (relaxed ones: f of the real-valued
    weights), the codes after every sweep (relaxed ones: their nearest levels) and
    the final codes.  A relaxed sweep minimizes f exactly along each coordinate, so
    it never increases f.  p = 300 ends on a ragged block; a zero row of X makes a
    dead column, which stays on its level."""
    q, p, n, bits, iters = 160, 300, 2048, 3, 7
    W = inputs.layer_weights(q, p, dtype=w_dtype, seed=64 + relax, device="cuda")
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=64 + relax, device="cuda",
                            heavy_frac=0.01, heavy_mult=30.0, zero_rows=zero_rows)
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, bits, iters, record_sweeps=True, want_norm=True, relax_period=relax)
    assert qe.qe_sync_status() == qe.QE_OK
    W64, S64 = parity.f64(W), parity.f64(Sg)
    wx = float(np.einsum("ij,jk,ik->", W64, S64, W64))
    s, z = parity.check_grid(out["scales"], out["zeros"], W64, bits)
    ref = O.alg1(W64, S64, s, z, bits, iters, record=True, relax_period=relax)
    obj = out["obj"].cpu().numpy()
    parity.check_obj(obj, ref["obj"], what="objective with relaxed sweeps", atol=1e-7 * wx)
    sweep = out["sweep_codes"].cpu().numpy()
    for t in range(iters):
        m = parity.code_match(sweep[t], ref["sweep_codes"][t])
        assert m >= 0.995, f"sweep {t + 1}: codes match {m:.5f}"
    m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
    assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"
    for t in range(1, iters - 1):
        if (t + 1) % relax == 0:
            assert obj[t] <= obj[t - 1] * (1 + 1e-6) + 1e-9 * wx, f"relaxed sweep {t + 1} increased f"


def test_layer_relax_period_not_below_iters_is_plain():
    W, X, Sg, out = _layer_case(96, 200, 1024, torch.bfloat16, 4, 5, seed=65)
    r = qe.qe_quantize_layer(W, Sg, 4, 5, record_sweeps=True, relax_period=5)
    assert qe.qe_sync_status() == qe.QE_OK
    assert torch.equal(r["sweep_codes"], out["sweep_codes"])
    assert torch.equal(r["obj"], out["obj"])


@pytest.mark.parametrize("bits", [1, 2, 3, 4, 5, 7, 8])
def test_pack_codes_bit_exact(bits):
    """Packed codes equal the oracle's bit stream byte for byte (ragged rows: p = 1001),
    and unpacking gives the codes back; also for the codes of a quantized layer."""
    q, p = 37, 1001
    g = torch.Generator(device="cuda").manual_seed(bits)
    codes = torch.randint(0, 2 ** bits, (q, p), dtype=torch.uint8, device="cuda", generator=g)
    packed = qe.qe_pack_codes(codes, bits)
    assert np.array_equal(packed.cpu().numpy(), oracle.pack_codes(codes.cpu().numpy(), bits))
    assert torch.equal(qe.qe_unpack_codes(packed, p, bits), codes)
    if bits in (2, 3, 4):
        W, X, Sg, out = _layer_case(64, 300, 1024, torch.bfloat16, bits, 2, seed=66)
        pk = qe.qe_pack_codes(out["codes"], bits)
        assert np.array_equal(pk.cpu().numpy(), oracle.pack_codes(out["codes"].cpu().numpy(), bits))
        assert torch.equal(qe.qe_unpack_codes(pk, 300, bits), out["codes"])


def _threshold_input(kind, N, seed):
    rng = np.random.default_rng(seed)
    if kind == "normal":
        return rng.standard_normal(N).astype(np.float32)
    if kind == "ties":           # few distinct magnitudes: the threshold falls inside a tie group
        return rng.integers(-50, 51, N).astype(np.float32)
    if kind == "sparse":         # mostly exact zeros (and a few -0.0): s may exceed the nonzeros
        T = rng.standard_normal(N).astype(np.float32)
        T[rng.random(N) < 0.97] = 0.0
        T[rng.random(N) < 0.01] = -0.0
        return T
    if kind == "wide":           # 70 decades, denormals included
        return (rng.standard_normal(N) * 10.0 ** rng.uniform(-44, 26, N)).astype(np.float32)
    raise ValueError(kind)


@pytest.mark.parametrize("kind,N,frac", [("normal", 10007, 0.01), ("normal", 10007, 1.0), ("ties", 50001, 0.013),
                                         ("sparse", 40000, 0.05), ("wide", 30011, 0.3),
                                         ("ties", 3_000_003, 0.01), ("normal", (1 << 24) + 3, 0.01)])
def test_hard_threshold_bit_exact(kind, N, frac):
    """P_s (Eq. iht-update) on its own against the oracle's: the kept indices and values
    bit for bit, ties at the threshold to the smaller index across many compaction
    chunks, zeros never kept; also from a T that is not 16-byte aligned."""
    T = _threshold_input(kind, N + 1, seed=N % 1000 + 70)
    s = int(round(frac * N))
    Tg = torch.from_numpy(T).cuda()
    for view, Th in ((Tg[:N], T[:N]), (Tg[1:], T[1:])):
        idx, val = qe.qe_hard_threshold(view, s)
        want = O.topk(Th.astype(np.float64), s)
        got = idx.cpu().numpy()
        assert got.shape == want.shape and np.array_equal(got, want), kind
        assert np.array_equal(val.cpu().numpy().view(np.uint32), Th[want].view(np.uint32))


def test_hard_threshold_degenerate():
    """s = 0, all-zero T, s = N, N = 1 and N = 3 (no 16-byte body)."""
    T = torch.zeros(1000, device="cuda")
    assert qe.qe_hard_threshold(T, 0)[0].numel() == 0
    assert qe.qe_hard_threshold(T, 1000)[0].numel() == 0
    for N in (1, 3, 17):
        Th = np.arange(1, N + 1, dtype=np.float32)[::-1].copy() * np.float32(-1.5)
        for s in range(N + 1):
            idx, val = qe.qe_hard_threshold(torch.from_numpy(Th).cuda(), s)
            assert np.array_equal(idx.cpu().numpy(), O.topk(Th.astype(np.float64), s))
            assert np.array_equal(val.cpu().numpy(), Th[idx.cpu().numpy()])


@pytest.mark.parametrize("block_width,group_size", [(256, 256), (128, 128), (128, 256)])
def test_layer_grouped_grids(block_width, group_size):
    """Grouped grids (one grid per row and group of columns) against the oracle's
    grouped Algorithm 1: the per-group scales and zero-points bit for bit,
    teacher-forced decisions, the objective of the GPU's own state and the
    free-running objective and codes.  Groups differ in range by a factor 6; p =
    704 ends on a ragged group."""
    q, p, bits, iters = 160, 704, 3, 4
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=67, device="cuda")
    W[:, 256:384] *= 6.0
    X = inputs.calib_inputs(p, 4096, dtype=torch.bfloat16, seed=67, device="cuda", heavy_frac=0.01,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, bits, iters, record_sweeps=True, block_width=block_width,
                               group_size=group_size)
    assert qe.qe_sync_status() == qe.QE_OK
    W64, S64 = parity.f64(W), parity.f64(Sg)
    wx = float(np.einsum("ij,jk,ik->", W64, S64, W64))
    s, z = O.grid(W64, bits, group_size=group_size)
    assert out["scales"].shape == (q, -(-p // group_size))
    assert np.array_equal(out["scales"].cpu().numpy(), s) and np.array_equal(out["zeros"].cpu().numpy(), z)
    sweep = out["sweep_codes"].cpu().numpy()
    parity.teacher_forced(W64, S64, s, z, bits, sweep, group_size=group_size)
    forced = O.alg1(W64, S64, s, z, bits, iters, forced=sweep, group_size=group_size)
    parity.check_obj(out["obj"].cpu().numpy(), forced["obj"], what="objective (GPU state, groups)",
                     atol=1e-7 * wx)
    ref = O.alg1(W64, S64, s, z, bits, iters, group_size=group_size)
    parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="objective (free-running, groups)",
                     atol=1e-7 * wx)
    m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
    assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"


def test_layer_group_of_all_columns_is_the_plain_layer():
    W, X, Sg, out = _layer_case(96, 300, 1024, torch.bfloat16, 4, 3, seed=68)
    r = qe.qe_quantize_layer(W, Sg, 4, 3, record_sweeps=True, group_size=512)
    assert qe.qe_sync_status() == qe.QE_OK
    assert r["scales"].shape == (96,)
    assert torch.equal(r["sweep_codes"], out["sweep_codes"]) and torch.equal(r["obj"], out["obj"])


def test_layer_dead_columns_round_to_nearest():
    dead = (5, 77, 130)
    W, X, Sg, out = _layer_case(96, 160, 1024, torch.float32, 4, 3, seed=12, zero_rows=dead)
    _check_layer(W, Sg, out, 4, 3)
    W64 = parity.f64(W)
    rtn = O.rtn(W64, out["scales"].cpu().numpy(), out["zeros"].cpu().numpy(), 4)
    codes = out["codes"].cpu().numpy()
    for j in dead:
        assert np.array_equal(codes[:, j], rtn[:, j])


@pytest.mark.parametrize("bits", [2, 8])
def test_layer_extreme_bits(bits):
    W, X, Sg, out = _layer_case(64, 128, 1024, torch.float32, bits, 3, seed=13)
    _check_layer(W, Sg, out, bits, 3)


def test_layer_tiny_and_single_column():
    for q, p in [(1, 1), (3, 5), (1, 70), (129, 1)]:
        W, X, Sg, out = _layer_case(q, p, 256, torch.float32, 3, 2, seed=q * 100 + p)
        _check_layer(W, Sg, out, 3, 2)


def test_layer_warm_start():
    q, p, n, bits, iters = 128, 192, 2048, 3, 3
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=21, device="cuda")
    X = inputs.calib_inputs(p, n, dtype=torch.bfloat16, seed=21, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0, corr_rank=4)
    Sg = qe.qe_build_sigma(X)
    W64 = parity.f64(W)
    s, z = O.grid(W64, bits)
    init = O.rtn(W64, s, z, bits)
    out = qe.qe_quantize_layer(W, Sg, bits, iters, init_codes=torch.from_numpy(init).cuda(),
                               record_sweeps=True, want_norm=True)
    assert qe.qe_sync_status() == qe.QE_OK
    _check_layer(W, Sg, out, bits, iters, init_codes=init, free_running=False)


def test_config1_opt125m_full():
    cfg = inputs.CONFIGS["opt125m_768x768"]
    W = cfg.weights("cuda")
    X = cfg.inputs("cuda")
    Sg = qe.qe_build_sigma(X)
    out = qe.qe_quantize_layer(W, Sg, cfg.bits[0], cfg.iters, record_sweeps=True, want_norm=True)
    assert qe.qe_sync_status() == qe.QE_OK
    _sigma_check(Sg, parity.f64(X))
    _check_layer(W, Sg, out, cfg.bits[0], cfg.iters)


def test_deterministic_repeat():
    W, X, Sg, out = _layer_case(150, 200, 1024, torch.bfloat16, 3, 3, seed=31, corr_rank=4)
    out2 = qe.qe_quantize_layer(W, Sg, 3, 3)
    torch.cuda.synchronize()
    assert torch.equal(out["codes"], out2["codes"])
    assert torch.equal(out["obj"], out2["obj"])
    S2 = qe.qe_build_sigma(X)
    torch.cuda.synchronize()
    assert torch.equal(S2, Sg)


def test_nonfinite_input_is_reported():
    W = inputs.layer_weights(16, 32, dtype=torch.float32, seed=1, device="cuda")
    W[3, 7] = float("nan")
    X = inputs.calib_inputs(32, 128, dtype=torch.float32, seed=1, device="cuda")
    Sg = qe.qe_build_sigma(X)
    qe.qe_quantize_layer(W, Sg, 4, 1)
    assert qe.qe_sync_status() == qe.QE_ERR_NUMERIC
    assert qe.qe_sync_status() == qe.QE_OK          # the latch is cleared


# ---------------------------------------------------------------------------
# qe_quantize_layer_outlier
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("q,p,bits,frac", [(96, 192, 3, 0.01), (130, 260, 2, 0.02), (70, 203, 3, 0.01),
                                         (8, 4200, 3, 0.01)])
def test_outlier_parity_small(q, p, bits, frac):
    iters, power_iters = 4, 200
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=41, device="cuda", planted_frac=frac,
                             planted_std=0.3)
    X = inputs.calib_inputs(p, 2048, dtype=torch.bfloat16, seed=41, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    s_budget = int(round(frac * q * p))
    out = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, s_budget, power_iters=power_iters,
                                       record_sweeps=True)
    assert qe.qe_sync_status() == qe.QE_OK
    W64, S64 = parity.f64(W), parity.f64(Sg)
    ref = O.outlier(W64, S64, bits, iters, s_budget, power_iters)
    assert np.array_equal(out["scales"].cpu().numpy(), ref["scale"])
    assert np.array_equal(out["zeros"].cpu().numpy(), ref["zero"])
    parity.check_obj(out["obj_cd"].cpu().numpy(), ref["obj_cd"], what="g after CD")
    parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="g after IHT")
    m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
    assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"
    nnz = int(out["H_nnz"].item())
    assert nnz == ref["nnz"]
    idx = out["H_idx"][:nnz].cpu().numpy()
    assert np.all(np.diff(idx) > 0)
    ref_idx = np.nonzero(ref["H"].ravel())[0]
    same = np.intersect1d(idx, ref_idx).size
    assert same >= 0.999 * nnz
    Hd = np.zeros(q * p)
    Hd[idx] = out["H_val"][:nnz].cpu().numpy()
    common = np.intersect1d(idx, ref_idx)
    assert np.allclose(Hd[common], ref["H"].ravel()[common], rtol=1e-3, atol=1e-6)
    # Lemma 3: the IHT half never increases g
    assert np.all(out["obj"].cpu().numpy() <= out["obj_cd"].cpu().numpy() * (1 + 1e-6))
    # teacher-forced, iteration by iteration from the GPU's own state
    _outlier_replay(W, Sg, bits, iters, s_budget, power_iters, False, out)


def _outlier_replay(W, Sg, bits, iters, s_budget, power_iters, structured, out):
    """The GPU's Algorithm 4 trajectory replayed through the oracle one iteration at a
    time from the GPU's own state (parity.outlier_replay); H after every iteration
    comes from runs stopped there, which must be prefixes of the full run."""
    runs = [qe.qe_quantize_layer_outlier(W, Sg, bits, k, s_budget, power_iters=power_iters,
                                         structured=structured) for k in range(1, iters)] + [out]
    assert qe.qe_sync_status() == qe.QE_OK
    for o in runs[:-1]:
        k = o["obj"].numel()
        assert torch.equal(o["obj"], out["obj"][:k])
    W64, S64 = parity.f64(W), parity.f64(Sg)
    q, p = W64.shape
    if structured:
        cols = O.topk_columns(W64, s_budget // q)
        H0 = np.zeros_like(W64)
        H0[:, cols] = W64[:, cols]
    else:
        k0 = O.topk(W64, s_budget)
        H0 = np.zeros(W64.size)
        H0[k0] = W64.ravel()[k0]
        H0 = H0.reshape(q, p)
    eta = 1.0 / (2.0 * O.power_lambda(S64, power_iters))
    nnz = [int(o["H_nnz"].item()) for o in runs]
    hidx = [o["H_idx"][:m].cpu().numpy() for o, m in zip(runs, nnz)]
    hval = [o["H_val"][:m].cpu().numpy() for o, m in zip(runs, nnz)]
    return parity.outlier_replay(W64, S64, out["scales"].cpu().numpy(), out["zeros"].cpu().numpy(), bits,
                                 out["sweep_codes"].cpu().numpy(), hidx, hval, H0, eta, s_budget, structured)


def _planted_columns(W, cols, std, seed):
    g = torch.Generator().manual_seed(seed)
    noise = torch.randn(W.shape[0], len(cols), generator=g) * std
    W[:, cols] = (W[:, cols].float() + noise.to(W.device)).to(W.dtype)
    return W


@pytest.mark.parametrize("q,p,bits,ncols", [(96, 192, 3, 3), (130, 260, 2, 5)])
def test_structured_outlier_parity_small(q, p, bits, ncols):
    """Whole-column outliers (Sec. 4.3): the kept columns, grid, objectives, codes
    and H values against the oracle."""
    iters, power_iters = 4, 200
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=43, device="cuda")
    W = _planted_columns(W, [5, 40, 77, 121, 150][:ncols], 0.3, 43)
    X = inputs.calib_inputs(p, 2048, dtype=torch.bfloat16, seed=43, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    s_budget = ncols * q + 7
    out = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, s_budget, power_iters=power_iters,
                                       structured=True, record_sweeps=True)
    assert qe.qe_sync_status() == qe.QE_OK
    W64, S64 = parity.f64(W), parity.f64(Sg)
    _outlier_replay(W, Sg, bits, iters, s_budget, power_iters, True, out)
    ref = O.outlier(W64, S64, bits, iters, s_budget, power_iters, structured=True)
    assert np.array_equal(out["scales"].cpu().numpy(), ref["scale"])
    assert np.array_equal(out["zeros"].cpu().numpy(), ref["zero"])
    parity.check_obj(out["obj_cd"].cpu().numpy(), ref["obj_cd"], what="g after CD")
    parity.check_obj(out["obj"].cpu().numpy(), ref["obj"], what="g after IHT")
    m = parity.code_match(out["codes"].cpu().numpy(), ref["codes"])
    assert m >= parity.CODE_MATCH, f"codes match {m:.5f}"
    nnz = int(out["H_nnz"].item())
    assert nnz == ref["nnz"] == q * ncols
    idx = out["H_idx"][:nnz].cpu().numpy()
    assert np.all(np.diff(idx) > 0)
    gpu_cols = np.unique(idx % p)
    ref_cols = np.nonzero(np.any(ref["H"] != 0, axis=0))[0]
    assert np.array_equal(gpu_cols, ref_cols)
    Hd = np.zeros(q * p)
    Hd[idx] = out["H_val"][:nnz].cpu().numpy()
    assert np.allclose(Hd, ref["H"].ravel(), rtol=1e-3, atol=1e-6)
    assert np.all(out["obj"].cpu().numpy() <= out["obj_cd"].cpu().numpy() * (1 + 1e-6))


def test_structured_outlier_below_one_column_matches_plain_layer():
    q, p, bits, iters = 64, 128, 3, 3
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=52, device="cuda")
    X = inputs.calib_inputs(p, 1024, dtype=torch.bfloat16, seed=52, device="cuda", corr_rank=4)
    Sg = qe.qe_build_sigma(X)
    a = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, 0)
    b = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, q - 1, structured=True)
    torch.cuda.synchronize()
    assert torch.equal(a["codes"], b["codes"]) and int(b["H_nnz"].item()) == 0
    assert np.array_equal(a["obj"].cpu().numpy(), b["obj"].cpu().numpy())


@pytest.mark.parametrize("p", [1024, 203])
def test_outlier_sweep_modes_identical(p):
    """The per-iteration sweeps after the first take their mode (rows in lockstep or each
    on its own) from the previous sweep's change counts; every mode takes the same
    decisions in the same order, so the results agree bit for bit with always-lockstep
    (free_changes = -1) and always-free (a huge threshold) runs."""
    q, bits, iters = 256, 3, 6
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=91, device="cuda", planted_frac=0.01,
                             planted_std=0.3)
    X = inputs.calib_inputs(p, 4096, dtype=torch.bfloat16, seed=91, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    s_budget = int(0.01 * q * p)
    outs = [qe.qe_quantize_layer_outlier(W, Sg, bits, iters, s_budget, free_changes=f) for f in (-1, 0, 1 << 20)]
    assert qe.qe_sync_status() == qe.QE_OK
    ref = outs[0]
    for o in outs[1:]:
        assert torch.equal(o["codes"], ref["codes"])
        assert torch.equal(o["obj"], ref["obj"]) and torch.equal(o["obj_cd"], ref["obj_cd"])
        n = int(ref["H_nnz"].item())
        assert int(o["H_nnz"].item()) == n
        assert torch.equal(o["H_idx"][:n], ref["H_idx"][:n]) and torch.equal(o["H_val"][:n], ref["H_val"][:n])


def test_outlier_warm_start_and_without_obj_cd():
    """A warm start (init_codes) and a call without obj_cd refresh R from the codes
    with no fused objective.  The run stays valid: the IHT half never increases g
    (Lemma 3), g never increases (Lemma 2 from a feasible start), and g of the final
    state recomputed in fp64 matches; without obj_cd the objective is the same."""
    q, p, bits, iters, frac = 96, 192, 3, 4, 0.01
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=43, device="cuda", planted_frac=frac,
                             planted_std=0.3)
    X = inputs.calib_inputs(p, 2048, dtype=torch.bfloat16, seed=43, device="cuda", heavy_frac=0.02,
                            heavy_mult=30.0)
    Sg = qe.qe_build_sigma(X)
    s_budget = int(round(frac * q * p))
    first = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, s_budget, power_iters=200)
    out = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, s_budget, power_iters=200,
                                       init_codes=first["codes"])
    assert qe.qe_sync_status() == qe.QE_OK
    obj, obj_cd = out["obj"].cpu().numpy(), out["obj_cd"].cpu().numpy()
    assert np.all(obj <= obj_cd * (1 + 1e-6)), "IHT step increased g (Lemma 3)"
    assert np.all(np.diff(obj) <= 1e-6 * obj[:-1])
    nnz = int(out["H_nnz"].item())
    H = torch.zeros(q * p, dtype=torch.float64, device="cuda")
    H[out["H_idx"][:nnz]] = out["H_val"][:nnz].double()
    What = out["scales"].double()[:, None] * (out["codes"].double() - out["zeros"].double()[:, None])
    D = W.double() - What - H.view(q, p)
    g = float(torch.sum((D @ Sg.double()) * D).item())
    parity.check_obj(obj[-1], g, what="g of the final state (fp64)")
    # the same call through the C ABI with obj_cd = NULL
    L = qe.load()
    codes = torch.empty(q, p, dtype=torch.uint8, device="cuda")
    sc = torch.empty(q, dtype=torch.float32, device="cuda")
    zp = torch.empty(q, dtype=torch.float32, device="cuda")
    ob = torch.empty(iters, dtype=torch.float64, device="cuda")
    hv = torch.empty(s_budget, dtype=torch.float32, device="cuda")
    hi = torch.empty(s_budget, dtype=torch.int64, device="cuda")
    hn = torch.zeros(1, dtype=torch.int64, device="cuda")
    o = qe.QEOpts()
    o.power_iters = 200
    o.init_codes = first["codes"].data_ptr()
    st = L.qe_quantize_layer_outlier(W.data_ptr(), qe.QE_BF16, q, p, p, Sg.data_ptr(), bits, iters, s_budget,
                                     ctypes.byref(o), codes.data_ptr(), sc.data_ptr(), zp.data_ptr(),
                                     hv.data_ptr(), hi.data_ptr(), hn.data_ptr(), ob.data_ptr(), None,
                                     ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == qe.QE_OK
    assert qe.qe_sync_status() == qe.QE_OK
    assert torch.equal(ob, out["obj"]) and torch.equal(codes, out["codes"])


def test_outlier_zero_budget_matches_plain_layer():
    q, p, bits, iters = 64, 128, 3, 3
    W = inputs.layer_weights(q, p, dtype=torch.bfloat16, seed=51, device="cuda")
    X = inputs.calib_inputs(p, 1024, dtype=torch.bfloat16, seed=51, device="cuda", corr_rank=4)
    Sg = qe.qe_build_sigma(X)
    a = qe.qe_quantize_layer(W, Sg, bits, iters)
    b = qe.qe_quantize_layer_outlier(W, Sg, bits, iters, 0)
    torch.cuda.synchronize()
    assert torch.equal(a["codes"], b["codes"])
    assert int(b["H_nnz"].item()) == 0
    assert np.allclose(a["obj"].cpu().numpy(), b["obj"].cpu().numpy(), rtol=1e-6)
