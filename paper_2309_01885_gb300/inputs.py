"""Seeded synthetic layers shaped like the paper's calibration workloads.

This module only draws random numbers; it holds none of the method's
arithmetic.  Both the CUDA path and the fp64 oracle are fed from it.

The paper calibrates on 128 C4 sequences of 2048 tokens (n = 262144, Sec. 5)
and quantizes OPT / BLOOM / Falcon / LLaMA-shaped linear layers.  Neither the
dataset nor the weights are available here, so every input is synthetic:

* W ~ N(0, 0.02^2) (fp32 or bf16), optionally with a fraction of entries
  multiplied by a factor (``w_outlier_frac`` / ``w_outlier_mult``) or with
  planted N(0, sigma^2) values *added* at a fraction of positions
  (``planted_frac`` / ``planted_std``);
* X ~ N(0, 1), p x n feature-major, with a fraction of input channels (whole
  rows of X) multiplied by ``heavy_mult``; optionally correlated as
  X = Z + U (V^T Z) with rank ``corr_rank`` to couple the coordinates hard.

Draws use ``torch.Generator(device).manual_seed(1000 * seed + stream)`` with
streams W = 1, X = 2, heavy-channel pick = 3, W-outlier pick = 4, planted
values = 5, correlation factors = 6.  fp32 draws are cast to bf16 with
round-to-nearest-even where a bf16 tensor is asked for.
"""
from __future__ import annotations

import dataclasses

import torch

STREAM_W, STREAM_X, STREAM_HEAVY, STREAM_WPICK, STREAM_PLANT, STREAM_CORR = 1, 2, 3, 4, 5, 6


def _gen(device, seed: int, stream: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(1000 * int(seed) + int(stream))
    return g


def _count(frac: float, total: int) -> int:
    return int(round(frac * total))


def layer_weights(q: int, p: int, *, dtype=torch.float32, seed: int = 0, device="cpu",
                  std: float = 0.02, w_outlier_frac: float = 0.0, w_outlier_mult: float = 10.0,
                  planted_frac: float = 0.0, planted_std: float = 0.3) -> torch.Tensor:
    """W (q x p) of the requested dtype."""
    W = torch.randn(q, p, generator=_gen(device, seed, STREAM_W), device=device,
                    dtype=torch.float32) * std
    if w_outlier_frac > 0:
        k = _count(w_outlier_frac, q * p)
        pick = torch.randperm(q * p, generator=_gen(device, seed, STREAM_WPICK), device=device)[:k]
        W.view(-1)[pick] *= w_outlier_mult
    if planted_frac > 0:
        k = _count(planted_frac, q * p)
        pick = torch.randperm(q * p, generator=_gen(device, seed, STREAM_WPICK), device=device)[:k]
        vals = torch.randn(k, generator=_gen(device, seed, STREAM_PLANT), device=device,
                           dtype=torch.float32) * planted_std
        W.view(-1)[pick] += vals
    return W.to(dtype)


def calib_inputs(p: int, n: int, *, dtype=torch.float32, seed: int = 0, device="cpu",
                 heavy_frac: float = 0.0, heavy_mult: float = 1.0, corr_rank: int = 0,
                 zero_rows=()) -> torch.Tensor:
    """X (p x n, feature-major) of the requested dtype."""
    X = torch.randn(p, n, generator=_gen(device, seed, STREAM_X), device=device,
                    dtype=torch.float32)
    if corr_rank > 0:
        g = _gen(device, seed, STREAM_CORR)
        U = torch.randn(p, corr_rank, generator=g, device=device) / (p ** 0.5)
        V = torch.randn(p, corr_rank, generator=g, device=device) * 2.0
        X = X + U @ (V.t() @ X)
    if heavy_frac > 0:
        k = _count(heavy_frac, p)
        pick = torch.randperm(p, generator=_gen(device, seed, STREAM_HEAVY), device=device)[:k]
        X[pick] *= heavy_mult
    for r in zero_rows:
        X[r] = 0
    return X.to(dtype)


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    """One synthetic layer workload."""
    name: str
    q: int
    p: int
    n: int
    w_dtype: torch.dtype
    x_dtype: torch.dtype
    bits: tuple
    iters: int
    heavy_frac: float
    heavy_mult: float = 30.0
    w_outlier_frac: float = 0.0
    w_outlier_mult: float = 10.0
    planted_frac: float = 0.0
    planted_std: float = 0.3
    outlier_budget_frac: float = 0.0   # s = round(frac * q * p), round-half-even
    seed: int = 0

    @property
    def s_budget(self) -> int:
        return int(round(self.outlier_budget_frac * self.q * self.p))

    def weights(self, device="cpu") -> torch.Tensor:
        return layer_weights(self.q, self.p, dtype=self.w_dtype, seed=self.seed, device=device,
                             w_outlier_frac=self.w_outlier_frac,
                             w_outlier_mult=self.w_outlier_mult,
                             planted_frac=self.planted_frac, planted_std=self.planted_std)

    def inputs(self, device="cpu") -> torch.Tensor:
        return calib_inputs(self.p, self.n, dtype=self.x_dtype, seed=self.seed, device=device,
                            heavy_frac=self.heavy_frac, heavy_mult=self.heavy_mult)


# The synthetic workloads: an OPT-125m-sized layer (oracle-sized), a LLaMA-7B
# attention projection, the LLaMA-7B MLP pair, the Falcon-180B QKV and down
# projections, and the outlier-aware variant of the LLaMA-7B projection at 3 bits
# with 1% outliers and at 2 bits with 2%.
CONFIGS = {
    "opt125m_768x768": LayerConfig("opt125m_768x768", 768, 768, 4096, torch.float32,
                                   torch.float32, (4,), 5, heavy_frac=0.01, heavy_mult=20.0,
                                   w_outlier_frac=0.001, w_outlier_mult=10.0),
    "llama7b_proj_4096x4096": LayerConfig("llama7b_proj_4096x4096", 4096, 4096, 262144,
                                          torch.bfloat16, torch.bfloat16, (3, 4), 20,
                                          heavy_frac=0.005),
    "llama7b_up_11008x4096": LayerConfig("llama7b_up_11008x4096", 11008, 4096, 262144,
                                         torch.bfloat16, torch.bfloat16, (4,), 20,
                                         heavy_frac=0.005),
    "llama7b_down_4096x11008": LayerConfig("llama7b_down_4096x11008", 4096, 11008, 262144,
                                           torch.bfloat16, torch.bfloat16, (4,), 20,
                                           heavy_frac=0.005),
    "falcon180b_qkv_15360x14848": LayerConfig("falcon180b_qkv_15360x14848", 15360, 14848, 65536,
                                              torch.bfloat16, torch.bfloat16, (3,), 10,
                                              heavy_frac=0.005),
    "falcon180b_down_14848x59392": LayerConfig("falcon180b_down_14848x59392", 14848, 59392, 65536,
                                               torch.bfloat16, torch.bfloat16, (3,), 10,
                                               heavy_frac=0.005),
    "llama7b_proj_outlier_4096x4096": LayerConfig("llama7b_proj_outlier_4096x4096", 4096, 4096,
                                                  262144, torch.bfloat16, torch.bfloat16, (3,), 20,
                                                  heavy_frac=0.005, planted_frac=0.01,
                                                  planted_std=0.3, outlier_budget_frac=0.01),
    # the 2-bit regime of Sec. 5 (2 bits with 2% outliers): the same path at b = 2, twice the budget
    "llama7b_proj_outlier2b_4096x4096": LayerConfig("llama7b_proj_outlier2b_4096x4096", 4096, 4096,
                                                    262144, torch.bfloat16, torch.bfloat16, (2,), 20,
                                                    heavy_frac=0.005, planted_frac=0.02,
                                                    planted_std=0.3, outlier_budget_frac=0.02),
}
