"""Seeded synthetic inputs with the shapes and value distributions of the
CurveFP workloads.

This module holds no CurveFP arithmetic: it only draws random tensors.  Both
the oracle checks and the CUDA path take their inputs from here, so that the
two sides see identical data.  The paper's own tensors (real LLM weights,
activations and gradients, Sec. 4.2-4.4) are not available; these stand in
for them with the distributions named per workload.

Seeds: A = 1, B = 2, X = 3, W = 4, dY = 5; outlier masks use seed + 100.
"""
from __future__ import annotations

import numpy as np


def normal(shape, seed: int, std: float = 1.0) -> np.ndarray:
    """N(0, std^2) float32."""
    rng = np.random.default_rng(seed)
    out = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        out *= np.float32(std)
    return out


def outlier_channels(shape, seed: int, frac: float = 0.01, gain: float = 20.0) -> np.ndarray:
    """N(0,1) activations [tokens x channels] where a seeded choice of
    round(frac * channels) channels (columns) is scaled by ``gain``."""
    x = normal(shape, seed)
    rng = np.random.default_rng(seed + 100)
    n_out = int(round(frac * shape[1]))
    cols = rng.choice(shape[1], size=n_out, replace=False)
    x[:, cols] *= np.float32(gain)
    return x


def elementwise_outliers(shape, seed: int, p: float = 0.001, gain: float = 100.0) -> np.ndarray:
    """N(0,1) where each element independently (probability p) is scaled by
    ``gain``."""
    x = normal(shape, seed)
    rng = np.random.default_rng(seed + 100)
    mask = rng.random(size=shape, dtype=np.float32) < p
    x[mask] *= np.float32(gain)
    return x


def heavy_tailed_grad(shape, seed: int, scale: float = 1e-3, nu: float = 3.0) -> np.ndarray:
    """Output-gradient stand-in: scale * Student-t(nu)."""
    rng = np.random.default_rng(seed)
    return (scale * rng.standard_t(nu, size=shape)).astype(np.float32)


def lognormal_channels(shape, seed: int, sigma: float = 1.5) -> np.ndarray:
    """Z * diag(s): Z ~ N(0,1) [tokens x channels], s_c ~ LogNormal(0, sigma)."""
    z = normal(shape, seed)
    rng = np.random.default_rng(seed + 100)
    s = rng.lognormal(mean=0.0, sigma=sigma, size=shape[1]).astype(np.float32)
    return z * s[None, :]


# --- named workloads --------------------------------------------------------

def small_e4c3(M: int = 128, N: int = 128, K: int = 256):
    """CurveFP8 E4C3 block-32 case: A[M x K], B[K x N], both N(0,1)."""
    return normal((M, K), 1), normal((K, N), 2)


def llama7b_linear(tokens: int = 2048, d_in: int = 4096, d_out: int = 4096):
    """CurveFP7 E3C3 linear: W[d_out x d_in] ~ N(0, 0.02^2); X[tokens x d_in]
    ~ N(0,1) with 1 % outlier channels x20.  Y = X W^T."""
    return outlier_channels((tokens, d_in), 3), normal((d_out, d_in), 4, 0.02)


def training_triplet(tokens: int = 4096, d_in: int = 4096, d_out: int = 11008):
    """CurveFP8 training GEMMs: X[tokens x d_in] ~ N(0,1),
    W[d_in x d_out] ~ N(0, 0.02^2), dY[tokens x d_out] = 1e-3 * t_3."""
    return (normal((tokens, d_in), 3), normal((d_in, d_out), 4, 0.02),
            heavy_tailed_grad((tokens, d_out), 5))


def ffn_sweep(M: int, K: int = 4096, N: int = 14336):
    """CurveFP7 E3C3 FFN: W[K x N] ~ N(0, 0.02^2); X[M x K] with
    LogNormal(0, 1.5)-scaled channels."""
    return lognormal_channels((M, K), 3), normal((K, N), 4, 0.02)


def bandwidth_tensor(n: int, cols: int = 4096, seed: int = 3) -> np.ndarray:
    """Quantize-only sweep tensor (n elements as [n/cols x cols]) ~ N(0,1)
    with 0.1 % x100 element outliers.  Returned as float32; BF16 callers
    round it once."""
    return elementwise_outliers((n // cols, cols), seed)


def bandwidth_tensor_cuda(n: int, cols: int = 4096, seed: int = 3):
    """Device-side generator for the quantize-only sweep (sizes up to 2^30
    elements are too slow to draw on the host): BF16 [n/cols x cols], N(0,1)
    with each element independently (p = 0.001) scaled by 100.  Uses torch's
    CUDA generator, so values differ from ``bandwidth_tensor`` but follow the
    same distribution."""
    import torch

    g = torch.Generator(device="cuda").manual_seed(seed)
    x = torch.randn((n // cols, cols), device="cuda", generator=g, dtype=torch.float32)
    mask = torch.rand((n // cols, cols), device="cuda", generator=g) < 0.001
    x = torch.where(mask, x * 100.0, x)
    del mask
    return x.to(torch.bfloat16)


def training_triplet_cuda(tokens: int = 4096, d_in: int = 4096, d_out: int = 11008, seed: int = 3):
    """Device-side draw of the training-GEMM tensors (same distributions as
    ``training_triplet``, torch's CUDA generator): X[tokens x d_in] ~ N(0,1),
    W[d_in x d_out] ~ N(0, 0.02^2), dY[tokens x d_out] = 1e-3 * t_3 with
    t_3 = Z / sqrt(chi^2_3 / 3)."""
    import torch

    g = torch.Generator(device="cuda").manual_seed(seed)
    x = torch.randn((tokens, d_in), device="cuda", generator=g)
    w = torch.randn((d_in, d_out), device="cuda", generator=g) * 0.02
    z = torch.randn((tokens, d_out), device="cuda", generator=g)
    chi2 = torch.zeros_like(z)
    for _ in range(3):
        chi2 += torch.randn((tokens, d_out), device="cuda", generator=g) ** 2
    dy = 1e-3 * z / torch.sqrt(chi2 / 3.0)
    return x, w, dy


def ffn_cuda(M: int, K: int = 4096, N: int = 14336, seed: int = 3):
    """Device-side draw of an FFN-sweep case (same distributions as
    ``ffn_sweep``): X[M x K] = Z diag(s), s_c ~ LogNormal(0, 1.5);
    W[K x N] ~ N(0, 0.02^2)."""
    import torch

    g = torch.Generator(device="cuda").manual_seed(seed)
    z = torch.randn((M, K), device="cuda", generator=g)
    s = torch.exp(1.5 * torch.randn((K,), device="cuda", generator=g))
    w = torch.randn((K, N), device="cuda", generator=g) * 0.02
    return z * s[None, :], w
