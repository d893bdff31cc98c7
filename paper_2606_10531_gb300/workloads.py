"""Seeded synthetic inputs shaped like the paper's LLM layers.

This module only draws random numbers and rounds them to the storage
types; it contains none of the quantizer's arithmetic. Tests feed the same
NumPy-drawn bits to the CUDA library and to the CPU oracle; the benchmark
draws the same distributions directly on the device with torch generators
(bit-identity with the oracle is not needed there).

Each matrix of a workload has its own seed stream
``SeedSequence(seed, spawn_key=(matrix_index, part))`` with one part per
tensor (W, A, b, X, dY, codes), so any tensor can be drawn alone.

Distributions (std, not variance, in every N(0, s)):
  * W ~ N(0, 0.02) fp32 (training workloads), N(0, 0.015) with a Bernoulli(0.001)
    mask of entries replaced by 0.015 * Student-t(nu=4) (bulk-encode workload);
  * A = 0.01 I + N(0, 1e-3) (d x d), b ~ N(0, 1e-3) (d);
  * X, dY ~ N(0, 1) rounded to bf16; the 7B-projection workload scales
    round(0.01 n) seeded input channels of X by 20 (activation outliers);
  * packed deployment codes: uniform random bytes (4 uniform codes each);
  * proxy Hessian for LDLQ (stands in for the calibration statistics E[x x^T] of
    1,024 RedPajama samples, which are absent): H0 = S (K/2 + V V^T/(2r)) S with
    K_ij = 0.9^|i-j| (neighbouring-channel correlation), V ~ N(0,1) of rank r = 8
    (a few dominant activation directions) and S = diag(1, with round(0.01 n)
    seeded outlier channels scaled by 20); H = H0 + 0.01 mean(diag H0) I (1%
    dampening), rounded to fp32.
"""
from __future__ import annotations

import dataclasses

import numpy as np

PARTS = {"W": 0, "A": 1, "b": 2, "X": 3, "dY": 4, "codes": 5, "outliers": 6, "hessian": 7}


@dataclasses.dataclass(frozen=True)
class Matrix:
    name: str
    m: int          # output rows
    n: int          # input dim (grouped along n)
    d: int          # group size
    N: int          # tokens
    w_std: float = 0.02
    heavy_tail: bool = False     # bulk-encode workload: Student-t entries
    outlier_frac: float = 0.0    # fraction of X channels scaled by outlier_scale
    outlier_scale: float = 20.0


def tiny_layer(N: int = 64, m: int = 512, n: int = 512, d: int = 4):
    """Single LC-VQ linear, 512x512, d=4, 64 tokens (oracle-sized)."""
    return [Matrix("tiny", m, n, d, N)]


def llama2_7b_projections(d: int, N: int = 4096):
    """Llama-2-7B projections q/k/v/o 4096x4096, gate/up 11008x4096, down 4096x11008; 1% outlier channels."""
    h, f = 4096, 11008
    shapes = [("q", h, h), ("k", h, h), ("v", h, h), ("o", h, h), ("gate", f, h), ("up", f, h), ("down", h, f)]
    return [Matrix(nm, m, n, d, N, outlier_frac=0.01) for nm, m, n in shapes]


def llama3_8b_layer(d: int = 8, N: int = 8 * 2048):
    """Llama-3-8B decoder layer: hidden 4096, GQA k/v 1024x4096, MLP 14336; 8 x 2048 tokens."""
    h, kv, f = 4096, 1024, 14336
    shapes = [("q", h, h), ("k", kv, h), ("v", kv, h), ("o", h, h), ("gate", f, h), ("up", f, h), ("down", h, f)]
    return [Matrix(nm, m, n, d, N) for nm, m, n in shapes]


def llama3_70b_gate_decode(batch: int):
    """Llama-3-70B gate projection 28672x8192 as packed 2-bit codes, d=8, `batch` tokens."""
    return [Matrix("gate70b", 28672, 8192, 8, batch)]


def llama3_70b_layer_encode(d: int = 8):
    """All linears of a Llama-3-70B layer for bulk encode; heavy-tailed fp32 weights."""
    h, kv, f = 8192, 1024, 28672
    shapes = [("q", h, h), ("k", kv, h), ("v", kv, h), ("o", h, h), ("gate", f, h), ("up", f, h), ("down", h, f)]
    return [Matrix(nm, m, n, d, 0, w_std=0.015, heavy_tail=True) for nm, m, n in shapes]


def llama3_70b_gate_ldlq(d: int = 8):
    """LDLQ initialisation of the Llama-3-70B gate projection 28672x8192 (heavy-tailed fp32 weights)."""
    return [Matrix("gate70b", 28672, 8192, d, 0, w_std=0.015, heavy_tail=True)]


def llama3_8b_gate_ldlq(d: int = 8):
    """LDLQ initialisation of the Llama-3-8B gate projection 14336x4096 (heavy-tailed fp32 weights)."""
    return [Matrix("gate8b", 14336, 4096, d, 0, w_std=0.015, heavy_tail=True)]


HESSIAN_RHO, HESSIAN_RANK, HESSIAN_DAMP = 0.9, 8, 0.01


# ----------------------------------------------------------------------------- NumPy draws

def _rng(seed: int, index: int, part: str) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence(seed, spawn_key=(index, PARTS[part])))


def bf16_bits(x) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest even) and return the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_to_f32(bits) -> np.ndarray:
    """Exact fp32 value of bf16 bit patterns."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def draw_W(mx: Matrix, seed: int, index: int) -> np.ndarray:
    rng = _rng(seed, index, "W")
    W = rng.normal(0.0, mx.w_std, size=(mx.m, mx.n)).astype(np.float32)
    if mx.heavy_tail:
        mask = rng.random((mx.m, mx.n)) < 0.001
        W[mask] = (mx.w_std * rng.standard_t(4.0, size=int(mask.sum()))).astype(np.float32)
    return W


def draw_A(mx: Matrix, seed: int, index: int) -> np.ndarray:
    rng = _rng(seed, index, "A")
    return (0.01 * np.eye(mx.d) + rng.normal(0.0, 1e-3, size=(mx.d, mx.d))).astype(np.float32)


def draw_b(mx: Matrix, seed: int, index: int) -> np.ndarray:
    rng = _rng(seed, index, "b")
    return rng.normal(0.0, 1e-3, size=(mx.d,)).astype(np.float32)


def draw_X(mx: Matrix, seed: int, index: int, tokens: int | None = None) -> np.ndarray:
    """Activations [N][n] as bf16 bit patterns (uint16)."""
    N = mx.N if tokens is None else tokens
    rng = _rng(seed, index, "X")
    X = rng.normal(0.0, 1.0, size=(N, mx.n)).astype(np.float32)
    if mx.outlier_frac > 0:
        k = int(round(mx.outlier_frac * mx.n))
        ch = _rng(seed, index, "outliers").choice(mx.n, size=k, replace=False)
        X[:, ch] *= np.float32(mx.outlier_scale)
    return bf16_bits(X)


def draw_dY(mx: Matrix, seed: int, index: int, tokens: int | None = None) -> np.ndarray:
    """Upstream gradient [N][m] as bf16 bit patterns (uint16)."""
    N = mx.N if tokens is None else tokens
    rng = _rng(seed, index, "dY")
    return bf16_bits(rng.normal(0.0, 1.0, size=(N, mx.m)).astype(np.float32))


def draw_packed_codes(mx: Matrix, seed: int, index: int) -> np.ndarray:
    """Uniform random packed codes [m][n/4] (each byte = 4 independent uniform 2-bit codes)."""
    rng = _rng(seed, index, "codes")
    return rng.integers(0, 256, size=(mx.m, mx.n // 4), dtype=np.uint8)


def draw_hessian(n: int, seed: int, index: int) -> np.ndarray:
    """Synthetic symmetric positive definite proxy Hessian [n][n] fp32 (recipe in the module doc)."""
    rng = _rng(seed, index, "hessian")
    V = rng.standard_normal((n, HESSIAN_RANK))
    s = np.ones(n)
    s[rng.choice(n, size=int(round(0.01 * n)), replace=False)] = 20.0
    i = np.arange(n)
    K = HESSIAN_RHO ** np.abs(i[:, None] - i[None, :]).astype(np.float64)
    H0 = s[:, None] * (0.5 * K + (0.5 / HESSIAN_RANK) * (V @ V.T)) * s[None, :]
    H = H0 + HESSIAN_DAMP * np.mean(np.diag(H0)) * np.eye(n)
    return H.astype(np.float32)


# ----------------------------------------------------------------------------- device draws

def _torch_gen(torch, device, seed: int, index: int, part: str):
    g = torch.Generator(device=device)
    g.manual_seed(int(np.random.SeedSequence(seed, spawn_key=(index, PARTS[part])).generate_state(1)[0]))
    return g


def torch_W(torch, mx: Matrix, seed: int, index: int, device):
    g = _torch_gen(torch, device, seed, index, "W")
    W = torch.randn((mx.m, mx.n), generator=g, device=device, dtype=torch.float32).mul_(mx.w_std)
    if mx.heavy_tail:
        mask = torch.rand((mx.m, mx.n), generator=g, device=device) < 0.001
        k = int(mask.sum().item())
        z = torch.randn(k, generator=g, device=device)
        chi2 = torch.randn((k, 4), generator=g, device=device).square_().sum(1)
        W[mask] = mx.w_std * z / torch.sqrt(chi2 / 4.0)
    return W


def torch_A(torch, mx: Matrix, seed: int, index: int, device):
    g = _torch_gen(torch, device, seed, index, "A")
    return 0.01 * torch.eye(mx.d, device=device) + 1e-3 * torch.randn((mx.d, mx.d), generator=g, device=device)


def torch_b(torch, mx: Matrix, seed: int, index: int, device):
    g = _torch_gen(torch, device, seed, index, "b")
    return 1e-3 * torch.randn(mx.d, generator=g, device=device)


def torch_X(torch, mx: Matrix, seed: int, index: int, device, tokens: int | None = None):
    N = mx.N if tokens is None else tokens
    g = _torch_gen(torch, device, seed, index, "X")
    X = torch.randn((N, mx.n), generator=g, device=device, dtype=torch.float32)
    if mx.outlier_frac > 0:
        k = int(round(mx.outlier_frac * mx.n))
        go = _torch_gen(torch, device, seed, index, "outliers")
        ch = torch.randperm(mx.n, generator=go, device=device)[:k]
        X[:, ch] *= mx.outlier_scale
    return X.to(torch.bfloat16)


def torch_dY(torch, mx: Matrix, seed: int, index: int, device, tokens: int | None = None):
    N = mx.N if tokens is None else tokens
    g = _torch_gen(torch, device, seed, index, "dY")
    return torch.randn((N, mx.m), generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def torch_packed_codes(torch, mx: Matrix, seed: int, index: int, device):
    g = _torch_gen(torch, device, seed, index, "codes")
    return torch.randint(0, 256, (mx.m, mx.n // 4), generator=g, device=device, dtype=torch.int32).to(torch.uint8)


def torch_hessian(torch, n: int, seed: int, index: int, device):
    """Device draw of the synthetic proxy Hessian (same recipe as draw_hessian, torch generator)."""
    g = _torch_gen(torch, device, seed, index, "hessian")
    V = torch.randn((n, HESSIAN_RANK), generator=g, device=device, dtype=torch.float32)
    s = torch.ones(n, device=device, dtype=torch.float32)
    s[torch.randperm(n, generator=g, device=device)[:int(round(0.01 * n))]] = 20.0
    i = torch.arange(n, device=device, dtype=torch.float32)
    H = torch.pow(torch.tensor(HESSIAN_RHO, device=device), (i[:, None] - i[None, :]).abs())
    H.mul_(0.5).addmm_(V, V.t(), alpha=0.5 / HESSIAN_RANK)
    H.mul_(s[:, None]).mul_(s[None, :])
    H.diagonal().add_(HESSIAN_DAMP * H.diagonal().mean())
    return H
