"""Helpers shared by the GPU parity tests: moving seeded NumPy inputs to the device as the
exact same bits, reading results back, and the comparison rules of the parity bar."""
import numpy as np

import oracle
from paper_2606_10531_gb300 import workloads as wl


def torch():
    import torch as _t
    return _t


def dev(a):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(a)).cuda()


def dev_bf16(bits):
    """uint16 bf16 bit patterns -> device bf16 tensor (same bits)."""
    t = torch()
    return t.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(t.bfloat16)


def host_bf16(x):
    """device bf16 tensor -> exact fp64 values."""
    t = torch()
    bits = x.contiguous().view(t.int16).cpu().numpy().view(np.uint16)
    return wl.bf16_to_f32(bits).astype(np.float64)


def empty_bf16(*shape):
    t = torch()
    return t.empty(shape, dtype=t.bfloat16, device="cuda")


def max_rel(x, ref):
    """max_i |x_i - ref_i| / max_i |ref_i| (the tensor-wide relative error of the parity bar)."""
    x = np.asarray(x, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    den = np.max(np.abs(ref))
    return float(np.max(np.abs(x - ref)) / (den if den > 0 else 1.0))


def digit_product_bound(Xf, Z, A, b, d, ref, levels=8191, sigmas=7.0):
    """Elementwise error bound of the packed product on its integer-digit path (2-16 tokens): each
    element of X' = X_g A is rounded per token to a multiple of D_t = max|X'_t| / levels, off by at
    most D_t / 2 and independently of the others, so output (t, r) is off by the code-weighted sum of
    these roundings (standard deviation D_t sqrt(sum_c z_rc^2 / 12)), bounded here at `sigmas`
    standard deviations, plus the bf16 rounding of the output (at most 2^-9 of it, doubled for the
    fp32 sums) and a floor of 1e-7 max|ref| for outputs near zero."""
    Xp, _ = oracle.activation_transform(Xf, A, b, d)
    D = np.abs(Xp).max(axis=1) / levels
    spread = np.sqrt((np.asarray(Z, np.float64) ** 2).sum(axis=1) / 12.0)
    ref = np.asarray(ref, np.float64)
    return sigmas * D[:, None] * spread[None, :] + 2.0 ** -8 * np.abs(ref) + 1e-7 * np.abs(ref).max()


def within(x, ref, bound):
    """Largest |x - ref| / bound over the elements (the check passes at <= 1)."""
    x = np.asarray(x, np.float64)
    return float(np.max(np.abs(x - np.asarray(ref, np.float64)) / bound))


def config_A(d, rng):
    return (0.01 * np.eye(d) + rng.normal(0, 1e-3, (d, d))).astype(np.float32)


def config_b(d, rng):
    return rng.normal(0, 1e-3, d).astype(np.float32)


TOL_BF16 = 2e-2        # bf16 GEMM outputs and gradients vs the fp64 oracle (max relative error)
TOL_DECODE_F32 = 1e-6  # fp32 decoded weights (absolute)


def ldlq_latent_bound(W, Z, U, A, b, d):
    """Elementwise bound on |u_fp32 - u_exact| for the LDLQ latents u = A^{-1}(T - b) of a sweep whose
    history is Z, when the kernel forms every target in fp32 (standard forward-error analysis,
    gamma_k = k u / (1 - k u), u = 2^-24):
        e_j = w_j - (A z_j + b)   fp32: |de| <= gamma_{d+2} (|W| + |W_hat|)
        T   = W + E U             fp32 sums of at most n + 1 terms:
              |dT| <= gamma_{n+d+3} ((|W| + |W_hat|) |U| + |W|)
        u   = A^{-1}(T - b)       fp32, A^{-1} to relative 1e-6:
              |du| <= |A^{-1}| (|dT| + (gamma_{d+1} + 1e-6) (|T| + |b|))
    """
    u32 = 2.0 ** -24
    gam = lambda k: k * u32 / (1 - k * u32)  # noqa: E731
    W64 = np.asarray(W, np.float64)
    m, n = W64.shape
    import oracle
    What = oracle.decode(Z, A, b, d)
    Ua = np.abs(np.asarray(U, np.float64))
    T = W64 + (W64 - What) @ np.asarray(U, np.float64)
    dT = gam(n + d + 3) * ((np.abs(W64) + np.abs(What)) @ Ua + np.abs(W64))
    Ai = np.abs(np.linalg.inv(np.asarray(A, np.float64)))
    rhs = dT + (gam(d + 1) + 1e-6) * (np.abs(T) + np.abs(np.tile(np.asarray(b, np.float64), n // d)))
    return (rhs.reshape(m, n // d, d) @ Ai.T).reshape(m, n)
