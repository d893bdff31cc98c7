"""Helpers shared by the GPU parity tests: moving seeded NumPy inputs to the device as the
exact same bits, reading results back, and the comparison rules of the parity bar."""
import numpy as np

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
