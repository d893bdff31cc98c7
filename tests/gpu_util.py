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
