"""Python binding of liblcq, the GB300 (sm_103a) LC-VQ linear layer.

Thin ctypes marshalling over the C ABI declared in include/lcq.h: every
function here has the name of its C entry point, takes torch tensors, and
passes their device pointers, sizes and the current CUDA stream. No step of
the computation runs in Python or PyTorch; if liblcq.so is missing the import
fails instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG_DIR, "liblcq.so")

LCQ_OK = 0
STATUS_NAMES = {0: "LCQ_OK", 1: "LCQ_ERR_NULL", 2: "LCQ_ERR_SHAPE", 3: "LCQ_ERR_ALIGN", 4: "LCQ_ERR_UNSUPPORTED",
                5: "LCQ_ERR_WORKSPACE", 6: "LCQ_ERR_CUDA", 7: "LCQ_ERR_SINGULAR", 8: "LCQ_ERR_TIMEOUT",
                9: "LCQ_ERR_ARG", 10: "LCQ_ERR_LIMIT"}
LCQ_OP_ENCODE, LCQ_OP_LINEAR_FWD, LCQ_OP_LINEAR_BWD, LCQ_OP_GEMM_PACKED2B, LCQ_OP_GEMM_PACKED2B_HADAMARD = 1, 2, 3, 4, 5
LCQ_OP_ENCODE_BATCH = 6
LCQ_OP_LDL_FACTOR, LCQ_OP_LDLQ = 7, 8
LCQ_ENCODE_BATCH_MAX = 16
LCQ_STE_IDENTITY, LCQ_STE_CLIPPED, LCQ_STE_DGE = 0, 1, 2

# Every symbol include/lcq.h declares.
EXPORTS = ("lcq_workspace_size", "lcq_encode", "lcq_decode", "lcq_pack2b", "lcq_linear_fwd", "lcq_linear_bwd",
           "lcq_gemm_packed2b", "lcq_device_status", "lcq_status_string", "lcq_launch_count", "lcq_trace_enable",
           "lcq_trace_read", "lcq_gemm_packed2b_noalloc", "lcq_last_cuda_error", "lcq_selftest_wait_timeout",
           "lcq_init_codebook", "lcq_init_latent", "lcq_hadamard", "lcq_gemm_packed2b_hadamard", "lcq_encode_batch",
           "lcq_ldl_factor", "lcq_ldlq", "lcq_activation_transform")
KERNEL_KINDS = ("encode", "quant_decode", "decode", "pack", "gemm_fwd", "gemm_dx", "gemm_dw", "reduce",
                "gemv_prep", "gemv", "ldl_factor", "ldlq", "xform")


class LCQError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        detail = _status_string(status)
        if status == 6:
            try:
                detail += ": " + lib().lcq_last_cuda_error().decode()
            except Exception:  # noqa: BLE001 - only decorates the message
                pass
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)} ({detail})")


class lcq_opts(ctypes.Structure):
    _fields_ = [("latent_scale", ctypes.c_float), ("latent_offset", ctypes.c_float),
                ("ste_mode", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("dge_k", ctypes.c_float), ("dge_grad_max", ctypes.c_float)]


_P = ctypes.c_void_p
_I64 = ctypes.c_int64


class lcq_encode_item(ctypes.Structure):
    _fields_ = [("W", _P), ("m", _I64), ("n", _I64), ("A", _P), ("b", _P), ("packed", _P), ("codes", _P),
                ("latent", _P), ("mse", _P)]
_SIG = {
    "lcq_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I64, _I64, _I64, ctypes.c_int]),
    "lcq_encode": (ctypes.c_int, [_P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "lcq_encode_batch": (ctypes.c_int, [ctypes.POINTER(lcq_encode_item), ctypes.c_int, ctypes.c_int, _P,
                                        ctypes.c_size_t, _P]),
    "lcq_decode": (ctypes.c_int, [_P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P]),
    "lcq_ldl_factor": (ctypes.c_int, [_P, _I64, ctypes.c_int, _P, _P, _P, ctypes.c_size_t, _P]),
    "lcq_ldlq": (ctypes.c_int, [_P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "lcq_pack2b": (ctypes.c_int, [_P, _I64, _I64, _P, _P]),
    "lcq_activation_transform": (ctypes.c_int, [_P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P]),
    "lcq_linear_fwd": (ctypes.c_int, [_P, _I64, _P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P, _P,
                                      ctypes.c_size_t, _P]),
    "lcq_linear_bwd": (ctypes.c_int, [_P, _P, _P, _P, _I64, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P, _P, _P,
                                      _P, ctypes.c_size_t, _P]),
    "lcq_gemm_packed2b": (ctypes.c_int, [_P, _I64, _P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, ctypes.c_size_t,
                                         _P]),
    "lcq_gemm_packed2b_noalloc": (ctypes.c_int, [_P, _I64, _P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P, _P]),
    "lcq_device_status": (ctypes.c_int, [_P, _P, ctypes.POINTER(ctypes.c_int32), ctypes.c_int]),
    "lcq_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "lcq_last_cuda_error": (ctypes.c_char_p, []),
    "lcq_selftest_wait_timeout": (ctypes.c_int, [_P, _P]),
    "lcq_init_codebook": (ctypes.c_int, [_P, ctypes.c_int, _P, _P, _P]),
    "lcq_hadamard": (ctypes.c_int, [_P, _I64, _I64, _P, _P]),
    "lcq_gemm_packed2b_hadamard": (ctypes.c_int, [_P, _I64, _P, _I64, _I64, ctypes.c_int, _P, _P, _P, _P,
                                                  ctypes.c_size_t, _P]),
    "lcq_init_latent": (ctypes.c_int, [_P, _I64, _I64, _P, ctypes.POINTER(ctypes.c_float),
                                       ctypes.POINTER(ctypes.c_float), _P]),
    "lcq_launch_count": (ctypes.c_uint64, []),
    "lcq_trace_enable": (ctypes.c_int, [ctypes.c_int]),
    "lcq_trace_read": (ctypes.c_int, [ctypes.c_int, ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(ctypes.c_double)]),
}


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load liblcq.so and declare the C signatures. Raises if it is missing."""
    if not os.path.exists(path):
        raise ImportError(f"liblcq.so not found at {path}; build it with paper_2606_10531_gb300.build.build()")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIG.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = load_library()
    return _lib


def _status_string(status: int) -> str:
    try:
        return lib().lcq_status_string(status).decode()
    except Exception:  # noqa: BLE001 - only used to decorate an error message
        return "?"


def _check(status: int, where: str):
    if status != LCQ_OK:
        raise LCQError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _opts(latent_scale=1.0, latent_offset=0.0, ste_mode=LCQ_STE_IDENTITY, dge_k=0.0, dge_grad_max=0.0):
    return lcq_opts(float(latent_scale), float(latent_offset), int(ste_mode), 0, float(dge_k), float(dge_grad_max))


# ----------------------------------------------------------------------------- entry points

def lcq_workspace_size(op: int, N: int, m: int, n: int, d: int) -> int:
    return int(lib().lcq_workspace_size(op, N, m, n, d))


def workspace(op: int, N: int, m: int, n: int, d: int, device="cuda"):
    """Allocate (through PyTorch) a workspace tensor large enough for `op`, zero-initialised."""
    import torch
    return torch.zeros(max(lcq_workspace_size(op, N, m, n, d), 256), dtype=torch.uint8, device=device)


def lcq_encode(W, A, b, d: int, ws, packed=None, codes=None, latent=None, mse=None, stream=None):
    m, n = W.shape
    _check(lib().lcq_encode(_ptr(W), m, n, d, _ptr(A), _ptr(b), _ptr(packed), _ptr(codes), _ptr(latent), _ptr(mse),
                            _ptr(ws), ws.numel(), _stream(stream)), "lcq_encode")


def lcq_encode_batch(items, d: int, ws, stream=None):
    """items: sequence of dicts with W, A, b and optional packed, codes, latent, mse tensors (as lcq_encode)."""
    arr = (lcq_encode_item * len(items))()
    for k, it in enumerate(items):
        m, n = it["W"].shape
        addr = lambda t: None if t is None else t.data_ptr()  # noqa: E731
        arr[k] = lcq_encode_item(addr(it["W"]), m, n, addr(it["A"]), addr(it["b"]), addr(it.get("packed")),
                                 addr(it.get("codes")), addr(it.get("latent")), addr(it.get("mse")))
    _check(lib().lcq_encode_batch(arr, len(items), d, _ptr(ws), ws.numel(), _stream(stream)), "lcq_encode_batch")


def lcq_ldl_factor(H, d: int, U, ws, D=None, stream=None):
    n = H.shape[0]
    _check(lib().lcq_ldl_factor(_ptr(H), n, d, _ptr(U), _ptr(D), _ptr(ws), ws.numel(), _stream(stream)),
           "lcq_ldl_factor")


def lcq_ldlq(W, A, b, U, d: int, ws, packed=None, codes=None, latent=None, mse=None, stream=None):
    m, n = W.shape
    _check(lib().lcq_ldlq(_ptr(W), m, n, d, _ptr(A), _ptr(b), _ptr(U), _ptr(packed), _ptr(codes), _ptr(latent),
                          _ptr(mse), _ptr(ws), ws.numel(), _stream(stream)), "lcq_ldlq")


def lcq_decode(packed, n: int, d: int, A, b, W_hat_f32=None, W_hat_bf16=None, stream=None):
    m = packed.shape[0]
    _check(lib().lcq_decode(_ptr(packed), m, n, d, _ptr(A), _ptr(b), _ptr(W_hat_f32), _ptr(W_hat_bf16),
                            _stream(stream)), "lcq_decode")


def lcq_activation_transform(X, d: int, A, b, Xp=None, r=None, stream=None):
    """X' = X_g A (bf16, into Xp) and r = sum_g X_g . b (fp32, into r) per token; either output may be None."""
    N, n = X.shape
    _check(lib().lcq_activation_transform(_ptr(X), N, n, d, _ptr(A), _ptr(b), _ptr(Xp), _ptr(r), _stream(stream)),
           "lcq_activation_transform")


def lcq_pack2b(codes, packed, stream=None):
    m, n = codes.shape
    _check(lib().lcq_pack2b(_ptr(codes), m, n, _ptr(packed), _stream(stream)), "lcq_pack2b")


def lcq_linear_fwd(X, P, d: int, A, b, Y, ws, packed_saved=None, latent_scale=1.0, latent_offset=0.0,
                   ste_mode=LCQ_STE_IDENTITY, stream=None):
    N = X.shape[0]
    m, n = P.shape
    o = _opts(latent_scale, latent_offset, ste_mode)
    _check(lib().lcq_linear_fwd(_ptr(X), N, _ptr(P), m, n, d, _ptr(A), _ptr(b), ctypes.byref(o), _ptr(Y),
                                _ptr(packed_saved), _ptr(ws), ws.numel(), _stream(stream)), "lcq_linear_fwd")


def lcq_linear_bwd(X, dY, packed_saved, m: int, n: int, d: int, A, b, dP, dA, db, ws, dX=None, P=None,
                   latent_scale=1.0, latent_offset=0.0, ste_mode=LCQ_STE_IDENTITY, dge_k=0.0, dge_grad_max=0.0,
                   stream=None):
    N = X.shape[0]
    o = _opts(latent_scale, latent_offset, ste_mode, dge_k, dge_grad_max)
    _check(lib().lcq_linear_bwd(_ptr(X), _ptr(dY), _ptr(packed_saved), _ptr(P), N, m, n, d, _ptr(A), _ptr(b),
                                ctypes.byref(o), _ptr(dX), _ptr(dP), _ptr(dA), _ptr(db), _ptr(ws), ws.numel(),
                                _stream(stream)), "lcq_linear_bwd")


def lcq_gemm_packed2b(X, packed, n: int, d: int, A, b, Y, ws, stream=None):
    N = X.shape[0]
    m = packed.shape[0]
    _check(lib().lcq_gemm_packed2b(_ptr(X), N, _ptr(packed), m, n, d, _ptr(A), _ptr(b), _ptr(Y), _ptr(ws),
                                   ws.numel(), _stream(stream)), "lcq_gemm_packed2b")


def lcq_gemm_packed2b_noalloc(X, packed, n: int, d: int, A, b, Y, device_status=None, stream=None):
    """Deployment product with the library's static scratch instead of a workspace (N <= 16, n <= 32768).
    For callers that must not allocate device memory; overlapping calls race on the shared scratch."""
    N = X.shape[0]
    m = packed.shape[0]
    _check(lib().lcq_gemm_packed2b_noalloc(_ptr(X), N, _ptr(packed), m, n, d, _ptr(A), _ptr(b), _ptr(Y),
                                           _ptr(device_status), _stream(stream)), "lcq_gemm_packed2b_noalloc")


def lcq_device_status(ws, clear: bool = False, stream=None) -> int:
    out = ctypes.c_int32(0)
    _check(lib().lcq_device_status(_ptr(ws), _stream(stream), ctypes.byref(out), int(bool(clear))),
           "lcq_device_status")
    return int(out.value)


def lcq_selftest_wait_timeout(ws, stream=None):
    """Run the bounded-wait self-test kernel (about 2 s); the workspace status then reads LCQ_ERR_TIMEOUT."""
    _check(lib().lcq_selftest_wait_timeout(_ptr(ws), _stream(stream)), "lcq_selftest_wait_timeout")


def lcq_hadamard(inp, out, stream=None):
    rows, n = inp.shape
    _check(lib().lcq_hadamard(_ptr(inp), rows, n, _ptr(out), _stream(stream)), "lcq_hadamard")


def lcq_gemm_packed2b_hadamard(X, packed, n: int, d: int, A, b, Y, ws, stream=None):
    N = X.shape[0]
    m = packed.shape[0]
    _check(lib().lcq_gemm_packed2b_hadamard(_ptr(X), N, _ptr(packed), m, n, d, _ptr(A), _ptr(b), _ptr(Y), _ptr(ws),
                                            ws.numel(), _stream(stream)), "lcq_gemm_packed2b_hadamard")


def lcq_init_codebook(G, d: int, A, b, stream=None):
    _check(lib().lcq_init_codebook(_ptr(G), d, _ptr(A), _ptr(b), _stream(stream)), "lcq_init_codebook")


def lcq_init_latent(packed, n: int, P, stream=None):
    """Writes P = s (z - t) (Eq. xavier_preprocess); returns (s, t) for lcq_linear_fwd's latent affine."""
    m = packed.shape[0]
    s_, t_ = ctypes.c_float(0.0), ctypes.c_float(0.0)
    _check(lib().lcq_init_latent(_ptr(packed), m, n, _ptr(P), ctypes.byref(s_), ctypes.byref(t_), _stream(stream)),
           "lcq_init_latent")
    return float(s_.value), float(t_.value)


def lcq_launch_count() -> int:
    return int(lib().lcq_launch_count())


def lcq_trace_enable(on: bool = True):
    _check(lib().lcq_trace_enable(int(bool(on))), "lcq_trace_enable")


def lcq_trace_read() -> dict:
    """{kernel kind: (launches, total milliseconds)} of the events recorded since tracing was enabled."""
    out = {}
    for k, name in enumerate(KERNEL_KINDS):
        cnt, ms = ctypes.c_uint64(0), ctypes.c_double(0.0)
        _check(lib().lcq_trace_read(k, ctypes.byref(cnt), ctypes.byref(ms)), "lcq_trace_read")
        if cnt.value:
            out[name] = (int(cnt.value), float(ms.value))
    return out
