"""The allocation-free deployment product against the workspace version.

lcq_gemm_packed2b_noalloc serves callers that must not allocate device memory (a process
that gives all device memory to its own pool at start-up, a C caller without a device
allocator): its scratch is a static device array inside the library. This file is named to
be collected last, so that a run stopping at its first failure has run every other test.
It must pass both alone in a fresh process and after the rest of the suite."""
import ctypes

import numpy as np
import pytest

import paper_2606_10531_gb300 as lcq
from paper_2606_10531_gb300 import workloads as wl
from tests.gpu_util import TOL_BF16, config_A, config_b, dev, dev_bf16, empty_bf16, host_bf16, max_rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_10531_gb300 import build
    build.build()
    lcq.lib()


def _case(N, m, n, d, seed):
    rng = np.random.default_rng(seed)
    packed = rng.integers(0, 256, (m, n // 4), dtype=np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    Xb = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    return dev_bf16(Xb), dev(packed), dev(A), dev(b)


def _noalloc_c_abi(X, packed, n, d, A, b, Y, status):
    """Direct C-ABI call (no Python-side workspace anywhere); status may be None (NULL)."""
    import torch
    L = lcq.lib()
    return L.lcq_gemm_packed2b_noalloc(ctypes.c_void_p(X.data_ptr()), X.shape[0], ctypes.c_void_p(packed.data_ptr()),
                                       packed.shape[0], n, d, ctypes.c_void_p(A.data_ptr()),
                                       ctypes.c_void_p(b.data_ptr()), ctypes.c_void_p(Y.data_ptr()),
                                       ctypes.c_void_p(status.data_ptr() if status is not None else None),
                                       ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def test_noalloc_matches_workspace_version_on_two_calls_in_a_row():
    """Both entry points run the same kernels on the same inputs, so the results are bit-identical.
    Each problem is called twice in a row: the second call reuses the static scratch the first left."""
    import torch
    # the largest problem the static scratch holds (16 tokens, n = 32768), then smaller ones
    for (N, m, n, d, seed) in [(16, 1000, 4096, 8, 11), (3, 777, 2048, 4, 12), (16, 300, 32768, 8, 15),
                               (1, 333, 8192, 8, 16)]:
        X, packed, A, b = _case(N, m, n, d, seed)
        Y_ref = empty_bf16(N, m)
        ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
        lcq.lcq_gemm_packed2b(X, packed, n, d, A, b, Y_ref, ws)
        for call in range(2):
            Y = empty_bf16(N, m)
            status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
            assert _noalloc_c_abi(X, packed, n, d, A, b, Y, status if call == 0 else None) == 0
            torch.cuda.synchronize()
            if call == 0:
                assert int(status.item()) == 0
            assert torch.equal(Y, Y_ref), (N, m, n, d, call)
        assert max_rel(host_bf16(Y), host_bf16(Y_ref)) <= TOL_BF16


def test_noalloc_rejects_problems_beyond_its_scratch():
    import torch
    X, packed, A, b = _case(17, 64, 512, 8, 13)
    Y = empty_bf16(17, 64)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert _noalloc_c_abi(X, packed, 512, 8, A, b, Y, status) == 10      # LCQ_ERR_LIMIT: N > 16
    X, packed, A, b = _case(1, 8, 32776, 8, 14)
    Y = empty_bf16(1, 8)
    assert _noalloc_c_abi(X, packed, 32776, 8, A, b, Y, status) == 10    # LCQ_ERR_LIMIT: n > 32768


def test_noalloc_rejects_bad_arguments_before_enqueueing():
    """Invalid arguments return their error code and enqueue nothing, so the status word that the
    previous call left in the static scratch stays as it was (read back through a valid call)."""
    import torch
    X, packed, A, b = _case(2, 64, 512, 8, 17)
    Y = empty_bf16(2, 64)
    assert _noalloc_c_abi(X, packed, 512, 5, A, b, Y, None) == 4         # LCQ_ERR_UNSUPPORTED: d = 5
    assert _noalloc_c_abi(X, packed, 500, 8, A, b, Y, None) == 2         # LCQ_ERR_SHAPE: n % 8 != 0
    L = lcq.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = L.lcq_gemm_packed2b_noalloc(ctypes.c_void_p(X.data_ptr()), 2, ctypes.c_void_p(packed.data_ptr()), 64, 512, 8,
                                     None, ctypes.c_void_p(b.data_ptr()), ctypes.c_void_p(Y.data_ptr()), None, stream)
    assert rc == 1                                                        # LCQ_ERR_NULL: A missing
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    assert _noalloc_c_abi(X, packed, 512, 8, A, b, Y, status) == 0
    torch.cuda.synchronize()
    assert int(status.item()) == 0
