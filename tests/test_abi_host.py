"""Host-only checks of the C ABI: the library loads, exports every symbol include/lcq.h
declares, and rejects bad arguments synchronously, before anything is enqueued on a GPU.
The pointers used here are never dereferenced: validation fails first."""
import ctypes
import os
import re

import pytest

import paper_2606_10531_gb300 as lcq
from paper_2606_10531_gb300 import build as lcq_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lcq.h")

OK, NULL, SHAPE, ALIGN, UNSUP, WS, ARG = 0, 1, 2, 3, 4, 5, 9
FAKE = 0x7F0000000000          # 256-byte aligned fake device address (never dereferenced)


@pytest.fixture(scope="module")
def L():
    lcq_build.build()
    return lcq.load_library()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(lcq_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_six_hot_path_calls():
    names = declared_functions()
    for want in ("lcq_encode", "lcq_decode", "lcq_linear_fwd", "lcq_linear_bwd", "lcq_pack2b", "lcq_gemm_packed2b"):
        assert want in names


def test_library_exports_every_declared_symbol(L):
    names = declared_functions()
    assert names, "no declarations parsed"
    for name in names:
        assert hasattr(L, name), name
    assert set(names) <= set(lcq.EXPORTS)


def test_status_strings(L):
    for s in range(0, 10):
        assert L.lcq_status_string(s)
    assert L.lcq_status_string(0) == b"ok"


def test_workspace_size_monotone_and_rejects_bad_d(L):
    for op in (1, 2, 3, 4):
        a = L.lcq_workspace_size(op, 16, 64, 64, 8)
        b = L.lcq_workspace_size(op, 32, 128, 128, 8)
        assert 0 < a <= b
    assert L.lcq_workspace_size(2, 16, 64, 64, 5) == 0
    assert L.lcq_workspace_size(99, 16, 64, 64, 4) == 0
    # forward workspace holds the bf16 decoded weights
    assert L.lcq_workspace_size(2, 1, 4096, 4096, 8) >= 4096 * 4096 * 2


def _encode(L, W=FAKE, m=8, n=16, d=4, A=FAKE, b=FAKE, packed=FAKE, ws=FAKE, ws_bytes=1 << 20):
    return L.lcq_encode(W, m, n, d, A, b, packed, None, None, None, ws, ws_bytes, None)


def test_encode_validation(L):
    assert _encode(L, d=5) == UNSUP
    assert _encode(L, n=12) == SHAPE          # n % 8 != 0
    assert _encode(L, m=-1) == SHAPE
    assert _encode(L, W=None) == NULL
    assert _encode(L, A=None) == NULL
    assert _encode(L, W=FAKE + 4) == ALIGN
    assert _encode(L, packed=FAKE + 8) == ALIGN
    assert _encode(L, ws=None) == WS
    assert _encode(L, ws_bytes=16) == WS
    assert _encode(L, ws=FAKE + 16) == ALIGN   # workspace must be 256-byte aligned


def test_linear_validation(L):
    o = lcq.lcq_opts(1.0, 0.0, 0, 0, 0.0, 0.0)
    big = 1 << 30
    fwd = lambda **k: L.lcq_linear_fwd(k.get("X", FAKE), k.get("N", 4), k.get("P", FAKE), k.get("m", 8),  # noqa: E731
                                       k.get("n", 16), k.get("d", 8), FAKE, FAKE, k.get("o", ctypes.byref(o)),
                                       k.get("Y", FAKE), None, FAKE, k.get("ws_bytes", big), None)
    assert fwd(d=3) == UNSUP
    assert fwd(N=-2) == SHAPE
    assert fwd(X=None) == NULL
    assert fwd(Y=FAKE + 2) == ALIGN
    assert fwd(ws_bytes=8) == WS
    bad = lcq.lcq_opts(0.0, 0.0, 0, 0, 0.0, 0.0)
    assert fwd(o=ctypes.byref(bad)) == ARG
    bad_mode = lcq.lcq_opts(1.0, 0.0, 7, 0, 0.0, 0.0)
    assert fwd(o=ctypes.byref(bad_mode)) == UNSUP
    bwd = lambda **k: L.lcq_linear_bwd(FAKE, FAKE, FAKE, k.get("P", None), 4, k.get("m", 8), 16, 8, FAKE,  # noqa: E731
                                       FAKE, k.get("o", None), None, FAKE, k.get("dA", FAKE), FAKE, FAKE, big, None)
    assert fwd(m=12) != SHAPE                       # the forward takes any output width m
    assert bwd(m=12) == SHAPE                       # the backward's dY rows are TMA operands: m % 8 == 0
    clipped = lcq.lcq_opts(1.0, 0.0, 1, 0, 0.0, 0.0)
    assert bwd(o=ctypes.byref(clipped)) == NULL     # CLIPPED needs P
    dge = lcq.lcq_opts(1.0, 0.0, 2, 0, 5.0, 3.0)
    assert bwd(o=ctypes.byref(dge)) == NULL         # DGE needs P
    assert bwd(dA=None) == NULL


def test_packed_and_decode_validation(L):
    assert L.lcq_pack2b(FAKE, 4, 6, FAKE, None) == SHAPE
    assert L.lcq_pack2b(None, 4, 8, FAKE, None) == NULL
    assert L.lcq_decode(FAKE, 4, 16, 8, FAKE, FAKE, None, None, None) == NULL
    assert L.lcq_decode(FAKE, 4, 16, 6, FAKE, FAKE, FAKE, None, None) == UNSUP
    assert L.lcq_gemm_packed2b(FAKE, 1, FAKE, 8, 16, 8, FAKE, FAKE, FAKE, FAKE, 8, None) == WS


def test_empty_problems_need_no_device(L):
    # nothing to do: returns before touching CUDA
    assert L.lcq_decode(None, 0, 16, 8, FAKE, FAKE, None, None, None) == OK
    assert L.lcq_pack2b(None, 0, 16, None, None) == OK


def test_encode_batch_validation(L):
    ws_ok = FAKE
    big = 1 << 30
    items = (lcq.lcq_encode_item * 2)()
    for k in range(2):
        items[k] = lcq.lcq_encode_item(FAKE, 8, 16, FAKE, FAKE, FAKE, None, None, None)
    eb = lambda arr=items, count=2, d=4, ws=ws_ok, ws_bytes=big: L.lcq_encode_batch(arr, count, d, ws, ws_bytes, None)  # noqa: E731
    assert eb(arr=None) == NULL
    assert eb(count=0) == SHAPE
    assert eb(count=17) == SHAPE
    assert eb(d=5) == UNSUP
    assert eb(ws_bytes=16) == WS
    bad = (lcq.lcq_encode_item * 2)()
    bad[0] = lcq.lcq_encode_item(FAKE, 8, 16, FAKE, FAKE, FAKE, None, None, None)
    bad[1] = lcq.lcq_encode_item(FAKE, 8, 12, FAKE, FAKE, FAKE, None, None, None)     # n % 8 != 0
    assert eb(arr=bad) == SHAPE
    bad[1] = lcq.lcq_encode_item(FAKE, 8, 16, None, FAKE, FAKE, None, None, None)     # A missing
    assert eb(arr=bad) == NULL
    bad[1] = lcq.lcq_encode_item(FAKE + 4, 8, 16, FAKE, FAKE, FAKE, None, None, None)  # W misaligned
    assert eb(arr=bad) == ALIGN
    assert L.lcq_workspace_size(6, 0, 0, 0, 8) == 0
    assert L.lcq_workspace_size(6, 17, 0, 0, 8) == 0
    assert 0 < L.lcq_workspace_size(6, 1, 0, 0, 8) < L.lcq_workspace_size(6, 7, 0, 0, 8)


def test_rotation_transform_ldlq_and_init_validation(L):
    big = 1 << 30
    assert L.lcq_hadamard(FAKE, 2, 12, FAKE, None) == SHAPE          # n % 8 != 0
    assert L.lcq_hadamard(None, 0, 16, None, None) == OK             # empty: no device
    assert L.lcq_hadamard(None, 2, 16, FAKE, None) == NULL
    assert L.lcq_hadamard(FAKE + 4, 2, 16, FAKE, None) == ALIGN

    def gh(X=FAKE, N=2, n=64, d=8, A=FAKE, ws=FAKE, ws_bytes=big):
        return L.lcq_gemm_packed2b_hadamard(X, N, FAKE, 8, n, d, A, FAKE, FAKE, ws, ws_bytes, None)
    assert gh(d=5) == UNSUP
    assert gh(N=-1) == SHAPE
    assert gh(n=60) == SHAPE
    assert gh(X=None) == NULL
    assert gh(A=None) == NULL
    assert gh(ws_bytes=16) == WS
    assert gh(ws=FAKE + 16) == ALIGN                                 # workspace must be 256-byte aligned

    def xf(N=4, n=64, d=8, A=FAKE, Xp=FAKE, r=FAKE):
        return L.lcq_activation_transform(FAKE, N, n, d, A, FAKE, Xp, r, None)
    assert xf(d=6) == UNSUP
    assert xf(N=-1) == SHAPE
    assert xf(N=0) == OK
    assert xf(Xp=None, r=None) == NULL                              # nothing to write
    assert xf(r=FAKE + 4) == ALIGN
    assert xf(A=None) == NULL

    assert L.lcq_ldl_factor(FAKE, 64, 5, FAKE, FAKE, FAKE, big, None) == UNSUP
    assert L.lcq_ldl_factor(FAKE, 0, 8, FAKE, FAKE, FAKE, big, None) == OK
    assert L.lcq_ldl_factor(FAKE, 65544, 8, FAKE, FAKE, FAKE, big, None) == SHAPE   # n > 65536
    assert L.lcq_ldl_factor(None, 64, 8, FAKE, FAKE, FAKE, big, None) == NULL
    assert L.lcq_ldl_factor(FAKE, 64, 8, FAKE, FAKE, FAKE, 16, None) == WS

    def lq(n=64, A=FAKE, U=FAKE, ws_bytes=big):
        return L.lcq_ldlq(FAKE, 64, n, 8, A, FAKE, U, FAKE, None, None, None, FAKE, ws_bytes, None)
    assert lq(n=60) == SHAPE
    assert lq(U=None) == NULL
    assert lq(A=None) == NULL
    assert lq(ws_bytes=16) == WS

    assert L.lcq_init_codebook(FAKE, 6, FAKE, FAKE, None) == UNSUP
    assert L.lcq_init_codebook(None, 8, FAKE, FAKE, None) == NULL
    assert L.lcq_init_latent(FAKE, 4, 6, FAKE, None, None, None) == SHAPE   # n % 4 != 0
    assert L.lcq_init_latent(FAKE, 0, 0, FAKE, None, None, None) == SHAPE


@pytest.mark.parametrize("m,n", [(0, 16), (4096, 0), (0, 14336)])
def test_init_latent_constants_match_the_oracle(L, m, n):
    """The preprocessing constants of Eq. xavier_preprocess (s = 2a/3, t = 3/2, a = sqrt(6/(m+n))) are
    computed on the host; for an empty matrix the call returns them without touching a device. s is
    the oracle's fp64 value rounded to fp32."""
    import numpy as np
    import oracle
    s, t = ctypes.c_float(-1.0), ctypes.c_float(-1.0)
    assert L.lcq_init_latent(None, m, n, None, ctypes.byref(s), ctypes.byref(t), None) == OK
    _, s_ref, t_ref = oracle.init_latent(np.zeros((m, n), np.uint8), m, n)
    assert s.value == float(np.float32(s_ref))
    assert t.value == t_ref == 1.5


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(ImportError, match="liblcq.so not found"):
        lcq.load_library(str(tmp_path / "liblcq.so"))


def test_product_package_never_reaches_the_oracle():
    """The binding and the library sources import, link or execute nothing under oracle/."""
    pkg = os.path.join(ROOT, "paper_2606_10531_gb300")
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath or "__pycache__" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp", ".c")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b|oracle/|brute\.c|lcvq", text, flags=re.M), f


def test_no_kernel_spills_registers(L):
    """ptxas resource reports of the build: no entry function spills registers (no exemptions)."""
    import re as _re
    if not all(os.path.exists(lcq_build.ptxas_report(s)) for s in lcq_build.SOURCES):
        lcq_build.build(force=True)
    entries = 0
    for src in lcq_build.SOURCES:
        cur = None
        for line in open(lcq_build.ptxas_report(src)):
            m = _re.search(r"Compiling entry function '(\S+)'", line)
            if m:
                cur = m.group(1)
                entries += 1
                continue
            m = _re.search(r"(\d+) bytes spill stores, (\d+) bytes spill loads", line)
            if m and cur:
                assert m.group(1) == m.group(2) == "0", (src, cur, line.strip())
    assert entries > 20
