"""Parity of every liblcq entry point against the CPU oracle on oracle-sized inputs that
span several tiles, chunks and ragged tails, plus the degenerate cases.

Matching rules: codes and packed bytes bit-exact (encode excludes latent values within 1e-5
of a rounding boundary and reports how many); fp32 decoded weights within 1e-6 absolute;
bf16 outputs and all gradients within 2e-2 of max|ref| (fp64 oracle)."""
import numpy as np
import pytest

import oracle
import paper_2606_10531_gb300 as lcq
from paper_2606_10531_gb300 import workloads as wl
from tests.gpu_util import (TOL_BF16, TOL_DECODE_F32, config_A, config_b, dev, dev_bf16, digit_product_bound, empty_bf16,
                            host_bf16, max_rel, within)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_10531_gb300 import build
    build.build()
    lcq.lib()


def T():
    import torch
    return torch


# ----------------------------------------------------------------------------- encode

ENCODE_CASES = [
    (512, 512, 4),      # the oracle-sized single layer
    (37, 24, 4),        # ragged: 888 weights, partial 16-weight slice
    (129, 4104, 8),     # several 16 KB chunks, ragged tail
    (300, 1000, 8),
    (1, 8, 8),          # one group
]


@pytest.mark.parametrize("m,n,d", ENCODE_CASES)
def test_encode_matches_oracle(m, n, d):
    torch = T()
    rng = np.random.default_rng(1000 + m + n + d)
    W = rng.normal(0, 0.02, (m, n)).astype(np.float32)
    heavy = rng.random((m, n)) < 0.01
    W[heavy] = (0.02 * rng.standard_t(4, heavy.sum())).astype(np.float32)
    A, b = config_A(d, rng), config_b(d, rng)
    ref = oracle.encode(W, A, b, d)

    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, n, d)
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    codes = torch.empty((m, n), dtype=torch.uint8, device="cuda")
    latent = torch.empty((m, n), dtype=torch.float32, device="cuda")
    mse = torch.empty(1, dtype=torch.float64, device="cuda")
    lcq.lcq_encode(dev(W), dev(A), dev(b), d, ws, packed=packed, codes=codes, latent=latent, mse=mse)
    assert lcq.lcq_device_status(ws) == 0

    z = codes.cpu().numpy()
    keep = ~ref["near"]
    mismatch = int(np.sum((z != ref["codes"]) & keep))
    assert mismatch == 0, f"{mismatch} codes differ away from rounding boundaries"
    assert set(np.unique(z)) <= {0, 1, 2, 3}
    assert np.array_equal(oracle.unpack2b(packed.cpu().numpy(), n)[keep], z[keep])
    assert np.array_equal(oracle.unpack2b(packed.cpu().numpy(), n), z)
    u = latent.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(u - ref["latent"]) <= 1e-5 * np.maximum(1.0, np.abs(ref["latent"])))
    # MSE of the GPU's own codes, oracle arithmetic; and vs the oracle's MSE
    mse_own = oracle.mse(W, z, A, b, d)
    assert abs(mse.item() - mse_own) <= 1e-4 * mse_own
    assert abs(mse.item() - ref["mse"]) <= 1e-4 * ref["mse"] + 1e-12
    print(f"near-boundary codes excluded: {int(np.sum(ref['near']))} of {m * n}")


@pytest.mark.parametrize("d", [4, 8])
@pytest.mark.parametrize("cond", [1e3, 1e6, 3e7])
def test_encode_inverse_accuracy_ill_conditioned(d, cond):
    # With b = 0 and a one-hot group w = e_g, the latent is u = A^{-1} e_g exactly (every other product
    # is an exact zero), so the latent output exposes the device's A^{-1} column by column. It must be
    # the fp64 inverse rounded to fp32, whatever the conditioning (the widest case takes the fp64
    # elimination path).
    torch = T()
    rng = np.random.default_rng(int(cond) + d)
    Q1, _ = np.linalg.qr(rng.normal(size=(d, d)))
    Q2, _ = np.linalg.qr(rng.normal(size=(d, d)))
    A = (0.02 * Q1 @ np.diag(np.logspace(0, -np.log10(cond), d)) @ Q2.T).astype(np.float32)
    b = np.zeros(d, dtype=np.float32)
    m = 4
    W = np.tile(np.eye(d, dtype=np.float32).reshape(1, d * d), (m, 1))      # groups e_0 .. e_{d-1}
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, d * d, d)
    latent = torch.empty((m, d * d), dtype=torch.float32, device="cuda")
    mse = torch.empty(1, dtype=torch.float64, device="cuda")
    lcq.lcq_encode(dev(W), dev(A), dev(b), d, ws, latent=latent, mse=mse)
    assert lcq.lcq_device_status(ws) == 0
    inv = oracle.inverse(A)                                  # fp64
    got = latent.cpu().numpy().astype(np.float64).reshape(m, d, d)   # [row][group g][k] = A^{-1}[k][g]
    for r in range(m):
        # fp32 rounding of each entry, plus the forward error of any fp64 inverse (~cond * 1e-16 of its norm)
        tol = 2.5e-7 * np.abs(inv) + 2e-8 * np.max(np.abs(inv))
        assert np.all(np.abs(got[r].T - inv) <= tol), f"max err/tol {np.max(np.abs(got[r].T - inv) / tol)}"


@pytest.mark.parametrize("d", [4, 8])
def test_encode_batch_matches_single_calls_and_oracle(d):
    # the batch gives, matrix by matrix, exactly what lcq_encode gives; and both match the oracle
    torch = T()
    rng = np.random.default_rng(77 + d)
    shapes = [(512, 512), (37, 24), (129, 4104), (0, 64), (300, 1000), (64, 8), (700, 2048), (5, 40),
              (1024, 512), (33, 96), (16, 16), (250, 1024)]      # 12 matrices: some warps invert two
    items, singles, refs = [], [], []
    for k, (m, n) in enumerate(shapes):
        W = rng.normal(0, 0.02, (m, n)).astype(np.float32)
        A, b = config_A(d, rng), config_b(d, rng)
        it = {"W": dev(W), "A": dev(A), "b": dev(b),
              "packed": torch.empty((m, n // 4), dtype=torch.uint8, device="cuda"),
              "codes": torch.empty((m, n), dtype=torch.uint8, device="cuda") if k % 2 == 0 else None,
              "latent": torch.empty((m, n), dtype=torch.float32, device="cuda") if k % 3 == 0 else None,
              "mse": torch.full((1,), -1.0, dtype=torch.float64, device="cuda") if k != 5 else None}
        items.append(it)
        one = {kk: (torch.empty_like(v) if kk in ("packed", "codes", "latent", "mse") and v is not None else v)
               for kk, v in it.items()}
        singles.append(one)
        refs.append((W, A, b))
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE_BATCH, len(items), 0, 0, d)
    for _ in range(2):                    # twice: the per-matrix counters must come back to zero
        lcq.lcq_encode_batch(items, d, ws)
    assert lcq.lcq_device_status(ws) == 0
    for it, one, (W, A, b) in zip(items, singles, refs):
        m, n = W.shape
        ws1 = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, n, d)
        lcq.lcq_encode(one["W"], one["A"], one["b"], d, ws1, packed=one["packed"], codes=one["codes"],
                       latent=one["latent"], mse=one["mse"])
        for key in ("packed", "codes", "latent"):
            if it[key] is not None:
                assert torch.equal(it[key], one[key]), key
        if it["mse"] is not None:
            assert it["mse"].item() == one["mse"].item()
        if m * n == 0:
            if it["mse"] is not None:
                assert it["mse"].item() == 0.0
            continue
        ref = oracle.encode(W, A, b, d)
        z = oracle.unpack2b(it["packed"].cpu().numpy(), n)
        keep = ~ref["near"]
        assert int(np.sum((z != ref["codes"]) & keep)) == 0
        if it["mse"] is not None:
            assert abs(it["mse"].item() - ref["mse"]) <= 1e-4 * ref["mse"] + 1e-12


def test_encode_nonfinite_inputs():
    torch = T()
    d, m, n = 8, 4, 32
    rng = np.random.default_rng(5)
    W = rng.normal(0, 0.02, (m, n)).astype(np.float32)
    W[0, :3] = [np.nan, np.inf, -np.inf]
    A, b = config_A(d, rng), config_b(d, rng)
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, n, d)
    codes = torch.empty((m, n), dtype=torch.uint8, device="cuda")
    lcq.lcq_encode(dev(W), dev(A), dev(b), d, ws, codes=codes)
    ref = oracle.encode(np.where(np.isfinite(W), W, 0), A, b, d)  # rows 1.. are finite
    z = codes.cpu().numpy()
    assert np.array_equal(z[1:], ref["codes"][1:])
    assert set(np.unique(z)) <= {0, 1, 2, 3}
    # group 0 holds the non-finite values: every latent coordinate mixing them is NaN/inf
    Ainv = np.linalg.inv(A.astype(np.float64))
    with np.errstate(invalid="ignore"):
        u0 = Ainv @ (W[0, :8].astype(np.float64) - b)
    assert np.array_equal(z[0, :8], oracle.round_clamp(u0))


def test_encode_singular_A_sets_status():
    torch = T()
    d, m, n = 4, 8, 16
    A = np.eye(d, dtype=np.float32)
    A[2] = 0.0
    W = np.random.default_rng(0).normal(0, 0.02, (m, n)).astype(np.float32)
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, n, d)
    codes = torch.full((m, n), 7, dtype=torch.uint8, device="cuda")
    lcq.lcq_encode(dev(W), dev(A), dev(np.zeros(d, np.float32)), d, ws, codes=codes)
    assert lcq.lcq_device_status(ws, clear=True) == 7   # LCQ_ERR_SINGULAR
    assert int(codes.max()) == 0
    assert lcq.lcq_device_status(ws) == 0


def test_encode_empty_writes_zero_mse():
    torch = T()
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, 0, 16, 4)
    mse = torch.full((1,), 5.0, dtype=torch.float64, device="cuda")
    A = dev(np.eye(4, dtype=np.float32))
    lcq.lcq_encode(torch.empty((0, 16), device="cuda"), A, dev(np.zeros(4, np.float32)), 4, ws, mse=mse)
    assert mse.item() == 0.0


# ----------------------------------------------------------------------------- decode / pack

@pytest.mark.parametrize("m,n,d", [(64, 512, 4), (33, 40, 8), (1, 8, 8), (257, 1032, 4)])
def test_decode_matches_oracle(m, n, d):
    torch = T()
    rng = np.random.default_rng(m * 7 + n)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    ref = oracle.decode(Z, A, b, d)
    f32 = torch.empty((m, n), dtype=torch.float32, device="cuda")
    h16 = empty_bf16(m, n)
    lcq.lcq_decode(dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), W_hat_f32=f32, W_hat_bf16=h16)
    assert np.max(np.abs(f32.cpu().numpy() - ref)) <= TOL_DECODE_F32
    # bf16: within half a bf16 ulp of the exact value, plus the fp32 error
    got = host_bf16(h16)
    assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0 ** -8 + TOL_DECODE_F32)


@pytest.mark.parametrize("m,n", [(64, 512), (3, 4), (5, 12), (17, 1028)])
def test_pack2b_matches_oracle(m, n):
    torch = T()
    Z = np.random.default_rng(m + n).integers(0, 256, (m, n)).astype(np.uint8)   # high bits must be ignored
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    lcq.lcq_pack2b(dev(Z), packed)
    assert np.array_equal(packed.cpu().numpy(), oracle.pack2b(Z & 3))


# ----------------------------------------------------------------------------- training layer

LINEAR_CASES = [
    # N tokens, m out, n in, d; the GEMMs run 256 x 256 tiles on pairs of CTAs
    (64, 512, 512, 4),     # the oracle-sized layer of the workload list
    (200, 384, 320, 8),    # 1 x 2 pair tiles, ragged in M and N, 5 K-blocks
    (130, 136, 72, 4),     # ragged everywhere, K tail of 8
    (1, 8, 8, 8),          # one token, one group
    (520, 1024, 256, 8),   # 3 x 4 pair tiles with two TMEM accumulators in flight
    # on 76 pairs (152 SMs) every GEMM of this case ends in a partial wave whose tiles run as 256 x 128
    # halves: forward 16 x 5 pair tiles, dX 16 x 16, dW 5 x 16
    (4096, 1280, 4096, 8),
    # ragged in M, N and K (K tails of 8, 40 and 32) with split last waves in the forward (16 x 5 pair
    # tiles) and dW (5 x 17)
    (4000, 1256, 4104, 4),
]


def _linear_inputs(N, m, n, d, seed):
    rng = np.random.default_rng(seed)
    W = rng.normal(0, 0.02, (m, n)).astype(np.float32)
    A, b = config_A(d, rng), config_b(d, rng)
    P = oracle.encode(W, A, b, d)["latent"].astype(np.float32)   # proxy weights = latent of W
    X = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    dY = wl.bf16_bits(rng.normal(0, 1, (N, m)).astype(np.float32))
    return P, A, b, X, dY


@pytest.mark.parametrize("N,m,n,d", LINEAR_CASES)
@pytest.mark.parametrize("ste", ["identity", "clipped", "dge"])
def test_linear_fwd_bwd_match_oracle(N, m, n, d, ste):
    torch = T()
    P, A, b, Xb, dYb = _linear_inputs(N, m, n, d, seed=N * 31 + m + n + d)
    X, dY = wl.bf16_to_f32(Xb), wl.bf16_to_f32(dYb)
    s, t = (1.0, 0.0) if ste == "identity" else (0.5, 0.75)
    mode = {"identity": lcq.LCQ_STE_IDENTITY, "clipped": lcq.LCQ_STE_CLIPPED, "dge": lcq.LCQ_STE_DGE}[ste]
    Z = oracle.quantize(P, s, t)
    Yref = oracle.linear_fwd(X, Z, A, b, d)
    g = oracle.linear_bwd(X, dY, Z, A, b, d, P=P, s=s, t=t, ste=ste)

    Pd, Ad, bd, Xd, dYd = dev(P), dev(A), dev(b), dev_bf16(Xb), dev_bf16(dYb)
    Y = empty_bf16(N, m)
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    wsf = lcq.workspace(lcq.LCQ_OP_LINEAR_FWD, N, m, n, d)
    lcq.lcq_linear_fwd(Xd, Pd, d, Ad, bd, Y, wsf, packed_saved=packed, latent_scale=s, latent_offset=t,
                       ste_mode=mode)
    assert np.array_equal(packed.cpu().numpy(), oracle.pack2b(Z)), "quantized integer weights differ"
    assert max_rel(host_bf16(Y), Yref) <= TOL_BF16

    wsb = lcq.workspace(lcq.LCQ_OP_LINEAR_BWD, N, m, n, d)
    dX = empty_bf16(N, n)
    dP = torch.empty((m, n), dtype=torch.float32, device="cuda")
    dA = torch.empty((d, d), dtype=torch.float32, device="cuda")
    db = torch.empty(d, dtype=torch.float32, device="cuda")
    lcq.lcq_linear_bwd(Xd, dYd, packed, m, n, d, Ad, bd, dP, dA, db, wsb, dX=dX, P=Pd, latent_scale=s,
                       latent_offset=t, ste_mode=mode)
    assert lcq.lcq_device_status(wsb) == 0 and lcq.lcq_device_status(wsf) == 0
    errs = {"dX": max_rel(host_bf16(dX), g["dX"]), "dP": max_rel(dP.cpu().numpy(), g["dP"]),
            "dA": max_rel(dA.cpu().numpy(), g["dA"]), "db": max_rel(db.cpu().numpy(), g["db"])}
    assert all(e <= TOL_BF16 for e in errs.values()), errs


def test_linear_forward_any_output_width():
    """The forward takes any number of output rows m (here 1250: Y's rows are not 16-byte aligned, so
    the GEMM epilogue stores them element by element); the backward, whose dY rows are TMA operands,
    rejects m % 8 != 0 before it enqueues anything."""
    torch = T()
    N, m, n, d = 4000, 1250, 4104, 4
    P, A, b, Xb, dYb = _linear_inputs(N, m, n, d, seed=4242)
    Z = oracle.quantize(P)
    Yref = oracle.linear_fwd(wl.bf16_to_f32(Xb), Z, A, b, d)
    Y = empty_bf16(N, m)
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    wsf = lcq.workspace(lcq.LCQ_OP_LINEAR_FWD, N, m, n, d)
    lcq.lcq_linear_fwd(dev_bf16(Xb), dev(P), d, dev(A), dev(b), Y, wsf, packed_saved=packed)
    assert lcq.lcq_device_status(wsf) == 0
    assert np.array_equal(packed.cpu().numpy(), oracle.pack2b(Z))
    assert max_rel(host_bf16(Y), Yref) <= TOL_BF16
    wsb = lcq.workspace(lcq.LCQ_OP_LINEAR_BWD, N, m, n, d)
    dP = torch.empty((m, n), dtype=torch.float32, device="cuda")
    dA = torch.empty((d, d), dtype=torch.float32, device="cuda")
    db = torch.empty(d, dtype=torch.float32, device="cuda")
    with pytest.raises(lcq.LCQError) as e:
        lcq.lcq_linear_bwd(dev_bf16(Xb), dev_bf16(dYb), packed, m, n, d, dev(A), dev(b), dP, dA, db, wsb)
    assert e.value.status == 2                     # LCQ_ERR_SHAPE


def test_linear_backward_is_bitwise_reproducible():
    torch = T()
    N, m, n, d = 300, 512, 256, 8
    P, A, b, Xb, dYb = _linear_inputs(N, m, n, d, seed=77)
    Ad, bd, Xd, dYd = dev(A), dev(b), dev_bf16(Xb), dev_bf16(dYb)
    packed = dev(oracle.pack2b(oracle.quantize(P)))
    wsb = lcq.workspace(lcq.LCQ_OP_LINEAR_BWD, N, m, n, d)
    outs = []
    for _ in range(2):
        dP = torch.empty((m, n), dtype=torch.float32, device="cuda")
        dA = torch.empty((d, d), dtype=torch.float32, device="cuda")
        db = torch.empty(d, dtype=torch.float32, device="cuda")
        lcq.lcq_linear_bwd(Xd, dYd, packed, m, n, d, Ad, bd, dP, dA, db, wsb)
        outs.append((dP.cpu().numpy(), dA.cpu().numpy(), db.cpu().numpy()))
    for a, c in zip(outs[0], outs[1]):
        assert np.array_equal(a, c)


def test_linear_empty_tokens_gives_zero_gradients():
    torch = T()
    m, n, d = 16, 32, 8
    A = dev(config_A(d, np.random.default_rng(3)))
    b = dev(np.zeros(d, np.float32))
    X = torch.empty((0, n), dtype=torch.bfloat16, device="cuda")
    dY = torch.empty((0, m), dtype=torch.bfloat16, device="cuda")
    packed = torch.zeros((m, n // 4), dtype=torch.uint8, device="cuda")
    dP = torch.full((m, n), 3.0, device="cuda")
    dA = torch.full((d, d), 3.0, device="cuda")
    db = torch.full((d,), 3.0, device="cuda")
    ws = lcq.workspace(lcq.LCQ_OP_LINEAR_BWD, 0, m, n, d)
    lcq.lcq_linear_bwd(X, dY, packed, m, n, d, A, b, dP, dA, db, ws)
    assert float(dP.abs().max()) == 0 and float(dA.abs().max()) == 0 and float(db.abs().max()) == 0
    Y = torch.empty((0, m), dtype=torch.bfloat16, device="cuda")
    wsf = lcq.workspace(lcq.LCQ_OP_LINEAR_FWD, 0, m, n, d)
    lcq.lcq_linear_fwd(X, torch.zeros((m, n), device="cuda"), d, A, b, Y, wsf)


# ----------------------------------------------------------------------------- deployment product

@pytest.mark.parametrize("N", [1, 2, 3, 4, 5, 16, 17, 40])
@pytest.mark.parametrize("m,n,d", [(200, 512, 8), (64, 1024, 4), (70, 200, 4), (8, 8, 8), (1000, 4096, 8),
                                   (300, 8192, 4)])
def test_gemm_packed2b_matches_oracle(N, m, n, d):
    torch = T()
    rng = np.random.default_rng(N * 1000 + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    Xb = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
    lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert max_rel(host_bf16(Y), ref) <= TOL_BF16


# With n % 64 == 0 (n <= 32768), one token takes the integer (dp2a) kernel: activations as int16 with
# one scale per token (a bound on max|X'|), exact int32 sums. Its only errors are the int16 rounding
# (at most 2^-16 of the bound per element) and the bf16 output rounding (2^-9 relative), so it is held
# to a tighter bound than the bf16 parity bar, on heavy-tailed activations (1% of the columns x50).
# Two to four tokens take the tcgen05 kernel (exact integer digits, below), held to the elementwise
# bound of its rounding (digit_product_bound). (300, 28672) puts 56 activation tiles in shared memory
# next to the code ring.
TOL_DP = 4e-3


@pytest.mark.parametrize("N", [1, 2, 3, 4])
@pytest.mark.parametrize("m,n,d", [(1000, 4096, 8), (300, 8192, 4), (300, 28672, 8), (16, 64, 8), (4000, 512, 4)])
def test_gemm_packed2b_few_tokens_heavy_tailed(N, m, n, d):
    rng = np.random.default_rng(7 * N + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n))
    X[:, rng.random(n) < 0.01] *= 50.0
    Xb = wl.bf16_bits(X.astype(np.float32))
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
    lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_device_status(ws) == 0
    if N == 1:
        assert max_rel(host_bf16(Y), ref) <= TOL_DP
    else:
        assert within(host_bf16(Y), ref, digit_product_bound(wl.bf16_to_f32(Xb), Z, A, b, d, ref)) <= 1.0


# Shapes the integer kernels do not take (n % 64 != 0, or n > 32768) run the mma.sync kernel: X' in
# bf16, fp32 accumulation, the bf16 parity bar. n = 32832 streams its codes through the TMA ring.
@pytest.mark.parametrize("N", [2, 5, 8])
@pytest.mark.parametrize("m,n,d", [(300, 200, 4), (129, 1000, 8), (64, 32832, 8)])
def test_gemm_packed2b_mma_sync_shapes(N, m, n, d):
    rng = np.random.default_rng(13 * N + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    Xb = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
    lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_device_status(ws) == 0
    assert max_rel(host_bf16(Y), ref) <= TOL_BF16


def test_gemm_packed2b_one_token_zero_activations():
    # a half-zero token, and an all-zero token (scale 0)
    rng = np.random.default_rng(5)
    m, n, d, N = 256, 2048, 8, 1
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    for zero in ("half", "all"):
        X = rng.normal(0, 1, (N, n))
        X[0, :1024] = 0.0
        if zero == "all":
            X[0, :] = 0.0
        Xb = wl.bf16_bits(X.astype(np.float32))
        ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
        Y = empty_bf16(N, m)
        ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
        lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
        got = host_bf16(Y)
        if zero == "all":
            assert np.all(got == 0.0)
        else:
            assert max_rel(got, ref) <= TOL_DP


def test_gemm_packed2b_two_tokens_independent_scales():
    # two tokens, one all zero (outputs exactly 0), then one 1e4 x larger than the other: each token is
    # scaled on its own, so neither loses precision to the other
    rng = np.random.default_rng(11)
    m, n, d = 500, 4096, 8
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    for case in ("zero", "scaled"):
        X = rng.normal(0, 1, (2, n))
        if case == "zero":
            X[1, :] = 0.0
        else:
            X[1, :] *= 1e4
        Xb = wl.bf16_bits(X.astype(np.float32))
        ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
        Y = empty_bf16(2, m)
        ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, 2, m, n, d)
        lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
        assert lcq.lcq_device_status(ws) == 0
        got = host_bf16(Y)
        bound = digit_product_bound(wl.bf16_to_f32(Xb), Z, A, b, d, ref)
        assert within(got[0], ref[0], bound[0]) <= 1.0
        if case == "zero":
            assert np.all(got[1] == 0.0)
        else:
            assert within(got[1], ref[1], bound[1]) <= 1.0


# ----------------------------------------------------------------------------- failure detection

def test_bounded_wait_reports_timeout_and_context_stays_usable():
    """A wait on a flag nothing sets gives up after its limit and reports LCQ_ERR_TIMEOUT (8)."""
    import time
    torch = T()
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    t0 = time.time()
    lcq.lcq_selftest_wait_timeout(ws)
    assert lcq.lcq_device_status(ws, clear=True) == 8
    assert 1.0 < time.time() - t0 < 30.0
    assert lcq.lcq_device_status(ws) == 0
    # the context still works: a normal call afterwards
    Z = np.random.default_rng(1).integers(0, 4, (4, 16)).astype(np.uint8)
    packed = torch.empty((4, 4), dtype=torch.uint8, device="cuda")
    lcq.lcq_pack2b(dev(Z), packed)
    assert np.array_equal(packed.cpu().numpy(), oracle.pack2b(Z))


# ----------------------------------------------------------------------------- initialisation

@pytest.mark.parametrize("d", [4, 8])
def test_init_codebook_matches_oracle(d):
    torch = T()
    G = np.linalg.qr(np.random.default_rng(40 + d).normal(size=(d, d)))[0].astype(np.float32)
    A = torch.empty((d, d), dtype=torch.float32, device="cuda")
    b = torch.empty(d, dtype=torch.float32, device="cuda")
    lcq.lcq_init_codebook(dev(G), d, A, b)
    Aref, bref = oracle.init_codebook(G.astype(np.float64))
    np.testing.assert_allclose(A.cpu().numpy(), Aref, rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(b.cpu().numpy(), bref, rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("m,n", [(4096, 4096), (37, 24), (300, 1028)])
def test_init_latent_matches_oracle_and_requantizes_to_the_same_codes(m, n):
    torch = T()
    d = 4
    Z = np.random.default_rng(m + n).integers(0, 4, (m, n)).astype(np.uint8)
    packed = dev(oracle.pack2b(Z))
    P = torch.empty((m, n), dtype=torch.float32, device="cuda")
    s, t = lcq.lcq_init_latent(packed, n, P)
    Pref, sref, tref = oracle.init_latent(Z, m, n)
    assert abs(s - sref) <= 1e-7 * sref and t == tref
    np.testing.assert_allclose(P.cpu().numpy(), Pref, rtol=2e-7, atol=1e-9)
    # forward quantization with the returned (s, t) gives back exactly the integer weights
    if n % 8 == 0:
        A = dev(np.eye(d, dtype=np.float32))
        bz = dev(np.zeros(d, np.float32))
        N = 1
        X = torch.zeros((N, n), dtype=torch.bfloat16, device="cuda")
        Y = torch.empty((N, m), dtype=torch.bfloat16, device="cuda")
        saved = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
        ws = lcq.workspace(lcq.LCQ_OP_LINEAR_FWD, N, m, n, d)
        lcq.lcq_linear_fwd(X, P, d, A, bz, Y, ws, packed_saved=saved, latent_scale=s, latent_offset=t)
        assert np.array_equal(saved.cpu().numpy(), oracle.pack2b(Z))


# ----------------------------------------------------------------------------- Hadamard rotation

@pytest.mark.parametrize("rows,n", [(3, 8), (5, 96), (3, 64), (2, 1024), (2, 8192), (4, 14336), (3, 6144), (1, 16384),
                                    (2, 65536)])
def test_hadamard_rotation_matches_oracle(rows, n):
    torch = T()
    X = np.random.default_rng(rows + n).normal(size=(rows, n)).astype(np.float32)
    out = torch.empty((rows, n), dtype=torch.float32, device="cuda")
    lcq.lcq_hadamard(dev(X), out)
    np.testing.assert_allclose(out.cpu().numpy(), oracle.hadamard_rotate(X, n), rtol=1e-4, atol=1e-5)
    lcq.lcq_hadamard(out, out)                    # in place, and H H = I
    np.testing.assert_allclose(out.cpu().numpy(), X, rtol=1e-4, atol=1e-5)


# One token, n = 8192 and enough rows per unit: the rotation runs in the one-token kernel's prologue
# (one launch instead of two), in fp32 before the int16 activations, so the dp bound applies.
@pytest.mark.parametrize("d", [4, 8])
def test_gemm_packed2b_hadamard_fused_prologue(d):
    m, n, N = 7296, 8192, 1
    rng = np.random.default_rng(31 + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n))
    X[:, rng.random(n) < 0.01] *= 50.0
    Xb = wl.bf16_bits(X.astype(np.float32))
    ref = oracle.gemm_packed2b_hadamard(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B_HADAMARD, N, m, n, d)
    before = lcq.lcq_launch_count()
    lcq.lcq_gemm_packed2b_hadamard(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_launch_count() - before == 1          # no separate rotation kernel
    assert lcq.lcq_device_status(ws) == 0
    assert max_rel(host_bf16(Y), ref) <= TOL_DP


@pytest.mark.parametrize("N", [1, 16])
@pytest.mark.parametrize("m,n,d", [(200, 512, 8), (70, 200, 4), (300, 8192, 8)])
def test_gemm_packed2b_hadamard_matches_oracle(N, m, n, d):
    rng = np.random.default_rng(N * 7 + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    Xb = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    ref = oracle.gemm_packed2b_hadamard(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B_HADAMARD, N, m, n, d)
    lcq.lcq_gemm_packed2b_hadamard(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert max_rel(host_bf16(Y), ref) <= TOL_BF16


# 1-16 tokens with n % 64 == 0 and n <= 32768 (but one token at n = 8192): the rotation runs in the
# tcgen05 kernel's prep kernel, so the call is two launches (prep and product) and no rotation kernel.
# The rotated activations then take the digit path, so each output is held to digit_product_bound of
# the rotated X. Rotation blocks: 2^6 (n = 576, lanes only), 2^9 (n = 512, every bit in registers or
# shuffles), then one shared-memory pass of 2, 4, 8 or 16 points (n = 3072, 14336, 4096, and 2^13 in
# three blocks at n = 24576) or two passes (16 + 2 points at n = 16384, 16 + 4 at n = 32768).
@pytest.mark.parametrize("N", [1, 2, 7, 16])
@pytest.mark.parametrize("m,n,d", [(300, 576, 8), (129, 512, 4), (1000, 14336, 8), (77, 24576, 4), (260, 32768, 8),
                                   (513, 8192, 8), (90, 3072, 8), (140, 4096, 4), (64, 16384, 8)])
def test_gemm_packed2b_hadamard_tcgen05_prep(N, m, n, d):
    if N == 1 and n == 8192:
        pytest.skip("one token at n = 8192 rotates in the one-token kernel (test above)")
    rng = np.random.default_rng(13 * N + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n))
    X[:, rng.random(n) < 0.01] *= 50.0
    Xb = wl.bf16_bits(X.astype(np.float32))
    Xr = oracle.hadamard_rotate(wl.bf16_to_f32(Xb), n)      # rotated once: reference and bound
    ref = oracle.gemm_packed2b(Xr, oracle.pack2b(Z), A, b, d, n)   # = gemm_packed2b_hadamard(X)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B_HADAMARD, N, m, n, d)
    before = lcq.lcq_launch_count()
    lcq.lcq_gemm_packed2b_hadamard(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_launch_count() - before == 2
    assert lcq.lcq_device_status(ws) == 0
    bound = digit_product_bound(Xr, Z, A, b, d, ref)
    assert within(host_bf16(Y), ref, bound) <= 1.0


# 2-16 tokens with n % 64 == 0 take the tcgen05 kernel (kind::mxf4): the codes are fp4 operands in
# tensor memory and the activations exact integer digits, q = rint(X' 8191 / max|X'_t|) per token, so
# its only errors are that rounding (at most 2^-14 of max|X'_t| per element) and the bf16 output
# rounding: each output is held to the bound those two give (digit_product_bound), on heavy-tailed
# activations.
# The shapes cover ragged rows (not a multiple of 32 or 128), a partial last 512-column tile, ranges
# of one to eight 32-row slices, and more rows than one wave of CTAs holds (several ranges per CTA).
@pytest.mark.parametrize("N", [2, 5, 8, 9, 12, 16])
@pytest.mark.parametrize("m,n,d", [(1000, 4096, 8), (300, 8192, 4), (77, 576, 8), (129, 1088, 4), (2500, 512, 8),
                                   (40000, 64, 8)])
def test_gemm_packed2b_tcgen05_heavy_tailed(N, m, n, d):
    rng = np.random.default_rng(11 * N + m + n + d)
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n))
    X[:, rng.random(n) < 0.01] *= 50.0
    Xb = wl.bf16_bits(X.astype(np.float32))
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    Y = empty_bf16(N, m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
    lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(oracle.pack2b(Z)), n, d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_device_status(ws) == 0
    assert within(host_bf16(Y), ref, digit_product_bound(wl.bf16_to_f32(Xb), Z, A, b, d, ref)) <= 1.0


def test_gemm_packed2b_tcgen05_zero_token_and_repeat():
    """A token of zeros (scale 0) beside others; two calls in a row give identical bytes (the
    accumulators hold exact integer sums, so the result does not depend on the order of the sums)."""
    torch = T()
    rng = np.random.default_rng(5)
    N, m, n, d = 12, 700, 2048, 8
    Z = rng.integers(0, 4, (m, n)).astype(np.uint8)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n)).astype(np.float32)
    X[3] = 0.0
    Xb = wl.bf16_bits(X)
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), oracle.pack2b(Z), A, b, d, n)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, N, m, n, d)
    Y1, Y2 = empty_bf16(N, m), empty_bf16(N, m)
    Xd, Pd, Ad, bd = dev_bf16(Xb), dev(oracle.pack2b(Z)), dev(A), dev(b)
    lcq.lcq_gemm_packed2b(Xd, Pd, n, d, Ad, bd, Y1, ws)
    lcq.lcq_gemm_packed2b(Xd, Pd, n, d, Ad, bd, Y2, ws)
    assert torch.equal(Y1, Y2)
    assert float(Y1[3].float().abs().max()) == 0.0
    assert within(host_bf16(Y1), ref, digit_product_bound(wl.bf16_to_f32(Xb), Z, A, b, d, ref)) <= 1.0


# ----------------------------------------------------------------------------- activation transform

def _xform_bounds(Xf, ref_p, A, b, d):
    """Elementwise error bounds of the transform against fp64: X' is an fp32 sum of d products (error
    at most gamma_d sum |x a|) rounded to bf16 (8 significant bits: half an ulp is at most 2^-8 of the
    value); r is an fp32 sum of n products, bounded by gamma_n-sized multiples of sum |x b|
    (u = 2^-24)."""
    N, n = Xf.shape
    u = 2.0 ** -24
    Xg = np.abs(Xf.astype(np.float64)).reshape(N, n // d, d)
    absxa = (Xg @ np.abs(A.astype(np.float64))).reshape(N, n)
    absxb = (Xg @ np.abs(b.astype(np.float64))).sum(axis=1)
    sum_err = 2 * d * u * absxa
    return 2.0 ** -8 * (np.abs(ref_p) + sum_err) + sum_err, 2 * (n + 8) * u * absxb


@pytest.mark.parametrize("d", [4, 8])
@pytest.mark.parametrize("N,n", [(64, 512), (3, 200), (33, 4104), (1, 8)])
def test_activation_transform_matches_oracle(N, n, d):
    torch = T()
    if n % d:
        pytest.skip("n % d")
    rng = np.random.default_rng(N + n + d)
    A, b = config_A(d, rng), config_b(d, rng)
    X = rng.normal(0, 1, (N, n))
    X[:, rng.random(n) < 0.01] *= 50.0
    Xb = wl.bf16_bits(X.astype(np.float32))
    Xf = wl.bf16_to_f32(Xb)
    ref_p, ref_r = oracle.activation_transform(Xf, A, b, d)
    Xp = empty_bf16(N, n)
    r = torch.empty(N, dtype=torch.float32, device="cuda")
    lcq.lcq_activation_transform(dev_bf16(Xb), d, dev(A), dev(b), Xp=Xp, r=r)
    bp, br = _xform_bounds(Xf, ref_p, A, b, d)
    assert np.all(np.abs(host_bf16(Xp) - ref_p) <= bp)
    assert np.all(np.abs(r.cpu().numpy().astype(np.float64) - ref_r) <= br)


def test_activation_transform_single_output_and_empty():
    torch = T()
    rng = np.random.default_rng(3)
    d, N, n = 8, 5, 64
    A, b = config_A(d, rng), config_b(d, rng)
    Xb = wl.bf16_bits(rng.normal(0, 1, (N, n)).astype(np.float32))
    r = torch.full((N,), 7.0, dtype=torch.float32, device="cuda")
    lcq.lcq_activation_transform(dev_bf16(Xb), d, dev(A), dev(b), r=r)      # X' not written (NULL)
    ref_p, ref_r = oracle.activation_transform(wl.bf16_to_f32(Xb), A, b, d)
    np.testing.assert_allclose(r.cpu().numpy(), ref_r, rtol=1e-5, atol=1e-7)
    Xp = empty_bf16(N, n)
    lcq.lcq_activation_transform(dev_bf16(Xb), d, dev(A), dev(b), Xp=Xp)     # r not written (NULL)
    assert max_rel(host_bf16(Xp), ref_p) <= 4e-3
    E = torch.empty((0, n), dtype=torch.bfloat16, device="cuda")
    lcq.lcq_activation_transform(E, d, dev(A), dev(b), r=torch.empty(0, device="cuda"))
