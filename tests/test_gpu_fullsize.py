"""Parity at the full sizes of the benchmarked workloads, through the same C-ABI calls bench.py makes.

The oracle cannot recompute every output of these layers in seconds, so each test checks what it
can exactly: the quantized codes over the whole matrix, sampled rows of every product computed one
by one in fp64, and the weight-gradient sums through identities that hold at any size:
    db[j]    = sum_t rowsum(dY)[t] * sum_g X[t, g*d + j]
    dA[j][k] = sum_{t,g} X[t, g*d + j] * (dY Z)[t, g*d + k]
Tolerances are those of the small parity tests (2e-2 of max|ref| for bf16 products and gradients)."""
import numpy as np
import pytest

import oracle
import paper_2606_10531_gb300 as lcq
from paper_2606_10531_gb300 import workloads as wl
from tests.gpu_util import (TOL_BF16, dev, dev_bf16, digit_product_bound, empty_bf16, host_bf16, ldlq_latent_bound,
                            max_rel, within)

pytestmark = pytest.mark.gpu

SEED = 0
SAMPLES = 32      # tokens and weight rows recomputed one by one in fp64


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_10531_gb300 import build
    build.build()
    lcq.lib()


def _latent_chunked(W, A, b, d, rows=2048):
    out = np.empty(W.shape, dtype=np.float32)
    for r0 in range(0, W.shape[0], rows):
        out[r0:r0 + rows] = oracle.latent(W[r0:r0 + rows], A, b, d).astype(np.float32)
    return out


def _check_linear(mx, index):
    import torch
    m, n, d, N = mx.m, mx.n, mx.d, mx.N
    W = wl.draw_W(mx, SEED, index)
    A, b = wl.draw_A(mx, SEED, index), wl.draw_b(mx, SEED, index)
    Xb, dYb = wl.draw_X(mx, SEED, index), wl.draw_dY(mx, SEED, index)
    P = _latent_chunked(W, A, b, d)
    del W
    Z = oracle.quantize(P)

    Xd, dYd, Ad, bd = dev_bf16(Xb), dev_bf16(dYb), dev(A), dev(b)
    Y = empty_bf16(N, m)
    saved = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    wsf = lcq.workspace(lcq.LCQ_OP_LINEAR_FWD, N, m, n, d)
    lcq.lcq_linear_fwd(Xd, dev(P), d, Ad, bd, Y, wsf, packed_saved=saved)
    assert np.array_equal(saved.cpu().numpy(), oracle.pack2b(Z)), "integer weights differ"
    dX = empty_bf16(N, n)
    dP = torch.empty((m, n), dtype=torch.float32, device="cuda")
    dA = torch.empty((d, d), dtype=torch.float32, device="cuda")
    db = torch.empty(d, dtype=torch.float32, device="cuda")
    wsb = lcq.workspace(lcq.LCQ_OP_LINEAR_BWD, N, m, n, d)
    lcq.lcq_linear_bwd(Xd, dYd, saved, m, n, d, Ad, bd, dP, dA, db, wsb, dX=dX)
    assert lcq.lcq_device_status(wsf) == 0 and lcq.lcq_device_status(wsb) == 0

    X, dY = wl.bf16_to_f32(Xb).astype(np.float64), wl.bf16_to_f32(dYb).astype(np.float64)
    W_hat = oracle.decode(Z, A, b, d)
    rng = np.random.default_rng(1234 + index)
    k = SAMPLES
    toks = rng.choice(N, k, replace=False)
    rows = rng.choice(m, k, replace=False)
    # sampled rows of Y = X W_hat^T and dX = dY W_hat
    Yg, dXg = host_bf16(Y), host_bf16(dX)
    assert max_rel(Yg[toks], X[toks] @ W_hat.T) <= TOL_BF16
    assert max_rel(dXg[toks], dY[toks] @ W_hat) <= TOL_BF16
    # sampled rows of dP = (dY^T X)_g A
    dW_rows = dY[:, rows].T @ X                                    # k x n
    dP_ref = (dW_rows.reshape(k, n // d, d) @ A.astype(np.float64)).reshape(k, n)
    assert max_rel(dP.cpu().numpy()[rows], dP_ref) <= TOL_BF16
    # db, dA through their row-sum identities (any size), in fp64
    rho = dY.sum(axis=1)
    sig = X.reshape(N, n // d, d).sum(axis=1)
    assert max_rel(db.cpu().numpy(), rho @ sig) <= TOL_BF16
    T = dY @ Z.astype(np.float64)                                  # dY Z, N x n
    dA_ref = X.reshape(N * (n // d), d).T @ T.reshape(N * (n // d), d)
    assert max_rel(dA.cpu().numpy(), dA_ref) <= TOL_BF16


def test_llama3_8b_gate_fwd_bwd_full_size():
    mats = wl.llama3_8b_layer()
    _check_linear(mats[4], 4)         # gate 14336 x 4096, d = 8, 16384 tokens


def test_llama3_8b_down_fwd_bwd_full_size():
    mats = wl.llama3_8b_layer()
    _check_linear(mats[6], 6)         # down 4096 x 14336: K = 14336 in the forward, the widest dW epilogue


def test_llama3_8b_k_fwd_bwd_full_size():
    mats = wl.llama3_8b_layer()
    _check_linear(mats[1], 1)         # k 1024 x 4096: eight 128-row blocks of weight rows


def test_llama2_7b_gate_fwd_bwd_full_size_d4_outliers():
    mats = wl.llama2_7b_projections(d=4)
    _check_linear(mats[4], 4)         # gate 11008 x 4096, d = 4, 4096 tokens, 1% outlier channels x20


def test_llama2_7b_gate_fwd_bwd_full_size_d8_outliers():
    mats = wl.llama2_7b_projections(d=8)
    _check_linear(mats[4], 4)         # gate 11008 x 4096, d = 8, 4096 tokens, 1% outlier channels x20


@pytest.mark.parametrize("B", [1, 2, 4, 16])
def test_llama3_70b_gate_packed_product_full_size(B):
    mx = wl.llama3_70b_gate_decode(B)[0]
    packed = wl.draw_packed_codes(mx, SEED, 0)
    A, b = wl.draw_A(mx, SEED, 0), wl.draw_b(mx, SEED, 0)
    Xb = wl.draw_X(mx, SEED, B)
    Y = empty_bf16(B, mx.m)
    ws = lcq.workspace(lcq.LCQ_OP_GEMM_PACKED2B, B, mx.m, mx.n, mx.d)
    lcq.lcq_gemm_packed2b(dev_bf16(Xb), dev(packed), mx.n, mx.d, dev(A), dev(b), Y, ws)
    assert lcq.lcq_device_status(ws) == 0
    rows = np.random.default_rng(99 + B).choice(mx.m, 64, replace=False)
    ref = oracle.gemm_packed2b(wl.bf16_to_f32(Xb), packed[rows], A, b, mx.d, mx.n)   # B x 64
    # every B here takes an integer kernel: int16 activations at one token (the one-token bar), exact
    # integer digits above (the elementwise bound of their rounding)
    if B == 1:
        assert max_rel(host_bf16(Y)[:, rows], ref) <= 4e-3
    else:
        Z = oracle.unpack2b(packed[rows], mx.n)
        bound = digit_product_bound(wl.bf16_to_f32(Xb), Z, A, b, mx.d, ref)
        assert within(host_bf16(Y)[:, rows], ref, bound) <= 1.0


def test_llama3_70b_gate_bulk_encode_full_size():
    import torch
    mx = wl.llama3_70b_layer_encode()[4]       # gate 28672 x 8192, heavy-tailed, d = 8
    W = wl.draw_W(mx, SEED, 4)
    A, b = wl.draw_A(mx, SEED, 4), wl.draw_b(mx, SEED, 4)
    packed = torch.empty((mx.m, mx.n // 4), dtype=torch.uint8, device="cuda")
    mse = torch.empty(1, dtype=torch.float64, device="cuda")
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, mx.m, mx.n, mx.d)
    lcq.lcq_encode(dev(W), dev(A), dev(b), mx.d, ws, packed=packed, mse=mse)
    assert lcq.lcq_device_status(ws) == 0
    got = packed.cpu().numpy()
    sq, mismatch, near = 0.0, 0, 0
    for r0 in range(0, mx.m, 2048):
        ref = oracle.encode(W[r0:r0 + 2048], A, b, mx.d)
        z = oracle.unpack2b(got[r0:r0 + 2048], mx.n)
        keep = ~ref["near"]
        mismatch += int(np.sum((z != ref["codes"]) & keep))
        near += int(np.sum(ref["near"]))
        sq += ref["mse"] * z.size
    assert mismatch == 0
    ref_mse = sq / (mx.m * mx.n)
    assert abs(mse.item() - ref_mse) <= 1e-4 * ref_mse
    print(f"near-boundary codes excluded: {near} of {mx.m * mx.n}")


def test_llama3_70b_gate_ldlq_full_size():
    """LDLQ of the Llama-3-70B gate (28672 x 8192, d = 8) with the synthetic proxy Hessian, through the
    calls bench.py times. The factor is checked by reconstructing sampled entries of H from U and D
    (any size); the sweep, on sampled rows, by its decisions against its own fp32 latents (exact) and
    those latents against the oracle's fp64 latents of the same history and U (fp32 error bound), and
    by its MSE over all rows."""
    import torch
    mx = wl.llama3_70b_gate_ldlq()[0]
    m, n, d = mx.m, mx.n, mx.d
    H = wl.draw_hessian(n, SEED, 0)
    W = wl.draw_W(mx, SEED, 0)
    A, b = wl.draw_A(mx, SEED, 0), wl.draw_b(mx, SEED, 0)
    U = torch.empty((n, n), dtype=torch.float32, device="cuda")
    D = torch.empty((n // d, d, d), dtype=torch.float32, device="cuda")
    wsf = lcq.workspace(lcq.LCQ_OP_LDL_FACTOR, 0, 0, n, d)
    lcq.lcq_ldl_factor(dev(H), d, U, wsf, D=D)
    codes = torch.empty((m, n), dtype=torch.uint8, device="cuda")
    latent = torch.empty((m, n), dtype=torch.float32, device="cuda")
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    mse = torch.empty(1, dtype=torch.float64, device="cuda")
    wss = lcq.workspace(lcq.LCQ_OP_LDLQ, 0, m, n, d)
    lcq.lcq_ldlq(dev(W), dev(A), dev(b), U, d, wss, packed=packed, codes=codes, latent=latent, mse=mse)
    assert lcq.lcq_device_status(wsf) == 0 and lcq.lcq_device_status(wss) == 0

    Uh = U.cpu().numpy().astype(np.float64)
    Dh = D.cpu().numpy().astype(np.float64)
    M = Uh + np.eye(n)
    rng = np.random.default_rng(4242)
    pairs = [(int(i), int(j)) for i, j in zip(rng.integers(0, n, 64), rng.integers(0, n, 64))] + [(0, 0), (n - 1, n - 1)]
    Hmax = float(np.abs(H).max())
    worst = 0.0
    for i, j in pairs:
        kmin = max(i, j) // d
        acc = 0.0
        for k in range(kmin, n // d):
            s = slice(k * d, (k + 1) * d)
            acc += M[i, s] @ Dh[k] @ M[j, s]
        worst = max(worst, abs(acc - float(H[i, j])) / Hmax)
    print(f"factor: max sampled |(M D M^T - H)_ij| / max|H| = {worst:.2e}")
    assert worst < 1e-4

    rows = np.concatenate([[0, m - 1], rng.choice(m, 30, replace=False)])
    Z = codes.cpu().numpy()
    assert np.array_equal(packed.cpu().numpy()[rows], oracle.pack2b(Z[rows]))
    lat_gpu = latent[torch.as_tensor(rows, device="cuda")].cpu().numpy()
    assert np.array_equal(oracle.round_clamp(lat_gpu), Z[rows])
    lat = oracle.ldlq_latent_given_codes(W[rows], Z[rows], Uh, A, b, d)
    bound = ldlq_latent_bound(W[rows], Z[rows], Uh, A, b, d)
    err = np.abs(lat_gpu.astype(np.float64) - lat)
    flips = int(np.sum(oracle.round_clamp(lat) != Z[rows]))
    print(f"sweep: latent error max {err.max():.2e} (median bound {np.median(bound):.2e}), "
          f"max error / bound {np.max(err / bound):.3f}; {flips} of {lat.size} decisions round otherwise "
          f"in fp64, all within the bound of a boundary")
    assert np.all(err <= bound)
    sq = 0.0
    for r0 in range(0, m, 2048):
        sq += float(np.sum((W[r0:r0 + 2048].astype(np.float64) - oracle.decode(Z[r0:r0 + 2048], A, b, d)) ** 2))
    ref_mse = sq / (m * n)
    assert abs(mse.item() - ref_mse) <= 1e-5 * ref_mse


def test_llama3_70b_layer_bulk_encode_batch_full_size():
    """The bulk encode that bench.py times: all seven linears of a Llama-3-70B layer (855,638,016
    weights, d = 8, heavy-tailed) in one lcq_encode_batch call with packed codes and MSE per matrix,
    checked against the oracle matrix by matrix in row chunks (codes bit-exact away from rounding
    boundaries, MSE to 1e-4 relative)."""
    import torch
    mats = wl.llama3_70b_layer_encode()
    items, host = [], []
    for i, mx in enumerate(mats):
        W = wl.draw_W(mx, SEED + 1000, i)
        A, b = wl.draw_A(mx, SEED + 1000, i), wl.draw_b(mx, SEED + 1000, i)
        packed = torch.empty((mx.m, mx.n // 4), dtype=torch.uint8, device="cuda")
        mse = torch.empty(1, dtype=torch.float64, device="cuda")
        items.append({"W": dev(W), "A": dev(A), "b": dev(b), "packed": packed, "mse": mse})
        host.append((mx, W, A, b))
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE_BATCH, len(items), 0, 0, mats[0].d)
    lcq.lcq_encode_batch(items, mats[0].d, ws)
    assert lcq.lcq_device_status(ws) == 0
    near_total = 0
    for (mx, W, A, b), it in zip(host, items):
        got = it["packed"].cpu().numpy()
        it["W"] = None
        sq, mismatch = 0.0, 0
        for r0 in range(0, mx.m, 2048):
            ref = oracle.encode(W[r0:r0 + 2048], A, b, mx.d)
            z = oracle.unpack2b(got[r0:r0 + 2048], mx.n)
            keep = ~ref["near"]
            mismatch += int(np.sum((z != ref["codes"]) & keep))
            near_total += int(np.sum(ref["near"]))
            sq += ref["mse"] * z.size
        assert mismatch == 0, mx.name
        ref_mse = sq / (mx.m * mx.n)
        assert abs(it["mse"].item() - ref_mse) <= 1e-4 * ref_mse, mx.name
    print(f"near-boundary codes excluded: {near_total} of {sum(mx.m * mx.n for mx in mats)}")


@pytest.mark.parametrize("index", [0, 6])
def test_llama3_8b_activation_transform_full_size(index):
    """The activation transform of the reformulated forward (Eq. def:forward_x) at the training shapes
    of the Llama-3-8B layer (16384 tokens; n = 4096 for q, n = 14336 for down): sampled tokens against
    the oracle in fp64, within the bf16 rounding of X' and the fp32 sum bound of r."""
    import torch
    from tests.test_gpu_parity import _xform_bounds
    mx = wl.llama3_8b_layer()[index]
    Xb = wl.draw_X(mx, SEED, index)
    A, b = wl.draw_A(mx, SEED, index), wl.draw_b(mx, SEED, index)
    Xp = empty_bf16(mx.N, mx.n)
    r = torch.empty(mx.N, dtype=torch.float32, device="cuda")
    lcq.lcq_activation_transform(dev_bf16(Xb), mx.d, dev(A), dev(b), Xp=Xp, r=r)
    toks = np.random.default_rng(7 + index).choice(mx.N, SAMPLES, replace=False)
    Xf = wl.bf16_to_f32(Xb[toks])
    ref_p, ref_r = oracle.activation_transform(Xf, A, b, mx.d)
    bp, br = _xform_bounds(Xf, ref_p, A, b, mx.d)
    got_p = host_bf16(Xp[torch.as_tensor(toks, device="cuda")])
    assert np.all(np.abs(got_p - ref_p) <= bp)
    assert np.all(np.abs(r.cpu().numpy()[toks].astype(np.float64) - ref_r) <= br)
