"""Parity of the LDLQ initialisation (lcq_ldl_factor, lcq_ldlq) against the CPU oracle.

Factor: U and D against the fp64 oracle's factor of the same fp32 Hessian, relative to their largest
entry; exact zeros on and below the block diagonal.

Sweep: both sides get the same fp32 U. A decision of the sweep depends on every earlier decision
of its row, so a single near-boundary rounding that differs would change the rest of the row
legitimately. The checks are:
  * decisions in the kernel's precision: every code is clip(round(.)) of the fp32 latent the kernel
    reports, bit for bit;
  * latents: with the GPU's codes as the history, the oracle's fp64 latents of every target
    (ldlq_latent_given_codes) lie within the fp32 forward-error bound of the GPU's latents
    (tests.gpu_util.ldlq_latent_bound);
  * identity: rows whose oracle sweep has no latent value within 1e-5 of a boundary match the
    oracle's codes bit for bit (small sizes).
"""
import numpy as np
import pytest

import oracle
import paper_2606_10531_gb300 as lcq
from paper_2606_10531_gb300 import workloads as wl
from tests.gpu_util import config_A, config_b, dev, ldlq_latent_bound

pytestmark = pytest.mark.gpu

EPS_BOUNDARY = 1e-5
TOL_FACTOR = 3e-5      # fp32 blocked factorisation vs fp64, relative to max |entry| (see the test)


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


def ldlq_weights(m, n, rng):
    """Bulk-encode weight recipe: N(0, 0.015) with 0.1% entries 0.015 * t(4)."""
    W = rng.normal(0, 0.015, (m, n)).astype(np.float32)
    heavy = rng.random((m, n)) < 0.001
    W[heavy] = (0.015 * rng.standard_t(4, heavy.sum())).astype(np.float32)
    return W


def gpu_factor(H, d, want_D=True):
    torch = T()
    n = H.shape[0]
    U = torch.empty((n, n), dtype=torch.float32, device="cuda")
    D = torch.empty((n // d, d, d), dtype=torch.float32, device="cuda") if want_D else None
    ws = lcq.workspace(lcq.LCQ_OP_LDL_FACTOR, 0, 0, n, d)
    lcq.lcq_ldl_factor(dev(H), d, U, ws, D=D)
    assert lcq.lcq_device_status(ws) == 0
    return U, D


def gpu_sweep(W, A, b, U, d, with_codes=True, with_latent=True):
    torch = T()
    m, n = W.shape
    ws = lcq.workspace(lcq.LCQ_OP_LDLQ, 0, m, n, d)
    packed = torch.empty((m, n // 4), dtype=torch.uint8, device="cuda")
    codes = torch.empty((m, n), dtype=torch.uint8, device="cuda") if with_codes else None
    latent = torch.empty((m, n), dtype=torch.float32, device="cuda") if with_latent else None
    mse = torch.empty(1, dtype=torch.float64, device="cuda")
    Ud = U if isinstance(U, torch.Tensor) else dev(U)
    lcq.lcq_ldlq(dev(W), dev(A), dev(b), Ud, d, ws, packed=packed, codes=codes, latent=latent, mse=mse)
    status = lcq.lcq_device_status(ws)
    return packed, codes, latent, mse, status


def check_decisions(W, Z, lat_gpu, U, A, b, d):
    """The kernel's decisions against its own fp32 latents (exact) and those latents against the
    oracle's fp64 latents of the same history (fp32 error bound). Returns max |du| / bound."""
    assert np.array_equal(oracle.round_clamp(lat_gpu), Z)
    lat = oracle.ldlq_latent_given_codes(W, Z, U, A, b, d)
    bound = ldlq_latent_bound(W, Z, U, A, b, d)
    ratio = np.abs(lat_gpu.astype(np.float64) - lat) / bound
    assert ratio.max() <= 1.0, f"latent off by {ratio.max():.2f} x its fp32 bound at {np.unravel_index(ratio.argmax(), ratio.shape)}"
    return float(ratio.max())


@pytest.mark.parametrize("n,d", [(64, 4), (200, 8), (384, 4), (520, 8)])
def test_ldl_factor_matches_oracle(n, d):
    """The factor of the synthetic Hessian (cond ~1e4). fp32 elimination: the entries of U and D agree
    with the fp64 factor to a few n * 2^-24 relative to the largest entry (measured at most 3.3e-6 for
    these sizes on a GB300); the bound leaves a factor of 10."""
    H = wl.draw_hessian(n, 7, n)
    U_ref, D_ref = oracle.ldl_block(H.astype(np.float64), d)
    U, D = gpu_factor(H, d)
    U = U.cpu().numpy().astype(np.float64)
    D = D.cpu().numpy().astype(np.float64)
    blk = np.arange(n) // d
    assert np.all(U[blk[:, None] >= blk[None, :]] == 0.0)
    errU = np.abs(U - U_ref).max() / np.abs(U_ref).max()
    errD = np.abs(D - D_ref).max() / np.abs(D_ref).max()
    print(f"n={n} d={d}: max |dU|/max|U| = {errU:.2e}, max |dD|/max|D| = {errD:.2e}")
    assert errU < TOL_FACTOR and errD < TOL_FACTOR


SWEEP_CASES = [
    (64, 128, 4),       # one row tile, one chunk
    (100, 264, 8),      # ragged rows, partial last chunk (8 columns: one partial slice)
    (130, 520, 4),      # three row tiles, five chunks
    (256, 1024, 8),
    (70, 392, 8),       # last chunk of 8 columns after three full chunks
]


@pytest.mark.parametrize("m,n,d", SWEEP_CASES)
def test_ldlq_sweep_matches_oracle(m, n, d):
    rng = np.random.default_rng(500 + m + n + d)
    W = ldlq_weights(m, n, rng)
    A, b = config_A(d, rng), config_b(d, rng)
    H = wl.draw_hessian(n, 11, n).astype(np.float64)
    U32 = oracle.ldl_block(H, d)[0].astype(np.float32)
    ref = oracle.ldlq(W, U32, A, b, d)
    packed, codes, latent, mse, status = gpu_sweep(W, A, b, U32, d)
    assert status == 0
    Z = codes.cpu().numpy()
    assert np.array_equal(packed.cpu().numpy(), oracle.pack2b(Z))
    assert Z.max() <= 3
    ratio = check_decisions(W, Z, latent.cpu().numpy(), U32, A, b, d)
    clean = ~ref["near"].any(axis=1)
    assert np.array_equal(Z[clean], ref["codes"][clean])
    mse_ref = float(np.mean((W.astype(np.float64) - oracle.decode(Z, A, b, d)) ** 2))
    assert float(mse.item()) == pytest.approx(mse_ref, rel=1e-5)
    print(f"m={m} n={n} d={d}: latent error {ratio:.3f} of its bound, {int((~clean).sum())} rows with a "
          f"boundary case, equal rows {int(clean.sum())}")


@pytest.mark.parametrize("d", [4, 8])
def test_ldlq_factor_and_sweep_end_to_end(d):
    """GPU factor feeding the GPU sweep, checked against the oracle's fp64 factor: the decisions are
    valid for the oracle's U up to the factor's own error, so the exclusion band here is the latent
    shift that error can cause (checked against the measured max of |U_gpu - U_oracle| |E| sums)."""
    m, n = 96, 384
    rng = np.random.default_rng(77 + d)
    W = ldlq_weights(m, n, rng)
    A, b = config_A(d, rng), config_b(d, rng)
    H = wl.draw_hessian(n, 13, d)
    U_ref = oracle.ldl_block(H.astype(np.float64), d)[0]
    U, _ = gpu_factor(H, d, want_D=False)
    packed, codes, latent, mse, status = gpu_sweep(W, A, b, U, d)
    assert status == 0
    Z = codes.cpu().numpy()
    check_decisions(W, Z, latent.cpu().numpy(), U.cpu().numpy(), A, b, d)
    lat_gpuU = oracle.ldlq_latent_given_codes(W, Z, U.cpu().numpy(), A, b, d)
    lat_refU = oracle.ldlq_latent_given_codes(W, Z, U_ref, A, b, d)
    band = max(EPS_BOUNDARY, 4.0 * float(np.abs(lat_gpuU - lat_refU).max()))
    near = oracle.near_boundary(lat_refU, band)
    bad = (oracle.round_clamp(lat_refU) != Z) & ~near
    assert not bad.any()
    assert band < 1e-2
    print(f"d={d}: exclusion band {band:.2e}, {int(near.sum())} decisions inside it")


@pytest.mark.parametrize("d", [4, 8])
def test_ldlq_without_feedback_is_the_encoder(d):
    """U = 0 (block-diagonal Hessian): LDLQ rounds every group on its own, as lcq_encode does."""
    torch = T()
    m, n = 130, 264
    rng = np.random.default_rng(91 + d)
    W = ldlq_weights(m, n, rng)
    A, b = config_A(d, rng), config_b(d, rng)
    _, codes, _, mse, status = gpu_sweep(W, A, b, np.zeros((n, n), np.float32), d)
    assert status == 0
    ws = lcq.workspace(lcq.LCQ_OP_ENCODE, 0, m, n, d)
    enc = torch.empty((m, n), dtype=torch.uint8, device="cuda")
    lcq.lcq_encode(dev(W), dev(A), dev(b), d, ws, codes=enc)
    ref = oracle.encode(W, A, b, d)
    Z, E = codes.cpu().numpy(), enc.cpu().numpy()
    far = ~ref["near"]
    assert np.array_equal(Z[far], E[far]) and np.array_equal(Z[far], ref["codes"][far])


def test_ldlq_singular_A_sets_status_and_zero_codes():
    d, m, n = 8, 64, 128
    rng = np.random.default_rng(5)
    W = ldlq_weights(m, n, rng)
    A = np.zeros((d, d), np.float32)
    H = wl.draw_hessian(n, 3, 0).astype(np.float64)
    U32 = oracle.ldl_block(H, d)[0].astype(np.float32)
    packed, codes, _, _, status = gpu_sweep(W, A, config_b(d, rng), U32, d)
    assert status == 7                                   # LCQ_ERR_SINGULAR
    assert int(codes.max().item()) == 0 and int(packed.max().item()) == 0


def test_ldl_factor_of_a_singular_matrix_sets_status():
    torch = T()
    n, d = 64, 8
    U = torch.empty((n, n), dtype=torch.float32, device="cuda")
    ws = lcq.workspace(lcq.LCQ_OP_LDL_FACTOR, 0, 0, n, d)
    lcq.lcq_ldl_factor(dev(np.zeros((n, n), np.float32)), d, U, ws)
    assert lcq.lcq_device_status(ws) == 7


def test_ldlq_empty():
    torch = T()
    d, n = 8, 64
    mse = torch.full((1,), 5.0, dtype=torch.float64, device="cuda")
    ws = lcq.workspace(lcq.LCQ_OP_LDLQ, 0, 0, n, d)
    W = torch.empty((0, n), dtype=torch.float32, device="cuda")
    U = torch.zeros((n, n), dtype=torch.float32, device="cuda")
    lcq.lcq_ldlq(W, dev(config_A(d, np.random.default_rng(1))), dev(np.zeros(d, np.float32)), U, d, ws, mse=mse)
    assert float(mse.item()) == 0.0


def test_ldl_factor_captured_in_a_cuda_graph():
    """The factorisation forks each panel onto a library side stream and joins it back with events:
    captured into a CUDA graph and replayed it gives the eager result, and work after the replay on
    the capturing stream sees every output."""
    torch = T()
    n, d = 520, 8
    H = dev(wl.draw_hessian(n, 17, n))
    U_eager, D_eager = gpu_factor(H.cpu().numpy(), d)
    U = torch.empty((n, n), dtype=torch.float32, device="cuda")
    D = torch.empty((n // d, d, d), dtype=torch.float32, device="cuda")
    ws = lcq.workspace(lcq.LCQ_OP_LDL_FACTOR, 0, 0, n, d)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        lcq.lcq_ldl_factor(H, d, U, ws, D=D)          # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    U.zero_(), D.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        lcq.lcq_ldl_factor(H, d, U, ws, D=D)
        checksum = U.abs().sum() + D.abs().sum()      # on the capturing stream, after the join
    g.replay()
    torch.cuda.synchronize()
    assert lcq.lcq_device_status(ws) == 0
    assert torch.equal(U, U_eager) and torch.equal(D, D_eager)
    assert float(checksum) == pytest.approx(float(U_eager.abs().sum() + D_eager.abs().sum()), rel=1e-6)
