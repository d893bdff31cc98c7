"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test ties one oracle function to a closed form, a textbook special
case, brute force on tiny inputs, finite differences, or a hand-worked
fixture in tests/golden/. Together they fail on a dropped term, a wrong
sign, a transposed operand or a wrong index in any oracle function.
"""
import itertools
import math

import numpy as np
import pytest

import oracle
from tests.golden_io import read_keyed, read_rows

RNG = np.random.default_rng(12345)


def config_like_A(d, rng):
    return 0.01 * np.eye(d) + rng.normal(0, 1e-3, (d, d))


# ----------------------------------------------------------------------------- encode / quantize

def test_round_clamp_table_matches_textbook(golden_dir):
    rows = read_rows("round_clamp_table.txt")
    v = np.array([float(r[0]) for r in rows])
    want = np.array([int(r[1]) for r in rows], dtype=np.uint8)
    assert np.array_equal(oracle.round_clamp(v), want)
    # Python's round() is round-half-to-even: the scalar textbook rule.
    assert [min(max(round(x), 0), 3) for x in v] == list(want)


def test_identity_codebook_reduces_to_scalar_round_clamp():
    """A = I, B = 0: LC-VQ encode is scalar clamp(round(w)) (SQ special case, Sec. 3.2)."""
    for d in (4, 8):
        W = RNG.uniform(-1.5, 4.5, (6, 8 * d))
        codes = oracle.encode(W, np.eye(d), np.zeros(d), d)["codes"]
        scalar = np.array([[min(max(round(w), 0), 3) for w in row] for row in W], dtype=np.uint8)
        assert np.array_equal(codes, scalar)


def test_encode_worked_example(golden_dir):
    g = read_keyed("encode_worked_d4.txt")
    d = int(g["d"][0])
    A = g["A"].reshape(d, d)
    out = oracle.encode(g["w"].reshape(1, -1), A, g["B"], d)
    np.testing.assert_allclose(out["latent"].ravel(), g["u"], rtol=0, atol=1e-12)
    assert np.array_equal(out["codes"].ravel(), g["z"].astype(np.uint8))
    np.testing.assert_allclose(oracle.decode(out["codes"], A, g["B"], d).ravel(), g["w_hat"], atol=1e-12)


def test_codes_lie_in_level_set_including_nan_and_inf():
    for d in (4, 8):
        A = config_like_A(d, RNG)
        W = RNG.normal(0, 0.05, (16, 4 * d))
        W[0, :3] = [np.nan, np.inf, -np.inf]
        out = oracle.encode(W, A, RNG.normal(0, 1e-3, d), d)
        assert out["codes"].dtype == np.uint8
        assert set(np.unique(out["codes"])) <= {0, 1, 2, 3}
    z = oracle.round_clamp(np.array([np.nan, np.inf, -np.inf]))
    assert list(z) == [0, 3, 0]


@pytest.mark.parametrize("d", [4, 8])
def test_reencoding_a_decoded_codeword_returns_its_codes(d):
    """Codewords are fixed points of the encoder: encode(decode(z)) = z."""
    for A in (config_like_A(d, RNG), oracle.init_codebook(np.linalg.qr(RNG.normal(size=(d, d)))[0])[0]):
        b = RNG.normal(0, 1e-3, d)
        Z = RNG.integers(0, 4, (32, 16 * d)).astype(np.uint8)
        W = oracle.decode(Z, A, b, d)
        assert np.array_equal(oracle.encode(W, A, b, d)["codes"], Z)


@pytest.mark.parametrize("d,m,n", [(4, 16, 64), (8, 4, 32)])
def test_bruteforce_nearest_equals_rounding_for_diagonal_positive_A(d, m, n):
    """For diagonal positive A the distance separates per coordinate, so the exhaustive
    4^d search of Eq. vq_assign must pick exactly the rounded-and-clamped latent."""
    A = np.diag(RNG.uniform(0.005, 0.02, d))
    b = RNG.normal(0, 1e-3, d)
    W = RNG.normal(0.015, 0.02, (m, n))
    codes_bf, _ = oracle.brute_nearest(W, A, b, d)
    out = oracle.encode(W, A, b, d)
    assert not out["near"].any()
    assert np.array_equal(codes_bf, out["codes"])


@pytest.mark.parametrize("d", [4, 8])
def test_rounding_never_beats_exhaustive_search_for_general_A(d):
    A = config_like_A(d, RNG) + RNG.normal(0, 4e-3, (d, d))
    b = RNG.normal(0, 1e-3, d)
    W = RNG.normal(0, 0.02, (3, 4 * d))
    codes_bf, dist_bf = oracle.brute_nearest(W, A, b, d)
    Zr = oracle.encode(W, A, b, d)["codes"]
    dist_r = ((W - oracle.decode(Zr, A, b, d)) ** 2).reshape(3, 4, d).sum(-1)
    assert np.all(dist_r >= dist_bf - 1e-15)
    # the brute force really is the minimum: its codes decode to its distance
    np.testing.assert_allclose(((W - oracle.decode(codes_bf, A, b, d)) ** 2).reshape(3, 4, d).sum(-1), dist_bf,
                               rtol=1e-12)


def test_near_boundary_mask_marks_only_half_integers_inside_range():
    u = np.array([0.5, 1.5 + 5e-6, 2.5 - 9e-6, 3.5, -0.5, 1.49, 0.0])
    assert list(oracle.near_boundary(u)) == [True, True, True, False, False, False, False]


def test_quantize_latent_affine_reading():
    """s = 1, t = 0 is the literal Eq. quant_param; with s, t it rounds P/s + t formed in fp32."""
    P = np.array([[-0.6, 0.2, 0.7, 1.5, 2.4999, 3.9, 2.5, 100.0]], dtype=np.float32)
    assert list(oracle.quantize(P)[0]) == [0, 0, 1, 2, 2, 3, 2, 3]
    s, t = 0.25, 1.5
    want = [min(max(round(float(np.float32(np.float32(p) * np.float32(4.0)) + np.float32(1.5))), 0), 3)
            for p in P[0]]
    assert list(oracle.quantize(P, s, t)[0]) == want


def test_mse_definition_and_zero_on_codewords():
    d = 4
    A, b = config_like_A(d, RNG), RNG.normal(0, 1e-3, d)
    Z = RNG.integers(0, 4, (8, 32))
    assert oracle.mse(oracle.decode(Z, A, b, d), Z, A, b, d) < 1e-30
    W = RNG.normal(0, 0.02, (8, 32))
    out = oracle.encode(W, A, b, d)
    direct = sum((W[r, c] - oracle.decode(out["codes"], A, b, d)[r, c]) ** 2 for r in range(8) for c in range(32)) / 256
    assert math.isclose(out["mse"], direct, rel_tol=1e-12)


# ----------------------------------------------------------------------------- decode

def test_decode_worked_example(golden_dir):
    g = read_keyed("decode_worked_d4.txt")
    d = int(g["d"][0])
    W_hat = oracle.decode(g["z"].reshape(1, d), g["A"].reshape(d, d), g["B"], d)
    np.testing.assert_allclose(W_hat.ravel(), g["w_hat"], rtol=0, atol=1e-12)


@pytest.mark.parametrize("d", [4, 8])
def test_decode_permutation_A_moves_codes_in_stated_direction(d):
    """A[j][(j+1) % d] = 1: w_hat_j = z_{(j+1) mod d} within every group (catches a transposed A)."""
    A = np.zeros((d, d))
    for j in range(d):
        A[j, (j + 1) % d] = 1.0
    Z = RNG.integers(0, 4, (5, 3 * d))
    W_hat = oracle.decode(Z, A, np.zeros(d), d)
    for r in range(5):
        for g in range(3):
            for j in range(d):
                assert W_hat[r, g * d + j] == Z[r, g * d + (j + 1) % d]


@pytest.mark.parametrize("d", [4, 8])
def test_initialised_codebook_has_zero_mean_and_identity_covariance(d, golden_dir):
    """Eq. init_ab: over all 4^d codewords the codebook mean is 0 and its covariance is I."""
    c = read_keyed("init_constants.txt")
    G = np.linalg.qr(np.random.default_rng(7).normal(size=(d, d)))[0]
    A, B = oracle.init_codebook(G)
    np.testing.assert_allclose(A, c["s"][0] * G, rtol=1e-15)
    allz = np.array(list(itertools.product(range(4), repeat=d)), dtype=np.uint8)   # 4^d x d
    C = oracle.decode(allz, A, B, d)      # one group per row
    np.testing.assert_allclose(C.mean(0), 0.0, atol=1e-12)
    np.testing.assert_allclose(np.cov(C.T, bias=True), np.eye(d), atol=1e-12)


# ----------------------------------------------------------------------------- forward

def test_forward_matches_explicit_loops_on_tiny_input():
    N, m, n, d = 2, 3, 8, 4
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    Z = RNG.integers(0, 4, (m, n))
    X = RNG.normal(size=(N, n))
    Y = oracle.linear_fwd(X, Z, A, b, d)
    for t in range(N):
        for r in range(m):
            acc = 0.0
            for g in range(n // d):
                for j in range(d):
                    w = b[j] + sum(A[j][k] * Z[r][g * d + k] for k in range(d))
                    acc += X[t][g * d + j] * w
            assert math.isclose(Y[t, r], acc, rel_tol=1e-12, abs_tol=1e-12)


def test_forward_one_hot_rows_select_decoded_weights():
    """X = e_c: Y[:, r] = W_hat[r, c] (fixes the Y = X W_hat^T orientation)."""
    d, m, n = 4, 5, 12
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    Z = RNG.integers(0, 4, (m, n))
    Y = oracle.linear_fwd(np.eye(n), Z, A, b, d)
    np.testing.assert_allclose(Y, oracle.decode(Z, A, b, d).T, atol=1e-13)


@pytest.mark.parametrize("d", [4, 8])
def test_forward_equals_reformulated_sum(d):
    """Eq. def:forward_x: Y = sum_i (X_i A) W_{z,i}^T + sum_i (X_i B) 1^T."""
    N, m, n = 7, 9, 6 * d
    A, b = config_like_A(d, RNG), RNG.normal(0, 1e-3, d)
    Z = RNG.integers(0, 4, (m, n))
    X = RNG.normal(size=(N, n))
    Y = np.zeros((N, m))
    for i in range(n // d):
        Xi = X[:, i * d:(i + 1) * d]
        Y += (Xi @ A) @ Z[:, i * d:(i + 1) * d].T + np.outer(Xi @ b, np.ones(m))
    np.testing.assert_allclose(oracle.linear_fwd(X, Z, A, b, d), Y, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("d", [4, 8])
def test_activation_transform_reproduces_the_decoded_product(d):
    """X' Z^T + r 1^T equals X W_hat^T computed through decode (Eq. def:forward vs def:forward_x): a
    transposed A, a dropped bias term or a wrong group stride breaks the identity."""
    N, m, n = 5, 7, 4 * d
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    Z = RNG.integers(0, 4, (m, n))
    X = RNG.normal(size=(N, n))
    Xp, r = oracle.activation_transform(X, A, b, d)
    np.testing.assert_allclose(Xp @ Z.T + r[:, None], oracle.linear_fwd(X, Z, A, b, d), rtol=1e-12, atol=1e-12)


def test_activation_transform_special_cases():
    """A = I, b = 0 leaves X unchanged with r = 0; a one-hot token e_c (c = g d + j) gives row j of A in
    group g and r = b_j; r is X times b repeated over the groups."""
    d, N, n = 4, 3, 12
    X = RNG.normal(size=(N, n))
    Xp, r = oracle.activation_transform(X, np.eye(d), np.zeros(d), d)
    np.testing.assert_array_equal(Xp, X)
    np.testing.assert_array_equal(r, np.zeros(N))
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    for c in (0, 5, 11):
        e = np.zeros((1, n))
        e[0, c] = 1.0
        Xp, r = oracle.activation_transform(e, A, b, d)
        g, j = divmod(c, d)
        expect = np.zeros(n)
        expect[g * d:(g + 1) * d] = A[j]
        np.testing.assert_allclose(Xp[0], expect, atol=0)
        assert r[0] == b[j]
    Xp, r = oracle.activation_transform(X, A, b, d)
    np.testing.assert_allclose(r, X @ np.tile(b, n // d), rtol=1e-13)


def test_packed_product_equals_unpacked_product():
    d, m, n = 8, 6, 32
    A, b = config_like_A(d, RNG), RNG.normal(0, 1e-3, d)
    Z = RNG.integers(0, 4, (m, n)).astype(np.uint8)
    X = RNG.normal(size=(3, n))
    np.testing.assert_allclose(oracle.gemm_packed2b(X, oracle.pack2b(Z), A, b, d, n),
                               oracle.linear_fwd(X, Z, A, b, d), rtol=1e-14)


# ----------------------------------------------------------------------------- backward

def _loss(X, A, b, Zc, dY, d):
    """<dY, Y> with z continuous (the STE treats the integer weights as real)."""
    m, n = Zc.shape
    W_hat = (Zc.reshape(m, n // d, d) @ A.T + b).reshape(m, n)
    return float(np.sum(dY * (X @ W_hat.T)))


@pytest.mark.parametrize("d", [4, 8])
def test_backward_equals_central_finite_differences(d):
    """L = <dY, Y> is linear in each of X, A, B and z, so central differences are exact."""
    N, m, n = 3, 4, 2 * d
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    Z = RNG.integers(0, 4, (m, n)).astype(np.float64)
    X, dY = RNG.normal(size=(N, n)), RNG.normal(size=(N, m))
    g = oracle.linear_bwd(X, dY, Z, A, b, d)
    h = 0.5

    def fd(arr, idx, f):
        old = arr[idx]
        arr[idx] = old + h
        up = f()
        arr[idx] = old - h
        dn = f()
        arr[idx] = old
        return (up - dn) / (2 * h)

    L = lambda: _loss(X, A, b, Z, dY, d)  # noqa: E731
    for idx in np.ndindex(X.shape):
        assert math.isclose(g["dX"][idx], fd(X, idx, L), rel_tol=1e-9, abs_tol=1e-9)
    for idx in np.ndindex(A.shape):
        assert math.isclose(g["dA"][idx], fd(A, idx, L), rel_tol=1e-9, abs_tol=1e-9)
    for idx in np.ndindex(b.shape):
        assert math.isclose(g["db"][idx], fd(b, idx, L), rel_tol=1e-9, abs_tol=1e-9)
    for idx in np.ndindex(Z.shape):
        assert math.isclose(g["dP"][idx], fd(Z, idx, L), rel_tol=1e-9, abs_tol=1e-9)


def test_ste_latent_scale_divides_gradient():
    """With z = P/s + t treated as identity-rounded, dL/dP = dL/dz / s (chain rule)."""
    d, s, t = 4, 0.25, 1.5
    N, m, n = 2, 3, 8
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    P = RNG.normal(size=(m, n))
    X, dY = RNG.normal(size=(N, n)), RNG.normal(size=(N, m))
    Z = oracle.quantize(P, s, t)
    g = oracle.linear_bwd(X, dY, Z, A, b, d, P=P, s=s, t=t)
    h = 0.5
    for idx in [(0, 0), (1, 3), (2, 7)]:
        Zc = Z.astype(np.float64)
        Zc[idx] += h / s
        up = _loss(X, A, b, Zc, dY, d)
        Zc[idx] -= 2 * h / s
        dn = _loss(X, A, b, Zc, dY, d)
        assert math.isclose(g["dP"][idx], (up - dn) / (2 * h), rel_tol=1e-9, abs_tol=1e-12)


def test_clipped_ste_masks_outside_clip_range_only():
    d, N, m, n = 4, 2, 2, 8
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    P = np.array([[-0.6, -0.5, 0.0, 1.7, 3.5, 3.6, 9.0, 2.0]] * 2, dtype=np.float32)
    X, dY = RNG.normal(size=(N, n)), RNG.normal(size=(N, m))
    Z = oracle.quantize(P)
    full = oracle.linear_bwd(X, dY, Z, A, b, d)["dP"]
    clip = oracle.linear_bwd(X, dY, Z, A, b, d, P=P, ste="clipped")["dP"]
    keep = np.array([False, True, True, True, True, False, False, True])
    assert np.all(clip[:, ~keep] == 0)
    np.testing.assert_array_equal(clip[:, keep], full[:, keep])


# ----------------------------------------------------------------------------- packing

def test_pack_golden_bytes(golden_dir):
    rows = read_rows("pack_bytes.txt")
    Z = np.array([[int(v) for v in r[:4]] for r in rows], dtype=np.uint8)
    want = np.array([int(r[4], 16) for r in rows], dtype=np.uint8)
    assert np.array_equal(oracle.pack2b(Z).ravel(), want)


def test_pack_unpack_round_trip():
    Z = RNG.integers(0, 4, (7, 64)).astype(np.uint8)
    P = oracle.pack2b(Z)
    assert P.shape == (7, 16)
    assert np.array_equal(oracle.unpack2b(P, 64), Z)


# ----------------------------------------------------------------------------- DGE (Sec. 3.3, Eq. dge)

def test_dge_surrogate_endpoints_and_slope_closed_forms(golden_dir):
    """f(0) = 0, f(delta/2) = delta/2, f(delta) = delta; f'(0) = f'(delta) = 1/k; f' = df/dx."""
    for k in (1.0, 3.0, 5.0):
        for delta in (1.0, 2.0):
            assert math.isclose(oracle.dge_f(0.0, k, delta), 0.0, abs_tol=1e-15)
            assert math.isclose(oracle.dge_f(delta / 2, k, delta), delta / 2, abs_tol=1e-15)
            assert math.isclose(oracle.dge_f(delta, k, delta), delta, rel_tol=1e-15)
            assert math.isclose(oracle.dge_fprime(0.0, k, delta), 1.0 / k, rel_tol=1e-15)
            assert math.isclose(oracle.dge_fprime(delta, k, delta), 1.0 / k, rel_tol=1e-15)
            for x in (0.1 * delta, 0.3 * delta, 0.7 * delta, 0.95 * delta):
                h = 1e-6 * delta
                fd = (oracle.dge_f(x + h, k, delta) - oracle.dge_f(x - h, k, delta)) / (2 * h)
                assert math.isclose(oracle.dge_fprime(x, k, delta), fd, rel_tol=1e-6)
    # the slope diverges at the boundary (the reason the implementation caps it)
    assert np.isinf(oracle.dge_fprime(0.5, 5.0))


def test_dge_with_k1_is_the_identity_estimator_inside_the_range():
    """k = 1 makes f(x) = x, slope 1: DGE reduces to the straight-through estimator on [0, 3)."""
    v = np.array([-0.7, -0.1, 0.0, 0.4, 1.5, 2.9, 3.0, 3.6])
    g = oracle.dge_grad(v, k=1.0, grad_max=10.0)
    assert list(g) == [0.0, 0.0, 1.0, 1.0, 1.0, 1.0, 0.0, 0.0]
    d, N, m, n = 4, 2, 3, 8
    A, b = RNG.normal(size=(d, d)), RNG.normal(size=d)
    P = RNG.uniform(0.01, 2.99, (m, n)).astype(np.float32)
    X, dY = RNG.normal(size=(N, n)), RNG.normal(size=(N, m))
    Z = oracle.quantize(P)
    ste = oracle.linear_bwd(X, dY, Z, A, b, d)["dP"]
    dge = oracle.linear_bwd(X, dY, Z, A, b, d, P=P, ste="dge", dge_k=1.0, dge_grad_max=10.0)["dP"]
    np.testing.assert_allclose(dge, ste, rtol=1e-15)


def test_dge_slope_is_periodic_and_capped():
    v = np.array([0.2, 1.2, 2.2, 0.5, 1.5, 0.49999])
    g = oracle.dge_grad(v, k=5.0, grad_max=3.0)
    np.testing.assert_allclose(g[:3], g[0], rtol=1e-12)
    assert g[3] == 3.0 and g[4] == 3.0 and g[5] == 3.0


# ----------------------------------------------------------------------------- initialisation (N2)

def test_xavier_preprocess_constants_and_levels(golden_dir):
    c = read_keyed("xavier_constants.txt")
    m, n = int(c["m"][0]), int(c["n"][0])
    P, s, t = oracle.init_latent(np.array([[0, 1, 2, 3]]), m, n)
    assert math.isclose(s, c["s"][0], rel_tol=1e-14) and t == c["t"][0]
    a = c["a"][0]
    np.testing.assert_allclose(P[0], [-a, -a / 3, a / 3, a], rtol=1e-14)


def test_xavier_preprocess_preserves_the_integer_weights():
    """Sec. 3.4: quantizing the preprocessed latents with the same (s, t) returns the integer weights."""
    for (m, n) in ((4096, 4096), (14336, 4096), (1024, 4096)):
        Z = RNG.integers(0, 4, (16, 64)).astype(np.uint8)
        P, s, t = oracle.init_latent(Z, m, n)
        assert np.array_equal(oracle.quantize(P.astype(np.float32), s, t), Z)


# ----------------------------------------------------------------------------- Hadamard rotation (N3)

def test_hadamard_blocks_are_the_largest_power_of_two_dividing_n():
    assert [oracle.hadamard_block(n) for n in (8, 24, 4096, 8192, 11008, 14336, 28672)] == \
        [8, 8, 4096, 8192, 256, 2048, 4096]


@pytest.mark.parametrize("n", [8, 24, 64, 96])
def test_hadamard_rotation_is_orthogonal_and_self_inverse(n):
    X = RNG.normal(size=(3, n))
    Xr = oracle.hadamard_rotate(X, n)
    np.testing.assert_allclose(np.linalg.norm(Xr, axis=1), np.linalg.norm(X, axis=1), rtol=1e-12)
    np.testing.assert_allclose(oracle.hadamard_rotate(Xr, n), X, atol=1e-12)
    # the first row of a Sylvester block is constant: column 0 of each block is the block mean times sqrt(bsz)
    bsz = oracle.hadamard_block(n)
    np.testing.assert_allclose(Xr[:, 0], X[:, :bsz].sum(axis=1) / np.sqrt(bsz), rtol=1e-12)


def test_rotation_cancels_through_the_product():
    """Rotating the activations and the weights by the same orthogonal H leaves Y unchanged:
    gemm_packed2b_hadamard(X H, codes) = gemm_packed2b(X, codes) since H H = I."""
    d, m, n = 4, 5, 32
    A, b = config_like_A(d, RNG), RNG.normal(0, 1e-3, d)
    Z = RNG.integers(0, 4, (m, n)).astype(np.uint8)
    X = RNG.normal(size=(2, n))
    np.testing.assert_allclose(oracle.gemm_packed2b_hadamard(oracle.hadamard_rotate(X, n), oracle.pack2b(Z), A, b, d, n),
                               oracle.gemm_packed2b(X, oracle.pack2b(Z), A, b, d, n), rtol=1e-12, atol=1e-14)


# ----------------------------------------------------------------------------- LDLQ initialisation

def _ar1(n, rho):
    i = np.arange(n)
    return rho ** np.abs(i[:, None] - i[None, :]).astype(np.float64)


def test_ldl_block_of_ar1_correlation_is_its_closed_form():
    """H_ij = rho^|i-j| (a stationary AR(1) covariance). Running the process backwards,
    x_i = rho x_{i+1} + sqrt(1 - rho^2) e_i, gives the scalar factor M_ij = rho^(j-i) (j >= i),
    D = diag(1 - rho^2, ..., 1 - rho^2, 1). The d-block factor is M B^-1, B D B^T with
    B = blockdiag(M_kk); by the Markov property only the first column of each off-diagonal
    block of U is non-zero: U[r, kd] = rho^(kd - r)."""
    rho, n = 0.7, 24
    H = _ar1(n, rho)
    U1, D1 = oracle.ldl_block(H, 1)
    i = np.arange(n)
    want_U1 = np.where(i[None, :] > i[:, None], rho ** (i[None, :] - i[:, None]).astype(float), 0.0)
    assert np.allclose(U1, want_U1, rtol=0, atol=1e-13)
    want_D1 = np.full(n, 1 - rho * rho)
    want_D1[-1] = 1.0
    assert np.allclose(D1[:, 0, 0], want_D1, rtol=0, atol=1e-13)
    for d in (4, 8):
        U, D = oracle.ldl_block(H, d)
        want_U = np.zeros((n, n))
        for k in range(1, n // d):
            want_U[:k * d, k * d] = rho ** (k * d - np.arange(k * d)).astype(float)
        assert np.allclose(U, want_U, rtol=0, atol=1e-13)
        for k in range(n // d):
            Mkk = np.triu(rho ** np.abs(np.subtract.outer(np.arange(d), np.arange(d))).astype(float))
            Dk = np.diag(want_D1[k * d:(k + 1) * d])
            assert np.allclose(D[k], Mkk @ Dk @ Mkk.T, rtol=0, atol=1e-13)


@pytest.mark.parametrize("d", [4, 8])
def test_ldl_block_reconstructs_spd_matrices(d):
    from paper_2606_10531_gb300 import workloads as wl
    rng = np.random.default_rng(7)
    Q = rng.normal(size=(64, 64))
    for H in (Q @ Q.T + 0.5 * np.eye(64), wl.draw_hessian(64, 0, 3).astype(np.float64)):
        U, D = oracle.ldl_block(H, d)
        n = H.shape[0]
        blk = np.arange(n) // d
        assert np.all(U[blk[:, None] >= blk[None, :]] == 0.0)       # strictly upper block-triangular
        Dfull = np.zeros((n, n))
        for k in range(n // d):
            assert np.allclose(D[k], D[k].T, rtol=0, atol=1e-12 * np.abs(D[k]).max())
            assert np.linalg.eigvalsh(D[k]).min() > 0
            Dfull[k * d:(k + 1) * d, k * d:(k + 1) * d] = D[k]
        M = U + np.eye(n)
        assert np.allclose(M @ Dfull @ M.T, H, rtol=0, atol=1e-11 * np.abs(H).max())


def _ldlq_case(m, n, d, seed, H=None):
    from paper_2606_10531_gb300 import workloads as wl
    rng = np.random.default_rng(seed)
    W = rng.normal(0.0, 0.015, (m, n))
    A = config_like_A(d, rng)
    b = rng.normal(0.0, 1e-3, d)
    if H is None:
        H = wl.draw_hessian(n, seed, 0).astype(np.float64)
    return W, A, b, H


@pytest.mark.parametrize("d", [4, 8])
def test_ldlq_with_block_diagonal_hessian_is_the_rounding_encoder(d):
    """No correlation between column groups: U = 0, no feedback, LDLQ = plain rounding."""
    rng = np.random.default_rng(11)
    n = 8 * d
    H = np.zeros((n, n))
    for k in range(n // d):
        Q = rng.normal(size=(d, d))
        H[k * d:(k + 1) * d, k * d:(k + 1) * d] = Q @ Q.T + np.eye(d)
    W, A, b, _ = _ldlq_case(16, n, d, 5, H)
    U, _ = oracle.ldl_block(H, d)
    assert np.all(U == 0.0)
    r = oracle.ldlq(W, U, A, b, d)
    e = oracle.encode(W, A, b, d)
    assert np.array_equal(r["codes"], e["codes"])
    assert r["mse"] == pytest.approx(e["mse"], rel=1e-12)


@pytest.mark.parametrize("d", [4, 8])
def test_ldlq_equals_the_optq_schur_complement_form(d):
    """QuIP shows LDLQ equals OPTQ: after the groups before k are fixed, the remaining columns are
    completed optimally, W_R - (W_hat_Q - W_Q) H_QR H_RR^-1, and group k is rounded from that.
    Computed here from H by linear solves, independently of the factorisation."""
    W, A, b, H = _ldlq_case(12, 8 * d, d, 21)
    m, n = W.shape
    Ainv = np.linalg.inv(A)
    What = np.zeros((m, n))
    Z = np.zeros((m, n), dtype=np.uint8)
    T = np.zeros((m, n))
    for k in range(n // d):
        q, r = slice(0, k * d), slice(k * d, n)
        TR = W[:, r] - (What[:, q] - W[:, q]) @ np.linalg.solve(H[r, r], H[q, r].T).T
        Tk = TR[:, :d]
        z = np.clip(np.rint((Tk - b) @ Ainv.T), 0, 3)
        Z[:, k * d:(k + 1) * d] = z
        What[:, k * d:(k + 1) * d] = z @ A.T + b
        T[:, k * d:(k + 1) * d] = Tk
    U, _ = oracle.ldl_block(H, d)
    res = oracle.ldlq(W, U, A, b, d)
    assert np.abs(res["target"] - T).max() < 1e-12
    assert np.array_equal(res["codes"], Z)
    assert not res["near"].any()


@pytest.mark.parametrize("d", [4, 8])
def test_ldlq_proxy_loss_is_the_d_weighted_sum_of_rounding_errors(d):
    """(W_hat - W)(U + I) = eta with eta_k = W_hat_k - T_k, so
    tr((W_hat - W) H (W_hat - W)^T) = sum_{r,k} eta_{r,k} D_k eta_{r,k}^T."""
    W, A, b, H = _ldlq_case(20, 16 * d, d, 31)
    U, D = oracle.ldl_block(H, d)
    res = oracle.ldlq(W, U, A, b, d)
    eta = (res["W_hat"] - res["target"]).reshape(W.shape[0], -1, d)
    rhs = float(np.einsum("rkj,kji,rki->", eta, D, eta))
    assert oracle.proxy_loss(W, res["W_hat"], H) == pytest.approx(rhs, rel=1e-9)


def test_ldlq_given_codes_reproduces_the_sweep_targets():
    W, A, b, H = _ldlq_case(24, 64, 8, 41)
    U, _ = oracle.ldl_block(H, 8)
    res = oracle.ldlq(W, U, A, b, 8)
    lat = oracle.ldlq_latent_given_codes(W, res["codes"], U, A, b, 8)
    assert np.abs(lat - res["latent"]).max() < 1e-10
    assert np.array_equal(oracle.round_clamp(lat), res["codes"])


def test_ldlq_keeps_codewords_fixed():
    """A matrix that is itself decoded codewords has zero error at every step: LDLQ returns its codes."""
    rng = np.random.default_rng(3)
    d = 8
    A = config_like_A(d, rng)
    b = rng.normal(0.0, 1e-3, d)
    Z0 = rng.integers(0, 4, (10, 64)).astype(np.uint8)
    W = oracle.decode(Z0, A, b, d)
    _, _, _, H = _ldlq_case(1, 64, d, 2)
    U, _ = oracle.ldl_block(H, d)
    assert np.array_equal(oracle.ldlq(W, U, A, b, d)["codes"], Z0)


def test_ldlq_lowers_the_proxy_loss_against_plain_rounding():
    """The feedback is what LDLQ adds: on a correlated Hessian its proxy loss is below that of
    rounding every group on its own (seeded instance)."""
    d = 8
    W, A, b, H = _ldlq_case(64, 256, d, 51)
    U, _ = oracle.ldl_block(H, d)
    res = oracle.ldlq(W, U, A, b, d)
    plain = oracle.decode(oracle.encode(W, A, b, d)["codes"], A, b, d)
    assert oracle.proxy_loss(W, res["W_hat"], H) < 0.9 * oracle.proxy_loss(W, plain, H)
