"""Plain fp64 CPU oracle of the LC-VQ linear layer (LC-QAT, arxiv 2606.10531).

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports this module:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its CPU
baseline and reference legs) may use it. It shares no code, table or helper
with the CUDA library; the two meet only through the seeded input
generators, which hold none of the method's arithmetic.

Every function is a literal restatement of one definition of the paper, in
the paper's notation, using NumPy fp64 and library primitives (matmul,
inverse) with no blocking, fusion or reordering:

  * codebook            c = A z + B, z in {0,1,2,3}^d          (Sec. 2.2, Eq. lc_codebook)
  * nearest codeword    i_g = argmin_k ||w_g - c_k||^2          (Sec. 2.1, Eq. vq_assign)
  * integer weights     W_z = clip(round(W_p), 0, 2^b - 1)      (Sec. 3.2, Eq. quant_param)
  * column grouping     G = n/d groups of d consecutive columns (Sec. 3.2)
  * decode              W_hat^T = [A W_{z,i}^T + B 1^T]_i       (Sec. 3.2, Eq. def:forward)
  * forward             Y = X W_hat^T (nn.Linear orientation)   (Sec. 3.2, Eq. def:forward_x)
  * activation side     X'_g = X_g A, r = sum_g X_g . B          (Sec. 3.2, Eq. def:forward_x)
  * backward            exact gradients of the linear map, with the
                        straight-through estimator dW_z/dW_p = 1 (Sec. 3.3)
  * LDLQ initialisation column groups quantized in order, each target
                        corrected by the earlier groups' errors through the
                        block U D U^T factor of the proxy Hessian (Sec. 2.2)

Readings where the paper is silent or inconsistent:
  * encode maps a real weight group to latent coordinates u = A^{-1}(w - B)
    and rounds/clamps u (Sec. 2.2 "rounding and clamping", Babai rounding);
  * round is round-half-to-even; NaN latent values encode to 0;
  * Y = X W_hat^T (the printed "Y = X W_hat" is shape-inconsistent);
  * the optional latent affine z = clip(round(P/s + t)) with dP = dZ/s
    reconciles Eq. quant_param with Eq. xavier_preprocess; s=1, t=0 is the
    literal Eq. quant_param. P/s + t is evaluated in fp32 (the precision in
    which the integer decision is taken on both sides): fl(fl(P*fl(1/s)) + t);
  * packed storage: 4 codes per byte, column c in bits 2(c mod 4)..+1 of
    byte floor(c/4), least significant first.
  * LDLQ (Sec. 2.2 names the algorithm, QuIP, and gives no formula): the
    block form with d x d blocks, the LC-VQ rounding encoder as the group
    quantizer, and errors W - W_hat measured against the original weights.
"""
from __future__ import annotations

import numpy as np

BITS = 2                       # b = 2 (Sec. 3.2, Eq. quant_param)
ZMAX = (1 << BITS) - 1         # 2^b - 1 = 3, largest level of {0,1,2,3}
COND_LIMIT = 1e8               # A with a larger condition number is "singular"


class SingularMatrix(ValueError):
    pass


def _f64(x):
    return np.asarray(x, dtype=np.float64)


def _grouped(M: np.ndarray, d: int) -> np.ndarray:
    """View an m x n matrix as (m, G, d): G = n/d groups of d consecutive columns (Sec. 3.2)."""
    m, n = M.shape
    if n % d:
        raise ValueError(f"n={n} is not a multiple of the group size d={d}")
    return M.reshape(m, n // d, d)


def inverse(A) -> np.ndarray:
    """A^{-1} in fp64 by the library LU inverse; refuses ill-conditioned A."""
    A64 = _f64(A)
    if not np.all(np.isfinite(A64)) or np.linalg.cond(A64) > COND_LIMIT:
        raise SingularMatrix("A is singular or ill-conditioned")
    return np.linalg.inv(A64)


def round_clamp(V) -> np.ndarray:
    """clip(round(v), 0, 2^b - 1) element-wise (Eq. quant_param); round half to even; NaN -> 0."""
    V64 = _f64(V)
    R = np.clip(np.rint(V64), 0, ZMAX)
    R = np.where(np.isnan(V64), 0.0, R)
    return R.astype(np.uint8)


def latent(W, A, b, d: int) -> np.ndarray:
    """Latent coordinates u_g = A^{-1}(w_g - B) of every weight group (Sec. 2.2 reading).

    Returns an (m, n) fp64 matrix laid out like W.
    """
    W64 = _f64(W)
    m, n = W64.shape
    Ainv = inverse(A)
    Wg = _grouped(W64, d) - _f64(b)            # w_g - B
    U = Wg @ Ainv.T                            # row-vector form of A^{-1} (w_g - B)
    return U.reshape(m, n)


def near_boundary(U, eps: float = 1e-5) -> np.ndarray:
    """Mask of latent values within eps of a decision boundary k + 1/2 of clamp(round(.)).

    Only 0.5, 1.5 and 2.5 are boundaries on {0,1,2,3}: below 0 and above 3
    the clamp absorbs the rounding.
    """
    U64 = _f64(U)
    mask = np.zeros(U64.shape, dtype=bool)
    for k in range(ZMAX):
        mask |= np.abs(U64 - (k + 0.5)) < eps
    return mask


def encode(W, A, b, d: int) -> dict:
    """LC-VQ encoder: z_g = clip(round(A^{-1}(w_g - B)), 0, 3) (Sec. 2.2; Eq. lc_codebook).

    Returns codes (uint8, m x n), latent u (fp64), the near-boundary mask and
    the reconstruction MSE mean((W - W_hat)^2).
    """
    U = latent(W, A, b, d)
    Z = round_clamp(U)
    return {"codes": Z, "latent": U, "near": near_boundary(U), "mse": mse(W, Z, A, b, d)}


def quantize(P, s: float = 1.0, t: float = 0.0) -> np.ndarray:
    """Integer weights W_z = clip(round(P/s + t), 0, 3) (Eq. quant_param; s=1, t=0 literal).

    P/s + t is formed in fp32 as fl(fl(P * fl(1/s)) + t): the precision in
    which the integer decision is made.
    """
    P32 = np.asarray(P, dtype=np.float32)
    inv_s = np.float32(1.0) / np.float32(s)
    V = (P32 * inv_s).astype(np.float32) + np.float32(t)
    return round_clamp(V.astype(np.float32))


def decode(Z, A, b, d: int) -> np.ndarray:
    """Affine decode w_hat_g = A z_g + B for every group (Eq. def:forward), fp64 (m x n)."""
    Z64 = _f64(Z)
    m, n = Z64.shape
    What = _grouped(Z64, d) @ _f64(A).T + _f64(b)   # row-vector form of A z_g + B
    return What.reshape(m, n)


def mse(W, Z, A, b, d: int) -> float:
    """Reconstruction error mean over all weights of (W - W_hat)^2 (fp64)."""
    W64 = _f64(W)
    if W64.size == 0:
        return 0.0
    return float(np.mean((W64 - decode(Z, A, b, d)) ** 2))


def linear_fwd(X, Z, A, b, d: int) -> np.ndarray:
    """Layer output Y = X W_hat^T with W_hat decoded from the integer weights (Eq. def:forward)."""
    return _f64(X) @ decode(Z, A, b, d).T


def activation_transform(X, A, b, d: int):
    """Activation side of the reformulated forward (Sec. 3.2, Eq. def:forward_x): per token and
    group of d columns, the row vector X_g A, and the bias term r = sum_g X_g . B, so that
    X W_hat^T = X' Z^T + r 1^T. Returns (X' (N x n), r (N,)) in fp64."""
    X64 = _f64(X)
    Xg = _grouped(X64, d)                      # (N, G, d)
    Xp = (Xg @ _f64(A)).reshape(X64.shape)
    r = (Xg @ _f64(b)).sum(axis=1)
    return Xp, r


DGE_K = 5.0          # sharpness k of the differentiable gradient estimator (Sec. 4.4)
DGE_GRAD_MAX = 3.0   # reading: cap on f'(x), which diverges at the rounding boundary (parity unpinned)


def dge_f(x, k: float = DGE_K, delta: float = 1.0):
    """Differentiable surrogate of rounding on one interval (Sec. 3.3, Eq. dge):
    f(x) = delta/2 * (1 + sign(2x/delta - 1) * |2x/delta - 1|^(1/k))."""
    y = 2.0 * _f64(x) / delta - 1.0
    return delta / 2.0 * (1.0 + np.sign(y) * np.abs(y) ** (1.0 / k))


def dge_fprime(x, k: float = DGE_K, delta: float = 1.0):
    """f'(x) = (1/k) * |2x/delta - 1|^(1/k - 1) (Sec. 3.3); infinite at x = delta/2."""
    y = np.abs(2.0 * _f64(x) / delta - 1.0)
    with np.errstate(divide="ignore"):
        return (1.0 / k) * y ** (1.0 / k - 1.0)


def dge_grad(V, k: float = DGE_K, grad_max: float = DGE_GRAD_MAX):
    """dz/dv of the DGE surrogate of clip(round(v), 0, 3) with delta = 1 (reading):
    on [0, 3) v = n + x with x = v - floor(v), the surrogate is n + f(x) and its slope f'(x),
    capped at grad_max; outside [0, 3) clip(round(.)) is flat and the slope is 0."""
    V64 = _f64(V)
    x = V64 - np.floor(V64)
    g = np.minimum(dge_fprime(x, k), grad_max)
    return np.where((V64 >= 0.0) & (V64 < ZMAX), g, 0.0)


def linear_bwd(X, dY, Z, A, b, d: int, P=None, s: float = 1.0, t: float = 0.0,
               ste: str = "identity", dge_k: float = DGE_K, dge_grad_max: float = DGE_GRAD_MAX) -> dict:
    """Gradients of L with dL/dY = dY through Y = X W_hat^T, W_hat = decode(Z).

    The layer is linear in X, A, B and in z treated as a real vector, so:
        dW_hat = dY^T X
        dX     = dY W_hat
        dz_g   = A^T dw_hat_g          (row-vector form: dw_hat_g @ A)
        dA     = sum_{r,g} dw_hat_{r,g} z_{r,g}^T
        dB     = sum_{r,g} dw_hat_{r,g}
    and the straight-through estimator dW_z/dW_p = 1 (Sec. 3.3) gives
    dP = dZ / s; with ste="clipped" the gradient is zeroed where
    P/s + t lies outside [-1/2, 2^b - 1/2]; with ste="dge" it is scaled by the
    slope of the differentiable gradient estimator at v = P/s + t (dge_grad).
    """
    X64, dY64, A64 = _f64(X), _f64(dY), _f64(A)
    What = decode(Z, A, b, d)
    dWhat = dY64.T @ X64
    dX = dY64 @ What
    dWg = _grouped(dWhat, d)
    Zg = _grouped(_f64(Z), d)
    dZ = (dWg @ A64).reshape(dWhat.shape)
    dA = np.einsum("rgj,rgk->jk", dWg, Zg)
    db = dWg.sum(axis=(0, 1))
    dP = dZ / s
    if ste == "clipped":
        if P is None:
            raise ValueError("ste='clipped' needs P")
        P32 = np.asarray(P, dtype=np.float32)
        V = ((P32 * (np.float32(1.0) / np.float32(s))).astype(np.float32) + np.float32(t)).astype(np.float64)
        dP = np.where((V >= -0.5) & (V <= ZMAX + 0.5), dP, 0.0)
    elif ste == "dge":
        if P is None:
            raise ValueError("ste='dge' needs P")
        P32 = np.asarray(P, dtype=np.float32)
        V = ((P32 * (np.float32(1.0) / np.float32(s))).astype(np.float32) + np.float32(t)).astype(np.float64)
        dP = dP * dge_grad(V, dge_k, dge_grad_max)
    elif ste != "identity":
        raise ValueError(f"unknown ste mode {ste!r}")
    return {"dX": dX, "dP": dP, "dA": dA, "db": db, "dW_hat": dWhat}


def pack2b(Z) -> np.ndarray:
    """Pack 2-bit codes 4 per byte: column c -> bits 2(c mod 4) of byte floor(c/4), LSB first."""
    Zu = np.asarray(Z, dtype=np.uint8)
    m, n = Zu.shape
    if n % 4:
        raise ValueError("n must be a multiple of 4 to pack")
    Q = Zu.reshape(m, n // 4, 4).astype(np.uint32)
    out = np.zeros((m, n // 4), dtype=np.uint32)
    for q in range(4):
        out |= (Q[:, :, q] & 3) << (2 * q)
    return out.astype(np.uint8)


def unpack2b(packed, n: int) -> np.ndarray:
    """Inverse of pack2b."""
    Pk = np.asarray(packed, dtype=np.uint8)
    m = Pk.shape[0]
    Z = np.zeros((m, n // 4, 4), dtype=np.uint8)
    for q in range(4):
        Z[:, :, q] = (Pk >> (2 * q)) & 3
    return Z.reshape(m, n)


def gemm_packed2b(X, packed, A, b, d: int, n: int) -> np.ndarray:
    """Deployment product Y = X W_hat^T from packed codes: unpack, decode, multiply."""
    return linear_fwd(X, unpack2b(packed, n), A, b, d)


def init_codebook(G, bits: int = BITS):
    """A = s G, B = -s G mu 1 with mu = (2^b - 1)/2 and s = sqrt(12/(2^{2b} - 1)) (Eq. init_ab)."""
    G64 = _f64(G)
    mu = ((1 << bits) - 1) / 2.0
    s = np.sqrt(12.0 / ((1 << (2 * bits)) - 1))
    A = s * G64
    B = -s * G64 @ (mu * np.ones(G64.shape[0]))
    return A, B


def init_latent(Z, m: int, n: int, bits: int = BITS):
    """Latent (proxy) weights from integer weights, Eq. xavier_preprocess: W_p = s (W_z - t) with
    s = 2a/(2^b - 1), t = (2^b - 1)/2, a = sqrt(6/(m+n)). Returns (W_p fp64, s, t)."""
    a = np.sqrt(6.0 / (m + n))
    L = (1 << bits) - 1
    s = 2.0 * a / L
    t = L / 2.0
    return s * (_f64(Z) - t), s, t


def hadamard_block(n: int, max_block: int = 32768) -> int:
    """Block size of the incoherence rotation (reading): the largest power of two dividing n, at most max_block."""
    bsz = 1
    while n % (bsz * 2) == 0 and bsz * 2 <= max_block:
        bsz *= 2
    return bsz


def hadamard_rotate(M, n: int):
    """Right-multiply the rows of M by the normalized block-diagonal Walsh-Hadamard matrix H of size n
    (blocks of hadamard_block(n)); H is symmetric and orthogonal (Sec. 2.2 incoherence processing, reading)."""
    import scipy.linalg
    bsz = hadamard_block(n)
    Hb = scipy.linalg.hadamard(bsz).astype(np.float64) / np.sqrt(bsz)
    M64 = _f64(M)
    rows = M64.shape[0]
    return (M64.reshape(rows, n // bsz, bsz) @ Hb).reshape(rows, n)


def gemm_packed2b_hadamard(X, packed, A, b, d: int, n: int) -> np.ndarray:
    """Deployment product with online rotation of the activations: Y = (X H) W_hat^T, where the
    codes encode the rotated weights W H (App. Inference Speed: Hadamard transform, then the product)."""
    return gemm_packed2b(hadamard_rotate(X, n), packed, A, b, d, n)


def brute_nearest(W, A, b, d: int):
    """Exhaustive nearest codeword over all 4^d codewords (Eq. vq_assign on Eq. lc_codebook).

    Runs the C searcher in oracle/brute.c. Returns (codes uint8 m x n, squared distance per group).
    """
    from . import _native
    return _native.brute_nearest(W, A, b, d)


# ----------------------------------------------------------------------------- LDLQ initialisation
#
# Sec. 2.2 initialises the codes with LDLQ (QuIP, Chee et al. 2023): the column groups of W are
# quantized one after another, and each group's target is its own weights plus the accumulated
# reconstruction error of the groups before it, fed forward through the factor of the proxy
# Hessian H. With groups of d columns (the block form used for vector quantizers, QuIP#):
#
#     H = (U + I) D (U + I)^T      U strictly upper block-triangular (d x d blocks), D block diagonal
#     T_k = W_k + sum_{j<k} (W_j - W_hat_j) U_{j,k}            (target of column group k)
#     z_k = clip(round(A^{-1}(T_k - B)), 0, 3),  W_hat_k = A z_k + B   (the LC-VQ rounding encoder)
#
# With U = 0 (H block diagonal) this is the plain encoder. The reconstruction error of the result
# satisfies (W_hat - W)(U + I) = eta, eta_k = W_hat_k - T_k, so the proxy loss
# tr((W_hat - W) H (W_hat - W)^T) equals sum_k sum_r eta_{r,k} D_k eta_{r,k}^T.

def ldl_block(H, d: int):
    """Block U D U^T factorisation H = (U + I) D (U + I)^T of a symmetric positive definite matrix
    (the factorisation LDLQ feeds its errors through; Sec. 2.2, LDLQ).

    Eliminates the d x d blocks from the last to the first: D_k is the current Schur-complement
    block, the column block above it is U_{<k,k} = S_{<k,k} D_k^{-1}, and the leading blocks are
    replaced by their Schur complement S_{<k,<k} - S_{<k,k} D_k^{-1} S_{k,<k}.
    Returns U (n x n fp64, zero on and below the block diagonal) and D (G x d x d fp64).
    """
    S = _f64(H).copy()
    n = S.shape[0]
    if S.shape != (n, n) or n % d:
        raise ValueError("H must be n x n with n a multiple of d")
    G = n // d
    U = np.zeros((n, n))
    D = np.zeros((G, d, d))
    for k in reversed(range(G)):
        blk = slice(k * d, (k + 1) * d)
        D[k] = S[blk, blk]
        if k == 0:
            break
        lead = slice(0, k * d)
        Uk = S[lead, blk] @ np.linalg.inv(D[k])
        U[lead, blk] = Uk
        S[lead, lead] -= Uk @ S[blk, lead]
    return U, D


def ldlq(W, U, A, b, d: int) -> dict:
    """LDLQ sweep with the LC-VQ rounding encoder as the group quantizer (Sec. 2.2, LDLQ):
    column groups k = 0 .. G-1 in order, target T_k = W_k + sum_{j<k} (W_j - W_hat_j) U_{j,k}.

    U is the strictly upper block factor of ldl_block. Returns the codes (uint8 m x n), the latent
    coordinates of the targets u = A^{-1}(T - B) (fp64, for the near-boundary mask), the targets T,
    the reconstruction MSE mean((W - W_hat)^2) and W_hat.
    """
    W64, U64, A64, b64 = _f64(W), _f64(U), _f64(A), _f64(b)
    m, n = W64.shape
    if n % d:
        raise ValueError(f"n={n} is not a multiple of the group size d={d}")
    Ainv = inverse(A)
    What = np.zeros((m, n))
    T = np.zeros((m, n))
    Ulat = np.zeros((m, n))
    Z = np.zeros((m, n), dtype=np.uint8)
    for k in range(n // d):
        blk = slice(k * d, (k + 1) * d)
        Tk = W64[:, blk] + (W64[:, :k * d] - What[:, :k * d]) @ U64[:k * d, blk]
        uk = (Tk - b64) @ Ainv.T                  # row-vector form of A^{-1} (T_k - B)
        zk = round_clamp(uk)
        Z[:, blk] = zk
        What[:, blk] = zk.astype(np.float64) @ A64.T + b64
        T[:, blk] = Tk
        Ulat[:, blk] = uk
    return {"codes": Z, "latent": Ulat, "near": near_boundary(Ulat), "target": T, "W_hat": What,
            "mse": float(np.mean((W64 - What) ** 2)) if W64.size else 0.0}


def ldlq_latent_given_codes(W, Z, U, A, b, d: int) -> np.ndarray:
    """Latent coordinates A^{-1}(T_k - B) of every LDLQ target when the earlier groups were decided
    as Z (Sec. 2.2, LDLQ): T = W + (W - decode(Z)) U with U strictly upper block-triangular, so
    T_k only sees groups j < k. A valid LDLQ result satisfies round_clamp(latent) == Z."""
    W64 = _f64(W)
    m, n = W64.shape
    T = W64 + (W64 - decode(Z, A, b, d)) @ _f64(U)
    return ((_grouped(T, d) - _f64(b)) @ inverse(A).T).reshape(m, n)


def proxy_loss(W, W_hat, H) -> float:
    """tr((W_hat - W) H (W_hat - W)^T), the layer-output error LDLQ minimises for E[x x^T] = H."""
    E = _f64(W_hat) - _f64(W)
    return float(np.einsum("ri,ij,rj->", E, _f64(H), E))
