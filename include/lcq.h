/*
 * lcq.h - C ABI of liblcq, the GB300 (sm_103a) LC-VQ linear layer.
 *
 * LC-QAT (arxiv 2606.10531) stores a weight matrix W (m x n, nn.Linear
 * orientation: m outputs, n inputs) as 2-bit integer weights z in {0,1,2,3}
 * grouped in d consecutive input columns, plus one affine map (A, B) per
 * matrix (Sec. 2.2 Eq. lc_codebook; Sec. 3.2 Eq. def:forward):
 *
 *     w_hat[r, g*d + j] = sum_k A[j][k] * z[r, g*d + k] + B[j]
 *
 * Conventions shared by every call:
 *   - Tensors are caller-owned DEVICE pointers, row-major and contiguous,
 *     16-byte aligned (LCQ_ERR_ALIGN otherwise). A is d x d fp32 row-major,
 *     b (the paper's B) is d fp32. bf16 tensors are passed as uint16_t bit
 *     patterns.
 *   - d must be 4 or 8 (LCQ_ERR_UNSUPPORTED); n must be a multiple of 8
 *     (and of d); m, n, N >= 0. Empty problems are valid and write the
 *     mathematically correct (zero) results.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream). Every call
 *     is asynchronous and stream-ordered; argument validation is
 *     synchronous and happens before anything is enqueued.
 *   - The library never allocates device memory. Calls that need scratch
 *     take `ws`/`ws_bytes`, a caller-owned device buffer of at least
 *     lcq_workspace_size(op, ...) bytes (LCQ_ERR_WORKSPACE otherwise). The
 *     first 256 bytes of a workspace hold a device status word that kernels
 *     set on device-detected errors (LCQ_ERR_SINGULAR, LCQ_ERR_TIMEOUT);
 *     read it with lcq_device_status(). The header must be zero before a
 *     workspace is first used (lcq_encode also keeps a counter there that
 *     returns to zero at the end of every call); after a device-detected
 *     error, zero it again. A workspace must not be shared by calls that may
 *     run concurrently.
 *   - Packed codes: 4 per byte; column c of a row sits in bits
 *     2*(c mod 4) .. 2*(c mod 4)+1 of byte c/4 of that row (LSB first);
 *     a packed matrix is m x (n/4) bytes.
 */
#ifndef LCQ_H
#define LCQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum lcq_status {
    LCQ_OK = 0,
    LCQ_ERR_NULL = 1,        /* a required pointer is NULL                              */
    LCQ_ERR_SHAPE = 2,       /* negative size, n % d != 0, n % 8 != 0                   */
    LCQ_ERR_ALIGN = 3,       /* a tensor pointer is not 16-byte aligned                 */
    LCQ_ERR_UNSUPPORTED = 4, /* d not in {4, 8}, unknown STE mode                       */
    LCQ_ERR_WORKSPACE = 5,   /* workspace NULL or smaller than lcq_workspace_size()     */
    LCQ_ERR_CUDA = 6,        /* a CUDA runtime call or kernel launch failed             */
    LCQ_ERR_SINGULAR = 7,    /* device-detected: A (or a block of D, LDLQ) not invertible */
    LCQ_ERR_TIMEOUT = 8,     /* device-detected: a bounded pipeline wait gave up        */
    LCQ_ERR_ARG = 9,         /* any other invalid argument (e.g. latent_scale == 0)     */
    LCQ_ERR_LIMIT = 10       /* problem larger than the static scratch of a _noalloc call */
} lcq_status;

/* Operation selector for lcq_workspace_size(). */
typedef enum lcq_op {
    LCQ_OP_ENCODE = 1,
    LCQ_OP_LINEAR_FWD = 2,
    LCQ_OP_LINEAR_BWD = 3,
    LCQ_OP_GEMM_PACKED2B = 4,
    LCQ_OP_GEMM_PACKED2B_HADAMARD = 5,
    LCQ_OP_ENCODE_BATCH = 6,         /* N = number of matrices; m, n unused */
    LCQ_OP_LDL_FACTOR = 7,           /* n, d; N, m unused */
    LCQ_OP_LDLQ = 8                  /* m, n, d; N unused */
} lcq_op;

/* Gradient estimators for dP through the rounding (Sec. 3.3). */
typedef enum lcq_ste_mode {
    LCQ_STE_IDENTITY = 0, /* dW_z/dW_p = 1 everywhere (the paper's STE)                  */
    LCQ_STE_CLIPPED = 1,  /* zero where P/s + t lies outside [-1/2, 7/2]                 */
    LCQ_STE_DGE = 2       /* differentiable gradient estimator (Eq. dge), see lcq_opts */
} lcq_ste_mode;

/*
 * Options of the training calls. NULL means {1, 0, LCQ_STE_IDENTITY, 0, 5, 3}.
 * LCQ_STE_DGE scales dP by the slope of the estimator at v = P/s + t: on [0, 3),
 * with x = v - floor(v) (interval delta = 1), min(dge_grad_max, (1/k)|2x - 1|^(1/k - 1));
 * 0 outside [0, 3). dge_k and dge_grad_max <= 0 select the defaults k = 5 (the
 * paper's setting) and a cap of 3 (the paper does not state a cap).
 */
typedef struct lcq_opts {
    float latent_scale;   /* s: integer weights are clip(round(P/s + t), 0, 3); must be != 0 */
    float latent_offset;  /* t                                                                 */
    int32_t ste_mode;     /* lcq_ste_mode                                                      */
    int32_t reserved;     /* must be 0                                                         */
    float dge_k;          /* DGE sharpness k                                                   */
    float dge_grad_max;   /* DGE slope cap                                                     */
} lcq_opts;

/*
 * Bytes of device workspace an operation needs for the given sizes
 * (N = tokens, m = output rows, n = input dim, d = group size). Returns 0
 * for an unknown op. The size only grows with each argument.
 */
size_t lcq_workspace_size(int op, int64_t N, int64_t m, int64_t n, int d);

/*
 * lcq_encode - map real weights to 2-bit latent codes (Sec. 2.2: codewords
 * A z + B; z obtained by rounding and clamping; Eq. quant_param with b = 2).
 *
 *   u[r, g*d + k] = sum_j Ainv[k][j] * (W[r, g*d + j] - b[j]),  Ainv = A^{-1}
 *   z = clip(round_half_even(u), 0, 3)   (NaN -> 0, +inf -> 3, -inf -> 0)
 *
 * W       [m][n] fp32 input.
 * packed  [m][n/4] uint8 output, or NULL.
 * codes   [m][n] uint8 output (one code per byte), or NULL.
 * latent  [m][n] fp32 output u, or NULL.
 * mse     device double, receives mean((W - (A z + b))^2) over all m*n
 *         weights (0 when m*n == 0), or NULL.
 * A^{-1} is formed on the device to fp32 accuracy (fp32 Gauss-Jordan refined
 * by Newton steps with a double-float residual; fp64 Gauss-Jordan when A is
 * badly conditioned); if A is singular the device status word becomes
 * LCQ_ERR_SINGULAR and every code is 0. Needs lcq_workspace_size(LCQ_OP_ENCODE, 0, m, n, d) bytes of ws.
 */
lcq_status lcq_encode(const float *W, int64_t m, int64_t n, int d, const float *A, const float *b,
                      uint8_t *packed, uint8_t *codes, float *latent, double *mse,
                      void *ws, size_t ws_bytes, void *stream);

/* One matrix of lcq_encode_batch: the arguments of lcq_encode for it. */
typedef struct lcq_encode_item {
    const float *W;        /* [m][n] fp32 input                              */
    int64_t m, n;          /* n a multiple of 8                              */
    const float *A, *b;    /* its affine map (d x d row-major, d)            */
    uint8_t *packed;       /* [m][n/4] uint8 output, or NULL                 */
    uint8_t *codes;        /* [m][n] uint8 output, or NULL                   */
    float *latent;         /* [m][n] fp32 output, or NULL                    */
    double *mse;           /* device double output, or NULL                  */
} lcq_encode_item;

#define LCQ_ENCODE_BATCH_MAX 16

/*
 * lcq_encode_batch - lcq_encode of several matrices (the bulk encode of all linears of a layer: PTQ
 * initialisation, per-step requantisation). Every output is exactly the one lcq_encode gives for the
 * same matrix. The matrices share the group size d. When no item asks for the MSE they stream through
 * one persistent launch, so the per-call costs (launch, forming A^{-1}, filling the ring) are paid
 * once for the batch; when any item asks for it, each matrix gets its own launch (measured faster),
 * and each launch after the first starts while the previous one drains (programmatic dependent
 * launch); work enqueued after the call still sees every output.
 *
 * items  host array of `count` matrices, 1 <= count <= LCQ_ENCODE_BATCH_MAX; each item is
 *        validated as lcq_encode validates its arguments. The items must be independent: no item's
 *        outputs may overlap another item's inputs or outputs.
 * Needs lcq_workspace_size(LCQ_OP_ENCODE_BATCH, count, 0, 0, d) bytes of ws. The workspace header
 * holds one counter per matrix, which returns to zero at the end of every call (the header must be
 * zero before first use). If any A is singular the status word becomes LCQ_ERR_SINGULAR and that
 * matrix's codes are 0.
 */
lcq_status lcq_encode_batch(const lcq_encode_item *items, int count, int d, void *ws, size_t ws_bytes,
                            void *stream);

/*
 * lcq_ldl_factor - block U D U^T factorisation of a proxy Hessian, the factor LDLQ feeds its errors
 * through (Sec. 2.2 initialises the codes with LDLQ):
 *
 *     H = (U + I) D (U + I)^T
 *
 * U is strictly upper block-triangular in d x d blocks (zero on and below the block diagonal), D is
 * block diagonal. Computed in fp32 through the Cholesky factorisation H = R R^T in reverse index order
 * (R upper triangular; 128-column panels from the last to the first): with Rd the block diagonal of R,
 * U + I = R Rd^-1 and D_k = R_kk R_kk^T. D_k is written as the Schur-complement block it factors.
 * If a pivot of D_k is not positive (H not positive definite), the status word becomes
 * LCQ_ERR_SINGULAR and that block's contributions are zero.
 *
 * H  [n][n] fp32, symmetric positive definite; only its upper triangle (i <= j) is read.
 * U  [n][n] fp32 output; every element is written.
 * D  [n/d][d][d] fp32 output (block k is D_k), or NULL.
 * Needs lcq_workspace_size(LCQ_OP_LDL_FACTOR, 0, 0, n, d) bytes of ws (a copy of H, about 4 n^2 bytes).
 * Streams: each panel's factorisation runs on a library-owned high-priority stream (one per device),
 * forked from and joined back to `stream` by events, so work enqueued on `stream` after the call sees
 * every output and the call can be captured into a CUDA graph. Concurrent calls are safe; they share
 * that stream's order.
 */
lcq_status lcq_ldl_factor(const float *H, int64_t n, int d, float *U, float *D, void *ws, size_t ws_bytes,
                          void *stream);

/*
 * lcq_ldlq - LDLQ initialisation of the codes (Sec. 2.2): the column groups k = 0, 1, ... of W are
 * rounded in order by the LC-VQ encoder, each from a target that carries the earlier groups' errors
 * forward through the factor U of lcq_ldl_factor (rows are independent):
 *
 *     T_k = W_k + sum_{j<k} (W_j - W_hat_j) U_{j,k},    z_k = clip(round_half_even(A^{-1}(T_k - b)), 0, 3),
 *     W_hat_k = A z_k + b                               (W_k: the d columns of group k)
 *
 * W       [m][n] fp32 input.
 * U       [n][n] fp32; only the entries above the block diagonal are read.
 * packed  [m][n/4] uint8 output, or NULL.
 * codes   [m][n] uint8 output (one code per byte), or NULL.
 * latent  [m][n] fp32 output: u = A^{-1}(T_k - b), the value each code was rounded from, or NULL.
 * mse     device double, receives mean((W - W_hat)^2) (0 when m*n == 0), or NULL.
 * Arithmetic is fp32; the feedback sums of a target run over up to n terms, in another order than a
 * sequential evaluation. If A is singular the status word becomes LCQ_ERR_SINGULAR and every code is 0.
 * Needs lcq_workspace_size(LCQ_OP_LDLQ, 0, m, n, d) bytes of ws (the error history, 4 n bytes per
 * row of m rounded up to 64 rows).
 */
lcq_status lcq_ldlq(const float *W, int64_t m, int64_t n, int d, const float *A, const float *b, const float *U,
                    uint8_t *packed, uint8_t *codes, float *latent, double *mse, void *ws, size_t ws_bytes,
                    void *stream);

/*
 * lcq_decode - affine decode of packed codes (Sec. 3.2 Eq. def:forward):
 *   W_hat[r, g*d + j] = sum_k A[j][k] * z[r, g*d + k] + b[j]
 * packed [m][n/4] uint8 input. W_hat_f32 [m][n] fp32 and/or W_hat_bf16 [m][n]
 * bf16 outputs (either may be NULL, not both). Needs no workspace.
 */
lcq_status lcq_decode(const uint8_t *packed, int64_t m, int64_t n, int d, const float *A, const float *b,
                      float *W_hat_f32, uint16_t *W_hat_bf16, void *stream);

/*
 * lcq_activation_transform - activation side of the reformulated forward (Sec. 3.2,
 * Eq. def:forward_x), for every token t and group g of d columns:
 *   X'[t, g*d + k] = sum_j X[t, g*d + j] * A[j][k]     (the row vector X_g times A)
 *   r[t]           = sum_g sum_j X[t, g*d + j] * b[j]
 * so that X W_hat^T = X' Z^T + r 1^T for the decoded weights W_hat_g = A z_g + b.
 * X [N][n] bf16 input; Xp [N][n] bf16 output (rounded to nearest even) or NULL;
 * r [N] fp32 output or NULL (not both NULL unless N = 0). r is summed in a
 * fixed order (bitwise reproducible). Needs no workspace.
 */
lcq_status lcq_activation_transform(const uint16_t *X, int64_t N, int64_t n, int d, const float *A, const float *b,
                                    uint16_t *Xp, float *r, void *stream);

/*
 * lcq_pack2b - storage of the 2-bit codes (Sec. 2.1: in the 2-bit setting each
 * dimension takes one of 4 values, so four codes fill a byte). Packs
 * one-code-per-byte codes [m][n] into [m][n/4] bytes in the library's bit
 * order (see the header comment). Only the two low bits of each input byte are
 * used. n must be a multiple of 4. Needs no workspace.
 */
lcq_status lcq_pack2b(const uint8_t *codes, int64_t m, int64_t n, uint8_t *packed, void *stream);

/*
 * lcq_linear_fwd - forward pass of one LC-VQ linear layer (Sec. 3.2,
 * Eq. quant_param and Eq. def:forward; output orientation of nn.Linear):
 *   Z = clip(round(P/s + t), 0, 3)      (P/s + t formed in fp32 as fl(fl(P*fl(1/s)) + t))
 *   W_hat = A Z_g + b per group          (rounded to bf16 as the GEMM operand)
 *   Y = X W_hat^T                        (bf16 tensor-core GEMM, fp32 accumulation)
 * X [N][n] bf16, P [m][n] fp32 latent (proxy) weights, Y [N][m] bf16 output,
 * packed_saved [m][n/4] uint8 output (the integer weights, for the backward;
 * may be NULL). Needs lcq_workspace_size(LCQ_OP_LINEAR_FWD, N, m, n, d).
 */
lcq_status lcq_linear_fwd(const uint16_t *X, int64_t N, const float *P, int64_t m, int64_t n, int d,
                          const float *A, const float *b, const lcq_opts *opts,
                          uint16_t *Y, uint8_t *packed_saved, void *ws, size_t ws_bytes, void *stream);

/*
 * lcq_linear_bwd - straight-through backward of one LC-VQ linear layer
 * (Sec. 3.3; exact gradients of the linear map of Eq. def:forward):
 *   dW_hat = dY^T X                                      (fp32, never stored)
 *   dX     = dY W_hat                                    [N][n] bf16
 *   dP[r, g*d + k] = (1/s) * sum_j dW_hat[r, g*d + j] A[j][k]  (masked in CLIPPED mode)
 *   dA[j][k] = sum_{r,g} dW_hat[r, g*d + j] * z[r, g*d + k]     [d][d] fp32
 *   db[j]    = sum_{r,g} dW_hat[r, g*d + j]                     [d] fp32
 * X [N][n] bf16, dY [N][m] bf16, packed_saved [m][n/4] from lcq_linear_fwd,
 * P [m][n] fp32 (read only in CLIPPED and DGE modes; may be NULL otherwise).
 * dX may be NULL (skips the dX GEMM). dA and db are overwritten, not
 * accumulated; the sums are taken in a fixed order (bitwise reproducible).
 * m must be a multiple of 8 as well as n (LCQ_ERR_SHAPE otherwise, before
 * anything is enqueued): dY's rows are read by TMA in 16-byte units.
 * Needs lcq_workspace_size(LCQ_OP_LINEAR_BWD, N, m, n, d).
 */
lcq_status lcq_linear_bwd(const uint16_t *X, const uint16_t *dY, const uint8_t *packed_saved, const float *P,
                          int64_t N, int64_t m, int64_t n, int d, const float *A, const float *b,
                          const lcq_opts *opts, uint16_t *dX, float *dP, float *dA, float *db,
                          void *ws, size_t ws_bytes, void *stream);

/*
 * lcq_gemm_packed2b - deployment product from packed 2-bit codes through the
 * reformulated forward (Sec. 3.2 Eq. def:forward_x):
 *   Y = sum_g (X_g A) Z_g^T + sum_g (X_g b) 1^T  ( = X W_hat^T )
 * X [N][n] bf16 activations (any N; built for N <= 16 tokens), packed
 * [m][n/4] uint8 codes, Y [N][m] bf16 output. How X_g A is rounded before
 * the product depends on the shape:
 *   - n % 64 == 0 and n <= 32768, one token: to int16 with one scale per
 *     token, exact integer sums;
 *   - the same n, 2-16 tokens: to q = rint(X' 8191 / max|X'_t|) per token
 *     (five base-8 digits, the tensor cores' fp4 operands), exact integer
 *     sums;
 *   - any other shape: to bf16, fp32 accumulation.
 * Needs lcq_workspace_size(LCQ_OP_GEMM_PACKED2B, N, m, n, d).
 */
lcq_status lcq_gemm_packed2b(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n,
                             int d, const float *A, const float *b, uint16_t *Y,
                             void *ws, size_t ws_bytes, void *stream);

/*
 * lcq_gemm_packed2b_noalloc - lcq_gemm_packed2b for callers that cannot
 * allocate device memory. The paper has no counterpart: this entry point
 * exists for callers that hand all device memory to their own fixed pool at
 * start-up and must not allocate afterwards (for example a serving process
 * with a hard memory budget), and for C callers with no device allocator.
 *
 * Same arguments and results as lcq_gemm_packed2b, without ws/ws_bytes: the
 * scratch lives in one static device array of 1.25 MiB + 4 KiB that every GPU
 * which loads the library holds until the process exits. The call itself
 * allocates nothing (no cudaMalloc, cudaFree or allocating library routine).
 *   - Limits: N <= 16 tokens and n <= 32768; larger problems return
 *     LCQ_ERR_LIMIT before anything is enqueued.
 *   - device_status: optional device int32 that receives the call's device
 *     status word (LCQ_OK or a device-detected error); may be NULL.
 *   - Every call shares the array and it keeps the last call's contents;
 *     the call clears what must start at zero. Calls that can overlap on the
 *     GPU (other streams, other host threads) race on the array.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make it before any
 *     stream capture.
 */
lcq_status lcq_gemm_packed2b_noalloc(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n,
                                     int d, const float *A, const float *b, uint16_t *Y,
                                     int32_t *device_status, void *stream);

/*
 * lcq_hadamard - incoherence rotation of Sec. 2.2 (Hadamard transform following QuIP#), read as a
 * normalized block-diagonal Walsh-Hadamard matrix H whose block is the largest power of two dividing
 * n (at most 32768): out[r] = in[r] H for each of `rows` rows of length n (fp32, device; in may equal
 * out). H is symmetric and orthogonal, so rotating twice restores the input. Used to rotate weights
 * before lcq_encode when the deployment product rotates the activations (lcq_gemm_packed2b_hadamard).
 */
lcq_status lcq_hadamard(const float *in, int64_t rows, int64_t n, float *out, void *stream);

/*
 * lcq_gemm_packed2b_hadamard - deployment product with online rotation of the activations
 * (App. Inference Speed: Hadamard transform, then the fused affine-dequant product):
 *   Y = (X H) W_hat^T, with the codes encoding the rotated weights W H (see lcq_hadamard).
 * Arguments as lcq_gemm_packed2b; needs lcq_workspace_size(LCQ_OP_GEMM_PACKED2B_HADAMARD, N, m, n, d).
 * The rotated activations are kept in fp32. The rotation runs inside the product where a product
 * kernel takes the shape: one token at n = 8192 in the one-token kernel's prologue, 1-16 tokens with
 * n % 64 == 0 and n <= 32768 in the tcgen05 kernel's prep (two launches per call); other shapes rotate
 * into the workspace in a kernel of their own first.
 */
lcq_status lcq_gemm_packed2b_hadamard(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n,
                                      int d, const float *A, const float *b, uint16_t *Y,
                                      void *ws, size_t ws_bytes, void *stream);

/*
 * lcq_init_codebook - codebook initialisation of Sec. 2.2 Eq. init_ab for b = 2:
 *   A = s G,  b = -s G mu 1,  mu = (2^b - 1)/2 = 1.5,  s = sqrt(12 / (2^{2b} - 1)) = sqrt(0.8)
 * G [d][d] fp32 (a random orthogonal matrix chosen by the caller), A [d][d] and b [d] fp32 outputs;
 * all device pointers. Over all 4^d codewords the codebook then has mean 0 and covariance G G^T.
 */
lcq_status lcq_init_codebook(const float *G, int d, float *A, float *b, void *stream);

/*
 * lcq_init_latent - latent (proxy) weights from integer weights, Sec. 3.4 Eq. xavier_preprocess:
 *   P = s (z - t),  s = 2a / (2^b - 1),  t = (2^b - 1) / 2,  a = sqrt(6 / (m + n))
 * packed [m][n/4] uint8 codes in, P [m][n] fp32 out (device). *s_out and *t_out (host, may be NULL)
 * receive s and t as used (fp32): passing them as lcq_opts.latent_scale / latent_offset makes
 * lcq_linear_fwd quantize P back to exactly the same codes.
 */
lcq_status lcq_init_latent(const uint8_t *packed, int64_t m, int64_t n, float *P, float *s_out, float *t_out,
                           void *stream);

/*
 * lcq_device_status - synchronise `stream`, then copy the workspace's device
 * status word (LCQ_OK or a device-detected lcq_status) to *status_out and,
 * if clear != 0, reset it to LCQ_OK.
 */
lcq_status lcq_device_status(const void *ws, void *stream, int32_t *status_out, int clear);

/*
 * lcq_selftest_wait_timeout - exercise the bounded-wait error path on the GPU
 * (measurement and reliability support; the paper has no counterpart). One
 * CTA waits on an mbarrier phase that nothing completes, using the same
 * bounded wait as every pipeline of the library; after about 2 seconds it gives
 * up, sets LCQ_ERR_TIMEOUT in the workspace status word and returns, leaving
 * the context usable. ws: at least 256 bytes of device memory.
 */
lcq_status lcq_selftest_wait_timeout(void *ws, void *stream);

/* Static description of a status code; never NULL. */
const char *lcq_status_string(lcq_status s);

/* Text of the CUDA error behind the most recent LCQ_ERR_CUDA in this process ("no error" if none). */
const char *lcq_last_cuda_error(void);

/* Number of kernels this library has launched in the calling process. */
uint64_t lcq_launch_count(void);

/*
 * Kernel tracing with CUDA events (measurement support; not part of the
 * paper's method). While enabled, every kernel the library launches is
 * bracketed by two events recorded on the launching stream; records beyond
 * LCQ_TRACE_CAPACITY are dropped. lcq_trace_enable(1) clears the records and
 * starts recording, lcq_trace_enable(0) stops. Not thread-safe: trace from one
 * host thread at a time.
 */
#define LCQ_TRACE_CAPACITY 4096
typedef enum lcq_kernel_kind {
    LCQ_K_ENCODE = 0,        /* encode stream kernel                         */
    LCQ_K_QUANT_DECODE = 1,  /* forward prologue: quantize + decode to bf16  */
    LCQ_K_DECODE = 2,        /* decode packed codes                          */
    LCQ_K_PACK = 3,          /* pack one-code-per-byte codes                 */
    LCQ_K_GEMM_FWD = 4,      /* tensor-core GEMM, Y = X W_hat^T              */
    LCQ_K_GEMM_DX = 5,       /* tensor-core GEMM, dX = dY W_hat              */
    LCQ_K_GEMM_DW = 6,       /* tensor-core GEMM, dW_hat = dY^T X + dP/dA/db */
    LCQ_K_REDUCE = 7,        /* fixed-order dA/db reduction                  */
    LCQ_K_GEMV_PREP = 8,     /* reserved (the transform is timed inside GEMV) */
    LCQ_K_GEMV = 9,          /* packed product: activation transform + main  */
    LCQ_K_LDL_FACTOR = 10,   /* LDLQ: block U D U^T factorisation (all its launches) */
    LCQ_K_LDLQ = 11,         /* LDLQ: error-feedback sweep                   */
    LCQ_K_XFORM = 12,        /* activation transform X' = X_g A, r = X_g . b  */
    LCQ_K_NUM_KINDS = 13
} lcq_kernel_kind;
lcq_status lcq_trace_enable(int on);
/*
 * Synchronise on the recorded events and report, for one kernel kind, the
 * number of recorded launches and the sum of their durations in milliseconds.
 */
lcq_status lcq_trace_read(int kind, uint64_t *launches, double *total_ms);

#ifdef __cplusplus
}
#endif

#endif /* LCQ_H */
