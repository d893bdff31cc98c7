// Host-side internal interface between the C ABI (lcq_api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/lcq.h"

namespace lcq {

void count_launch();
// cuTensorMapEncodeTiled from the driver (looked up once); nullptr if unavailable.
void *tensor_map_encoder();
// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) once per kernel and device.
cudaError_t ensure_dynamic_smem(const void *fn, int bytes);
// Record the start / end event of a kernel of the given lcq_kernel_kind on `st` (no-op unless tracing).
void trace_begin(int kind, cudaStream_t st);
void trace_end(int kind, cudaStream_t st);

struct EncodeArgs {
    const float *W;
    int64_t m, n;
    const float *A, *b;
    uint8_t *packed, *codes;
    float *latent;
    double *mse;
    double *partials;     // [grid] per-CTA sums of squared residuals
    unsigned *counter;    // zero between calls: the last CTA wraps it back (atomicInc)
    int32_t *status;
    // programmatic dependent launch inside lcq_encode_batch (independent matrices): bit 0 = let the
    // next launch start early, bit 1 = launched early (waits for the previous grid before it exits,
    // so completion stays in stream order). 0 for a single lcq_encode.
    int pdl = 0;
};

constexpr int kEncodeBatchMax = 16;   // = LCQ_ENCODE_BATCH_MAX
constexpr int kEncodeBatchPartials = 2048;   // per-matrix partials slots in a batch workspace (>= grid)

struct EncodeBatchItem {
    const float *W;
    int64_t m, n;
    const float *A, *b;
    uint8_t *packed, *codes;
    float *latent;
    double *mse;
    int64_t chunk0;       // first chunk of this matrix in the batch's chunk list
    int64_t nchunks;
};

struct EncodeBatchArgs {
    EncodeBatchItem item[kEncodeBatchMax];
    int count;
    int64_t total_chunks;
    double *partials;     // [count][grid] per-CTA sums of squared residuals
    unsigned *counters;   // [count], zero between calls (atomicInc wraps them back)
    int32_t *status;
};

// LDLQ (Sec. 2.2): block U D U^T factorisation of the proxy Hessian, and the error-feedback sweep.
struct LdlFactorArgs {
    const float *H;           // [n][n] symmetric positive definite (upper triangle read)
    int64_t n;
    int d;
    float *U;                 // [n][n] output, zero on and below the block diagonal
    float *D;                 // [n/d][d][d] output, or null
    float *scratch;           // ldl_factor_scratch_bytes(n)
    int32_t *status;
};
size_t ldl_factor_scratch_bytes(int64_t n);
cudaError_t launch_ldl_factor(const LdlFactorArgs &a, cudaStream_t st);

struct LdlqArgs {
    const float *W;
    int64_t m, n;
    int d;
    const float *A, *b, *U;
    uint8_t *packed, *codes;
    float *latent;
    double *mse;
    float *E;                 // error history, ldlq_history_bytes(m, n)
    double *partials;         // [ldlq_tiles(m)]
    int32_t *status;
};
int64_t ldlq_tiles(int64_t m);
size_t ldlq_history_bytes(int64_t m, int64_t n);
cudaError_t launch_ldlq(const LdlqArgs &a, cudaStream_t st);

// Chunk size (fp32 weights) of the encode pipeline.
int64_t encode_chunk_size();

struct QuantDecodeArgs {
    const float *P;
    int64_t m, n;
    const float *A, *b;
    float inv_s, t;
    uint8_t *packed;      // may be NULL
    uint16_t *W_hat;      // bf16 [m][n]
    int32_t *status;
};

struct DecodeArgs {
    const uint8_t *packed;
    int64_t m, n;
    const float *A, *b;
    float *W_f32;
    uint16_t *W_bf16;
};

int encode_max_blocks(int num_sms);
cudaError_t launch_encode(const EncodeArgs &a, int d, int num_sms, cudaStream_t st);
cudaError_t launch_encode_batch(const EncodeBatchArgs &a, int d, int num_sms, cudaStream_t st);
cudaError_t launch_quant_decode(const QuantDecodeArgs &a, int d, int num_sms, cudaStream_t st);
cudaError_t launch_decode(const DecodeArgs &a, int d, int num_sms, cudaStream_t st);
cudaError_t launch_pack2b(const uint8_t *codes, int64_t total, uint8_t *packed, int num_sms, cudaStream_t st);
cudaError_t launch_xform(const uint16_t *X, int64_t N, int64_t n, int d, const float *A, const float *b, uint16_t *Xp,
                         float *r, cudaStream_t st);
cudaError_t launch_wait_timeout_selftest(int32_t *status, cudaStream_t st);
cudaError_t launch_init_codebook(const float *G, int d, float *A, float *b, cudaStream_t st);
cudaError_t launch_init_latent(const uint8_t *packed, int64_t total, float s, float t, float *P, int num_sms,
                               cudaStream_t st);
cudaError_t launch_reduce_partials(const float *partials, int nparts, int d, float *dA, float *db, cudaStream_t st);

// ---------------------------------------------------------------- tensor-core GEMM
// C[M][N] = sum_k A(m, k) * B(n, k), bf16 operands, fp32 accumulation in TMEM.
// Operand X is "K-major" when stored [rows][K] (K contiguous) and "MN-major"
// when stored [K][rows].
enum GemmEpilogue { EPI_STORE_BF16 = 0, EPI_DW = 1 };

struct GemmOperand {
    const uint16_t *ptr;
    int64_t ld;          // elements between consecutive rows of the stored matrix
    bool mn_major;
};

struct DwEpilogue {
    const uint8_t *packed;   // [M][N/4] codes of the weight matrix
    const float *A;          // d x d
    const float *P;          // [M][N] latent weights (CLIPPED STE only), else NULL
    float *dP;               // [M][N]
    float *partials;         // [grid][d*d + d]
    float inv_s, t;
    int ste_mode;
    int d;
    float dge_inv_k;         // 1/k
    float dge_exp;           // 1/k - 1
    float dge_cap;
};

struct GemmProblem {
    int64_t M, N, K;
    GemmOperand a, b;
    uint16_t *C;             // EPI_STORE_BF16: [M][ldc] bf16
    int64_t ldc;
    DwEpilogue dw;
    int32_t *status;
    int trace_kind;          // lcq_kernel_kind recorded by the tracer
};

// Number of CTAs the persistent GEMM uses for this problem (partials rows for EPI_DW).
int gemm_grid(int64_t M, int64_t N, int num_sms);
cudaError_t launch_gemm(const GemmProblem &p, GemmEpilogue epi, int num_sms, cudaStream_t st);

// ---------------------------------------------------------------- packed 2-bit GEMV / small GEMM
struct PackedGemvArgs {
    const uint16_t *X;       // [N][n] bf16
    const float *Xf;         // [N][n] fp32 activations used instead of X when not NULL
    int64_t N, m, n;
    const uint8_t *packed;   // [m][n/4]
    const float *A, *b;
    uint16_t *Y;             // [N][m] bf16
    uint16_t *Xp;            // workspace: transformed activations [N][npad]
    float *corr;             // workspace: per-token constant, partial sums [N][nprep]
    int32_t *status;
    bool rotate = false;     // rotate X by the block Walsh-Hadamard transform in the product's prologue
};
// Argument checks of lcq_gemm_packed2b other than the workspace (LCQ_OK or the error it returns).
lcq_status check_gemm_packed2b_args(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n, int d,
                                    const float *A, const float *b, const uint16_t *Y);
size_t packed_gemv_workspace(int64_t N, int64_t n);
size_t packed_gemv_corr_offset(int64_t N, int64_t n);
cudaError_t launch_packed_gemv(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st);
// The tcgen05 (kind::mxf4) product for 1-16 tokens and n % 64 == 0, with its digits and constants in
// the workspace at a.Xp. Returns false (nothing launched) when it does not apply; err holds a launch
// error otherwise.
size_t packed_gemv_fp4_workspace(int64_t N, int64_t n);
bool launch_packed_gemv_fp4(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st, cudaError_t &err);
// The rotated product with the rotation inside the product: in the one-token kernel's prologue, else
// in the tcgen05 kernel's prep kernel (1-16 tokens). Returns false (nothing launched) when neither
// applies; err holds a launch error otherwise.
bool launch_packed_gemv_rotated(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st, cudaError_t &err);
// Row-wise normalized block Walsh-Hadamard rotation (block = largest power of two dividing n, <= 32768).
int hadamard_block_size(int64_t n);
cudaError_t launch_hadamard(const void *in, bool in_bf16, int64_t rows, int64_t n, float *out, cudaStream_t st);

}  // namespace lcq
