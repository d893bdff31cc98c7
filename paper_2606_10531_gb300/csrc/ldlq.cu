// LDLQ initialisation of the codes (Sec. 2.2 adopts LDLQ, QuIP): the column groups of W are
// quantized in order, each group's target being its weights plus the earlier groups' errors fed
// through the block U D U^T factor of the proxy Hessian H:
//
//     H = (U + I) D (U + I)^T,   T_k = W_k + sum_{j<k} (W_j - W_hat_j) U_{j,k},
//     z_k = clip(round(A^{-1}(T_k - b)), 0, 3),   W_hat_k = A z_k + b.
//
// Factorisation (ldl_panel_kernel, ldl_gemm_k128_kernel, ldl_syrk_kernel): H = R R^T with R upper
// triangular (a Cholesky factorisation in reverse index order), from which D_k = R_kk R_kk^T and
// U = R Rd^-1 - I (Rd = the block diagonal of R). Right-looking over 128-column panels from the last
// to the first: one CTA factors a panel's diagonal block in shared memory and forms W = R_PP^-1; the
// column block above it, Z = S_QP W^T (with U_QP = Z Rd^-1 in the same kernel), and the Schur update
// S_QQ -= Z Z^T (upper triangle only) are fp32 SIMT GEMMs.
//
// Sweep (ldlq_sweep_kernel): rows are independent, so one CTA takes 64 rows through every column
// chunk of 128 columns. For chunk c it first forms the feedback of all earlier columns as a GEMM,
// F = E_{<c} U_{<c,c} (E = W - W_hat, this CTA's own error history, written by it in earlier chunks),
// then rounds the chunk's groups in order, adding the in-chunk feedback as it goes. One producer
// thread streams 32-row slices of U (and of the error history) through a TMA ring; the error history
// of the previous chunk is loaded only after the compute threads have published it (an mbarrier
// phase per chunk, after a generic-to-async proxy fence).
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "invert.cuh"

namespace lcq {

// ================================================================== factorisation

constexpr int kLdlPanel = 128;        // panel width (columns), a multiple of 8
constexpr int kLdlThreads = 256;
constexpr int kLdlLd = kLdlPanel + 4; // rows 16-byte aligned, consecutive rows 4 banks apart
constexpr int kLdlRinvLd = 72;        // floats between the groups of R_kk^-1 (8 banks apart)
constexpr int kLdlBarColumns = 1;     // named barrier: the column block of R is complete

// The panel's diagonal block is factored as S = R R^T with R upper triangular (a Cholesky factorisation
// in reverse index order, group by group). The block factor follows from it without d x d inversions:
// D_k = R_kk R_kk^T and U = R Rd^-1 - I (Rd = block diagonal of R). The panel hands W = R^-1 and the
// R_kk^-1 to the trailing update: Z = S_QP W^T is the factor's column block above the panel,
// U_QP = Z Rd^-1 and the Schur update is S_QQ -= Z Z^T.
struct LdlPanelSmem {
    float S[kLdlPanel][kLdlLd];       // Schur block (block-upper part current); row block k becomes W's once consumed
    float R[kLdlPanel][kLdlLd];       // R's column blocks above the diagonal blocks, as they are formed
    float RT[8][kLdlPanel];           // the current column block of R, transposed
    float Rinv[kLdlPanel / 4][kLdlRinvLd];   // R_kk^-1 per group (D x D row-major, upper triangular)
};

__device__ __forceinline__ void ldl_named_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void ldl_named_arrive(int id, int count) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// One warp: S_kk = R_kk R_kk^T (upper triangle of S_kk read) and R_kk^-1. Every lane factors the block
// in registers (pivots from the last index to the first); lane j then forms column j of R_kk^-1. A pivot
// that is not positive relative to the block's largest entry (or a non-finite block) sets
// LCQ_ERR_SINGULAR and leaves R_kk^-1 zero.
template <int D>
__device__ void ldl_factor_group(LdlPanelSmem &s, int k, float *Dk, int32_t *status) {
    const int lane = threadIdx.x & 31, kd = k * D;
    if (Dk) {
        for (int e = lane; e < D * D; e += 32) {
            const int i = e / D, j = e % D;
            Dk[e] = i <= j ? s.S[kd + i][kd + j] : s.S[kd + j][kd + i];
        }
    }
    float a[D][D];                                 // upper triangle
    float amax = 0.0f;
#pragma unroll
    for (int i = 0; i < D; ++i)
#pragma unroll
        for (int j = i; j < D; ++j) {
            a[i][j] = s.S[kd + i][kd + j];
            amax = fmaxf(amax, fabsf(a[i][j]));
        }
    bool ok = amax > 0.0f && isfinite(amax);
    float ip[D];                                   // 1 / R_pp
#pragma unroll
    for (int p = D - 1; p >= 0; --p) {
        const float piv = a[p][p];
        ok = ok && piv > 1e-12f * amax;
        ip[p] = rsqrtf(fmaxf(piv, 1e-30f));
#pragma unroll
        for (int i = 0; i <= p; ++i) a[i][p] *= ip[p];          // column p of R
#pragma unroll
        for (int i = 0; i < p; ++i)
#pragma unroll
            for (int j = i; j < p; ++j) a[i][j] = fmaf(-a[i][p], a[j][p], a[i][j]);
    }
    // column `lane` of R_kk^-1 by back substitution
    float x[D];
#pragma unroll
    for (int q = 0; q < D; ++q) x[q] = q == lane ? ip[q] : 0.0f;
#pragma unroll
    for (int r = D - 2; r >= 0; --r) {
        float acc = 0.0f;
#pragma unroll
        for (int l = r + 1; l < D; ++l) acc = fmaf(a[r][l], x[l], acc);
        if (r < lane) x[r] = -acc * ip[r];
    }
    if (lane < D) {
#pragma unroll
        for (int r = 0; r < D; ++r) s.Rinv[k][r * D + lane] = ok ? x[r] : 0.0f;
    }
    if (lane == 0 && !ok) set_status(status, LCQ_ERR_SINGULAR);
    __syncwarp();
}

// Row i of the column block k of R: R_{i,k} = S_{i,k} R_kk^-T, outputs 4h .. 4h+3 (into R and RT).
template <int D>
__device__ __forceinline__ void ldl_column_quad(LdlPanelSmem &s, int k, int i, int h) {
    const int kd = k * D;
    float sv[D];
#pragma unroll
    for (int q = 0; q < D; q += 4) {
        const float4 v = *reinterpret_cast<const float4 *>(&s.S[i][kd + q]);
        sv[q] = v.x; sv[q + 1] = v.y; sv[q + 2] = v.z; sv[q + 3] = v.w;
    }
    float o[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const float *rr = &s.Rinv[k][(4 * h + t) * D];     // row 4h+t of R_kk^-1 (zero below the diagonal)
        float acc = 0.0f;
#pragma unroll
        for (int q = 0; q < D; q += 4) {
            const float4 r4 = *reinterpret_cast<const float4 *>(rr + q);
            acc = fmaf(sv[q], r4.x, acc);
            acc = fmaf(sv[q + 1], r4.y, acc);
            acc = fmaf(sv[q + 2], r4.z, acc);
            acc = fmaf(sv[q + 3], r4.w, acc);
        }
        o[t] = acc;
    }
    *reinterpret_cast<float4 *>(&s.R[i][kd + 4 * h]) = make_float4(o[0], o[1], o[2], o[3]);
#pragma unroll
    for (int t = 0; t < 4; ++t) s.RT[4 * h + t][i] = o[t];
}

// Row block k of W = R^-1 (into S's row block k, whose Schur entries are consumed): W_kk = R_kk^-1 and
// W_{k,j} = -R_kk^-1 sum_{k<l<=j} R_{k,l} W_{l,j}; needs W's row blocks after k. Threads t < nthr in
// pairs: a pair takes one column, each summing every other 4-row chunk of it.
template <int D>
__device__ __forceinline__ void ldl_w_row_block(LdlPanelSmem &s, int k, int P, int t, int nthr) {
    const int kd = k * D;
    for (int e = t; e < D * D; e += nthr) s.S[kd + e / D][kd + e % D] = s.Rinv[k][e];
    const int items = 2 * (P - kd - D);
    for (int base = 0; base < items; base += nthr) {           // uniform trip count: the pair exchange below
        const int e = base + t;
        const int half = e & 1, col = kd + D + (e >> 1);
        const int cend = e < items ? (col / D + 1) * D : kd + D;
        float T[D];
#pragma unroll
        for (int q = 0; q < D; ++q) T[q] = 0.0f;
        for (int cs = kd + D + 4 * half; cs < cend; cs += 8) {
            const float w0 = s.S[cs][col], w1 = s.S[cs + 1][col], w2 = s.S[cs + 2][col], w3 = s.S[cs + 3][col];
#pragma unroll
            for (int q = 0; q < D; ++q) {
                const float4 rv = *reinterpret_cast<const float4 *>(&s.R[kd + q][cs]);
                T[q] = fmaf(rv.x, w0, fmaf(rv.y, w1, fmaf(rv.z, w2, fmaf(rv.w, w3, T[q]))));
            }
        }
#pragma unroll
        for (int q = 0; q < D; ++q) T[q] += __shfl_xor_sync(0xffffffffu, T[q], 1);
        if (e < items) {
#pragma unroll
            for (int rr = 0; rr < D / 2; ++rr) {
                const int r = half * (D / 2) + rr;
                float acc = 0.0f;
#pragma unroll
                for (int q = 0; q < D; ++q) acc = fmaf(s.Rinv[k][r * D + q], T[q], acc);
                s.S[kd + r][col] = -acc;
            }
        }
    }
}

// Factor the diagonal block S[c0:c0+P, c0:c0+P] (upper triangle read) of the current Schur complement.
// Writes U's panel block, D (if requested), W = R^-1 (P x P, leading dimension kLdlPanel, zero below
// the diagonal) and the R_kk^-1 (P/D blocks of D x D).
// Iteration k (from G down to 1; G = P / D): with the column block R_{<k,k} = S_{<k,k} R_kk^-T formed,
// warp 0 updates the next diagonal block S_{k-1,k-1} -= R_{k-1,k} R_{k-1,k}^T and factors it, while
// warps 1.. apply the rest of the Schur update S_{<k,<k} -= R_{<k,k} R_{<k,k}^T (block-upper part, one
// D x D block per thread), write U_{<k,k} = R_{<k,k} R_kk^-1 and form W's row block k.
template <int D>
__global__ void __launch_bounds__(kLdlThreads)
ldl_panel_kernel(const float *__restrict__ S, int64_t n, int64_t c0, int P, float *__restrict__ U,
                 float *__restrict__ Dout, float *__restrict__ Wout, float *__restrict__ RinvOut, int32_t *status) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    LdlPanelSmem &s = *reinterpret_cast<LdlPanelSmem *>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = P / D, P4 = P / 4;
    constexpr int NQ = D / 4;                      // output quads per row of a column block
    constexpr int kWork = kLdlThreads - 32;        // threads of warps 1..
    // the block-upper part of S in 16-byte chunks, eight loads in flight per thread
    {
        constexpr int kBatch = 8;
        const int total = P * P4;
        for (int e0 = tid; e0 < total; e0 += kLdlThreads * kBatch) {
            float4 v[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int e = e0 + u * kLdlThreads;
                const int i = e / P4, j = (e % P4) * 4;
                v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (e < total && j / D >= i / D)
                    v[u] = __ldg(reinterpret_cast<const float4 *>(S + (c0 + i) * n + c0 + j));
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int e = e0 + u * kLdlThreads;
                const int i = e / P4, j = (e % P4) * 4;
                if (e < total && j / D >= i / D) *reinterpret_cast<float4 *>(&s.S[i][j]) = v[u];
            }
        }
    }
    __syncthreads();
    for (int k = G; k >= 1; --k) {
        const int kd = k * D, kp = kd - D;
        const bool cols = k < G;                   // the column block k exists (R_kk known)
        if (warp == 0) {
            if (cols) {
                if (lane < D * NQ) ldl_column_quad<D>(s, k, kp + lane / NQ, lane % NQ);
                __syncwarp();
                ldl_named_arrive(kLdlBarColumns, kLdlThreads);
                for (int e = lane; e < D * D; e += 32) {
                    const int r = e / D, c = e % D;
                    float acc = s.S[kp + r][kp + c];
#pragma unroll
                    for (int q = 0; q < D; ++q) acc = fmaf(-s.RT[q][kp + r], s.RT[q][kp + c], acc);
                    s.S[kp + r][kp + c] = acc;
                }
                __syncwarp();
            }
            ldl_factor_group<D>(s, k - 1, Dout ? Dout + (c0 / D + k - 1) * D * D : nullptr, status);
        } else if (cols) {
            const int t = tid - 32;
            for (int e = t; e < kp * NQ; e += kWork) ldl_column_quad<D>(s, k, e / NQ, e % NQ);
            ldl_named_sync(kLdlBarColumns, kLdlThreads);
            // Schur update: blocks (gi, gj), gi <= gj < k, in row-major order, all but the last, (k-1, k-1)
            const int nblk = k * (k + 1) / 2 - 1;
            for (int e = t; e < nblk; e += kWork) {
                int gi = 0, rem = e;
                while (rem >= k - gi) { rem -= k - gi; ++gi; }
                const int gj = gi + rem;
                float c[D][D];
#pragma unroll
                for (int r = 0; r < D; ++r)
#pragma unroll
                    for (int q = 0; q < D; q += 4) {
                        const float4 v = *reinterpret_cast<const float4 *>(&s.S[gi * D + r][gj * D + q]);
                        c[r][q] = v.x; c[r][q + 1] = v.y; c[r][q + 2] = v.z; c[r][q + 3] = v.w;
                    }
#pragma unroll
                for (int q = 0; q < D; ++q) {
                    float av[D], bv[D];
#pragma unroll
                    for (int u = 0; u < D; u += 4) {
                        const float4 a4 = *reinterpret_cast<const float4 *>(&s.RT[q][gi * D + u]);
                        const float4 b4 = *reinterpret_cast<const float4 *>(&s.RT[q][gj * D + u]);
                        av[u] = a4.x; av[u + 1] = a4.y; av[u + 2] = a4.z; av[u + 3] = a4.w;
                        bv[u] = b4.x; bv[u + 1] = b4.y; bv[u + 2] = b4.z; bv[u + 3] = b4.w;
                    }
#pragma unroll
                    for (int r = 0; r < D; ++r)
#pragma unroll
                        for (int cc = 0; cc < D; ++cc) c[r][cc] = fmaf(-av[r], bv[cc], c[r][cc]);
                }
#pragma unroll
                for (int r = 0; r < D; ++r)
#pragma unroll
                    for (int q = 0; q < D; q += 4)
                        *reinterpret_cast<float4 *>(&s.S[gi * D + r][gj * D + q]) =
                            make_float4(c[r][q], c[r][q + 1], c[r][q + 2], c[r][q + 3]);
            }
            // U_{<k,k} = R_{<k,k} R_kk^-1, one row per thread
            for (int i = t; i < kd; i += kWork) {
                float rv[D];
#pragma unroll
                for (int q = 0; q < D; q += 4) {
                    const float4 v = *reinterpret_cast<const float4 *>(&s.R[i][kd + q]);
                    rv[q] = v.x; rv[q + 1] = v.y; rv[q + 2] = v.z; rv[q + 3] = v.w;
                }
                float o[D];
#pragma unroll
                for (int jj = 0; jj < D; ++jj) {
                    float acc = 0.0f;
#pragma unroll
                    for (int q = 0; q <= jj; ++q) acc = fmaf(rv[q], s.Rinv[k][q * D + jj], acc);
                    o[jj] = acc;
                }
                float *dst = U + (c0 + i) * n + c0 + kd;
#pragma unroll
                for (int q = 0; q < D; q += 4)
                    *reinterpret_cast<float4 *>(dst + q) = make_float4(o[q], o[q + 1], o[q + 2], o[q + 3]);
            }
            ldl_w_row_block<D>(s, k, P, t, kWork);
        }
        __syncthreads();
    }
    ldl_w_row_block<D>(s, 0, P, tid, kLdlThreads);
    __syncthreads();
    // W (zero below the block diagonal and below the diagonal of W_kk, which S holds as zeros) and R_kk^-1
    for (int e = tid; e < P * P4; e += kLdlThreads) {
        const int i = e / P4, j = (e % P4) * 4;
        const float4 v = j / D >= i / D ? *reinterpret_cast<const float4 *>(&s.S[i][j]) : make_float4(0.f, 0.f, 0.f, 0.f);
        *reinterpret_cast<float4 *>(Wout + i * kLdlPanel + j) = v;
    }
    for (int e = tid; e < G * D * D; e += kLdlThreads) RinvOut[e] = s.Rinv[e / (D * D)][e % (D * D)];
}

// The trailing update's GEMMs. All have K = kLdlPanel = 128 (the panel width; only the first panel can
// be narrower, and no update follows it) and both operands K-contiguous (C += A B^T form).
//
// ldl_gemm_k128_kernel: C[i][j] = beta C[i][j] + alpha sum_k A[i][k] B[j][k] on a 64 x 64 tile, the
// whole K of both operands copied to shared memory up front by cp.async (one load latency per tile:
// these run on the critical path between two panels). Thread (ty, tx) computes rows ty + 16 i and
// columns tx + 16 j (i, j < 4), reading its operand rows 16 bytes of K at a time. EPI_D > 0 (alpha = 1,
// beta = 0, N a multiple of EPI_D): also U2 = C blockdiag(Rinv) with the EPI_D x EPI_D blocks Rinv[g]
// (U2[i][j] = sum_q C[i][gD + q] Rinv[g][q][j - gD], g = j / EPI_D).
constexpr int kGemmTile = 64, kGemmKAll = kLdlPanel, kGemmLd = kGemmKAll + 4;

struct GemmK128Smem {
    float As[kGemmTile][kGemmLd];     // A tile, row-major (rows 16-byte aligned, 4 banks apart)
    float Bs[kGemmTile][kGemmLd];
};
static_assert(kGemmTile * (kGemmTile + 4) <= kGemmTile * kGemmLd, "the C tile reuses As");

__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gsrc, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem_dst)), "l"(gsrc),
                 "r"(valid ? 16 : 0)
                 : "memory");
}

template <int EPI_D>
__global__ void __launch_bounds__(256)
ldl_gemm_k128_kernel(const float *__restrict__ Am, int64_t lda, const float *__restrict__ Bm, int64_t ldb,
                     float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, float alpha, float beta,
                     const float *__restrict__ Rinv, float *__restrict__ U2, int64_t ldu2) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    GemmK128Smem &s = *reinterpret_cast<GemmK128Smem *>(smem_raw);
    const int64_t i0 = static_cast<int64_t>(blockIdx.y) * kGemmTile, j0 = static_cast<int64_t>(blockIdx.x) * kGemmTile;
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    // 64 rows x 32 16-byte chunks per operand: rows (tid >> 3) + 32 v, chunks (tid & 7) + 8 u; rows past
    // the matrix are zero-filled (the source address stays the operand's first row)
#pragma unroll
    for (int v = 0; v < 2; ++v)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int r = (tid >> 3) + 32 * v, q = (tid & 7) + 8 * u;
            const bool va = i0 + r < M, vb = j0 + r < N;
            cp_async16(&s.As[r][4 * q], Am + (va ? (i0 + r) * lda : 0) + 4 * q, va);
            cp_async16(&s.Bs[r][4 * q], Bm + (vb ? (j0 + r) * ldb : 0) + 4 * q, vb);
        }
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    float acc[4][4] = {};
#pragma unroll 4
    for (int k = 0; k < kGemmKAll; k += 4) {
        float4 a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            a[i] = *reinterpret_cast<const float4 *>(&s.As[ty + 16 * i][k]);
            b[i] = *reinterpret_cast<const float4 *>(&s.Bs[tx + 16 * i][k]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                acc[i][j] = fmaf(a[i].x, b[j].x, acc[i][j]);
                acc[i][j] = fmaf(a[i].y, b[j].y, acc[i][j]);
                acc[i][j] = fmaf(a[i].z, b[j].z, acc[i][j]);
                acc[i][j] = fmaf(a[i].w, b[j].w, acc[i][j]);
            }
    }
    if constexpr (EPI_D > 0) {
        // the C tile through shared memory: a group of EPI_D columns spans several threads
        __syncthreads();
        float(*Cs)[kGemmTile + 4] = reinterpret_cast<float(*)[kGemmTile + 4]>(&s.As[0][0]);
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) Cs[ty + 16 * i][tx + 16 * j] = acc[i][j];
        __syncthreads();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int lc = tx + 16 * j;
            const int64_t c = j0 + lc;
            if (c >= N) continue;
            const int jj = static_cast<int>(c % EPI_D), lg = lc - jj;
            const float *Rg = Rinv + (c / EPI_D) * EPI_D * EPI_D + jj;
            float rq[EPI_D];
#pragma unroll
            for (int q = 0; q < EPI_D; ++q) rq[q] = __ldg(Rg + q * EPI_D);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t r = i0 + ty + 16 * i;
                if (r >= M) continue;
                float u = 0.0f;
#pragma unroll
                for (int q = 0; q < EPI_D; ++q) u = fmaf(Cs[ty + 16 * i][lg + q], rq[q], u);
                U2[r * ldu2 + c] = u;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = i0 + ty + 16 * i;
        if (r >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t c = j0 + tx + 16 * j;
            if (c >= N) continue;
            float *p = C + r * ldc + c;
            *p = beta == 0.0f ? alpha * acc[i][j] : fmaf(alpha, acc[i][j], beta * *p);
        }
    }
}

// ldl_syrk_kernel: the leading square of the Schur update, C -= Z Z^T on the tiles (ti <= tj) of a
// 128 x 128 tiling of the m x m upper triangle (m a multiple of 4; one CTA per tile, blockIdx.x the
// tile's index in row-major order). K = 128 in steps of 16: cp.async copies the steps' rows of both
// operands into a 4-stage raw ring three steps ahead; each step is transposed in shared memory
// (As[k][row]) for conflict-free 16-byte operand reads; 8 x 8 outputs per thread (rows ty*4 + {0..3,
// 64..67}, likewise the columns), accumulated with packed fp32x2 FMAs. The epilogue passes the tile
// through shared memory so that all of a thread's C loads are in flight at once.
constexpr int kSyrkTile = 128, kSyrkK = 16, kSyrkLd = kSyrkTile + 4, kSyrkRaw = 4;
constexpr int kSyrkSteps = kLdlPanel / kSyrkK;

struct SyrkSmem {
    float raw[kSyrkRaw][2][kSyrkTile][kSyrkK];   // [stage][operand][row][k], as copied
    float T[2][2][kSyrkK][kSyrkLd];              // [buffer][operand][k][row]
};
static_assert(sizeof(float) * kSyrkTile * kSyrkTile <= sizeof(float) * kSyrkRaw * 2 * kSyrkTile * kSyrkK,
              "the epilogue's C tile reuses the raw ring");

__global__ void __launch_bounds__(256, 2)
ldl_syrk_kernel(const float *__restrict__ Zm, int64_t ldz, float *__restrict__ C, int64_t ldc, int64_t m, int nt) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    SyrkSmem &s = *reinterpret_cast<SyrkSmem *>(smem_raw);
    int ti = 0, rem = static_cast<int>(blockIdx.x);
    while (rem >= nt - ti) { rem -= nt - ti; ++ti; }
    const int tj = ti + rem;
    const int64_t i0 = static_cast<int64_t>(ti) * kSyrkTile, j0 = static_cast<int64_t>(tj) * kSyrkTile;
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    // copies: rows (tid >> 2) + 64 v of each operand, 16-byte chunk (tid & 3) of the step's 16 columns;
    // rows past m are zero-filled (the source address stays the operand's first row)
    const int lr = tid >> 2, lq = tid & 3;
    const auto issue = [&](int step) {
        if (step < kSyrkSteps) {
            const int k0 = step * kSyrkK, st = step % kSyrkRaw;
#pragma unroll
            for (int v = 0; v < 2; ++v) {
                const int r = lr + 64 * v;
                const bool va = i0 + r < m, vb = j0 + r < m;
                cp_async16(&s.raw[st][0][r][4 * lq], Zm + (va ? (i0 + r) * ldz : 0) + k0 + 4 * lq, va);
                cp_async16(&s.raw[st][1][r][4 * lq], Zm + (vb ? (j0 + r) * ldz : 0) + k0 + 4 * lq, vb);
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    issue(0);
    issue(1);
    issue(2);
    float2 acc[8][4];                                  // acc[i][j] holds columns 2j, 2j + 1 (packed FMAs)
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = make_float2(0.0f, 0.0f);
#pragma unroll 1
    for (int step = 0; step < kSyrkSteps; ++step) {
        asm volatile("cp.async.wait_group 2;" ::: "memory");   // this step's copies have landed
        __syncthreads();                                      // ... for every thread; step - 1 is consumed
        issue(step + 3);                                      // into the raw stage step - 1 used
        const int st = step % kSyrkRaw, tb = step & 1;
#pragma unroll
        for (int o = 0; o < 2; ++o)
#pragma unroll
            for (int v = 0; v < 2; ++v) {
                const int r = lr + 64 * v;
                const float4 x = *reinterpret_cast<const float4 *>(&s.raw[st][o][r][4 * lq]);
                s.T[tb][o][4 * lq][r] = x.x;
                s.T[tb][o][4 * lq + 1][r] = x.y;
                s.T[tb][o][4 * lq + 2][r] = x.z;
                s.T[tb][o][4 * lq + 3][r] = x.w;
            }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kSyrkK; ++kk) {
            const float4 a0 = *reinterpret_cast<const float4 *>(&s.T[tb][0][kk][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4 *>(&s.T[tb][0][kk][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4 *>(&s.T[tb][1][kk][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4 *>(&s.T[tb][1][kk][64 + tx * 4]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float2 bv[4] = {make_float2(b0.x, b0.y), make_float2(b0.z, b0.w), make_float2(b1.x, b1.y),
                                  make_float2(b1.z, b1.w)};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float2 ai = make_float2(av[i], av[i]);
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = __ffma2_rn(ai, bv[j], acc[i][j]);
            }
        }
    }
    // the tile through shared memory (the raw ring is free: every copy has been consumed)
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    float(*Cs)[kSyrkTile] = reinterpret_cast<float(*)[kSyrkTile]>(&s.raw[0][0][0][0]);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int r = i < 4 ? ty * 4 + i : 64 + ty * 4 + i - 4;
        *reinterpret_cast<float4 *>(&Cs[r][tx * 4]) = make_float4(acc[i][0].x, acc[i][0].y, acc[i][1].x, acc[i][1].y);
        *reinterpret_cast<float4 *>(&Cs[r][64 + tx * 4]) = make_float4(acc[i][2].x, acc[i][2].y, acc[i][3].x, acc[i][3].y);
    }
    __syncthreads();
    // 16-byte chunk e = tid + 256 u of the tile: row e / 32, columns 4 (e % 32) .. + 3
    constexpr int kChunks = kSyrkTile * kSyrkTile / 4 / 256;
    float4 cv[kChunks];
#pragma unroll
    for (int u = 0; u < kChunks; ++u) {
        const int e = tid + 256 * u, r = e >> 5, c = 4 * (e & 31);
        cv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i0 + r < m && j0 + c < m) cv[u] = *reinterpret_cast<const float4 *>(C + (i0 + r) * ldc + j0 + c);
    }
#pragma unroll
    for (int u = 0; u < kChunks; ++u) {
        const int e = tid + 256 * u, r = e >> 5, c = 4 * (e & 31);
        if (i0 + r < m && j0 + c < m) {     // m % 4 == 0: a 4-column chunk is all in or all out
            const float4 z = *reinterpret_cast<const float4 *>(&Cs[r][c]);
            float4 v = cv[u];
            v.x -= z.x; v.y -= z.y; v.z -= z.z; v.w -= z.w;
            *reinterpret_cast<float4 *>(C + (i0 + r) * ldc + j0 + c) = v;
        }
    }
}

size_t ldl_factor_scratch_bytes(int64_t n) {
    const auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
    const size_t nn = static_cast<size_t>(n);
    return al(nn * nn * 4) + al(nn * kLdlPanel * 4) + 2 * al(size_t(kLdlPanel) * kLdlPanel * 4);
}

static cudaError_t gemm_k128(const float *A, int64_t lda, const float *B, int64_t ldb, float *C, int64_t ldc,
                             int64_t M, int64_t N, float alpha, float beta, const float *Rinv, float *U2, int64_t ldu2,
                             int epi_d, cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    void (*fn)(const float *, int64_t, const float *, int64_t, float *, int64_t, int64_t, int64_t, float, float,
               const float *, float *, int64_t) =
        epi_d == 8 ? ldl_gemm_k128_kernel<8> : epi_d == 4 ? ldl_gemm_k128_kernel<4> : ldl_gemm_k128_kernel<0>;
    const int smem = static_cast<int>(sizeof(GemmK128Smem));
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(fn), smem);
    if (e != cudaSuccess) return e;
    dim3 grid(static_cast<unsigned>((N + kGemmTile - 1) / kGemmTile), static_cast<unsigned>((M + kGemmTile - 1) / kGemmTile));
    fn<<<grid, 256, smem, st>>>(A, lda, B, ldb, C, ldc, M, N, alpha, beta, Rinv, U2, ldu2);
    count_launch();
    return cudaGetLastError();
}

// C[0:m, 0:m] -= Z Z^T on the upper tiles (Z: m x kLdlPanel, leading dimension ldz).
static cudaError_t syrk_upper(const float *Z, int64_t ldz, float *C, int64_t ldc, int64_t m, cudaStream_t st) {
    if (m <= 0) return cudaSuccess;
    const int nt = static_cast<int>((m + kSyrkTile - 1) / kSyrkTile);
    const int smem = static_cast<int>(sizeof(SyrkSmem));
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(ldl_syrk_kernel), smem);
    if (e != cudaSuccess) return e;
    ldl_syrk_kernel<<<static_cast<unsigned>(nt * (nt + 1) / 2), 256, smem, st>>>(Z, ldz, C, ldc, m, nt);
    count_launch();
    return cudaGetLastError();
}

// The side stream of the factorisation's look-ahead: one per device, created once with the highest
// priority. Calls enqueue
// under a lock and fork/join through events of their own, so concurrent calls only share its order.
static std::mutex g_ldl_side_mu;
static cudaError_t ldl_side_stream(cudaStream_t &out) {
    static cudaStream_t per_device[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!per_device[dev]) {
        // the highest priority: the one-CTA panel takes the first SM slot the trailing GEMM frees
        int lo = 0, hi = 0;
        if ((e = cudaDeviceGetStreamPriorityRange(&lo, &hi)) != cudaSuccess) return e;
        if ((e = cudaStreamCreateWithPriority(&per_device[dev], cudaStreamNonBlocking, hi)) != cudaSuccess) return e;
    }
    out = per_device[dev];
    return cudaSuccess;
}
struct LdlEvents {
    cudaEvent_t fork = nullptr, join = nullptr;
    ~LdlEvents() {
        if (fork) cudaEventDestroy(fork);
        if (join) cudaEventDestroy(join);
    }
};

// Right-looking from the last panel. After a panel, its column block (Y = S_QP M^-T, U_QP) and the
// update of the next panel's columns run first; the next panel's factorisation then runs on a side
// stream while the rest of the Schur update (the leading square) runs on the caller's stream.
cudaError_t launch_ldl_factor(const LdlFactorArgs &a, cudaStream_t st) {
    const int64_t n = a.n;
    const size_t nn = static_cast<size_t>(n);
    const auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
    float *S = a.scratch;
    float *Z = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(S) + al(nn * nn * 4));
    float *W = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(Z) + al(nn * kLdlPanel * 4));
    float *Rinv = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(W) + al(size_t(kLdlPanel) * kLdlPanel * 4));
    void (*panel)(const float *, int64_t, int64_t, int, float *, float *, float *, float *, int32_t *) =
        a.d == 4 ? ldl_panel_kernel<4> : ldl_panel_kernel<8>;
    const int smem = static_cast<int>(sizeof(LdlPanelSmem));
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(panel), smem);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_ldl_side_mu);
    cudaStream_t side;
    if ((e = ldl_side_stream(side)) != cudaSuccess) return e;
    LdlEvents ev;
    if ((e = cudaEventCreateWithFlags(&ev.fork, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&ev.join, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaMemcpyAsync(S, a.H, nn * nn * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(a.U, 0, nn * nn * 4, st)) != cudaSuccess) return e;
    int64_t c1 = n;
    int64_t c0 = c1 > kLdlPanel ? c1 - kLdlPanel : 0;
    panel<<<1, kLdlThreads, smem, st>>>(S, n, c0, static_cast<int>(c1 - c0), a.U, a.D, W, Rinv, a.status);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    bool side_pending = false;
    while (c0 > 0) {
        const int P = static_cast<int>(c1 - c0);
        const int64_t p0 = c0 > kLdlPanel ? c0 - kLdlPanel : 0;
        const int Pn = static_cast<int>(c0 - p0);
        if (side_pending && (e = cudaStreamWaitEvent(st, ev.join, 0)) != cudaSuccess) return e;
        // the factor's column block above the panel, Z = S_QP W^T, and U_QP = Z Rd^-1 (P = kLdlPanel here)
        if ((e = gemm_k128(S + c0, n, W, kLdlPanel, Z, kLdlPanel, c0, P, 1.0f, 0.0f, Rinv, a.U + c0, n, a.d, st)) !=
            cudaSuccess)
            return e;
        // the next panel's columns of S_QQ -= Z Z^T (rows 0 .. c0, columns p0 .. c0)
        if ((e = gemm_k128(Z, kLdlPanel, Z + p0 * kLdlPanel, kLdlPanel, S + p0, n, c0, Pn, -1.0f, 1.0f, nullptr, nullptr,
                           0, 0, st)) != cudaSuccess)
            return e;
        // the next panel on the side stream, after all of the above (it overwrites W and the R_kk^-1)
        if ((e = cudaEventRecord(ev.fork, st)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(side, ev.fork, 0)) != cudaSuccess) return e;
        panel<<<1, kLdlThreads, smem, side>>>(S, n, p0, Pn, a.U, a.D, W, Rinv, a.status);
        count_launch();
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        if ((e = cudaEventRecord(ev.join, side)) != cudaSuccess) return e;
        side_pending = true;
        // the rest of the update, the leading p0 x p0 square (upper tiles), meanwhile
        if ((e = syrk_upper(Z, kLdlPanel, S, n, p0, st)) != cudaSuccess) return e;
        c1 = c0;
        c0 = p0;
    }
    if (side_pending && (e = cudaStreamWaitEvent(st, ev.join, 0)) != cudaSuccess) return e;
    return cudaSuccess;
}

// ================================================================== sweep

constexpr int kSwR = 64;              // rows per CTA
constexpr int kSwC = 256;             // columns per chunk (8 slices of 32)
constexpr int kSwBK = 16;             // rows of U / of the error history per ring stage
constexpr int kSwStages = 4;
constexpr int kSwWarps = 8;           // compute warps; + 1 producer warp
constexpr int kSwThreads = 32 * (kSwWarps + 1);
constexpr int kSwS = 32;              // columns of a rounding slice: warp q rounds slice q
constexpr int kSwSlices = kSwC / kSwS;
constexpr int kSwTLd = kSwC + 4;      // padded row of the target tile (conflict-free 16-byte access)
static_assert(kSwSlices == kSwWarps, "one rounding slice per compute warp");

struct SweepSmem {
    float ring_u[kSwStages][kSwBK][kSwC];    // U[k0 .. k0+15][c0 .. c0+255]
    float ring_e[kSwStages][kSwBK][kSwR];    // E[k0 .. k0+15][64 rows] (history, k-major)
    float W[kSwSlices][kSwR][32];            // the chunk's weights: one 128B-swizzled box per slice
    float T[kSwR][kSwTLd];                   // feedback of the earlier chunks, then targets - weights, then errors
    float A[64], Ainv[64], b[8];
    InvScratch inv;
    double red[kSwWarps];
    uint64_t full[kSwStages], empty[kSwStages], edone, wfull;
};

__device__ __forceinline__ void sweep_bar() {
    asm volatile("bar.sync 1, %0;" ::"r"(32 * kSwWarps) : "memory");
}
// the warps taking part in the errors of slice s: warps s .. 7
__device__ __forceinline__ void slice_bar(int s) {
    asm volatile("bar.sync %0, %1;" ::"r"(2 + s), "r"(32 * (kSwWarps - s)) : "memory");
}
// shared-memory load the compiler must not hoist (keeps the d x d constants out of registers)
__device__ __forceinline__ float lds_nohoist(const float *p) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(smem_u32(p)));
    return v;
}
__device__ __forceinline__ float4 lds4_nohoist(const float *p) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(smem_u32(p)));
    return v;
}
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}
// 16-byte chunk c16 of row r of a 128B-swizzled box (rows of 128 bytes)
__device__ __forceinline__ const float4 *swz128(const float (*box)[32], int r, int c16) {
    return reinterpret_cast<const float4 *>(&box[r][0]) + (c16 ^ (r & 7));
}

struct SweepParams {
    const float *A, *b;
    int64_t m, n;
    uint8_t *packed, *codes;
    float *latent;             // [m][n] latent coordinates of the targets, or null
    float *E;                  // [tiles][n][kSwR] error history
    double *partials;          // [tiles] per-CTA sum of squared errors, or null
    int32_t *status;
};

template <int D>
__global__ void __launch_bounds__(kSwThreads, 1)
ldlq_sweep_kernel(const __grid_constant__ CUtensorMap tmU, const __grid_constant__ CUtensorMap tmE,
                  const __grid_constant__ CUtensorMap tmW, const SweepParams p) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    SweepSmem &s = *reinterpret_cast<SweepSmem *>(align_smem_1024(smem_raw));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t n = p.n, tile = blockIdx.x;
    const int nchunks = static_cast<int>((n + kSwC - 1) / kSwC);
    if (tid == 0) {
        for (int i = 0; i < kSwStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kSwWarps);
        }
        mbar_init(&s.edone, 32 * kSwWarps);
        mbar_init(&s.wfull, 1);
        fence_barrier_init();
    }
    if (tid < D * D) s.A[tid] = s.inv.A[tid] = p.A[tid];
    if (tid < D) s.b[tid] = p.b[tid];
    __syncthreads();

    if (warp == kSwWarps) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            prefetch_tensormap(&tmU);
            prefetch_tensormap(&tmE);
            prefetch_tensormap(&tmW);
            int st = 0;
            uint32_t ph = 0;
            for (int c = 0; c < nchunks; ++c) {
                const int c0 = c * kSwC;
                const int cend = static_cast<int>(n < c0 + kSwC ? n : c0 + kSwC);
                for (int k0 = 0; k0 < cend; k0 += kSwBK) {
                    const bool gemm = k0 < c0;
                    if (k0 == (c0 > 0 ? c0 - kSwC : 0)) {
                        // the previous chunk is done (its errors published, its weights read):
                        // this chunk's weights may replace them
                        if (c > 0 && !mbar_wait(&s.edone, (c - 1) & 1, p.status)) return;
                        const int nbox = (cend - c0 + 31) / 32;
                        mbar_arrive_expect_tx(&s.wfull, nbox * sizeof(s.W[0]));
                        for (int q = 0; q < nbox; ++q)
                            tma_load_2d(&s.W[q][0][0], &tmW, c0 + 32 * q, static_cast<int32_t>(tile * kSwR), &s.wfull);
                    }
                    if (!mbar_wait(&s.empty[st], ph ^ 1, p.status)) return;
                    mbar_arrive_expect_tx(&s.full[st], gemm ? sizeof(s.ring_u[0]) + sizeof(s.ring_e[0]) : sizeof(s.ring_u[0]));
                    tma_load_2d(&s.ring_u[st][0][0], &tmU, c0, k0, &s.full[st]);
                    if (gemm) tma_load_2d(&s.ring_e[st][0][0], &tmE, 0, static_cast<int32_t>(tile * n + k0), &s.full[st]);
                    if (++st == kSwStages) { st = 0; ph ^= 1; }
                }
            }
        }
        return;
    }

    // ---------------------------------------------------------------- compute
    if (warp == 0) invert_warp<D>(s.inv);
    sweep_bar();
    if (tid < D * D) s.Ainv[tid] = s.inv.Ainv[tid];
    if (tid == 0 && s.inv.singular && blockIdx.x == 0) set_status(p.status, LCQ_ERR_SINGULAR);
    sweep_bar();

    // feedback GEMM: warp w computes rows 8w .. 8w+7, lane l columns 4l .. 4l+3 and 128+4l .. 128+4l+3.
    // rounding: warp q owns slice q (columns 32q .. 32q+31) of rows l and l + 32.
    const int q = warp;
    int st = 0;
    uint32_t ph = 0;
    bool ok = true;
    double sq = 0.0;

    for (int c = 0; c < nchunks; ++c) {
        const int c0 = c * kSwC;
        const int cw = static_cast<int>(n - c0 < kSwC ? n - c0 : kSwC);
        const int col0 = c0 + kSwS * q;                // this thread's first column
        // feedback of the earlier chunks: F = E_{<c0} U_{<c0, chunk}, packed fp32 FMAs (two columns each)
        float2 acc[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i][j] = make_float2(0.0f, 0.0f);
        for (int k0 = 0; k0 < c0; k0 += kSwBK) {
            if (ok && !mbar_wait(&s.full[st], ph, p.status)) ok = false;
            if (ok) {
#pragma unroll 4
                for (int kk = 0; kk < kSwBK; ++kk) {
                    const float4 a0 = *reinterpret_cast<const float4 *>(&s.ring_e[st][kk][8 * warp]);
                    const float4 a1 = *reinterpret_cast<const float4 *>(&s.ring_e[st][kk][8 * warp + 4]);
                    const float4 b0 = *reinterpret_cast<const float4 *>(&s.ring_u[st][kk][4 * lane]);
                    const float4 b1 = *reinterpret_cast<const float4 *>(&s.ring_u[st][kk][128 + 4 * lane]);
                    const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
                    const float2 bv[4] = {make_float2(b0.x, b0.y), make_float2(b0.z, b0.w), make_float2(b1.x, b1.y),
                                          make_float2(b1.z, b1.w)};
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const float2 ai = make_float2(av[i], av[i]);
#pragma unroll
                        for (int j = 0; j < 4; ++j) acc[i][j] = __ffma2_rn(ai, bv[j], acc[i][j]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[st]);
            if (++st == kSwStages) { st = 0; ph ^= 1; }
        }
        sweep_bar();                                   // the previous chunk's readers of T are done
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            *reinterpret_cast<float4 *>(&s.T[8 * warp + i][4 * lane]) = make_float4(acc[i][0].x, acc[i][0].y, acc[i][1].x, acc[i][1].y);
            *reinterpret_cast<float4 *>(&s.T[8 * warp + i][128 + 4 * lane]) = make_float4(acc[i][2].x, acc[i][2].y, acc[i][3].x, acc[i][3].y);
        }
        sweep_bar();
        if (ok && !mbar_wait(&s.wfull, c & 1, p.status)) ok = false;
        uint64_t bits[2] = {0ull, 0ull};             // this thread's 32 codes of rows lane, lane + 32
        float csq = 0.0f;
        // the chunk's slices in order: slice s (its 32 rows of U's diagonal block in one or two ring
        // stages) is rounded by warp s in place in T (target - weight -> error); its errors then reach
        // the later slices through U's diagonal block
        for (int sl = 0; sl * kSwS < cw; ++sl) {
            const int span = cw - kSwS * sl < kSwS ? cw - kSwS * sl : kSwS;   // valid columns of the slice
            const int nst = (span + kSwBK - 1) / kSwBK;
            const int stA = st;
            if (ok && !mbar_wait(&s.full[st], ph, p.status)) ok = false;
            if (++st == kSwStages) { st = 0; ph ^= 1; }
            int stB = stA;
            if (nst == 2) {
                stB = st;
                if (ok && !mbar_wait(&s.full[st], ph, p.status)) ok = false;
                if (++st == kSwStages) { st = 0; ph ^= 1; }
            }
            // row i (0 .. 31) of the slice in U's diagonal block
            const auto urow = [&](int i) -> const float * {
                return i < kSwBK ? &s.ring_u[stA][i][0] : &s.ring_u[stB][i - kSwBK][0];
            };
            if (q == sl) {
                // both rows of this lane, group by group; each row of A^{-1} and A is loaded once (16-byte
                // shared-memory loads) for the two rows
                float4 *t4[2] = {reinterpret_cast<float4 *>(&s.T[lane][kSwS * sl]),
                                 reinterpret_cast<float4 *>(&s.T[lane + 32][kSwS * sl])};
                float bb[D];
#pragma unroll
                for (int hh = 0; hh < D / 4; ++hh) {
                    const float4 v = lds4_nohoist(&s.b[4 * hh]);
                    bb[4 * hh] = v.x; bb[4 * hh + 1] = v.y; bb[4 * hh + 2] = v.z; bb[4 * hh + 3] = v.w;
                }
#pragma unroll 1
                for (int j = 0; j < span / D; ++j) {
                    float tb[2][D], w[2][D];
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        const int r = lane + 32 * rr;
#pragma unroll
                        for (int hh = 0; hh < D / 4; ++hh) {
                            const float4 fv = t4[rr][j * (D / 4) + hh];
                            const float4 wv = *swz128(s.W[sl], r, j * (D / 4) + hh);
                            w[rr][4 * hh] = wv.x; w[rr][4 * hh + 1] = wv.y; w[rr][4 * hh + 2] = wv.z; w[rr][4 * hh + 3] = wv.w;
                            tb[rr][4 * hh] = (wv.x + fv.x) - bb[4 * hh];
                            tb[rr][4 * hh + 1] = (wv.y + fv.y) - bb[4 * hh + 1];
                            tb[rr][4 * hh + 2] = (wv.z + fv.z) - bb[4 * hh + 2];
                            tb[rr][4 * hh + 3] = (wv.w + fv.w) - bb[4 * hh + 3];
                        }
                    }
                    // u = A^{-1} (t - b) (written out as it is formed) and z = clip(round(u), 0, 3)
                    uint32_t z[2][D];
#pragma unroll
                    for (int i = 0; i < D; ++i) {
                        float ar[D];
#pragma unroll
                        for (int hh = 0; hh < D / 4; ++hh) {
                            const float4 v = lds4_nohoist(&s.Ainv[i * D + 4 * hh]);
                            ar[4 * hh] = v.x; ar[4 * hh + 1] = v.y; ar[4 * hh + 2] = v.z; ar[4 * hh + 3] = v.w;
                        }
#pragma unroll
                        for (int rr = 0; rr < 2; ++rr) {
                            float v = 0.0f;
#pragma unroll
                            for (int jj = 0; jj < D; ++jj) v = fmaf(ar[jj], tb[rr][jj], v);
                            z[rr][i] = round_clamp3(v);
                            const int64_t grow = tile * kSwR + lane + 32 * rr;
                            if (p.latent && grow < p.m) p.latent[grow * n + col0 + j * D + i] = v;
                        }
                    }
                    // e = w - (A z + b)
                    float e[2][D];
#pragma unroll
                    for (int i = 0; i < D; ++i) {
                        float ar[D];
#pragma unroll
                        for (int hh = 0; hh < D / 4; ++hh) {
                            const float4 v = lds4_nohoist(&s.A[i * D + 4 * hh]);
                            ar[4 * hh] = v.x; ar[4 * hh + 1] = v.y; ar[4 * hh + 2] = v.z; ar[4 * hh + 3] = v.w;
                        }
#pragma unroll
                        for (int rr = 0; rr < 2; ++rr) {
                            float wh = bb[i];
#pragma unroll
                            for (int jj = 0; jj < D; ++jj) wh = fmaf(ar[jj], static_cast<float>(z[rr][jj]), wh);
                            e[rr][i] = w[rr][i] - wh;
                        }
                    }
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        const int64_t grow = tile * kSwR + lane + 32 * rr;
                        uint32_t zb = 0;
#pragma unroll
                        for (int i = 0; i < D; ++i) zb |= z[rr][i] << (2 * i);
                        bits[rr] |= static_cast<uint64_t>(zb) << (2 * j * D);
                        if (grow < p.m) {
#pragma unroll
                            for (int i = 0; i < D; ++i) csq = fmaf(e[rr][i], e[rr][i], csq);
                        }
#pragma unroll
                        for (int hh = 0; hh < D / 4; ++hh)
                            t4[rr][j * (D / 4) + hh] = make_float4(e[rr][4 * hh], e[rr][4 * hh + 1], e[rr][4 * hh + 2], e[rr][4 * hh + 3]);
                    }
                    // later groups of this slice, 16 bytes of the rows at a time (U shared by the two rows)
                    for (int c4 = (j + 1) * (D / 4); c4 < span / 4; ++c4) {
                        float4 v0 = t4[0][c4], v1 = t4[1][c4];
#pragma unroll
                        for (int i = 0; i < D; ++i) {
                            const float4 uv = *reinterpret_cast<const float4 *>(urow(j * D + i) + kSwS * sl + 4 * c4);
                            v0.x = fmaf(e[0][i], uv.x, v0.x); v0.y = fmaf(e[0][i], uv.y, v0.y);
                            v0.z = fmaf(e[0][i], uv.z, v0.z); v0.w = fmaf(e[0][i], uv.w, v0.w);
                            v1.x = fmaf(e[1][i], uv.x, v1.x); v1.y = fmaf(e[1][i], uv.y, v1.y);
                            v1.z = fmaf(e[1][i], uv.z, v1.z); v1.w = fmaf(e[1][i], uv.w, v1.w);
                        }
                        t4[0][c4] = v0;
                        t4[1][c4] = v1;
                    }
                }
            }
            if (sl < kSwSlices - 1 && q >= sl) slice_bar(sl);
            if (q > sl) {
                // T[r][this slice] += e_slice U[slice rows][this thread's columns], both rows per U load, the
                // slice's 32 columns in two halves of 16
#pragma unroll 1
                for (int hc = 0; hc < 2; ++hc) {
                    float2 acc2[2][kSwS / 4];
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        const float4 *own = reinterpret_cast<const float4 *>(&s.T[lane + 32 * rr][kSwS * q + 16 * hc]);
#pragma unroll
                        for (int c4 = 0; c4 < kSwS / 8; ++c4) {
                            const float4 v = own[c4];
                            acc2[rr][2 * c4] = make_float2(v.x, v.y);
                            acc2[rr][2 * c4 + 1] = make_float2(v.z, v.w);
                        }
                    }
#pragma unroll 1
                    for (int i4 = 0; i4 < span / 4; ++i4) {
                        const float4 e0 = reinterpret_cast<const float4 *>(&s.T[lane][kSwS * sl])[i4];
                        const float4 e1 = reinterpret_cast<const float4 *>(&s.T[lane + 32][kSwS * sl])[i4];
                        const float ev0[4] = {e0.x, e0.y, e0.z, e0.w}, ev1[4] = {e1.x, e1.y, e1.z, e1.w};
#pragma unroll
                        for (int ii = 0; ii < 4; ++ii) {
                            const float4 *ur = reinterpret_cast<const float4 *>(urow(4 * i4 + ii) + kSwS * q + 16 * hc);
                            const float2 x0 = make_float2(ev0[ii], ev0[ii]), x1 = make_float2(ev1[ii], ev1[ii]);
#pragma unroll
                            for (int c4 = 0; c4 < kSwS / 8; ++c4) {
                                const float4 uv = ur[c4];
                                const float2 ua = make_float2(uv.x, uv.y), ub = make_float2(uv.z, uv.w);
                                acc2[0][2 * c4] = __ffma2_rn(x0, ua, acc2[0][2 * c4]);
                                acc2[0][2 * c4 + 1] = __ffma2_rn(x0, ub, acc2[0][2 * c4 + 1]);
                                acc2[1][2 * c4] = __ffma2_rn(x1, ua, acc2[1][2 * c4]);
                                acc2[1][2 * c4 + 1] = __ffma2_rn(x1, ub, acc2[1][2 * c4 + 1]);
                            }
                            asm volatile("" ::: "memory");
                        }
                    }
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        float4 *ownw = reinterpret_cast<float4 *>(&s.T[lane + 32 * rr][kSwS * q + 16 * hc]);
#pragma unroll
                        for (int c4 = 0; c4 < kSwS / 8; ++c4)
                            ownw[c4] = make_float4(acc2[rr][2 * c4].x, acc2[rr][2 * c4].y, acc2[rr][2 * c4 + 1].x,
                                                   acc2[rr][2 * c4 + 1].y);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&s.empty[stA]);
                if (nst == 2) mbar_arrive(&s.empty[stB]);
            }
        }
        // this thread's columns: error history (k-major) from T, codes
        if (col0 < n) {
#pragma unroll
            for (int rr = 0; rr < 2; ++rr) {
                const int r = lane + 32 * rr;
                const int64_t grow = tile * kSwR + r;
                float *Eh = p.E + (tile * n + col0) * kSwR + r;
                const float4 *ev = reinterpret_cast<const float4 *>(&s.T[r][kSwS * q]);
#pragma unroll
                for (int c4 = 0; c4 < kSwS / 4; ++c4) {
                    if (col0 + 4 * c4 >= n) break;
                    const float4 v = ev[c4];
                    Eh[(4 * c4 + 0) * kSwR] = v.x;
                    Eh[(4 * c4 + 1) * kSwR] = v.y;
                    Eh[(4 * c4 + 2) * kSwR] = v.z;
                    Eh[(4 * c4 + 3) * kSwR] = v.w;
                }
                if (grow < p.m && p.packed) {
                    uint8_t *pk = p.packed + grow * (n / 4) + col0 / 4;
                    if (col0 + kSwS <= n && (reinterpret_cast<uintptr_t>(pk) & 7u) == 0) {
                        *reinterpret_cast<uint2 *>(pk) =
                            make_uint2(static_cast<uint32_t>(bits[rr]), static_cast<uint32_t>(bits[rr] >> 32));
                    } else {
                        for (int i = 0; i < kSwS && col0 + i < n; i += 4)
                            pk[i / 4] = static_cast<uint8_t>((bits[rr] >> (2 * i)) & 0xFFu);
                    }
                }
                if (grow < p.m && p.codes) {
                    uint8_t *cd = p.codes + grow * n + col0;
                    for (int i = 0; i < kSwS && col0 + i < n; ++i)
                        cd[i] = static_cast<uint8_t>((bits[rr] >> (2 * i)) & 3u);
                }
            }
        }
        sq += static_cast<double>(csq);
        fence_proxy_async_global();
        mbar_arrive(&s.edone);
    }
    if (p.partials) {
        for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        if (lane == 0) s.red[warp] = sq;
        sweep_bar();
        if (tid == 0) {
            double tot = 0.0;
            for (int i = 0; i < kSwWarps; ++i) tot += s.red[i];
            p.partials[blockIdx.x] = tot;
        }
    }
}

// mse = sum of the per-CTA partials (fixed order) / count
__global__ void ldlq_mse_kernel(const double *partials, int nparts, double count, double *mse) {
    __shared__ double red[256];
    double v = 0.0;
    for (int i = threadIdx.x; i < nparts; i += 256) v += partials[i];
    red[threadIdx.x] = v;
    __syncthreads();
    for (int o = 128; o; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) *mse = count > 0.0 ? red[0] / count : 0.0;
}

int64_t ldlq_tiles(int64_t m) { return (m + kSwR - 1) / kSwR; }
size_t ldlq_history_bytes(int64_t m, int64_t n) {
    return static_cast<size_t>(ldlq_tiles(m)) * kSwR * static_cast<size_t>(n) * 4;
}

static bool make_map_f32(CUtensorMap *map, const float *base, uint64_t inner, uint64_t outer, uint64_t ld_elems,
                         uint32_t box_inner, uint32_t box_outer, bool swizzle128 = false) {
    auto enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {ld_elems * 4};
    cuuint32_t box[2] = {box_inner, box_outer}, estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t launch_ldlq(const LdlqArgs &a, cudaStream_t st) {
    const int64_t tiles = ldlq_tiles(a.m);
    CUtensorMap tmU, tmE, tmW;
    if (!make_map_f32(&tmU, a.U, a.n, a.n, a.n, kSwC, kSwBK) ||
        !make_map_f32(&tmE, a.E, kSwR, static_cast<uint64_t>(tiles * a.n), kSwR, kSwR, kSwBK) ||
        !make_map_f32(&tmW, a.W, a.n, a.m, a.n, 32, kSwR, true))
        return cudaErrorInvalidValue;
    SweepParams p{a.A, a.b, a.m, a.n, a.packed, a.codes, a.latent, a.E, a.mse ? a.partials : nullptr, a.status};
    void (*k)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const SweepParams) =
        a.d == 4 ? ldlq_sweep_kernel<4> : ldlq_sweep_kernel<8>;
    const int smem = static_cast<int>(sizeof(SweepSmem)) + 1024;
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), smem);
    if (e != cudaSuccess) return e;
    k<<<static_cast<unsigned>(tiles), kSwThreads, smem, st>>>(tmU, tmE, tmW, p);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (a.mse) {
        ldlq_mse_kernel<<<1, 256, 0, st>>>(a.partials, static_cast<int>(tiles),
                                           static_cast<double>(a.m) * static_cast<double>(a.n), a.mse);
        count_launch();
        e = cudaGetLastError();
    }
    return e;
}

}  // namespace lcq
