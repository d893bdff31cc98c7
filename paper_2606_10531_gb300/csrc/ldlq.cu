// LDLQ initialisation of the codes (Sec. 2.2 adopts LDLQ, QuIP): the column groups of W are
// quantized in order, each group's target being its weights plus the earlier groups' errors fed
// through the block U D U^T factor of the proxy Hessian H:
//
//     H = (U + I) D (U + I)^T,   T_k = W_k + sum_{j<k} (W_j - W_hat_j) U_{j,k},
//     z_k = clip(round(A^{-1}(T_k - b)), 0, 3),   W_hat_k = A z_k + b.
//
// Factorisation (ldl_panel_kernel, ldl_gemm_nt_kernel): right-looking over 128-column panels from
// the last to the first. A panel's diagonal block is factored by one CTA in shared memory; the
// column block above it and the Schur-complement update of the leading matrix are fp32 SIMT GEMMs
// (Y = S_QP M^-T, U_QP = S_QP M^-T D^-1, S_QQ -= Y U_QP^T; upper triangle only, the panel kernel
// mirrors it).
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
constexpr int kLdlLd = kLdlPanel + 1;

struct LdlPanelSmem {
    float S[kLdlPanel][kLdlLd];       // Schur block of the panel (symmetrised); later M^-1
    float Up[kLdlPanel][kLdlLd];      // U of the panel (strictly upper d x d blocks)
    float Dinv[kLdlPanel / 4][64];    // D_k^{-1} per group
    InvScratch inv;
};

// Factor the diagonal block S[c0:c0+P, c0:c0+P] (upper triangle read, mirrored) of the current
// Schur complement: U and D of the panel's groups, eliminated from the last group to the first; then
// M^-1 = (I + U_PP)^-1 by block back substitution, and D^-1 M^-1. Writes U's panel block, D (if
// requested), Minv and Binv (P x P, leading dimension kLdlPanel).
template <int D>
__global__ void __launch_bounds__(kLdlThreads)
ldl_panel_kernel(const float *__restrict__ S, int64_t n, int64_t c0, int P, float *__restrict__ U,
                 float *__restrict__ Dout, float *__restrict__ Minv, float *__restrict__ Binv, int32_t *status) {
    extern __shared__ __align__(16) uint8_t smem_raw[];
    LdlPanelSmem &s = *reinterpret_cast<LdlPanelSmem *>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int G = P / D;
    for (int e = tid; e < P * P; e += kLdlThreads) {
        const int i = e / P, j = e % P;
        const int64_t lo = i <= j ? i : j, hi = i <= j ? j : i;
        s.S[i][j] = S[(c0 + lo) * n + c0 + hi];
        s.Up[i][j] = 0.0f;
    }
    __syncthreads();
    // D_k^{-1} of the last group; then per group k (from the last): U_{<k,k} = S_{<k,k} D_k^{-1}, the
    // next diagonal block D_{k-1} updated first, and its inversion (warp 0) overlapped with the rest of
    // the Schur update S_{<k,<k} -= U_{<k,k} S_{k,<k} (warps 1..). Only the block-upper triangle is
    // kept current (S_{k,<k} is read as S_{<k,k}^T).
    const auto invert_group = [&](int k) {
        const int kd = k * D;
        for (int e = tid; e < D * D; e += 32) s.inv.A[e] = s.S[kd + e / D][kd + e % D];
        __syncwarp();
        invert_warp<D, InvScratch, true>(s.inv);
        for (int e = tid; e < D * D; e += 32) {
            s.Dinv[k][e] = s.inv.Ainv[e];
            if (Dout) Dout[(c0 / D + k) * D * D + e] = s.inv.A[e];
        }
        if (tid == 0 && s.inv.singular) set_status(status, LCQ_ERR_SINGULAR);
    };
    if (warp == 0) invert_group(G - 1);
    __syncthreads();
    for (int k = G - 1; k >= 1; --k) {
        const int kd = k * D, kp = kd - D;
        // U_{<k,k} = S_{<k,k} D_k^{-1}
        for (int e = tid; e < kd * D; e += kLdlThreads) {
            const int i = e / D, j = e % D;
            float acc = 0.0f;
#pragma unroll
            for (int q = 0; q < D; ++q) acc = fmaf(s.S[i][kd + q], s.Dinv[k][q * D + j], acc);
            s.Up[i][kd + j] = acc;
        }
        __syncthreads();
        // the next diagonal block, D_{k-1} -= U_{k-1,k} S_{k,k-1}
        for (int e = tid; e < D * D; e += kLdlThreads) {
            const int i = kp + e / D, j = kp + e % D;
            float acc = s.S[i][j];
#pragma unroll
            for (int q = 0; q < D; ++q) acc = fmaf(-s.Up[i][kd + q], s.S[j][kd + q], acc);
            s.S[i][j] = acc;
        }
        __syncthreads();
        if (warp == 0) {
            invert_group(k - 1);
        } else {
            // the rest of the block-upper triangle of S_{<k,<k}
            for (int e = tid - 32; e < kd * kd; e += kLdlThreads - 32) {
                const int i = e / kd, j = e % kd;
                const int bi = i / D, bj = j / D;
                if (bi > bj || (bi == k - 1 && bj == k - 1)) continue;
                float acc = s.S[i][j];
#pragma unroll
                for (int q = 0; q < D; ++q) acc = fmaf(-s.Up[i][kd + q], s.S[j][kd + q], acc);
                s.S[i][j] = acc;
            }
        }
        __syncthreads();
    }
    // U's panel block (the zero blocks stay as the caller cleared them)
    for (int e = tid; e < P * P; e += kLdlThreads) {
        const int i = e / P, j = e % P;
        if (i / D < j / D) U[(c0 + i) * n + c0 + j] = s.Up[i][j];
    }
    // X = M^-1, M = I + Up unit block-upper triangular: X_k = E_k - sum_{j>k} Up_{k,j} X_j, block rows
    // from the last; X is block-upper triangular too, so X_k[., col] needs the blocks up to col's only
    for (int k = G - 1; k >= 0; --k) {
        const int kd = k * D;
        for (int e = tid; e < D * P; e += kLdlThreads) {
            const int r = kd + e / P, col = e % P;
            float acc;
            if (col < kd + D) {
                acc = (r == col) ? 1.0f : 0.0f;
            } else {
                // four partial sums (the block boundaries are multiples of D >= 4)
                float a4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                const int cend = (col / D + 1) * D;
                for (int c = kd + D; c < cend; c += 4)
#pragma unroll
                    for (int q = 0; q < 4; ++q) a4[q] = fmaf(-s.Up[r][c + q], s.S[c + q][col], a4[q]);
                acc = (a4[0] + a4[1]) + (a4[2] + a4[3]);
            }
            s.S[r][col] = acc;
        }
        __syncthreads();
    }
    for (int e = tid; e < P * P; e += kLdlThreads) {
        const int i = e / P, j = e % P;
        Minv[i * kLdlPanel + j] = s.S[i][j];
        const int k = i / D, r = i % D;
        float acc = 0.0f;
#pragma unroll
        for (int q = 0; q < D; ++q) acc = fmaf(s.Dinv[k][r * D + q], s.S[k * D + q][j], acc);
        Binv[i * kLdlPanel + j] = acc;
    }
}

// C[i][j] = beta C[i][j] + alpha sum_k A[i][k] B[j][k] for i < M, j < N (K a multiple of 16; rows
// of A and B 16-byte aligned). upper: skip the 64 x 64 tiles that lie wholly below the diagonal.
constexpr int kGemmTile = 64, kGemmK = 16, kGemmPad = 68;

__global__ void __launch_bounds__(256)
ldl_gemm_nt_kernel(const float *__restrict__ Am, int64_t lda, const float *__restrict__ Bm, int64_t ldb,
                   float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, int K, float alpha, float beta,
                   int upper) {
    const int64_t i0 = static_cast<int64_t>(blockIdx.y) * kGemmTile, j0 = static_cast<int64_t>(blockIdx.x) * kGemmTile;
    if (upper && i0 > j0 + kGemmTile - 1) return;
    __shared__ __align__(16) float As[kGemmK][kGemmPad];
    __shared__ __align__(16) float Bs[kGemmK][kGemmPad];
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    const int lr = tid >> 2, lk = (tid & 3) * 4;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += kGemmK) {
        float4 va = make_float4(0.f, 0.f, 0.f, 0.f), vb = va;
        if (i0 + lr < M) va = *reinterpret_cast<const float4 *>(Am + (i0 + lr) * lda + k0 + lk);
        if (j0 + lr < N) vb = *reinterpret_cast<const float4 *>(Bm + (j0 + lr) * ldb + k0 + lk);
        As[lk + 0][lr] = va.x; As[lk + 1][lr] = va.y; As[lk + 2][lr] = va.z; As[lk + 3][lr] = va.w;
        Bs[lk + 0][lr] = vb.x; Bs[lk + 1][lr] = vb.y; Bs[lk + 2][lr] = vb.z; Bs[lk + 3][lr] = vb.w;
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kGemmK; ++kk) {
            const float4 a = *reinterpret_cast<const float4 *>(&As[kk][ty * 4]);
            const float4 b = *reinterpret_cast<const float4 *>(&Bs[kk][tx * 4]);
            const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = i0 + ty * 4 + i;
        if (r >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t c = j0 + tx * 4 + j;
            if (c >= N) continue;
            float *p = C + r * ldc + c;
            *p = beta == 0.0f ? alpha * acc[i][j] : fmaf(alpha, acc[i][j], beta * *p);
        }
    }
}

size_t ldl_factor_scratch_bytes(int64_t n) {
    const auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
    const size_t nn = static_cast<size_t>(n);
    return al(nn * nn * 4) + al(nn * kLdlPanel * 4) + 2 * al(size_t(kLdlPanel) * kLdlPanel * 4);
}

static cudaError_t gemm_nt(const float *A, int64_t lda, const float *B, int64_t ldb, float *C, int64_t ldc, int64_t M,
                           int64_t N, int K, float alpha, float beta, bool upper, cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    dim3 grid(static_cast<unsigned>((N + kGemmTile - 1) / kGemmTile), static_cast<unsigned>((M + kGemmTile - 1) / kGemmTile));
    ldl_gemm_nt_kernel<<<grid, 256, 0, st>>>(A, lda, B, ldb, C, ldc, M, N, K, alpha, beta, upper ? 1 : 0);
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
    float *Y = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(S) + al(nn * nn * 4));
    float *Minv = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(Y) + al(nn * kLdlPanel * 4));
    float *Binv = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(Minv) + al(size_t(kLdlPanel) * kLdlPanel * 4));
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
    panel<<<1, kLdlThreads, smem, st>>>(S, n, c0, static_cast<int>(c1 - c0), a.U, a.D, Minv, Binv, a.status);
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    bool side_pending = false;
    while (c0 > 0) {
        const int P = static_cast<int>(c1 - c0);
        const int64_t p0 = c0 > kLdlPanel ? c0 - kLdlPanel : 0;
        const int Pn = static_cast<int>(c0 - p0);
        if (side_pending && (e = cudaStreamWaitEvent(st, ev.join, 0)) != cudaSuccess) return e;
        // Y = S_QP M^-T, U_QP = S_QP (D^-1 M^-1)^T (P = kLdlPanel here)
        if ((e = gemm_nt(S + c0, n, Minv, kLdlPanel, Y, kLdlPanel, c0, P, P, 1.0f, 0.0f, false, st)) != cudaSuccess) return e;
        if ((e = gemm_nt(S + c0, n, Binv, kLdlPanel, a.U + c0, n, c0, P, P, 1.0f, 0.0f, false, st)) != cudaSuccess) return e;
        // the next panel's columns of S_QQ -= Y U_QP^T (rows 0 .. c0, columns p0 .. c0)
        if ((e = gemm_nt(Y, kLdlPanel, a.U + p0 * n + c0, n, S + p0, n, c0, Pn, P, -1.0f, 1.0f, false, st)) != cudaSuccess)
            return e;
        // the next panel on the side stream, after all of the above (it overwrites M^-1, D^-1 M^-1)
        if ((e = cudaEventRecord(ev.fork, st)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(side, ev.fork, 0)) != cudaSuccess) return e;
        panel<<<1, kLdlThreads, smem, side>>>(S, n, p0, Pn, a.U, a.D, Minv, Binv, a.status);
        count_launch();
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        if ((e = cudaEventRecord(ev.join, side)) != cudaSuccess) return e;
        side_pending = true;
        // the rest of the update, the leading p0 x p0 square (upper tiles), meanwhile
        if ((e = gemm_nt(Y, kLdlPanel, a.U + c0, n, S, n, p0, p0, P, -1.0f, 1.0f, true, st)) != cudaSuccess) return e;
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
        uint32_t bits[2][2] = {{0u, 0u}, {0u, 0u}};
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
                    // u = A^{-1} (t - b) and z = clip(round(u), 0, 3)
                    float u[2][D];
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
                            u[rr][i] = v;
                            z[rr][i] = round_clamp3(v);
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
                        if (p.latent && grow < p.m) {
#pragma unroll
                            for (int i = 0; i < D; ++i) p.latent[grow * n + col0 + j * D + i] = u[rr][i];
                        }
                        uint32_t zb = 0;
#pragma unroll
                        for (int i = 0; i < D; ++i) zb |= z[rr][i] << (2 * i);
                        bits[rr][(j * D) >> 4] |= zb << (2 * ((j * D) & 15));
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
                // T[r][this slice] += e_slice U[slice rows][this thread's columns], both rows per U load
                float2 acc2[2][kSwS / 2];
#pragma unroll
                for (int rr = 0; rr < 2; ++rr) {
                    const float4 *own = reinterpret_cast<const float4 *>(&s.T[lane + 32 * rr][kSwS * q]);
#pragma unroll
                    for (int c4 = 0; c4 < kSwS / 4; ++c4) {
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
                        const float4 *ur = reinterpret_cast<const float4 *>(urow(4 * i4 + ii) + kSwS * q);
                        const float2 x0 = make_float2(ev0[ii], ev0[ii]), x1 = make_float2(ev1[ii], ev1[ii]);
#pragma unroll
                        for (int c4 = 0; c4 < kSwS / 4; ++c4) {
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
                    float4 *ownw = reinterpret_cast<float4 *>(&s.T[lane + 32 * rr][kSwS * q]);
#pragma unroll
                    for (int c4 = 0; c4 < kSwS / 4; ++c4)
                        ownw[c4] = make_float4(acc2[rr][2 * c4].x, acc2[rr][2 * c4].y, acc2[rr][2 * c4 + 1].x, acc2[rr][2 * c4 + 1].y);
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
                        *reinterpret_cast<uint2 *>(pk) = make_uint2(bits[rr][0], bits[rr][1]);
                    } else {
                        for (int i = 0; i < kSwS && col0 + i < n; i += 4)
                            pk[i / 4] = static_cast<uint8_t>((bits[rr][i >> 4] >> (2 * (i & 15))) & 0xFFu);
                    }
                }
                if (grow < p.m && p.codes) {
                    uint8_t *cd = p.codes + grow * n + col0;
                    for (int i = 0; i < kSwS && col0 + i < n; ++i)
                        cd[i] = static_cast<uint8_t>((bits[rr][i >> 4] >> (2 * (i & 15))) & 3u);
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
