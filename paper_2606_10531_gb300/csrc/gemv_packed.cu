// Deployment product from packed 2-bit codes through the reformulated forward
// (Sec. 3.2 Eq. def:forward_x):
//
//   Y[t][r] = sum_c X'[t][c] z[r][c] + sum_g X_g[t] . b,     X'_g = X_g A  (per group of d columns)
//
// so the integer codes themselves are the weight operand and A acts on the few activation rows.
//
// prep kernel  (one CTA per token): X' in bf16, written in the column order and scale the
//              main kernel's register fragments expect, and the per-token constant corr[t].
// main kernel  streams the codes once from HBM with 16-byte loads, turns each 32-bit word of 16
//              codes into eight bf16x2 tensor-core fragments with one LOP3 each (no table, no
//              shared memory) and accumulates with mma.sync m16n8k16 (rows of W x tokens).
//
// Code -> bf16 conversion: OR-ing a 2-bit field into the mantissa of bf16 128.0 (0x4300) gives
// the exact value 128 + z * 4^p when the field sits at mantissa bit 2p (p = 0, 1, 2). Word w holds
// code e of its 16 columns at bits 2e; fragment register k (k = 0..7) pairs code k (low half) with
// code k + 8 (high half), read from w, w >> 6 or w >> 12 at field position p_k = {0,1,2,0,1,2,0,1}[k].
// The factor 4^p_k is folded into X' (X'_scaled = X' * 4^-p_k, exact power-of-two scaling) and the
// constant 128 * sum_c X'_scaled[t][c] is removed through corr[t].
#include "common.cuh"
#include "internal.h"

namespace lcq {

constexpr int kGemvRowBlocks = 4;                 // 16-row MMA blocks per warp
constexpr int kGemvRows = 16 * kGemvRowBlocks;    // rows of W per CTA
constexpr int kGemvWarps = 8;                     // K is split over the CTA's warps
constexpr int kSuper = 256;                       // columns per warp step (64 bytes per row)

__host__ __device__ inline int64_t gemv_npad(int64_t n) { return (n + kSuper - 1) / kSuper * kSuper; }

// Field position (power-of-4 scale) of fragment register k.
__device__ __forceinline__ int frag_shift(int k) { return (k % 3 == 2) ? 2 : ((k % 3 == 1) ? 1 : 0); }

template <int D>
__global__ void __launch_bounds__(256)
gemv_prep_kernel(const uint16_t *__restrict__ X, int64_t n, int64_t npad, const float *__restrict__ A,
                 const float *__restrict__ b, uint16_t *__restrict__ Xp, float *__restrict__ corr) {
    __shared__ float red[2][8];
    const int64_t t = blockIdx.x;
    float Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) Am[i] = __ldg(A + i);
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = __ldg(b + i);
    const uint16_t *xrow = X + t * n;
    uint32_t *out = reinterpret_cast<uint32_t *>(Xp + t * npad);
    float S = 0.0f, r = 0.0f;
    for (int64_t blk = threadIdx.x; blk < npad / 16; blk += blockDim.x) {
        float xp[16];
        const int64_t c0 = blk * 16;
        if (c0 + 16 <= n) {
            float x[16];
            const uint4 *src = reinterpret_cast<const uint4 *>(xrow + c0);
            const uint4 u0 = __ldg(src), u1 = __ldg(src + 1);
            const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                x[2 * i] = __uint_as_float(w[i] << 16);
                x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
            }
#pragma unroll
            for (int g = 0; g < 16 / D; ++g) {
#pragma unroll
                for (int k = 0; k < D; ++k) {
                    float acc = 0.0f;
#pragma unroll
                    for (int j = 0; j < D; ++j) acc = fmaf(x[g * D + j], Am[j * D + k], acc);
                    xp[g * D + k] = acc;
                }
#pragma unroll
                for (int j = 0; j < D; ++j) r = fmaf(x[g * D + j], bv[j], r);
            }
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) xp[i] = 0.0f;
            for (int64_t g0 = c0; g0 < n; g0 += D) {
                for (int k = 0; k < D; ++k) {
                    float acc = 0.0f;
                    for (int j = 0; j < D; ++j) {
                        const float xv = __uint_as_float(static_cast<uint32_t>(xrow[g0 + j]) << 16);
                        acc = fmaf(xv, Am[j * D + k], acc);
                    }
                    xp[g0 - c0 + k] = acc;
                }
                for (int j = 0; j < D; ++j)
                    r = fmaf(__uint_as_float(static_cast<uint32_t>(xrow[g0 + j]) << 16), bv[j], r);
            }
        }
        uint32_t words[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float sc = 1.0f / static_cast<float>(1 << (2 * frag_shift(k)));
            const __nv_bfloat16 lo = __float2bfloat16_rn(xp[k] * sc);
            const __nv_bfloat16 hi = __float2bfloat16_rn(xp[k + 8] * sc);
            S += __bfloat162float(lo) + __bfloat162float(hi);
            words[k] = static_cast<uint32_t>(*reinterpret_cast<const uint16_t *>(&lo)) |
                       (static_cast<uint32_t>(*reinterpret_cast<const uint16_t *>(&hi)) << 16);
        }
        uint4 *dst = reinterpret_cast<uint4 *>(out + blk * 8);
        dst[0] = make_uint4(words[0], words[1], words[2], words[3]);
        dst[1] = make_uint4(words[4], words[5], words[6], words[7]);
    }
    for (int o = 16; o; o >>= 1) {
        S += __shfl_xor_sync(0xffffffffu, S, o);
        r += __shfl_xor_sync(0xffffffffu, r, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { red[0][warp] = S; red[1][warp] = r; }
    __syncthreads();
    if (threadIdx.x == 0) {
        float s2 = 0.0f, r2 = 0.0f;
        for (int w = 0; w < static_cast<int>(blockDim.x / 32); ++w) { s2 += red[0][w]; r2 += red[1][w]; }
        corr[t] = r2 - 128.0f * s2;
    }
}

__device__ __forceinline__ uint32_t lop_or_and(uint32_t a, uint32_t mask) {
    // (a & mask) | 0x43004300 in one LOP3
    uint32_t d;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(a), "r"(mask), "r"(0x43004300u));
    return d;
}

__device__ __forceinline__ void codes_to_frags(uint32_t w, uint32_t (&f)[8]) {
    const uint32_t w6 = w >> 6, w12 = w >> 12;
    f[0] = lop_or_and(w, 0x00030003u);
    f[1] = lop_or_and(w, 0x000C000Cu);
    f[2] = lop_or_and(w, 0x00300030u);
    f[3] = lop_or_and(w6, 0x00030003u);
    f[4] = lop_or_and(w6, 0x000C000Cu);
    f[5] = lop_or_and(w6, 0x00300030u);
    f[6] = lop_or_and(w12, 0x00030003u);
    f[7] = lop_or_and(w12, 0x000C000Cu);
}

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <bool VEC>
__device__ __forceinline__ uint4 load_codes(const uint8_t *row_ptr, int64_t byte0, int64_t nbytes) {
    if (VEC && byte0 + 16 <= nbytes) return __ldcs(reinterpret_cast<const uint4 *>(row_ptr + byte0));
    uint32_t w[4] = {0, 0, 0, 0};
    for (int e = 0; e < 16; ++e)
        if (byte0 + e < nbytes) w[e >> 2] |= static_cast<uint32_t>(row_ptr[byte0 + e]) << (8 * (e & 3));
    return make_uint4(w[0], w[1], w[2], w[3]);
}

template <bool VEC>
__global__ void __launch_bounds__(32 * kGemvWarps)
packed_gemv_kernel(const uint8_t *__restrict__ packed, int64_t m, int64_t n, int64_t N, const uint16_t *__restrict__ Xp,
                   int64_t npad, const float *__restrict__ corr, uint16_t *__restrict__ Y) {
    __shared__ float red[kGemvWarps][kGemvRows][17];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, tid = lane & 3;
    const int64_t row0 = static_cast<int64_t>(blockIdx.x) * kGemvRows;
    const int64_t tok0 = static_cast<int64_t>(blockIdx.y) * 16;
    const int ntok = static_cast<int>(N - tok0 < 16 ? N - tok0 : 16);
    const bool two = ntok > 8;
    const int64_t nbytes = n / 4;
    const int64_t nsc = npad / kSuper;

    float acc[kGemvRowBlocks][2][4];
#pragma unroll
    for (int i = 0; i < kGemvRowBlocks; ++i)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[i][nt][e] = 0.0f;

    const uint32_t *xp0 = reinterpret_cast<const uint32_t *>(Xp + (tok0 + g) * npad);
    const uint32_t *xp1 = reinterpret_cast<const uint32_t *>(Xp + (tok0 + g + 8) * npad);
    const bool has0 = g < ntok, has1 = g + 8 < ntok;

    for (int64_t sc = warp; sc < nsc; sc += kGemvWarps) {
        const int64_t byte0 = sc * 64 + 16 * tid;
        uint4 cw[kGemvRowBlocks][2];
#pragma unroll
        for (int i = 0; i < kGemvRowBlocks; ++i)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int64_t row = row0 + 16 * i + g + 8 * hh;
                cw[i][hh] = row < m ? load_codes<VEC>(packed + row * nbytes, byte0, nbytes) : make_uint4(0, 0, 0, 0);
            }
        const int64_t blk0 = sc * 16 + 4 * tid;   // 16-column block of this lane's first word
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint2 bq0[4], bq1[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                bq0[h] = has0 ? __ldg(reinterpret_cast<const uint2 *>(xp0 + (blk0 + q) * 8 + 2 * h)) : make_uint2(0, 0);
                bq1[h] = has1 ? __ldg(reinterpret_cast<const uint2 *>(xp1 + (blk0 + q) * 8 + 2 * h)) : make_uint2(0, 0);
            }
#pragma unroll
            for (int i = 0; i < kGemvRowBlocks; ++i) {
                const uint32_t wlo = q == 0 ? cw[i][0].x : q == 1 ? cw[i][0].y : q == 2 ? cw[i][0].z : cw[i][0].w;
                const uint32_t whi = q == 0 ? cw[i][1].x : q == 1 ? cw[i][1].y : q == 2 ? cw[i][1].z : cw[i][1].w;
                uint32_t flo[8], fhi[8];
                codes_to_frags(wlo, flo);
                codes_to_frags(whi, fhi);
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    mma_bf16_16816(acc[i][0], flo[2 * h], fhi[2 * h], flo[2 * h + 1], fhi[2 * h + 1], bq0[h].x, bq0[h].y);
                    if (two)
                        mma_bf16_16816(acc[i][1], flo[2 * h], fhi[2 * h], flo[2 * h + 1], fhi[2 * h + 1], bq1[h].x,
                                       bq1[h].y);
                }
            }
        }
    }

    // cross-warp (K-split) reduction in a fixed order
#pragma unroll
    for (int i = 0; i < kGemvRowBlocks; ++i)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            red[warp][16 * i + g][nt * 8 + 2 * tid] = acc[i][nt][0];
            red[warp][16 * i + g][nt * 8 + 2 * tid + 1] = acc[i][nt][1];
            red[warp][16 * i + g + 8][nt * 8 + 2 * tid] = acc[i][nt][2];
            red[warp][16 * i + g + 8][nt * 8 + 2 * tid + 1] = acc[i][nt][3];
        }
    __syncthreads();
    for (int o = threadIdx.x; o < kGemvRows * 16; o += blockDim.x) {
        const int rl = o % kGemvRows, tl = o / kGemvRows;
        const int64_t row = row0 + rl;
        if (row >= m || tl >= ntok) continue;
        float s = 0.0f;
#pragma unroll
        for (int w = 0; w < kGemvWarps; ++w) s += red[w][rl][tl];
        s += corr[tok0 + tl];
        const __nv_bfloat16 h = __float2bfloat16_rn(s);
        Y[(tok0 + tl) * m + row] = *reinterpret_cast<const uint16_t *>(&h);
    }
}

size_t packed_gemv_workspace(int64_t N, int64_t n) {
    const size_t xp = static_cast<size_t>(N) * static_cast<size_t>(gemv_npad(n)) * 2;
    const size_t cr = static_cast<size_t>(N) * 4;
    return ((xp + 255) / 256) * 256 + ((cr + 255) / 256) * 256;
}

cudaError_t launch_packed_gemv(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st) {
    (void)num_sms;
    const int64_t npad = gemv_npad(a.n);
    trace_begin(LCQ_K_GEMV_PREP, st);
    if (d == 4) gemv_prep_kernel<4><<<static_cast<unsigned>(a.N), 256, 0, st>>>(a.X, a.n, npad, a.A, a.b, a.Xp, a.corr);
    else gemv_prep_kernel<8><<<static_cast<unsigned>(a.N), 256, 0, st>>>(a.X, a.n, npad, a.A, a.b, a.Xp, a.corr);
    trace_end(LCQ_K_GEMV_PREP, st);
    count_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 grid(static_cast<unsigned>((a.m + kGemvRows - 1) / kGemvRows), static_cast<unsigned>((a.N + 15) / 16));
    const bool vec = (a.n % 64) == 0;
    trace_begin(LCQ_K_GEMV, st);
    if (vec) packed_gemv_kernel<true><<<grid, 32 * kGemvWarps, 0, st>>>(a.packed, a.m, a.n, a.N, a.Xp, npad, a.corr, a.Y);
    else packed_gemv_kernel<false><<<grid, 32 * kGemvWarps, 0, st>>>(a.packed, a.m, a.n, a.N, a.Xp, npad, a.corr, a.Y);
    trace_end(LCQ_K_GEMV, st);
    count_launch();
    return cudaGetLastError();
}

}  // namespace lcq
