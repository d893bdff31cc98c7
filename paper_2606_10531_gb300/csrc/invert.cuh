// A^{-1} of a small (d x d, d <= 8) matrix by one warp, to fp32 accuracy: register Gauss-Jordan
// elimination in fp32, refined by Newton steps whose residual is accumulated in double-float, with
// an fp64 elimination as the fallback for badly conditioned input. Used by the encoders (A^{-1} of
// the codebook map) and by the LDLQ sweep.
//
// The scratch type Smem must provide: float A[64] (input, row-major d x d), float Ainv[64] (output),
// float M[64] (output: A^T A), double gj[8][16], float gjf[8][16] (work), int singular (output).
#pragma once

#include "common.cuh"

namespace lcq {

struct InvScratch {
    float A[64];
    float Ainv[64];
    float M[64];
    double gj[8][16];
    float gjf[8][16];
    int singular;
};

// One warp: A^{-1} by Gauss-Jordan elimination with partial pivoting in fp64, rounded to fp32.
// Sets s.singular if a pivot is (relatively) zero. Slow on this part (fp64 latency), so it is the
// fallback of invert_warp.
template <int D, typename Smem>
__device__ void invert_fp64_warp(Smem &s) {
    const int lane = threadIdx.x & 31;
    double amax = 0.0;
    for (int e = lane; e < D * 2 * D; e += 32) {
        const int r = e / (2 * D), c = e % (2 * D);
        const double v = c < D ? static_cast<double>(s.A[r * D + c]) : (c - D == r ? 1.0 : 0.0);
        s.gj[r][c] = v;
        if (c < D) amax = fmax(amax, fabs(v));
    }
    for (int o = 16; o; o >>= 1) amax = fmax(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    __syncwarp();
    int singular = !(amax > 0.0) || !isfinite(amax);
    for (int c = 0; c < D && !singular; ++c) {
        double best = -1.0;
        int prow = c;
        for (int r = c; r < D; ++r) {
            const double v = fabs(s.gj[r][c]);
            if (v > best) { best = v; prow = r; }
        }
        if (!(best > 1e-12 * amax) || !isfinite(best)) { singular = 1; break; }
        if (prow != c && lane < 2 * D) {
            const double t = s.gj[c][lane];
            s.gj[c][lane] = s.gj[prow][lane];
            s.gj[prow][lane] = t;
        }
        __syncwarp();
        const double piv = s.gj[c][c];
        __syncwarp();
        if (lane < 2 * D) s.gj[c][lane] /= piv;
        __syncwarp();
        double f[4];
        int cnt = 0;
        for (int e = lane; e < D * 2 * D; e += 32, ++cnt) f[cnt] = s.gj[e / (2 * D)][c];
        __syncwarp();
        cnt = 0;
        for (int e = lane; e < D * 2 * D; e += 32, ++cnt) {
            const int r = e / (2 * D), cc = e % (2 * D);
            if (r != c) s.gj[r][cc] -= f[cnt] * s.gj[c][cc];
        }
        __syncwarp();
    }
    for (int e = lane; e < D * D; e += 32) {
        const int r = e / D, c = e % D;
        s.Ainv[e] = singular ? 0.0f : static_cast<float>(s.gj[r][D + c]);
    }
    if (lane == 0) s.singular = singular;
    __syncwarp();
}

// Error-free transformations in fp32: a*b = p + e exactly (FMA), and a + b = s + err exactly (TwoSum).
__device__ __forceinline__ void two_prod(float a, float b, float &p, float &e) {
    p = a * b;
    e = fmaf(a, b, -p);
}
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &err) {
    s = a + b;
    const float bb = s - a;
    err = (a - (s - bb)) + (b - bb);
}

// One warp: A^{-1} and M = A^T A (fp32).
//  1. Gauss-Jordan elimination with partial pivoting in fp32, in registers: lane r + D h (r < D,
//     h < 2D/8) holds columns 8h .. 8h+7 of row r of [A | I]; pivots, row swaps and the pivot row
//     are exchanged with warp shuffles.
//  2. Newton steps X <- X + X R with the residual R = I - A X accumulated in double-float (fp32 pairs:
//     FMA-exact products, TwoSum accumulation): each step squares the residual (I - A X' = R^2) without
//     fp64 arithmetic, which is slow on this part. One step suffices for well-conditioned A.
//  3. If the residual does not reach the acceptance bound within four steps (A badly conditioned, or
//     non-finite), the fp64 elimination runs instead.
// Sets s.singular if a pivot is (relatively) zero.
template <int D, typename Smem>
__device__ void invert_warp(Smem &s) {
    constexpr int H = 2 * D / 8;                 // 8-column blocks of [A | I]
    const int lane = threadIdx.x & 31;
    const int r = lane % D, h = lane / D;
    const bool act = lane < D * H;
    float row[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const int c = 8 * h + j;
        row[j] = !act ? 0.0f : (c < D ? s.A[r * D + c] : (c - D == r ? 1.0f : 0.0f));
    }
    for (int e = lane; e < D * D; e += 32) {
        const int i = e / D, j = e % D;
        float acc = 0.0f;
        for (int k = 0; k < D; ++k) acc = fmaf(s.A[k * D + i], s.A[k * D + j], acc);
        s.M[e] = acc;
    }
    float amax = 0.0f;
#pragma unroll
    for (int j = 0; j < 8; ++j)
        if (8 * h + j < D) amax = fmaxf(amax, fabsf(row[j]));
    for (int o = 16; o; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    int singular = !(amax > 0.0f) || !isfinite(amax);
#pragma unroll
    for (int c = 0; c < D; ++c) {
        if (singular) break;
        // pivot: largest |a[r][c]| over rows r >= c (column c sits in block 0, lane r)
        float v = (act && h == 0 && r >= c) ? fabsf(row[c]) : -1.0f;
        int idx = r;
        for (int o = 16; o; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, v, o);
            const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
            if (ov > v || (ov == v && oi < idx)) { v = ov; idx = oi; }
        }
        if (!(static_cast<double>(v) > 1e-12 * static_cast<double>(amax)) || !isfinite(v)) { singular = 1; break; }
        const int prow = idx;
        // swap rows c and prow, within each column block
        const int src = (r == c) ? prow : (r == prow ? c : r);
#pragma unroll
        for (int j = 0; j < 8; ++j) row[j] = __shfl_sync(0xffffffffu, row[j], src + D * h);
        const float piv = __shfl_sync(0xffffffffu, row[c], c);     // a[c][c], block 0
        const float rinv = 1.0f / piv;
        if (r == c) {
#pragma unroll
            for (int j = 0; j < 8; ++j) row[j] *= rinv;
        }
        const float f = __shfl_sync(0xffffffffu, row[c], r);       // a[r][c] of this lane's row
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float pc = __shfl_sync(0xffffffffu, row[j], c + D * h);   // pivot row, same block
            if (r != c) row[j] = fmaf(-f, pc, row[j]);
        }
    }
    if (singular) {
        for (int e = lane; e < D * D; e += 32) s.Ainv[e] = 0.0f;
        if (lane == 0) s.singular = 1;
        __syncwarp();
        return;
    }
    // X = right half of [I | A^{-1}]
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        const int c = 8 * h + j;
        if (act && c >= D) s.gjf[r][c - D] = row[j];
    }
    __syncwarp();
    // Acceptance: the residual of any fp32-stored inverse has a rounding floor of about
    // cond(A) 2^-24; stop after the update whose residual was within 8x that floor (capped at 1e-4,
    // beyond which the fp64 elimination is used), cond(A) estimated as ||A||_inf ||X||_inf.
    float arow = 0.0f, xrow = 0.0f;
    if (lane < D) {
        for (int k = 0; k < D; ++k) {
            arow += fabsf(s.A[lane * D + k]);
            xrow += fabsf(s.gjf[lane][k]);
        }
    }
    for (int o = 16; o; o >>= 1) {
        arow = fmaxf(arow, __shfl_xor_sync(0xffffffffu, arow, o));
        xrow = fmaxf(xrow, __shfl_xor_sync(0xffffffffu, xrow, o));
    }
    const float accept = fmaxf(1e-6f, fminf(8.0f * arow * xrow * 5.9604645e-8f, 1e-4f));
    bool ok = false;
    for (int pass = 0; pass < 4; ++pass) {
        float res = 0.0f;
        float Rv[2] = {0.0f, 0.0f};
        for (int q = 0; q < 2; ++q) {
            const int e = lane + 32 * q;
            if (e < D * D) {
                const int i = e / D, j = e % D;
                float hi = (i == j) ? 1.0f : 0.0f, lo = 0.0f;
                for (int k = 0; k < D; ++k) {
                    float pp, pe, t, te;
                    two_prod(s.A[i * D + k], s.gjf[k][j], pp, pe);
                    two_sum(hi, -pp, t, te);
                    hi = t;
                    lo += te - pe;
                }
                Rv[q] = hi + lo;
                res = fmaxf(res, fabsf(Rv[q]));
            }
        }
        for (int o = 16; o; o >>= 1) res = fmaxf(res, __shfl_xor_sync(0xffffffffu, res, o));
        if (!(res <= 0.5f)) break;                              // not converging (or non-finite): fall back
        for (int q = 0; q < 2; ++q) {
            const int e = lane + 32 * q;
            if (e < D * D) s.gjf[e / D][D + e % D] = Rv[q];      // R beside X
        }
        __syncwarp();
        float Xn[2] = {0.0f, 0.0f};
        for (int q = 0; q < 2; ++q) {
            const int e = lane + 32 * q;
            if (e < D * D) {
                const int i = e / D, j = e % D;
                float corr = 0.0f;
                for (int k = 0; k < D; ++k) corr = fmaf(s.gjf[i][k], s.gjf[k][D + j], corr);
                Xn[q] = s.gjf[i][j] + corr;
            }
        }
        __syncwarp();
        for (int q = 0; q < 2; ++q) {
            const int e = lane + 32 * q;
            if (e < D * D) s.gjf[e / D][e % D] = Xn[q];
        }
        __syncwarp();
        if (res <= accept) { ok = true; break; }
    }
    if (!ok) {
        invert_fp64_warp<D>(s);
        return;
    }
    for (int e = lane; e < D * D; e += 32) s.Ainv[e] = s.gjf[e / D][e % D];
    if (lane == 0) s.singular = 0;
    __syncwarp();
}

}  // namespace lcq
