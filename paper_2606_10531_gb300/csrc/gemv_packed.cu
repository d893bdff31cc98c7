// Deployment product from packed 2-bit codes through the reformulated forward
// (Sec. 3.2 Eq. def:forward_x):
//
//   Y[t][r] = sum_c X'[t][c] z[r][c] + sum_g X_g[t] . b,     X'_g = X_g A  (per group of d columns)
//
// so the integer codes themselves are the weight operand and A acts on the few activation rows.
// With n % 64 == 0 and n <= 32768, one token takes the dp2a kernel below and 2-16 tokens the tcgen05
// kernel (gemv_fp4.cu); the mma.sync kernels below take every other shape.
//
// prep kernel  (256 16-column blocks per CTA): X' in bf16, written in the column order and scale
//              the main kernel's register fragments expect (tile-major for the tma variant), and
//              per-CTA partials of the per-token constant corr[t].
// main kernel  streams the codes once from HBM, turns each 32-bit word of 16 codes into eight
//              bf16x2 tensor-core fragments with one LOP3 each (no table) and accumulates with
//              mma.sync m16n8k16 (16 rows of W x 8 tokens). The codes operand is converted in
//              registers, so the bandwidth-bound stream never round-trips through a bf16 copy.
//   tma variant (n % 64 == 0): persistent CTAs; one producer thread streams (rows x 512 columns)
//              code tiles, each with the tile's 512 columns of X' (one bulk copy), through a
//              shared-memory ring (2-D TMA copies, 128-byte swizzle, bank-conflict-free fragment
//              reads); each consumer warp owns whole rows of the unit over all columns, so a row's
//              sum stays in registers. Launched with programmatic dependent launch so the code
//              stream starts while the prep kernel still runs; the X' copies wait for it.
//   generic variant: plain 16-byte loads (byte loads at a ragged row end), any n % 8 == 0.
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

constexpr int kGemvRowBlocks = 4;                 // generic variant: 16-row MMA blocks per warp
constexpr int kGemvRows = 16 * kGemvRowBlocks;    // generic variant: rows of W per CTA
constexpr int kGemvWarps = 8;                     // generic variant: K is split over the CTA's warps
constexpr int kSuper = 256;                       // generic variant: columns per warp step
constexpr int kPadCols = 512;                     // X' rows are zero-padded to a multiple of this
constexpr int kPrepCols = 4096;                   // columns per prep CTA (256 threads x 16)
constexpr int kTmaStages = 8;                     // ring stages (at most)
constexpr int kTileCols = 512;                    // 128 bytes of codes per row per stage
constexpr size_t kGemvSmemLimit = 227 * 1024;

__host__ __device__ inline int64_t gemv_npad(int64_t n) { return (n + kPadCols - 1) / kPadCols * kPadCols; }
__host__ __device__ inline int64_t gemv_nprep(int64_t n) { return (gemv_npad(n) + kPrepCols - 1) / kPrepCols; }

// Field position (power-of-4 scale) of fragment register k.
__device__ __forceinline__ int frag_shift(int k) { return (k % 3 == 2) ? 2 : ((k % 3 == 1) ? 1 : 0); }

// The 16 activations of the block starting at column c0 of token row t (zero past n; n % 8 == 0).
// X is bf16 [N][n] (uint16 bit patterns) or, with f32in, fp32 [N][n] (rotated activations).
__device__ __forceinline__ void load_block(const void *__restrict__ Xv, bool f32in, int64_t n, int64_t t, int64_t c0,
                                           float (&x)[16]) {
    if (c0 + 16 <= n) {
        if (f32in) {
            const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(Xv) + t * n + c0);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 f = __ldg(src + q);
                x[4 * q] = f.x; x[4 * q + 1] = f.y; x[4 * q + 2] = f.z; x[4 * q + 3] = f.w;
            }
        } else {
            const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(Xv) + t * n + c0);
            const uint4 u0 = __ldg(src), u1 = __ldg(src + 1);
            const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                x[2 * i] = __uint_as_float(w[i] << 16);
                x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
            }
        }
    } else {
        // ragged end, 8 columns at a time
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const bool in = c0 + 8 * h < n;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int64_t c = c0 + 8 * h + i;
                x[8 * h + i] = !in ? 0.0f
                               : f32in ? static_cast<const float *>(Xv)[t * n + c]
                                       : __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(Xv)[t * n + c]) << 16);
            }
        }
    }
}

// X' = X_g A of one 16-column block (groups of D columns), and the block's share r of sum_g X_g . b.
template <int D>
__device__ __forceinline__ void xform_block(const float (&x)[16], const float (&Am)[D * D], const float (&bv)[D],
                                            float (&xp)[16], float &r) {
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
}

template <int D, bool F32IN>
__device__ __forceinline__ void prep_block(const void *__restrict__ Xv, int64_t n, int64_t t, int64_t c0,
                                           const float (&Am)[D * D], const float (&bv)[D], float (&xp)[16],
                                           float &r) {
    float x[16];
    load_block(Xv, F32IN, n, t, c0, x);
    xform_block<D>(x, Am, bv, xp, r);
}

// Per-CTA sum of v over the 256 threads, written by thread 0 (fixed order).
__device__ __forceinline__ void block_sum_256(float v, float *out) {
    __shared__ float red[8];
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = 0.0f;
        for (int w = 0; w < 8; ++w) s += red[w];
        *out = s;
    }
}

// TILED: X' in the tile-major order of the TMA variant ([npad / 512][N][512], 16-byte chunks of a
// token's tile row permuted as its consumers read them); otherwise [N][npad] in block order.
template <int D, bool F32IN, bool TILED>
__global__ void __launch_bounds__(256)
gemv_prep_kernel(const void *__restrict__ Xv, int64_t n, int64_t npad, const float *__restrict__ A,
                 const float *__restrict__ b, uint16_t *__restrict__ Xp, float *__restrict__ corrpart) {
    // let the dependent main kernel start streaming codes right away (it waits for our results itself)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t t = blockIdx.x;
    float Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) Am[i] = __ldg(A + i);
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = __ldg(b + i);
    float S = 0.0f, r = 0.0f;
    const int64_t blk = static_cast<int64_t>(blockIdx.y) * 256 + threadIdx.x;
    if (blk < npad / 16) {
        float xp[16];
        prep_block<D, F32IN>(Xv, n, t, blk * 16, Am, bv, xp, r);
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
        const uint4 c0 = make_uint4(words[0], words[1], words[2], words[3]);
        const uint4 c1 = make_uint4(words[4], words[5], words[6], words[7]);
        if (TILED) {
            // block bi of tile kc: chunks 2 (bi % 8) and 2 (bi % 8) + 1 of lane group bi / 8
            const int64_t kc = blk / 32;
            const int bi = static_cast<int>(blk % 32), q4 = bi / 8;
            const int sig = (2 * q4 + static_cast<int>(t & 1)) & 7;
            uint4 *row = reinterpret_cast<uint4 *>(Xp + (kc * gridDim.x + t) * kTileCols);
            row[16 * q4 + ((2 * (bi % 8)) ^ sig)] = c0;
            row[16 * q4 + ((2 * (bi % 8) + 1) ^ sig)] = c1;
        } else {
            uint4 *dst = reinterpret_cast<uint4 *>(Xp + t * npad) + blk * 2;
            dst[0] = c0;
            dst[1] = c1;
        }
    }
    block_sum_256(r - 128.0f * S, corrpart + t * gridDim.y + blockIdx.y);
}

// corr[t] = sum of the prep CTAs' partials, in a fixed order.
__device__ __forceinline__ float token_corr(const float *corrpart, int64_t t, int64_t nprep) {
    float s = 0.0f;
    for (int64_t c = 0; c < nprep; ++c) s += corrpart[t * nprep + c];
    return s;
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
    // not volatile: a pure function of its operands, so independent accumulator chains can be interleaved
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
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
                   int64_t npad, const float *__restrict__ corrpart, int64_t nprep, uint16_t *__restrict__ Y) {
    __shared__ float red[kGemvWarps][kGemvRows][17];
    asm volatile("griddepcontrol.wait;" ::: "memory");
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

    const bool has0 = g < ntok, has1 = g + 8 < ntok;
    const uint32_t *xp0 = reinterpret_cast<const uint32_t *>(Xp + (tok0 + (has0 ? g : 0)) * npad);
    const uint32_t *xp1 = reinterpret_cast<const uint32_t *>(Xp + (tok0 + (has1 ? g + 8 : 0)) * npad);

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
        s += token_corr(corrpart, tok0 + tl, nprep);
        const __nv_bfloat16 h = __float2bfloat16_rn(s);
        Y[(tok0 + tl) * m + row] = *reinterpret_cast<const uint16_t *>(&h);
    }
}

// ------------------------------------------------------------------ TMA-streamed variant
//
// Persistent CTAs. One producer thread streams each (R rows x 512 columns) code tile (2-D TMA copy,
// 128-byte swizzle) together with the matching 512 columns of X' of the launch's tokens (one bulk
// copy) through a shared-memory ring. Consumer warp w owns RBW 16-row blocks of every tile, over all
// 512 columns, so a row's sum stays in one warp's registers (with KS = 2 two warps split the tiles of
// a unit by parity and add their sums once per unit).
//
// Fragment reads. Lane (g, q4) (g = lane / 4, q4 = lane % 4) reads the 16-byte chunks 2 q4 and
// 2 q4 + 1 of its rows g and g + 8 of a block: a chunk holds four 16-column code words, and word v of
// chunk c supplies the lane's A fragments of four MMAs (16 columns x 16 rows each). The swizzle puts
// chunk c of row r at c ^ (r % 8), so a quarter-warp's eight 16-byte reads hit eight distinct bank
// groups. X' of a tile is stored per token as 64 chunks of 16 bytes; lane (g, q4) reads token g's
// chunks [16 q4, 16 q4 + 16) (the activations of its own 128 columns, in word order), each at
// position 16 q4 + (i ^ ((2 q4 + g % 2) % 8)) so that those reads are conflict-free as well; the prep
// kernel writes X' in exactly this order.
//
// Two accumulators per (row block, token tile) alternate over the four MMAs of a word, which halves
// the dependent-MMA chains a warp waits on.


struct GemvTmaParams {
    int64_t m, ntok_all, npad, nprep;
    int ntok, t0, units, nkc, stages;
    const uint16_t *Xp;       // tile-major X': [npad / 512][ntok_all][512]
    const float *corrpart;    // [ntok][nprep] (token t0 of this launch)
    uint16_t *Y;              // [ntok][m] (token t0 of this launch)
    int32_t *status;
};

// Shared-memory layout (offsets from the 1024-byte aligned base): code ring, X' ring, KS = 2
// exchange buffer, barriers.
struct GemvTmaLayout {
    size_t acts, red, bars, total;
};
__host__ __device__ inline GemvTmaLayout gemv_tma_layout(int R, int stages, int nt, int cwr, int rbw, int ks) {
    GemvTmaLayout L;
    L.acts = static_cast<size_t>(stages) * static_cast<size_t>(R) * 128;
    L.red = L.acts + static_cast<size_t>(stages) * static_cast<size_t>(8 * nt) * 1024;
    L.bars = L.red + (ks > 1 ? static_cast<size_t>(cwr) * 32 * static_cast<size_t>(rbw * nt * 8) * 4 : 0);
    L.total = L.bars + 2 * kTmaStages * 8;
    return L;
}

// Named-barrier arrival that also tells whether any participating thread had pred set.
__device__ __forceinline__ bool bar_any(int id, int count, bool pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(count)
        : "memory");
    return r != 0;
}

// NT: 8-token MMA tiles (1: <= 8 tokens, 2: <= 16). CWR: consumer warps per K phase; RBW: 16-row
// blocks per warp; KS: K phases (tiles of a unit split by kc % KS). Unit rows R = CWR * 16 * RBW.
template <int NT, int CWR, int RBW, int KS>
__global__ void __launch_bounds__(32 * (CWR * KS + 1), 1)
packed_gemv_tma_kernel(const __grid_constant__ CUtensorMap tmC, const GemvTmaParams p) {
    constexpr int CW = CWR * KS;
    constexpr int R = CWR * 16 * RBW;
    constexpr uint32_t kCodeBytes = static_cast<uint32_t>(R) * 128u;
    constexpr uint32_t kActStride = 8u * NT * 1024u;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *base = align_smem_1024(smem_raw);
    const GemvTmaLayout L = gemv_tma_layout(R, p.stages, NT, CWR, RBW, KS);
    uint8_t *acts = base + L.acts;
    float *red = reinterpret_cast<float *>(base + L.red);
    uint64_t *full = reinterpret_cast<uint64_t *>(base + L.bars);
    uint64_t *empty = full + kTmaStages;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t act_bytes = static_cast<uint32_t>(p.ntok) * 1024u;
    const int my_units = p.units > static_cast<int>(blockIdx.x)
                             ? (p.units - 1 - static_cast<int>(blockIdx.x)) / static_cast<int>(gridDim.x) + 1
                             : 0;
    const int tiles = my_units * p.nkc;
    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmC);
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], CWR);
        }
        fence_barrier_init();
    }
    __syncthreads();

    if (warp == 0) {
        // ---------------------------------------------------------------- producer
        if (lane == 0) {
            auto tile_at = [&](int T, int &u, int &kc) {
                u = static_cast<int>(blockIdx.x) + (T / p.nkc) * static_cast<int>(gridDim.x);
                kc = T % p.nkc;
            };
            auto act_src = [&](int kc) {
                return p.Xp + (static_cast<int64_t>(kc) * p.ntok_all + p.t0) * kTileCols;
            };
            // The code tiles of the first stages go out before X' exists (the prep kernel may still
            // be running); their X' copies follow once it has completed.
            const int P = tiles < p.stages ? tiles : p.stages;
            for (int T = 0; T < P; ++T) {
                int u, kc;
                tile_at(T, u, kc);
                mbar_arrive_expect_tx(&full[T], kCodeBytes + act_bytes);
                tma_load_2d(base + static_cast<size_t>(T) * kCodeBytes, &tmC, kc * 128, u * R, &full[T]);
            }
            asm volatile("griddepcontrol.wait;" ::: "memory");
            for (int T = 0; T < P; ++T) {
                int u, kc;
                tile_at(T, u, kc);
                bulk_g2s(acts + static_cast<size_t>(T) * kActStride, act_src(kc), act_bytes, &full[T]);
            }
            int st = P % p.stages;
            uint32_t ph = P == p.stages ? 1u : 0u;
            for (int T = P; T < tiles; ++T) {
                int u, kc;
                tile_at(T, u, kc);
                if (!mbar_wait(&empty[st], ph ^ 1, p.status)) return;
                mbar_arrive_expect_tx(&full[st], kCodeBytes + act_bytes);
                tma_load_2d(base + static_cast<size_t>(st) * kCodeBytes, &tmC, kc * 128, u * R, &full[st]);
                bulk_g2s(acts + static_cast<size_t>(st) * kActStride, act_src(kc), act_bytes, &full[st]);
                if (++st == p.stages) { st = 0; ph ^= 1; }
            }
        }
        return;
    }

    // -------------------------------------------------------------------- consumers
    asm volatile("griddepcontrol.wait;" ::: "memory");   // corr partials of the prep kernel
    const int cwarp = warp - 1;
    const int rg = cwarp % CWR, ks = cwarp / CWR;
    const int g = lane >> 2, q4 = lane & 3;
    // X' rows of the tile's unused token slots are zero in every stage (the copies never write them),
    // so the lanes of those tokens read zero fragments without a select
    {
        const int zrows = 8 * NT - p.ntok;
        for (int o = threadIdx.x - 32; o < p.stages * zrows * 64; o += 32 * CW) {
            const int s_ = o / (zrows * 64), rem = o % (zrows * 64);
            reinterpret_cast<uint4 *>(acts + static_cast<size_t>(s_) * kActStride +
                                      static_cast<size_t>(p.ntok + rem / 64) * 1024)[rem % 64] = make_uint4(0, 0, 0, 0);
        }
        asm volatile("bar.sync 1, %0;" ::"r"(32 * CW) : "memory");
    }
    float corr[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int t = 8 * nt + 2 * q4 + e;
            corr[nt][e] = t < p.ntok ? token_corr(p.corrpart, t, p.nprep) : 0.0f;
        }
    }
    // byte offsets inside a stage: this lane's first code chunk (row g of its first block) and its
    // X' chunks (token g); the chunk index i of X' is stored at i ^ sig
    const uint32_t code_off = static_cast<uint32_t>((rg * RBW * 16 + g) * 128);
    const uint32_t act_off = static_cast<uint32_t>(g * 1024 + q4 * 256);
    const uint32_t sig = static_cast<uint32_t>((2 * q4 + (g & 1)) & 7);

    int st = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int ul = 0; ul < my_units && ok; ++ul) {
        const int u = static_cast<int>(blockIdx.x) + ul * static_cast<int>(gridDim.x);
        float acc[RBW][NT][2][4];
#pragma unroll
        for (int i = 0; i < RBW; ++i)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int a = 0; a < 2; ++a)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[i][nt][a][e] = 0.0f;

        for (int kc = 0; kc < p.nkc; ++kc) {
            if (KS == 1 || kc % KS == ks) {
                if (!mbar_wait(&full[st], ph, p.status)) { ok = false; break; }
                const uint8_t *ctile = base + static_cast<size_t>(st) * kCodeBytes + code_off;
                const uint8_t *atile = acts + static_cast<size_t>(st) * kActStride + act_off;
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    const uint32_t cchunk = static_cast<uint32_t>(((2 * q4 + j) ^ g) << 4);
                    uint4 cw[RBW][2];
#pragma unroll
                    for (int i = 0; i < RBW; ++i)
#pragma unroll
                        for (int r8 = 0; r8 < 2; ++r8)
                            cw[i][r8] = *reinterpret_cast<const uint4 *>(ctile + (i * 16 + 8 * r8) * 128 + cchunk);
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        uint4 bx[NT][2];
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                            for (int hf = 0; hf < 2; ++hf) {
                                const uint32_t ci = static_cast<uint32_t>(8 * j) + ((static_cast<uint32_t>(2 * v + hf)) ^ sig);
                                bx[nt][hf] = *reinterpret_cast<const uint4 *>(atile + nt * 8 * 1024 + ci * 16);
                            }
                        // all blocks' fragments first, then the MMAs with the blocks innermost, so
                        // consecutive MMAs are independent
                        uint32_t f0[RBW][8], f8[RBW][8];
#pragma unroll
                        for (int i = 0; i < RBW; ++i) {
                            const uint32_t w0 = v == 0 ? cw[i][0].x : v == 1 ? cw[i][0].y : v == 2 ? cw[i][0].z : cw[i][0].w;
                            const uint32_t w8 = v == 0 ? cw[i][1].x : v == 1 ? cw[i][1].y : v == 2 ? cw[i][1].z : cw[i][1].w;
                            codes_to_frags(w0, f0[i]);
                            codes_to_frags(w8, f8[i]);
                        }
#pragma unroll
                        for (int h = 0; h < 4; ++h)
#pragma unroll
                            for (int i = 0; i < RBW; ++i)
#pragma unroll
                                for (int nt = 0; nt < NT; ++nt) {
                                    const uint4 &b = bx[nt][h >> 1];
                                    const uint32_t b0 = (h & 1) ? b.z : b.x, b1 = (h & 1) ? b.w : b.y;
                                    mma_bf16_16816(acc[i][nt][h & 1], f0[i][2 * h], f8[i][2 * h], f0[i][2 * h + 1],
                                                   f8[i][2 * h + 1], b0, b1);
                                }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[st]);
            }
            if (++st == p.stages) { st = 0; ph ^= 1; }
        }
        if (KS == 1 && !ok) break;
        // sum of the two accumulators; with KS = 2 the second phase's warps hand theirs over
#pragma unroll
        for (int i = 0; i < RBW; ++i)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[i][nt][0][e] += acc[i][nt][1][e];
        if (KS > 1) {
            float *mine = red + static_cast<size_t>(rg) * 32 * (RBW * NT * 4) + lane;
            if (ks == 1 && ok) {
#pragma unroll
                for (int i = 0; i < RBW; ++i)
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int e = 0; e < 4; ++e) mine[32 * ((i * NT + nt) * 4 + e)] = acc[i][nt][0][e];
            }
            // every consumer warp reaches both barriers of a unit, also after a failed wait, and
            // all of them leave together if any wait failed
            const bool failed = bar_any(1, 32 * CW, !ok);
            if (ks == 0 && !failed) {
#pragma unroll
                for (int i = 0; i < RBW; ++i)
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                        for (int e = 0; e < 4; ++e) acc[i][nt][0][e] += mine[32 * ((i * NT + nt) * 4 + e)];
            }
            asm volatile("bar.sync 1, %0;" ::"r"(32 * CW) : "memory");
            if (failed) break;
            if (ks != 0) continue;
        }
        const int64_t row0 = static_cast<int64_t>(u) * R + (rg * RBW) * 16 + g;
#pragma unroll
        for (int i = 0; i < RBW; ++i)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int64_t row = row0 + 16 * i + 8 * (e >> 1);
                    const int t = 8 * nt + 2 * q4 + (e & 1);
                    if (row < p.m && t < p.ntok) {
                        const __nv_bfloat16 hv = __float2bfloat16_rn(acc[i][nt][0][e] + corr[nt][e & 1]);
                        p.Y[static_cast<int64_t>(t) * p.m + row] = *reinterpret_cast<const uint16_t *>(&hv);
                    }
                }
    }
}

// ------------------------------------------------------------------ integer (dp2a) variant, one token
//
// With one token a tensor-core MMA spends most of its width on padding, and the fragment conversion
// costs more than the product. This variant works on the CUDA cores instead: a code word of 16
// columns is split into four byte-spread words with one shift and four ANDs,
//   s0 = w & 0x03030303 (columns 0,4,8,12)       s1 = w & 0x0C0C0C0C (columns 1,5,9,13, times 4)
//   s2 = (w >> 4) & 0x03030303 (columns 2,6,...)  s3 = (w >> 4) & 0x0C0C0C0C (columns 3,7,..., times 4)
// and each dp2a multiplies two of those bytes with two int16 activations (exact int32 sums).
//
// Activations: the consumer warps compute X' = X_g A themselves (no separate prep kernel) and store
// it in shared memory as int16 with one scale for the token, s = max|X| * max_k sum_j |A[j][k]| /
// 32767, a bound on max|X'| known before X' is formed. Column c of a 16-column block holds
// round(X'[c] / s) for c % 4 in {0, 2} and round(X'[c] / (4 s)) for c % 4 in {1, 3} (those codes
// arrive multiplied by 4). The eight 32-bit words of a block hold the column pairs (0,4) (8,12)
// (1,5) (9,13) (2,6) (10,14) (3,7) (11,15), the pairs one dp2a multiplies with bytes (0,1) or (2,3)
// of a spread code word; a 512-column tile stores the first halves of its 32 blocks, then the second
// halves (conflict-free 16-byte reads).
//
// Codes: one producer thread streams (R rows x 512 columns) tiles through a TMA ring (128-byte
// swizzle). Lane l owns code word l (16 columns) of rows warp + CW j (CW consumer warps), so a warp
// reads one whole 128-byte row per load, and the lane's position in a swizzled row is the same for
// all its rows (CW is a multiple of 8). The int32 sums run over the whole unit and are added over the
// 32 lanes of a row with exact integer warp reductions (two accumulators, each over half the row's
// columns: below 2^31 for n <= 32768), then scaled once.
//
// Launched with programmatic dependent launch: the code stream starts while the previous kernel in
// the stream finishes; the consumers wait for it (griddepcontrol.wait) before reading X.

constexpr int kFp4MinTokens = 1;          // the tcgen05 fp4 kernel takes more tokens than this
constexpr int kDpMaxTokens = 1;            // two tokens measured slower than the tensor-core kernel
constexpr int kDpWarps = 16;               // consumer warps (a multiple of 8)
constexpr int64_t kDpMaxN = 32768;         // integer row sums stay below 2^31
constexpr int kDpPrefill = 2;              // ring stages filled before the activations are loaded
constexpr size_t kDpSmemLimit = 227 * 1024;

struct GemvDpParams {
    const void *X;            // [n] bf16 bit patterns, or fp32 when f32in
    const float *A, *b;
    int64_t m, n;
    int d, f32in;
    int hb;                   // > 0: rotate X by the block Walsh-Hadamard transform of this block size first
    int R, units, nkc, stages;
    uint16_t *Y;              // [m]
    int32_t *status;
};

// Shared-memory layout of the dp kernel (offsets from the 1024-byte aligned base).
struct DpSmemLayout {
    size_t xq, red, ab, bars, total;
};
__host__ __device__ inline DpSmemLayout dp_smem_layout(int R, int stages, int nkc) {
    DpSmemLayout L;
    L.xq = static_cast<size_t>(stages) * static_cast<size_t>(R) * 128;
    L.red = L.xq + static_cast<size_t>(nkc) * 1024;
    L.ab = L.red + 2 * kDpWarps * 4;                                 // per-warp max|X| and sum X_g . b
    L.bars = (L.ab + (64 + 8 + 1) * 4 + 15) / 16 * 16;               // A (d x d), b (d), max_k sum_j |A|
    L.total = L.bars + (2 * kTmaStages + 1) * 8;    // full[], empty[], xready
    return L;
}

// acc += the two int16 halves of a times bytes 0, 1 (lo) or 2, 3 (hi) of b, accumulated in place
__device__ __forceinline__ void dp2a_lo(uint32_t a, uint32_t b, int32_t &acc) {
    asm("dp2a.lo.s32.u32 %0, %1, %2, %0;" : "+r"(acc) : "r"(a), "r"(b));
}
__device__ __forceinline__ void dp2a_hi(uint32_t a, uint32_t b, int32_t &acc) {
    asm("dp2a.hi.s32.u32 %0, %1, %2, %0;" : "+r"(acc) : "r"(a), "r"(b));
}

// acc0/acc1 += the 16 columns of code word w times one 16-column block (two uint4) of activations.
__device__ __forceinline__ void dp_word(uint32_t w, const uint4 &xa, const uint4 &xb, int32_t &acc0, int32_t &acc1) {
    const uint32_t w4 = w >> 4;
    const uint32_t s0 = w & 0x03030303u, s1 = w & 0x0C0C0C0Cu, s2 = w4 & 0x03030303u, s3 = w4 & 0x0C0C0C0Cu;
    dp2a_lo(xa.x, s0, acc0);
    dp2a_hi(xa.y, s0, acc1);
    dp2a_lo(xa.z, s1, acc0);
    dp2a_hi(xa.w, s1, acc1);
    dp2a_lo(xb.x, s2, acc0);
    dp2a_hi(xb.y, s2, acc1);
    dp2a_lo(xb.z, s3, acc0);
    dp2a_hi(xb.w, s3, acc1);
}

// int16 activations of one 16-column block (lane l of tile `tile`): X' = X_g A, scaled by inv
// (times 1/4 for columns c % 4 in {1, 3}), stored in the pair order of dp_word. Returns the block's
// share of sum_g X_g . b added to r.
template <int D>
__device__ __forceinline__ void dp_quantize(const float (&x)[16], const float *ab_s, uint8_t *xq_s, float inv, int tile,
                                            int lane, float &r) {
    // X'_g = X_g A, one row of A (16-byte loads from shared memory) at a time, so that the loads of
    // the next row overlap the FMAs of this one; the rows j < D/2 and j >= D/2 accumulate separately
    // (half-length dependency chains), added at the end
    float xp[16], xq[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) xp[i] = xq[i] = 0.0f;
    float r2 = 0.0f;
#pragma unroll
    for (int j = 0; j < D; ++j) {
        float (&acc)[16] = j < D / 2 ? xp : xq;
        float &racc = j < D / 2 ? r : r2;
        float arow[D];
#pragma unroll
        for (int h = 0; h < D / 4; ++h) {
            const float4 v = reinterpret_cast<const float4 *>(ab_s + j * D)[h];
            arow[4 * h] = v.x; arow[4 * h + 1] = v.y; arow[4 * h + 2] = v.z; arow[4 * h + 3] = v.w;
        }
        const float bj = ab_s[D * D + j];
#pragma unroll
        for (int g = 0; g < 16 / D; ++g) {
            const float xj = x[g * D + j];
            const float2 xx = make_float2(xj, xj);
#pragma unroll
            for (int k = 0; k < D; k += 2) {
                const float2 v = __ffma2_rn(xx, make_float2(arow[k], arow[k + 1]), make_float2(acc[g * D + k], acc[g * D + k + 1]));
                acc[g * D + k] = v.x;
                acc[g * D + k + 1] = v.y;
            }
            racc = fmaf(xj, bj, racc);
        }
    }
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
        const float2 v = __fadd2_rn(make_float2(xp[i], xp[i + 1]), make_float2(xq[i], xq[i + 1]));
        xp[i] = v.x;
        xp[i + 1] = v.y;
    }
    r += r2;
    // round to int16: v + 1.5 * 2^23 holds round(v) (ties to even) in its low mantissa bits for
    // |v| < 2^22, so the low 16 bits are the two's-complement int16. |v| <= 32767 (1 + 16 * 2^-24) for
    // finite X: |X'| <= max|X| max_k sum_j |A_jk| up to the FMA rounding, and inv is that bound's
    // 32767 / bound to 2 ulp, so round(v) stays in [-32767, 32767] without a clamp
    constexpr int kFirst[8] = {0, 8, 1, 9, 2, 10, 3, 11};
    constexpr float kMagic = 12582912.0f;
    uint32_t words[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int cc = kFirst[k];
        const float f = (cc & 1) ? 0.25f * inv : inv;
        const float lo = fmaf(xp[cc], f, kMagic);
        const float hi = fmaf(xp[cc + 4], f, kMagic);
        words[k] = __byte_perm(__float_as_uint(lo), __float_as_uint(hi), 0x5410);
    }
    uint4 *dst = reinterpret_cast<uint4 *>(xq_s + static_cast<size_t>(tile) * 1024);
    dst[lane] = make_uint4(words[0], words[1], words[2], words[3]);
    dst[32 + lane] = make_uint4(words[4], words[5], words[6], words[7]);
}

__device__ __forceinline__ float absmax16(const float (&x)[16], float mx) {
#pragma unroll
    for (int i = 0; i < 16; ++i) mx = fmaxf(mx, fabsf(x[i]));
    return mx;
}

// Block Walsh-Hadamard rotation of the token in the prologue (Sec. 3.3 rotated deployment), for
// n = 32 * 16 * kDpWarps: consumer thread t holds columns 16 t .. 16 t + 15, so the bits of a column
// index are (warp, lane, register). H_B factors over the index bits (one (u, v) -> (u + v, u - v)
// stage per bit below log2 B): the 4 register bits in registers, the 5 lane bits by warp shuffles, the
// warp bits after one exchange through shared memory (thread t then holds columns t + 512 w, w = 0..15)
// and one back. Unnormalised; the caller scales by 1 / sqrt(B).
__device__ __forceinline__ void wht_reg16(float (&x)[16], int step0, int hb) {
    // butterflies over the register index for element strides step0 * {1, 2, 4, 8} below hb
#pragma unroll
    for (int r = 1; r < 16; r *= 2) {
        if (step0 * r >= hb) break;
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if ((i & r) == 0) {
                const float u = x[i], v = x[i + r];
                x[i] = u + v;
                x[i + r] = u - v;
            }
    }
}
__device__ __forceinline__ void wht_lanes(float (&x)[16], int lane, int hb) {
#pragma unroll
    for (int s = 1; s < 32; s *= 2) {
        if (16 * s >= hb) break;
        const bool upper = (lane & s) != 0;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float v = __shfl_xor_sync(0xffffffffu, x[i], s);
            x[i] = upper ? v - x[i] : x[i] + v;
        }
    }
}

// RPT: rows per thread per tile (a unit has R = kDpWarps * RPT rows).
template <int RPT>
__global__ void __launch_bounds__(32 * (kDpWarps + 1), 1)
packed_gemv_dp_kernel(const __grid_constant__ CUtensorMap tmC, const GemvDpParams p) {
    constexpr int CW = kDpWarps;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *base = align_smem_1024(smem_raw);
    const DpSmemLayout L = dp_smem_layout(p.R, p.stages, p.nkc);
    float *red_s = reinterpret_cast<float *>(base + L.red);   // [2][CW]: max|X|, then sum X_g . b
    float *ab_s = reinterpret_cast<float *>(base + L.ab);
    uint64_t *full = reinterpret_cast<uint64_t *>(base + L.bars);
    uint64_t *empty = full + kTmaStages;
    uint64_t *xready = empty + kTmaStages;    // the consumers have loaded X
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t stage_bytes = static_cast<uint32_t>(p.R) * 128u;
    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmC);
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], CW);
        }
        mbar_init(xready, 1);
        fence_barrier_init();
    }
    __syncthreads();
    // the next kernel in the stream may start launching; it waits for our completion before it
    // reads anything we write
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp == 0) {
        // ---------------------------------------------------------------- producer: code tiles -> ring
        if (lane == 0) {
            int st = 0;
            uint32_t ph = 0;
            for (int u = blockIdx.x; u < p.units; u += gridDim.x) {
                for (int kc = 0; kc < p.nkc; ++kc) {
                    if (!mbar_wait(&empty[st], ph ^ 1, p.status)) return;
                    mbar_arrive_expect_tx(&full[st], stage_bytes);
                    tma_load_2d(base + static_cast<size_t>(st) * stage_bytes, &tmC, kc * 128, u * p.R, &full[st]);
                    // only a short head start of the code stream before the consumers' X loads: a full
                    // ring in flight delays those loads (measured)
                    if (u == static_cast<int>(blockIdx.x) && kc == kDpPrefill - 1) {
                        if (!mbar_wait(xready, 0, p.status)) return;
                        // the consumers' generic accesses to the later stages (the rotation's
                        // exchange buffer) come before the copies that refill them
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    }
                    if (++st == p.stages) { st = 0; ph ^= 1; }
                }
            }
        }
        return;
    }

    // -------------------------------------------------------------------- consumers
    const int cw = warp - 1, ct = threadIdx.x - 32;
    const auto bar_consumers = [] { asm volatile("bar.sync 1, %0;" ::"r"(32 * CW) : "memory"); };
    // A and b are weights like the codes: read before the wait, only X comes from the previous kernel;
    // so is max_k sum_j |A[j][k]| (lane k of every warp)
    if (ct < p.d * p.d + p.d) ab_s[ct] = ct < p.d * p.d ? __ldg(p.A + ct) : __ldg(p.b + (ct - p.d * p.d));
    float acol = 0.0f;
    if (lane < p.d)
        for (int j = 0; j < p.d; ++j) acol += fabsf(__ldg(p.A + j * p.d + lane));
    for (int o = 16; o; o >>= 1) acol = fmaxf(acol, __shfl_xor_sync(0xffffffffu, acol, o));
    asm volatile("griddepcontrol.wait;" ::: "memory");
    float scale, corr;
    {
        // pass 1: A, b to shared memory; max|X| per warp. Lane l of warp cw reads the 16-column block l
        // of tiles cw, cw + CW, ...; the first block stays in registers for pass 2.
        const int D = p.d;
        const bool f32in = p.f32in != 0;
        float x0[16];
        float mx = 0.0f;
        if (cw < p.nkc) load_block(p.X, f32in, p.n, 0, (static_cast<int64_t>(cw) * 32 + lane) * 16, x0);
        if (p.hb > 0) {
            // the rotation (launcher: nkc == CW, so every consumer thread holds one 16-column block);
            // ring stages kDpPrefill.. are still empty (the producer waits for xready before filling
            // them) and serve as the exchange buffer
            wht_reg16(x0, 1, p.hb);
            wht_lanes(x0, lane, p.hb);
            if (p.hb > 32 * 16) {
                float *xs = reinterpret_cast<float *>(base + static_cast<size_t>(kDpPrefill) * stage_bytes);
                const int t = cw * 32 + lane;
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    reinterpret_cast<float4 *>(xs + 16 * t)[q] = make_float4(x0[4 * q], x0[4 * q + 1], x0[4 * q + 2], x0[4 * q + 3]);
                bar_consumers();
                float y[16];
#pragma unroll
                for (int w = 0; w < 16; ++w) y[w] = w < CW ? xs[t + 512 * w] : 0.0f;
                wht_reg16(y, 512, p.hb);
#pragma unroll
                for (int w = 0; w < 16; ++w)
                    if (w < CW) xs[t + 512 * w] = y[w];
                bar_consumers();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 v = reinterpret_cast<const float4 *>(xs + 16 * t)[q];
                    x0[4 * q] = v.x; x0[4 * q + 1] = v.y; x0[4 * q + 2] = v.z; x0[4 * q + 3] = v.w;
                }
            }
            const float nrm = rsqrtf(static_cast<float>(p.hb));
#pragma unroll
            for (int i = 0; i < 16; ++i) x0[i] *= nrm;
        }
        if (cw < p.nkc) mx = absmax16(x0, mx);
        for (int tile = cw + CW; tile < p.nkc; tile += CW) {
            float x[16];
            load_block(p.X, f32in, p.n, 0, (static_cast<int64_t>(tile) * 32 + lane) * 16, x);
            mx = absmax16(x, mx);
        }
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if (lane == 0) red_s[cw] = mx;
        bar_consumers();
        if (ct == 0) mbar_arrive(xready);
        // pass 2: the token's scale s = max|X| * max_k sum_j |A[j][k]| / 32767 (a bound on max|X'|),
        // then X' -> int16. The maxima by warp shuffles (no serial chains of shared-memory loads).
        float xmax = lane < CW ? red_s[lane] : 0.0f;
        for (int o = 16; o; o >>= 1) xmax = fmaxf(xmax, __shfl_xor_sync(0xffffffffu, xmax, o));
        const float bound = xmax * acol;
        scale = bound * (1.0f / 32767.0f);
        // inv need not be exactly 1 / scale: |X'| * inv stays <= 32767 up to rounding (clamped)
        const float inv = bound > 0.0f ? __fdividef(32767.0f, bound) : 0.0f;
        uint8_t *xq_s = base + L.xq;
        float r = 0.0f;
        if (cw < p.nkc) {
            if (D == 8) dp_quantize<8>(x0, ab_s, xq_s, inv, cw, lane, r);
            else dp_quantize<4>(x0, ab_s, xq_s, inv, cw, lane, r);
        }
        for (int tile = cw + CW; tile < p.nkc; tile += CW) {
            float x[16];
            load_block(p.X, f32in, p.n, 0, (static_cast<int64_t>(tile) * 32 + lane) * 16, x);
            if (D == 8) dp_quantize<8>(x, ab_s, xq_s, inv, tile, lane, r);
            else dp_quantize<4>(x, ab_s, xq_s, inv, tile, lane, r);
        }
        for (int o = 16; o; o >>= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
        if (lane == 0) red_s[CW + cw] = r;
        bar_consumers();
        corr = lane < CW ? red_s[CW + lane] : 0.0f;
        for (int o = 16; o; o >>= 1) corr += __shfl_xor_sync(0xffffffffu, corr, o);
    }

    // this lane's word in any of its rows: 16-byte chunk (lane / 4) ^ (row % 8), row % 8 = warp % 8
    const int lane_word = (((lane >> 2) ^ (cw & 7)) << 2) + (lane & 3);
    const uint32_t *ring_w = reinterpret_cast<const uint32_t *>(base) + cw * 32 + lane_word;
    const uint4 *xq_v = reinterpret_cast<const uint4 *>(base + L.xq) + lane;
    // per-tile bookkeeping kept to a minimum (the loop is issue-bound): barrier addresses as 32-bit
    // shared addresses, the tile pointer advanced instead of recomputed
    const uint32_t full_a = smem_u32(full), empty_a = smem_u32(empty);
    int st = 0;
    uint32_t ph = 0;
    const uint32_t *tile = ring_w;
    bool ok = true;
    for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
        int32_t acc[RPT][2];
#pragma unroll
        for (int j = 0; j < RPT; ++j) acc[j][0] = acc[j][1] = 0;

        const uint4 *xv = xq_v;
        for (int kc = 0; kc < p.nkc; ++kc) {
            // this lane's 16 activation columns of tile kc (fetched before waiting for the code tile)
            const uint4 xa = xv[0], xb = xv[32];
            xv += 64;
            if (!mbar_wait_u32(full_a + 8u * st, ph, p.status)) { ok = false; break; }
            uint32_t w[RPT];
#pragma unroll
            for (int j = 0; j < RPT; ++j) w[j] = tile[j * CW * 32];
#pragma unroll
            for (int j = 0; j < RPT; ++j) dp_word(w[j], xa, xb, acc[j][0], acc[j][1]);
            __syncwarp();
            if (lane == 0) mbar_arrive_u32(empty_a + 8u * st);
            if (++st == p.stages) {
                st = 0;
                ph ^= 1;
                tile = ring_w;
            } else {
                tile += RPT * CW * 32;
            }
        }
        if (!ok) break;
        // sum the 32 lanes of each row (exact integer warp reductions: each accumulator covers half the
        // row's columns, below 2^31 for n <= 32768), scale, + corr, bf16 store
        const int64_t row0 = static_cast<int64_t>(u) * p.R + cw;
#pragma unroll
        for (int j = 0; j < RPT; ++j) {
            const int32_t s0 = __reduce_add_sync(0xffffffffu, acc[j][0]);
            const int32_t s1 = __reduce_add_sync(0xffffffffu, acc[j][1]);
            const int64_t row = row0 + static_cast<int64_t>(CW) * j;
            if (lane == 0 && row < p.m) {
                const float v = static_cast<float>(static_cast<int64_t>(s0) + static_cast<int64_t>(s1));
                const __nv_bfloat16 h = __float2bfloat16_rn(fmaf(v, scale, corr));
                p.Y[row] = *reinterpret_cast<const uint16_t *>(&h);
            }
        }
    }
}

// ------------------------------------------------------------------ host side

// ------------------------------------------------------------------ block Walsh-Hadamard rotation
//
// out[r, blk*B + j] = (1/sqrt(B)) sum_i in[r, blk*B + i] * H_B[i][j] (Sylvester H, symmetric). The
// transform factors over the bits of the index: one stage per bit combines each pair of elements whose
// indices differ in that bit only, (u, v) -> (u + v, u - v). in may equal out (each block is read whole
// before it is written).
//
// Blocks of B >= 64: one CTA of T = B / E threads per (row, block); element idx = t + T i sits in
// register i of thread t. Index bits [log2 T, log2 B) are combined in registers, bits [0, 5) (the lane)
// with warp shuffles, and bits [5, log2 T) (the warp) after one exchange through shared memory, where
// each thread takes elements that differ only in those bits and then writes its results.
// Blocks of B <= 32: one thread per block, all stages in registers.

template <int E>
__device__ __forceinline__ void wht_registers(float (&x)[E]) {
#pragma unroll
    for (int h = 1; h < E; h <<= 1)
#pragma unroll
        for (int i = 0; i < E; ++i)
            if ((i & h) == 0) {
                const float u = x[i], v = x[i + h];
                x[i] = u + v;
                x[i + h] = u - v;
            }
}

template <typename InT>
__device__ __forceinline__ float load_act(const InT *p, int64_t i) {
    if constexpr (sizeof(InT) == 2)
        return __uint_as_float(static_cast<uint32_t>(p[i]) << 16);
    else
        return p[i];
}

template <int LB>
struct WhtShape {
    static constexpr int B = 1 << LB;
    static constexpr int E = LB >= 14 ? 32 : (LB >= 9 ? 16 : B / 32);   // elements per thread
    static constexpr int T = B / E;                                        // threads, 32 .. 1024
    static constexpr int LT = LB >= 14 ? LB - 5 : (LB >= 9 ? LB - 4 : 5);
    static constexpr int W = LT - 5;                                       // warp index bits
};

template <int LB, typename InT>
__global__ void __launch_bounds__(WhtShape<LB>::T)
hadamard_block_kernel(const InT *__restrict__ in, int64_t n, float *out) {
    using S = WhtShape<LB>;
    constexpr int E = S::E, T = S::T, W = S::W;
    static_assert(S::B == E * T && (1 << S::LT) == T && (1 << W) <= E, "bad shape");
    extern __shared__ float hbuf[];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * n + static_cast<int64_t>(blockIdx.y) * S::B;
    const float scale = rsqrtf(static_cast<float>(S::B));
    float x[E];
#pragma unroll
    for (int i = 0; i < E; ++i) x[i] = load_act(in, base + t + T * i);
    wht_registers<E>(x);                                   // bits [LT, LB)
#pragma unroll
    for (int h = 1; h < 32; h <<= 1) {                     // bits [0, 5)
        const bool hi = (lane & h) != 0;
#pragma unroll
        for (int i = 0; i < E; ++i) {
            const float o = __shfl_xor_sync(0xffffffffu, x[i], h);
            x[i] = hi ? o - x[i] : x[i] + o;
        }
    }
    if constexpr (W == 0) {
#pragma unroll
        for (int i = 0; i < E; ++i) out[base + t + T * i] = x[i] * scale;
    } else {
        // bits [5, LT): element lane | k << 5 | (warp | g << W) << LT, k < 2^W, g < E / 2^W
#pragma unroll
        for (int i = 0; i < E; ++i) hbuf[t + T * i] = x[i];
        __syncthreads();
        constexpr int K = 1 << W, G = E / K;
#pragma unroll
        for (int g = 0; g < G; ++g) {
            float y[K];
            const int hi_part = (warp | (g << W)) << S::LT;
#pragma unroll
            for (int k = 0; k < K; ++k) y[k] = hbuf[lane | (k << 5) | hi_part];
            wht_registers<K>(y);
#pragma unroll
            for (int k = 0; k < K; ++k) out[base + (lane | (k << 5) | hi_part)] = y[k] * scale;
        }
    }
}

template <int LB, typename InT>
__global__ void __launch_bounds__(256)
hadamard_small_kernel(const InT *__restrict__ in, int64_t rows, int64_t n, float *out) {
    constexpr int B = 1 << LB;
    const int64_t nb = n >> LB;
    const int64_t blk = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
    if (blk >= rows * nb) return;
    const int64_t base = (blk / nb) * n + (blk % nb) * B;
    float x[B];
#pragma unroll
    for (int i = 0; i < B; ++i) x[i] = load_act(in, base + i);
    wht_registers<B>(x);
    const float scale = rsqrtf(static_cast<float>(B));
#pragma unroll
    for (int i = 0; i < B; ++i) out[base + i] = x[i] * scale;
}

int hadamard_block_size(int64_t n) {
    int bsz = 1;
    while (n % (2 * bsz) == 0 && 2 * bsz <= 32768) bsz *= 2;
    return bsz;
}

template <int LB, typename InT>
static cudaError_t launch_wht(const InT *in, int64_t rows, int64_t n, float *out, cudaStream_t st) {
    if constexpr (LB <= 5) {
        const int64_t blocks = rows * (n >> LB);
        hadamard_small_kernel<LB, InT><<<static_cast<unsigned>((blocks + 255) / 256), 256, 0, st>>>(in, rows, n, out);
    } else {
        using S = WhtShape<LB>;
        const size_t smem = S::W > 0 ? static_cast<size_t>(S::B) * 4 : 0;
        if (smem) {
            const cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(hadamard_block_kernel<LB, InT>),
                                                      static_cast<int>(smem));
            if (e != cudaSuccess) return e;
        }
        dim3 grid(static_cast<unsigned>(rows), static_cast<unsigned>(n >> LB));
        hadamard_block_kernel<LB, InT><<<grid, S::T, smem, st>>>(in, n, out);
    }
    return cudaGetLastError();
}

template <typename InT>
static cudaError_t launch_wht_any(const InT *in, int64_t rows, int64_t n, float *out, cudaStream_t st) {
    switch (hadamard_block_size(n)) {
        case 1: return launch_wht<0>(in, rows, n, out, st);
        case 2: return launch_wht<1>(in, rows, n, out, st);
        case 4: return launch_wht<2>(in, rows, n, out, st);
        case 8: return launch_wht<3>(in, rows, n, out, st);
        case 16: return launch_wht<4>(in, rows, n, out, st);
        case 32: return launch_wht<5>(in, rows, n, out, st);
        case 64: return launch_wht<6>(in, rows, n, out, st);
        case 128: return launch_wht<7>(in, rows, n, out, st);
        case 256: return launch_wht<8>(in, rows, n, out, st);
        case 512: return launch_wht<9>(in, rows, n, out, st);
        case 1024: return launch_wht<10>(in, rows, n, out, st);
        case 2048: return launch_wht<11>(in, rows, n, out, st);
        case 4096: return launch_wht<12>(in, rows, n, out, st);
        case 8192: return launch_wht<13>(in, rows, n, out, st);
        case 16384: return launch_wht<14>(in, rows, n, out, st);
        default: return launch_wht<15>(in, rows, n, out, st);
    }
}

cudaError_t launch_hadamard(const void *in, bool in_bf16, int64_t rows, int64_t n, float *out, cudaStream_t st) {
    const cudaError_t e = in_bf16 ? launch_wht_any(static_cast<const uint16_t *>(in), rows, n, out, st)
                                  : launch_wht_any(static_cast<const float *>(in), rows, n, out, st);
    count_launch();
    return e;
}

size_t packed_gemv_workspace(int64_t N, int64_t n) {
    const size_t xp = static_cast<size_t>(N) * static_cast<size_t>(gemv_npad(n)) * 2;
    const size_t cr = static_cast<size_t>(N) * static_cast<size_t>(gemv_nprep(n)) * 4;
    const size_t mma_sync_path = ((xp + 255) / 256) * 256 + ((cr + 255) / 256) * 256;
    const size_t fp4_path = packed_gemv_fp4_workspace(N, n);
    return mma_sync_path > fp4_path ? mma_sync_path : fp4_path;
}

size_t packed_gemv_corr_offset(int64_t N, int64_t n) {
    const size_t xp = static_cast<size_t>(N) * static_cast<size_t>(gemv_npad(n)) * 2;
    return ((xp + 255) / 256) * 256;
}

// Tensor-core variant configurations: (token tiles, warps per K phase, row blocks per warp, K
// phases). The unit has CWR * 16 * RBW rows; the launcher picks the configuration whose units
// balance best over the CTAs.
struct GemvTmaConfig {
    int nt, cwr, rbw, ks;
    void (*kernel)(const CUtensorMap, const GemvTmaParams);
};
// In order of preference; a later entry wins only if its units balance at least half a percent better.
static const GemvTmaConfig kGemvTmaConfigs[] = {
    {1, 4, 3, 2, packed_gemv_tma_kernel<1, 4, 3, 2>}, {1, 4, 2, 2, packed_gemv_tma_kernel<1, 4, 2, 2>},
    {1, 4, 1, 2, packed_gemv_tma_kernel<1, 4, 1, 2>}, {2, 4, 3, 2, packed_gemv_tma_kernel<2, 4, 3, 2>},
    {2, 4, 2, 2, packed_gemv_tma_kernel<2, 4, 2, 2>}, {2, 4, 1, 2, packed_gemv_tma_kernel<2, 4, 1, 2>},
};

static const GemvTmaConfig *choose_tma_config(int64_t m, int ctas, int nt) {
    const GemvTmaConfig *best = nullptr;
    double best_eff = -1.0;
    for (const GemvTmaConfig &c : kGemvTmaConfigs) {
        if (c.nt != nt) continue;
        const int R = c.cwr * 16 * c.rbw;
        const int64_t units = (m + R - 1) / R;
        const int64_t rounds = (units + ctas - 1) / ctas;
        const double eff = static_cast<double>(units) / static_cast<double>(rounds * (units < ctas ? units : ctas));
        const double rows_eff = static_cast<double>(m) / static_cast<double>(units * R);
        const double busy = static_cast<double>(units < ctas ? units : ctas) / static_cast<double>(ctas);
        const double e = eff * rows_eff * busy;
        if (e > best_eff + 0.005) { best_eff = e; best = &c; }
    }
    return best;
}

// Rows per thread per tile the dp2a kernel is instantiated for (a unit has kDpWarps * RPT rows).
static const int kDpRpts[] = {16, 12, 8, 6, 4, 3, 2, 1};

// Rows per unit for the dp2a variant: balance the units over the CTAs, and prefer all SMs busy.
static int choose_rows_dp(int64_t m, int ctas) {
    int best = kDpWarps;
    double best_eff = -1.0;
    for (int rpt : kDpRpts) {
        const int R = kDpWarps * rpt;
        const int64_t units = (m + R - 1) / R;
        const int64_t rounds = (units + ctas - 1) / ctas;
        const double eff = static_cast<double>(units) / static_cast<double>(rounds * (units < ctas ? units : ctas));
        const double rows_eff = static_cast<double>(m) / static_cast<double>(units * R);
        const double busy = static_cast<double>(units < ctas ? units : ctas) / static_cast<double>(ctas);
        const double e = eff * rows_eff * busy;
        if (e > best_eff + 1e-9) { best_eff = e; best = R; }
    }
    return best;
}

static bool make_codes_map(CUtensorMap *map, const uint8_t *packed, int64_t m, int64_t n, int R) {
    void *fnp = tensor_map_encoder();
    if (!fnp) return false;
    auto enc = reinterpret_cast<CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                             const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                             CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                             CUtensorMapFloatOOBfill)>(fnp);
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(n / 4), static_cast<cuuint64_t>(m)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(n / 4)};
    cuuint32_t box[2] = {128, static_cast<cuuint32_t>(R)};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(packed), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename... KArgs, typename... Args>
static cudaError_t launch_pdl(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k, std::forward<Args>(args)...);
}

// dp2a variant for one token. Leaves `done` false (and launches nothing) when the activations do
// not fit in shared memory next to a ring of at least three stages.
// Rows per unit, ring stages and rotation block of the dp kernel for this call; false when the kernel
// does not apply (the activations would not fit next to a ring of three stages, or a requested
// prologue rotation lacks its one-block-per-thread layout or exchange buffer).
static bool dp_plan(const PackedGemvArgs &a, int num_sms, int &R, int &stages, int &nkc, int &hb) {
    nkc = static_cast<int>(gemv_npad(a.n) / kTileCols);
    R = choose_rows_dp(a.m, num_sms);
    stages = kTmaStages;
    while (stages >= 3 && dp_smem_layout(R, stages, nkc).total + 1024 > kDpSmemLimit) --stages;
    if (stages < 3) return false;
    hb = 0;
    if (a.rotate) {
        // the prologue rotation wants one 16-column block per consumer thread and an exchange buffer
        // in the ring stages the producer fills only after the activations are in
        if (a.Xf || nkc != kDpWarps ||
            static_cast<size_t>(stages - kDpPrefill) * static_cast<size_t>(R) * 128 < static_cast<size_t>(a.n) * 4)
            return false;
        hb = hadamard_block_size(a.n);
    }
    return true;
}

static cudaError_t launch_packed_gemv_dp(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st, bool &done) {
    done = false;
    int R, stages, nkc, hb;
    if (!dp_plan(a, num_sms, R, stages, nkc, hb)) return cudaSuccess;
    CUtensorMap map;
    if (!make_codes_map(&map, a.packed, a.m, a.n, R)) return cudaErrorInvalidValue;
    GemvDpParams p;
    p.X = a.Xf ? static_cast<const void *>(a.Xf) : static_cast<const void *>(a.X);
    p.A = a.A;
    p.b = a.b;
    p.m = a.m;
    p.n = a.n;
    p.d = d;
    p.f32in = a.Xf != nullptr;
    p.hb = hb;
    p.R = R;
    p.units = static_cast<int>((a.m + R - 1) / R);
    p.nkc = nkc;
    p.stages = stages;
    p.Y = a.Y;
    p.status = a.status;
    const int grid = p.units < num_sms ? p.units : num_sms;
    const size_t smem = dp_smem_layout(R, stages, nkc).total + 1024;
    void (*k)(const CUtensorMap, const GemvDpParams) = nullptr;
    switch (R / kDpWarps) {
        case 16: k = packed_gemv_dp_kernel<16>; break;
        case 12: k = packed_gemv_dp_kernel<12>; break;
        case 8: k = packed_gemv_dp_kernel<8>; break;
        case 6: k = packed_gemv_dp_kernel<6>; break;
        case 4: k = packed_gemv_dp_kernel<4>; break;
        case 3: k = packed_gemv_dp_kernel<3>; break;
        case 2: k = packed_gemv_dp_kernel<2>; break;
        default: k = packed_gemv_dp_kernel<1>; break;
    }
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(k, dim3(grid), dim3(32 * (kDpWarps + 1)), smem, st, map, p);
    count_launch();
    if (e != cudaSuccess) return e;
    done = true;
    return cudaSuccess;
}

bool launch_packed_gemv_rotated(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st, cudaError_t &err) {
    err = cudaSuccess;
    PackedGemvArgs r = a;
    r.rotate = true;
    r.Xf = nullptr;
    int R, stages, nkc, hb;
    if (a.n % 64 == 0 && a.n <= kDpMaxN && a.m >= 16 && a.N == kDpMaxTokens && dp_plan(r, num_sms, R, stages, nkc, hb)) {
        // one token: the rotation runs in the dp kernel's prologue
        bool done = false;
        trace_begin(LCQ_K_GEMV, st);
        err = launch_packed_gemv_dp(r, d, num_sms, st, done);
        if (err == cudaSuccess) {
            trace_end(LCQ_K_GEMV, st);
            err = cudaGetLastError();
        }
        return true;
    }
    // 1-16 tokens, n % 64 == 0, n <= 32768: the rotation runs in the tcgen05 kernel's prep kernel (a
    // begin mark left when that kernel does not apply is overwritten by the next one)
    trace_begin(LCQ_K_GEMV, st);
    if (!launch_packed_gemv_fp4(r, d, num_sms, st, err)) return false;
    if (err == cudaSuccess) {
        trace_end(LCQ_K_GEMV, st);
        err = cudaGetLastError();
    }
    return true;
}

cudaError_t launch_packed_gemv(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t npad = gemv_npad(a.n), nprep = gemv_nprep(a.n);
    trace_begin(LCQ_K_GEMV, st);
    if (a.N > kFp4MinTokens) {
        // 2-16 tokens, n % 64 == 0, n <= 32768: codes as fp4 tensor-core operands in tensor memory
        // (tcgen05); faster than the mma.sync kernel below at every token count from 2 (70B gate:
        // 14.5-14.9 against 18.4-18.6 us at 2-8 tokens), which keeps the other shapes
        cudaError_t e = cudaSuccess;
        if (launch_packed_gemv_fp4(a, d, num_sms, st, e)) {
            if (e != cudaSuccess) return e;
            trace_end(LCQ_K_GEMV, st);
            return cudaGetLastError();
        }
    }
    if (a.n % 64 == 0 && a.n <= kDpMaxN && a.m >= 16 && a.N == kDpMaxTokens) {
        bool done = false;
        const cudaError_t e = launch_packed_gemv_dp(a, d, num_sms, st, done);
        if (e != cudaSuccess) return e;
        if (done) {
            trace_end(LCQ_K_GEMV, st);
            return cudaGetLastError();
        }
    }
    const bool tiled = a.n % 64 == 0 && a.m >= 16;
    dim3 pgrid(static_cast<unsigned>(a.N), static_cast<unsigned>(nprep));
    using PrepFn = void (*)(const void *, int64_t, int64_t, const float *, const float *, uint16_t *, float *);
    PrepFn prep;
    if (a.Xf)
        prep = d == 4 ? (tiled ? gemv_prep_kernel<4, true, true> : gemv_prep_kernel<4, true, false>)
                      : (tiled ? gemv_prep_kernel<8, true, true> : gemv_prep_kernel<8, true, false>);
    else
        prep = d == 4 ? (tiled ? gemv_prep_kernel<4, false, true> : gemv_prep_kernel<4, false, false>)
                      : (tiled ? gemv_prep_kernel<8, false, true> : gemv_prep_kernel<8, false, false>);
    prep<<<pgrid, 256, 0, st>>>(a.Xf ? static_cast<const void *>(a.Xf) : static_cast<const void *>(a.X), a.n, npad,
                                a.A, a.b, a.Xp, a.corr);
    count_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (tiled) {
        for (int64_t t0 = 0; t0 < a.N; t0 += 16) {
            const int64_t ntok = (a.N - t0) < 16 ? (a.N - t0) : 16;
            const GemvTmaConfig *c = choose_tma_config(a.m, num_sms, ntok > 8 ? 2 : 1);
            const int R = c->cwr * 16 * c->rbw;
            CUtensorMap map;
            if (!make_codes_map(&map, a.packed, a.m, a.n, R)) return cudaErrorInvalidValue;
            int stages = kTmaStages;
            while (stages > 2 && gemv_tma_layout(R, stages, c->nt, c->cwr, c->rbw, c->ks).total + 1024 > kGemvSmemLimit)
                --stages;
            GemvTmaParams p;
            p.m = a.m;
            p.ntok_all = a.N;
            p.npad = npad;
            p.nprep = nprep;
            p.ntok = static_cast<int>(ntok);
            p.t0 = static_cast<int>(t0);
            p.units = static_cast<int>((a.m + R - 1) / R);
            p.nkc = static_cast<int>(npad / kTileCols);
            p.stages = stages;
            p.Xp = a.Xp;
            p.corrpart = a.corr + t0 * nprep;
            p.Y = a.Y + t0 * a.m;
            p.status = a.status;
            const int grid = p.units < num_sms ? p.units : num_sms;
            const size_t smem = gemv_tma_layout(R, stages, c->nt, c->cwr, c->rbw, c->ks).total + 1024;
            e = ensure_dynamic_smem(reinterpret_cast<const void *>(c->kernel), static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            e = launch_pdl(c->kernel, dim3(grid), dim3(32 * (c->cwr * c->ks + 1)), smem, st, map, p);
            count_launch();
            if (e != cudaSuccess) return e;
        }
    } else {
        dim3 grid(static_cast<unsigned>((a.m + kGemvRows - 1) / kGemvRows), static_cast<unsigned>((a.N + 15) / 16));
        const bool vec = (a.n % 64) == 0;
        if (vec)
            e = launch_pdl(packed_gemv_kernel<true>, grid, dim3(32 * kGemvWarps), 0, st, a.packed, a.m, a.n, a.N,
                           static_cast<const uint16_t *>(a.Xp), npad, static_cast<const float *>(a.corr), nprep, a.Y);
        else
            e = launch_pdl(packed_gemv_kernel<false>, grid, dim3(32 * kGemvWarps), 0, st, a.packed, a.m, a.n, a.N,
                           static_cast<const uint16_t *>(a.Xp), npad, static_cast<const float *>(a.corr), nprep, a.Y);
        count_launch();
        if (e != cudaSuccess) return e;
    }
    trace_end(LCQ_K_GEMV, st);
    return cudaGetLastError();
}

}  // namespace lcq
