// Deployment product from packed 2-bit codes on the 5th-generation tensor cores (tcgen05,
// kind::mxf4), through the reformulated forward of Sec. 3.2 (Eq. def:forward_x):
//
//   Y[t][r] = sum_c X'[t][c] z[r][c] + sum_g X_g[t] . b,     X'_g = X_g A  (per group of d columns)
//
// Operands. A 2-bit code z placed in the low half of a 4-bit field is the e2m1 (fp4) value z / 2,
// exactly, so 16 packed codes become 16 fp4 elements with one shift and two ANDs:
//   w & 0x33333333          -> codes 0, 2, 4, .., 14 of the word in nibbles 0..7
//   (w >> 2) & 0x33333333   -> codes 1, 3, 5, .., 15
// The activations are made exact integers and split into digits that e2m1 also holds exactly:
// per token, q = rint(X' / D_t) with D_t = max|X'_t| / 8191, and q = sum_j d_j 8^j with balanced
// digits d_j in [-4, 3] (j = 0..4). Every product (z/2) d_j is exact and every partial sum is a
// multiple of 1/2 far below 2^24, so the fp32 accumulators hold sum_c (z/2) d_j exactly, and
//   Y[t][r] = 2 D_t sum_j 8^j acc[r][(t, j)] + sum_g X_g[t] . b.
// The only rounding is that of X' to q (at most D_t / 2 per element) and of the final sums.
//
// Roles (one CTA per SM, persistent over contiguous ranges of at most 256 rows, whole K per range):
//   warp 0      code producer: per 512-column tile, a 2-D TMA copy of the range's code rows (one box of
//               up to 256 rows, 128-byte swizzle) into the code ring. The converters free a code stage
//               as soon as they have read it, so the ring streams from HBM at its own pace; its first
//               stages fill while the prep kernel still runs (programmatic dependent launch).
//   warp 10     digit producer: after the prep kernel has completed, the tile's activation digits (two
//               128-byte-wide boxes) into the digit ring; a digit stage is freed by the MMAs reading it.
//   warp 1      TMEM owner and MMA issuer: per tile and 128-row block, eight
//               tcgen05.mma.kind::mxf4.block_scale (M = 128, N = 5 x tokens rounded up to 16,
//               K = 64), A (codes) from tensor memory, B (digits) from the digit ring, every block
//               scale 1. It never touches shared memory while MMAs are queued (such an access waits for
//               them): the converters hand each tile over through a named barrier.
//   warps 2-9   converters, two teams of four (warps 2-5 and 6-9) taking alternate tiles, so that the
//               per-tile chain of one team (code loads, mbarrier checks, stores, barrier) overlaps the
//               other's: a warp expands the 512 codes of its TMEM lane quarter's rows of both 128-row
//               blocks from the code ring into the tile's fp4 A slot in tensor memory (slot = team),
//               waits for the tile's digits, then joins the named barrier of that slot. They also run
//               the epilogue of a range (warp of team t: block t): tcgen05.ld of the accumulator, the
//               digit sum and scales, bf16 stores.
// Every wait on an mbarrier gives up after kWaitLimitNs (status LCQ_ERR_TIMEOUT); every warp still
// reaches every named barrier of every tile, so no warp waits forever on one.
#include "common.cuh"
#include "internal.h"

namespace lcq {

namespace {

constexpr int kF4Digits = 5;               // balanced base-8 digits per activation
constexpr float kF4QMax = 8191.0f;         // |q| bound; 5 digits in [-4, 3] cover [-18724, 14043]
constexpr int kF4DigitBias = 18724;        // 4 (1 + 8 + 64 + 512 + 4096): q + bias has octal digits d_j + 4
constexpr int kF4MaxTokens = 16;
constexpr int kF4TileCols = 512;           // codes per row and ring stage (128 bytes)
constexpr int kF4SliceRows = 32;           // rows per code box
constexpr int kF4MaxSlices = 8;            // rows per range <= 256: two 128-row MMA blocks
constexpr int kF4ConvWarps = 8;            // two teams of one warp per TMEM lane quarter
constexpr int kF4Conv0 = 2;                // first converter warp
constexpr int kF4DigitWarp = kF4Conv0 + kF4ConvWarps;
constexpr int kF4Threads = 32 * (kF4DigitWarp + 1);
constexpr int kF4CodeStagesMax = 8;
constexpr int kF4DigitStagesMax = 4;
constexpr int kF4MinCodeStages = 5;       // code stages kept before digit stages are given up
constexpr int kF4PreStages = 8;           // code tiles requested before the prep kernel has completed
constexpr uint32_t kF4TmemCols = 512;
// Tensor memory columns: accumulators of the two row blocks, block scales of A and B, the A ring
// (slot s, block rb at kF4ColA + 128 s + 64 rb: 8 columns per K step of 64 fp4 elements).
constexpr uint32_t kF4ColD1 = 128, kF4ColSFA = 224, kF4ColSFB = 240, kF4ColA = 256;
// Named barriers (0 is __syncthreads): A slot s full = 1 + s; accumulator read = 3.
constexpr int kF4BarAFull = 1, kF4BarDFree = 3;
constexpr int kF4TeamWarps = kF4ConvWarps / 2;   // converter warps per tile (two teams)
constexpr int kF4BarAFullCount = 32 * (kF4TeamWarps + 1);
constexpr int kF4BarDFreeCount = 32 * (8 + 1);   // the eight epilogue warps and the issuer
constexpr size_t kF4SmemLimit = 227 * 1024;
constexpr size_t kF4SmemMin = 120 * 1024;

__host__ __device__ inline int f4_nb(int ntok) { return (ntok * kF4Digits + 15) / 16 * 16; }

struct F4Params {
    int64_t m;
    int slices, ranges, tiles, ntok, NB, cstages, dstages;
    uint32_t code_bytes, act_bytes;
    const float *scale;      // [ntok] 2 max|X'_t| / 8191
    const float *corr;       // [ntok] sum_g X_g[t] . b
    uint16_t *Y;             // [ntok][m]
    int32_t *status;
};

// kind::mxf4 instruction descriptor: A and B e2m1, ue8m0 block scales, both K-major, fp32 D.
__host__ __device__ constexpr uint32_t idesc_mxf4(int M, int N) {
    return (1u << 7)                                   // A format: e2m1
           | (1u << 10)                                // B format: e2m1
           | (static_cast<uint32_t>(N >> 3) << 17)     // N / 8
           | (1u << 23)                                // scale factor format: ue8m0
           | (static_cast<uint32_t>(M >> 4) << 24);    // M / 16
}

// D[tmem] (+)= (A[tmem] x SFA) * (B[smem] x SFB)^T, K = 64, two scale factors per row and K step.
__device__ __forceinline__ void umma_mxf4_ts(uint32_t d, uint32_t a, uint64_t bdesc, uint32_t idesc, uint32_t sfa,
                                             uint32_t sfb, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %6, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::mxf4.block_scale.scale_vec::2X [%0], [%1], %2, %3, [%4], [%5], p;\n\t}" ::"r"(d),
        "r"(a), "l"(bdesc), "r"(idesc), "r"(sfa), "r"(sfb), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
        "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
        "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, uint32_t v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %1, %1, %1, %1, %1, %1, %1};" ::"r"(taddr), "r"(v)
        : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float *v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Bounded wait for a thread that need not react quickly (the producers): it sleeps between polls so
// that it takes no issue slots from the converter warps sharing its SM sub-partition.
__device__ __noinline__ bool mbar_wait_backoff(uint64_t *bar, uint32_t parity, int32_t *status) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        __nanosleep(64);
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 15u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
            set_status(status, LCQ_ERR_TIMEOUT);
            return false;
        }
    }
}

// A warp waits on an mbarrier phase through one lane (the others meet it at __syncwarp, which orders
// the phase's writes before their reads); returns the warp-uniform outcome. Skips the wait once a
// previous one failed (ok == false).
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, bool ok, int32_t *status) {
    uint32_t r = ok ? 1u : 0u;
    if (ok && (threadIdx.x & 31) == 0) r = mbar_wait(bar, parity, status) ? 1u : 0u;
    r = __shfl_sync(0xffffffffu, r, 0);
    return r != 0;
}

// One lane of the (converged) warp returns true: warp-uniform issue of tcgen05 instructions.
__device__ __forceinline__ bool elect_one() {
    uint32_t pred;
    asm volatile(
        "{\n\t.reg .pred e;\n\t"
        "elect.sync _|e, 0xffffffff;\n\t"
        "selp.u32 %0, 1, 0, e;\n\t}"
        : "=r"(pred));
    return pred != 0;
}

__device__ __forceinline__ void named_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void named_arrive(int id, int count) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// e2m1 bit pattern of a balanced base-8 digit d in [-4, 3], one per byte, byte d + 4 of {lo, hi}
// (a byte-permute table): -4 -> 0xE, -3 -> 0xD, -2 -> 0xC, -1 -> 0xA, 0 -> 0x0, 1 -> 0x2, 2 -> 0x4,
// 3 -> 0x5
constexpr uint32_t kE2m1BytesLo = 0x0A0C0D0Eu, kE2m1BytesHi = 0x05040200u;

// Rows [s0, s1) of 32-row slices form range r of `ranges` (balanced split of `slices`).
__host__ __device__ inline void f4_range(int r, int slices, int ranges, int &s0, int &s1) {
    s0 = static_cast<int>(static_cast<int64_t>(r) * slices / ranges);
    s1 = static_cast<int>(static_cast<int64_t>(r + 1) * slices / ranges);
}

// ---------------------------------------------------------------------------------- prep kernel
//
// One CTA per token, one pass: each thread forms X' = X_g A for up to kF4PrepGroups groups of 16
// columns (kept in registers), the CTA reduces max|X'| and the bias term sum_g X_g . b, then every
// thread turns its values into q = rint(X' * 8191 / max) and the five digits, stored as e2m1 nibbles
// in the MMA's K order: within 16 columns, K position 8 p + i carries column 2 i + p (the order the
// code expansion produces). Digit row t * 5 + j of tile k is 256 bytes at dig[(k * NB + t * 5 + j) *
// 256]; the last token's CTA also zeroes rows 5 ntok .. NB - 1. With the online rotation (ROT), the
// token's row is rotated by the block Walsh-Hadamard transform first, in this same layout (f4_rotate).

constexpr int kF4PrepThreads = 512;
constexpr int kF4PrepGroups = 4;           // groups of 16 columns per thread: n <= 32768

template <int D, bool F32IN>
__device__ __forceinline__ void f4_load16(const void *__restrict__ Xv, int64_t n, int64_t t, int64_t c0,
                                          float (&x)[16]) {
    if (c0 + 16 <= n) {
        if (F32IN) {
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
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int64_t c = c0 + i;
            x[i] = c >= n ? 0.0f
                   : F32IN ? static_cast<const float *>(Xv)[t * n + c]
                           : __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t *>(Xv)[t * n + c]) << 16);
        }
    }
}

// Element e of the row sits in shared memory at word e ^ (((e >> 5) & 3) << 2): the 16-byte chunks of
// each 64-byte group are permuted by bits 5-6 of the index, so that the 16-byte stores and loads of a
// quarter warp, whose threads hold 16 consecutive elements each, fall on eight distinct 4-bank groups.
__device__ __forceinline__ int64_t f4_swz(int64_t e) { return e ^ (((e >> 5) & 3) << 2); }

// Radix-K butterflies of the Walsh-Hadamard transform over index bits [bit0, bit0 + log2 K) of the
// row in shared memory: each thread takes the K elements of a group that differ only in those bits.
// Consecutive threads take consecutive low indices (bit0 >= 9), so a warp's accesses hit 32 banks (the
// permutation above moves words within aligned runs of 32; bits >= bit0 leave it unchanged).
template <int K>
__device__ __forceinline__ void f4_wht_pass(float *buf, int64_t n, int bit0) {
    const int64_t groups = n / K;
    const int64_t low = (int64_t(1) << bit0) - 1;
    for (int64_t g = threadIdx.x; g < groups; g += kF4PrepThreads) {
        const int64_t base = f4_swz((g & low) | ((g >> bit0) << bit0) * K);
        float y[K];
#pragma unroll
        for (int k = 0; k < K; ++k) y[k] = buf[base + (static_cast<int64_t>(k) << bit0)];
#pragma unroll
        for (int h = 1; h < K; h <<= 1)
#pragma unroll
            for (int k = 0; k < K; ++k)
                if ((k & h) == 0) {
                    const float u = y[k], v = y[k + h];
                    y[k] = u + v;
                    y[k + h] = u - v;
                }
#pragma unroll
        for (int k = 0; k < K; ++k) buf[base + (static_cast<int64_t>(k) << bit0)] = y[k];
    }
}

// Normalized block Walsh-Hadamard rotation of one token's row (the online rotation of the rotated
// deployment product, Sec. 2.2 / App. Inference Speed) on the prep layout: column (threadIdx.x + 512 gg)
// * 16 + i sits in x[gg][i]. The block is 2^lb columns (6 <= lb <= 15, the largest power of two dividing
// n), so the transform factors over index bits 0 .. lb-1, one butterfly stage (u, v) -> (u + v, u - v)
// per bit, in any order: bits 0-3 in registers, bits 4-8 (the lane) by warp shuffles, bits 9 .. lb-1
// (warp and gg) through the row in shared memory (n floats, permuted as f4_swz states), up to four bits
// per pass. A column's partner in a bit below lb lies in its own block, so columns past the row's end
// never feed real ones. The result is scaled by 2^(-lb/2).
__device__ __forceinline__ void f4_rotate(float (&x)[kF4PrepGroups][16], int64_t n, int lb, float *buf) {
    const int ngg = static_cast<int>((n / 16 + kF4PrepThreads - 1) / kF4PrepThreads);
#pragma unroll
    for (int gg = 0; gg < kF4PrepGroups; ++gg) {
        if (gg >= ngg) continue;
#pragma unroll
        for (int h = 1; h < 16; h <<= 1)
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if ((i & h) == 0) {
                    const float u = x[gg][i], v = x[gg][i + h];
                    x[gg][i] = u + v;
                    x[gg][i + h] = u - v;
                }
    }
    const int lane = threadIdx.x & 31;
    const int hmax = lb >= 9 ? 32 : 1 << (lb - 4);   // lane bit h is column bit 4 + log2 h
#pragma unroll
    for (int h = 1; h < 32; h <<= 1) {
        if (h >= hmax) break;
        // the upper lane of a pair forms o - x, the lower x + o: one fma by -1 or 1 (exact, one rounding)
        const float sgn = (lane & h) ? -1.0f : 1.0f;
#pragma unroll
        for (int gg = 0; gg < kF4PrepGroups; ++gg) {
            if (gg >= ngg) continue;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float o = __shfl_xor_sync(0xffffffffu, x[gg][i], h);
                x[gg][i] = fmaf(sgn, x[gg][i], o);
            }
        }
    }
    if (lb > 9) {
#pragma unroll
        for (int gg = 0; gg < kF4PrepGroups; ++gg) {
            const int64_t c0 = (threadIdx.x + static_cast<int64_t>(gg) * kF4PrepThreads) * 16;
            if (c0 >= n) continue;
            float4 *dst = reinterpret_cast<float4 *>(buf + c0);
            const int sw = static_cast<int>(c0 >> 5) & 3;   // bits 5-6 of the group's indices
#pragma unroll
            for (int q = 0; q < 4; ++q)
                dst[q ^ sw] = make_float4(x[gg][4 * q], x[gg][4 * q + 1], x[gg][4 * q + 2], x[gg][4 * q + 3]);
        }
        for (int bit0 = 9; bit0 < lb; bit0 += 4) {
            __syncthreads();
            switch (lb - bit0) {
                case 1: f4_wht_pass<2>(buf, n, bit0); break;
                case 2: f4_wht_pass<4>(buf, n, bit0); break;
                case 3: f4_wht_pass<8>(buf, n, bit0); break;
                default: f4_wht_pass<16>(buf, n, bit0); break;
            }
        }
        __syncthreads();
#pragma unroll
        for (int gg = 0; gg < kF4PrepGroups; ++gg) {
            const int64_t c0 = (threadIdx.x + static_cast<int64_t>(gg) * kF4PrepThreads) * 16;
            if (c0 >= n) continue;
            const float4 *src = reinterpret_cast<const float4 *>(buf + c0);
            const int sw = static_cast<int>(c0 >> 5) & 3;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 f = src[q ^ sw];
                x[gg][4 * q] = f.x; x[gg][4 * q + 1] = f.y; x[gg][4 * q + 2] = f.z; x[gg][4 * q + 3] = f.w;
            }
        }
    }
    const float s = rsqrtf(static_cast<float>(1 << lb));
#pragma unroll
    for (int gg = 0; gg < kF4PrepGroups; ++gg)
#pragma unroll
        for (int i = 0; i < 16; ++i) x[gg][i] *= s;
}

// ROT: rotate the token's bf16 row by the block Walsh-Hadamard transform of block 2^lb first (dynamic
// shared memory: n floats when lb > 9).
template <int D, bool F32IN, bool ROT>
__global__ void __launch_bounds__(kF4PrepThreads)
fp4_prep_kernel(const void *__restrict__ Xv, int64_t n, int tiles, int ntok, int NB, const float *__restrict__ A,
                const float *__restrict__ b, uint8_t *__restrict__ dig, float *__restrict__ scale,
                float *__restrict__ corr, int lb) {
    // the main kernel may start streaming codes right away; it waits for these results itself
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ float sA[D * D], sb[D];
    __shared__ float red_max[kF4PrepThreads / 32], red_sum[kF4PrepThreads / 32];
    __shared__ float s_inv;
    const int64_t t = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t ngroups = static_cast<int64_t>(tiles) * (kF4TileCols / 16);
    // A and b are weights like the codes: read before the wait. This kernel is itself launched as a
    // programmatic dependent of the previous kernel in the stream (it may become resident while that
    // one runs): X, and the workspace this kernel writes, are touched only after that kernel completed.
    if (threadIdx.x < D * D) sA[threadIdx.x] = __ldg(A + threadIdx.x);
    if (threadIdx.x < D) sb[threadIdx.x] = __ldg(b + threadIdx.x);
    asm volatile("griddepcontrol.wait;" ::: "memory");
    float xv[kF4PrepGroups][16];
#pragma unroll
    for (int gg = 0; gg < kF4PrepGroups; ++gg) {
        const int64_t gi = threadIdx.x + static_cast<int64_t>(gg) * kF4PrepThreads;
        if (gi < ngroups) f4_load16<D, F32IN>(Xv, n, t, gi * 16, xv[gg]);
        else if (ROT) {
#pragma unroll
            for (int i = 0; i < 16; ++i) xv[gg][i] = 0.0f;
        }
    }
    if (ROT) {
        extern __shared__ __align__(16) float rot_buf[];
        f4_rotate(xv, n, lb, rot_buf);
    }
    __syncthreads();

    float amax = 0.0f, r = 0.0f;
#pragma unroll
    for (int gg = 0; gg < kF4PrepGroups; ++gg) {
        const int64_t gi = threadIdx.x + static_cast<int64_t>(gg) * kF4PrepThreads;
        if (gi >= ngroups) continue;
        float xp[16];
#pragma unroll
        for (int g = 0; g < 16 / D; ++g) {
            // outputs in pairs (k, k + 1) by packed fp32x2 FMAs: each lane's FMA sequence over j is
            // the scalar one
#pragma unroll
            for (int k = 0; k < D; k += 2) {
                float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    const float xj = xv[gg][g * D + j];
                    acc = __ffma2_rn(make_float2(xj, xj), make_float2(sA[j * D + k], sA[j * D + k + 1]), acc);
                }
                xp[k + g * D] = acc.x;
                xp[k + 1 + g * D] = acc.y;
            }
#pragma unroll
            for (int j = 0; j < D; ++j) r = fmaf(xv[gg][g * D + j], sb[j], r);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            xv[gg][i] = xp[i];
            amax = fmaxf(amax, fabsf(xp[i]));
        }
    }
    for (int o = 16; o; o >>= 1) {
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        r += __shfl_xor_sync(0xffffffffu, r, o);
    }
    if (lane == 0) { red_max[warp] = amax; red_sum[warp] = r; }
    __syncthreads();
    if (threadIdx.x == 0) {
        float m_ = 0.0f, s_ = 0.0f;
        for (int w = 0; w < kF4PrepThreads / 32; ++w) { m_ = fmaxf(m_, red_max[w]); s_ += red_sum[w]; }
        // NaN or inf activations give a non-finite scale, which carries into every output of the token
        scale[t] = 2.0f * (m_ / kF4QMax);
        corr[t] = s_;
        s_inv = m_ > 0.0f ? kF4QMax / m_ : 0.0f;
    }
    __syncthreads();
    const float inv = s_inv;

#pragma unroll
    for (int gg = 0; gg < kF4PrepGroups; ++gg) {
        const int64_t gi = threadIdx.x + static_cast<int64_t>(gg) * kF4PrepThreads;
        if (gi >= ngroups) continue;
        // q + 4 (1 + 8 + 64 + 512 + 4096) lies in [10533, 26915]: its five octal digits, each minus 4,
        // are the balanced digits of q (the representation is unique), so digit j is octal field j
        uint32_t u[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float v = fminf(fmaxf(xv[gg][i] * inv, -kF4QMax), kF4QMax);   // NaN -> one of the bounds
            u[i] = static_cast<uint32_t>(__float2int_rn(v) + kF4DigitBias);
        }
        const int64_t tile = gi / (kF4TileCols / 16);
        const int slot = static_cast<int>(gi % (kF4TileCols / 16));
#pragma unroll
        for (int j = 0; j < kF4Digits; ++j) {
            uint32_t lo = 0, hi = 0;   // K positions 0..7 and 8..15 of the group
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                // field j of u (bit-field extract), its e2m1 pattern from the byte table (byte
                // permute; the field selects byte f of kE2m1Bytes), inserted at the column's K position
                // (bit-field insert of the low 4 bits): column i = 2 u + p sits at K position 8 p + u
                uint32_t f, nib;
                asm("bfe.u32 %0, %1, %2, 3;" : "=r"(f) : "r"(u[i]), "r"(3 * j));
                asm("prmt.b32 %0, %1, %2, %3;" : "=r"(nib) : "r"(kE2m1BytesLo), "r"(kE2m1BytesHi), "r"(f));
                const int pos = 8 * (i & 1) + (i >> 1);
                if (pos < 8) asm("bfi.b32 %0, %1, %2, %3, 4;" : "=r"(lo) : "r"(nib), "r"(lo), "r"(4 * pos));
                else asm("bfi.b32 %0, %1, %2, %3, 4;" : "=r"(hi) : "r"(nib), "r"(hi), "r"(4 * (pos - 8)));
            }
            uint8_t *dst = dig + (tile * NB + t * kF4Digits + j) * 256 + slot * 8;
            *reinterpret_cast<uint2 *>(dst) = make_uint2(lo, hi);
        }
    }
    if (t == ntok - 1) {
        const int z0 = ntok * kF4Digits, zr = NB - z0;
        const int64_t total = static_cast<int64_t>(tiles) * zr * 16;   // 16-byte chunks
        for (int64_t o = threadIdx.x; o < total; o += kF4PrepThreads) {
            const int64_t k = o / (zr * 16);
            const int rem = static_cast<int>(o % (zr * 16));
            reinterpret_cast<uint4 *>(dig + (k * NB + z0 + rem / 16) * 256)[rem % 16] = make_uint4(0, 0, 0, 0);
        }
    }
}

// ---------------------------------------------------------------------------------- main kernel

__global__ void __launch_bounds__(kF4Threads, 1)
packed_gemv_fp4_kernel(const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmB,
                       const F4Params p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t *cring = align_smem_1024(smem_raw);                                     // [cstages][code_bytes]
    uint8_t *dring = cring + static_cast<size_t>(p.cstages) * p.code_bytes;          // [dstages][act_bytes]
    uint64_t *cfull = reinterpret_cast<uint64_t *>(dring + static_cast<size_t>(p.dstages) * p.act_bytes);
    uint64_t *cempty = cfull + kF4CodeStagesMax;   // one arrival per warp of the tile's team: codes read
    uint64_t *dfull = cempty + kF4CodeStagesMax;
    uint64_t *dempty = dfull + kF4DigitStagesMax;  // the MMAs reading the digits completed
    uint64_t *aempty = dempty + kF4DigitStagesMax; // [2] the MMAs of the tile in A slot s completed
    uint64_t *accfull = aempty + 2;                // the range's MMAs completed
    uint64_t *done = accfull + 1;                  // teardown: every MMA completed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int my_ranges = p.ranges > static_cast<int>(blockIdx.x)
                              ? (p.ranges - 1 - static_cast<int>(blockIdx.x)) / static_cast<int>(gridDim.x) + 1
                              : 0;
    const int total_tiles = my_ranges * p.tiles;

    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmC);
        prefetch_tensormap(&tmB);
        for (int i = 0; i < p.cstages; ++i) {
            mbar_init(&cfull[i], 1);
            mbar_init(&cempty[i], kF4TeamWarps);
        }
        for (int i = 0; i < p.dstages; ++i) {
            mbar_init(&dfull[i], 1);
            mbar_init(&dempty[i], 1);
        }
        for (int i = 0; i < 2; ++i) mbar_init(&aempty[i], 1);
        mbar_init(accfull, 1);
        mbar_init(done, 1);
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kF4TmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tb = *tmem_slot;
    // every block scale factor is 1 (ue8m0 0x7F): the first four converter warps fill their lane
    // quarter of the scale-factor columns of A and B
    if (warp >= kF4Conv0 && warp < kF4Conv0 + 4) {
        const uint32_t lq = tb + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        tmem_st8(lq + kF4ColSFA, 0x7F7F7F7Fu);
        tmem_st8(lq + kF4ColSFA + 8, 0x7F7F7F7Fu);
        tmem_st8(lq + kF4ColSFB, 0x7F7F7F7Fu);
        tmem_st8(lq + kF4ColSFB + 8, 0x7F7F7F7Fu);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // the next kernel in the stream may start launching (the next call's prep waits for this kernel's
    // completion before it reads or writes anything)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // Tiles are numbered T = 0, 1, .. over this CTA's ranges in order; each role keeps its ring
    // stages, phases and A slot (T mod 2) as running counters, and computes the rows of a range once
    // per range.
    if (warp == 0) {
        // ---------------------------------------------------------------- code producer
        if (lane == 0) {
            int T = 0, cs = 0;
            uint32_t cph = 0;
            bool ok = true;
            for (int ri = 0; ri < my_ranges && ok; ++ri) {
                int s0, s1;
                f4_range(static_cast<int>(blockIdx.x) + ri * static_cast<int>(gridDim.x), p.slices, p.ranges, s0, s1);
                // one box of code_bytes / 128 rows from the range's first row (rows past the range or
                // past m come along unused: zero-filled past m)
                for (int k = 0; k < p.tiles; ++k, ++T) {
                    // only the first tiles go out before the prep kernel completes: code copies from
                    // every SM queue the prep kernel's own memory traffic behind them. With the prep
                    // resident early (it overlaps the previous kernel) and the first two tiles stored
                    // before their digits are checked, eight tiles measured fastest (seven to ten alike,
                    // 0.9 us ahead of four)
                    if (T == kF4PreStages) asm volatile("griddepcontrol.wait;" ::: "memory");
                    if (T >= p.cstages && !mbar_wait_backoff(&cempty[cs], cph ^ 1, p.status)) { ok = false; break; }
                    mbar_arrive_expect_tx(&cfull[cs], p.code_bytes);
                    tma_load_2d(cring + static_cast<size_t>(cs) * p.code_bytes, &tmC, k * 128, s0 * kF4SliceRows,
                                &cfull[cs]);
                    if (++cs == p.cstages) { cs = 0; cph ^= 1; }
                }
            }
        }
    } else if (warp == kF4DigitWarp) {
        // ---------------------------------------------------------------- digit producer
        if (lane == 0) {
            asm volatile("griddepcontrol.wait;" ::: "memory");   // the prep kernel's digits are complete
            int T = 0, ds = 0;
            uint32_t dph = 0;
            bool ok = true;
            for (int ri = 0; ri < my_ranges && ok; ++ri) {
                for (int k = 0; k < p.tiles; ++k, ++T) {
                    if (T >= p.dstages && !mbar_wait_backoff(&dempty[ds], dph ^ 1, p.status)) { ok = false; break; }
                    uint8_t *dst = dring + static_cast<size_t>(ds) * p.act_bytes;
                    mbar_arrive_expect_tx(&dfull[ds], p.act_bytes);
                    tma_load_2d(dst, &tmB, 0, k * p.NB, &dfull[ds]);
                    tma_load_2d(dst + p.act_bytes / 2, &tmB, 128, k * p.NB, &dfull[ds]);
                    if (++ds == p.dstages) { ds = 0; dph ^= 1; }
                }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        // The whole warp runs the loop and one elected lane issues: warp-uniform control flow with the
        // tile's descriptors formed before its MMAs lets them issue back to back (about 24 cycles per
        // MMA at N = 32, measured, against about 64 for a divergent lane-0 branch).
        const uint32_t idesc = idesc_mxf4(128, p.NB);
        const uint32_t sfa = tb + kF4ColSFA, sfb = tb + kF4ColSFB;
        const uint64_t dbase = smem_desc_sw128(smem_u32(dring), 16, 1024);
        const uint64_t hstep = static_cast<uint64_t>(p.act_bytes >> 5);   // second 128-byte half: NB x 128 B
        const uint64_t astep = static_cast<uint64_t>(p.act_bytes >> 4);   // next digit stage
        int ds = 0, slot = 0;
        uint64_t bstage = dbase;
        for (int ri = 0; ri < my_ranges; ++ri) {
            int s0, s1;
            f4_range(static_cast<int>(blockIdx.x) + ri * static_cast<int>(gridDim.x), p.slices, p.ranges, s0, s1);
            const bool two = (s1 - s0) > 4;
            for (int k = 0; k < p.tiles; ++k) {
                named_sync(kF4BarAFull + slot, kF4BarAFullCount);
                tc_fence_after();
                const uint32_t a0 = tb + kF4ColA + static_cast<uint32_t>(slot * 128);
                const uint32_t acc0 = k > 0 ? 1u : 0u;
                uint64_t bd[8];
#pragma unroll
                for (int s = 0; s < 8; ++s) bd[s] = bstage + static_cast<uint64_t>(s >> 2) * hstep + static_cast<uint64_t>((s & 3) * 2);
                if (elect_one()) {
#pragma unroll
                    for (int s = 0; s < 8; ++s) umma_mxf4_ts(tb, a0 + 8 * s, bd[s], idesc, sfa, sfb, s ? 1u : acc0);
                    if (two) {
#pragma unroll
                        for (int s = 0; s < 8; ++s)
                            umma_mxf4_ts(tb + kF4ColD1, a0 + 64 + 8 * s, bd[s], idesc, sfa, sfb, s ? 1u : acc0);
                    }
                    umma_commit(&aempty[slot]);
                    umma_commit(&dempty[ds]);
                    if (k == p.tiles - 1) umma_commit(accfull);
                }
                __syncwarp();
                slot ^= 1;
                if (++ds == p.dstages) { ds = 0; bstage = dbase; } else { bstage += astep; }
            }
            // before the next range overwrites the accumulators, the epilogue has read them
            if (ri + 1 < my_ranges) named_sync(kF4BarDFree, kF4BarDFreeCount);
        }
        // every MMA of this thread has completed before the teardown frees tensor memory
        if (total_tiles > 0) {
            if (elect_one()) umma_commit(done);
            __syncwarp();
            if (lane == 0) mbar_wait(done, 0, p.status);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------------- converters and epilogue
        // Two teams of four warps take alternate tiles (team = T mod 2 = the A slot), so that one team
        // converts while the other's tile waits on its barrier; a warp converts its TMEM lane quarter's
        // rows of both 128-row blocks. In the epilogue, team t reads block t.
        const int ci = warp - kF4Conv0;
        const int q = warp & 3;                       // TMEM lane quarter this warp may access
        const int team = ci >> 2;
        const uint32_t lane_base = tb + (static_cast<uint32_t>(32 * q) << 16);
        const uint32_t a_base = lane_base + kF4ColA;
        bool ok = true;                               // false after a failed wait: no more waits
        int T = 0, cs = 0, ds = 0;
        uint32_t cph = 0, dph = 0;
        const int lrow0 = q * 32 + lane;              // row of block 0 within the range; block 1: + 128
        const uint8_t *crow = cring + lrow0 * 128;
        const int sw = lane & 7;                      // 128-byte swizzle phase of both rows
        for (int ri = 0; ri < my_ranges; ++ri) {
            int s0, s1;
            f4_range(static_cast<int>(blockIdx.x) + ri * static_cast<int>(gridDim.x), p.slices, p.ranges, s0, s1);
            // this warp's 32 rows of block rb belong to the range
            const bool live0 = q < (s1 - s0), live1 = (4 + q) < (s1 - s0);
            for (int k = 0; k < p.tiles; ++k, ++T) {
                if ((T & 1) == team) {
                    const int slot = T & 1;
                    ok = warp_wait(&cfull[cs], cph, ok, p.status);
                    uint4 v[2][8];
                    if (ok) {
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            if (live0) v[0][c] = *reinterpret_cast<const uint4 *>(crow + ((c ^ sw) << 4));
                            if (live1) v[1][c] = *reinterpret_cast<const uint4 *>(crow + 128 * 128 + ((c ^ sw) << 4));
                        }
                    }
                    // the code stage is free once every converter warp of the team has read its part
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&cempty[cs]);
                    // the slot is free once the MMAs of tile T - 2 completed (aempty phase (T / 2 + 1) mod 2);
                    // the digits are checked only before the barrier, so the first two tiles leave the
                    // code ring while the prep kernel still runs
                    if (T >= 2) ok = warp_wait(&aempty[slot], static_cast<uint32_t>(((T >> 1) + 1) & 1), ok, p.status);
                    tc_fence_after();
#pragma unroll
                    for (int rb = 0; rb < 2; ++rb) {
                        if (ok && (rb ? live1 : live0)) {
                            uint32_t f[2][32];
#pragma unroll
                            for (int c = 0; c < 8; ++c) {
                                const uint32_t w[4] = {v[rb][c].x, v[rb][c].y, v[rb][c].z, v[rb][c].w};
#pragma unroll
                                for (int u = 0; u < 4; ++u) {
                                    f[c >> 2][8 * (c & 3) + 2 * u] = w[u] & 0x33333333u;
                                    f[c >> 2][8 * (c & 3) + 2 * u + 1] = (w[u] >> 2) & 0x33333333u;
                                }
                            }
#pragma unroll
                            for (int h = 0; h < 2; ++h)
                                tmem_st32(a_base + static_cast<uint32_t>(slot * 128 + rb * 64 + h * 32), f[h]);
                        }
                    }
                    if (ok && (live0 || live1)) asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                    // the issuer reads the digits once the converters have seen them land
                    ok = warp_wait(&dfull[ds], dph, ok, p.status);
                    tc_fence_before();
                    named_sync(kF4BarAFull + slot, kF4BarAFullCount);
                }
                if (++cs == p.cstages) { cs = 0; cph ^= 1; crow = cring + lrow0 * 128; } else { crow += p.code_bytes; }
                if (++ds == p.dstages) { ds = 0; dph ^= 1; }
            }
            {
                // ------------------------------------------------------------ epilogue of the range
                const int rb = team;
                const bool live = rb ? live1 : live0;
                const int lrow = rb * 128 + lrow0;
                if (ri == 0) asm volatile("griddepcontrol.wait;" ::: "memory");   // scale and corr of the prep kernel
                // the token scales and bias terms are read while the range's last MMAs run
                float sc[kF4MaxTokens], co[kF4MaxTokens];
#pragma unroll
                for (int t = 0; t < kF4MaxTokens; ++t) {
                    sc[t] = t < p.ntok ? __ldg(p.scale + t) : 0.0f;
                    co[t] = t < p.ntok ? __ldg(p.corr + t) : 0.0f;
                }
                ok = warp_wait(accfull, ri & 1, ok, p.status);
                tc_fence_after();
                // column c of the accumulator is digit c % 5 of token c / 5: sum_j 8^j acc_j per token,
                // in increasing column order, 16 columns per load
                float y[kF4MaxTokens];
#pragma unroll
                for (int t = 0; t < kF4MaxTokens; ++t) y[t] = 0.0f;
                if (ok && live) {
#pragma unroll
                    for (int c0 = 0; c0 < kF4MaxTokens * kF4Digits; c0 += 16) {
                        if (c0 < p.NB) {
                            float v[16];
                            tmem_ld16(lane_base + (rb ? kF4ColD1 : 0u) + static_cast<uint32_t>(c0), v);
                            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                            for (int c = 0; c < 16; ++c) {
                                const int col = c0 + c;
                                const float w = col % 5 == 0 ? 1.0f : col % 5 == 1 ? 8.0f : col % 5 == 2 ? 64.0f
                                                : col % 5 == 3 ? 512.0f : 4096.0f;
                                y[col / 5] = fmaf(v[c], w, y[col / 5]);
                            }
                        }
                    }
                }
                tc_fence_before();
                if (ri + 1 < my_ranges) named_arrive(kF4BarDFree, kF4BarDFreeCount);
                const int64_t grow = static_cast<int64_t>(s0) * kF4SliceRows + lrow;
                if (ok && live && grow < p.m) {
#pragma unroll
                    for (int t = 0; t < kF4MaxTokens; ++t) {
                        if (t < p.ntok) {
                            const float yt = fmaf(y[t], sc[t], co[t]);
                            const __nv_bfloat16 h = __float2bfloat16_rn(yt);
                            p.Y[static_cast<int64_t>(t) * p.m + grow] = *reinterpret_cast<const uint16_t *>(&h);
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tb, kF4TmemCols);
    }
}

// ---------------------------------------------------------------------------------- host side

struct F4Plan {
    int tiles, NB, slices, ranges, grid, cstages, dstages;
    uint32_t code_bytes, act_bytes;
    size_t smem;
};

bool f4_plan(int64_t N, int64_t m, int64_t n, int num_sms, F4Plan &pl) {
    if (N < 1 || N > kF4MaxTokens || m < 1 || n < 64 || n % 64 != 0) return false;
    if (n > static_cast<int64_t>(kF4PrepThreads) * kF4PrepGroups * 16) return false;   // prep keeps X' in registers
    pl.tiles = static_cast<int>((n + kF4TileCols - 1) / kF4TileCols);
    pl.NB = f4_nb(static_cast<int>(N));
    const int64_t slices = (m + kF4SliceRows - 1) / kF4SliceRows;
    if (slices > (int64_t(1) << 30)) return false;
    pl.slices = static_cast<int>(slices);
    // one SM per prep CTA is left to the prep kernel: its CTAs (one per token) cannot share an SM with
    // a CTA of this kernel, which would otherwise start only after them and finish last
    const int64_t G = num_sms > 2 * N ? num_sms - N : (num_sms > 0 ? num_sms : 1);
    const int64_t waves = (slices + kF4MaxSlices * G - 1) / (kF4MaxSlices * G);
    pl.ranges = static_cast<int>(slices < G * waves ? slices : G * waves);
    pl.grid = static_cast<int>(pl.ranges < G ? pl.ranges : G);
    const int max_slices = (pl.slices + pl.ranges - 1) / pl.ranges;
    pl.code_bytes = static_cast<uint32_t>(max_slices) * 4096u;
    pl.act_bytes = static_cast<uint32_t>(pl.NB) * 256u;
    // as many code stages as fit next to up to four digit stages (at least kF4MinCodeStages code
    // stages while there are more than two digit stages)
    const size_t fixed = 1024 + 1024;   // barriers and the TMEM slot; alignment slack
    auto code_stages = [&](int d) {
        const size_t rest = kF4SmemLimit - fixed - static_cast<size_t>(d) * pl.act_bytes;
        const size_t c = rest / pl.code_bytes;
        return static_cast<int>(c < static_cast<size_t>(kF4CodeStagesMax) ? c : kF4CodeStagesMax);
    };
    pl.dstages = kF4DigitStagesMax;
    pl.cstages = code_stages(pl.dstages);
    while (pl.cstages < kF4MinCodeStages && pl.dstages > 2) pl.cstages = code_stages(--pl.dstages);
    if (pl.cstages < 2) return false;
    pl.smem = static_cast<size_t>(pl.cstages) * pl.code_bytes + static_cast<size_t>(pl.dstages) * pl.act_bytes + fixed;
    // at least half the shared memory, so one CTA per SM owns all 512 tensor-memory columns
    if (pl.smem < kF4SmemMin) pl.smem = kF4SmemMin;
    return pl.smem <= kF4SmemLimit;
}

size_t f4_digits_bytes(int64_t N, int64_t n) {
    const int64_t tiles = (n + kF4TileCols - 1) / kF4TileCols;
    return static_cast<size_t>(tiles) * static_cast<size_t>(f4_nb(static_cast<int>(N))) * 256u;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool f4_map_u8(CUtensorMap *map, const void *ptr, uint64_t inner, uint64_t outer, uint32_t box_inner,
               uint32_t box_outer) {
    void *fnp = tensor_map_encoder();
    if (!fnp) return false;
    auto enc = reinterpret_cast<EncodeTiledFn>(fnp);
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {inner};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(ptr), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

size_t packed_gemv_fp4_workspace(int64_t N, int64_t n) {
    if (N < 1 || N > kF4MaxTokens) return 0;
    return ((f4_digits_bytes(N, n) + 255) / 256) * 256 + 256;
}

bool launch_packed_gemv_fp4(const PackedGemvArgs &a, int d, int num_sms, cudaStream_t st, cudaError_t &err) {
    err = cudaSuccess;
    F4Plan pl;
    if (!f4_plan(a.N, a.m, a.n, num_sms, pl)) return false;
    uint8_t *dig = reinterpret_cast<uint8_t *>(a.Xp);
    float *scale = reinterpret_cast<float *>(dig + ((f4_digits_bytes(a.N, a.n) + 255) / 256) * 256);
    float *corr = scale + kF4MaxTokens;

    CUtensorMap mc, mb;
    if (!f4_map_u8(&mc, a.packed, static_cast<uint64_t>(a.n / 4), static_cast<uint64_t>(a.m), 128, pl.code_bytes / 128) ||
        !f4_map_u8(&mb, dig, 256, static_cast<uint64_t>(pl.tiles) * static_cast<uint64_t>(pl.NB), 128,
                   static_cast<uint32_t>(pl.NB))) {
        err = cudaErrorInvalidValue;
        return true;
    }
    using PrepFn = void (*)(const void *, int64_t, int, int, int, const float *, const float *, uint8_t *, float *,
                            float *, int);
    PrepFn prep = a.rotate ? (d == 4 ? fp4_prep_kernel<4, false, true> : fp4_prep_kernel<8, false, true>)
                  : a.Xf   ? (d == 4 ? fp4_prep_kernel<4, true, false> : fp4_prep_kernel<8, true, false>)
                           : (d == 4 ? fp4_prep_kernel<4, false, false> : fp4_prep_kernel<8, false, false>);
    int lb = 0;
    size_t prep_smem = 0;
    if (a.rotate) {
        // n % 64 == 0 and n <= 32768 (the plan), so the block is 2^6 .. 2^15 columns
        while ((a.n >> (lb + 1)) << (lb + 1) == a.n && lb < 15) ++lb;
        prep_smem = lb > 9 ? static_cast<size_t>(a.n) * sizeof(float) : 0;
        if (prep_smem) {
            err = ensure_dynamic_smem(reinterpret_cast<const void *>(prep), static_cast<int>(prep_smem));
            if (err != cudaSuccess) return true;
        }
    }
    {
        // a programmatic dependent of the previous kernel in the stream: it may become resident on the
        // SMs this kernel's grid leaves free while that kernel still runs, and waits for it on the device
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(a.N));
        cfg.blockDim = dim3(kF4PrepThreads);
        cfg.dynamicSmemBytes = prep_smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        err = cudaLaunchKernelEx(&cfg, prep, a.Xf ? static_cast<const void *>(a.Xf) : static_cast<const void *>(a.X),
                                 a.n, pl.tiles, static_cast<int>(a.N), pl.NB, a.A, a.b, dig, scale, corr, lb);
        count_launch();
        if (err == cudaSuccess) err = cudaGetLastError();
        if (err != cudaSuccess) return true;
    }

    F4Params p;
    p.m = a.m;
    p.slices = pl.slices;
    p.ranges = pl.ranges;
    p.tiles = pl.tiles;
    p.ntok = static_cast<int>(a.N);
    p.NB = pl.NB;
    p.cstages = pl.cstages;
    p.dstages = pl.dstages;
    p.code_bytes = pl.code_bytes;
    p.act_bytes = pl.act_bytes;
    p.scale = scale;
    p.corr = corr;
    p.Y = a.Y;
    p.status = a.status;
    err = ensure_dynamic_smem(reinterpret_cast<const void *>(packed_gemv_fp4_kernel), static_cast<int>(pl.smem));
    if (err != cudaSuccess) return true;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(pl.grid));
    cfg.blockDim = dim3(kF4Threads);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    err = cudaLaunchKernelEx(&cfg, packed_gemv_fp4_kernel, mc, mb, p);
    count_launch();
    if (err == cudaSuccess) err = cudaGetLastError();
    return true;
}

}  // namespace lcq
