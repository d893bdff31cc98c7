// HBM-bound element-wise kernels of the LC-VQ layer:
//   encode         W -> latent u = A^{-1}(W_g - b), codes clip(round(u),0,3), MSE   (Sec. 2.2)
//   quant_decode   P -> Z = clip(round(P/s + t),0,3) packed, W_hat = A Z_g + b bf16 (Eq. quant_param, def:forward)
//   decode         packed Z -> W_hat fp32 / bf16                                      (Eq. def:forward)
//   pack2b         one code per byte -> 4 codes per byte
//   reduce_partials  fixed-order sum of per-CTA dA/db partials
//
// encode and quant_decode stream their fp32 input through a shared-memory ring
// filled by the bulk-copy (TMA) engine: one producer thread issues 33 KB
// cp.async.bulk copies, eleven compute warps consume them. In encode, thread t takes
// the groups t, t + T, ... of a chunk (conflict-free shared-memory reads); in quant_decode
// each compute thread owns 24 consecutive weights, i.e. whole groups for d = 4 and 8.
#include "common.cuh"
#include "internal.h"
#include "invert.cuh"

namespace lcq {

// Encode is bound by its FMA-pipe issue at three warps per SM sub-partition (four would cap the
// registers at 128): three groups of 8 weights per thread and stage measured faster than two
// (encode with the MSE 0.722 against 0.750 ms on the Llama-3-70B layer) and than four, and so did
// these warps against 15 compute warps at one or two groups each.
constexpr int kComputeWarps = 11;                                // + 1 producer = 12 warps, 3 per SM sub-partition
constexpr int kPerThread = 24;                                   // weights per compute thread per stage
constexpr int kChunk = 32 * kComputeWarps * kPerThread;          // fp32 weights per stage (33 KB)
constexpr int kStreamStages = 6;                                 // 198 KB ring (single-matrix kernels)
constexpr int kBatchStages = 5;                                  // 165 KB ring (batched encode)
constexpr int kStreamThreads = 32 * (1 + kComputeWarps);
static_assert(kPerThread % 8 == 0, "a compute thread's weights are whole 8-weight groups (16-byte stores)");
constexpr float kRoundMagic = 12582912.0f;                       // 1.5 * 2^23

struct StreamSmem {
    float buf[kStreamStages][kChunk];
    uint64_t full[kStreamStages];
    uint64_t empty[kStreamStages];
    float Ainv[64];
    float A[64];
    float M[64];        // A^T A (encode MSE)
    float b[8];
    double gj[8][16];   // fp64 elimination (fallback)
    float gjf[8][16];   // Newton iterate X (columns 0..d-1) and residual R (columns d..2d-1)
    double dred[kComputeWarps];
    int singular;
};

__device__ __forceinline__ void compute_bar() {
    asm volatile("bar.sync 1, %0;" ::"r"(32 * kComputeWarps) : "memory");
}

// Producer loop (one thread): stream chunks blockIdx.x, +gridDim.x, ... of `src`.
__device__ void stream_producer(StreamSmem &s, const float *src, int64_t total, int32_t *status) {
    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    int i = 0;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++i) {
        const int st = i % kStreamStages;
        const uint32_t ph = (i / kStreamStages) & 1;
        if (!mbar_wait(&s.empty[st], ph ^ 1, status)) return;
        const int64_t base = c * kChunk;
        const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
        const uint32_t bytes = static_cast<uint32_t>(cnt * 4);
        mbar_arrive_expect_tx(&s.full[st], bytes);
        bulk_g2s(s.buf[st], src + base, bytes, &s.full[st]);
    }
}

// ------------------------------------------------------------------ encode
//
// Per group (d weights): v = w - b; u = A^{-1} v (packed fp32x2 FMAs over pairs of rows of A^{-1});
// z = clip(round_half_even(u), 0, 3) taken on the fp32 pipe: t = u + 1.5*2^23 rounds u to an
// integer (round to nearest even), clamping t to [1.5*2^23, 1.5*2^23 + 3] clamps the integer,
// whose value is then the low two bits of t (NaN -> 0: fmaxf drops the NaN).
// Squared residual ||w - (A z + b)||^2 = ||A (u - z)||^2 = e^T (A^T A) e with e = u - z.

// Insert the two low bits of `src` (the code: tc = 1.5*2^23 + z) into `dst` at bit `pos` (ALU pipe).
__device__ __forceinline__ uint32_t bfi2(uint32_t src, uint32_t dst, int pos) {
    uint32_t r;
    asm("bfi.b32 %0, %1, %2, %3, 2;" : "=r"(r) : "r"(src), "r"(dst), "r"(pos));
    return r;
}

// Upper triangle of M = A^T A in the order the paired quadratic form consumes it (see quad_form).
template <int D>
struct QuadCoef {
    float2 pair[D * D / 4];   // (Mu[i][j], Mu[i+1][j]) for even i, j = i+1..D-1
    float diag[D / 2];        // Mu[i][i] for even i
};

// q = e^T M e = sum_i e_i s_i with s_i = M_ii e_i + 2 sum_{j>i} M_ij e_j, rows taken in pairs (i, i+1) so
// that every column j > i feeds both rows with one packed fp32x2 FMA.
template <int D>
__device__ __forceinline__ float quad_form(const QuadCoef<D> &c, const float (&e)[D]) {
    float2 eb[D];
#pragma unroll
    for (int j = 0; j < D; ++j) eb[j] = make_float2(e[j], e[j]);
    float2 q2 = make_float2(0.0f, 0.0f);
    int idx = 0;
#pragma unroll
    for (int i = 0; i < D; i += 2) {
        float2 s2 = make_float2(c.diag[i / 2] * e[i], 0.0f);
#pragma unroll
        for (int j = i + 1; j < D; ++j) s2 = __ffma2_rn(c.pair[idx++], eb[j], s2);
        q2 = __ffma2_rn(make_float2(e[i], e[i + 1]), s2, q2);
    }
    return q2.x + q2.y;
}

template <int D, bool kMse>
__device__ __forceinline__ void encode_group(const float *w, const float2 (&Ai2)[D / 2][D], const QuadCoef<D> &qc,
                                             const float2 (&c2)[D / 2], uint32_t &zacc, int zshift, float (&u)[D],
                                             float &sq) {
    // u = A^{-1} w + c with c = -A^{-1} b
    float2 u2[D / 2];
#pragma unroll
    for (int kp = 0; kp < D / 2; ++kp) {
        float2 acc = c2[kp];
#pragma unroll
        for (int j = 0; j < D; ++j) acc = __ffma2_rn(Ai2[kp][j], make_float2(w[j], w[j]), acc);
        u2[kp] = acc;
        u[2 * kp] = acc.x;
        u[2 * kp + 1] = acc.y;
    }
    float e[D];
#pragma unroll
    for (int kp = 0; kp < D / 2; ++kp) {
        const float2 t = __fadd2_rn(u2[kp], make_float2(kRoundMagic, kRoundMagic));
        const float tc0 = fminf(fmaxf(t.x, kRoundMagic), kRoundMagic + 3.0f);
        const float tc1 = fminf(fmaxf(t.y, kRoundMagic), kRoundMagic + 3.0f);
        zacc = bfi2(__float_as_uint(tc0), zacc, zshift + 4 * kp);
        zacc = bfi2(__float_as_uint(tc1), zacc, zshift + 4 * kp + 2);
        if (kMse) {
            const float2 zf = __fadd2_rn(make_float2(tc0, tc1), make_float2(-kRoundMagic, -kRoundMagic));
            const float2 ee = __ffma2_rn(zf, make_float2(-1.0f, -1.0f), u2[kp]);
            e[2 * kp] = ee.x;
            e[2 * kp + 1] = ee.y;
        }
    }
    if (kMse) sq += quad_form<D>(qc, e);
}

// The per-thread copy of a matrix's encode constants: A^{-1} as row pairs (columns swapped for the
// threads that read the halves of their groups swapped), c = -A^{-1} b, and the quadratic-form
// coefficients of A^T A.
template <int D>
__device__ __forceinline__ void load_encode_constants(const float *Ainv, const float *M, const float *b, int hswap,
                                                      float2 (&Ai2)[D / 2][D], float2 (&c2)[D / 2], QuadCoef<D> &qc) {
#pragma unroll
    for (int kp = 0; kp < D / 2; ++kp)
#pragma unroll
        for (int j = 0; j < D; ++j) {
            const int jc = j ^ (4 * hswap);
            Ai2[kp][j] = make_float2(Ainv[(2 * kp) * D + jc], Ainv[(2 * kp + 1) * D + jc]);
        }
#pragma unroll
    for (int kp = 0; kp < D / 2; ++kp) {
        float c0 = 0.0f, c1 = 0.0f;
#pragma unroll
        for (int j = 0; j < D; ++j) {
            c0 = fmaf(-Ainv[(2 * kp) * D + j], b[j], c0);
            c1 = fmaf(-Ainv[(2 * kp + 1) * D + j], b[j], c1);
        }
        c2[kp] = make_float2(c0, c1);
    }
    int idx = 0;
#pragma unroll
    for (int i = 0; i < D; i += 2) {
        qc.diag[i / 2] = M[i * D + i];
        // row i gets 2*M[i][j] for j > i; row i+1 gets M[i+1][i+1] at j = i+1, 2*M[i+1][j] beyond
#pragma unroll
        for (int j = i + 1; j < D; ++j)
            qc.pair[idx++] = make_float2(2.0f * M[i * D + j], (j == i + 1 ? 1.0f : 2.0f) * M[(i + 1) * D + j]);
    }
}

// Encode one chunk held in shared memory (cnt weights starting at flat index base of a matrix).
// Thread t encodes the groups t, t + T, ... of the chunk (T compute threads), so consecutive threads
// read consecutive groups. For d = 8 a group is two 16-byte units; threads with bit 2 of t set read
// the second unit first, which puts the eight 16-byte reads of a quarter warp in distinct banks (their
// constants were loaded with the columns swapped to match).
template <int D, bool kMse>
__device__ __forceinline__ void encode_chunk(const float *buf, int64_t base, int64_t cnt, int t, int hswap,
                                             const float2 (&Ai2)[D / 2][D], const QuadCoef<D> &qc,
                                             const float2 (&c2)[D / 2], uint8_t *packed, uint8_t *codes, float *latent,
                                             float &sq) {
    constexpr int kGroupsPerThread = kPerThread / D;
    constexpr int kThreads = 32 * kComputeWarps;
    const int ngroups = static_cast<int>(cnt / D);   // n % 8 == 0: whole groups
#pragma unroll
    for (int k = 0; k < kGroupsPerThread; ++k) {
        const int g = t + k * kThreads;
        if (g < ngroups) {
            const float4 *src = reinterpret_cast<const float4 *>(buf + g * D);
            float w[D];
            if (D == 8) {
                const float4 f0 = src[hswap], f1 = src[1 - hswap];
                w[0] = f0.x; w[1] = f0.y; w[2] = f0.z; w[3] = f0.w;
                w[4] = f1.x; w[5] = f1.y; w[6] = f1.z; w[7] = f1.w;
            } else {
                const float4 f0 = src[0];
                w[0] = f0.x; w[1] = f0.y; w[2] = f0.z; w[3] = f0.w;
            }
            float u[D];
            float gsq = 0.0f;
            uint32_t p = 0;
            encode_group<D, kMse>(w, Ai2, qc, c2, p, 0, u, gsq);
            sq += gsq;
            const int64_t gidx = base + static_cast<int64_t>(g) * D;   // flat index of the group's first weight
            if (packed) {
                if (D == 8) *reinterpret_cast<uint16_t *>(packed + gidx / 4) = static_cast<uint16_t>(p);
                else packed[gidx / 4] = static_cast<uint8_t>(p);
            }
            if (codes) {
                uint32_t ww[D / 4];
#pragma unroll
                for (int q = 0; q < D / 4; ++q) {
                    const uint32_t f = (p >> (8 * q)) & 0xFFu;
                    ww[q] = (f & 3u) | (((f >> 2) & 3u) << 8) | (((f >> 4) & 3u) << 16) | (((f >> 6) & 3u) << 24);
                }
                if (D == 8) *reinterpret_cast<uint2 *>(codes + gidx) = make_uint2(ww[0], ww[D / 4 - 1]);
                else *reinterpret_cast<uint32_t *>(codes + gidx) = ww[0];
            }
            if (latent) {
                float4 *dst = reinterpret_cast<float4 *>(latent + gidx);
#pragma unroll
                for (int q = 0; q < D / 4; ++q) dst[q] = make_float4(u[4 * q], u[4 * q + 1], u[4 * q + 2], u[4 * q + 3]);
            }
        }
    }
}


// End of a matrix's share of a CTA: the compute threads' sums of squared residuals become one
// per-CTA partial (fixed order); the CTA that arrives last (counter wraps back to zero, atomicInc)
// sums the partials in a fixed order and writes the mean. All compute warps call it together; dred
// must not be reused until every compute warp has passed the next compute_bar.
__device__ __forceinline__ void mse_flush(float &sq, double *dred, double *partials, unsigned *counter, double *mse,
                                          int64_t total) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
    if (lane == 0) dred[warp - 1] = static_cast<double>(sq);
    sq = 0.0f;
    compute_bar();
    if (warp == 1) {
        unsigned prev = 0;
        if (lane == 0) {
            double acc = 0.0;
            for (int w = 0; w < kComputeWarps; ++w) acc += dred[w];
            partials[blockIdx.x] = acc;
            __threadfence();
            prev = atomicInc(counter, gridDim.x - 1);
        }
        prev = __shfl_sync(0xffffffffu, prev, 0);
        if (prev == gridDim.x - 1) {
            __threadfence();
            double tot = 0.0;
            for (unsigned q = lane; q < gridDim.x; q += 32) tot += __ldcg(partials + q);
            for (int o = 16; o; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
            if (lane == 0 && mse) *mse = total > 0 ? tot / static_cast<double>(total) : 0.0;
        }
    }
}

template <int D, bool kMse, bool kLatent>
__global__ void __launch_bounds__(kStreamThreads, 1)
encode_kernel(EncodeArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    StreamSmem &s = *reinterpret_cast<StreamSmem *>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t total = a.m * a.n;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStreamStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kComputeWarps);
        }
        fence_barrier_init();
    }
    if (threadIdx.x < D * D) s.A[threadIdx.x] = a.A[threadIdx.x];
    if (threadIdx.x < D) s.b[threadIdx.x] = a.b[threadIdx.x];
    __syncthreads();
    if (a.pdl & 1) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp == 0) {
        if (lane == 0) stream_producer(s, a.W, total, a.status);
        if (a.pdl & 2) asm volatile("griddepcontrol.wait;" ::: "memory");
        return;
    }
    // compute warps
    if (warp == 1) invert_warp<D>(s);
    compute_bar();
    if (s.singular && blockIdx.x == 0 && threadIdx.x == 32) set_status(a.status, LCQ_ERR_SINGULAR);

    const int t = threadIdx.x - 32;
    const int hswap = (D == 8) ? ((t >> 2) & 1) : 0;
    float2 Ai2[D / 2][D], c2[D / 2];
    QuadCoef<D> qc;
    load_encode_constants<D>(s.Ainv, s.M, s.b, hswap, Ai2, c2, qc);

    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    float sq = 0.0f;
    int i = 0;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++i) {
        const int st = i % kStreamStages;
        if (!mbar_wait(&s.full[st], (i / kStreamStages) & 1, a.status)) break;
        const int64_t base = c * kChunk;
        const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
        encode_chunk<D, kMse>(s.buf[st], base, cnt, t, hswap, Ai2, qc, c2, a.packed, a.codes,
                              kLatent ? a.latent : nullptr, sq);
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[st]);
    }
    if (kMse) mse_flush(sq, s.dred, a.partials, a.counter, a.mse, total);
    if (a.pdl & 2) asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ------------------------------------------------------------------ batched encode (codes, latents)
//
// Several matrices (same d) in one persistent launch: their chunks form one list, streamed through
// the ring in order; CTA b takes chunks b, b + G, ... of the list (G CTAs), so it visits the matrices in
// order. Compute warp w forms A^{-1} of matrices w - 1, w - 1 + kComputeWarps, ... in parallel. Used
// when no matrix asks for the MSE (see launch_encode_batch).

struct InvSlot {
    float A[64];
    float Ainv[64];
    float M[64];
    float b[8];
    float gjf[8][16];
    double gj[8][16];
    int singular;
};

struct EncBatchSmem {
    float buf[kBatchStages][kChunk];
    uint64_t full[kBatchStages];
    uint64_t empty[kBatchStages];
    InvSlot inv[kEncodeBatchMax];
};

__device__ __forceinline__ int batch_item_of(const EncodeBatchArgs &a, int64_t c, int from) {
    int j = from;
    while (j + 1 < a.count && c >= a.item[j + 1].chunk0) ++j;
    return j;
}

// One matrix of a batched encode, for one CTA: its constants and its chunks (the sequence the
// producer streams).
template <int D, bool kLatent>
__device__ __forceinline__ void encode_batch_matrix(EncBatchSmem &s, const EncodeBatchArgs &a, int j, int &it, bool &ok) {
    const int lane = threadIdx.x & 31;
    const int t = threadIdx.x - 32;
    const int hswap = (D == 8) ? ((t >> 2) & 1) : 0;
    float2 Ai2[D / 2][D], c2[D / 2];
    QuadCoef<D> qc;
    float sq = 0.0f;
    const int64_t chunk0 = a.item[j].chunk0, chunk1 = chunk0 + a.item[j].nchunks;
    const int64_t total = a.item[j].m * a.item[j].n;
    // this CTA's first chunk of matrix j: the first c >= chunk0 with c = blockIdx.x (mod gridDim.x)
    const int64_t G = gridDim.x;
    const int64_t first = chunk0 + ((static_cast<int64_t>(blockIdx.x) - chunk0) % G + G) % G;
    if (first < chunk1) {
        load_encode_constants<D>(s.inv[j].Ainv, s.inv[j].M, s.inv[j].b, hswap, Ai2, c2, qc);
        uint8_t *const packed = a.item[j].packed;
        uint8_t *const codes = a.item[j].codes;
        float *const latent = kLatent ? a.item[j].latent : nullptr;
        for (int64_t c = first; c < chunk1 && ok; c += G, ++it) {
            const int st = it % kBatchStages;
            if (!mbar_wait(&s.full[st], (it / kBatchStages) & 1, a.status)) { ok = false; break; }
            const int64_t base = (c - chunk0) * kChunk;
            const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
            encode_chunk<D, false>(s.buf[st], base, cnt, t, hswap, Ai2, qc, c2, packed, codes, latent, sq);
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[st]);
        }
    }
}

template <int D, bool kLatent>
__global__ void __launch_bounds__(kStreamThreads, 1)
encode_batch_kernel(const __grid_constant__ EncodeBatchArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    EncBatchSmem &s = *reinterpret_cast<EncBatchSmem *>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kBatchStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kComputeWarps);
        }
        fence_barrier_init();
    }
    for (int e = threadIdx.x; e < a.count * (D * D + D); e += blockDim.x) {
        const int j = e / (D * D + D), r = e % (D * D + D);
        if (r < D * D) s.inv[j].A[r] = a.item[j].A[r];
        else s.inv[j].b[r - D * D] = a.item[j].b[r - D * D];
    }
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) {
            int it = 0, j = -1;
            int64_t next0 = 0, chunk0 = 0, total = 0;
            const float *W = nullptr;
            for (int64_t c = blockIdx.x; c < a.total_chunks; c += gridDim.x, ++it) {
                if (c >= next0) {   // this chunk belongs to a later matrix: cache its fields
                    j = batch_item_of(a, c, j < 0 ? 0 : j);
                    chunk0 = a.item[j].chunk0;
                    total = a.item[j].m * a.item[j].n;
                    W = a.item[j].W;
                    next0 = j + 1 < a.count ? a.item[j + 1].chunk0 : a.total_chunks;
                }
                const int st = it % kBatchStages;
                if (!mbar_wait(&s.empty[st], ((it / kBatchStages) & 1) ^ 1, a.status)) return;
                const int64_t base = (c - chunk0) * kChunk;
                const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
                const uint32_t bytes = static_cast<uint32_t>(cnt * 4);
                mbar_arrive_expect_tx(&s.full[st], bytes);
                bulk_g2s(s.buf[st], W + base, bytes, &s.full[st]);
            }
        }
        return;
    }
    // compute warps: every matrix's A^{-1}, one matrix per warp at a time
    for (int j = warp - 1; j < a.count; j += kComputeWarps) invert_warp<D>(s.inv[j]);
    compute_bar();
    if (blockIdx.x == 0 && threadIdx.x == 32) {
        for (int j = 0; j < a.count; ++j)
            if (s.inv[j].singular) set_status(a.status, LCQ_ERR_SINGULAR);
    }

    int it = 0;   // position in this CTA's chunk sequence (ring stage and phase), continued across matrices
    bool ok = true;
    for (int j = 0; j < a.count; ++j) encode_batch_matrix<D, kLatent>(s, a, j, it, ok);
}

// ------------------------------------------------------------------ quantize + decode (forward prologue)

template <int D>
__global__ void __launch_bounds__(kStreamThreads, 1)
quant_decode_kernel(QuantDecodeArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    StreamSmem &s = *reinterpret_cast<StreamSmem *>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t total = a.m * a.n;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStreamStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kComputeWarps);
        }
        fence_barrier_init();
    }
    __syncthreads();
    if (warp == 0) {
        if (lane == 0) stream_producer(s, a.P, total, a.status);
        return;
    }
    float Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) Am[i] = __ldg(a.A + i);
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = __ldg(a.b + i);
    const float inv_s = a.inv_s, tt = a.t;

    const int t = threadIdx.x - 32;
    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    int i = 0;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++i) {
        const int st = i % kStreamStages;
        if (!mbar_wait(&s.full[st], (i / kStreamStages) & 1, a.status)) break;
        const int64_t base = c * kChunk;
        const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
        const int64_t off = static_cast<int64_t>(t) * kPerThread;
        if (off < cnt) {
            const int valid = static_cast<int>((cnt - off) < kPerThread ? (cnt - off) : kPerThread);
            const float *src = s.buf[st] + off;
            uint32_t z[kPerThread];
            float wh[kPerThread];
#pragma unroll
            for (int q = 0; q < kPerThread / 4; ++q) {
                const float4 f = (q * 4 < valid) ? reinterpret_cast<const float4 *>(src)[q] : make_float4(0, 0, 0, 0);
                z[4 * q + 0] = round_clamp3(__fadd_rn(__fmul_rn(f.x, inv_s), tt));
                z[4 * q + 1] = round_clamp3(__fadd_rn(__fmul_rn(f.y, inv_s), tt));
                z[4 * q + 2] = round_clamp3(__fadd_rn(__fmul_rn(f.z, inv_s), tt));
                z[4 * q + 3] = round_clamp3(__fadd_rn(__fmul_rn(f.w, inv_s), tt));
            }
#pragma unroll
            for (int g = 0; g < kPerThread / D; ++g) {
#pragma unroll
                for (int j = 0; j < D; ++j) {
                    float acc = bv[j];
#pragma unroll
                    for (int k = 0; k < D; ++k) acc = fmaf(Am[j * D + k], static_cast<float>(z[g * D + k]), acc);
                    wh[g * D + j] = acc;
                }
            }
            const int64_t gidx = base + off;
            if (valid == kPerThread) {
                // gidx is a multiple of 8 (kChunk and kPerThread are): 16-bit words of packed codes at
                // an even byte offset, 16-byte runs of bf16
                if (a.packed) {
                    uint16_t *pk = reinterpret_cast<uint16_t *>(a.packed + gidx / 4);
#pragma unroll
                    for (int h = 0; h < kPerThread / 8; ++h) {
                        uint32_t p = 0;
#pragma unroll
                        for (int k = 0; k < 8; ++k) p |= z[8 * h + k] << (2 * k);
                        pk[h] = static_cast<uint16_t>(p);
                    }
                }
                uint4 *dst = reinterpret_cast<uint4 *>(a.W_hat + gidx);
#pragma unroll
                for (int q = 0; q < kPerThread / 8; ++q)
                    dst[q] = make_uint4(pack_bf16x2(wh[8 * q], wh[8 * q + 1]), pack_bf16x2(wh[8 * q + 2], wh[8 * q + 3]),
                                        pack_bf16x2(wh[8 * q + 4], wh[8 * q + 5]), pack_bf16x2(wh[8 * q + 6], wh[8 * q + 7]));
            } else {
#pragma unroll
                for (int k = 0; k < kPerThread; k += 4) {
                    if (k < valid) {
                        if (a.packed)
                            a.packed[(gidx + k) / 4] =
                                static_cast<uint8_t>(z[k] | (z[k + 1] << 2) | (z[k + 2] << 4) | (z[k + 3] << 6));
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const __nv_bfloat16 h = __float2bfloat16_rn(wh[k + e]);
                            a.W_hat[gidx + k + e] = *reinterpret_cast<const uint16_t *>(&h);
                        }
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[st]);
    }
}

// ------------------------------------------------------------------ decode

// One group of d weights per lane, so that a warp's store of its 32 groups is one contiguous run
// (512 bytes of bf16 at d = 8): W_hat = A z + b with packed fp32x2 FMAs (rows 2jp, 2jp + 1 of A per
// pair, k in order from b: the plain sum's rounding); a code becomes an exact float as (2^23 + z) - 2^23,
// its bits OR-ed into 2^23's mantissa. Each lane keeps kDecGroups groups' codes in flight.
constexpr int kDecGroups = 8;

template <int D>
__device__ __forceinline__ void decode_group(uint32_t codes, const float2 (&A2)[D / 2][D], const float2 (&b2)[D / 2],
                                             float (&wh)[D]) {
    float z[D];
#pragma unroll
    for (int k = 0; k < D; ++k) z[k] = __uint_as_float(0x4B000000u | ((codes >> (2 * k)) & 3u)) - 8388608.0f;
#pragma unroll
    for (int jp = 0; jp < D / 2; ++jp) {
        float2 acc = b2[jp];
#pragma unroll
        for (int k = 0; k < D; ++k) acc = __ffma2_rn(A2[jp][k], make_float2(z[k], z[k]), acc);
        wh[2 * jp] = acc.x;
        wh[2 * jp + 1] = acc.y;
    }
}

template <int D>
__global__ void __launch_bounds__(256)
decode_kernel(DecodeArgs a) {
    float2 A2[D / 2][D], b2[D / 2];
#pragma unroll
    for (int jp = 0; jp < D / 2; ++jp) {
#pragma unroll
        for (int k = 0; k < D; ++k) A2[jp][k] = make_float2(__ldg(a.A + (2 * jp) * D + k), __ldg(a.A + (2 * jp + 1) * D + k));
        b2[jp] = make_float2(__ldg(a.b + 2 * jp), __ldg(a.b + 2 * jp + 1));
    }
    const int64_t ngroups = a.m * a.n / D;            // n % d == 0: whole groups
    const int lane = threadIdx.x & 31;
    const int64_t warp0 = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
    const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    constexpr int64_t kSpan = 32 * kDecGroups;         // groups a warp takes per iteration
    for (int64_t g0 = warp0 * kSpan; g0 < ngroups; g0 += nwarps * kSpan) {
        uint32_t cw[kDecGroups];
#pragma unroll
        for (int i = 0; i < kDecGroups; ++i) {
            const int64_t g = g0 + i * 32 + lane;
            cw[i] = 0;
            if (g < ngroups) {
                if (D == 8) cw[i] = __ldg(reinterpret_cast<const uint16_t *>(a.packed) + g);
                else cw[i] = __ldg(a.packed + g);
            }
        }
#pragma unroll
        for (int i = 0; i < kDecGroups; ++i) {
            const int64_t g = g0 + i * 32 + lane;
            if (g >= ngroups) continue;
            float wh[D];
            decode_group<D>(cw[i], A2, b2, wh);
            if (a.W_f32) {
                float4 *dst = reinterpret_cast<float4 *>(a.W_f32 + g * D);
#pragma unroll
                for (int q = 0; q < D / 4; ++q) dst[q] = make_float4(wh[4 * q], wh[4 * q + 1], wh[4 * q + 2], wh[4 * q + 3]);
            }
            if (a.W_bf16) {
                if (D == 8) {
                    *reinterpret_cast<uint4 *>(a.W_bf16 + g * D) =
                        make_uint4(pack_bf16x2(wh[0], wh[1]), pack_bf16x2(wh[2], wh[3]), pack_bf16x2(wh[4], wh[5]),
                                   pack_bf16x2(wh[6], wh[7]));
                } else {
                    *reinterpret_cast<uint2 *>(a.W_bf16 + g * D) = make_uint2(pack_bf16x2(wh[0], wh[1]), pack_bf16x2(wh[2], wh[3]));
                }
            }
        }
    }
}

// ------------------------------------------------------------------ pack

__global__ void __launch_bounds__(256)
pack2b_kernel(const uint8_t *__restrict__ codes, int64_t total, uint8_t *__restrict__ packed) {
    const int64_t nslices = (total + 15) / 16;
    for (int64_t sl = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; sl < nslices;
         sl += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gidx = sl * 16;
        if (total - gidx >= 16) {
            const uint4 q = __ldg(reinterpret_cast<const uint4 *>(codes + gidx));
            const uint32_t w[4] = {q.x, q.y, q.z, q.w};
            uint32_t p = 0;
#pragma unroll
            for (int k = 0; k < 16; ++k) p |= ((w[k >> 2] >> (8 * (k & 3))) & 3u) << (2 * k);
            *reinterpret_cast<uint32_t *>(packed + gidx / 4) = p;
        } else {
            for (int64_t k = gidx; k < total; k += 4) {
                uint32_t p = 0;
                for (int e = 0; e < 4; ++e) p |= (codes[k + e] & 3u) << (2 * e);
                packed[k / 4] = static_cast<uint8_t>(p);
            }
        }
    }
}

// ------------------------------------------------------------------ dA / db final reduction

// One warp per value: lane l sums partials l, l + 32, ... in order, then a fixed butterfly adds the
// lanes, so the result is the same on every run (no atomics) and all of a lane's loads are in flight.
__global__ void __launch_bounds__(256)
reduce_partials_kernel(const float *__restrict__ partials, int nparts, int d, float *dA, float *db) {
    const int nvals = d * d + d;
    const int i = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (i >= nvals) return;                   // whole warps: i is uniform across the warp
    float acc = 0.0f;
#pragma unroll 8
    for (int p = lane; p < nparts; p += 32) acc += __ldg(partials + static_cast<int64_t>(p) * nvals + i);
    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) {
        if (i < d * d) dA[i] = acc;
        else db[i - d * d] = acc;
    }
}

// ------------------------------------------------------------------ initialisation (Eq. init_ab, Eq. xavier_preprocess)

__global__ void init_codebook_kernel(const float *__restrict__ G, int d, float *A, float *b) {
    const float sc = sqrtf(12.0f / 15.0f);   // s = sqrt(12 / (2^{2b} - 1)), b = 2
    const int i = threadIdx.x;
    if (i < d * d) A[i] = sc * G[i];
    if (i < d) {
        float acc = 0.0f;
        for (int k = 0; k < d; ++k) acc += G[i * d + k];
        b[i] = -sc * 1.5f * acc;             // -s G (mu 1), mu = 1.5
    }
}

__global__ void __launch_bounds__(256)
init_latent_kernel(const uint8_t *__restrict__ packed, int64_t total, float s, float t, float *__restrict__ P) {
    const int64_t nslices = (total + 15) / 16;
    for (int64_t sl = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; sl < nslices;
         sl += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gidx = sl * 16;
        const int valid = static_cast<int>((total - gidx) < 16 ? (total - gidx) : 16);
        uint32_t w = 0;
        if (valid == 16) {
            w = __ldg(reinterpret_cast<const uint32_t *>(packed + gidx / 4));
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (k < valid / 4) w |= static_cast<uint32_t>(packed[gidx / 4 + k]) << (8 * k);
        }
        float v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = s * (static_cast<float>((w >> (2 * k)) & 3u) - t);
        if (valid == 16) {
            float4 *dst = reinterpret_cast<float4 *>(P + gidx);
#pragma unroll
            for (int q = 0; q < 4; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        } else {
#pragma unroll
            for (int k = 0; k < 16; ++k)
                if (k < valid) P[gidx + k] = v[k];
        }
    }
}

cudaError_t launch_init_codebook(const float *G, int d, float *A, float *b, cudaStream_t st) {
    init_codebook_kernel<<<1, 64, 0, st>>>(G, d, A, b);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_init_latent(const uint8_t *packed, int64_t total, float s, float t, float *P, int num_sms,
                               cudaStream_t st) {
    const int64_t nslices = (total + 15) / 16;
    int64_t grid = (nslices + 255) / 256;
    if (grid > 8LL * num_sms) grid = 8LL * num_sms;
    if (grid < 1) grid = 1;
    init_latent_kernel<<<static_cast<int>(grid), 256, 0, st>>>(packed, total, s, t, P);
    count_launch();
    return cudaGetLastError();
}

// ------------------------------------------------------------------ bounded-wait self-test

// One thread waits on an mbarrier whose phase nothing completes: mbar_wait gives up after its
// time limit, records LCQ_ERR_TIMEOUT and the kernel returns normally.
__global__ void wait_timeout_selftest_kernel(int32_t *status) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_barrier_init();
        (void)mbar_wait(&bar, 0, status);
    }
}

cudaError_t launch_wait_timeout_selftest(int32_t *status, cudaStream_t st) {
    wait_timeout_selftest_kernel<<<1, 32, 0, st>>>(status);
    count_launch();
    return cudaGetLastError();
}

// ------------------------------------------------------------------ host launchers

static int stream_grid(int64_t total, int num_sms) {
    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    int64_t g = num_sms;   // persistent: one CTA (a 198 KB ring) per SM
    if (nchunks < g) g = nchunks;
    return static_cast<int>(g < 1 ? 1 : g);
}

int encode_max_blocks(int num_sms) { return num_sms; }

cudaError_t launch_encode(const EncodeArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t total = a.m * a.n;
    const int grid = stream_grid(total, num_sms);
    const size_t smem = sizeof(StreamSmem);
    const bool mse = a.mse != nullptr;
    const bool lat = a.latent != nullptr;
    void (*k)(EncodeArgs) = nullptr;
    if (d == 4) {
        k = mse ? (lat ? encode_kernel<4, true, true> : encode_kernel<4, true, false>)
                : (lat ? encode_kernel<4, false, true> : encode_kernel<4, false, false>);
    } else {
        k = mse ? (lat ? encode_kernel<8, true, true> : encode_kernel<8, true, false>)
                : (lat ? encode_kernel<8, false, true> : encode_kernel<8, false, false>);
    }
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    trace_begin(LCQ_K_ENCODE, st);
    if (a.pdl & 2) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(grid);
        cfg.blockDim = dim3(kStreamThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, k, a);
    } else {
        k<<<grid, kStreamThreads, smem, st>>>(a);
        e = cudaSuccess;
    }
    trace_end(LCQ_K_ENCODE, st);
    count_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

int64_t encode_chunk_size() { return kChunk; }

cudaError_t launch_encode_batch(const EncodeBatchArgs &a, int d, int num_sms, cudaStream_t st) {
    bool mse = false, lat = false;
    for (int i = 0; i < a.count; ++i) {
        mse = mse || a.item[i].mse != nullptr;
        lat = lat || a.item[i].latent != nullptr;
    }
    if (mse) {
        // With the reconstruction MSE, the single-matrix kernel measured faster per matrix than the
        // fused batch kernel (whose MSE variant compiles to ~25% more instructions per group), so each
        // matrix gets its own launch, with its own partials and counter in the batch workspace. The
        // matrices are independent, so each launch after the first is a programmatic dependent launch
        // that starts as the previous one drains; the last one does not let anything start early, so
        // the work after the batch sees all of it.
        int last = -1;
        for (int i = 0; i < a.count; ++i) {
            const EncodeBatchItem &it = a.item[i];
            if (it.m * it.n != 0) {
                last = i;
            } else if (it.mse) {
                const cudaError_t e = cudaMemsetAsync(it.mse, 0, sizeof(double), st);
                if (e != cudaSuccess) return e;
            }
        }
        bool first = true;
        for (int i = 0; i < a.count; ++i) {
            const EncodeBatchItem &it = a.item[i];
            if (it.m * it.n == 0) continue;
            EncodeArgs e;
            e.W = it.W; e.m = it.m; e.n = it.n; e.A = it.A; e.b = it.b;
            e.packed = it.packed; e.codes = it.codes; e.latent = it.latent; e.mse = it.mse;
            e.partials = a.partials + static_cast<int64_t>(i) * kEncodeBatchPartials;
            e.counter = a.counters + i;
            e.status = a.status;
            e.pdl = (i != last ? 1 : 0) | (first ? 0 : 2);
            first = false;
            const cudaError_t r = launch_encode(e, d, num_sms, st);
            if (r != cudaSuccess) return r;
        }
        return cudaSuccess;
    }
    const int grid = static_cast<int>(a.total_chunks < num_sms ? (a.total_chunks > 0 ? a.total_chunks : 1) : num_sms);
    const size_t smem = sizeof(EncBatchSmem);
    void (*k)(const EncodeBatchArgs) = d == 4 ? (lat ? encode_batch_kernel<4, true> : encode_batch_kernel<4, false>)
                                              : (lat ? encode_batch_kernel<8, true> : encode_batch_kernel<8, false>);
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    trace_begin(LCQ_K_ENCODE, st);
    k<<<grid, kStreamThreads, smem, st>>>(a);
    trace_end(LCQ_K_ENCODE, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_quant_decode(const QuantDecodeArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t total = a.m * a.n;
    const int grid = stream_grid(total, num_sms);
    const size_t smem = sizeof(StreamSmem);
    void (*k)(QuantDecodeArgs) = d == 4 ? quant_decode_kernel<4> : quant_decode_kernel<8>;
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    trace_begin(LCQ_K_QUANT_DECODE, st);
    k<<<grid, kStreamThreads, smem, st>>>(a);
    trace_end(LCQ_K_QUANT_DECODE, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t nspans = (a.m * a.n / d + 32 * kDecGroups - 1) / (32 * kDecGroups);   // one warp each
    int64_t grid = (nspans + 7) / 8;
    if (grid > 8LL * num_sms) grid = 8LL * num_sms;
    if (grid < 1) grid = 1;
    trace_begin(LCQ_K_DECODE, st);
    if (d == 4) decode_kernel<4><<<static_cast<int>(grid), 256, 0, st>>>(a);
    else decode_kernel<8><<<static_cast<int>(grid), 256, 0, st>>>(a);
    trace_end(LCQ_K_DECODE, st);
    count_launch();
    return cudaGetLastError();
}

// Activation transform (Sec. 3.2, Eq. def:forward_x): one warp per token row. A lane takes the row's
// 8-column units lane, lane + 32, ... (one 16-byte load of bf16 each), four loads in flight before
// their arithmetic; it forms X' = X_g A for the unit's groups and adds X_g . b into its share of r,
// which the warp sums by a fixed butterfly.
constexpr int kXformWarps = 8;

template <int D>
__device__ __forceinline__ void xform_unit(const uint4 v, const float (&Am)[D * D], const float (&bv)[D], uint4 &out,
                                           float &racc) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float x[8], y[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
#pragma unroll
    for (int g = 0; g < 8 / D; ++g) {
#pragma unroll
        for (int k = 0; k < D; ++k) {
            float acc = 0.0f;
#pragma unroll
            for (int j = 0; j < D; ++j) acc = fmaf(x[g * D + j], Am[j * D + k], acc);
            y[g * D + k] = acc;
        }
#pragma unroll
        for (int j = 0; j < D; ++j) racc = fmaf(x[g * D + j], bv[j], racc);
    }
    out = make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]), pack_bf16x2(y[4], y[5]), pack_bf16x2(y[6], y[7]));
}

template <int D>
__global__ void __launch_bounds__(32 * kXformWarps)
xform_kernel(const uint16_t *__restrict__ X, int64_t N, int64_t n, const float *__restrict__ A,
             const float *__restrict__ b, uint16_t *__restrict__ Xp, float *__restrict__ r) {
    __shared__ float sA[D * D], sb[D];
    if (threadIdx.x < D * D) sA[threadIdx.x] = __ldg(A + threadIdx.x);
    if (threadIdx.x < D) sb[threadIdx.x] = __ldg(b + threadIdx.x);
    __syncthreads();
    float Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) Am[i] = sA[i];
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = sb[i];
    const int lane = threadIdx.x & 31;
    const int64_t t = static_cast<int64_t>(blockIdx.x) * kXformWarps + (threadIdx.x >> 5);
    if (t >= N) return;
    const uint4 *src = reinterpret_cast<const uint4 *>(X + t * n);
    uint4 *dst = Xp ? reinterpret_cast<uint4 *>(Xp + t * n) : nullptr;
    const int64_t units = n / 8;
    float racc = 0.0f;
    int64_t u = lane;
    for (; u + 96 < units; u += 128) {
        uint4 v[4], o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __ldg(src + u + 32 * i);
#pragma unroll
        for (int i = 0; i < 4; ++i) xform_unit<D>(v[i], Am, bv, o[i], racc);
        if (dst) {
#pragma unroll
            for (int i = 0; i < 4; ++i) dst[u + 32 * i] = o[i];
        }
    }
    for (; u < units; u += 32) {
        uint4 o;
        xform_unit<D>(__ldg(src + u), Am, bv, o, racc);
        if (dst) dst[u] = o;
    }
    for (int o = 16; o; o >>= 1) racc += __shfl_xor_sync(0xffffffffu, racc, o);
    if (r && lane == 0) r[t] = racc;
}

cudaError_t launch_xform(const uint16_t *X, int64_t N, int64_t n, int d, const float *A, const float *b, uint16_t *Xp,
                         float *r, cudaStream_t st) {
    trace_begin(LCQ_K_XFORM, st);
    const unsigned grid = static_cast<unsigned>((N + kXformWarps - 1) / kXformWarps);
    if (d == 4) xform_kernel<4><<<grid, 32 * kXformWarps, 0, st>>>(X, N, n, A, b, Xp, r);
    else xform_kernel<8><<<grid, 32 * kXformWarps, 0, st>>>(X, N, n, A, b, Xp, r);
    trace_end(LCQ_K_XFORM, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_pack2b(const uint8_t *codes, int64_t total, uint8_t *packed, int num_sms, cudaStream_t st) {
    const int64_t nslices = (total + 15) / 16;
    int64_t grid = (nslices + 255) / 256;
    if (grid > 8LL * num_sms) grid = 8LL * num_sms;
    if (grid < 1) grid = 1;
    trace_begin(LCQ_K_PACK, st);
    pack2b_kernel<<<static_cast<int>(grid), 256, 0, st>>>(codes, total, packed);
    trace_end(LCQ_K_PACK, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_reduce_partials(const float *partials, int nparts, int d, float *dA, float *db, cudaStream_t st) {
    trace_begin(LCQ_K_REDUCE, st);
    const int nvals = d * d + d;
    reduce_partials_kernel<<<(nvals * 32 + 255) / 256, 256, 0, st>>>(partials, nparts, d, dA, db);
    trace_end(LCQ_K_REDUCE, st);
    count_launch();
    return cudaGetLastError();
}

}  // namespace lcq
