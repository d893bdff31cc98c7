// HBM-bound element-wise kernels of the LC-VQ layer:
//   encode         W -> latent u = A^{-1}(W_g - b), codes clip(round(u),0,3), MSE   (Sec. 2.2)
//   quant_decode   P -> Z = clip(round(P/s + t),0,3) packed, W_hat = A Z_g + b bf16 (Eq. quant_param, def:forward)
//   decode         packed Z -> W_hat fp32 / bf16                                      (Eq. def:forward)
//   pack2b         one code per byte -> 4 codes per byte
//   reduce_partials  fixed-order sum of per-CTA dA/db partials
//
// encode and quant_decode stream their fp32 input through a shared-memory ring
// filled by the bulk-copy (TMA) engine: one producer thread issues 16 KB
// cp.async.bulk copies, eight compute warps consume them. Each compute thread
// owns 16 consecutive weights of a chunk, i.e. whole groups for d = 4 and 8.
#include "common.cuh"
#include "internal.h"

namespace lcq {

constexpr int kChunk = 4096;                 // fp32 weights per stage (16 KB)
constexpr int kStages = 4;
constexpr int kComputeWarps = 8;
constexpr int kStreamThreads = 32 * (1 + kComputeWarps);
constexpr int kPerThread = kChunk / (32 * kComputeWarps);   // 16
static_assert(kPerThread == 16, "each compute thread owns 16 weights");

struct StreamSmem {
    float buf[kStages][kChunk];
    uint64_t full[kStages];
    uint64_t empty[kStages];
    float Ainv[64];
    float A[64];
    float b[8];
    double gj[8][16];
    float red[kComputeWarps];
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
        const int st = i % kStages;
        const uint32_t ph = (i / kStages) & 1;
        if (!mbar_wait(&s.empty[st], ph ^ 1, status)) return;
        const int64_t base = c * kChunk;
        const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
        const uint32_t bytes = static_cast<uint32_t>(cnt * 4);
        mbar_arrive_expect_tx(&s.full[st], bytes);
        bulk_g2s(s.buf[st], src + base, bytes, &s.full[st]);
    }
}

// One warp: A^{-1} by Gauss-Jordan elimination with partial pivoting in fp64,
// rounded to fp32. Sets s.singular if a pivot is (relatively) zero.
template <int D>
__device__ void invert_warp(StreamSmem &s) {
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
        // pivot search over rows c..D-1
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
        for (int e = lane; e < D * 2 * D; e += 32, ++cnt) {
            const int r = e / (2 * D);
            f[cnt] = s.gj[r][c];
        }
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
}

// ------------------------------------------------------------------ encode

template <int D, bool kMse>
__device__ __forceinline__ void encode_group(const float *w, const float (&Ai)[D * D], const float (&Am)[D * D],
                                             const float (&bv)[D], uint32_t (&z)[D], float (&u)[D], float &sq) {
    float v[D];
#pragma unroll
    for (int j = 0; j < D; ++j) v[j] = w[j] - bv[j];
#pragma unroll
    for (int k = 0; k < D; ++k) {
        float acc = 0.0f;
#pragma unroll
        for (int j = 0; j < D; ++j) acc = fmaf(Ai[k * D + j], v[j], acc);
        u[k] = acc;
        z[k] = round_clamp3(acc);
    }
    if (kMse) {
#pragma unroll
        for (int j = 0; j < D; ++j) {
            float r = v[j];
#pragma unroll
            for (int k = 0; k < D; ++k) r = fmaf(-Am[j * D + k], static_cast<float>(z[k]), r);
            sq = fmaf(r, r, sq);
        }
    }
}

template <int D, bool kMse>
__global__ void __launch_bounds__(kStreamThreads, 1)
encode_kernel(EncodeArgs a) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    StreamSmem &s = *reinterpret_cast<StreamSmem *>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t total = a.m * a.n;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], kComputeWarps);
        }
        fence_barrier_init();
    }
    if (threadIdx.x < D * D) s.A[threadIdx.x] = a.A[threadIdx.x];
    if (threadIdx.x < D) s.b[threadIdx.x] = a.b[threadIdx.x];
    __syncthreads();

    if (warp == 0) {
        if (lane == 0) stream_producer(s, a.W, total, a.status);
        return;
    }
    // compute warps
    if (warp == 1) invert_warp<D>(s);
    compute_bar();
    if (s.singular && blockIdx.x == 0 && threadIdx.x == 32) set_status(a.status, LCQ_ERR_SINGULAR);

    float Ai[D * D], Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) { Ai[i] = s.Ainv[i]; Am[i] = s.A[i]; }
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = s.b[i];

    const int t = threadIdx.x - 32;
    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    float sq = 0.0f;
    int i = 0;
    for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++i) {
        const int st = i % kStages;
        if (!mbar_wait(&s.full[st], (i / kStages) & 1, a.status)) break;
        const int64_t base = c * kChunk;
        const int64_t cnt = (total - base < kChunk) ? (total - base) : kChunk;
        const int64_t off = static_cast<int64_t>(t) * kPerThread;
        if (off < cnt) {
            const int valid = static_cast<int>((cnt - off) < kPerThread ? (cnt - off) : kPerThread);
            const float *src = s.buf[st] + off;
            float w[kPerThread];
#pragma unroll
            for (int q = 0; q < kPerThread / 4; ++q) {
                const float4 f = (q * 4 < valid) ? reinterpret_cast<const float4 *>(src)[q] : make_float4(0, 0, 0, 0);
                w[4 * q] = f.x; w[4 * q + 1] = f.y; w[4 * q + 2] = f.z; w[4 * q + 3] = f.w;
            }
            uint32_t zz[kPerThread];
            float uu[kPerThread];
#pragma unroll
            for (int g = 0; g < kPerThread / D; ++g) {
                uint32_t z[D];
                float u[D];
                float gsq = 0.0f;
                encode_group<D, kMse>(w + g * D, Ai, Am, bv, z, u, gsq);
                if (g * D < valid) sq += gsq;
#pragma unroll
                for (int k = 0; k < D; ++k) { zz[g * D + k] = z[k]; uu[g * D + k] = u[k]; }
            }
            const int64_t gidx = base + off;   // flat weight index, multiple of 16
            if (valid == kPerThread) {
                if (a.packed) {
                    uint32_t p = 0;
#pragma unroll
                    for (int k = 0; k < kPerThread; ++k) p |= zz[k] << (2 * k);
                    *reinterpret_cast<uint32_t *>(a.packed + gidx / 4) = p;
                }
                if (a.codes) {
                    uint4 q;
                    q.x = zz[0] | (zz[1] << 8) | (zz[2] << 16) | (zz[3] << 24);
                    q.y = zz[4] | (zz[5] << 8) | (zz[6] << 16) | (zz[7] << 24);
                    q.z = zz[8] | (zz[9] << 8) | (zz[10] << 16) | (zz[11] << 24);
                    q.w = zz[12] | (zz[13] << 8) | (zz[14] << 16) | (zz[15] << 24);
                    *reinterpret_cast<uint4 *>(a.codes + gidx) = q;
                }
                if (a.latent) {
                    float4 *dst = reinterpret_cast<float4 *>(a.latent + gidx);
#pragma unroll
                    for (int q = 0; q < 4; ++q) dst[q] = make_float4(uu[4 * q], uu[4 * q + 1], uu[4 * q + 2], uu[4 * q + 3]);
                }
            } else {
#pragma unroll
                for (int k = 0; k < kPerThread; k += 4) {
                    if (k < valid) {
                        if (a.packed)
                            a.packed[(gidx + k) / 4] =
                                static_cast<uint8_t>(zz[k] | (zz[k + 1] << 2) | (zz[k + 2] << 4) | (zz[k + 3] << 6));
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            if (a.codes) a.codes[gidx + k + e] = static_cast<uint8_t>(zz[k + e]);
                            if (a.latent) a.latent[gidx + k + e] = uu[k + e];
                        }
                    }
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[st]);
    }

    if (kMse) {
        for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        if (lane == 0) s.dred[warp - 1] = static_cast<double>(sq);
        compute_bar();
        if (t == 0) {
            double acc = 0.0;
            for (int w = 0; w < kComputeWarps; ++w) acc += s.dred[w];
            a.partials[blockIdx.x] = acc;
            __threadfence();
            const unsigned prev = atomicAdd(a.counter, 1u);
            if (prev == gridDim.x - 1) {
                __threadfence();
                double tot = 0.0;
                for (unsigned p = 0; p < gridDim.x; ++p) tot += __ldcg(a.partials + p);
                *a.mse = total > 0 ? tot / static_cast<double>(total) : 0.0;
            }
        }
    }
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
        for (int i = 0; i < kStages; ++i) {
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
        const int st = i % kStages;
        if (!mbar_wait(&s.full[st], (i / kStages) & 1, a.status)) break;
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
                if (a.packed) {
                    uint32_t p = 0;
#pragma unroll
                    for (int k = 0; k < kPerThread; ++k) p |= z[k] << (2 * k);
                    *reinterpret_cast<uint32_t *>(a.packed + gidx / 4) = p;
                }
                uint4 *dst = reinterpret_cast<uint4 *>(a.W_hat + gidx);
                dst[0] = make_uint4(pack_bf16x2(wh[0], wh[1]), pack_bf16x2(wh[2], wh[3]), pack_bf16x2(wh[4], wh[5]),
                                    pack_bf16x2(wh[6], wh[7]));
                dst[1] = make_uint4(pack_bf16x2(wh[8], wh[9]), pack_bf16x2(wh[10], wh[11]),
                                    pack_bf16x2(wh[12], wh[13]), pack_bf16x2(wh[14], wh[15]));
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

template <int D>
__global__ void __launch_bounds__(256)
decode_kernel(DecodeArgs a) {
    float Am[D * D], bv[D];
#pragma unroll
    for (int i = 0; i < D * D; ++i) Am[i] = __ldg(a.A + i);
#pragma unroll
    for (int i = 0; i < D; ++i) bv[i] = __ldg(a.b + i);
    const int64_t total = a.m * a.n;
    const int64_t nslices = (total + 15) / 16;
    for (int64_t sl = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; sl < nslices;
         sl += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gidx = sl * 16;
        const int valid = static_cast<int>((total - gidx) < 16 ? (total - gidx) : 16);
        uint32_t p;
        if (valid == 16) {
            p = __ldg(reinterpret_cast<const uint32_t *>(a.packed + gidx / 4));
        } else {
            p = 0;
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (k < valid / 4) p |= static_cast<uint32_t>(a.packed[gidx / 4 + k]) << (8 * k);
        }
        float wh[16];
#pragma unroll
        for (int g = 0; g < 16 / D; ++g) {
#pragma unroll
            for (int j = 0; j < D; ++j) {
                float acc = bv[j];
#pragma unroll
                for (int k = 0; k < D; ++k)
                    acc = fmaf(Am[j * D + k], static_cast<float>((p >> (2 * (g * D + k))) & 3u), acc);
                wh[g * D + j] = acc;
            }
        }
        if (valid == 16) {
            if (a.W_f32) {
                float4 *dst = reinterpret_cast<float4 *>(a.W_f32 + gidx);
#pragma unroll
                for (int q = 0; q < 4; ++q) dst[q] = make_float4(wh[4 * q], wh[4 * q + 1], wh[4 * q + 2], wh[4 * q + 3]);
            }
            if (a.W_bf16) {
                uint4 *dst = reinterpret_cast<uint4 *>(a.W_bf16 + gidx);
                dst[0] = make_uint4(pack_bf16x2(wh[0], wh[1]), pack_bf16x2(wh[2], wh[3]), pack_bf16x2(wh[4], wh[5]),
                                    pack_bf16x2(wh[6], wh[7]));
                dst[1] = make_uint4(pack_bf16x2(wh[8], wh[9]), pack_bf16x2(wh[10], wh[11]),
                                    pack_bf16x2(wh[12], wh[13]), pack_bf16x2(wh[14], wh[15]));
            }
        } else {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                if (k < valid) {
                    if (a.W_f32) a.W_f32[gidx + k] = wh[k];
                    if (a.W_bf16) {
                        const __nv_bfloat16 h = __float2bfloat16_rn(wh[k]);
                        a.W_bf16[gidx + k] = *reinterpret_cast<const uint16_t *>(&h);
                    }
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

__global__ void reduce_partials_kernel(const float *__restrict__ partials, int nparts, int d, float *dA, float *db) {
    const int nvals = d * d + d;
    for (int i = threadIdx.x; i < nvals; i += blockDim.x) {
        float acc = 0.0f;
        for (int p = 0; p < nparts; ++p) acc += partials[static_cast<int64_t>(p) * nvals + i];
        if (i < d * d) dA[i] = acc;
        else db[i - d * d] = acc;
    }
}

// ------------------------------------------------------------------ host launchers

static int stream_grid(int64_t total, int num_sms) {
    const int64_t nchunks = (total + kChunk - 1) / kChunk;
    int64_t g = 2LL * num_sms;
    if (nchunks < g) g = nchunks;
    return static_cast<int>(g < 1 ? 1 : g);
}

size_t encode_partials_offset() { return 256; }

int encode_max_blocks(int num_sms) { return 2 * num_sms; }

cudaError_t launch_encode(const EncodeArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t total = a.m * a.n;
    const int grid = stream_grid(total, num_sms);
    const size_t smem = sizeof(StreamSmem);
    const bool mse = a.mse != nullptr;
    void (*k)(EncodeArgs) = nullptr;
    if (d == 4) k = mse ? encode_kernel<4, true> : encode_kernel<4, false>;
    else k = mse ? encode_kernel<8, true> : encode_kernel<8, false>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
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
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    trace_begin(LCQ_K_QUANT_DECODE, st);
    k<<<grid, kStreamThreads, smem, st>>>(a);
    trace_end(LCQ_K_QUANT_DECODE, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeArgs &a, int d, int num_sms, cudaStream_t st) {
    const int64_t nslices = (a.m * a.n + 15) / 16;
    int64_t grid = (nslices + 255) / 256;
    if (grid > 8LL * num_sms) grid = 8LL * num_sms;
    if (grid < 1) grid = 1;
    trace_begin(LCQ_K_DECODE, st);
    if (d == 4) decode_kernel<4><<<static_cast<int>(grid), 256, 0, st>>>(a);
    else decode_kernel<8><<<static_cast<int>(grid), 256, 0, st>>>(a);
    trace_end(LCQ_K_DECODE, st);
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
    reduce_partials_kernel<<<1, 128, 0, st>>>(partials, nparts, d, dA, db);
    trace_end(LCQ_K_REDUCE, st);
    count_launch();
    return cudaGetLastError();
}

}  // namespace lcq
