// Persistent bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM), fed by TMA.
//
//   C[M][N] = sum_k A(m, k) * B(n, k)        fp32 accumulation in tensor memory
//
// One CTA per SM, 192 threads:
//   warp 0      TMA producer: 4-stage ring of (128 x 64) A and (256 x 64) B bf16 tiles, 128B swizzle
//   warp 1      TMEM owner (512 columns = two 128 x 256 fp32 accumulators) and single-thread MMA issuer
//   warps 2..5  epilogue: tcgen05.ld the accumulator (one TMEM lane quarter per warp) and
//               either store bf16 C, or run the LC-VQ weight-gradient epilogue (EPI_DW):
//                 dP_g = (1/s) * dW_hat_g A        (straight-through estimator, Sec. 3.3)
//                 dA  += dW_hat_g z_g^T,  db += dW_hat_g   (per-thread, reduced per CTA at the end)
// The two accumulators let the epilogue of tile i overlap the main loop of tile i+1.
// Operands may be K-major ([rows][K]) or MN-major ([K][rows]); both layouts are read by TMA
// with 128-byte swizzle and described to the tensor core with the matching smem descriptor.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "internal.h"

namespace lcq {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_STAGE = BM * BK * 2;   // 16 KB
constexpr int B_STAGE = BN * BK * 2;   // 32 KB
constexpr int kGemmThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr int kGroupM = 16;            // tile raster: groups of 16 M-tiles sweep all N-tiles

struct GemmSmem {
    uint8_t a[STAGES][A_STAGE];
    uint8_t b[STAGES][B_STAGE];
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint32_t tmem_base;
    float Am[64];
    float red[4][72];
};

struct GemmParams {
    int M, N, K;
    uint16_t *C;
    int64_t ldc;
    DwEpilogue dw;
    int32_t *status;
};

__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int &tm, int &tn) {
    const int span = kGroupM * num_n;
    const int g = tile / span;
    const int first_m = g * kGroupM;
    const int gsize = min(num_m - first_m, kGroupM);
    const int r = tile - g * span;
    tm = first_m + r % gsize;
    tn = r / gsize;
}

template <bool MN>
__device__ __forceinline__ uint64_t operand_desc(uint32_t stage_base, int kstep) {
    if (MN) {
        // [chunk of 64 rows][64 k-rows][128 B]: next 64-row chunk at 8 KB, next 8 k-rows at 1 KB,
        // a K=16 step advances 16 k-rows (2 KB).
        return smem_desc_sw128(stage_base + kstep * 2048, 8192, 1024);
    } else {
        // [rows][128 B] with 8-row swizzle atoms of 1 KB; a K=16 step advances 32 B inside the atom.
        return smem_desc_sw128(stage_base + kstep * 32, 16, 1024);
    }
}

template <bool MN, int ROWS>
__device__ __forceinline__ void load_operand(uint8_t *dst, const CUtensorMap *map, int row0, int k0, uint64_t *bar) {
    if (MN) {
#pragma unroll
        for (int c = 0; c < ROWS / 64; ++c) tma_load_2d(dst + c * 8192, map, row0 + c * 64, k0, bar);
    } else {
        tma_load_2d(dst, map, k0, row0, bar);
    }
}

template <int EPI, int D, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kGemmThreads, 1)
gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const GemmParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte alignment of the stage buffers is required by the 128B swizzle atoms.
    GemmSmem &s = *reinterpret_cast<GemmSmem *>(align_smem_1024(smem_raw));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int num_m = (p.M + BM - 1) / BM, num_n = (p.N + BN - 1) / BN;
    const int num_tiles = num_m * num_n;
    const int num_kb = (p.K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmA);
        prefetch_tensormap(&tmB);
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.tfull[i], 1);
            mbar_init(&s.tempty[i], 4);
        }
        fence_barrier_init();
    }
    if (EPI == EPI_DW && threadIdx.x < D * D) s.Am[threadIdx.x] = p.dw.A[threadIdx.x];
    if (warp == 1) {
        tmem_alloc(&s.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s.tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------------ TMA producer
            int it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
                int tm, tn;
                tile_coords(tile, num_m, num_n, tm, tn);
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int st = it % STAGES;
                    if (!mbar_wait(&s.empty[st], ((it / STAGES) & 1) ^ 1, p.status)) { ok = false; break; }
                    mbar_arrive_expect_tx(&s.full[st], A_STAGE + B_STAGE);
                    load_operand<A_MN, BM>(s.a[st], &tmA, tm * BM, kb * BK, &s.full[st]);
                    load_operand<B_MN, BN>(s.b[st], &tmB, tn * BN, kb * BK, &s.full[st]);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------------------ MMA issuer
            constexpr uint32_t idesc = idesc_bf16(BM, BN, A_MN, B_MN);
            int it = 0, tcount = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++tcount) {
                const int acc = tcount & 1;
                if (!mbar_wait(&s.tempty[acc], ((tcount >> 1) & 1) ^ 1, p.status)) break;
                tc_fence_after();
                const uint32_t dtm = tmem + acc * BN;
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int st = it % STAGES;
                    if (!mbar_wait(&s.full[st], (it / STAGES) & 1, p.status)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t abase = smem_u32(s.a[st]), bbase = smem_u32(s.b[st]);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        umma_bf16(dtm, operand_desc<A_MN>(abase, k), operand_desc<B_MN>(bbase, k), idesc,
                                  (kb | k) != 0);
                    }
                    umma_commit(&s.empty[st]);
                }
                umma_commit(&s.tfull[acc]);
            }
        }
    } else {
        // ---------------------------------------------------------------- epilogue (warps 2..5)
        const int q = warp & 3;   // TMEM lane quarter this warp may access
        float dA[EPI == EPI_DW ? D * D : 1], db[EPI == EPI_DW ? D : 1];
        float Am[EPI == EPI_DW ? D * D : 1];
        if (EPI == EPI_DW) {
#pragma unroll
            for (int i = 0; i < D * D; ++i) { dA[i] = 0.0f; Am[i] = s.Am[i]; }
#pragma unroll
            for (int i = 0; i < D; ++i) db[i] = 0.0f;
        }
        int tcount = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++tcount) {
            int tm, tn;
            tile_coords(tile, num_m, num_n, tm, tn);
            const int acc = tcount & 1;
            if (!mbar_wait(&s.tfull[acc], (tcount >> 1) & 1, p.status)) break;
            tc_fence_after();
            const int row = tm * BM + q * 32 + lane;
            const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + acc * BN;
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                float v[32];
                __syncwarp();   // tcgen05.ld is warp-collective: reconverge after the bounds checks
                tmem_ld32(taddr + c * 32, v);
                const int col0 = tn * BN + c * 32;
                if (row >= p.M || col0 >= p.N) continue;
                if (EPI == EPI_STORE_BF16) {
                    uint16_t *dst = p.C + static_cast<int64_t>(row) * p.ldc + col0;
                    if (col0 + 32 <= p.N) {
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            reinterpret_cast<uint4 *>(dst)[u] =
                                make_uint4(pack_bf16x2(v[8 * u + 0], v[8 * u + 1]), pack_bf16x2(v[8 * u + 2], v[8 * u + 3]),
                                           pack_bf16x2(v[8 * u + 4], v[8 * u + 5]), pack_bf16x2(v[8 * u + 6], v[8 * u + 7]));
                        }
                    } else {
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            if (col0 + e < p.N) {
                                const __nv_bfloat16 h = __float2bfloat16_rn(v[e]);
                                dst[e] = *reinterpret_cast<const uint16_t *>(&h);
                            }
                        }
                    }
                } else {
                    // weight-gradient epilogue: this thread holds dW_hat[row][col0 .. col0+31]
                    const int64_t nq = p.N / 4;   // packed bytes per row
                    const uint8_t *zrow = p.dw.packed + static_cast<int64_t>(row) * nq + col0 / 4;
                    uint32_t zw[2];
                    const bool full32 = col0 + 32 <= p.N;
                    if (full32 && (nq % 8) == 0) {
                        const uint2 t2 = *reinterpret_cast<const uint2 *>(zrow);
                        zw[0] = t2.x; zw[1] = t2.y;
                    } else {
                        zw[0] = zw[1] = 0;
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            if (col0 + 4 * e < p.N) zw[e >> 2] |= static_cast<uint32_t>(zrow[e]) << (8 * (e & 3));
                    }
                    float *dprow = p.dw.dP + static_cast<int64_t>(row) * p.N + col0;
                    const float *prow = p.dw.P ? p.dw.P + static_cast<int64_t>(row) * p.N + col0 : nullptr;
#pragma unroll
                    for (int g = 0; g < 32 / D; ++g) {
                        if (col0 + g * D >= p.N) break;
                        float z[D], out[D];
#pragma unroll
                        for (int k = 0; k < D; ++k) {
                            const int e = g * D + k;
                            z[k] = static_cast<float>((zw[e >> 4] >> (2 * (e & 15))) & 3u);
                        }
#pragma unroll
                        for (int k = 0; k < D; ++k) {
                            float t = 0.0f;
#pragma unroll
                            for (int j = 0; j < D; ++j) t = fmaf(v[g * D + j], Am[j * D + k], t);
                            out[k] = t * p.dw.inv_s;
                        }
                        if (p.dw.ste_mode == LCQ_STE_CLIPPED) {
#pragma unroll
                            for (int k = 0; k < D; ++k) {
                                const float u = __fadd_rn(__fmul_rn(prow[g * D + k], p.dw.inv_s), p.dw.t);
                                if (!(u >= -0.5f && u <= 3.5f)) out[k] = 0.0f;
                            }
                        } else if (p.dw.ste_mode == LCQ_STE_DGE) {
                            // slope of the differentiable gradient estimator (Eq. dge) at v, delta = 1
#pragma unroll
                            for (int k = 0; k < D; ++k) {
                                const float u = __fadd_rn(__fmul_rn(prow[g * D + k], p.dw.inv_s), p.dw.t);
                                const float x = u - floorf(u);
                                const float y = fabsf(2.0f * x - 1.0f);
                                float gs = fminf(p.dw.dge_cap, p.dw.dge_inv_k * exp2f(p.dw.dge_exp * log2f(y)));
                                if (!(u >= 0.0f && u < 3.0f)) gs = 0.0f;
                                out[k] *= gs;
                            }
                        }
#pragma unroll
                        for (int k = 0; k < D; k += 4)
                            *reinterpret_cast<float4 *>(dprow + g * D + k) = make_float4(out[k], out[k + 1], out[k + 2], out[k + 3]);
#pragma unroll
                        for (int j = 0; j < D; ++j) {
                            db[j] += v[g * D + j];
#pragma unroll
                            for (int k = 0; k < D; ++k) dA[j * D + k] = fmaf(v[g * D + j], z[k], dA[j * D + k]);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.tempty[acc]);
        }
        if (EPI == EPI_DW) {
            // fixed-order reduction: lanes (butterfly), then the 4 warps in order
            constexpr int NV = D * D + D;
#pragma unroll
            for (int i = 0; i < NV; ++i) {
                float x = i < D * D ? dA[i] : db[i - D * D];
                for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
                if (lane == 0) s.red[q][i] = x;
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (warp == 2) {
                for (int i = lane; i < NV; i += 32) {
                    const float x = ((s.red[0][i] + s.red[1][i]) + s.red[2][i]) + s.red[3][i];
                    p.dw.partials[static_cast<int64_t>(blockIdx.x) * NV + i] = x;
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ------------------------------------------------------------------ host side

static PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(tensor_map_encoder());
}

// rows x K operand stored K-major ([rows][ld]) or MN-major ([K][ld]); box rows_box x 64.
static bool make_map(CUtensorMap *map, const GemmOperand &op, int64_t rows, int64_t K, int rows_box) {
    auto enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2], strides[1];
    cuuint32_t box[2], estr[2] = {1, 1};
    if (op.mn_major) {
        dims[0] = static_cast<cuuint64_t>(rows);
        dims[1] = static_cast<cuuint64_t>(K);
        box[0] = 64;
        box[1] = 64;
    } else {
        dims[0] = static_cast<cuuint64_t>(K);
        dims[1] = static_cast<cuuint64_t>(rows);
        box[0] = 64;
        box[1] = static_cast<cuuint32_t>(rows_box);
    }
    strides[0] = static_cast<cuuint64_t>(op.ld) * 2;
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(op.ptr), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int gemm_grid(int64_t M, int64_t N, int num_sms) {
    const int64_t tiles = ((M + BM - 1) / BM) * ((N + BN - 1) / BN);
    return static_cast<int>(tiles < num_sms ? (tiles < 1 ? 1 : tiles) : num_sms);
}

template <int EPI, int D, bool A_MN, bool B_MN>
static cudaError_t launch_one(const CUtensorMap &ma, const CUtensorMap &mb, const GemmParams &gp, int grid,
                              int trace_kind, cudaStream_t st) {
    auto k = gemm_kernel<EPI, D, A_MN, B_MN>;
    const int smem = static_cast<int>(sizeof(GemmSmem) + 1024);
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), smem);
    if (e != cudaSuccess) return e;
    trace_begin(trace_kind, st);
    k<<<grid, kGemmThreads, smem, st>>>(ma, mb, gp);
    trace_end(trace_kind, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmProblem &p, GemmEpilogue epi, int num_sms, cudaStream_t st) {
    CUtensorMap ma, mb;
    if (!make_map(&ma, p.a, p.M, p.K, BM) || !make_map(&mb, p.b, p.N, p.K, BN)) return cudaErrorInvalidValue;
    GemmParams gp;
    gp.M = static_cast<int>(p.M);
    gp.N = static_cast<int>(p.N);
    gp.K = static_cast<int>(p.K);
    gp.C = p.C;
    gp.ldc = p.ldc;
    gp.dw = p.dw;
    gp.status = p.status;
    const int grid = gemm_grid(p.M, p.N, num_sms);
    if (epi == EPI_STORE_BF16) {
        if (!p.a.mn_major && !p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, false, false>(ma, mb, gp, grid, p.trace_kind, st);
        if (!p.a.mn_major && p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, false, true>(ma, mb, gp, grid, p.trace_kind, st);
        if (p.a.mn_major && p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, true, true>(ma, mb, gp, grid, p.trace_kind, st);
        return launch_one<EPI_STORE_BF16, 1, true, false>(ma, mb, gp, grid, p.trace_kind, st);
    }
    if (!(p.a.mn_major && p.b.mn_major)) return cudaErrorInvalidValue;
    if (p.dw.d == 4) return launch_one<EPI_DW, 4, true, true>(ma, mb, gp, grid, p.trace_kind, st);
    return launch_one<EPI_DW, 8, true, true>(ma, mb, gp, grid, p.trace_kind, st);
}

}  // namespace lcq
