// Persistent bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM), fed by TMA, run by pairs
// of CTAs (clusters of two) over 256 x 256 output tiles.
//
//   C[M][N] = sum_k A(m, k) * B(n, k)        fp32 accumulation in tensor memory
//
// Per CTA, one per SM, 192 threads:
//   warp 0      TMA producer: a 7-stage ring of this CTA's halves of the tile, rows r*128.. of A and
//               rows r*128.. of B (128 x 64 bf16 each, 128B swizzle; r = rank in the pair)
//   warp 1      TMEM owner (512 columns = two 128 x 256 fp32 accumulators, allocated by the pair
//               together) and, in the leader CTA, the single-thread issuer of
//               tcgen05.mma.cta_group::2 (M = 256, N = 256), which reads both CTAs' halves and writes
//               each CTA's 128 accumulator rows into its own tensor memory
//   warps 2..5  epilogue: tcgen05.ld this CTA's accumulator rows (one TMEM lane quarter per warp) and
//               either store bf16 C, or run the LC-VQ weight-gradient epilogue (EPI_DW):
//                 dP_g = (1/s) * dW_hat_g A        (straight-through estimator, Sec. 3.3)
//                 dA  += dW_hat_g z_g^T,  db += dW_hat_g   (per-thread, reduced per CTA at the end)
// The two accumulators let the epilogue of tile i overlap the main loop of tile i+1. Holding half of
// B per SM leaves room for seven stages of operand data in flight (four with a whole 128 x 256 tile per
// CTA), which is what the main loop waits on.
// Operands may be K-major ([rows][K]) or MN-major ([K][rows]); both layouts are read by TMA
// with 128-byte swizzle and described to the tensor core with the matching smem descriptor.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "internal.h"

namespace lcq {

constexpr int BK = 64;
constexpr int kGemmThreads = 192;
constexpr uint32_t kTmemCols = 512;

struct GemmParams {
    int M, N, K;
    uint16_t *C;
    int64_t ldc;
    DwEpilogue dw;
    int32_t *status;
};

__device__ __forceinline__ void tile_coords_group(int tile, int num_m, int num_n, int group_m, int &tm, int &tn) {
    const int span = group_m * num_n;
    const int g = tile / span;
    const int first_m = g * group_m;
    const int gsize = min(num_m - first_m, group_m);
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

template <int EPI, int D>
__device__ __forceinline__ void epilogue_chunk(const GemmParams &p, const float (&v)[32], int row, int col0,
                                               const float (&Am)[EPI == EPI_DW ? D * D : 1],
                                               float (&dA)[EPI == EPI_DW ? D * D : 1],
                                               float (&db)[EPI == EPI_DW ? D : 1]) {
    if (row >= p.M || col0 >= p.N) return;
    if (EPI == EPI_STORE_BF16) {
        uint16_t *dst = p.C + static_cast<int64_t>(row) * p.ldc + col0;
        // 16-byte stores need a 16-byte aligned row start: the row stride of C (the output width) need
        // not be a multiple of 8
        if (col0 + 32 <= p.N && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
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

// End of a CTA's weight-gradient epilogue: fixed-order reduction of the per-thread dA, db (lanes by a
// butterfly, then the four warps in order) into this CTA's partials.
template <int D>
__device__ __forceinline__ void epilogue_dw_reduce(const float (&dA)[D * D], const float (&db)[D], float (*red)[72], int q,
                                                   int warp, int lane, float *partials) {
    constexpr int NV = D * D + D;
#pragma unroll
    for (int i = 0; i < NV; ++i) {
        float x = i < D * D ? dA[i] : db[i - D * D];
        for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
        if (lane == 0) red[q][i] = x;
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (warp == 2) {
        for (int i = lane; i < NV; i += 32) {
            const float x = ((red[0][i] + red[1][i]) + red[2][i]) + red[3][i];
            partials[static_cast<int64_t>(blockIdx.x) * NV + i] = x;
        }
    }
}

// ------------------------------------------------------------------ paired kernel (cta_group::2)
//
// 256 x 256 tiles per pair of CTAs (a cluster of two). CTA r of the pair holds rows r*128.. of the
// tile's A and rows r*128.. of its B in its own shared memory (32 KB per stage, so seven stages fit;
// a whole 128 x 256 tile per CTA would take 48 KB per stage, four stages); the leader's
// tcgen05.mma.cta_group::2 (M = 256, N = 256) reads both CTAs' halves and writes each CTA's 128
// accumulator rows into that CTA's tensor memory. Both CTAs' TMA copies complete on the leader's full
// barrier (the copies' .cta_group::2 form, the barrier addressed through mapa), the leader's MMA
// commits arrive on both CTAs' empty and accumulator-full barriers (multicast), and both CTAs' epilogue
// warps arrive on the leader's accumulator-empty barrier. Each CTA's epilogue handles its own 128 rows.

constexpr int PM = 256, PN = 256, PH = 128;   // pair tile; rows of A and of B per CTA
constexpr int PSTAGES = 7;
constexpr int P_HALF = PH * BK * 2;            // 16 KB: one CTA's A (or B) rows of a stage
constexpr int kPairGroupM = 8;                 // pair-tile raster: groups of 8 M pair-tiles (2048 rows)

struct PairSmem {
    uint8_t a[PSTAGES][P_HALF];
    uint8_t b[PSTAGES][P_HALF];
    uint64_t full[PSTAGES];    // leader's: both CTAs' copies of the stage landed
    uint64_t empty[PSTAGES];   // each CTA's: the MMAs reading the stage completed
    uint64_t tfull[2];         // each CTA's: the accumulator is complete
    uint64_t tempty[2];        // leader's: both CTAs' epilogues have read the accumulator
    uint32_t tmem_base;
    float Am[64];
};

__device__ __forceinline__ uint32_t pair_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void pair_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared variable in the leader CTA (rank 0) of the pair.
__device__ __forceinline__ uint32_t leader_smem(const void *p) {
    uint32_t m;
    asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(m) : "r"(smem_u32(p)));
    return m;
}
// 2-D TMA copy into this CTA's shared memory, completing on the leader's mbarrier.
__device__ __forceinline__ void tma_load_2d_to_leader(void *dst, const CUtensorMap *map, int32_t c0, int32_t c1,
                                                      uint32_t leader_bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%2, "
        "%3}], [%4];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(leader_bar)
        : "memory");
}
template <bool MN>
__device__ __forceinline__ void load_half(uint8_t *dst, const CUtensorMap *map, int row0, int k0, uint32_t leader_bar) {
    if (MN) {
#pragma unroll
        for (int c = 0; c < PH / 64; ++c) tma_load_2d_to_leader(dst + c * 8192, map, row0 + c * 64, k0, leader_bar);
    } else {
        tma_load_2d_to_leader(dst, map, k0, row0, leader_bar);
    }
}
__device__ __forceinline__ void umma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive on the mbarrier at this shared address in both CTAs of the pair once the MMAs issued so far
// have completed.
__device__ __forceinline__ void umma_commit_both(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            smem_u32(bar)),
        "h"(static_cast<uint16_t>(3))
        : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// Work item w of pair cid (of G pairs): the whole tiles cid, cid + G, ...; then, when the tiles of the
// last, partial wave split into two 128-column halves still fit one wave (2R <= G), half tile cid of
// that wave (half = 0 or 1; -1 for a whole tile), so the last wave takes half the time.
struct PairWork {
    int tm, tn, half;
};
__device__ __forceinline__ bool pair_work(int w, int cid, int G, int num_m, int num_n, PairWork &o) {
    const int tiles = num_m * num_n;
    const int R = tiles % G;
    const bool split = R > 0 && 2 * R <= G;
    const int whole = split ? tiles - R : tiles;
    const int nwhole = whole > cid ? (whole - cid + G - 1) / G : 0;
    if (w < nwhole) {
        tile_coords_group(cid + w * G, num_m, num_n, kPairGroupM, o.tm, o.tn);
        o.half = -1;
        return true;
    }
    if (!split || w != nwhole || cid >= 2 * R) return false;
    tile_coords_group(whole + (cid >> 1), num_m, num_n, kPairGroupM, o.tm, o.tn);
    o.half = cid & 1;
    return true;
}

template <int EPI, int D, bool A_MN, bool B_MN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const __grid_constant__ CUtensorMap tmB64, const GemmParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    PairSmem &s = *reinterpret_cast<PairSmem *>(align_smem_1024(smem_raw));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = pair_rank();
    const int cid = static_cast<int>(blockIdx.x) >> 1, nclusters = static_cast<int>(gridDim.x) >> 1;
    const int num_m = (p.M + PM - 1) / PM, num_n = (p.N + PN - 1) / PN;
    const int num_kb = (p.K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmA);
        prefetch_tensormap(&tmB);
        if (!B_MN) prefetch_tensormap(&tmB64);
        for (int i = 0; i < PSTAGES; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.tfull[i], 1);
            mbar_init(&s.tempty[i], 8);   // the four epilogue warps of each CTA
        }
        fence_barrier_init();
    }
    if (EPI == EPI_DW && threadIdx.x < D * D) s.Am[threadIdx.x] = p.dw.A[threadIdx.x];
    if (warp == 1) {
        // the pair allocates together: both CTAs receive the same columns
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s.tmem_base)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    pair_sync();   // both CTAs' barriers are initialised before any copy or arrival reaches them
    tc_fence_after();
    const uint32_t tmem = s.tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------------ TMA producer (both CTAs)
            int it = 0;
            bool ok = true;
            PairWork wk;
            for (int w = 0; ok && pair_work(w, cid, nclusters, num_m, num_n, wk); ++w) {
                // a half tile's B: 64 rows per CTA of its 128 columns
                const int brows = wk.half < 0 ? PH : PH / 2;
                const int b0 = wk.tn * PN + (wk.half > 0 ? PN / 2 : 0) + static_cast<int>(rank) * brows;
                const uint32_t bytes = 2u * static_cast<uint32_t>(P_HALF + brows * BK * 2);   // the pair's A and B
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int st = it % PSTAGES;
                    if (!mbar_wait(&s.empty[st], ((it / PSTAGES) & 1) ^ 1, p.status)) { ok = false; break; }
                    if (rank == 0) mbar_arrive_expect_tx(&s.full[st], bytes);
                    const uint32_t fb = leader_smem(&s.full[st]);
                    load_half<A_MN>(s.a[st], &tmA, wk.tm * PM + static_cast<int>(rank) * PH, kb * BK, fb);
                    if (wk.half < 0) load_half<B_MN>(s.b[st], &tmB, b0, kb * BK, fb);
                    else if (B_MN) tma_load_2d_to_leader(s.b[st], &tmB, b0, kb * BK, fb);   // one 64-row chunk
                    else tma_load_2d_to_leader(s.b[st], &tmB64, kb * BK, b0, fb);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ------------------------------------------------------------ MMA issuer (leader)
            constexpr uint32_t idesc_whole = idesc_bf16(PM, PN, A_MN, B_MN);
            constexpr uint32_t idesc_half = idesc_bf16(PM, PN / 2, A_MN, B_MN);
            int it = 0, tcount = 0;
            bool ok = true;
            PairWork wk;
            for (int w = 0; ok && pair_work(w, cid, nclusters, num_m, num_n, wk); ++w, ++tcount) {
                const uint32_t idesc = wk.half < 0 ? idesc_whole : idesc_half;
                const int acc = tcount & 1;
                if (!mbar_wait(&s.tempty[acc], ((tcount >> 1) & 1) ^ 1, p.status)) break;
                tc_fence_after();
                const uint32_t dtm = tmem + acc * PN;
                for (int kb = 0; kb < num_kb; ++kb, ++it) {
                    const int st = it % PSTAGES;
                    if (!mbar_wait(&s.full[st], (it / PSTAGES) & 1, p.status)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t abase = smem_u32(s.a[st]), bbase = smem_u32(s.b[st]);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        umma_bf16_pair(dtm, operand_desc<A_MN>(abase, k), operand_desc<B_MN>(bbase, k), idesc,
                                       (kb | k) != 0);
                    }
                    umma_commit_both(&s.empty[st]);
                }
                umma_commit_both(&s.tfull[acc]);
            }
        }
    } else {
        // ---------------------------------------------------------------- epilogue (warps 2..5, both CTAs)
        const int q = warp & 3;   // TMEM lane quarter this warp may access
        float dA[EPI == EPI_DW ? D * D : 1], db[EPI == EPI_DW ? D : 1];
        float Am[EPI == EPI_DW ? D * D : 1];
        if (EPI == EPI_DW) {
#pragma unroll
            for (int i = 0; i < D * D; ++i) { dA[i] = 0.0f; Am[i] = s.Am[i]; }
#pragma unroll
            for (int i = 0; i < D; ++i) db[i] = 0.0f;
        }
        const uint32_t tempty_leader0 = leader_smem(&s.tempty[0]), tempty_leader1 = leader_smem(&s.tempty[1]);
        int tcount = 0;
        PairWork wk;
        for (int w = 0; pair_work(w, cid, nclusters, num_m, num_n, wk); ++w, ++tcount) {
            const int acc = tcount & 1;
            if (!mbar_wait(&s.tfull[acc], (tcount >> 1) & 1, p.status)) break;
            tc_fence_after();
            const int row = wk.tm * PM + static_cast<int>(rank) * PH + q * 32 + lane;
            const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + acc * PN;
            const int col_base = wk.tn * PN + (wk.half > 0 ? PN / 2 : 0);
            const int nchunks = wk.half < 0 ? PN / 32 : PN / 64;
#pragma unroll 1
            for (int c = 0; c < nchunks; ++c) {
                float v[32];
                __syncwarp();   // tcgen05.ld is warp-collective: reconverge after the bounds checks
                tmem_ld32(taddr + c * 32, v);
                epilogue_chunk<EPI, D>(p, v, row, col_base + c * 32, Am, dA, db);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acc ? tempty_leader1 : tempty_leader0);
        }
        // the ring is idle once this CTA's last accumulator is complete (every MMA reading either CTA's
        // stages has completed and no copy is pending): its first stage holds the reduction
        if (EPI == EPI_DW) epilogue_dw_reduce<D>(dA, db, reinterpret_cast<float (*)[72]>(s.a[0]), q, warp, lane, p.dw.partials);
    }

    tc_fence_before();
    __syncthreads();
    pair_sync();   // no copy, commit or arrival of either CTA is still headed for the other
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
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

// Pairs of CTAs (clusters of two) run the paired kernel; the grid is two CTAs per pair tile, at most
// one per SM.
int gemm_grid(int64_t M, int64_t N, int num_sms) {
    const int64_t tiles = ((M + PM - 1) / PM) * ((N + PN - 1) / PN);
    const int64_t pairs = num_sms / 2 > 0 ? num_sms / 2 : 1;
    return static_cast<int>(2 * (tiles < pairs ? (tiles < 1 ? 1 : tiles) : pairs));
}

template <int EPI, int D, bool A_MN, bool B_MN>
static cudaError_t launch_one(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mb64,
                              const GemmParams &gp, int grid, int trace_kind, cudaStream_t st) {
    auto k = gemm_pair_kernel<EPI, D, A_MN, B_MN>;
    const int smem = static_cast<int>(sizeof(PairSmem) + 1024);
    cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void *>(k), smem);
    if (e != cudaSuccess) return e;
    trace_begin(trace_kind, st);
    k<<<grid, kGemmThreads, smem, st>>>(ma, mb, mb64, gp);   // cluster dimensions (2, 1, 1) from the kernel
    trace_end(trace_kind, st);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmProblem &p, GemmEpilogue epi, int num_sms, cudaStream_t st) {
    // mb64: K-major B in 64-row boxes, for the halves of a split last wave
    CUtensorMap ma, mb, mb64;
    if (!make_map(&ma, p.a, p.M, p.K, PH) || !make_map(&mb, p.b, p.N, p.K, PH) || !make_map(&mb64, p.b, p.N, p.K, PH / 2))
        return cudaErrorInvalidValue;
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
        if (!p.a.mn_major && !p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, false, false>(ma, mb, mb64, gp, grid, p.trace_kind, st);
        if (!p.a.mn_major && p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, false, true>(ma, mb, mb64, gp, grid, p.trace_kind, st);
        if (p.a.mn_major && p.b.mn_major) return launch_one<EPI_STORE_BF16, 1, true, true>(ma, mb, mb64, gp, grid, p.trace_kind, st);
        return launch_one<EPI_STORE_BF16, 1, true, false>(ma, mb, mb64, gp, grid, p.trace_kind, st);
    }
    if (!(p.a.mn_major && p.b.mn_major)) return cudaErrorInvalidValue;
    if (p.dw.d == 4) return launch_one<EPI_DW, 4, true, true>(ma, mb, mb64, gp, grid, p.trace_kind, st);
    return launch_one<EPI_DW, 8, true, true>(ma, mb, mb64, gp, grid, p.trace_kind, st);
}

}  // namespace lcq
