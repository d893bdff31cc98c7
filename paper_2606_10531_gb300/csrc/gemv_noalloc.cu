// Allocation-free variant of the packed 2-bit deployment product.
//
// Some callers cannot allocate device memory for the library's scratch: a serving process that hands
// all device memory to its own fixed pool at start-up and must not allocate afterwards, or a C caller
// with no device allocator of its own. For them, lcq_gemm_packed2b_noalloc takes its scratch (the
// transformed activations, the per-token constant and the status word) from one file-scope device
// array instead of a caller-provided workspace. It never calls cudaMalloc, cudaFree or any
// allocating library routine.
//
// The array is shared by every call in the process: calls that may overlap on the GPU (different
// streams, or different host threads) race on it. The first call on each device looks up the array's
// device address with that device current; make that first call before any stream capture.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace lcq {

// Largest problem the static scratch holds: 16 tokens, n <= 32768 (see lcq.h).
constexpr int64_t kNoallocMaxTokens = 16;
constexpr int64_t kNoallocMaxN = 32768;
constexpr size_t kNoallocScratchBytes = (size_t(5) << 18) + 4096;   // 1.25 MiB + 4 KiB

static __device__ __align__(256) unsigned char g_gemv_scratch[kNoallocScratchBytes];

static std::mutex g_noalloc_mu;
static void *g_noalloc_addr[64] = {nullptr};

// Device address of g_gemv_scratch on the current device (looked up once per device).
static cudaError_t noalloc_scratch(void **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_gemv_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_addr[dev] = p;
    }
    *out = g_noalloc_addr[dev];
    return cudaSuccess;
}

}  // namespace lcq

extern "C" lcq_status lcq_gemm_packed2b_noalloc(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m,
                                                int64_t n, int d, const float *A, const float *b, uint16_t *Y,
                                                int32_t *device_status, void *stream) {
    using namespace lcq;
    // every argument is checked before the status word is cleared, so a rejected call enqueues nothing
    const lcq_status arg = check_gemm_packed2b_args(X, N, packed, m, n, d, A, b, Y);
    if (arg != LCQ_OK) return arg;
    if (N > kNoallocMaxTokens || n > kNoallocMaxN) return LCQ_ERR_LIMIT;
    if (device_status && (reinterpret_cast<uintptr_t>(device_status) & 3u)) return LCQ_ERR_ALIGN;
    const size_t need = lcq_workspace_size(LCQ_OP_GEMM_PACKED2B, N, m, n, d);
    if (need > kNoallocScratchBytes) return LCQ_ERR_LIMIT;
    void *scratch = nullptr;
    if (noalloc_scratch(&scratch) != cudaSuccess) return LCQ_ERR_CUDA;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // The status word at the start of the scratch must start each call at LCQ_OK.
    if (cudaMemsetAsync(scratch, 0, 256, st) != cudaSuccess) return LCQ_ERR_CUDA;
    const lcq_status s = lcq_gemm_packed2b(X, N, packed, m, n, d, A, b, Y, scratch, kNoallocScratchBytes, stream);
    if (s != LCQ_OK) return s;
    if (device_status &&
        cudaMemcpyAsync(device_status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return LCQ_ERR_CUDA;
    return LCQ_OK;
}
