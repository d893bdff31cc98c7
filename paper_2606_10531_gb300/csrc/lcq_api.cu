// C ABI of liblcq: argument validation, workspace carving and kernel dispatch.
// See include/lcq.h for the contract of every entry point.
#include <atomic>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace lcq {

static std::atomic<uint64_t> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// ---------------------------------------------------------------- CUDA-event kernel tracing
struct TraceRec {
    int kind;
    cudaEvent_t start, stop;
};
static bool g_trace_on = false;
static int g_trace_n = 0;
static TraceRec g_trace[LCQ_TRACE_CAPACITY];
static bool g_trace_pool_ready = false;

static bool trace_pool() {
    if (g_trace_pool_ready) return true;
    for (int i = 0; i < LCQ_TRACE_CAPACITY; ++i) {
        if (cudaEventCreate(&g_trace[i].start) != cudaSuccess) return false;
        if (cudaEventCreate(&g_trace[i].stop) != cudaSuccess) return false;
    }
    g_trace_pool_ready = true;
    return true;
}

void trace_begin(int kind, cudaStream_t st) {
    if (!g_trace_on || g_trace_n >= LCQ_TRACE_CAPACITY) return;
    g_trace[g_trace_n].kind = kind;
    cudaEventRecord(g_trace[g_trace_n].start, st);
}

void trace_end(int kind, cudaStream_t st) {
    if (!g_trace_on || g_trace_n >= LCQ_TRACE_CAPACITY || g_trace[g_trace_n].kind != kind) return;
    cudaEventRecord(g_trace[g_trace_n].stop, st);
    ++g_trace_n;
}

void *tensor_map_encoder() {
    static std::once_flag once;
    static void *fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = p;
    });
    return fn;
}

cudaError_t ensure_dynamic_smem(const void *fn, int bytes) {
    struct Entry {
        const void *fn;
        int dev, bytes;
    };
    static std::mutex mu;
    static Entry done[256];
    static int ndone = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < ndone; ++i)
        if (done[i].fn == fn && done[i].dev == dev && done[i].bytes >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && ndone < 256) done[ndone++] = {fn, dev, bytes};
    return e;
}

static int num_sms_current() {
    // per-device cache; calls from several host threads may fill an entry at once (same value)
    static std::atomic<int> cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (dev >= 0 && dev < 64) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    if (dev >= 0 && dev < 64) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

static inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
static inline bool al16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
static inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

constexpr size_t kHeader = 256;           // status word + counter
constexpr int kMaxGemmCtas = 1024;        // upper bound on the persistent GEMM grid

struct Header {
    int32_t status;
    uint32_t counter;
    uint32_t pad[14];
    uint32_t batch_counters[kEncodeBatchMax];   // lcq_encode_batch, one per matrix
};
static_assert(sizeof(Header) <= kHeader, "workspace header");

static lcq_status check_common(int64_t m, int64_t n, int d) {
    if (d != 4 && d != 8) return LCQ_ERR_UNSUPPORTED;
    if (m < 0 || n < 0) return LCQ_ERR_SHAPE;
    if (n % 8 != 0 || n % d != 0) return LCQ_ERR_SHAPE;
    if (m > (int64_t(1) << 31) || n > (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    return LCQ_OK;
}

// A tensor of `elems` elements: NULL allowed only when empty; must be 16-byte aligned.
static lcq_status check_tensor(const void *p, int64_t elems, bool required = true) {
    if (elems == 0) return LCQ_OK;
    if (!p) return required ? LCQ_ERR_NULL : LCQ_OK;
    if (!al16(p)) return LCQ_ERR_ALIGN;
    return LCQ_OK;
}

static lcq_status check_ws(void *ws, size_t ws_bytes, size_t need) {
    if (!ws) return LCQ_ERR_WORKSPACE;
    if (!al16(ws) || (reinterpret_cast<uintptr_t>(ws) & 255u)) return LCQ_ERR_ALIGN;
    if (ws_bytes < need) return LCQ_ERR_WORKSPACE;
    return LCQ_OK;
}

static std::atomic<int> g_last_cuda_error{0};

static lcq_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return LCQ_OK;
    g_last_cuda_error.store(static_cast<int>(e), std::memory_order_relaxed);
    return LCQ_ERR_CUDA;
}

static lcq_status opts_of(const lcq_opts *o, float &inv_s, float &t, int &ste, float *dge_k = nullptr,
                          float *dge_cap = nullptr) {
    float s = 1.0f, k = 5.0f, cap = 3.0f;
    t = 0.0f;
    ste = LCQ_STE_IDENTITY;
    if (o) {
        s = o->latent_scale;
        t = o->latent_offset;
        ste = o->ste_mode;
        if (o->reserved != 0) return LCQ_ERR_ARG;
        if (o->dge_k > 0.0f) k = o->dge_k;
        if (o->dge_grad_max > 0.0f) cap = o->dge_grad_max;
    }
    if (!(s != 0.0f) || !isfinite(s) || !isfinite(t) || !isfinite(k) || !isfinite(cap)) return LCQ_ERR_ARG;
    if (ste != LCQ_STE_IDENTITY && ste != LCQ_STE_CLIPPED && ste != LCQ_STE_DGE) return LCQ_ERR_UNSUPPORTED;
    inv_s = 1.0f / s;
    if (dge_k) *dge_k = k;
    if (dge_cap) *dge_cap = cap;
    return LCQ_OK;
}

// Argument checks of lcq_gemm_packed2b (everything but the workspace); also used by the
// allocation-free variant before it enqueues anything.
lcq_status check_gemm_packed2b_args(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n, int d,
                                    const float *A, const float *b, const uint16_t *Y) {
    lcq_status s = check_common(m, n, d);
    if (s != LCQ_OK) return s;
    if (N < 0 || N > (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    if ((s = check_tensor(X, N * n)) != LCQ_OK) return s;
    if ((s = check_tensor(packed, m * n)) != LCQ_OK) return s;
    if ((s = check_tensor(Y, N * m)) != LCQ_OK) return s;
    if (!A || !b) return LCQ_ERR_NULL;
    return LCQ_OK;
}

}  // namespace lcq

using namespace lcq;

#define LCQ_TRY(x)                          \
    do {                                    \
        lcq_status _s = (x);                \
        if (_s != LCQ_OK) return _s;        \
    } while (0)

extern "C" {

size_t lcq_workspace_size(int op, int64_t N, int64_t m, int64_t n, int d) {
    if (N < 0 || m < 0 || n < 0 || (d != 4 && d != 8)) return 0;
    const size_t mn = static_cast<size_t>(m) * static_cast<size_t>(n);
    switch (op) {
        case LCQ_OP_ENCODE:
            return kHeader + align256(sizeof(double) * 2 * 1024);
        case LCQ_OP_ENCODE_BATCH:
            if (N < 1 || N > kEncodeBatchMax) return 0;
            return kHeader + align256(sizeof(double) * kEncodeBatchPartials * static_cast<size_t>(N));
        case LCQ_OP_LINEAR_FWD:
            return kHeader + align256(mn * 2);
        case LCQ_OP_LINEAR_BWD:
            return kHeader + align256(mn * 2) + align256(sizeof(float) * kMaxGemmCtas * (d * d + d));
        case LCQ_OP_GEMM_PACKED2B:
            return kHeader + packed_gemv_workspace(N, n);
        case LCQ_OP_GEMM_PACKED2B_HADAMARD:
            return kHeader + align256(static_cast<size_t>(N) * static_cast<size_t>(n) * 4) + packed_gemv_workspace(N, n);
        case LCQ_OP_LDL_FACTOR:
            return kHeader + ldl_factor_scratch_bytes(n);
        case LCQ_OP_LDLQ:
            return kHeader + align256(ldlq_history_bytes(m, n)) + align256(sizeof(double) * ldlq_tiles(m));
        default:
            return 0;
    }
}

const char *lcq_status_string(lcq_status s) {
    switch (s) {
        case LCQ_OK: return "ok";
        case LCQ_ERR_NULL: return "a required pointer is NULL";
        case LCQ_ERR_SHAPE: return "invalid shape (negative size, n % d != 0 or n % 8 != 0)";
        case LCQ_ERR_ALIGN: return "pointer not 16-byte aligned (workspace: 256-byte)";
        case LCQ_ERR_UNSUPPORTED: return "unsupported parameter (d must be 4 or 8; STE mode)";
        case LCQ_ERR_WORKSPACE: return "workspace missing or too small";
        case LCQ_ERR_CUDA: return "CUDA runtime error";
        case LCQ_ERR_SINGULAR: return "A is singular";
        case LCQ_ERR_TIMEOUT: return "device pipeline wait timed out";
        case LCQ_ERR_ARG: return "invalid argument";
        case LCQ_ERR_LIMIT: return "problem exceeds the static scratch of the allocation-free call";
        default: return "unknown status";
    }
}

uint64_t lcq_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char *lcq_last_cuda_error(void) {
    const int e = g_last_cuda_error.load(std::memory_order_relaxed);
    return e == 0 ? "no error" : cudaGetErrorString(static_cast<cudaError_t>(e));
}

lcq_status lcq_trace_enable(int on) {
    if (on) {
        if (!trace_pool()) return LCQ_ERR_CUDA;
        g_trace_n = 0;
        g_trace_on = true;
    } else {
        g_trace_on = false;
    }
    return LCQ_OK;
}

lcq_status lcq_trace_read(int kind, uint64_t *launches, double *total_ms) {
    if (!launches || !total_ms) return LCQ_ERR_NULL;
    if (kind < 0 || kind >= LCQ_K_NUM_KINDS) return LCQ_ERR_ARG;
    uint64_t cnt = 0;
    double tot = 0.0;
    for (int i = 0; i < g_trace_n; ++i) {
        if (g_trace[i].kind != kind) continue;
        if (cudaEventSynchronize(g_trace[i].stop) != cudaSuccess) return LCQ_ERR_CUDA;
        float ms = 0.0f;
        if (cudaEventElapsedTime(&ms, g_trace[i].start, g_trace[i].stop) != cudaSuccess) return LCQ_ERR_CUDA;
        tot += ms;
        ++cnt;
    }
    *launches = cnt;
    *total_ms = tot;
    return LCQ_OK;
}

lcq_status lcq_device_status(const void *ws, void *stream, int32_t *status_out, int clear) {
    if (!ws || !status_out) return LCQ_ERR_NULL;
    cudaStream_t st = as_stream(stream);
    int32_t v = 0;
    if (cudaMemcpyAsync(&v, ws, sizeof(int32_t), cudaMemcpyDeviceToHost, st) != cudaSuccess) return LCQ_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return LCQ_ERR_CUDA;
    *status_out = v;
    if (clear) {
        if (cudaMemsetAsync(const_cast<void *>(ws), 0, sizeof(int32_t), st) != cudaSuccess) return LCQ_ERR_CUDA;
        if (cudaStreamSynchronize(st) != cudaSuccess) return LCQ_ERR_CUDA;
    }
    return LCQ_OK;
}

lcq_status lcq_hadamard(const float *in, int64_t rows, int64_t n, float *out, void *stream) {
    if (rows < 0 || n < 0 || n % 8 != 0) return LCQ_ERR_SHAPE;
    if (rows * n == 0) return LCQ_OK;
    LCQ_TRY(check_tensor(in, rows * n));
    LCQ_TRY(check_tensor(out, rows * n));
    return cuda_status(launch_hadamard(in, false, rows, n, out, as_stream(stream)));
}

lcq_status lcq_gemm_packed2b_hadamard(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n,
                                      int d, const float *A, const float *b, uint16_t *Y, void *ws, size_t ws_bytes,
                                      void *stream) {
    LCQ_TRY(check_common(m, n, d));
    if (N < 0 || N > (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    LCQ_TRY(check_tensor(X, N * n));
    LCQ_TRY(check_tensor(packed, m * n));
    LCQ_TRY(check_tensor(Y, N * m));
    if (!A || !b) return LCQ_ERR_NULL;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_GEMM_PACKED2B_HADAMARD, N, m, n, d)));
    cudaStream_t st = as_stream(stream);
    if (N * m == 0) return LCQ_OK;
    if (n == 0) return cuda_status(cudaMemsetAsync(Y, 0, sizeof(uint16_t) * N * m, st));
    Header *h = static_cast<Header *>(ws);
    float *Xr = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + kHeader);
    uint8_t *base = static_cast<uint8_t *>(ws) + kHeader + align256(static_cast<size_t>(N) * static_cast<size_t>(n) * 4);
    {
        // the rotation runs inside the product (the one-token kernel's prologue or the tcgen05
        // kernel's prep) where one of those kernels takes the shape
        PackedGemvArgs a;
        a.X = X; a.Xf = nullptr; a.N = N; a.m = m; a.n = n; a.packed = packed; a.A = A; a.b = b; a.Y = Y;
        a.Xp = reinterpret_cast<uint16_t *>(base);
        a.corr = reinterpret_cast<float *>(base + packed_gemv_corr_offset(N, n));
        a.status = &h->status;
        cudaError_t err;
        if (launch_packed_gemv_rotated(a, d, num_sms_current(), st, err)) return cuda_status(err);
        LCQ_TRY(cuda_status(err));
    }
    trace_begin(LCQ_K_GEMV, st);
    const cudaError_t e = launch_hadamard(X, true, N, n, Xr, st);
    trace_end(LCQ_K_GEMV, st);
    LCQ_TRY(cuda_status(e));
    PackedGemvArgs a;
    a.X = X; a.Xf = Xr; a.N = N; a.m = m; a.n = n; a.packed = packed; a.A = A; a.b = b; a.Y = Y;
    a.Xp = reinterpret_cast<uint16_t *>(base);
    a.corr = reinterpret_cast<float *>(base + packed_gemv_corr_offset(N, n));
    a.status = &h->status;
    return cuda_status(launch_packed_gemv(a, d, num_sms_current(), st));
}

lcq_status lcq_ldl_factor(const float *H, int64_t n, int d, float *U, float *D, void *ws, size_t ws_bytes,
                          void *stream) {
    LCQ_TRY(check_common(0, n, d));
    if (n == 0) return LCQ_OK;
    if (n > 65536) return LCQ_ERR_SHAPE;
    LCQ_TRY(check_tensor(H, n * n));
    LCQ_TRY(check_tensor(U, n * n));
    LCQ_TRY(check_tensor(D, n * d, false));
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_LDL_FACTOR, 0, 0, n, d)));
    cudaStream_t st = as_stream(stream);
    Header *h = static_cast<Header *>(ws);
    LdlFactorArgs a{H, n, d, U, D, reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + kHeader), &h->status};
    trace_begin(LCQ_K_LDL_FACTOR, st);
    const cudaError_t e = launch_ldl_factor(a, st);
    trace_end(LCQ_K_LDL_FACTOR, st);
    return cuda_status(e);
}

lcq_status lcq_ldlq(const float *W, int64_t m, int64_t n, int d, const float *A, const float *b, const float *U,
                    uint8_t *packed, uint8_t *codes, float *latent, double *mse, void *ws, size_t ws_bytes,
                    void *stream) {
    LCQ_TRY(check_common(m, n, d));
    const int64_t mn = m * n;
    LCQ_TRY(check_tensor(W, mn));
    LCQ_TRY(check_tensor(U, n * n));
    LCQ_TRY(check_tensor(packed, mn, false));
    LCQ_TRY(check_tensor(codes, mn, false));
    LCQ_TRY(check_tensor(latent, mn, false));
    if (!A || !b) return LCQ_ERR_NULL;
    if (ldlq_tiles(m) * n >= (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_LDLQ, 0, m, n, d)));
    cudaStream_t st = as_stream(stream);
    if (mn == 0) return mse ? cuda_status(cudaMemsetAsync(mse, 0, sizeof(double), st)) : LCQ_OK;
    Header *h = static_cast<Header *>(ws);
    uint8_t *base = static_cast<uint8_t *>(ws) + kHeader;
    LdlqArgs a{W, m, n, d, A, b, U, packed, codes, latent, mse, reinterpret_cast<float *>(base),
               reinterpret_cast<double *>(base + align256(ldlq_history_bytes(m, n))), &h->status};
    trace_begin(LCQ_K_LDLQ, st);
    const cudaError_t e = launch_ldlq(a, st);
    trace_end(LCQ_K_LDLQ, st);
    return cuda_status(e);
}

lcq_status lcq_init_codebook(const float *G, int d, float *A, float *b, void *stream) {
    if (d != 4 && d != 8) return LCQ_ERR_UNSUPPORTED;
    if (!G || !A || !b) return LCQ_ERR_NULL;
    return cuda_status(launch_init_codebook(G, d, A, b, as_stream(stream)));
}

lcq_status lcq_init_latent(const uint8_t *packed, int64_t m, int64_t n, float *P, float *s_out, float *t_out,
                           void *stream) {
    if (m < 0 || n < 0 || n % 4 != 0) return LCQ_ERR_SHAPE;
    if (m + n == 0) return LCQ_ERR_SHAPE;
    const double a = sqrt(6.0 / static_cast<double>(m + n));
    const float s = static_cast<float>(2.0 * a / 3.0);
    const float t = 1.5f;
    if (s_out) *s_out = s;
    if (t_out) *t_out = t;
    const int64_t mn = m * n;
    if (mn == 0) return LCQ_OK;
    LCQ_TRY(check_tensor(packed, mn));
    LCQ_TRY(check_tensor(P, mn));
    return cuda_status(launch_init_latent(packed, mn, s, t, P, num_sms_current(), as_stream(stream)));
}

lcq_status lcq_selftest_wait_timeout(void *ws, void *stream) {
    if (!ws) return LCQ_ERR_NULL;
    if (reinterpret_cast<uintptr_t>(ws) & 255u) return LCQ_ERR_ALIGN;
    Header *h = static_cast<Header *>(ws);
    return cuda_status(launch_wait_timeout_selftest(&h->status, as_stream(stream)));
}

lcq_status lcq_encode(const float *W, int64_t m, int64_t n, int d, const float *A, const float *b, uint8_t *packed,
                      uint8_t *codes, float *latent, double *mse, void *ws, size_t ws_bytes, void *stream) {
    LCQ_TRY(check_common(m, n, d));
    const int64_t mn = m * n;
    LCQ_TRY(check_tensor(W, mn));
    if (!A || !b) return LCQ_ERR_NULL;
    LCQ_TRY(check_tensor(packed, mn, false));
    LCQ_TRY(check_tensor(codes, mn, false));
    LCQ_TRY(check_tensor(latent, mn, false));
    if (mse && (reinterpret_cast<uintptr_t>(mse) & 7u)) return LCQ_ERR_ALIGN;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_ENCODE, 0, m, n, d)));
    cudaStream_t st = as_stream(stream);
    if (mn == 0) {
        if (mse) return cuda_status(cudaMemsetAsync(mse, 0, sizeof(double), st));
        return LCQ_OK;
    }
    Header *h = static_cast<Header *>(ws);
    EncodeArgs a;
    a.W = W; a.m = m; a.n = n; a.A = A; a.b = b;
    a.packed = packed; a.codes = codes; a.latent = latent; a.mse = mse;
    a.partials = reinterpret_cast<double *>(static_cast<uint8_t *>(ws) + kHeader);
    a.counter = &h->counter;
    a.status = &h->status;
    return cuda_status(launch_encode(a, d, num_sms_current(), st));
}

lcq_status lcq_encode_batch(const lcq_encode_item *items, int count, int d, void *ws, size_t ws_bytes, void *stream) {
    if (!items) return LCQ_ERR_NULL;
    if (count < 1 || count > kEncodeBatchMax) return LCQ_ERR_SHAPE;
    if (d != 4 && d != 8) return LCQ_ERR_UNSUPPORTED;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_ENCODE_BATCH, count, 0, 0, d)));
    EncodeBatchArgs a;
    std::memset(&a, 0, sizeof(a));
    const int64_t chunk = encode_chunk_size();
    int64_t c0 = 0;
    for (int i = 0; i < count; ++i) {
        const lcq_encode_item &it = items[i];
        LCQ_TRY(check_common(it.m, it.n, d));
        const int64_t mn = it.m * it.n;
        LCQ_TRY(check_tensor(it.W, mn));
        if (!it.A || !it.b) return LCQ_ERR_NULL;
        LCQ_TRY(check_tensor(it.packed, mn, false));
        LCQ_TRY(check_tensor(it.codes, mn, false));
        LCQ_TRY(check_tensor(it.latent, mn, false));
        if (it.mse && (reinterpret_cast<uintptr_t>(it.mse) & 7u)) return LCQ_ERR_ALIGN;
        EncodeBatchItem &e = a.item[i];
        e.W = it.W; e.m = it.m; e.n = it.n; e.A = it.A; e.b = it.b;
        e.packed = it.packed; e.codes = it.codes; e.latent = it.latent; e.mse = it.mse;
        e.chunk0 = c0;
        e.nchunks = (mn + chunk - 1) / chunk;
        c0 += e.nchunks;
    }
    a.count = count;
    a.total_chunks = c0;
    cudaStream_t st = as_stream(stream);
    if (c0 == 0) {
        // every matrix is empty: the MSE of an empty matrix is 0
        for (int i = 0; i < count; ++i)
            if (items[i].mse) LCQ_TRY(cuda_status(cudaMemsetAsync(items[i].mse, 0, sizeof(double), st)));
        return LCQ_OK;
    }
    Header *h = static_cast<Header *>(ws);
    a.partials = reinterpret_cast<double *>(static_cast<uint8_t *>(ws) + kHeader);
    a.counters = h->batch_counters;
    a.status = &h->status;
    return cuda_status(launch_encode_batch(a, d, num_sms_current(), st));
}

lcq_status lcq_decode(const uint8_t *packed, int64_t m, int64_t n, int d, const float *A, const float *b,
                      float *W_hat_f32, uint16_t *W_hat_bf16, void *stream) {
    LCQ_TRY(check_common(m, n, d));
    const int64_t mn = m * n;
    if (mn == 0) return LCQ_OK;
    LCQ_TRY(check_tensor(packed, mn));
    if (!A || !b) return LCQ_ERR_NULL;
    if (!W_hat_f32 && !W_hat_bf16) return LCQ_ERR_NULL;
    LCQ_TRY(check_tensor(W_hat_f32, mn, false));
    LCQ_TRY(check_tensor(W_hat_bf16, mn, false));
    DecodeArgs a;
    a.packed = packed; a.m = m; a.n = n; a.A = A; a.b = b; a.W_f32 = W_hat_f32; a.W_bf16 = W_hat_bf16;
    return cuda_status(launch_decode(a, d, num_sms_current(), as_stream(stream)));
}

lcq_status lcq_activation_transform(const uint16_t *X, int64_t N, int64_t n, int d, const float *A, const float *b,
                                    uint16_t *Xp, float *r, void *stream) {
    LCQ_TRY(check_common(0, n, d));
    if (N < 0 || N > (int64_t(1) << 31) - 1) return LCQ_ERR_SHAPE;
    if (N == 0) return LCQ_OK;
    if (!Xp && !r) return LCQ_ERR_NULL;
    LCQ_TRY(check_tensor(X, N * n));
    LCQ_TRY(check_tensor(Xp, N * n, false));
    LCQ_TRY(check_tensor(r, N, false));
    if (!A || !b) return LCQ_ERR_NULL;
    if (n == 0) return r ? cuda_status(cudaMemsetAsync(r, 0, sizeof(float) * N, as_stream(stream))) : LCQ_OK;
    return cuda_status(launch_xform(X, N, n, d, A, b, Xp, r, as_stream(stream)));
}

lcq_status lcq_pack2b(const uint8_t *codes, int64_t m, int64_t n, uint8_t *packed, void *stream) {
    if (m < 0 || n < 0) return LCQ_ERR_SHAPE;
    if (n % 4 != 0) return LCQ_ERR_SHAPE;
    const int64_t mn = m * n;
    if (mn == 0) return LCQ_OK;
    LCQ_TRY(check_tensor(codes, mn));
    LCQ_TRY(check_tensor(packed, mn));
    return cuda_status(launch_pack2b(codes, mn, packed, num_sms_current(), as_stream(stream)));
}

lcq_status lcq_linear_fwd(const uint16_t *X, int64_t N, const float *P, int64_t m, int64_t n, int d, const float *A,
                          const float *b, const lcq_opts *opts, uint16_t *Y, uint8_t *packed_saved, void *ws,
                          size_t ws_bytes, void *stream) {
    LCQ_TRY(check_common(m, n, d));
    if (N < 0 || N > (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    float inv_s, t;
    int ste;
    LCQ_TRY(opts_of(opts, inv_s, t, ste));
    LCQ_TRY(check_tensor(X, N * n));
    LCQ_TRY(check_tensor(P, m * n));
    LCQ_TRY(check_tensor(Y, N * m));
    LCQ_TRY(check_tensor(packed_saved, m * n, false));
    if (!A || !b) return LCQ_ERR_NULL;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_LINEAR_FWD, N, m, n, d)));
    cudaStream_t st = as_stream(stream);
    const int sms = num_sms_current();
    Header *h = static_cast<Header *>(ws);
    uint16_t *W_hat = reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(ws) + kHeader);
    if (m * n > 0) {
        QuantDecodeArgs q;
        q.P = P; q.m = m; q.n = n; q.A = A; q.b = b; q.inv_s = inv_s; q.t = t;
        q.packed = packed_saved; q.W_hat = W_hat; q.status = &h->status;
        LCQ_TRY(cuda_status(launch_quant_decode(q, d, sms, st)));
    }
    if (N * m == 0) return LCQ_OK;
    if (n == 0) return cuda_status(cudaMemsetAsync(Y, 0, sizeof(uint16_t) * N * m, st));
    GemmProblem g;
    std::memset(&g, 0, sizeof(g));
    g.M = N; g.N = m; g.K = n;
    g.a = {X, n, false};
    g.b = {W_hat, n, false};
    g.C = Y; g.ldc = m;
    g.status = &h->status;
    g.trace_kind = LCQ_K_GEMM_FWD;
    return cuda_status(launch_gemm(g, EPI_STORE_BF16, sms, st));
}

lcq_status lcq_linear_bwd(const uint16_t *X, const uint16_t *dY, const uint8_t *packed_saved, const float *P, int64_t N,
                          int64_t m, int64_t n, int d, const float *A, const float *b, const lcq_opts *opts,
                          uint16_t *dX, float *dP, float *dA, float *db, void *ws, size_t ws_bytes, void *stream) {
    LCQ_TRY(check_common(m, n, d));
    if (N < 0 || N > (int64_t(1) << 31)) return LCQ_ERR_SHAPE;
    // dY is a TMA operand of both backward GEMMs: its rows (m bf16) must span a multiple of 16 bytes
    if (m % 8 != 0) return LCQ_ERR_SHAPE;
    float inv_s, t, dge_k, dge_cap;
    int ste;
    LCQ_TRY(opts_of(opts, inv_s, t, ste, &dge_k, &dge_cap));
    LCQ_TRY(check_tensor(X, N * n));
    LCQ_TRY(check_tensor(dY, N * m));
    LCQ_TRY(check_tensor(packed_saved, m * n));
    LCQ_TRY(check_tensor(P, m * n, ste != LCQ_STE_IDENTITY));
    LCQ_TRY(check_tensor(dX, N * n, false));
    LCQ_TRY(check_tensor(dP, m * n));
    if (!A || !b || !dA || !db) return LCQ_ERR_NULL;
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_LINEAR_BWD, N, m, n, d)));
    cudaStream_t st = as_stream(stream);
    const int sms = num_sms_current();
    Header *h = static_cast<Header *>(ws);
    uint16_t *W_hat = reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(ws) + kHeader);
    float *partials = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + kHeader +
                                                align256(static_cast<size_t>(m) * static_cast<size_t>(n) * 2));

    // dX = dY W_hat
    if (dX && N * n > 0) {
        if (m == 0) {
            LCQ_TRY(cuda_status(cudaMemsetAsync(dX, 0, sizeof(uint16_t) * N * n, st)));
        } else {
            DecodeArgs da;
            da.packed = packed_saved; da.m = m; da.n = n; da.A = A; da.b = b; da.W_f32 = nullptr; da.W_bf16 = W_hat;
            LCQ_TRY(cuda_status(launch_decode(da, d, sms, st)));
            GemmProblem g;
            std::memset(&g, 0, sizeof(g));
            g.M = N; g.N = n; g.K = m;
            g.a = {dY, m, false};
            g.b = {W_hat, n, true};
            g.C = dX; g.ldc = n;
            g.status = &h->status;
            g.trace_kind = LCQ_K_GEMM_DX;
            LCQ_TRY(cuda_status(launch_gemm(g, EPI_STORE_BF16, sms, st)));
        }
    }
    // dW_hat = dY^T X  ->  dP, dA, db
    if (m * n == 0 || N == 0) {
        if (m * n > 0) LCQ_TRY(cuda_status(cudaMemsetAsync(dP, 0, sizeof(float) * m * n, st)));
        LCQ_TRY(cuda_status(cudaMemsetAsync(dA, 0, sizeof(float) * d * d, st)));
        return cuda_status(cudaMemsetAsync(db, 0, sizeof(float) * d, st));
    }
    GemmProblem g;
    std::memset(&g, 0, sizeof(g));
    g.M = m; g.N = n; g.K = N;
    g.a = {dY, m, true};
    g.b = {X, n, true};
    g.dw.packed = packed_saved;
    g.dw.A = A;
    g.dw.P = ste != LCQ_STE_IDENTITY ? P : nullptr;
    g.dw.dge_inv_k = 1.0f / dge_k;
    g.dw.dge_exp = 1.0f / dge_k - 1.0f;
    g.dw.dge_cap = dge_cap;
    g.dw.dP = dP;
    g.dw.partials = partials;
    g.dw.inv_s = inv_s;
    g.dw.t = t;
    g.dw.ste_mode = ste;
    g.dw.d = d;
    g.status = &h->status;
    g.trace_kind = LCQ_K_GEMM_DW;
    LCQ_TRY(cuda_status(launch_gemm(g, EPI_DW, sms, st)));
    return cuda_status(launch_reduce_partials(partials, gemm_grid(m, n, sms), d, dA, db, st));
}

lcq_status lcq_gemm_packed2b(const uint16_t *X, int64_t N, const uint8_t *packed, int64_t m, int64_t n, int d,
                             const float *A, const float *b, uint16_t *Y, void *ws, size_t ws_bytes, void *stream) {
    LCQ_TRY(check_gemm_packed2b_args(X, N, packed, m, n, d, A, b, Y));
    LCQ_TRY(check_ws(ws, ws_bytes, lcq_workspace_size(LCQ_OP_GEMM_PACKED2B, N, m, n, d)));
    cudaStream_t st = as_stream(stream);
    if (N * m == 0) return LCQ_OK;
    if (n == 0) return cuda_status(cudaMemsetAsync(Y, 0, sizeof(uint16_t) * N * m, st));
    Header *h = static_cast<Header *>(ws);
    uint8_t *base = static_cast<uint8_t *>(ws) + kHeader;
    PackedGemvArgs a;
    a.X = X; a.Xf = nullptr; a.N = N; a.m = m; a.n = n; a.packed = packed; a.A = A; a.b = b; a.Y = Y;
    a.Xp = reinterpret_cast<uint16_t *>(base);
    a.corr = reinterpret_cast<float *>(base + packed_gemv_corr_offset(N, n));
    a.status = &h->status;
    return cuda_status(launch_packed_gemv(a, d, num_sms_current(), st));
}

}  // extern "C"
