// aio_api.cu -- the C ABI (include/aio.h): argument validation, handles and their device
// workspaces, kernel launches, and the decode step captured as one CUDA graph.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "aio.h"
#include "aio_attn.h"
#include "aio_pld.h"
#include "aio_internal.h"

namespace {

constexpr uint32_t kLinearMagic = 0xA10113EAu;
constexpr uint32_t kStepMagic = 0xA1057E90u;
constexpr unsigned kCreateFlags = AIO_FLAG_ROWMAJOR | AIO_FLAG_NO_PDL | AIO_FLAG_STREAM_KERNEL | AIO_FLAG_TEST_STALL;
constexpr unsigned kStepFlags = AIO_STEP_GRAPH | AIO_STEP_PDL | AIO_STEP_PERSISTENT;
constexpr unsigned long long kWaitLimitNs = 1000000000ull;      // 1 s: a healthy wait takes microseconds
constexpr unsigned long long kTestWaitLimitNs = 20000000ull;    // 20 ms for AIO_FLAG_TEST_STALL

thread_local char g_last_error[512] = "";

aio_status fail(aio_status s, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return s;
}

#define AIO_CUDA(expr)                                                                             \
    do {                                                                                           \
        cudaError_t e_ = (expr);                                                                   \
        if (e_ != cudaSuccess) return fail(AIO_ERR_CUDA, "%s: %s", #expr, cudaGetErrorString(e_)); \
    } while (0)

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

bool test_alloc_failure() {
    const char* v = getenv("AIO_TEST_FAIL_ALLOC");
    return v && v[0] == '1';
}

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Device checks and one-time kernel attributes per device.
std::mutex g_prep_mu;
bool g_prepared[64] = {};

aio_status current_device(int* dev, int* sms) {
    AIO_CUDA(cudaGetDevice(dev));
    int major = 0, minor = 0;
    AIO_CUDA(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, *dev));
    AIO_CUDA(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, *dev));
    if (major != 10 || minor != 3)
        return fail(AIO_ERR_UNSUPPORTED, "device %d is sm_%d%d; libaio is built for sm_103a (GB300) only", *dev, major,
                    minor);
    AIO_CUDA(cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, *dev));
    std::lock_guard<std::mutex> lk(g_prep_mu);
    if (*dev < 0 || *dev >= 64) return fail(AIO_ERR_UNSUPPORTED, "device ordinal %d out of range", *dev);
    if (!g_prepared[*dev]) {
        AIO_CUDA(aio::prepare_kernels());
        g_prepared[*dev] = true;
    }
    return AIO_OK;
}

aio_status check_device(int dev) {
    int cur = -1;
    AIO_CUDA(cudaGetDevice(&cur));
    if (cur != dev) return fail(AIO_ERR_STATE, "object belongs to device %d but device %d is current", dev, cur);
    return AIO_OK;
}

}  // namespace

namespace aio {

Geometry geometry(int K, int N, int num_sms) {
    Geometry g;
    g.NG = (N + kRows - 1) / kRows;
    g.NKT = (K + kKT - 1) / kKT;
    g.T = static_cast<long long>(g.NG) * g.NKT;
    g.grid = num_sms;
    g.Z = g.grid * kWarps;
    return g;
}

size_t workspace_bytes(const Geometry& g, int M) {
    return round_up(static_cast<size_t>(g.Z) * kRows * M * sizeof(float), 256);
}

}  // namespace aio

struct aio_linear {
    uint32_t magic;
    int K, N, max_M;
    aio_wtype wt;
    unsigned flags;
    int device;
    aio::Geometry geo;
    aio::SmallGeometry small;   // small.ok: aio_linear_run launches one CTA per row group (aio_small.cu)
    void* ws;            // partial-sum slots, then the error word
    size_t ws_bytes;
    float* partial;      // partial-sum slots (empty pattern 0xFF at rest)
    int* err;
};

struct aio_step {
    uint32_t magic;
    int device, M, n;
    unsigned flags;
    bool persistent;
    bool chained;                        // some projection computes its x (the chained kernels run)
    bool phases;                         // attention, merge or SwiGLU phases (their kernel instances)
    bool i8;                             // weight type of every projection (persistent mode)
    int grid;
    std::vector<aio::StreamArgs> chain;  // per-projection launches (chain mode)
    std::vector<char> chain_i8;
    std::vector<aio::SmallGeometry> chain_small;   // chain mode: per-launch small-projection geometry
    aio::StreamArgs whole;               // one launch over the device descriptor array (persistent mode)
    void* ws;                            // workspaces, descriptors, done counters, error words
    size_t ws_bytes;
    int* errs;
    cudaGraph_t graph;
    cudaGraphExec_t exec;
};

namespace {

aio_status valid_linear(aio_linear_t h) {
    if (!h) return fail(AIO_ERR_INVALID_ARG, "null aio_linear_t");
    if (h->magic != kLinearMagic) return fail(AIO_ERR_STATE, "aio_linear_t is not a live handle");
    return AIO_OK;
}

// The descriptor of one projection with weights W [N, K] streamed over geometry geo: the one
// construction behind aio_linear_run, the decode steps and aio_linear_run_noalloc.
aio::ProjDesc make_desc_geo(const aio::Geometry& geo, int K, int N, bool rowmajor, const void* x, const void* W,
                            const void* scales, float* y, float* partial) {
    aio::ProjDesc d = {};
    d.x = static_cast<const uint16_t*>(x);
    d.w = static_cast<const uint8_t*>(W);
    d.scales = static_cast<const uint16_t*>(scales);
    d.y = y;
    d.partial = partial;
    d.T = geo.T;
    d.Tq = static_cast<int>(geo.T / geo.Z);
    d.Tr = static_cast<int>(geo.T % geo.Z);
    d.K = K;
    d.N = N;
    d.NG = geo.NG;
    d.NKT = geo.NKT;
    d.rowmajor = rowmajor ? 1 : 0;
    d.uniform = (!rowmajor && N % aio::kRows == 0 && K % aio::kKT == 0) ? 1 : 0;
    return d;
}

aio::ProjDesc make_desc(const aio_linear* h, const void* x, const void* W, const void* scales, float* y,
                        float* partial) {
    return make_desc_geo(h->geo, h->K, h->N, (h->flags & AIO_FLAG_ROWMAJOR) != 0, x, W, scales, y, partial);
}

// Launch arguments of a single-projection launch (no grid barrier, no done counters).
aio::StreamArgs single_args_geo(const aio::ProjDesc& d, int Z, int M, int* err, bool test_stall) {
    aio::StreamArgs a = {};
    a.projs = nullptr;
    a.one = d;
    a.done = nullptr;
    a.exit_count = nullptr;
    a.err = err;
    a.nproj = 1;
    a.M = M;
    a.Z = Z;
    a.test_stall = test_stall ? 1 : 0;
    a.wait_limit_ns = test_stall ? kTestWaitLimitNs : kWaitLimitNs;
    return a;
}

aio::StreamArgs single_args(const aio_linear* h, const aio::ProjDesc& d, int M, int* err) {
    return single_args_geo(d, h->geo.Z, M, err, (h->flags & AIO_FLAG_TEST_STALL) != 0);
}

// Shape and weight-type checks shared by aio_linear_create and aio_linear_run_noalloc.
aio_status validate_shape(int K, int N, aio_wtype wt) {
    if (K < 16 || K > (1 << 20) || K % 16 != 0) return fail(AIO_ERR_INVALID_ARG, "K=%d: need 16 <= K <= 2^20, K %% 16 == 0", K);
    if (N < 1 || N > (1 << 24)) return fail(AIO_ERR_INVALID_ARG, "N=%d: need 1 <= N <= 2^24", N);
    if (wt != AIO_W_BF16 && wt != AIO_W_INT8_PERCHANNEL) return fail(AIO_ERR_INVALID_ARG, "unknown weight type %d", (int)wt);
    return AIO_OK;
}

// Pointer checks of a run, shared by aio_linear_run, the decode steps and aio_linear_run_noalloc.
aio_status validate_io(aio_wtype wt, const void* x, const void* W, const void* scales, const float* y) {
    if (!x || !W || !y) return fail(AIO_ERR_INVALID_ARG, "x, W and y must be non-NULL");
    if (!aligned(x, 16) || !aligned(W, 16) || !aligned(y, 16))
        return fail(AIO_ERR_ALIGNMENT, "x, W and y must be 16-byte aligned");
    if (wt == AIO_W_INT8_PERCHANNEL) {
        if (!scales) return fail(AIO_ERR_INVALID_ARG, "int8 weights need per-channel scales");
        if (!aligned(scales, 2)) return fail(AIO_ERR_ALIGNMENT, "scales must be 2-byte aligned");
    } else if (scales) {
        return fail(AIO_ERR_INVALID_ARG, "bf16 weights take no scales (pass NULL)");
    }
    return AIO_OK;
}

aio_status validate_run(const aio_linear* h, const void* x, int M, const void* W, const void* scales, const float* y) {
    if (M < 1 || M > h->max_M) return fail(AIO_ERR_INVALID_ARG, "M=%d outside [1, max_M=%d]", M, h->max_M);
    return validate_io(h->wt, x, W, scales, y);
}

}  // namespace

extern "C" {

int aio_abi_version(void) { return AIO_ABI_VERSION; }

const char* aio_status_string(aio_status s) {
    switch (s) {
        case AIO_OK: return "AIO_OK";
        case AIO_ERR_INVALID_ARG: return "AIO_ERR_INVALID_ARG";
        case AIO_ERR_UNSUPPORTED: return "AIO_ERR_UNSUPPORTED";
        case AIO_ERR_ALIGNMENT: return "AIO_ERR_ALIGNMENT";
        case AIO_ERR_CUDA: return "AIO_ERR_CUDA";
        case AIO_ERR_OOM: return "AIO_ERR_OOM";
        case AIO_ERR_STATE: return "AIO_ERR_STATE";
        case AIO_ERR_DEVICE_TIMEOUT: return "AIO_ERR_DEVICE_TIMEOUT";
    }
    return "AIO_ERR_UNKNOWN";
}

const char* aio_last_error(void) { return g_last_error; }

aio_status aio_linear_create(aio_linear_t* out, int K, int N, aio_wtype wt, int max_M, unsigned flags) {
    if (!out) return fail(AIO_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    {
        const aio_status sv = validate_shape(K, N, wt);
        if (sv != AIO_OK) return sv;
    }
    if (max_M < 1 || max_M > aio::kMaxM) return fail(AIO_ERR_INVALID_ARG, "max_M=%d outside [1, 8]", max_M);
    if (flags & ~kCreateFlags) return fail(AIO_ERR_INVALID_ARG, "unknown flags 0x%x", flags & ~kCreateFlags);
    int dev = 0, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    aio::Geometry geo = aio::geometry(K, N, sms);
    const size_t ws = aio::workspace_bytes(geo, max_M);
    if (test_alloc_failure()) return fail(AIO_ERR_OOM, "workspace allocation failed (AIO_TEST_FAIL_ALLOC)");
    void* mem = nullptr;
    if (cudaMalloc(&mem, ws + 256) != cudaSuccess) {
        cudaGetLastError();
        return fail(AIO_ERR_OOM, "cudaMalloc(%zu) failed", ws + 256);
    }
    if (cudaMemset(mem, 0xFF, ws) != cudaSuccess || cudaMemset(static_cast<uint8_t*>(mem) + ws, 0, 256) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess) {
        cudaFree(mem);
        return fail(AIO_ERR_CUDA, "workspace initialisation failed");
    }
    aio_linear* h = new (std::nothrow) aio_linear();
    if (!h) {
        cudaFree(mem);
        return fail(AIO_ERR_OOM, "host allocation failed");
    }
    h->magic = kLinearMagic;
    h->K = K;
    h->N = N;
    h->max_M = max_M;
    h->wt = wt;
    h->flags = flags;
    h->device = dev;
    h->geo = geo;
    h->small = aio::small_geometry(K, N, wt == AIO_W_INT8_PERCHANNEL, (flags & AIO_FLAG_ROWMAJOR) != 0, sms);
    if (flags & AIO_FLAG_STREAM_KERNEL) h->small.ok = false;
    h->ws = mem;
    h->ws_bytes = ws + 256;
    h->partial = static_cast<float*>(mem);
    h->err = reinterpret_cast<int*>(static_cast<uint8_t*>(mem) + ws);
    *out = h;
    return AIO_OK;
}

aio_status aio_linear_packed_bytes(aio_linear_t h, size_t* w_bytes, size_t* scale_bytes) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    const size_t e = h->wt == AIO_W_BF16 ? 2 : 1;
    if (w_bytes) *w_bytes = static_cast<size_t>(h->N) * h->K * e;
    if (scale_bytes) *scale_bytes = h->wt == AIO_W_BF16 ? 0 : static_cast<size_t>(h->N) * 2;
    return AIO_OK;
}

aio_status aio_linear_launch_info(aio_linear_t h, int* grid, int* block, size_t* smem_bytes, long long* tiles) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    if (grid) *grid = h->small.ok ? h->small.grid : h->geo.grid;
    if (block) *block = aio::kThreads;
    if (smem_bytes) *smem_bytes = h->small.ok ? h->small.smem : static_cast<size_t>(aio::kSmemBytes);
    if (tiles) *tiles = h->geo.T;
    return AIO_OK;
}

static aio_status pack_common(aio_linear_t h, const void* src, void* dst, bool inverse, void* stream) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    if ((st = check_device(h->device)) != AIO_OK) return st;
    if (!src || !dst) return fail(AIO_ERR_INVALID_ARG, "weight pointers must be non-NULL");
    if (!aligned(src, 16) || !aligned(dst, 16)) return fail(AIO_ERR_ALIGNMENT, "weight pointers must be 16-byte aligned");
    const size_t e = h->wt == AIO_W_BF16 ? 2 : 1;
    const size_t bytes = static_cast<size_t>(h->N) * h->K * e;
    const uintptr_t a = reinterpret_cast<uintptr_t>(src), b = reinterpret_cast<uintptr_t>(dst);
    if (a < b + bytes && b < a + bytes) return fail(AIO_ERR_INVALID_ARG, "source and destination overlap");
    AIO_CUDA(aio::launch_pack(src, dst, h->N, h->K, static_cast<int>(e), inverse, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

aio_status aio_linear_pack(aio_linear_t h, const void* W_rowmajor, const void* scales, void* W_packed,
                           void* scales_packed, void* stream) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    if (h->wt == AIO_W_INT8_PERCHANNEL) {
        if (!scales || !scales_packed) return fail(AIO_ERR_INVALID_ARG, "int8 weights need scales and scales_packed");
        if (!aligned(scales, 2) || !aligned(scales_packed, 2)) return fail(AIO_ERR_ALIGNMENT, "scales must be 2-byte aligned");
    } else if (scales || scales_packed) {
        return fail(AIO_ERR_INVALID_ARG, "bf16 weights take no scales (pass NULL)");
    }
    if ((st = pack_common(h, W_rowmajor, W_packed, false, stream)) != AIO_OK) return st;
    if (h->wt == AIO_W_INT8_PERCHANNEL && scales != scales_packed)
        AIO_CUDA(cudaMemcpyAsync(scales_packed, scales, static_cast<size_t>(h->N) * 2, cudaMemcpyDeviceToDevice,
                                 static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

aio_status aio_linear_unpack(aio_linear_t h, const void* W_packed, void* W_rowmajor, void* stream) {
    return pack_common(h, W_packed, W_rowmajor, true, stream);
}

aio_status aio_linear_run(aio_linear_t h, const void* x, int M, int K, int N, const void* W, const void* scales,
                          float* y, void* stream) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    if (K != h->K || N != h->N) return fail(AIO_ERR_INVALID_ARG, "K=%d N=%d do not match the handle (K=%d N=%d)", K, N, h->K, h->N);
    if ((st = validate_run(h, x, M, W, scales, y)) != AIO_OK) return st;
    if ((st = check_device(h->device)) != AIO_OK) return st;
    const aio::StreamArgs a = single_args(h, make_desc(h, x, W, scales, y, h->partial), M, h->err);
    const bool i8 = h->wt == AIO_W_INT8_PERCHANNEL, pdl = !(h->flags & AIO_FLAG_NO_PDL);
    if (h->small.ok) {
        AIO_CUDA(aio::launch_small(a, i8, h->small, static_cast<cudaStream_t>(stream), pdl));
    } else {
        AIO_CUDA(aio::launch_stream(a, i8, h->geo.grid, static_cast<cudaStream_t>(stream), pdl, false));
    }
    return AIO_OK;
}

static aio_status read_errors(int device, const int* errs, int n, int* device_error) {
    aio_status st = check_device(device);
    if (st != AIO_OK) return st;
    AIO_CUDA(cudaDeviceSynchronize());
    std::vector<int> host(static_cast<size_t>(n));
    AIO_CUDA(cudaMemcpy(host.data(), errs, sizeof(int) * n, cudaMemcpyDeviceToHost));
    int e = 0;
    for (int v : host) e = e ? e : v;
    if (device_error) *device_error = e;
    if (e) return fail(AIO_ERR_DEVICE_TIMEOUT, "a bounded device wait expired (code %d)", e);
    return AIO_OK;
}

aio_status aio_linear_check(aio_linear_t h, int* device_error) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    return read_errors(h->device, h->err, 1, device_error);
}

aio_status aio_linear_reset(aio_linear_t h) {
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    if ((st = check_device(h->device)) != AIO_OK) return st;
    AIO_CUDA(cudaDeviceSynchronize());
    AIO_CUDA(cudaMemset(h->ws, 0xFF, h->ws_bytes - 256));   // partial slots: empty
    AIO_CUDA(cudaMemset(h->err, 0, 256));
    AIO_CUDA(cudaDeviceSynchronize());
    return AIO_OK;
}

aio_status aio_linear_destroy(aio_linear_t h) {
    if (!h) return AIO_OK;
    aio_status st = valid_linear(h);
    if (st != AIO_OK) return st;
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != h->device) cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    cudaFree(h->ws);
    if (cur != h->device) cudaSetDevice(cur);
    h->magic = 0;
    delete h;
    return AIO_OK;
}

static void step_free(aio_step* s) {
    if (!s) return;
    if (s->exec) cudaGraphExecDestroy(s->exec);
    if (s->graph) cudaGraphDestroy(s->graph);
    if (s->ws) cudaFree(s->ws);
    s->magic = 0;
    delete s;
}

static aio_status step_launch_all(aio_step* s, cudaStream_t stream) {
    if (s->persistent) {
        AIO_CUDA(aio::launch_stream(s->whole, s->i8, s->grid, stream, false, true, s->chained, s->phases));
        return AIO_OK;
    }
    for (int i = 0; i < s->n; ++i) {
        const bool pdl = i > 0 && (s->flags & AIO_STEP_PDL);
        if (s->chain_small[i].ok) {
            AIO_CUDA(aio::launch_small(s->chain[i], s->chain_i8[i] != 0, s->chain_small[i], stream, pdl));
        } else {
            AIO_CUDA(aio::launch_stream(s->chain[i], s->chain_i8[i] != 0, s->grid, stream, pdl, false, s->chained, s->phases));
        }
    }
    return AIO_OK;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Host checks of one projection's x preparation (see aio_decode_step_create_chained).
static aio_status validate_prep(const aio_linear* h, const aio_xprep& x, int M) {
    if (x.op == AIO_X_GIVEN) return AIO_OK;
    const int K = h->K;
    if (x.op == AIO_X_ATTENTION) {
        // x is written by the step's merge phase and then staged like a given x
        if (!x.src || !x.kv_cache || !x.L_past) return fail(AIO_ERR_INVALID_ARG, "ATTENTION needs src, kv_cache and L_past");
        if (x.n_heads < 1 || static_cast<long long>(x.n_heads) * aio::kHeadDim != K)
            return fail(AIO_ERR_INVALID_ARG, "ATTENTION needs K = 128 n_heads (K=%d, n_heads=%d)", K, x.n_heads);
        if (x.n_heads > h->geo.Z) return fail(AIO_ERR_UNSUPPORTED, "n_heads=%d above the %d warps of the grid", x.n_heads, h->geo.Z);
        if (x.L_max < M || static_cast<long long>(x.n_heads) * ((x.L_max + aio::kAttnPos - 1) / aio::kAttnPos) > (1LL << 30))
            return fail(AIO_ERR_INVALID_ARG, "ATTENTION needs M <= L_max and n_heads * L_max / 16 <= 2^30 (L_max=%d)", x.L_max);
        if (x.src_stride < 3LL * K) return fail(AIO_ERR_INVALID_ARG, "src_stride %d < 3K (%d)", x.src_stride, 3 * K);
        if (!aligned16(x.src) || !aligned16(x.kv_cache) || !aligned(x.L_past, 4) || x.src_stride % 4 != 0)
            return fail(AIO_ERR_ALIGNMENT, "src and kv_cache must be 16-byte aligned, L_past 4-byte, src_stride a multiple of 4");
        return AIO_OK;
    }
    if (x.op != AIO_X_RMSNORM && x.op != AIO_X_SWIGLU && x.op != AIO_X_SLICE)
        return fail(AIO_ERR_INVALID_ARG, "unknown x preparation %d", x.op);
    // a SwiGLU x that does not fit is computed by a grid-wide phase instead (see step_create)
    if (x.op != AIO_X_SWIGLU && static_cast<long long>(M) * (K + aio::kXsPad) * 2 > aio::kXsBytes)
        return fail(AIO_ERR_UNSUPPORTED, "a computed x needs M (K + 32) 2 <= %d bytes (M=%d, K=%d)", aio::kXsBytes, M, K);
    if (x.op == AIO_X_RMSNORM) {
        if (!x.h_in || !x.gamma) return fail(AIO_ERR_INVALID_ARG, "RMSNORM needs h_in and gamma");
        if (!(x.eps >= 0.0f) || !std::isfinite(x.eps)) return fail(AIO_ERR_INVALID_ARG, "eps must be finite and >= 0");
        if (x.h_out && (x.h_out == x.h_in || x.h_out == x.src))
            return fail(AIO_ERR_INVALID_ARG, "h_out must differ from h_in and src");
        if (!aligned16(x.h_in) || !aligned16(x.gamma) || !aligned16(x.h_out) || !aligned16(x.src))
            return fail(AIO_ERR_ALIGNMENT, "h_in, h_out, src and gamma must be 16-byte aligned");
        return AIO_OK;
    }
    if (!x.src) return fail(AIO_ERR_INVALID_ARG, "SWIGLU and SLICE need src");
    if (!aligned16(x.src) || x.src_stride % 4 != 0 || x.src_off % 4 != 0)
        return fail(AIO_ERR_ALIGNMENT, "src must be 16-byte aligned, src_stride and src_off multiples of 4");
    const long long need = x.op == AIO_X_SWIGLU ? 2LL * K : static_cast<long long>(x.src_off) + K;
    if (x.src_off < 0 || x.src_stride < need)
        return fail(AIO_ERR_INVALID_ARG, "columns [%lld, %lld) outside src_stride %d", need - K, need, x.src_stride);
    return AIO_OK;
}

// A SwiGLU x too large for the staging area: computed into the projection's x by its own phase.
static bool swiglu_phase(const aio_linear* h, const aio_xprep& x, int M) {
    return x.op == AIO_X_SWIGLU && static_cast<long long>(M) * (h->K + aio::kXsPad) * 2 > aio::kXsBytes;
}

static void apply_prep(aio::ProjDesc& d, const aio_xprep& x, bool own_phase) {
    if (x.op == AIO_X_ATTENTION || own_phase) return;   // an earlier phase writes x: staged (or read) as given
    d.xop = x.op;
    d.xsrc = x.src;
    d.xsrc_stride = x.op == AIO_X_RMSNORM ? d.K : x.src_stride;
    d.xsrc_off = x.src_off;
    d.h_in = x.h_in;
    d.h_out = x.h_out;
    d.gamma = static_cast<const uint16_t*>(x.gamma);
    d.eps = x.eps;
}

static aio_status step_create(aio_step_t* out, const aio_proj* projs, const aio_xprep* preps, int n_projs, int M,
                              unsigned flags) {
    if (!out) return fail(AIO_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!projs || n_projs < 1) return fail(AIO_ERR_INVALID_ARG, "need at least one projection");
    if (flags & ~kStepFlags) return fail(AIO_ERR_INVALID_ARG, "unknown step flags 0x%x", flags & ~kStepFlags);
    if (M < 1 || M > aio::kMaxM) return fail(AIO_ERR_INVALID_ARG, "M=%d outside [1, 8]", M);
    const bool persistent = (flags & AIO_STEP_PERSISTENT) != 0;
    int dev = -1;
    {
        aio_status st = valid_linear(projs[0].h);
        if (st != AIO_OK) return st;
        dev = projs[0].h->device;
    }
    const aio_wtype wt0 = projs[0].h->wt;
    size_t total = 0;
    std::vector<size_t> offs(static_cast<size_t>(n_projs));
    for (int i = 0; i < n_projs; ++i) {
        const aio_proj& p = projs[i];
        aio_status st = valid_linear(p.h);
        if (st != AIO_OK) return fail(st, "projection %d: %s", i, g_last_error);
        if (p.h->device != dev) return fail(AIO_ERR_STATE, "projection %d is on device %d, not %d", i, p.h->device, dev);
        if (persistent && p.h->wt != wt0)
            return fail(AIO_ERR_UNSUPPORTED, "a persistent step needs one weight type (projection %d differs)", i);
        if ((st = validate_run(p.h, p.x, M, p.W, p.scales, p.y)) != AIO_OK)
            return fail(st, "projection %d: %s", i, g_last_error);
        if (preps && (st = validate_prep(p.h, preps[i], M)) != AIO_OK)
            return fail(st, "projection %d: %s", i, g_last_error);
        offs[i] = total;
        total += aio::workspace_bytes(p.h->geo, M);
    }
    aio_status st = check_device(dev);
    if (st != AIO_OK) return st;
    const int grid = projs[0].h->geo.grid;
    bool chained = false;
    for (int i = 0; preps && i < n_projs; ++i) chained = chained || preps[i].op != AIO_X_GIVEN;
    if (chained && M > aio::kMaxChainM)
        return fail(AIO_ERR_UNSUPPORTED, "a chained step supports M <= %d (M=%d)", aio::kMaxChainM, M);
    bool phases = false;
    for (int i = 0; preps && i < n_projs; ++i)
        phases = phases || preps[i].op == AIO_X_ATTENTION || swiglu_phase(projs[i].h, preps[i], M);
    if (persistent) {
        int blocks = 0;
        AIO_CUDA(aio::occupancy(wt0 == AIO_W_INT8_PERCHANNEL, M, chained, phases, &blocks));
        if (blocks < 1) return fail(AIO_ERR_UNSUPPORTED, "the stream kernel cannot be resident on an SM");
    }
    // Phases: every projection, and before a projection whose x is attention over a KV cache, the
    // attention phase and its merge.
    int n_attn = 0, n_swiglu = 0;
    for (int i = 0; preps && i < n_projs; ++i) {
        n_attn += preps[i].op == AIO_X_ATTENTION ? 1 : 0;
        n_swiglu += swiglu_phase(projs[i].h, preps[i], M) ? 1 : 0;
    }
    const int n_phases = n_projs + 2 * n_attn + n_swiglu;
    const size_t apart_off = total;   // the attention phases' partial records (shared by the layers)
    if (n_attn) total += round_up(static_cast<size_t>(projs[0].h->geo.Z) * 2 * M * aio::kAttnRec * sizeof(float), 256);
    const size_t desc_off = total;
    total += round_up(sizeof(aio::ProjDesc) * n_phases, 256);
    const size_t done_off = total;
    total += round_up(sizeof(unsigned) * (n_phases + 1), 256);
    const size_t err_off = total;
    total += round_up(sizeof(int) * n_phases, 256);
    if (test_alloc_failure()) return fail(AIO_ERR_OOM, "workspace allocation failed (AIO_TEST_FAIL_ALLOC)");
    aio_step* s = new (std::nothrow) aio_step();
    if (!s) return fail(AIO_ERR_OOM, "host allocation failed");
    s->magic = kStepMagic;
    s->device = dev;
    s->M = M;
    s->n = n_phases;
    s->flags = flags;
    s->persistent = persistent;
    s->chained = chained;
    s->phases = phases;
    s->i8 = wt0 == AIO_W_INT8_PERCHANNEL;
    s->grid = grid;
    s->ws_bytes = total;
    if (cudaMalloc(&s->ws, total) != cudaSuccess) {
        cudaGetLastError();
        s->ws = nullptr;
        step_free(s);
        return fail(AIO_ERR_OOM, "cudaMalloc(%zu) failed", total);
    }
    uint8_t* base = static_cast<uint8_t*>(s->ws);
    s->errs = reinterpret_cast<int*>(base + err_off);
    std::vector<aio::ProjDesc> descs;
    for (int i = 0; i < n_projs; ++i) {
        const aio_proj& p = projs[i];
        const bool i8 = p.h->wt == AIO_W_INT8_PERCHANNEL;
        if (preps && preps[i].op == AIO_X_ATTENTION) {
            const aio_xprep& x = preps[i];
            aio::ProjDesc a = {};
            a.kind = aio::kPhaseAttn;
            a.x = static_cast<const uint16_t*>(p.x);
            a.K = a.N = p.h->K;
            a.NG = a.NKT = 1;
            a.xsrc = x.src;
            a.xsrc_stride = x.src_stride;
            a.kv = static_cast<uint16_t*>(x.kv_cache);
            a.Lpast = x.L_past;
            a.n_heads = x.n_heads;
            a.L_max = x.L_max;
            a.apart = reinterpret_cast<float*>(base + apart_off);
            a.aout = static_cast<uint16_t*>(const_cast<void*>(p.x));
            for (int kind : {aio::kPhaseAttn, aio::kPhaseMerge}) {
                a.kind = kind;
                descs.push_back(a);
                const int e = static_cast<int>(descs.size()) - 1;
                s->chain.push_back(aio::StreamArgs{});
                s->chain.back() = single_args(p.h, a, M, s->errs + e);
                s->chain_i8.push_back(i8 ? 1 : 0);
                s->chain_small.push_back(aio::SmallGeometry{});
            }
        }
        const bool own = preps && swiglu_phase(p.h, preps[i], M);
        if (own) {
            aio::ProjDesc g = {};
            g.kind = aio::kPhaseSwiGlu;
            g.x = static_cast<const uint16_t*>(p.x);
            g.K = g.N = p.h->K;
            g.NG = g.NKT = 1;
            g.xsrc = preps[i].src;
            g.xsrc_stride = preps[i].src_stride;
            g.aout = static_cast<uint16_t*>(const_cast<void*>(p.x));
            descs.push_back(g);
            s->chain.push_back(single_args(p.h, g, M, s->errs + (descs.size() - 1)));
            s->chain_i8.push_back(i8 ? 1 : 0);
            s->chain_small.push_back(aio::SmallGeometry{});
        }
        descs.push_back(make_desc(p.h, p.x, p.W, p.scales, p.y, reinterpret_cast<float*>(base + offs[i])));
        if (preps) apply_prep(descs.back(), preps[i], own);
        s->chain.push_back(single_args(p.h, descs.back(), M, s->errs + (descs.size() - 1)));
        s->chain_i8.push_back(i8 ? 1 : 0);
        // a plain projection of a step without computed x: the small-projection launch if it qualifies
        s->chain_small.push_back(chained ? aio::SmallGeometry{} : p.h->small);
    }
    // A projection whose x overlaps a buffer an earlier phase of the step writes (y, a computed x, a
    // residual stream, an attention or SwiGLU output, a KV cache) reads data written in the same
    // launch: it fences before staging x (generic stores, then async-proxy reads).
    {
        std::vector<std::pair<uintptr_t, uintptr_t>> written;
        auto add = [&](const void* p, size_t n) {
            if (p && n) written.emplace_back(reinterpret_cast<uintptr_t>(p), reinterpret_cast<uintptr_t>(p) + n);
        };
        for (aio::ProjDesc& d : descs) {
            const size_t xb = static_cast<size_t>(M) * d.K * 2;
            if (d.kind == aio::kPhaseProj) {
                const uintptr_t a = reinterpret_cast<uintptr_t>(d.x);
                for (const auto& r : written) d.xfence |= (a < r.second && r.first < a + xb) ? 1 : 0;
                add(d.y, static_cast<size_t>(M) * d.N * 4);
                if (d.xop != aio::kXGiven) add(d.x, xb);
                add(d.h_out, static_cast<size_t>(M) * d.K * 4);
            } else if (d.kind == aio::kPhaseAttn) {
                add(d.kv, static_cast<size_t>(2) * d.n_heads * d.L_max * aio::kHeadDim * 2);
            } else {
                add(d.aout, xb);
            }
        }
    }
    aio::StreamArgs w = {};
    w.projs = reinterpret_cast<const aio::ProjDesc*>(base + desc_off);
    w.done = reinterpret_cast<unsigned*>(base + done_off);
    w.exit_count = w.done + n_phases;
    w.err = s->errs;
    w.nproj = n_phases;
    w.M = M;
    w.Z = projs[0].h->geo.Z;
    w.test_stall = 0;
    w.wait_limit_ns = kWaitLimitNs;
    s->whole = w;
    if (cudaMemset(s->ws, 0xFF, desc_off) != cudaSuccess ||
        cudaMemset(base + desc_off, 0, total - desc_off) != cudaSuccess ||
        cudaMemcpy(base + desc_off, descs.data(), sizeof(aio::ProjDesc) * n_phases, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess) {
        step_free(s);
        return fail(AIO_ERR_CUDA, "step workspace initialisation failed");
    }
    if (flags & AIO_STEP_GRAPH) {
        cudaStream_t cs = nullptr;
        if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
            step_free(s);
            return fail(AIO_ERR_CUDA, "capture stream creation failed");
        }
        aio_status lst = AIO_OK;
        if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
            lst = fail(AIO_ERR_CUDA, "cudaStreamBeginCapture failed");
        } else {
            lst = step_launch_all(s, cs);
            cudaGraph_t g = nullptr;
            const cudaError_t ec = cudaStreamEndCapture(cs, &g);
            if (lst == AIO_OK && ec != cudaSuccess) lst = fail(AIO_ERR_CUDA, "cudaStreamEndCapture: %s", cudaGetErrorString(ec));
            s->graph = g;
            if (lst == AIO_OK) {
                const cudaError_t ei = cudaGraphInstantiate(&s->exec, s->graph, 0);
                if (ei != cudaSuccess) lst = fail(AIO_ERR_CUDA, "cudaGraphInstantiate: %s", cudaGetErrorString(ei));
            }
        }
        cudaStreamDestroy(cs);
        if (lst != AIO_OK) {
            cudaGetLastError();
            step_free(s);
            return lst;
        }
    }
    *out = s;
    return AIO_OK;
}

aio_status aio_decode_step_create(aio_step_t* out, const aio_proj* projs, int n_projs, int M, unsigned flags) {
    return step_create(out, projs, nullptr, n_projs, M, flags);
}

aio_status aio_decode_step_create_chained(aio_step_t* out, const aio_proj* projs, const aio_xprep* preps,
                                          int n_projs, int M, unsigned flags) {
    return step_create(out, projs, preps, n_projs, M, flags);
}

static aio_status valid_step(aio_step_t s) {
    if (!s) return fail(AIO_ERR_INVALID_ARG, "null aio_step_t");
    if (s->magic != kStepMagic) return fail(AIO_ERR_STATE, "aio_step_t is not a live step");
    return AIO_OK;
}

aio_status aio_decode_step(aio_step_t s, void* stream) {
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    if ((st = check_device(s->device)) != AIO_OK) return st;
    if (s->exec) {
        AIO_CUDA(cudaGraphLaunch(s->exec, static_cast<cudaStream_t>(stream)));
        return AIO_OK;
    }
    return step_launch_all(s, static_cast<cudaStream_t>(stream));
}

aio_status aio_decode_step_host(aio_step_t s, const void* x_host, void* x_dev, size_t x_bytes, const void* y_dev,
                                void* y_host, size_t y_bytes, void* stream) {
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    if ((x_bytes && (!x_host || !x_dev)) || (y_bytes && (!y_host || !y_dev)))
        return fail(AIO_ERR_INVALID_ARG, "a copy of non-zero size needs both of its pointers");
    if ((st = check_device(s->device)) != AIO_OK) return st;
    const cudaStream_t cs = static_cast<cudaStream_t>(stream);
    if (x_bytes) AIO_CUDA(cudaMemcpyAsync(x_dev, x_host, x_bytes, cudaMemcpyHostToDevice, cs));
    if ((st = aio_decode_step(s, stream)) != AIO_OK) return st;
    if (y_bytes) AIO_CUDA(cudaMemcpyAsync(y_host, y_dev, y_bytes, cudaMemcpyDeviceToHost, cs));
    return AIO_OK;
}

aio_status aio_decode_step_kernels(aio_step_t s, int* n_kernels) {
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    if (n_kernels) *n_kernels = s->persistent ? 1 : s->n;
    return AIO_OK;
}

aio_status aio_decode_step_reset(aio_step_t s) {
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    if ((st = check_device(s->device)) != AIO_OK) return st;
    const size_t desc_off = reinterpret_cast<const uint8_t*>(s->whole.projs) - static_cast<const uint8_t*>(s->ws);
    const size_t done_off = reinterpret_cast<const uint8_t*>(s->whole.done) - static_cast<const uint8_t*>(s->ws);
    AIO_CUDA(cudaDeviceSynchronize());
    AIO_CUDA(cudaMemset(s->ws, 0xFF, desc_off));   // partial-sum slots: empty
    AIO_CUDA(cudaMemset(static_cast<uint8_t*>(s->ws) + done_off, 0, s->ws_bytes - done_off));  // done, errors
    AIO_CUDA(cudaDeviceSynchronize());
    return AIO_OK;
}

aio_status aio_decode_step_check(aio_step_t s, int* device_error) {
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    return read_errors(s->device, s->errs, s->n, device_error);
}

aio_status aio_decode_step_destroy(aio_step_t s) {
    if (!s) return AIO_OK;
    aio_status st = valid_step(s);
    if (st != AIO_OK) return st;
    const int dev = s->device;
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != dev) cudaSetDevice(dev);
    cudaDeviceSynchronize();
    step_free(s);
    if (cur != dev) cudaSetDevice(cur);
    return AIO_OK;
}

aio_status aio_probe_read(const void* buf, size_t bytes, unsigned* out, void* stream) {
    if (!buf || !out) return fail(AIO_ERR_INVALID_ARG, "buf and out must be non-NULL");
    if (bytes == 0 || bytes % 4096 != 0) return fail(AIO_ERR_INVALID_ARG, "bytes must be a positive multiple of 4096");
    if (!aligned(buf, 16) || !aligned(out, 4)) return fail(AIO_ERR_ALIGNMENT, "buf must be 16-byte aligned, out 4-byte");
    int dev = 0, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    AIO_CUDA(aio::launch_probe(buf, static_cast<long long>(bytes / 4096), out, sms, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------------------------
// aio_linear_run_noalloc: the stream kernel's single-projection launch (aio_linear_run's launch for
// a handle created with AIO_FLAG_STREAM_KERNEL) with its cross-warp
// scratch (partial sums of row groups split between warps) in one static
// device array that is part of the library image, instead of a handle's cudaMalloc'd workspace.
// It is for callers that cannot allocate device memory where they call: a serving engine that has
// handed nearly all of HBM to its own pools (weights, KV cache), so that a cudaMalloc there fails,
// or a hot loop in which cudaMalloc / cudaFree would synchronise the device.

static __device__ __align__(256) unsigned char aio_noalloc_scratch[AIO_NOALLOC_SCRATCH_BYTES];

namespace {

std::mutex g_noalloc_mu;
void* g_noalloc_base[64] = {};   // device address of aio_noalloc_scratch, per device ordinal

// Looked up once per device, with that device current (the caller made it current).
aio_status noalloc_scratch(int dev, void** out) {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_base[dev]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, aio_noalloc_scratch);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(AIO_ERR_CUDA, "cudaGetSymbolAddress(scratch) on device %d: %s", dev, cudaGetErrorString(e));
        }
        if (!p || !aligned(p, 256)) return fail(AIO_ERR_CUDA, "static scratch on device %d is not 256-byte aligned", dev);
        g_noalloc_base[dev] = p;
    }
    *out = g_noalloc_base[dev];
    return AIO_OK;
}

}  // namespace

extern "C" aio_status aio_linear_run_noalloc(const void* x, int M, int K, int N, aio_wtype wt, unsigned flags,
                                             const void* W, const void* scales, float* y, int* device_error,
                                             void* stream) {
    aio_status st = validate_shape(K, N, wt);
    if (st != AIO_OK) return st;
    if (M < 1 || M > aio::kMaxM) return fail(AIO_ERR_INVALID_ARG, "M=%d outside [1, 8]", M);
    const unsigned allowed = AIO_FLAG_ROWMAJOR | AIO_FLAG_NO_PDL;
    if (flags & ~allowed) return fail(AIO_ERR_INVALID_ARG, "unknown flags 0x%x (ROWMAJOR and NO_PDL only)", flags & ~allowed);
    if (!device_error) return fail(AIO_ERR_INVALID_ARG, "device_error must be non-NULL");
    if ((st = validate_io(wt, x, W, scales, y)) != AIO_OK) return st;
    if (!aligned(device_error, 4)) return fail(AIO_ERR_ALIGNMENT, "device_error must be 4-byte aligned");
    int dev = 0, sms = 0;
    st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    const aio::Geometry geo = aio::geometry(K, N, sms);
    const size_t need = aio::workspace_bytes(geo, M);
    size_t limit = AIO_NOALLOC_SCRATCH_BYTES;
    if (const char* t = getenv("AIO_TEST_NOALLOC_BYTES"))   // test hook: a smaller limit
        limit = std::min(limit, static_cast<size_t>(strtoull(t, nullptr, 10)));
    if (need > limit)
        return fail(AIO_ERR_INVALID_ARG,
                    "K=%d N=%d M=%d needs %zu bytes of scratch; the static scratch holds %zu "
                    "(use aio_linear_create + aio_linear_run)", K, N, M, need, limit);
    void* base = nullptr;
    if ((st = noalloc_scratch(dev, &base)) != AIO_OK) return st;
    float* partial = static_cast<float*>(base);
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The partial-sum slots must start empty (all bytes 0xFF); a healthy run leaves them so, an
    // expired wait may not, and the array starts out zeroed.
    AIO_CUDA(cudaMemsetAsync(partial, 0xFF, need, s));
    const aio::ProjDesc d = make_desc_geo(geo, K, N, (flags & AIO_FLAG_ROWMAJOR) != 0, x, W, scales, y, partial);
    const aio::StreamArgs a = single_args_geo(d, geo.Z, M, device_error, false);
    AIO_CUDA(aio::launch_stream(a, wt == AIO_W_INT8_PERCHANNEL, geo.grid, s, !(flags & AIO_FLAG_NO_PDL), false));
    return AIO_OK;
}

// ------------------------------------------------------------------ decode attention
extern "C" aio_status aio_attention_workspace_bytes(int M, size_t* bytes) {
    if (!bytes) return fail(AIO_ERR_INVALID_ARG, "bytes is NULL");
    if (M < 1 || M > aio::kMaxM) return fail(AIO_ERR_INVALID_ARG, "M=%d outside [1, 8]", M);
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    *bytes = aio::attn_workspace_bytes(sms * aio::kWarps, M);
    return AIO_OK;
}

extern "C" aio_status aio_attention_decode(const float* q, int q_stride, const void* k_cache, const void* v_cache,
                                           int n_heads, int head_dim, int L_max, int L, int M, float* out,
                                           void* workspace, size_t workspace_bytes, void* stream) {
    if (!q || !k_cache || !v_cache || !out || !workspace)
        return fail(AIO_ERR_INVALID_ARG, "q, k_cache, v_cache, out and workspace must be non-NULL");
    if (head_dim != 128) return fail(AIO_ERR_UNSUPPORTED, "head_dim=%d: only 128 is supported", head_dim);
    if (M < 1 || M > aio::kMaxM) return fail(AIO_ERR_INVALID_ARG, "M=%d outside [1, 8]", M);
    if (n_heads < 1 || L < M || L > L_max)
        return fail(AIO_ERR_INVALID_ARG, "need n_heads >= 1 and M <= L <= L_max (n_heads=%d M=%d L=%d L_max=%d)",
                    n_heads, M, L, L_max);
    if (q_stride < n_heads * 128) return fail(AIO_ERR_INVALID_ARG, "q_stride=%d < n_heads * 128", q_stride);
    const uintptr_t mis = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_cache) |
                          reinterpret_cast<uintptr_t>(v_cache) | reinterpret_cast<uintptr_t>(out) |
                          reinterpret_cast<uintptr_t>(workspace);
    if ((mis & 15u) || q_stride % 4 != 0)
        return fail(AIO_ERR_ALIGNMENT, "q, the caches, out and workspace must be 16-byte aligned, q_stride a multiple of 4");
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    if (n_heads > sms * aio::kWarps)
        return fail(AIO_ERR_UNSUPPORTED, "n_heads=%d above %d (warps in the grid)", n_heads, sms * aio::kWarps);
    const size_t need = aio::attn_workspace_bytes(sms * aio::kWarps, M);
    if (workspace_bytes < need) return fail(AIO_ERR_INVALID_ARG, "workspace of %zu bytes, %zu needed", workspace_bytes, need);
    AIO_CUDA(aio::launch_attention(q, q_stride, k_cache, v_cache, n_heads, L_max, L, M, out, workspace, sms,
                                   kWaitLimitNs, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

extern "C" aio_status aio_attention_check(void* workspace, int* device_error) {
    if (!workspace) return fail(AIO_ERR_INVALID_ARG, "workspace is NULL");
    int dev = -1;
    AIO_CUDA(cudaGetDevice(&dev));
    AIO_CUDA(cudaDeviceSynchronize());
    int e = 0;
    AIO_CUDA(cudaMemcpy(&e, workspace, sizeof e, cudaMemcpyDeviceToHost));
    if (e) AIO_CUDA(cudaMemset(workspace, 0, sizeof e));
    if (device_error) *device_error = e;
    if (e) return fail(AIO_ERR_DEVICE_TIMEOUT, "a bounded device wait expired (code %d)", e);
    return AIO_OK;
}

// ------------------------------------------------------------------ prompt-lookup decoding
extern "C" aio_status aio_pld_draft(const int* tokens, int T, int N, int L, int* out, void* stream) {
    if (!tokens || !out) return fail(AIO_ERR_INVALID_ARG, "tokens and out must be non-NULL");
    if (T < 1 || N < 1 || N > aio::kPldMaxN || L < 1 || L > aio::kPldMaxL)
        return fail(AIO_ERR_INVALID_ARG, "need T >= 1, 1 <= N <= %d, 1 <= L <= %d (T=%d N=%d L=%d)", aio::kPldMaxN,
                    aio::kPldMaxL, T, N, L);
    if ((reinterpret_cast<uintptr_t>(tokens) | reinterpret_cast<uintptr_t>(out)) & 3u)
        return fail(AIO_ERR_ALIGNMENT, "tokens and out must be 4-byte aligned");
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    AIO_CUDA(aio::launch_pld_draft(tokens, T, N, L, out, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

extern "C" aio_status aio_argmax_rows(const float* logits, int M, int V, int stride, int* out, void* stream) {
    if (!logits || !out) return fail(AIO_ERR_INVALID_ARG, "logits and out must be non-NULL");
    if (M < 1 || M > 65535 || V < 1 || stride < V)
        return fail(AIO_ERR_INVALID_ARG, "need 1 <= M <= 65535, V >= 1, stride >= V (M=%d V=%d stride=%d)", M, V, stride);
    if ((reinterpret_cast<uintptr_t>(logits) | reinterpret_cast<uintptr_t>(out)) & 3u)
        return fail(AIO_ERR_ALIGNMENT, "logits and out must be 4-byte aligned");
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    AIO_CUDA(aio::launch_argmax(logits, M, V, stride, out, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

extern "C" aio_status aio_pld_accept(const int* argmax, const int* draft, int* result, void* stream) {
    if (!argmax || !draft || !result) return fail(AIO_ERR_INVALID_ARG, "argmax, draft and result must be non-NULL");
    if ((reinterpret_cast<uintptr_t>(argmax) | reinterpret_cast<uintptr_t>(draft) | reinterpret_cast<uintptr_t>(result)) & 3u)
        return fail(AIO_ERR_ALIGNMENT, "argmax, draft and result must be 4-byte aligned");
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    AIO_CUDA(aio::launch_pld_accept(argmax, draft, result, static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}

extern "C" aio_status aio_route(const float* logits, const int* category_tokens, int n_categories, int code_index,
                                int L_ctx, float tau, int* decision, void* stream) {
    if (!logits || !category_tokens || !decision)
        return fail(AIO_ERR_INVALID_ARG, "logits, category_tokens and decision must be non-NULL");
    if (n_categories < 1 || n_categories > 32 || code_index < 0 || code_index >= n_categories || L_ctx < 0 ||
        !(tau >= 0.0f) || !std::isfinite(tau))
        return fail(AIO_ERR_INVALID_ARG, "need 1 <= n_categories <= 32, 0 <= code_index < n_categories, L_ctx >= 0, "
                                         "finite tau >= 0");
    if ((reinterpret_cast<uintptr_t>(logits) | reinterpret_cast<uintptr_t>(category_tokens) |
         reinterpret_cast<uintptr_t>(decision)) & 3u)
        return fail(AIO_ERR_ALIGNMENT, "logits, category_tokens and decision must be 4-byte aligned");
    int dev = -1, sms = 0;
    aio_status st = current_device(&dev, &sms);
    if (st != AIO_OK) return st;
    AIO_CUDA(aio::launch_route(logits, category_tokens, n_categories, code_index, L_ctx, tau, decision,
                               static_cast<cudaStream_t>(stream)));
    return AIO_OK;
}
