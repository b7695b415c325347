// Internal declarations shared by the libaio translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace aio {

constexpr int kRows = 8;                    // rows per row group (AIO_ROWS_PER_GROUP)
constexpr int kKT = 256;                    // k columns per tile (AIO_K_TILE)
constexpr int kWarps = 8;                   // warps per CTA; every warp streams its own tile segment
constexpr int kThreads = kWarps * 32;
constexpr int kRingBytesPerWarp = 12 * 1024;  // per-warp shared-memory ring (3 bf16 tiles / 6 int8 tiles)
constexpr int kMaxStages = 6;
constexpr int kSmemBytes = kWarps * kRingBytesPerWarp + kWarps * kMaxStages * 8;
constexpr int kMaxM = 8;

constexpr int kDevErrTimeout = 1;

// Everything one launch of the linear kernel needs.  Geometry:
//   NG  = ceil(N / 8) row groups, NKT = ceil(K / 256) tiles per group, T = NG * NKT tiles
//   Z   = grid * kWarps warps; warp z streams tiles [z*T/Z, (z+1)*T/Z)
struct GemvArgs {
    const uint16_t* x;        // [M, K] bf16
    const uint8_t* w;         // packed (or row-major) weights
    const uint16_t* scales;   // [N] bf16 (int8 only)
    float* y;                 // [M, N] fp32
    float* partial;           // [Z][2][kRows * M] partial sums of row groups split between warps
    unsigned* counters;       // [NG] tiles accumulated so far per split row group; 0 between launches
    int* err;                 // device error word
    long long T;              // total tiles
    int M, K, N;
    int NG, NKT;
    int Z;
    int rowmajor;             // 1: W is row-major [N, K]
    int test_stall;           // 1: the grid's last warp skips its first copy (bounded-wait test)
    unsigned long long wait_limit_ns;
};

struct Geometry {
    int NG, NKT, grid, Z;
    long long T;
};

Geometry geometry(int K, int N, int num_sms);
size_t workspace_bytes(const Geometry& g, int M);   // partial + counters + error word, 256-B aligned parts
void carve_workspace(void* base, const Geometry& g, int M, float** partial, unsigned** counters, int** err);

cudaError_t prepare_kernels();  // per-device kernel attributes (dynamic shared memory)
cudaError_t launch_gemv(const GemvArgs& a, bool i8, int grid, cudaStream_t s, bool pdl);
cudaError_t launch_pack(const void* src, void* dst, int N, int K, int esize, bool inverse, cudaStream_t s);
cudaError_t launch_probe(const void* buf, long long chunks, unsigned* out, int grid, cudaStream_t s);

}  // namespace aio
