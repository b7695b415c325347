// Internal declarations shared by the libaio translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

// Build-time knobs (defaults are the shipped configuration).
#ifndef AIO_RING_KB
#define AIO_RING_KB 24          // shared-memory ring per warp, KB
#endif
#ifndef AIO_WARPS
#define AIO_WARPS 8             // warps per CTA (one CTA per SM)
#endif
#ifndef AIO_FFMA
#define AIO_FFMA 0              // 1: CUDA-core FFMA consumer instead of mma.sync (kept for comparison)
#endif
#ifndef AIO_SLOT_KB
#define AIO_SLOT_KB 8           // bytes per ring slot, KB: one bulk copy of consecutive tiles
#endif
// Ring slots a warp fills with chunks of the next projection once it has finished its tiles of the
// current one (AIO_AHEAD), and while it still has some (AIO_AHEAD_LIVE); the rest of the ring is
// filled when the next projection starts.  Separate values for int8 weights.
#ifndef AIO_AHEAD
#define AIO_AHEAD 2
#endif
#ifndef AIO_AHEAD_LIVE
#define AIO_AHEAD_LIVE 0
#endif
#ifndef AIO_AHEAD_I8
#define AIO_AHEAD_I8 2
#endif
#ifndef AIO_AHEAD_LIVE_I8
#define AIO_AHEAD_LIVE_I8 2
#endif
#ifndef AIO_XBAR_ONLY
#define AIO_XBAR_ONLY 1         // warps 1..7 learn of the grid barrier from the staged x's mbarrier (0: a shared flag)
#endif
#ifndef AIO_SLOT_KB_I8
#define AIO_SLOT_KB_I8 AIO_SLOT_KB   // the same for int8 weights (4 KB tiles)
#endif
// Plain launches with M >= AIO_WIDE_M token rows (int8 weights: M >= AIO_WIDE_M_I8) use a ring of
// AIO_RING_KB_WIDE per warp instead, so that the area left for staged x holds M rows of the
// 4096-column projections (and M <= 4 rows of K = 11008): at such widths a tile's x read from L2
// costs more than a ring slot.  Such launches refill a slot as soon as its tiles are in registers,
// so two slots keep as many copies in flight as three did.  int8 tiles take longer to compute per
// byte, which is why they gain from the wide layout from two rows up.  The chained kernels always use
// the narrow layout.
#ifndef AIO_RING_KB_WIDE
#define AIO_RING_KB_WIDE 16
#endif
#ifndef AIO_WIDE_M
#define AIO_WIDE_M 5
#endif
#ifndef AIO_WIDE_M_I8
#define AIO_WIDE_M_I8 2
#endif

namespace aio {

constexpr int kRows = 16;                   // rows per row group (AIO_ROWS_PER_GROUP)
constexpr int kKT = 256;                    // k columns per tile (AIO_K_TILE)
constexpr int kWarps = AIO_WARPS;           // every warp streams its own tile segment
constexpr int kThreads = kWarps * 32;
constexpr int kSlotBytes = AIO_SLOT_KB * 1024;
constexpr int kSlotBytesI8 = AIO_SLOT_KB_I8 * 1024;
constexpr int kMaxM = 8;
constexpr int kXsPad = 32;                         // elements between staged x rows beyond K (64 B)
constexpr int kSmemBytes = 227 * 1024;             // dynamic shared memory of every stream-kernel launch

// Shared memory of one CTA with a ring of RingKB per warp: the warps' rings, their slot barriers,
// CTA sync words and the x barrier, x-preparation scratch, then the staged x in the rest.
template <int RingKB>
struct SmemLayout {
    static constexpr int kRingBytes = RingKB * 1024;                 // per warp
    static constexpr int kStages = kRingBytes / kSlotBytes;          // bf16 ring slots per warp
    static constexpr int kStagesI8 = kRingBytes / kSlotBytesI8;      // int8 ring slots per warp
    static constexpr int kMaxStages = kStages > kStagesI8 ? kStages : kStagesI8;
    static constexpr int kSyncOffset = kWarps * kRingBytes + kWarps * kMaxStages * 8;   // CTA-level sync words
    static constexpr int kAuxOffset = kSyncOffset + 32;  // sync words (16 B), the x barrier (8 B), padding
    static constexpr int kAuxBytes = kWarps * kMaxM * 4; // per-warp, per-token partial sums (x preparation)
    static constexpr int kXsOffset = kAuxOffset + (kAuxBytes + 15) / 16 * 16;
    static constexpr int kXsBytes = kSmemBytes - kXsOffset;  // x staged when M * (K + kXsPad) * 2 fits
    static_assert(kSlotBytes % 8192 == 0 && kStages >= 2, "a slot holds whole tiles; a ring has >= 2 slots");
    static_assert(kSlotBytesI8 % 4096 == 0 && kStagesI8 >= 2, "a slot holds whole tiles; a ring has >= 2 slots");
    static_assert(kXsOffset % 16 == 0 && kXsBytes > 0, "ring does not fit in shared memory");
};
using NarrowLayout = SmemLayout<AIO_RING_KB>;       // launches of fewer token rows, and every chained launch
using WideLayout = SmemLayout<AIO_RING_KB_WIDE>;    // plain launches of M >= AIO_WIDE_M (int8: AIO_WIDE_M_I8)
// The layout of a launch of MT token rows, int8 or bf16 weights, chained or plain.
template <int MT, bool I8, bool CH>
constexpr bool kWideLaunch = !CH && MT >= (I8 ? AIO_WIDE_M_I8 : AIO_WIDE_M);
template <int MT, bool I8, bool CH>
using LayoutFor = SmemLayout<(kWideLaunch<MT, I8, CH> ? AIO_RING_KB_WIDE : AIO_RING_KB)>;
// The narrow layout's values, for code that runs at every width (the read probe, attention) and for
// the chained step, whose kernels exist for M <= 4 only.
constexpr int kRingBytesPerWarp = NarrowLayout::kRingBytes;
constexpr int kStages = NarrowLayout::kStages;
constexpr int kMaxStages = NarrowLayout::kMaxStages;
constexpr int kXsBytes = NarrowLayout::kXsBytes;

constexpr int kDevErrTimeout = 1;       // a bulk-copy wait expired
constexpr int kDevErrGridTimeout = 2;   // a wait for the previous projection expired
constexpr int kDevErrPrep = 3;          // x preparation asked for a projection whose x is not staged
constexpr int kDevErrAttn = 4;          // a chained step's attention: L_past + M outside [M, L_max]

// How a projection's x is obtained (the values of AIO_X_*).
constexpr int kXGiven = 0, kXRmsNorm = 1, kXSwiGlu = 2, kXSlice = 3, kXAttention = 4;

// Phases of a launch: a projection, or one of the two phases that compute an O projection's x by
// attention over a KV cache in a chained step (the partial results of every warp's units, then
// their merge).
constexpr int kPhaseProj = 0, kPhaseAttn = 1, kPhaseMerge = 2;
// ...or a phase that computes a projection's SwiGLU x into global memory, spread over the grid, when
// it does not fit the staging area (the projection then reads it as a given x).
constexpr int kPhaseSwiGlu = 3;

// Decode attention: heads of 128, units of 16 positions of one head (4 KB of K and 4 KB of V, one
// 8 KB ring slot), partial records of 128 weighted-V sums, the running max, the sum and padding.
constexpr int kHeadDim = 128;
constexpr int kAttnPos = 16;
constexpr int kAttnUnitBytes = kAttnPos * kHeadDim * 2;
constexpr int kAttnSlot = 2 * kAttnUnitBytes;
constexpr int kAttnRec = 132;
// Shared scratch of a chained step's attention merge (it borrows the staged-x area): each warp's
// weighted sums, running max and weight.
constexpr int kAttnMergeScratch = kWarps * 32 * 16 + kWarps * 8;

// One projection of a launch; read-only while the kernel runs.  Geometry:
//   NG  = ceil(N / 8) row groups, NKT = ceil(K / 256) tiles per group, T = NG * NKT tiles;
//   warp z of the Z warps in the grid streams tiles [z*T/Z, (z+1)*T/Z) of every projection.
struct ProjDesc {
    const uint16_t* x;        // [M, K] bf16
    const uint8_t* w;         // packed (or row-major) weights
    const uint16_t* scales;   // [N] bf16 (int8 only)
    float* y;                 // [M, N] fp32
    float* partial;           // [Z][kRows * M] partial sums of split row groups; 0xFF bytes when empty
    int Tq, Tr;               // T = Tq * Z + Tr (Z = warps in the grid): segment bounds in 32-bit arithmetic
    long long T;
    int K, N, NG, NKT;
    int rowmajor;             // 1: W is row-major [N, K]
    int uniform;              // 1: packed, N % 8 == 0 and K % 256 == 0, so tile t is bytes [t, t+1) * tile size
    // x preparation in a chained step (xop != kXGiven): x is computed by every CTA into its staged
    // copy (and by CTA 0 into x itself) from buffers earlier projections wrote.
    const float* xsrc;        // RMSNorm: added to h_in (may be null); SwiGLU, slice: the y read
    const float* h_in;        // RMSNorm: residual stream [M, K]
    float* h_out;             // RMSNorm: h_in + xsrc, written by CTA 0 (may be null)
    const uint16_t* gamma;    // RMSNorm: [K] bf16
    int xop;
    int xsrc_stride;          // elements per token row of xsrc
    int xsrc_off;             // slice: first column
    float eps;                // RMSNorm
    // Attention phases (kind kPhaseAttn / kPhaseMerge) before an O projection: q, k and v of the M
    // new tokens are the column thirds of the QKV output xsrc (xsrc_stride elements per row, head h
    // at columns [128 h, 128 h + 128) of each third).
    uint16_t* kv;             // the layer's cache [2][n_heads][L_max][128] bf16, K then V
    const int* Lpast;         // device int: positions in the cache before this step
    float* apart;             // partial records [Z][2][M][kAttnRec]
    uint16_t* aout;           // merge: the O projection's x [M][n_heads * 128] bf16; SwiGLU phase: x [M][K]
    int kind;                 // kPhase*
    int n_heads, L_max;
    int xfence;               // 1: x may be written earlier in the same launch (fence before staging it)
};
static_assert(sizeof(ProjDesc) % 16 == 0, "descriptor array stride");

// Kernel parameters.  A launch streams nproj projections back to back: projs[] in device memory,
// or the single descriptor `one` when projs is null.  Projection p+1 reads its x only after every
// CTA has finished projection p (done[p] == gridDim.x); done[] and the exit counter are zero at rest.
struct StreamArgs {
    const ProjDesc* projs;
    ProjDesc one;
    unsigned* done;           // [nproj] CTAs finished per projection (nproj > 1 only)
    unsigned* exit_count;     // CTAs that have left the kernel (nproj > 1 only)
    int* err;                 // device error word
    int nproj;
    int M;
    int Z;
    int test_stall;           // 1: the grid's last warp skips its first copy (bounded-wait test)
    unsigned long long wait_limit_ns;
};

struct Geometry {
    int NG, NKT, grid, Z;
    long long T;
};

Geometry geometry(int K, int N, int num_sms);
// Partial-sum slots of one launch: Z * kRows * M floats, rounded up to 256 bytes.  Every slot
// must hold the empty pattern (all bytes 0xFF) when a launch starts; a launch that completes
// without a device error leaves them so.
size_t workspace_bytes(const Geometry& g, int M);

cudaError_t prepare_kernels();  // per-device kernel attributes (dynamic shared memory)
// pdl: programmatic dependent launch; coop: cooperative launch (all CTAs co-resident).
using StreamFn = void (*)(const StreamArgs);
constexpr int kMaxChainM = 4;   // token rows of a chained step (its kernels are instantiated for M <= 4)
static_assert(!kWideLaunch<kMaxChainM, true, true> && !kWideLaunch<kMaxChainM, false, true>,
              "the chained step's staging limit is the narrow layout's");
static_assert(kAttnMergeScratch <= kXsBytes, "the attention merge's scratch fits the staging area");
StreamFn chain_stream_fn(bool i8, int M, bool phases);   // aio_chain.cu
StreamFn chain_phase_stream_fn(bool i8, int M);          // aio_chain_ph.cu
// chained: the chained kernels (x computed on the device); phases: with attention, merge or SwiGLU
// phases.
cudaError_t launch_stream(const StreamArgs& a, bool i8, int grid, cudaStream_t s, bool pdl, bool coop,
                          bool chained = false, bool phases = false);
cudaError_t occupancy(bool i8, int M, bool chained, bool phases, int* blocks_per_sm);
// A projection small enough to launch as one CTA per row group (aio_small.cu): packed weights, at most
// two CTAs per SM, at most 96 KB of weights per CTA (bf16 K <= 2048, int8 K <= 6144).
struct SmallGeometry {
    bool ok;       // the shape qualifies
    int grid;      // CTAs: one per row group
    int tpw;       // tiles per warp: ceil(NKT / 8)
    size_t smem;   // dynamic shared memory per CTA
};
SmallGeometry small_geometry(int K, int N, bool i8, bool rowmajor, int num_sms);
cudaError_t prepare_small_kernels();
cudaError_t launch_small(const StreamArgs& a, bool i8, const SmallGeometry& g, cudaStream_t s, bool pdl);
cudaError_t launch_pack(const void* src, void* dst, int N, int K, int esize, bool inverse, cudaStream_t s);
cudaError_t launch_probe(const void* buf, long long pages, unsigned* out, int grid, cudaStream_t s);

}  // namespace aio
