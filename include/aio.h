/*
 * aio.h -- C ABI of libaio: decode-step weight-streaming linear layers on GB300 (sm_103a).
 *
 * The computation (A-IO, arxiv 2604.09752): during autoregressive decoding every
 * generated token fetches every weight of every linear layer from HBM, so decode is
 * bound by HBM bandwidth (Sec. 2.1; Sec. 3.1).  Each projection computes
 *
 *     y[m, n] = sum_k x[m, k] * W[n, k]                         (y = x W^T)
 *
 * for M = 1 token row (plain decoding) or M = 2..8 rows (prompt-lookup verification,
 * Sec. 4.2).  W8A16 storage-only quantization (Sec. 2.4; Sec. 6.2) stores W as int8
 * codes q with one bf16 scale s[n] per output channel:
 *
 *     y[m, n] = s[n] * sum_k x[m, k] * q[n, k]
 *
 * Types and layouts (all row-major, all device pointers unless stated):
 *   x  [M, K]  bf16 (IEEE bfloat16 bit patterns), row stride K elements
 *   W  [N, K]  bf16, or int8 codes in [-127, 127] (-128 is also computed exactly)
 *   s  [N]     bf16 scales (int8 weights only)
 *   y  [M, N]  fp32, row stride N elements; fp32 accumulation
 *
 * Conventions shared by every entry point:
 *   - Every call returns an aio_status; on failure aio_last_error() (thread-local)
 *     holds a one-line description.  Argument errors are detected on the host
 *     before anything is launched; no entry point traps on the device.
 *   - Ownership: the caller owns every buffer it passes (x, W, scales, y, packed
 *     weights).  The library owns only its handles, their small device workspaces
 *     and captured graphs, and frees them in the matching *_destroy call.
 *   - Asynchrony: run / pack / step calls enqueue work on the given stream (a
 *     cudaStream_t passed as void*, NULL = legacy default stream) and return without
 *     synchronising.  Buffers must stay valid until the stream has executed the work.
 *   - Devices: a handle or step belongs to the device that was current when it was
 *     created; using it while another device is current returns AIO_ERR_STATE.
 *   - Device-side waits are bounded.  A wait that expires sets an error word that
 *     aio_linear_check / aio_decode_step_check / aio_attention_check report as
 *     AIO_ERR_DEVICE_TIMEOUT, with the code in *device_error: 1 a bulk-copy wait expired,
 *     2 a wait for the previous projection expired, 3 a chained step's computed x did not fit
 *     the staging area (refused on the host; the device check is a second guard), 4 a chained
 *     step's attention found L_past + M outside [M, L_max].
 */
#ifndef AIO_H
#define AIO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AIO_ABI_VERSION 8

typedef enum {
    AIO_OK = 0,
    AIO_ERR_INVALID_ARG = 1,     /* bad size, null pointer, M out of range, shape mismatch */
    AIO_ERR_UNSUPPORTED = 2,     /* device is not sm_103 (the library is built for sm_103a only) */
    AIO_ERR_ALIGNMENT = 3,       /* a pointer is not aligned as documented */
    AIO_ERR_CUDA = 4,            /* a CUDA runtime call failed; see aio_last_error() */
    AIO_ERR_OOM = 5,             /* workspace allocation failed */
    AIO_ERR_STATE = 6,           /* wrong device current, or handle used after destroy */
    AIO_ERR_DEVICE_TIMEOUT = 7   /* a bounded device-side wait expired (reported by *_check) */
} aio_status;

typedef enum {
    AIO_W_BF16 = 0,              /* W is bf16 */
    AIO_W_INT8_PERCHANNEL = 1    /* W is int8 codes, one bf16 scale per output channel */
} aio_wtype;

/* aio_linear_create flags */
#define AIO_FLAG_ROWMAJOR   0x1u   /* aio_linear_run reads W as plain row-major [N, K] (no packing) */
#define AIO_FLAG_NO_PDL     0x2u   /* launch without programmatic dependent launch */
#define AIO_FLAG_STREAM_KERNEL 0x4u /* aio_linear_run always takes the stream kernel (never the small-projection launch) */
#define AIO_FLAG_TEST_STALL 0x100u /* TEST ONLY: the grid's last warp skips its first weight copy,
                                      so its bounded wait (20 ms) expires and the run reports
                                      AIO_ERR_DEVICE_TIMEOUT; outputs are then undefined */

/* aio_decode_step_create flags */
#define AIO_STEP_GRAPH      0x1u   /* capture the step's launches into one CUDA graph (one launch per step) */
#define AIO_STEP_PDL        0x2u   /* chain mode: programmatic dependent launch between projections */
#define AIO_STEP_PERSISTENT 0x4u   /* one cooperative launch streams every projection: each SM keeps a deep
                                      ring of weight tiles in flight across projection boundaries, and a
                                      bounded grid-wide counter orders projection i+1's x reads after
                                      projection i.  Needs one weight type for all projections.  Without
                                      this flag the step is a chain of one launch per projection. */

/* Packed weight layout written by aio_linear_pack (a permutation of W, no padding):
 * rows are grouped 16 at a time and each group is cut into tiles of 256 k-columns;
 * tile (g, kt) starts at element 16*g*K + rows_g*256*kt, rows_g = min(16, N - 16g), and holds
 * the block W[16g : 16g+rows_g, 256kt : 256kt+len], len = min(256, K - 256kt): row-major when
 * ragged (rows_g < 16 or len < 256), otherwise in the stream kernel's fragment order: lane
 * L = 4r + c reads 16-byte piece j at byte j*512 + 16L.  bf16: piece s holds, with
 * k0 = 32(s/2) + 8c + 4(s%2), the pairs W[r][k0..k0+1], W[r+8][k0..k0+1], W[r][k0+2..k0+3],
 * W[r+8][k0+2..k0+3].  int8: piece j = 4h + u holds the 8-code runs W[r+8h][32t + 8c : +8] for
 * t = 2u then 2u + 1, each 4-code word stored as codes (0, 2, 1, 3). */
#define AIO_ROWS_PER_GROUP 16
#define AIO_K_TILE 256

typedef struct aio_linear* aio_linear_t;
typedef struct aio_step* aio_step_t;

/* One projection of a decode step (all device pointers, see the layouts above). */
typedef struct {
    aio_linear_t h;       /* shape and weight type */
    const void* x;        /* [M, K] bf16 */
    const void* W;        /* packed weights (or row-major if h was created with AIO_FLAG_ROWMAJOR) */
    const void* scales;   /* [N] bf16 for int8 weights, NULL for bf16 */
    float* y;             /* [M, N] fp32 */
} aio_proj;

/*
 * How a projection of a chained decoder step obtains its x (aio_xprep.op).  The paper names its
 * models (Sec. 4.2) but prints no block structure; these are the steps of a pre-norm decoder block
 * between its projections.  The device computes x at the start of the projection, after every
 * projection before it in the step has completed, rounds it to bf16 (nearest even) and uses it;
 * it also writes it to the projection's x buffer.  All arithmetic is fp32.
 */
#define AIO_X_GIVEN   0   /* x is an input the caller fills (the plain decode step) */
#define AIO_X_RMSNORM 1   /* h = h_in + src (src may be NULL), x = h * gamma / sqrt(mean(h^2) + eps) */
#define AIO_X_SWIGLU  2   /* x[m, k] = silu(src[m, k]) * src[m, K + k], silu(t) = t / (1 + exp(-t)) */
#define AIO_X_SLICE   3   /* x[m, k] = src[m, src_off + k] (attention over one position: V of QKV) */
#define AIO_X_ATTENTION 4 /* x = bf16(attention of the M new tokens over the layer's KV cache), q, k, v
                             the column thirds of src (the QKV output), see aio_xprep.kv_cache */

typedef struct {
    int op;               /* AIO_X_* */
    const float* src;     /* fp32 [M, src_stride]: RMSNORM the residual to add ([M, K], stride K, or
                             NULL), SWIGLU the gate+up output (gate in [0, K), up in [K, 2K)), SLICE
                             the output the columns come from */
    int src_stride;       /* elements per token row of src (SWIGLU, SLICE) */
    int src_off;          /* SLICE: first column (multiple of 4) */
    const float* h_in;    /* RMSNORM: residual stream [M, K] fp32 */
    float* h_out;         /* RMSNORM: h_in + src is stored here (fp32 [M, K]) when non-NULL; it must
                             not be h_in, and no projection of the step may read it as h_in before
                             the next grid-wide step boundary after this projection */
    const void* gamma;    /* RMSNORM: norm weight [K] bf16 */
    float eps;            /* RMSNORM: >= 0 */
    /* ATTENTION (decode attention over a KV cache, the long-context path of Sec. 3.3 and Sec. 5.1):
     * src is the QKV output, fp32 [M, src_stride >= 3K]; q, k and v of token m are its columns
     * [0, K), [K, 2K) and [2K, 3K), head h at columns [128 h, 128 h + 128) of each (K = 128 n_heads).
     * The device reads *L_past (set before the step; not changed by it), writes the new tokens' k
     * and v, rounded to bf16, at positions L_past .. L_past + M - 1 of the cache, and computes
     *   out[m, h] = sum_j softmax_j(q[m, h] . k[h, j] / sqrt(128)) v[h, j]  over j <= L_past + m,
     * in fp32 with an online softmax and a fixed merge order; x = bf16(out) (nearest even).  It
     * runs as two phases of the step before this projection, so the step grows by two grid-wide
     * steps (two kernels in chain mode).  L_past + M > L_max is reported as device error 4 and
     * leaves x undefined. */
    void* kv_cache;       /* ATTENTION: the layer's cache, bf16 [2][n_heads][L_max][128] (K, then V), device,
                             16-byte aligned; updated in place */
    const int* L_past;    /* ATTENTION: device int, positions already in the cache, 4-byte aligned */
    int n_heads;          /* ATTENTION: K / 128, at most the warps of the grid */
    int L_max;            /* ATTENTION: positions the cache holds */
} aio_xprep;

/* ABI version of the loaded library (AIO_ABI_VERSION at build time). */
int aio_abi_version(void);

/* Static description of an error code; never NULL. */
const char* aio_status_string(aio_status s);

/* Detail of the last failure on the calling thread ("" if none). */
const char* aio_last_error(void);

/*
 * Create a handle for one linear layer y = x W^T with W [N, K] (Sec. 2.1; Sec. 2.4 for int8).
 *   out    receives the handle (set to NULL on failure)
 *   K      16 <= K <= 1048576 and K % 16 == 0
 *   N      1 <= N <= 16777216
 *   wt     AIO_W_BF16 or AIO_W_INT8_PERCHANNEL
 *   max_M  1..8: the largest number of token rows later passed to aio_linear_run
 *   flags  AIO_FLAG_* bits
 * Allocates a small device workspace (cross-warp partial sums and an error word, set up here)
 * on the current device; synchronises that device.  Errors: INVALID_ARG, UNSUPPORTED,
 * OOM, CUDA.
 */
aio_status aio_linear_create(aio_linear_t* out, int K, int N, aio_wtype wt, int max_M, unsigned flags);

/* Bytes of the packed weight buffer (N*K*elem_size) and of the scale buffer (2*N for int8, else 0):
 * the bytes every decode step streams for this layer (Sec. 3.1), half of them for the int8 codes
 * of storage-only quantization (Sec. 2.4) plus their per-channel scales. */
aio_status aio_linear_packed_bytes(aio_linear_t h, size_t* w_bytes, size_t* scale_bytes);

/* Launch geometry of aio_linear_run: CTAs, threads per CTA, dynamic shared memory bytes,
 * and the number of weight tiles the grid streams.  Any pointer may be NULL. */
aio_status aio_linear_launch_info(aio_linear_t h, int* grid, int* block, size_t* smem_bytes, long long* tiles);

/*
 * Store a layer's weights for streaming (Sec. 2.1: every decode step reads them all from HBM; Sec.
 * 2.4: int8 weights are stored as codes plus scales and dequantized only inside the kernel).
 * Pack row-major W [N, K] (bf16 or int8, device) into the tiled layout above (device,
 * aio_linear_packed_bytes bytes, must not overlap W).  For int8, scales [N] bf16 are copied
 * to scales_packed (both device, or both NULL for bf16).  All pointers 16-byte aligned.
 * Asynchronous on stream.  Errors: INVALID_ARG, ALIGNMENT, STATE, CUDA.
 */
aio_status aio_linear_pack(aio_linear_t h, const void* W_rowmajor, const void* scales,
                           void* W_packed, void* scales_packed, void* stream);

/* Inverse of aio_linear_pack for the weights (used by tests): packed -> row-major [N, K]. */
aio_status aio_linear_unpack(aio_linear_t h, const void* W_packed, void* W_rowmajor, void* stream);

/*
 * y = x W^T for M token rows (Sec. 2.1; int8 with per-channel scales, Sec. 2.4).
 *   x       [M, K] bf16, 16-byte aligned
 *   M       1 <= M <= max_M of the handle
 *   K, N    must equal the handle's
 *   W       packed weights (row-major if the handle has AIO_FLAG_ROWMAJOR), 16-byte aligned
 *   scales  [N] bf16, 2-byte aligned, non-NULL exactly when the handle is int8
 *   y       [M, N] fp32, 16-byte aligned; fully overwritten
 * Uses the handle's workspace: runs of one handle must not overlap in time (issue them on
 * one stream, or order the streams).  With PDL (default) the kernel may start streaming W
 * while the previous kernel on the stream is still running; it reads x and writes y only
 * after that kernel has completed.
 * Two launches (Sec. 3.1: a projection launched on its own is bound by latency once its weights
 * are a few MB).  A small packed projection -- at most 2 x (SM count) row groups of 16 rows, and
 * K <= 2048 (bf16) or K <= 6144 (int8) -- runs as one CTA of 8 warps per row group: the warps split
 * the group's tiles, their partial sums meet in shared memory and are added in warp order, and two
 * such CTAs fit an SM, so a PDL launch loads its weights beside the previous one.  Every other
 * projection, and every handle created with AIO_FLAG_STREAM_KERNEL, takes the stream kernel (all
 * SMs, equal bytes per warp).  A decode step's per-projection launches (without
 * AIO_STEP_PERSISTENT, and without computed x) make the same choice.
 * Errors: INVALID_ARG, ALIGNMENT, STATE, CUDA.
 */
aio_status aio_linear_run(aio_linear_t h, const void* x, int M, int K, int N, const void* W,
                          const void* scales, float* y, void* stream);

/*
 * y = x W^T as the stream kernel computes it (aio_linear_run with AIO_FLAG_STREAM_KERNEL), without
 * a handle and without allocating anything.
 * The paper has no counterpart: this is a library entry for callers that cannot allocate device
 * memory where they call -- a serving engine that has handed nearly all of HBM to its own pools
 * (weights, KV cache), so that a cudaMalloc there fails, or a hot loop in which cudaMalloc /
 * cudaFree would synchronise the device.
 *   x, M, W, scales, y   as for aio_linear_run, with 1 <= M <= 8
 *   K, N          as for aio_linear_create
 *   wt            AIO_W_BF16 or AIO_W_INT8_PERCHANNEL
 *   flags         AIO_FLAG_ROWMAJOR and / or AIO_FLAG_NO_PDL
 *   device_error  device int, 4-byte aligned, owned by the caller.  It must hold 0 when the call
 *                 runs on the stream.  The kernel sets it non-zero if a bounded device-side wait
 *                 expired (y is then incomplete).  The library never clears it, so an error stays
 *                 visible to the caller across later calls; but while it is non-zero, later calls
 *                 that share the word give up at their first wait for another warp's partial sums
 *                 and leave y incomplete.  Clear it (e.g. cudaMemsetAsync) before reusing it.
 * Scratch: the cross-warp partial sums live in one static device array of
 * AIO_NOALLOC_SCRATCH_BYTES per device, part of the loaded library image.  A call needs
 * 16 * 4 * M * Z bytes of it, rounded up to 256, where Z = the device's SM count times the warps per
 * CTA (8 in the default build): on a 152-SM GB300 every M <= 8 fits (622592 bytes at M = 8).  A call
 * that needs more returns AIO_ERR_INVALID_ARG and launches nothing.
 * Each call enqueues a cudaMemsetAsync that empties the partial-sum slots it uses (all bytes 0xFF),
 * then the kernel.
 * Every call on a device shares that scratch: calls that overlap in time race and give wrong
 * results, so issue them on one stream or order their streams.
 * The first call on each device looks up the scratch address (cudaGetSymbolAddress) and sets the
 * kernels' attributes; make that first call before any stream capture begins.
 * Errors: INVALID_ARG, ALIGNMENT, UNSUPPORTED, CUDA.
 */
#define AIO_NOALLOC_SCRATCH_BYTES 1048576
aio_status aio_linear_run_noalloc(const void* x, int M, int K, int N, aio_wtype wt, unsigned flags,
                                  const void* W, const void* scales, float* y, int* device_error,
                                  void* stream);

/* Synchronise the device, then report the handle's device error word:
 * AIO_OK, or AIO_ERR_DEVICE_TIMEOUT (code also stored in *device_error if non-NULL). */
aio_status aio_linear_check(aio_linear_t h, int* device_error);

/* Empty the handle's partial-sum slots and clear its error word (needed only after a device error). */
aio_status aio_linear_reset(aio_linear_t h);

/* Free the handle of one linear layer (Sec. 2.1) and its workspace (synchronises the device).
 * NULL is accepted. */
aio_status aio_linear_destroy(aio_linear_t h);

/*
 * Build one decode step: the projections run in array order on one stream, projection i+1
 * reading its x only after projection i has completed (Sec. 3.1: every weight of every layer is
 * streamed once per token).  Pointer values are captured at creation: later calls rewrite the
 * buffers' contents, never their addresses.  1 <= M <= every handle's max_M.  The step owns a
 * private workspace per projection (so consecutive projections may overlap), a device copy of
 * the projection list, and per-projection completion counters; runs of one step must not overlap
 * in time.  flags: AIO_STEP_* bits.  Errors: INVALID_ARG, ALIGNMENT, STATE, UNSUPPORTED, OOM, CUDA.
 */
aio_status aio_decode_step_create(aio_step_t* out, const aio_proj* projs, int n_projs, int M, unsigned flags);

/*
 * The same, for a chained decoder step: projection i obtains its x as preps[i] says (AIO_X_*),
 * from buffers the caller filled or earlier projections of the step wrote; preps may be NULL (all
 * AIO_X_GIVEN).  projs[i].x receives the computed x.  A chained step takes M <= 4.  Every CTA computes
 * an RMSNORM or SLICE x itself into shared memory, so M * (K + 32) * 2 must not exceed the staging
 * area (35,360 bytes in the default build: M <= 4 for K = 4096): UNSUPPORTED otherwise.  A SWIGLU x
 * that does not fit (M >= 2 at K = 5632 or 11008) is computed by a grid-wide phase of its own into
 * projs[i].x instead (one more grid-wide step).  src, h_in, h_out and gamma must be 16-byte aligned,
 * src_stride and src_off multiples of 4: ALIGNMENT otherwise.  A missing pointer, a column range
 * outside src_stride, h_out == h_in or a negative eps: INVALID_ARG.  ATTENTION preparations: see
 * aio_xprep.  Device errors are reported as for aio_decode_step_create.
 */
aio_status aio_decode_step_create_chained(aio_step_t* out, const aio_proj* projs, const aio_xprep* preps,
                                          int n_projs, int M, unsigned flags);

/* Enqueue one decode step on stream (one graph launch with AIO_STEP_GRAPH). */
aio_status aio_decode_step(aio_step_t step, void* stream);

/*
 * One decode step from host memory (Sec. 3.1: one generated token): copy x_bytes from x_host to
 * x_dev, run the step, copy y_bytes from y_dev to y_host, all in order on stream.  x_dev and y_dev
 * are device buffers the step reads and writes (e.g. one arena holding every projection's x, and
 * one holding every y); x_host and y_host are host buffers, page-locked for the copies to be
 * asynchronous.  A size of 0 skips that copy.  Returns without synchronising: y_host is valid once
 * the stream has executed the work.  Errors: INVALID_ARG (a copy of non-zero size with a NULL
 * pointer), STATE, CUDA.
 */
aio_status aio_decode_step_host(aio_step_t step, const void* x_host, void* x_dev, size_t x_bytes, const void* y_dev,
                                void* y_host, size_t y_bytes, void* stream);

/* Number of kernels one aio_decode_step launches (1 in persistent mode, else one per projection). */
aio_status aio_decode_step_kernels(aio_step_t step, int* n_kernels);

/* Empty the step's partial-sum slots, clear its counters and error words (needed only after a device error). */
aio_status aio_decode_step_reset(aio_step_t step);

/* Synchronise the device, then report the step's device error word (see aio_linear_check). */
aio_status aio_decode_step_check(aio_step_t step, int* device_error);

/* Free a decode step (Sec. 3.1), its graph and its workspace (synchronises the device). NULL is
 * accepted. */
aio_status aio_decode_step_destroy(aio_step_t step);

/*
 * Decode attention over a KV cache (the long-context path the paper routes on: standard contexts
 * up to 2K tokens, long ones up to 32K, Sec. 3.3 and Sec. 5.1).  M new tokens sit at positions
 * L - M .. L - 1 of a cache holding L positions; token m attends to positions j <= L - M + m:
 *   out[m, h*128 + e] = sum_j softmax_j(q[m, h] . k[h, j] / sqrt(128)) v[h, j, e].
 * q:        fp32 [M, q_stride] (head h at columns [128 h, 128 h + 128)), device.
 * k_cache,
 * v_cache:  bf16 [n_heads][L_max][128], device (a run of positions of one head is contiguous).
 * out:      fp32 [M, n_heads * 128], device.
 * workspace: device scratch of aio_attention_workspace_bytes(M) bytes; its first 4 bytes are the
 *           device error word and must be zero before the first call (aio_attention_check
 *           clears it after reporting an error).  Calls sharing a workspace must not overlap.
 * Arithmetic is fp32 with an online softmax; the per-warp partial results are merged in a fixed
 * order, so results are reproducible.  Asynchronous on stream, allocates nothing.  The two kernels
 * launch with programmatic dependent launch: K and V start streaming before earlier work on the
 * stream has completed, while q is read and out, the workspace and the error word are written only
 * after it has.  Errors:
 * INVALID_ARG (NULL pointer, M outside [1, 8], L outside [M, L_max], q_stride < 128 n_heads,
 * workspace too small), UNSUPPORTED (head_dim != 128, n_heads above the grid's warp count),
 * ALIGNMENT (a pointer not 16-byte aligned, q_stride not a multiple of 4), CUDA.
 */
aio_status aio_attention_workspace_bytes(int M, size_t* bytes);
aio_status aio_attention_decode(const float* q, int q_stride, const void* k_cache, const void* v_cache, int n_heads,
                                int head_dim, int L_max, int L, int M, float* out, void* workspace,
                                size_t workspace_bytes, void* stream);

/* Synchronise the device, then report (and clear) the attention workspace's device error word. */
aio_status aio_attention_check(void* workspace, int* device_error);

/*
 * Prompt-lookup decoding around the verification pass (Sec. 4.2: n-gram window N = 6, look-ahead
 * L = 2).  All device pointers, asynchronous on stream, no allocation; the paper prints no
 * algorithm, so these state the reading.
 *
 * aio_pld_draft: tokens [T] int32.  Among positions i < T - 1, the one whose preceding tokens
 * share the longest suffix (n <= N tokens) with the whole sequence, the most recent among equals;
 * the draft is the up to L tokens after it (fewer at the end of the sequence, none without a
 * match).  out [3 + L] int32: draft length d, matched n, position i (-1 without a match), then the
 * d drafted tokens (-1 after them).  1 <= N <= 32, 1 <= L <= 7.
 *
 * aio_argmax_rows: out[m] = argmax over v < V of logits[m * stride + v] (fp32), the lowest index
 * among equal maxima; a NaN counts as the maximum (the first NaN wins).  1 <= M <= 65535.
 *
 * aio_pld_accept: greedy acceptance.  argmax [d + 1] holds the verification pass's argmax for the
 * last committed token followed by the d drafted tokens; draft is aio_pld_draft's out.  result [2]
 * int32: the number a of drafted tokens accepted (the longest agreeing prefix), then the model's
 * next token argmax[a]: a + 1 tokens commit.
 *
 * Errors: INVALID_ARG (NULL pointer, a size outside its range), ALIGNMENT (a pointer not 4-byte
 * aligned), UNSUPPORTED (not a GB300), CUDA.
 */
aio_status aio_pld_draft(const int* tokens, int T, int N, int L, int* out, void* stream);
aio_status aio_argmax_rows(const float* logits, int M, int V, int stride, int* out, void* stream);
aio_status aio_pld_accept(const int* argmax, const int* draft, int* result, void* stream);

/*
 * The request-level routing decision (Sec. 3.2, Sec. 3.3) from the probe's single-token output.
 * logits: the probe's fp32 logits over its vocabulary (device); category_tokens [n_categories]
 * int32 (device): the token id of each category in the classification template; code_index: the
 * category that is Code Generation.  On the device: the category is the argmax over the category
 * logits (lowest index among ties); H is the softmax entropy over them in nats (the paper gives no
 * base); the 1B model serves the request if it is Code Generation, L_ctx <= 2048 and H <= tau,
 * the 7B model otherwise; PLD is on for every category but Code Generation.  decision [4] int32:
 * category, model (1 or 7), PLD (1 on, 0 off), H as the bits of a float.  The paper's tau is 0.45.
 * Errors: INVALID_ARG (NULL pointer, n_categories outside [1, 32], code_index outside them,
 * negative L_ctx, tau negative or not finite), ALIGNMENT (a pointer not 4-byte aligned), CUDA.
 */
aio_status aio_route(const float* logits, const int* category_tokens, int n_categories, int code_index, int L_ctx,
                     float tau, int* decision, void* stream);

/*
 * Read-bandwidth probe: streams `bytes` from buf (device, 16-byte aligned, bytes a multiple of
 * 4096) through the same per-warp bulk-copy ring the linear kernels use, touching every chunk,
 * and XORs one word per chunk into *out (device uint32).  Measures the practical HBM read
 * ceiling for the roofline.  Asynchronous on stream.
 */
aio_status aio_probe_read(const void* buf, size_t bytes, unsigned* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AIO_H */
