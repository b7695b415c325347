// aio_stream.cuh -- the decode-step stream kernel: y = x W^T for M = 1..8 token rows, bf16 weights or
// int8 codes with per-output-channel bf16 scales (Sec. 2.1, Sec. 2.4), for one projection or for
// every projection of a decode step in one persistent launch (Sec. 3.1).
//
// The work is a stream of weight bytes from HBM with 1 (bf16) or 2 (int8) multiply-adds per byte per
// token row.  Design:
//
//   * Tiles.  W is cut into tiles of 16 rows x 256 k (8 KB bf16, 4 KB int8); consecutive tiles are
//     contiguous in the packed layout, so any run of them is one bulk copy.  The T tiles of a matrix
//     are split evenly over the Z warps of the grid: warp z streams tiles [z*T/Z, (z+1)*T/Z), so
//     every warp moves the same bytes to within one tile whatever N and K are.
//   * Rings.  One CTA per SM; each warp owns a shared-memory ring of slots.  Lane 0 issues one
//     cp.async.bulk per slot (global -> shared, L2 evict-first) completing on the slot's mbarrier;
//     the warp waits (bounded by %globaltimer), computes, and refills the slot.  The issue cursor
//     runs ahead across projection boundaries: weights never depend on x.  The wide launches (two
//     slots per warp: bf16 M >= 5, int8 M >= 2) read a slot into registers and refill it before
//     computing.
//   * x.  Once per CTA and projection, warp 0 stages x into shared memory (one bulk copy per token
//     row, rows padded by 64 B) when it fits; otherwise the lanes read x from global memory.
//   * Arithmetic on the tensor cores: mma.sync.m16n8k16, bf16 in, fp32 accumulate, with A = W
//     (the tile's 16 rows) and B = x (up to 8 tokens), so one MMA reduces 256 weights for every
//     token and the work per byte does not grow with M.  A k-permutation shared by A and B (see
//     tile_mma_frag) gives each lane runs of 8 consecutive k; full tiles are stored in fragment
//     order ([j][lane][16 B]), so W comes in with conflict-free 128-bit shared loads.  Four
//     accumulator chains keep MMAs in flight.  int8 codes become bf16 exactly (|q| <= 128 fits
//     bf16's 8 significant bits) with two bit operations and one bf16x2 subtraction per pair; the
//     per-channel scale multiplies the finished fp32 sum.
//   * Split row groups.  A row group whose tiles all lie in one warp's segment is written directly.
//     A group split between warps is owned by its first contributor, for which it is the last group
//     of its segment, so the owner reaches it at the end of the phase; the other contributors reach
//     it earlier, at the start of their segments.  They store their partial sums with relaxed
//     stores into slots that read 0xFFFFFFFF (a bit pattern no computed float takes) while empty,
//     and move on: no fence and no atomic on their path.  The owner polls the slots (bounded),
//     sums them in warp order (deterministic), writes y and empties the slots again.
//   * Projection order.  In a persistent step, projection p+1 reads x only after every CTA has
//     finished projection p: warps count in shared memory, the last warp of a CTA makes one global
//     increment, warp 0 of each CTA polls the global counter (bounded) and publishes it to its CTA.
//   * Programmatic dependent launch: the kernel signals dependents at entry and issues its first
//     weight copies before griddepcontrol.wait; x, y and the workspace are touched after it.
// Included by aio_gemv.cu (the plain step: x is an input) and aio_chain.cu (the chained step:
// x computed on the device); each instantiates its own kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <type_traits>

#include "aio_internal.h"

namespace aio {
namespace {

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on a phase of an mbarrier; false if limit_ns elapsed first.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned long long limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t start = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (globaltimer_ns() - start > limit_ns) return false;
    }
}

__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
        ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
        : "memory");
}

// The same without an L2 cache hint (activations: read by every CTA, keep the default policy).
__device__ __forceinline__ void bulk_g2s_plain(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ void st_relaxed_u32(void* p, uint32_t v) {
    asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t ld_relaxed_u32(const void* p) {
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Orders this thread's earlier generic-proxy accesses (and those it has observed) before its later
// async-proxy accesses, in every state space.
__device__ __forceinline__ void fence_proxy_async_all() { asm volatile("fence.proxy.async;" ::: "memory"); }

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ unsigned ld_acquire_cta_shared(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.cta.shared::cta.u32 %0, [%1];" : "=r"(v) : "r"(smem_addr(p)) : "memory");
    return v;
}

__device__ __forceinline__ void st_release_cta_shared(unsigned* p, unsigned v) {
    asm volatile("st.release.cta.shared::cta.u32 [%0], %1;" ::"r"(smem_addr(p)), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned atom_add_acq_rel_cta_shared(unsigned* p, unsigned v) {
    unsigned old;
    asm volatile("atom.acq_rel.cta.shared::cta.add.u32 %0, [%1], %2;" : "=r"(old) : "r"(smem_addr(p)), "r"(v) : "memory");
    return old;
}

// D (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
[[maybe_unused]] __device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The constants of the int8 -> bf16 conversion, held in registers: a hardware LOP3 takes at most
// one immediate, so (t & mask) | magic with both as immediates would cost two instructions.  The
// moves are volatile so the compiler keeps the values in registers.
struct I8Consts {
    uint32_t m7, m8, magic;   // 0x007F007F, 0x00800080, 0x43004300
};

__device__ __forceinline__ I8Consts i8_consts() {
    I8Consts k;
    asm volatile("mov.u32 %0, 0x007F007F;" : "=r"(k.m7));
    asm volatile("mov.u32 %0, 0x00800080;" : "=r"(k.m8));
    asm volatile("mov.u32 %0, 0x43004300;" : "=r"(k.magic));
    return k;
}

__device__ __forceinline__ uint32_t lop3_and_or(uint32_t t, uint32_t m, uint32_t c) {   // (t & m) | c
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(t), "r"(m), "r"(c));
    return r;
}

// Two int8 codes -> bf16x2, exactly.  t holds the codes in the low bytes of its 16-bit halves (the
// high bytes are ignored): 0x4300 | (q & 0x7F) is bf16 128 + (q & 0x7F), and 0x4300 | (q & 0x80)
// is bf16 128 or 256; their difference is q (an integer in [-128, 127], so the subtraction is exact).
[[maybe_unused]] __device__ __forceinline__ uint32_t i8x2_to_bf16x2(uint32_t t, const I8Consts& k) {
    const uint32_t a = lop3_and_or(t, k.m7, k.magic);
    const uint32_t b = lop3_and_or(t, k.m8, k.magic);
    uint32_t r;
    asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }

template <bool I8>
struct TileT {
    static constexpr int kEsize = I8 ? 1 : 2;
    static constexpr int kBytes = kRows * kKT * kEsize;    // 4096 (int8) or 8192 (bf16)
    static constexpr int kSlot = I8 ? kSlotBytesI8 : kSlotBytes;
    static constexpr int kChunk = kSlot / kBytes;          // tiles per ring slot
    static constexpr int kAhead = I8 ? AIO_AHEAD_I8 : AIO_AHEAD;
    static constexpr int kAheadLive = I8 ? AIO_AHEAD_LIVE_I8 : AIO_AHEAD_LIVE;
    static constexpr int kPieces = kBytes / 512;           // 16-byte pieces per lane per tile (8 or 16)
};

__device__ __forceinline__ const ProjDesc* proj_desc(const StreamArgs& s, int p) {
    return s.projs ? s.projs + p : &s.one;
}

// Byte offset of tile (g, kt) in the packed layout.
template <int E>
__device__ __forceinline__ size_t tile_offset(int K, int N, int g, int kt) {
    const int rows = min(kRows, N - g * kRows);
    return (static_cast<size_t>(g) * kRows * K + static_cast<size_t>(kt) * rows * kKT) * E;
}

// What the issuing lane needs of one phase, held in registers.  A projection: its packed weights,
// shape and tile grid.  An attention phase of a chained step streams units of 16 positions of one
// head instead (T = n_heads * nch units, unit u = head u / nch, positions 16 (u % nch) ...): w is
// the layer's KV cache, K = L_max, N = L (the cached positions including the new tokens), NKT = nch,
// uniform = n_heads, rowmajor = kIssueAttn.  Merge and SwiGLU phases stream nothing (T = 0).
struct IssueProj {
    const uint8_t* w;
    int Tq, Tr;           // T = Tq * Z + Tr
    int K, N, NKT;
    int uniform, rowmajor;
};
constexpr int kIssueAttn = 2;   // IssueProj::rowmajor of an attention phase

// Positions an attention phase covers, L = L_past + M, read from the device int the caller set
// before the launch; 0 when the cache cannot hold them (the phase then streams and computes nothing
// and reports kDevErrAttn).
__device__ __forceinline__ int attn_len(const ProjDesc* d, int M) {
    const int lp = __ldg(d->Lpast);
    return (lp >= 0 && lp <= d->L_max - M) ? lp + M : 0;
}

// Units and segment bounds of an attention (or merge) phase over Z warps.
__device__ __forceinline__ void attn_geom(const ProjDesc* d, int M, int Z, int& L, int& nch, int& Tq, int& Tr) {
    L = attn_len(d, M);
    nch = (L + kAttnPos - 1) / kAttnPos;
    const int U = d->kind == kPhaseAttn ? d->n_heads * nch : 0;
    Tq = U / Z;
    Tr = U - Tq * Z;
}

// The issue fields of a chained step's non-projection phase (out of line: it runs once per phase).
__device__ __noinline__ IssueProj load_issue_phase(const ProjDesc* d, int M, int Z) {
    IssueProj q;
    int L = 0, nch = 0;
    q.Tq = q.Tr = 0;   // merge and SwiGLU phases stream nothing
    if (d->kind == kPhaseAttn) attn_geom(d, M, Z, L, nch, q.Tq, q.Tr);
    q.w = reinterpret_cast<const uint8_t*>(d->kv);
    q.K = d->L_max;
    q.N = L;
    q.NKT = nch;
    q.uniform = d->n_heads;
    q.rowmajor = kIssueAttn;
    return q;
}

template <bool PH>
__device__ __forceinline__ IssueProj load_issue(const ProjDesc* d, int M, int Z) {
    if (PH && d->kind != kPhaseProj) return load_issue_phase(d, M, Z);
    IssueProj q;
    q.w = d->w;
    q.Tq = d->Tq;
    q.Tr = d->Tr;
    q.K = d->K;
    q.N = d->N;
    q.NKT = d->NKT;
    q.uniform = d->uniform;
    q.rowmajor = d->rowmajor;
    return q;
}

// Lane 0: the K rows then the V rows of attention unit u into one slot (K at dst, V at dst +
// kAttnUnitBytes), both 256 B per position, completing on the slot's barrier.
__device__ __noinline__ void issue_attn_unit(IssueProj d, int u, uint8_t* dst, uint64_t* bar, uint64_t pol) {
    const int h = u / d.NKT, c = u - h * d.NKT;
    const int p0 = c * kAttnPos, np = min(kAttnPos, d.N - p0);
    const uint32_t bytes = static_cast<uint32_t>(np * kHeadDim * 2);
    const size_t off = (static_cast<size_t>(h) * d.K + p0) * (kHeadDim * 2);
    const size_t voff = static_cast<size_t>(d.uniform) * d.K * (kHeadDim * 2);
    mbar_expect_tx(bar, 2 * bytes);
    bulk_g2s(dst, d.w + off, bytes, bar, pol);
    bulk_g2s(dst + kAttnUnitBytes, d.w + voff + off, bytes, bar, pol);
}

// First tile of warp z's segment (z = Z gives T): floor(z T / Z) = z Tq + floor(z Tr / Z), exact in
// 32-bit arithmetic (z Tq <= T < 2^31 and z Tr < Z^2).
__device__ __forceinline__ int seg(int z, int Z, int Tq, int Tr) { return z * Tq + (z * Tr) / Z; }

// Lane 0: arm the slot's barrier with the chunk's byte count and issue the copies of tiles
// [t, t + nt) of projection d.  Packed weights: one bulk copy.  Row-major weights: one copy per
// tile row, landing in the row-major form of that tile.
template <bool I8>
__device__ __noinline__ void issue_chunk_general(IssueProj d, int t, int nt, uint8_t* dst, uint64_t* bar,
                                                 uint64_t pol) {
    constexpr int E = TileT<I8>::kEsize;
    const int K = d.K, N = d.N, NKT = d.NKT;
    int g = t / NKT, kt = t - g * NKT;
    if (!d.rowmajor) {
        const int tl = t + nt - 1;
        const int gl = tl / NKT, ktl = tl - gl * NKT;
        const int rows_l = min(kRows, N - gl * kRows), klen_l = min(kKT, K - ktl * kKT);
        const size_t off = tile_offset<E>(K, N, g, kt);
        const size_t end = tile_offset<E>(K, N, gl, ktl) + static_cast<size_t>(rows_l) * klen_l * E;
        const uint32_t bytes = static_cast<uint32_t>(end - off);
        mbar_expect_tx(bar, bytes);
        bulk_g2s(dst, d.w + off, bytes, bar, pol);
        return;
    }
    uint32_t total = 0;
    {
        int gg = g, kk = kt;
        for (int j = 0; j < nt; ++j) {
            total += static_cast<uint32_t>(min(kRows, N - gg * kRows) * min(kKT, K - kk * kKT) * E);
            if (++kk == NKT) { kk = 0; ++gg; }
        }
    }
    mbar_expect_tx(bar, total);
    for (int j = 0; j < nt; ++j) {
        const int rows = min(kRows, N - g * kRows), klen = min(kKT, K - kt * kKT);
        for (int r = 0; r < rows; ++r) {
            const size_t off = (static_cast<size_t>(g * kRows + r) * K + static_cast<size_t>(kt) * kKT) * E;
            bulk_g2s(dst + r * klen * E, d.w + off, static_cast<uint32_t>(klen * E), bar, pol);
        }
        dst += rows * klen * E;
        if (++kt == NKT) { kt = 0; ++g; }
    }
}

template <bool I8>
__device__ __forceinline__ void issue_chunk(const IssueProj& d, int t, int nt, uint8_t* dst, uint64_t* bar,
                                            uint64_t pol) {
    constexpr int B = TileT<I8>::kBytes;
    if (d.uniform) {   // every tile full: tile t is bytes [t * B, (t + 1) * B)
        const uint32_t bytes = static_cast<uint32_t>(nt * B);
        mbar_expect_tx(bar, bytes);
        bulk_g2s(dst, d.w + static_cast<size_t>(t) * B, bytes, bar, pol);
        return;
    }
    issue_chunk_general<I8>(d, t, nt, dst, bar, pol);
}

// First page of a probe warp's range (64-bit: any buffer size).
__device__ __forceinline__ long long seg_start(long long z, int Z, long long T) { return z * T / Z; }

// A warp's walk over its tiles of every projection, one chunk (<= C consecutive tiles) at a time.
// It holds the issue fields of the current projection and, loaded one projection ahead, of the
// next, so crossing a projection boundary never waits on a descriptor load.
struct ChunkCursor {
    int p, t, te;
    IssueProj cur, nxt;
};

// Kernels with attention, merge or SwiGLU phases (PH) keep no copy of the next phase's fields:
// they load them at the boundary instead, which frees the registers their phase code needs.
template <bool PH>
__device__ __forceinline__ void cursor_init(ChunkCursor& c, const StreamArgs& s, int z, int Z) {
    c.cur = load_issue<PH>(proj_desc(s, 0), s.M, Z);
    if constexpr (!PH) c.nxt = s.nproj > 1 ? load_issue<PH>(proj_desc(s, 1), s.M, Z) : c.cur;
    c.p = 0;
    c.t = seg(z, Z, c.cur.Tq, c.cur.Tr);
    c.te = seg(z + 1, Z, c.cur.Tq, c.cur.Tr);
}

// Next chunk of the walk: its phase, first tile (or unit) and count; false at the end.  An
// attention unit fills a slot on its own.
template <bool PH>
__device__ __forceinline__ bool cursor_next(ChunkCursor& c, const StreamArgs& s, int z, int Z, int C, int& p,
                                            int& t, int& nt) {
    while (c.t >= c.te) {
        if (c.p + 1 >= s.nproj) return false;
        ++c.p;
        if constexpr (PH) {
            c.cur = load_issue<PH>(proj_desc(s, c.p), s.M, Z);
        } else {
            c.cur = c.nxt;
            if (c.p + 1 < s.nproj) c.nxt = load_issue<PH>(proj_desc(s, c.p + 1), s.M, Z);
        }
        c.t = seg(z, Z, c.cur.Tq, c.cur.Tr);
        c.te = seg(z + 1, Z, c.cur.Tq, c.cur.Tr);
    }
    p = c.p;
    t = c.t;
    nt = (PH && c.cur.rowmajor == kIssueAttn) ? 1 : min(C, c.te - c.t);
    c.t += nt;
    return true;
}

// The fields of one projection the consuming warp needs, held in registers.
struct Proj {
    const uint16_t* x;
    const uint16_t* scales;
    float* y;
    float* partial;
    long long T;
    int Tq, Tr;
    int M, K, N, NKT;
    int rowmajor, uniform;
    int xop;
    int xfence;   // plain kernels: fence before staging x (chained kernels always fence)
};

template <bool CH>
__device__ __forceinline__ Proj load_proj(const ProjDesc* d, int M) {
    Proj p;
    p.x = d->x;
    p.scales = d->scales;
    p.y = d->y;
    p.partial = d->partial;
    p.Tq = d->Tq;
    p.Tr = d->Tr;
    p.T = d->T;
    p.M = M;
    p.K = d->K;
    p.N = d->N;
    p.NKT = d->NKT;
    p.rowmajor = d->rowmajor;
    p.uniform = d->uniform;
    p.xop = d->xop;
    p.xfence = CH ? 1 : d->xfence;
    return p;
}

// ------------------------------------------------------------------ one tile on the tensor cores
// A tile is 16 rows x 256 k of W.  It takes 16 k-steps of mma.m16n8k16 with A = W (lane (g, c)
// supplies rows g and g + 8 of the tile) and B = x (lane (g, c) supplies token g), so one MMA
// reduces 256 weights for all M <= 8 tokens at once; D[row][token] accumulates in fp32.
// k-permutation: in k-step s, lane (g, c) holds the logical k pairs (2c, 2c+1) and (2c+8, 2c+9)
// of both operands, which are the physical k = 32(s/2) + 8c + 4(s%2) + {0, 1} and + {2, 3}.
// The map is a bijection onto the tile's 256 k and A and B share it, so the sum is unchanged.
// Per pair of k-steps t = s/2 a lane therefore reads 8 consecutive k at 32t + 8c of W rows g and
// g + 8 and of x token g; the four lanes of a token read 64 consecutive bytes of x (no shared-
// memory bank conflict).  k-step s accumulates into d[s % 4]: four MMA chains in flight.
constexpr int kRuns = kKT / 32;   // runs of 8 k per lane and row: x pieces per tile, bf16 pieces per row half

template <bool I8>
__device__ __forceinline__ void tile_mma_frag(float (&d)[4][4], const uint4 (&w)[TileT<I8>::kPieces],
                                              const uint4 (&xv)[kRuns], const I8Consts& kc) {
#pragma unroll
    for (int s = 0; s < kKT / 16; ++s) {
        const int t = s >> 1, q = s & 1;
        const uint4& xq = xv[t];
        const uint32_t b0 = q ? xq.z : xq.x;
        const uint32_t b1 = q ? xq.w : xq.y;
        uint32_t a0, a1, a2, a3;
        if constexpr (I8) {
            // piece t/2 of row g (kRuns/2 + t/2 of row g + 8); word 2(t%2) + q holds the step's 4 codes,
            // stored (0, 2, 1, 3): k pair (0, 1) in the low bytes of its halves, (2, 3) in the high
            const uint4& lo = w[t >> 1];
            const uint4& hi = w[kRuns / 2 + (t >> 1)];
            const int wi = (t & 1) * 2 + q;
            const uint32_t wl = wi == 0 ? lo.x : wi == 1 ? lo.y : wi == 2 ? lo.z : lo.w;
            const uint32_t wh = wi == 0 ? hi.x : wi == 1 ? hi.y : wi == 2 ? hi.z : hi.w;
            a0 = i8x2_to_bf16x2(wl, kc);
            a2 = i8x2_to_bf16x2(wl >> 8, kc);
            a1 = i8x2_to_bf16x2(wh, kc);
            a3 = i8x2_to_bf16x2(wh >> 8, kc);
        } else {
            // piece s is this step's A fragment in register order (see the packed layout)
            a0 = w[s].x;
            a1 = w[s].y;
            a2 = w[s].z;
            a3 = w[s].w;
        }
        mma_bf16(d[s & 3], a0, a1, a2, a3, b0, b1);
    }
}

#if AIO_FFMA
// ------------------------------------------------------------------ CUDA-core consumer (comparison)
// Built with AIO_DEFINES="AIO_FFMA=1".  Same layouts, ring, partition and fixups; only the tile
// arithmetic differs: lane (g, c) converts its weights of rows g and g + 8 at its k (the k order of
// the MMA path) to fp32 and accumulates acc(h, m) = sum W[row g + 8h][k] x[m][k] with FFMA for every
// token m, in d[(8h + m) / 4][(8h + m) % 4].  ffma_finish reduces over the four lanes of a row pair
// and returns the D layout of the MMA path.
__device__ __forceinline__ float& acc_at(float (&d)[4][4], int h, int m) { return d[(8 * h + m) >> 2][(8 * h + m) & 3]; }
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
// int8 code in byte i of u (u = stored word ^ 0x80808080) -> float, exactly: 2^23 + q + 128 - (2^23 + 128)
__device__ __forceinline__ float i8f(uint32_t u, uint32_t i) {
    return __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7440u | i)) - 8388736.0f;
}
__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) { return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w; }

template <bool I8, int MT, class XL>
__device__ __forceinline__ void tile_ffma(float (&d)[4][4], const uint4 (&w)[TileT<I8>::kPieces], XL xload) {
#pragma unroll
    for (int t = 0; t < kRuns; ++t) {
        uint4 xq[MT];
#pragma unroll
        for (int m = 0; m < MT; ++m) xq[m] = xload(m, t);
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            float wg[4], wh[4];   // k0 .. k0 + 3 of rows g and g + 8
            if constexpr (I8) {
                const int wi = (t & 1) * 2 + q;   // stored (0, 2, 1, 3)
                const uint32_t a = word_of(w[t >> 1], wi) ^ 0x80808080u;
                const uint32_t b = word_of(w[kRuns / 2 + (t >> 1)], wi) ^ 0x80808080u;
                wg[0] = i8f(a, 0); wg[1] = i8f(a, 2); wg[2] = i8f(a, 1); wg[3] = i8f(a, 3);
                wh[0] = i8f(b, 0); wh[1] = i8f(b, 2); wh[2] = i8f(b, 1); wh[3] = i8f(b, 3);
            } else {
                const uint4& a = w[2 * t + q];
                wg[0] = bf_lo(a.x); wg[1] = bf_hi(a.x); wg[2] = bf_lo(a.z); wg[3] = bf_hi(a.z);
                wh[0] = bf_lo(a.y); wh[1] = bf_hi(a.y); wh[2] = bf_lo(a.w); wh[3] = bf_hi(a.w);
            }
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                const uint32_t xa = q ? xq[m].z : xq[m].x, xb = q ? xq[m].w : xq[m].y;
                const float x0 = bf_lo(xa), x1 = bf_hi(xa), x2 = bf_lo(xb), x3 = bf_hi(xb);
                float& a0 = acc_at(d, 0, m);
                float& a1 = acc_at(d, 1, m);
                a0 = fmaf(wg[3], x3, fmaf(wg[2], x2, fmaf(wg[1], x1, fmaf(wg[0], x0, a0))));
                a1 = fmaf(wh[3], x3, fmaf(wh[2], x2, fmaf(wh[1], x1, fmaf(wh[0], x0, a1))));
            }
        }
    }
}

// Group end: sum over the lanes c of each row pair, then lane (g, c) returns D[g][2c], D[g][2c+1],
// D[g+8][2c], D[g+8][2c+1] (0 for tokens >= M), as the MMA path does.
template <int MT>
__device__ __forceinline__ void ffma_finish(float (&d)[4][4], float (&sum)[4], int lane) {
    float r0[8], r1[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        float a = m < MT ? acc_at(d, 0, m) : 0.0f, b = m < MT ? acc_at(d, 1, m) : 0.0f;
        if (m < MT) {
            a += __shfl_xor_sync(0xffffffffu, a, 1);
            a += __shfl_xor_sync(0xffffffffu, a, 2);
            b += __shfl_xor_sync(0xffffffffu, b, 1);
            b += __shfl_xor_sync(0xffffffffu, b, 2);
        }
        r0[m] = a;
        r1[m] = b;
    }
    const int c = lane & 3;
    sum[0] = c == 0 ? r0[0] : c == 1 ? r0[2] : c == 2 ? r0[4] : r0[6];
    sum[1] = c == 0 ? r0[1] : c == 1 ? r0[3] : c == 2 ? r0[5] : r0[7];
    sum[2] = c == 0 ? r1[0] : c == 1 ? r1[2] : c == 2 ? r1[4] : r1[6];
    sum[3] = c == 0 ? r1[1] : c == 1 ? r1[3] : c == 2 ? r1[5] : r1[7];
}

// Full tile, x staged: xs0 = shared address of token 0's x at k = 256 kt + 8c, xsb = row stride in bytes.
template <bool I8, int MT>
__device__ __forceinline__ void ffma_full_s(float (&d)[4][4], uint32_t waddr, uint32_t xs0, uint32_t xsb) {
    uint4 w[TileT<I8>::kPieces];
#pragma unroll
    for (int j = 0; j < TileT<I8>::kPieces; ++j) w[j] = lds128(waddr + j * 512);
    tile_ffma<I8, MT>(d, w, [&](int m, int t) { return lds128(xs0 + m * xsb + 64 * t); });
}

// Full tile, x in global memory: x0 = x + 256 kt + 8c (token 0), K = row stride.
template <bool I8, int MT>
__device__ __forceinline__ void ffma_full_g(float (&d)[4][4], const uint8_t* tile_lane, const uint16_t* x0, int K) {
    uint4 w[TileT<I8>::kPieces];
#pragma unroll
    for (int j = 0; j < TileT<I8>::kPieces; ++j) w[j] = *reinterpret_cast<const uint4*>(tile_lane + j * 512);
    tile_ffma<I8, MT>(d, w, [&](int m, int t) {
        return *reinterpret_cast<const uint4*>(x0 + static_cast<size_t>(m) * K + 32 * t);
    });
}
#endif  // AIO_FFMA

// Any tile: full packed tiles in fragment order (piece j at j * 512 + 16 lane); ragged tiles
// (rows < 16 or klen < 256) and row-major weights as the row-major block [rows][klen].  Pieces
// outside the tile are zero, and so is x outside [kbase, kbase + klen) or for tokens >= M.
// x is read from xp = x + token g's row (row stride xstride elements), staged or global.
// x_l2: xrow_ptr is global memory other CTAs may have written earlier in the launch (read at L2).
template <bool I8>
__device__ __forceinline__ void tile_mma(float (&d)[4][4], const uint8_t* tile, int rows, int klen, int kbase,
                                         int lane, const Proj& P, const uint16_t* xrow_ptr, const I8Consts& kc,
                                         int xstride = 0, bool x_l2 = false) {
    using TL = TileT<I8>;
    constexpr int NP = TL::kPieces;
    const int g = lane >> 2, c = lane & 3;
    const bool full = rows == kRows && klen == kKT && !P.rowmajor;
    uint4 w[NP];
#pragma unroll
    for (int j = 0; j < NP; ++j) {
        if (full) {
            w[j] = *reinterpret_cast<const uint4*>(tile + j * 512 + lane * 16);
        } else if constexpr (I8) {
            // piece j: row g + 8 (j / (kRuns/2)), runs t = 2 (j % (kRuns/2)) and t + 1, 8 codes each
            const int r = g + 8 * (j / (kRuns / 2)), ka = 64 * (j % (kRuns / 2)) + 8 * c, kb = ka + 32;
            const uint8_t* rowp = tile + static_cast<size_t>(r) * klen;
            const uint2 lo = (r < rows && ka < klen) ? *reinterpret_cast<const uint2*>(rowp + ka) : make_uint2(0u, 0u);
            const uint2 hi = (r < rows && kb < klen) ? *reinterpret_cast<const uint2*>(rowp + kb) : make_uint2(0u, 0u);
            // row-major codes: put each word in the (0, 2, 1, 3) order full tiles are stored in
            w[j] = make_uint4(__byte_perm(lo.x, 0u, 0x3120u), __byte_perm(lo.y, 0u, 0x3120u),
                              __byte_perm(hi.x, 0u, 0x3120u), __byte_perm(hi.y, 0u, 0x3120u));
        } else {
            // piece j = k-step j's A fragment: 4 bf16 at k0 of rows g and g + 8, as pairs
            const int k0 = 32 * (j >> 1) + 8 * c + 4 * (j & 1);
            const uint2 lo = (g < rows && k0 < klen)
                                 ? *reinterpret_cast<const uint2*>(tile + (static_cast<size_t>(g) * klen + k0) * 2)
                                 : make_uint2(0u, 0u);
            const uint2 hi = (g + 8 < rows && k0 < klen)
                                 ? *reinterpret_cast<const uint2*>(tile + (static_cast<size_t>(g + 8) * klen + k0) * 2)
                                 : make_uint2(0u, 0u);
            w[j] = make_uint4(lo.x, hi.x, lo.y, hi.y);
        }
    }
#if AIO_FFMA
    // xrow_ptr is token 0's row here, xstride the row stride (staged or global)
    tile_ffma<I8, kMaxM>(d, w, [&](int m, int t) {
        const int k = 32 * t + 8 * c;
        return (m < P.M && k < klen) ? *reinterpret_cast<const uint4*>(xrow_ptr + static_cast<size_t>(m) * xstride + kbase + k)
                                     : make_uint4(0u, 0u, 0u, 0u);
    });
#else
    uint4 xv[kRuns];
    const bool xrow = g < P.M;
#pragma unroll
    for (int t = 0; t < kRuns; ++t) {
        const int k = 32 * t + 8 * c;
        const uint4* xq = reinterpret_cast<const uint4*>(xrow_ptr + kbase + k);
        xv[t] = (xrow && k < klen) ? (x_l2 ? __ldcg(xq) : *xq) : make_uint4(0u, 0u, 0u, 0u);
    }
    tile_mma_frag<I8>(d, w, xv, kc);
#endif
}

// A full packed tile with x in global memory: xp = x + token min(g, M-1)'s row + 256 kt + 8c.
// Lanes g >= M load a real token's x (the same addresses as lanes of token M-1, served once):
// they only fill columns of D for tokens >= M, which are never written.  No select is needed.
// CG: x may have been written by other CTAs earlier in the launch (a chained step's SwiGLU phase),
// so it is read at L2 rather than through L1.
template <bool I8, bool CG = false>
__device__ __forceinline__ void tile_mma_full(float (&d)[4][4], const uint8_t* tile_lane, const uint16_t* xp,
                                              const I8Consts& kc) {
    using TL = TileT<I8>;
    uint4 w[TL::kPieces];
#pragma unroll
    for (int j = 0; j < TL::kPieces; ++j) w[j] = *reinterpret_cast<const uint4*>(tile_lane + j * 512);
    uint4 xv[kRuns];
#pragma unroll
    for (int t = 0; t < kRuns; ++t) {
        const uint4* xq = reinterpret_cast<const uint4*>(xp + 32 * t);
        xv[t] = CG ? __ldcg(xq) : *xq;
    }
    tile_mma_frag<I8>(d, w, xv, kc);
}

// A full packed tile with x staged in shared memory: waddr / xaddr are shared-window addresses of
// this lane's piece 0 of W and of x (token min(g, M-1), k = 256 kt + 8c); both come in with
// ld.shared.v4.  The four lanes of a token read 64 contiguous bytes of x, and lanes g >= M read the
// same addresses as token M-1's lanes (a broadcast), so the x loads are free of bank conflicts and
// need no select; those lanes only fill columns of D for tokens >= M, which are never written.
template <bool I8>
__device__ __forceinline__ void tile_mma_full_s(float (&d)[4][4], uint32_t waddr, uint32_t xaddr, const I8Consts& kc) {
    using TL = TileT<I8>;
    uint4 w[TL::kPieces];
#pragma unroll
    for (int j = 0; j < TL::kPieces; ++j) w[j] = lds128(waddr + j * 512);
    uint4 xv[kRuns];
#pragma unroll
    for (int t = 0; t < kRuns; ++t) xv[t] = lds128(xaddr + 64 * t);
    tile_mma_frag<I8>(d, w, xv, kc);
}

template <bool I8>
__device__ __forceinline__ float row_scale(const Proj& P, int n) {
    if constexpr (I8) {
        return bf16_to_f32(P.scales[n]);
    } else {
        return 1.0f;
    }
}

constexpr uint32_t kSlotEmpty = 0xFFFFFFFFu;   // a partial slot not written yet
constexpr int kGather = 8;                    // contributors whose slots an owner loads at once

// A partial sum as stored in a slot: NaNs become the quiet NaN 0x7FC00000, so no stored value is
// ever kSlotEmpty.
__device__ __forceinline__ uint32_t slot_bits(float v) {
    return v != v ? 0x7FC00000u : __float_as_uint(v);
}

// Warp z has finished its tiles of row group g: lane (g', c) holds d = D[row g'][token 2c],
// D[row g'][token 2c + 1], D[row g' + 8][token 2c], D[row g' + 8][token 2c + 1].  Writes y (group
// complete in this warp), stores the partial (split group, not the owner), or, as the owner, adds
// the other contributors' partials and writes y.  Returns false if a wait for a partial expired or
// the launch already failed.
template <bool I8, int MT>
__device__ __forceinline__ bool finish_group(const Proj& P, const StreamArgs& s, int Z, const float (&d)[4], int g,
                                             int rows, long long z, long long t0, long long t1, int lane) {
    const int gr = lane >> 2, m0 = 2 * (lane & 3);
    const int row0 = g * kRows;
    const long long gfirst = static_cast<long long>(g) * P.NKT;
    const long long tl = gfirst + P.NKT - 1;

    if (t0 <= gfirst && t1 > tl) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int m = m0 + (i & 1), r = gr + 8 * (i >> 1);
            if (m < P.M && r < rows) P.y[static_cast<size_t>(m) * P.N + row0 + r] = d[i] * row_scale<I8>(P, row0 + r);
        }
        return true;
    }

    constexpr int V = kRows * MT;   // values per partial slot (P.M == MT)
    if (t0 > gfirst) {
        // Not the owner: g is this warp's first group (its last split group it always owns), so
        // one slot per warp suffices.  Publish [token][row] and go on.
        float* part = P.partial + static_cast<size_t>(z) * V;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int m = m0 + (i & 1), r = gr + 8 * (i >> 1);
            if (m < P.M) st_relaxed_u32(part + m * kRows + r, slot_bits(d[i]));
        }
        return true;
    }

    // The owner: this warp holds tile gfirst.  The other contributors are the next warps up to the
    // owner of tile tl (segments are contiguous and in warp order).  Lane l handles the values
    // v = 32 j + l (token v / 16, row v % 16) for j < NV.
    long long zl = z;
    while (zl + 1 < Z && seg(static_cast<int>(zl) + 1, Z, P.Tq, P.Tr) <= tl) ++zl;
    constexpr int NV = (kRows * MT + 31) / 32;
    float sum[NV];
    bool act[NV];
#pragma unroll
    for (int j = 0; j < NV; ++j) {
        const int v = 32 * j + lane;
        const int m = v / kRows, r = v - m * kRows;
        const int src = ((r & 7) * 4 + (m >> 1)) & 31;   // the lane holding the owner's own value
        const int idx = (r >> 3) * 2 + (m & 1);
        const float o0 = __shfl_sync(0xffffffffu, d[0], src), o1 = __shfl_sync(0xffffffffu, d[1], src);
        const float o2 = __shfl_sync(0xffffffffu, d[2], src), o3 = __shfl_sync(0xffffffffu, d[3], src);
        act[j] = v < V && r < rows;
        sum[j] = idx == 0 ? o0 : idx == 1 ? o1 : idx == 2 ? o2 : o3;
    }
    bool ok = true;
    // Up to kGather contributors at a time: all their slots are loaded together (independent loads,
    // one round trip), the ones still empty are re-loaded together until every slot is written,
    // and the values are added in warp order.
    for (long long zb = z + 1; ok && zb <= zl; zb += kGather) {
        unsigned want = 0u;   // contributors with a non-empty segment (the others publish nothing)
        int sprev = seg(static_cast<int>(zb), Z, P.Tq, P.Tr);
#pragma unroll
        for (int i = 0; i < kGather; ++i) {
            if (zb + i <= zl) {
                const int snext = seg(static_cast<int>(zb + i) + 1, Z, P.Tq, P.Tr);
                if (snext > sprev) want |= 1u << i;
                sprev = snext;
            }
        }
        const uint32_t* slots = reinterpret_cast<const uint32_t*>(P.partial) + static_cast<size_t>(zb) * V + lane;
        uint32_t bits[NV][kGather];
        uint32_t pend = 0u;   // bit j * kGather + i: value j of contributor zb + i not written yet
#pragma unroll
        for (int j = 0; j < NV; ++j) {
#pragma unroll
            for (int i = 0; i < kGather; ++i) {
                bits[j][i] = 0u;
                if (act[j] && (want >> i & 1u)) bits[j][i] = ld_relaxed_u32(slots + i * V + 32 * j);
            }
        }
#pragma unroll
        for (int j = 0; j < NV; ++j)
#pragma unroll
            for (int i = 0; i < kGather; ++i)
                if (act[j] && (want >> i & 1u) && bits[j][i] == kSlotEmpty) pend |= 1u << (j * kGather + i);
        if (pend) {
            const uint64_t start = globaltimer_ns();
            while (pend && ok) {
                uint32_t still = 0u;
#pragma unroll
                for (int j = 0; j < NV; ++j) {
#pragma unroll
                    for (int i = 0; i < kGather; ++i) {
                        if (pend >> (j * kGather + i) & 1u) {
                            bits[j][i] = ld_relaxed_u32(slots + i * V + 32 * j);
                            if (bits[j][i] == kSlotEmpty) still |= 1u << (j * kGather + i);
                        }
                    }
                }
                pend = still;
                if (pend) ok = ld_relaxed_u32(s.err) == 0u && globaltimer_ns() - start <= s.wait_limit_ns;
            }
        }
        if (ok) {
#pragma unroll
            for (int j = 0; j < NV; ++j) {
#pragma unroll
                for (int i = 0; i < kGather; ++i) {
                    if (act[j] && (want >> i & 1u)) {
                        sum[j] += __uint_as_float(bits[j][i]);
                        st_relaxed_u32(P.partial + (static_cast<size_t>(zb + i) * V + 32 * j + lane), kSlotEmpty);
                    }
                }
            }
        }
    }
    if (ok) {
#pragma unroll
        for (int j = 0; j < NV; ++j) {
            const int v = 32 * j + lane;
            const int m = v / kRows, r = v - m * kRows;
            if (act[j]) P.y[static_cast<size_t>(m) * P.N + row0 + r] = sum[j] * row_scale<I8>(P, row0 + r);
        }
    }
    return __all_sync(0xffffffffu, ok);
}

// Lane 0 polls until *counter >= target (bounded by limit_ns); the result is broadcast to the warp.
__device__ __noinline__ bool poll_global(const unsigned* counter, unsigned target, unsigned long long limit_ns,
                                         int lane) {
    int ok = 1;
    if (lane == 0 && ld_acquire(counter) < target) {
        const uint64_t start = globaltimer_ns();
        while (ld_acquire(counter) < target) {
            if (globaltimer_ns() - start > limit_ns) {
                ok = 0;
                break;
            }
        }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Same for a CTA-local flag in shared memory.
__device__ __noinline__ bool poll_shared(const unsigned* flag, unsigned target, unsigned long long limit_ns,
                                         int lane) {
    int ok = 1;
    if (lane == 0 && ld_acquire_cta_shared(flag) < target) {
        const uint64_t start = globaltimer_ns();
        while (ld_acquire_cta_shared(flag) < target) {
            if (globaltimer_ns() - start > limit_ns) {
                ok = 0;
                break;
            }
            __nanosleep(32);
        }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// This warp has finished its part of a phase (a projection, or the whole kernel).  Warps count in
// shared memory with acquire-release semantics; the last warp of the CTA fences at device scope
// (cumulatively publishing what every warp of the CTA wrote in the phase) and makes the one global
// increment.  Returns the global counter's previous value in the last warp, ~0u elsewhere.
__device__ __forceinline__ unsigned cta_arrive(unsigned* cta_count, unsigned* global_count, int lane) {
    __syncwarp();
    unsigned g = 0xffffffffu;
    if (lane == 0) {
        if (atom_add_acq_rel_cta_shared(cta_count, 1u) == static_cast<unsigned>(kWarps - 1)) {
            *cta_count = 0u;   // no warp of this CTA can arrive again before this phase completes
            __threadfence();
            g = atomicAdd(global_count, 1u);
        }
    }
    return __shfl_sync(0xffffffffu, g, 0);
}

// ------------------------------------------------------------------ decode attention
// Shared by the attention kernel (aio_attn.cu) and the attention phases of a chained step.
__device__ __forceinline__ uint2 lds64(uint32_t addr) {
    uint2 v;
    asm volatile("ld.shared.v2.b32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

// Sum over the warp of 16 per-lane values a[0..15] (one per position); returns, in lane l, the
// total for position (l >> 1) & 15.  Each step halves the values a lane holds: lanes whose bit o is
// set keep the upper half and send the lower, the others the reverse, so 8 + 4 + 2 + 1 + 1 shuffles
// replace 16 separate 5-step butterflies.
__device__ __forceinline__ float warp_sum16_transpose(float (&a)[16], int lane) {
#pragma unroll
    for (int o = 16, n = 8; o >= 2; o >>= 1, n >>= 1) {
        const bool hi = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < n; ++i) {
            const float send = hi ? a[i] : a[i + n];
            const float keep = hi ? a[i + n] : a[i];
            a[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    return a[0] + __shfl_xor_sync(0xffffffffu, a[0], 1);
}

// One unit of np <= 16 positions [p0, p0 + np) of one head, staged in shared memory: K rows at
// kaddr - 8 lane (256 B apart), V rows kAttnUnitBytes later.  Token m sits at position q0 + m and
// sees positions j <= q0 + m.  Lane l holds dims [4l, 4l + 4) of each token's q (scaled by
// log2(e) / sqrt(128)) and of its running weighted V sum; mx and ls are the running base-2 max and
// sum of an online softmax.  K and V rows are read from shared memory once for all tokens, and
// each step of the softmax runs for every token before the next, so the tokens' chains interleave.
// PRELOAD: all 16 K and V rows are loaded first (more loads in flight, 64 more registers).
template <int MT, bool PRELOAD = true>
__device__ __forceinline__ void attn_unit(uint32_t kaddr, int p0, int np, int q0, const float4 (&q4)[MT],
                                          float (&mx)[MT], float (&ls)[MT], float4 (&acc)[MT], int lane) {
    const uint32_t vaddr = kaddr + kAttnUnitBytes;
    constexpr int NR = PRELOAD ? kAttnPos : 1;
    uint2 kr[NR], vr[NR];
    auto krow = [&](int j) -> uint2 {
        if constexpr (PRELOAD) return kr[j];
        return j < np ? lds64(kaddr + j * (kHeadDim * 2)) : make_uint2(0u, 0u);
    };
    auto vrow = [&](int j) -> uint2 {
        if constexpr (PRELOAD) return vr[j];
        return j < np ? lds64(vaddr + j * (kHeadDim * 2)) : make_uint2(0u, 0u);
    };
    if constexpr (PRELOAD) {
#pragma unroll
        for (int j = 0; j < kAttnPos; ++j) {
            kr[j] = j < np ? lds64(kaddr + j * (kHeadDim * 2)) : make_uint2(0u, 0u);
            vr[j] = j < np ? lds64(vaddr + j * (kHeadDim * 2)) : make_uint2(0u, 0u);
        }
    }
    // lanes 2p and 2p + 1 hold position p's score (base-2 logits)
    const int pos = (lane >> 1) & 15;
    float sc[MT], bm[MT];
    bool vis[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        float part[kAttnPos];
#pragma unroll
        for (int j = 0; j < kAttnPos; ++j) {
            const uint2 kj = krow(j);
            const float k0 = __uint_as_float(kj.x << 16), k1 = __uint_as_float(kj.x & 0xFFFF0000u);
            const float k2 = __uint_as_float(kj.y << 16), k3 = __uint_as_float(kj.y & 0xFFFF0000u);
            part[j] = fmaf(q4[m].w, k3, fmaf(q4[m].z, k2, fmaf(q4[m].y, k1, q4[m].x * k0)));
        }
        const float sm = warp_sum16_transpose(part, lane);
        vis[m] = pos < np && p0 + pos <= q0 + m;
        sc[m] = vis[m] ? sm : -INFINITY;
        bm[m] = sc[m];
    }
#pragma unroll
    for (int o = 2; o < 32; o <<= 1)
#pragma unroll
        for (int m = 0; m < MT; ++m) bm[m] = fmaxf(bm[m], __shfl_xor_sync(0xffffffffu, bm[m], o));
    float pr[MT], ps[MT];
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        const float nm = fmaxf(mx[m], bm[m]);
        const bool live = nm != -INFINITY;   // some position seen so far is visible
        const float alpha = live ? exp2f(mx[m] - nm) : 1.0f;   // 0 while mx is -inf
        pr[m] = live && vis[m] ? exp2f(sc[m] - nm) : 0.0f;
        ps[m] = pr[m];
        ls[m] *= alpha;
        acc[m] = make_float4(acc[m].x * alpha, acc[m].y * alpha, acc[m].z * alpha, acc[m].w * alpha);
        if (live) mx[m] = nm;
    }
#pragma unroll
    for (int o = 2; o < 32; o <<= 1)
#pragma unroll
        for (int m = 0; m < MT; ++m) ps[m] += __shfl_xor_sync(0xffffffffu, ps[m], o);
#pragma unroll
    for (int m = 0; m < MT; ++m) ls[m] += ps[m];
#pragma unroll
    for (int j = 0; j < kAttnPos; ++j) {
        const uint2 vj = vrow(j);
        const float v0 = __uint_as_float(vj.x << 16), v1 = __uint_as_float(vj.x & 0xFFFF0000u);
        const float v2 = __uint_as_float(vj.y << 16), v3 = __uint_as_float(vj.y & 0xFFFF0000u);
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            const float pj = __shfl_sync(0xffffffffu, pr[m], 2 * j);   // 0 past np: V is zero there too
            acc[m] = make_float4(fmaf(pj, v0, acc[m].x), fmaf(pj, v1, acc[m].y), fmaf(pj, v2, acc[m].z),
                                 fmaf(pj, v3, acc[m].w));
        }
    }
}

// ------------------------------------------------------------------ x of a chained step
__device__ __forceinline__ void named_barrier_sync() {
    asm volatile("bar.sync 1, %0;" ::"n"(kThreads) : "memory");
}

// Data another CTA wrote before the grid barrier: read at L2, never from a stale L1 line.
__device__ __forceinline__ float4 ldcg4(const float* p) { return __ldcg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ uint32_t bf16x2_rn(float lo, float hi) {
    return static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(lo))) |
           (static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(hi))) << 16);
}

// Four consecutive x values of one token at k = 4i, rounded to bf16: into this CTA's staged copy,
// and from CTA 0 into the projection's x buffer as well.
__device__ __forceinline__ void put_x4(uint16_t* xs_row, uint16_t* xg_row, int i, float a, float b, float c, float d,
                                       bool cta0) {
    const uint2 v = make_uint2(bf16x2_rn(a, b), bf16x2_rn(c, d));
    *reinterpret_cast<uint2*>(xs_row + 4 * i) = v;
    if (cta0) *reinterpret_cast<uint2*>(xg_row + 4 * i) = v;
}

// silu(t) = t / (1 + e^-t), evaluated with e^-|t| so that the exponential never overflows (for
// t < 0 it is t e^t / (1 + e^t)).
__device__ __forceinline__ float silu(float t) {
    const float e = __expf(-fabsf(t));
    return __fdividef(t >= 0.0f ? t : t * e, 1.0f + e);
}

// x of a projection in a chained decoder step, computed by every thread of the CTA into the staged
// copy xs (row stride xs_stride) after the grid barrier, from buffers earlier projections wrote:
//   RMSNorm: h = h_in + xsrc (fp32 add; CTA 0 stores h in h_out), x = bf16(h * gamma / rms(h)),
//            rms(h) = sqrt(sum h^2 / K + eps), the sum reduced in a fixed order;
//   SwiGLU:  x = bf16(silu(g) * u), g = xsrc[m, k], u = xsrc[m, K + k];
//   slice:   x = bf16(xsrc[m, off + k]).
// red holds kWarps x kMaxM floats of shared scratch.  Ends with a CTA-wide barrier.
template <int MT>
__device__ __forceinline__ void prep_x(const ProjDesc* d, uint16_t* xs, int xs_stride, float* red, int warp,
                                       int lane) {
    const int tid = warp * 32 + lane;
    const int K = d->K, n4 = K / 4, op = d->xop;
    const bool cta0 = blockIdx.x == 0;
    uint16_t* xg = const_cast<uint16_t*>(d->x);
    const float* src = d->xsrc;
    if (op == kXRmsNorm) {
        const float* hin = d->h_in;
        float* hout = d->h_out;
        const uint2* g4 = reinterpret_cast<const uint2*>(d->gamma);
        constexpr int kCache = 4;   // float4 of h per thread and token held in registers (K <= 4096)
        if constexpr (MT <= 2) {
            if (n4 <= kCache * kThreads) {
                // one pass over global memory: h, the residual and gamma are loaded together
                float4 hv[MT][kCache];
                uint2 gv[kCache];
                float ss[MT];
#pragma unroll
                for (int c = 0; c < kCache; ++c) {
                    const int i = tid + c * kThreads;
                    gv[c] = i < n4 ? __ldg(g4 + i) : make_uint2(0u, 0u);
                }
#pragma unroll
                for (int m = 0; m < MT; ++m) {
#pragma unroll
                    for (int c = 0; c < kCache; ++c) {
                        const int i = tid + c * kThreads;
                        float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                        if (i < n4) {
                            a = ldcg4(hin + m * K + 4 * i);
                            if (src) {
                                const float4 b = ldcg4(src + m * K + 4 * i);
                                a.x += b.x;
                                a.y += b.y;
                                a.z += b.z;
                                a.w += b.w;
                            }
                        }
                        hv[m][c] = a;
                    }
                }
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    float acc = 0.0f;
#pragma unroll
                    for (int c = 0; c < kCache; ++c) {
                        const float4 a = hv[m][c];
                        acc = fmaf(a.x, a.x, acc);
                        acc = fmaf(a.y, a.y, acc);
                        acc = fmaf(a.z, a.z, acc);
                        acc = fmaf(a.w, a.w, acc);
                        const int i = tid + c * kThreads;
                        if (cta0 && hout && i < n4) *reinterpret_cast<float4*>(hout + m * K + 4 * i) = a;
                    }
                    ss[m] = acc;
                }
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    float v = ss[m];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    if (lane == 0) red[warp * kMaxM + m] = v;
                }
                named_barrier_sync();
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    float tot = 0.0f;
#pragma unroll
                    for (int w = 0; w < kWarps; ++w) tot += red[w * kMaxM + m];
                    const float inv = 1.0f / sqrtf(tot / static_cast<float>(K) + d->eps);
#pragma unroll
                    for (int c = 0; c < kCache; ++c) {
                        const int i = tid + c * kThreads;
                        if (i < n4) {
                            const float4 a = hv[m][c];
                            const uint2 gb = gv[c];
                            put_x4(xs + m * xs_stride, xg + m * K, i, a.x * __uint_as_float(gb.x << 16) * inv,
                                   a.y * __uint_as_float(gb.x & 0xFFFF0000u) * inv,
                                   a.z * __uint_as_float(gb.y << 16) * inv,
                                   a.w * __uint_as_float(gb.y & 0xFFFF0000u) * inv, cta0);
                        }
                    }
                }
                named_barrier_sync();
                return;
            }
        }
        // general case: two passes over global memory
        float ss[MT];
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float acc = 0.0f;
#pragma unroll 4
            for (int i = tid; i < n4; i += kThreads) {
                float4 a = ldcg4(hin + m * K + 4 * i);
                if (src) {
                    const float4 b = ldcg4(src + m * K + 4 * i);
                    a.x += b.x;
                    a.y += b.y;
                    a.z += b.z;
                    a.w += b.w;
                }
                acc = fmaf(a.x, a.x, acc);
                acc = fmaf(a.y, a.y, acc);
                acc = fmaf(a.z, a.z, acc);
                acc = fmaf(a.w, a.w, acc);
                if (cta0 && hout) *reinterpret_cast<float4*>(hout + m * K + 4 * i) = a;
            }
            ss[m] = acc;
        }
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float v = ss[m];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) red[warp * kMaxM + m] = v;
        }
        named_barrier_sync();
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) tot += red[w * kMaxM + m];
            const float inv = 1.0f / sqrtf(tot / static_cast<float>(K) + d->eps);
#pragma unroll 4
            for (int i = tid; i < n4; i += kThreads) {
                float4 a = ldcg4(hin + m * K + 4 * i);
                if (src) {
                    const float4 b = ldcg4(src + m * K + 4 * i);
                    a.x += b.x;
                    a.y += b.y;
                    a.z += b.z;
                    a.w += b.w;
                }
                const uint2 gb = __ldg(g4 + i);
                put_x4(xs + m * xs_stride, xg + m * K, i, a.x * __uint_as_float(gb.x << 16) * inv,
                       a.y * __uint_as_float(gb.x & 0xFFFF0000u) * inv, a.z * __uint_as_float(gb.y << 16) * inv,
                       a.w * __uint_as_float(gb.y & 0xFFFF0000u) * inv, cta0);
            }
        }
    } else if (op == kXSwiGlu) {
        // all loads of a batch are issued before its stores (the stores could alias them)
        constexpr int B = 6;
        const int stride = d->xsrc_stride;
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            for (int i0 = tid; i0 < n4; i0 += B * kThreads) {
                float4 g[B], u[B];
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const int i = i0 + b * kThreads;
                    if (i < n4) {
                        g[b] = ldcg4(src + m * stride + 4 * i);
                        u[b] = ldcg4(src + m * stride + K + 4 * i);
                    }
                }
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const int i = i0 + b * kThreads;
                    if (i < n4)
                        put_x4(xs + m * xs_stride, xg + m * K, i, silu(g[b].x) * u[b].x, silu(g[b].y) * u[b].y,
                               silu(g[b].z) * u[b].z, silu(g[b].w) * u[b].w, cta0);
                }
            }
        }
    } else {
        constexpr int B = 8;
        const int stride = d->xsrc_stride, off = d->xsrc_off;
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            for (int i0 = tid; i0 < n4; i0 += B * kThreads) {
                float4 v[B];
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const int i = i0 + b * kThreads;
                    if (i < n4) v[b] = ldcg4(src + m * stride + off + 4 * i);
                }
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const int i = i0 + b * kThreads;
                    if (i < n4) put_x4(xs + m * xs_stride, xg + m * K, i, v[b].x, v[b].y, v[b].z, v[b].w, cta0);
                }
            }
        }
    }
    named_barrier_sync();
}

// The merge phase of a chained step's attention.  CTA c merges the (head, token) items c, c + G,
// ...: warp w takes the records w, w + 8, ... of the warps whose units cover the head, loads them 8
// at a time and combines them with a running maximum (each record's weighted sums rescaled by
// 2^(max_r - max)); warp 0 then combines the 8 warps' results in order, rescaled the same way,
// divides by the total weight and writes the head's slice of the O projection's x row as bf16.
// The order is fixed, whatever the timing.  Every warp of a CTA takes part (named barriers),
// whatever its state.
template <int MT>
__device__ __noinline__ void attn_merge(const ProjDesc* d, int Z, uint8_t* scratch, int warp, int lane) {
    const int L = attn_len(d, MT);
    if (L == 0) return;
    const int nch = (L + kAttnPos - 1) / kAttnPos;
    const int U = d->n_heads * nch, Tq = U / Z, Tr = U - Tq * Z;
    const int items = d->n_heads * MT, H = d->n_heads * kHeadDim;
    float4* wacc = reinterpret_cast<float4*>(scratch);           // [kWarps][32]
    float* wml = reinterpret_cast<float*>(wacc + kWarps * 32);    // [kWarps][2]: max, weight
    constexpr int B = 8;   // records a warp loads at once
    for (int it = blockIdx.x; it < items; it += gridDim.x) {
        const int h = it / MT, m = it - h * MT;
        const int ua = h * nch, ub = ua + nch - 1;   // the head's units
        // the warps holding units ua and ub (segment starts are nondecreasing in z)
        int zlo = static_cast<int>(static_cast<long long>(ua) * Z / U);
        while (zlo > 0 && seg(zlo, Z, Tq, Tr) > ua) --zlo;
        while (seg(zlo + 1, Z, Tq, Tr) <= ua) ++zlo;
        int zhi = static_cast<int>(static_cast<long long>(ub) * Z / U);
        while (zhi > 0 && seg(zhi, Z, Tq, Tr) > ub) --zhi;
        while (seg(zhi + 1, Z, Tq, Tr) <= ub) ++zhi;
        const int n = zhi - zlo + 1;
        float gm = -INFINITY, gl = 0.0f;
        float4 a = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        for (int i0 = warp; i0 < n; i0 += B * kWarps) {
            float rm[B], rl[B];
            float4 rv[B];
#pragma unroll
            for (int b = 0; b < B; ++b) {   // the records' loads, issued together
                const int i = i0 + b * kWarps;
                rm[b] = -INFINITY;
                rl[b] = 0.0f;
                rv[b] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                if (i < n) {
                    const int zz = zlo + i, s0 = seg(zz, Z, Tq, Tr);
                    if (seg(zz + 1, Z, Tq, Tr) > s0) {   // a non-empty segment: its first or second record
                        const float* r = d->apart + ((zz * 2 + (s0 / nch == h ? 0 : 1)) * MT + m) * kAttnRec;
                        rm[b] = __ldcg(r + 128);
                        rl[b] = __ldcg(r + 129);
                        rv[b] = ldcg4(r + 4 * lane);
                    }
                }
            }
#pragma unroll
            for (int b = 0; b < B; ++b) {   // combined in record order
                if (rm[b] == -INFINITY) continue;
                const float nm = fmaxf(gm, rm[b]);
                const float so = exp2f(gm - nm), sr = exp2f(rm[b] - nm);   // so = 0 while gm is -inf
                gl = gl * so + rl[b] * sr;
                a = make_float4(fmaf(rv[b].x, sr, a.x * so), fmaf(rv[b].y, sr, a.y * so), fmaf(rv[b].z, sr, a.z * so),
                                fmaf(rv[b].w, sr, a.w * so));
                gm = nm;
            }
        }
        wacc[warp * 32 + lane] = a;
        if (lane == 0) {
            wml[2 * warp] = gm;
            wml[2 * warp + 1] = gl;
        }
        named_barrier_sync();
        if (warp == 0) {
            float M_ = -INFINITY;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) M_ = fmaxf(M_, wml[2 * w]);
            float lt = 0.0f;
            float4 at = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
            for (int w = 0; w < kWarps; ++w) {
                const float mw = wml[2 * w];
                const float sw = mw == -INFINITY ? 0.0f : exp2f(mw - M_);
                lt = fmaf(wml[2 * w + 1], sw, lt);
                const float4 v = wacc[w * 32 + lane];
                at = make_float4(fmaf(v.x, sw, at.x), fmaf(v.y, sw, at.y), fmaf(v.z, sw, at.z), fmaf(v.w, sw, at.w));
            }
            const float inv = 1.0f / lt;
            *reinterpret_cast<uint2*>(d->aout + static_cast<size_t>(m) * H + h * kHeadDim + 4 * lane) =
                make_uint2(bf16x2_rn(at.x * inv, at.y * inv), bf16x2_rn(at.z * inv, at.w * inv));
        }
        named_barrier_sync();   // the warps' results are read before the next item rewrites them
    }
    fence_proxy_async_smem();   // the scratch writes precede the next phase's bulk copies into this area
}

// A warp's ring state, handed to and returned by the out-of-line attention phase.
struct RingCtx {
    ChunkCursor cur;
    int islot, in_flight, ahead, cslot;
    uint32_t cphase;
    bool first_issue, dead;
};

// The attention phase of a chained step, for one warp: attention of the M new tokens over the
// layer's cache, over this warp's units, each one ring slot of 16 positions of one head.  The new
// tokens' rows (positions L_past .. L - 1) were copied stale from the cache: they are replaced by k
// and v of the QKV output rounded to bf16, which are also written back to the cache.  A warp's units
// span at most two heads (n_heads <= Z), so it leaves at most two partial records.  The ring is
// refilled as in the projection phases (the issue and refill steps of the stream kernel, restated
// on the state passed in).
template <int MT, bool I8>
__device__ __noinline__ RingCtx attn_phase(RingCtx r, const StreamArgs& s, const ProjDesc* D, uint8_t* ring,
                                           uint64_t* bars, int z, int lane, uint64_t pol, int p) {
    using TL = TileT<I8>;
    using SL = LayoutFor<MT, I8, true>;   // phases run in chained kernels
    constexpr int C = TL::kChunk;
    constexpr int S = I8 ? SL::kStagesI8 : SL::kStages;
    const int Z = s.Z;
    auto issue_next = [&]() -> bool {
        int ip, it, nt;
        if (!cursor_next<true>(r.cur, s, z, Z, C, ip, it, nt)) return false;
        if (lane == 0) {
            if (r.cur.cur.rowmajor == kIssueAttn)
                issue_attn_unit(r.cur.cur, it, ring + r.islot * TL::kSlot, &bars[r.islot], pol);
            else
                issue_chunk<I8>(r.cur.cur, it, nt, ring + r.islot * TL::kSlot, &bars[r.islot], pol);
        }
        r.first_issue = false;
        r.islot = (r.islot + 1 == S) ? 0 : r.islot + 1;
        return true;
    };
    auto refill = [&]() {
        const bool later = r.cur.p > p || r.cur.t >= r.cur.te;
        if (later && r.ahead >= TL::kAheadLive) {
            --r.in_flight;
            return;
        }
        if (!issue_next()) {
            --r.in_flight;
        } else if (later) {
            ++r.ahead;
        }
    };
    int L, nch, Tq, Tr;
    attn_geom(D, MT, Z, L, nch, Tq, Tr);
    if (L == 0 && z == 0 && lane == 0) atomicCAS(s.err, 0, kDevErrAttn);
    const int u0 = seg(z, Z, Tq, Tr), u1 = seg(z + 1, Z, Tq, Tr);
    const int H = D->n_heads * kHeadDim, qs = D->xsrc_stride, Lp = L - MT;
    const float* qkv = D->xsrc;
    uint16_t* kvc = D->kv;
    const size_t voff = static_cast<size_t>(D->n_heads) * D->L_max * kHeadDim;
    const float qscale = 1.4426950408889634f / sqrtf(static_cast<float>(kHeadDim));   // log2(e) / sqrt(d)
    float4 q4[MT], acc[MT];
    float mx[MT], ls[MT];
    int head = -1, sidx = -1;
    auto flush = [&]() {
        if (head < 0) return;
        float* base = D->apart + (static_cast<size_t>(z) * 2 + sidx) * MT * kAttnRec;
#pragma unroll
        for (int m = 0; m < MT; ++m) {
            float* rec = base + m * kAttnRec;
            *reinterpret_cast<float4*>(rec + 4 * lane) = acc[m];
            if (lane == 0) {
                rec[128] = mx[m];
                rec[129] = ls[m];
            }
        }
    };
    int h = nch ? u0 / nch : 0, c = u0 - h * nch - 1;
    for (int u = u0; u < u1 && !r.dead; ++u) {
        if (++c == nch) {
            c = 0;
            ++h;
        }
        if (h != head) {
            flush();
            head = h;
            ++sidx;
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                const float4 t = ldcg4(qkv + static_cast<size_t>(m) * qs + h * kHeadDim + 4 * lane);
                q4[m] = make_float4(t.x * qscale, t.y * qscale, t.z * qscale, t.w * qscale);
                mx[m] = -INFINITY;
                ls[m] = 0.0f;
                acc[m] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            }
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[r.cslot], r.cphase, s.wait_limit_ns))) {
            if (lane == 0) atomicExch(s.err, kDevErrTimeout);
            r.dead = true;
            break;
        }
        const int p0 = c * kAttnPos, np = min(kAttnPos, L - p0);
        uint8_t* slot = ring + r.cslot * TL::kSlot;
        const int jn0 = max(p0, Lp), jn1 = p0 + np;
        if (jn0 < jn1) {
            for (int j = jn0; j < jn1; ++j) {
                const int m = j - Lp, row = j - p0;
                const float* src = qkv + static_cast<size_t>(m) * qs + h * kHeadDim + 4 * lane;
                const float4 kf = ldcg4(src + H), vf = ldcg4(src + 2 * H);
                const uint2 kb = make_uint2(bf16x2_rn(kf.x, kf.y), bf16x2_rn(kf.z, kf.w));
                const uint2 vb = make_uint2(bf16x2_rn(vf.x, vf.y), bf16x2_rn(vf.z, vf.w));
                *reinterpret_cast<uint2*>(slot + row * (kHeadDim * 2) + 8 * lane) = kb;
                *reinterpret_cast<uint2*>(slot + kAttnUnitBytes + row * (kHeadDim * 2) + 8 * lane) = vb;
                const size_t off = (static_cast<size_t>(h) * D->L_max + j) * kHeadDim + 4 * lane;
                *reinterpret_cast<uint2*>(kvc + off) = kb;
                *reinterpret_cast<uint2*>(kvc + voff + off) = vb;
            }
            fence_proxy_async_smem();   // these writes precede the slot's next bulk copy
            __syncwarp();               // every lane's rows are in place before any lane reads
        }
        attn_unit<MT, false>(smem_addr(slot) + 8 * lane, p0, np, Lp, q4, mx, ls, acc, lane);
        __syncwarp();   // every lane's reads of the slot are done before it is refilled
        r.cslot = (r.cslot + 1 == S) ? 0 : r.cslot + 1;
        r.cphase ^= (r.cslot == 0) ? 1u : 0u;
        refill();
    }
    flush();
    if (!r.dead) {
        while (r.ahead < TL::kAhead && r.in_flight < S && issue_next()) {
            ++r.in_flight;
            ++r.ahead;
        }
    } else {
        // wait (bounded) for this warp's copies still in flight, then stop issuing
        for (int j = 0; j < r.in_flight; ++j) {
            mbar_wait(&bars[r.cslot], r.cphase, s.wait_limit_ns);
            r.cslot = (r.cslot + 1 == S) ? 0 : r.cslot + 1;
            r.cphase ^= (r.cslot == 0) ? 1u : 0u;
        }
        r.in_flight = 0;
    }
    return r;
}

// The stream kernel: one CTA per SM, every warp streams its segment of every projection through
// its own bulk-copy ring.  All per-tile bookkeeping is incremental 32-bit arithmetic; divisions
// happen once per chunk (issue) or once per projection (consume).  CH: a chained step, where a
// projection's x may be computed on the device (prep_x); the plain step's kernels carry none of
// that code.  PH: a chained step that also has attention, merge or SwiGLU phases (their own
// instantiations, so that the chained kernels without them keep their registers for the projections).
template <int MT, bool I8, bool CH, bool PH = false>
__global__ void __launch_bounds__(kThreads, 1) aio_stream_kernel(const __grid_constant__ StreamArgs s) {
    using TL = TileT<I8>;
    using SL = LayoutFor<MT, I8, CH>;
    static_assert(CH || !PH, "phases belong to chained steps");
    static_assert(!PH || TL::kSlot >= kAttnSlot, "a ring slot holds one attention unit");
    constexpr int C = TL::kChunk;
    constexpr int S = I8 ? SL::kStagesI8 : SL::kStages;   // ring slots per warp
    constexpr int E = TL::kEsize;
    extern __shared__ __align__(1024) uint8_t smem[];
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * SL::kRingBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * SL::kRingBytes) + warp * SL::kMaxStages;
    // CTA-level sync words: [0] warps of this CTA done with the current phase, [1] highest projection
    // index whose predecessor is known complete (published by warp 0).
    unsigned* cta_sync = reinterpret_cast<unsigned*>(smem + SL::kSyncOffset);
    // x of the current projection, staged once per CTA when it fits (one bulk copy by warp 0).
    uint64_t* xbar = reinterpret_cast<uint64_t*>(smem + SL::kSyncOffset + 16);
    uint16_t* xs = reinterpret_cast<uint16_t*>(smem + SL::kXsOffset);
    [[maybe_unused]] float* red = reinterpret_cast<float*>(smem + SL::kAuxOffset);   // x preparation scratch

    griddep_launch_dependents();

    const long long z = static_cast<long long>(blockIdx.x) * kWarps + warp;
    const int Z = s.Z;
    if (lane == 0) {
#pragma unroll
        for (int i = 0; i < S; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (threadIdx.x == 0) {
        cta_sync[0] = 0u;
        cta_sync[1] = 0u;
        mbar_init(xbar, 1);
        fence_mbar_init();
    }
    __syncthreads();   // barriers and sync words are initialised (later CTA-wide barriers: prep_x only)
    const uint64_t pol = policy_evict_first();
    const I8Consts kc = i8_consts();

    // The issue cursor walks this warp's tiles of all projections in consumption order.
    ChunkCursor ring_cur;
    cursor_init<PH>(ring_cur, s, static_cast<int>(z), Z);
    int islot = 0;
    bool first_issue = true;
    const bool stall = s.test_stall && z == Z - 1;   // the grid's last warp always owns >= 1 tile
    auto issue_next = [&]() -> bool {
        int ip, it, nt;
        if (!cursor_next<PH>(ring_cur, s, static_cast<int>(z), Z, C, ip, it, nt)) return false;
        if (PH && ring_cur.cur.rowmajor == kIssueAttn) {
            if (lane == 0) issue_attn_unit(ring_cur.cur, it, ring + islot * TL::kSlot, &bars[islot], pol);
        } else if (lane == 0 && !(stall && first_issue)) {   // test hook: this slot's barrier never completes
            issue_chunk<I8>(ring_cur.cur, it, nt, ring + islot * TL::kSlot, &bars[islot], pol);
        }
        first_issue = false;
        islot = (islot + 1 == S) ? 0 : islot + 1;
        return true;
    };
    int in_flight = 0;
    for (int i = 0; i < S; ++i) {
        if (!issue_next()) break;
        ++in_flight;
    }
    // Chunks of projections after the one being consumed take at most TL::kAheadLive slots while
    // the warp still has tiles of the current one, TL::kAhead once it has finished them (its last
    // gather done); the rest of the ring is filled when the next projection starts.
    int ahead = 0;
    auto refill = [&](int p) {
        const bool later = ring_cur.p > p || ring_cur.t >= ring_cur.te;
        if (later && ahead >= TL::kAheadLive) {
            --in_flight;
            return;
        }
        if (!issue_next()) {
            --in_flight;
        } else if (later) {
            ++ahead;
        }
    };

    // With programmatic dependent launch, everything below (x, y, workspace) waits for the
    // previous grid on the stream.
    griddep_wait();

    const unsigned G = gridDim.x;
    int cslot = 0;
    uint32_t cphase = 0;
    uint32_t xphase = 0;
    bool dead = false;    // set after a timeout: stop consuming, keep signalling
    for (int p = 0; p < s.nproj; ++p) {
        Proj P = load_proj<CH>(proj_desc(s, p), MT);
        // the phase kind is reloaded where it is needed (the chained kernels are short of registers)
        auto kind_of = [&]() { return PH ? proj_desc(s, p)->kind : kPhaseProj; };
        const long long t0 = seg(static_cast<int>(z), Z, P.Tq, P.Tr), t1 = seg(static_cast<int>(z) + 1, Z, P.Tq, P.Tr);
        // Staged x rows are kXsPad elements apart beyond K, so two tokens read in one shared-memory
        // phase fall in different banks.
        const int xs_stride = P.K + kXsPad;
        const bool stage = kind_of() == kPhaseProj && P.M * xs_stride * 2 <= SL::kXsBytes;
        // Plain kernels: an x that no phase of the launch writes (the host checks every buffer the
        // step writes) was staged by this CTA's last warp at the end of the previous projection, so
        // that its copy overlaps the grid barrier; computing still waits for the barrier.
        const bool early = !CH && p > 0 && stage && !P.xfence;
        // Warp 0 stages x once every CTA has finished the previous projection (every warp of this
        // CTA has then finished reading the previous x and fenced its reads against async writes):
        // one bulk copy per token row.  When x may have been written by other CTAs earlier in the
        // launch (generic stores, ordered before the grid counter's acquire), a proxy fence orders
        // them before these async-proxy reads: in a chained step whenever x is staged as given (the
        // O projection after attention), in a plain step where the host found x aliased.
        auto stage_x = [&]() {
            if (stage && !early && (!CH || P.xop == kXGiven) && lane == 0) {
                if (CH || P.xfence) fence_proxy_async_all();
                mbar_expect_tx(xbar, static_cast<uint32_t>(P.M * P.K * 2));
                for (int m = 0; m < P.M; ++m)
                    bulk_g2s_plain(xs + m * xs_stride, P.x + static_cast<size_t>(m) * P.K,
                                   static_cast<uint32_t>(P.K * 2), xbar);
            }
        };
        if (p == 0 && warp == 0) stage_x();
        if (p > 0) {
            // Projection p reads x only after every CTA finished projection p-1.
            bool ok;
            if (warp == 0) {
                const bool polled = !dead && poll_global(&s.done[p - 1], G, s.wait_limit_ns, lane);
                ok = dead || polled;
                stage_x();
                if (lane == 0) st_release_cta_shared(&cta_sync[1], static_cast<unsigned>(p));
                if (polled && p > 1 && blockIdx.x == 0 && lane == 0) s.done[p - 2] = 0u;   // nobody polls it any more
            } else if (AIO_XBAR_ONLY && stage && !early && (!CH || P.xop == kXGiven)) {
                // warp 0 stages x only after the grid counter is complete, so the staged x's
                // barrier, waited on below, already orders this warp after the previous projection
                ok = true;
            } else {
                ok = poll_shared(&cta_sync[1], static_cast<unsigned>(p), s.wait_limit_ns, lane);
            }
            __syncwarp();
            if (!ok && !dead) {
                if (lane == 0) atomicExch(s.err, kDevErrGridTimeout);
                dead = true;
            }
        }
        if (stage && (!CH || P.xop == kXGiven)) {
            // every warp waits for the staged x (also so that no copy is in flight at exit)
            if (!__all_sync(0xffffffffu, mbar_wait(xbar, xphase, s.wait_limit_ns)) && !dead) {
                if (lane == 0) atomicExch(s.err, kDevErrTimeout);
                dead = true;
            }
            xphase ^= 1u;
        }
        if constexpr (CH) {
            if (P.xop != kXGiven) {
                // chained step: every warp of the CTA computes x (uniform over the CTA, dead or not)
                if (stage) {
                    prep_x<MT>(proj_desc(s, p), xs, xs_stride, red, warp, lane);
                } else if (!dead) {
                    if (lane == 0) atomicCAS(s.err, 0, kDevErrPrep);
                    dead = true;
                }
            }
        }
        ahead = 0;
        if (!dead) {
            while (in_flight < S && issue_next()) ++in_flight;
        }
        if constexpr (PH) {
            const int kind = kind_of();
            if (kind == kPhaseAttn) {
                RingCtx rc{ring_cur, islot, in_flight, ahead, cslot, cphase, first_issue, dead};
                rc = attn_phase<MT, I8>(rc, s, proj_desc(s, p), ring, bars, static_cast<int>(z), lane, pol, p);
                ring_cur = rc.cur;
                islot = rc.islot;
                in_flight = rc.in_flight;
                ahead = rc.ahead;
                cslot = rc.cslot;
                cphase = rc.cphase;
                first_issue = rc.first_issue;
                dead = rc.dead;
            } else if (kind == kPhaseMerge) {
                attn_merge<MT>(proj_desc(s, p), Z, reinterpret_cast<uint8_t*>(xs), warp, lane);
            } else if (kind == kPhaseSwiGlu) {
                // x[m, k] = bf16(silu(src[m, k]) * src[m, K + k]), four values per thread, over the grid
                const ProjDesc* D = proj_desc(s, p);
                const int K = D->K, n4 = K / 4, stride = D->xsrc_stride, total = MT * n4;
                for (int i = blockIdx.x * kThreads + threadIdx.x; i < total; i += gridDim.x * kThreads) {
                    const int m = i / n4, q = i - m * n4;
                    const float4 g = ldcg4(D->xsrc + static_cast<size_t>(m) * stride + 4 * q);
                    const float4 u = ldcg4(D->xsrc + static_cast<size_t>(m) * stride + K + 4 * q);
                    *reinterpret_cast<uint2*>(D->aout + static_cast<size_t>(m) * K + 4 * q) =
                        make_uint2(bf16x2_rn(silu(g.x) * u.x, silu(g.y) * u.y), bf16x2_rn(silu(g.z) * u.z, silu(g.w) * u.w));
                }
            }
        }
        if (kind_of() == kPhaseProj && !dead && t1 > t0) {
            float d[4][4] = {};
            const int NKT = P.NKT;
            const int last_len = P.K - (NKT - 1) * kKT;
            int t = static_cast<int>(t0);
            const int tend = static_cast<int>(t1);
            int g = t / NKT, kt = t - g * NKT;
            int rows = min(kRows, P.N - g * kRows);
            const int tok = lane >> 2;
            // x of this lane's token (rows >= M are never read): the staged copy or global memory
            [[maybe_unused]] const uint16_t* xrow_ptr = stage ? xs + tok * xs_stride : P.x + static_cast<size_t>(tok) * P.K;
            const int xtok = min(tok, MT - 1);   // full tiles: lanes of tokens >= M read token M-1's x
            [[maybe_unused]] const uint16_t* xlane = P.x + static_cast<size_t>(xtok) * P.K + 8 * (lane & 3);
            const uint32_t xs_lane = smem_addr(xs) + static_cast<uint32_t>((xtok * xs_stride + 8 * (lane & 3)) * 2);
            // The tile loop, compiled twice: FAST is the common case (every tile full, x staged), with
            // the tile shape, the x source and the row count known at compile time, so each tile
            // carries fewer branches; the general copy takes ragged, row-major and unstaged tiles.
            auto consume = [&](auto fast_tag) {
                constexpr bool FAST = decltype(fast_tag)::value;
                while (t < tend) {
                    if (!__all_sync(0xffffffffu, mbar_wait(&bars[cslot], cphase, s.wait_limit_ns))) {
                        if (lane == 0) atomicExch(s.err, kDevErrTimeout);
                        dead = true;
                        break;
                    }
                    const int nt = min(C, tend - t);
                    const uint8_t* tp = ring + cslot * TL::kSlot;
#if !AIO_FFMA
                    if constexpr (FAST && kWideLaunch<MT, I8, CH>) {
                        // Early release (the wide launches, whose rings have two slots):
                        // read the slot's tiles of W into registers and hand the slot back to the
                        // issuing lane before the arithmetic, so that its next copy is in flight while
                        // these tiles are computed.  Every lane's reads are ordered before lane 0's
                        // copy by the warp barrier and the proxy fence.
                        uint4 wr[C][TL::kPieces];
                        const uint32_t wa = smem_addr(tp) + lane * 16;
#pragma unroll
                        for (int j = 0; j < C; ++j)
#pragma unroll
                            for (int q = 0; q < TL::kPieces; ++q) wr[j][q] = lds128(wa + j * TL::kBytes + q * 512);
                        __syncwarp();
                        if (lane == 0) fence_proxy_async_smem();
                        cslot = (cslot + 1 == S) ? 0 : cslot + 1;
                        cphase ^= (cslot == 0) ? 1u : 0u;
                        refill(p);
#pragma unroll
                        for (int j = 0; j < C; ++j) {
                            if (j < nt) {
                                uint4 xv[kRuns];
#pragma unroll
                                for (int u = 0; u < kRuns; ++u) xv[u] = lds128(xs_lane + kt * (kKT * 2) + 64 * u);
                                tile_mma_frag<I8>(d, wr[j], xv, kc);
                                if (kt == NKT - 1 || t == tend - 1) {
                                    float sum[4];
#pragma unroll
                                    for (int i = 0; i < 4; ++i) sum[i] = (d[0][i] + d[1][i]) + (d[2][i] + d[3][i]);
                                    if (!finish_group<I8, MT>(P, s, Z, sum, g, kRows, z, t0, t1, lane)) {
                                        if (lane == 0) atomicCAS(s.err, 0, kDevErrTimeout);
                                        dead = true;
                                    }
#pragma unroll
                                    for (int q = 0; q < 4; ++q)
#pragma unroll
                                        for (int i = 0; i < 4; ++i) d[q][i] = 0.0f;
                                }
                                ++t;
                                if (++kt == NKT) {
                                    kt = 0;
                                    ++g;
                                }
                            }
                        }
                        continue;
                    }
#endif
#pragma unroll
                    for (int j = 0; j < C; ++j) {
                        if (j < nt) {
                            const int klen = FAST ? kKT : (kt == NKT - 1 ? last_len : kKT);
#if AIO_FFMA
                            if (FAST || (P.uniform && stage)) {
                                ffma_full_s<I8, MT>(d, smem_addr(tp) + lane * 16,
                                                    smem_addr(xs) + 16 * (lane & 3) + kt * (kKT * 2), xs_stride * 2);
                            } else if (P.uniform) {
                                ffma_full_g<I8, MT>(d, tp + lane * 16, P.x + 8 * (lane & 3) + kt * kKT, P.K);
                            } else {
                                tile_mma<I8>(d, tp, rows, klen, kt * kKT, lane, P, stage ? xs : P.x, kc,
                                             stage ? xs_stride : P.K);
                            }
#else
                            if (FAST || (P.uniform && stage)) {
                                tile_mma_full_s<I8>(d, smem_addr(tp) + lane * 16, xs_lane + kt * (kKT * 2), kc);
                            } else if (P.uniform) {
                                tile_mma_full<I8, PH>(d, tp + lane * 16, xlane + kt * kKT, kc);
                            } else {
                                tile_mma<I8>(d, tp, rows, klen, kt * kKT, lane, P, xrow_ptr, kc, 0, PH && !stage);
                            }
#endif
                            tp += FAST ? TL::kBytes : rows * klen * E;
                            if (kt == NKT - 1 || t == tend - 1) {
                                float sum[4];
#if AIO_FFMA
                                ffma_finish<MT>(d, sum, lane);
#else
#pragma unroll
                                for (int i = 0; i < 4; ++i) sum[i] = (d[0][i] + d[1][i]) + (d[2][i] + d[3][i]);
#endif
                                if (!finish_group<I8, MT>(P, s, Z, sum, g, FAST ? kRows : rows, z, t0, t1, lane)) {
                                    if (lane == 0) atomicCAS(s.err, 0, kDevErrTimeout);
                                    dead = true;
                                }
#pragma unroll
                                for (int q = 0; q < 4; ++q)
#pragma unroll
                                    for (int i = 0; i < 4; ++i) d[q][i] = 0.0f;
                            }
                            ++t;
                            if (++kt == NKT) {
                                kt = 0;
                                ++g;
                                if (!FAST) rows = min(kRows, P.N - g * kRows);
                            }
                        }
                    }
                    // Every lane's reads of the slot have returned (their values fed the MMAs above), so
                    // lane 0 may let the bulk copy overwrite it, as a consumer release would.
                    __syncwarp();
                    cslot = (cslot + 1 == S) ? 0 : cslot + 1;
                    cphase ^= (cslot == 0) ? 1u : 0u;
                    refill(p);
                }
            };
            if (P.uniform && stage) {
                consume(std::true_type{});
            } else {
                consume(std::false_type{});
            }
            if (!dead) {
                while (ahead < TL::kAhead && in_flight < S && issue_next()) {
                    ++in_flight;
                    ++ahead;
                }
            }
            if (dead) {
                // wait (bounded) for this warp's copies still in flight, then stop issuing
                for (int j = 0; j < in_flight; ++j) {
                    mbar_wait(&bars[cslot], cphase, s.wait_limit_ns);
                    cslot = (cslot + 1 == S) ? 0 : cslot + 1;
                    cphase ^= (cslot == 0) ? 1u : 0u;
                }
                in_flight = 0;
            }
        }
        if (stage) {
            __syncwarp();
            if (lane == 0) fence_proxy_async_smem();   // this warp's reads of xs precede the next staging
        }
        if (s.nproj > 1 && p + 1 < s.nproj) {
            const unsigned g = cta_arrive(&cta_sync[0], &s.done[p], lane);
            if constexpr (!CH) {
                if (g != 0xffffffffu && lane == 0) {
                    // the CTA's last warp: every warp has finished (and fenced) its reads of this
                    // projection's x, so the next one's may be staged now if nothing writes it
                    const Proj Q = load_proj<CH>(proj_desc(s, p + 1), MT);
                    const int qs = Q.K + kXsPad;
                    if (Q.M * qs * 2 <= SL::kXsBytes && !Q.xfence) {
                        mbar_expect_tx(xbar, static_cast<uint32_t>(Q.M * Q.K * 2));
                        for (int m = 0; m < Q.M; ++m)
                            bulk_g2s_plain(xs + m * qs, Q.x + static_cast<size_t>(m) * Q.K, static_cast<uint32_t>(Q.K * 2), xbar);
                    }
                }
            }
        }
    }
    if (s.nproj > 1) {
        const unsigned prev = cta_arrive(&cta_sync[0], s.exit_count, lane);
        if (lane == 0 && prev == G - 1) {
            // every CTA has left: clear the counters no warp could clear while others might poll them
            for (int q = max(0, s.nproj - 3); q < s.nproj; ++q) s.done[q] = 0u;
            *s.exit_count = 0u;
        }
    }
}

}  // namespace
}  // namespace aio
