// Device code of the paged tensor store: the batched page-table scatter
// (put), gather (get), gather with a fused fp32 -> bf16 round-to-nearest-even
// cast, and live-page moves (compaction). All four are one copy engine. A
// launch carries its descriptors in its own parameter space (up to ~31 KiB):
// no host->device descriptor copy.
//
// Work split: the segments of a launch are laid end to end in a "launch byte
// space" (each starting on a 32-byte granule). SMs do not all get the same
// share of HBM bandwidth: with one equal static share per resident CTA, the
// last CTAs of a large launch finished ~1.6x later than the first on GB300.
// So a launch balances its work one of two ways:
//   - a very large launch (>= 1 MiB per resident CTA) runs a persistent grid
//     whose CTAs take 32 KiB chunks one at a time from a counter in device
//     memory (the store's work counter for the launch's stream);
//   - any other launch (work == 0) runs one CTA per 64 KiB (at least the
//     resident CTAs, each with >= 16 KiB), each with an equal contiguous
//     share, and the hardware block scheduler hands CTAs to whichever SMs
//     free up first.
// Both leave all CTAs finishing within a chunk or a share of each other. A
// CTA walks its part in pieces of at most U = 32 KiB within one segment,
// mapping each piece to its page through the segment's page list: a piece
// stays in one page, unless the segment is a run of consecutive pages (then
// only its first page is listed), and with pages smaller than U one round
// of the copy covers several pages, each vector finding its own.
//
// HBM-bound by construction (2 bytes of traffic per payload byte, 1.5 for the
// cast): fully coalesced 16-byte accesses, enough bytes in flight per SM (8
// independent 16-byte loads per thread before the first store, 3-4 resident
// CTAs of 256 threads per SM: 96-128 KiB in flight; user addresses that are
// not 16-byte aligned are realigned in shared memory, or by warp shuffles for
// the cast), grids sized from the SM count, the occupancy and the launch's
// bytes (see the work split above), and programmatic dependent launch so
// that the next launch's set-up, and an L2 prefetch of each CTA's first
// source bytes, overlap the end of this one. The launch shape and cache policy were chosen by a sweep
// on GB300 (default caching beat streaming hints by ~1.5%; 8 vectors per
// thread beat 2 and 4).
#pragma once

#include <cstdint>

namespace t2i {

// Launch shape (overridable at compile time for tuning sweeps).
#ifndef T2I_TUNE_THREADS
#define T2I_TUNE_THREADS 256
#endif
#ifndef T2I_TUNE_VEC
#define T2I_TUNE_VEC 8
#endif
#ifndef T2I_TUNE_MIN_BLOCKS
#define T2I_TUNE_MIN_BLOCKS 4
#endif
#ifndef T2I_TUNE_MIN_BLOCKS_GET
#define T2I_TUNE_MIN_BLOCKS_GET 3
#endif
#ifndef T2I_TUNE_CACHE
#define T2I_TUNE_CACHE 1  // 0: streaming (.cs) loads and stores; 1: default caching; 2: loads bypass L1
#endif
constexpr int kThreads = T2I_TUNE_THREADS;          // threads per CTA
constexpr int kVecPerThread = T2I_TUNE_VEC;         // 16-byte vectors per thread per round of a copy loop
constexpr int kMinBlocks = T2I_TUNE_MIN_BLOCKS;     // resident CTAs per SM the register budget must allow
constexpr int kMinBlocksGet = T2I_TUNE_MIN_BLOCKS_GET;  // same, gather (its cast path needs a few more registers)
#ifndef T2I_TUNE_MIN_BLOCKS_GENERAL
#define T2I_TUNE_MIN_BLOCKS_GENERAL 3
#endif
// same, the any-alignment kernels (their pieces are staged in shared memory,
// 32 KiB per CTA, so that their loads need no more registers than the
// aligned kernels'). A sweep over 1 GiB at misaligned offsets: 3 resident
// CTAs per SM beat 4 by 1-2% on copies and by 12% on the cast into 2-byte
// aligned destinations; 5 lost 5-12%.
constexpr int kMinBlocksGeneral = T2I_TUNE_MIN_BLOCKS_GENERAL;
#ifndef T2I_TUNE_MIN_BLOCKS_GENERAL_GET
#define T2I_TUNE_MIN_BLOCKS_GENERAL_GET T2I_TUNE_MIN_BLOCKS_GENERAL
#endif
// same, the any-alignment get that may cast
constexpr int kMinBlocksGeneralGet = T2I_TUNE_MIN_BLOCKS_GENERAL_GET;
constexpr uint32_t kPieceBytes = kThreads * kVecPerThread * 16;  // U = 32 KiB: one round of the copy loop
constexpr uint32_t kGranule = 32;  // segment starts and CTA shares fall on 32-byte boundaries
constexpr uint64_t kMinCtaBytes = 16 * 1024;  // smallest share worth a CTA
#ifndef T2I_TUNE_STATIC_CTA_BYTES
#define T2I_TUNE_STATIC_CTA_BYTES (64ull << 10)
#endif
// share of a CTA in a large launch without chunks (a sweep: 32, 48, 64, 96,
// 128, 256 and 512 KiB; 64 KiB was best or within noise of the best on
// every workload)
constexpr uint64_t kStaticCtaBytes = T2I_TUNE_STATIC_CTA_BYTES;
#ifndef T2I_TUNE_GET_COPY_KERNEL
#define T2I_TUNE_GET_COPY_KERNEL 1
#endif
constexpr bool kGetCopyKernel = T2I_TUNE_GET_COPY_KERNEL != 0;  // gets without casts run gather_copy_kernel
#ifndef T2I_TUNE_CAST_SHUFFLE
#define T2I_TUNE_CAST_SHUFFLE 1  // casts into unaligned destinations realign by warp shuffles (0: in shared memory)
#endif
#ifndef T2I_TUNE_CAST_SHUFFLE_STEPS
#define T2I_TUNE_CAST_SHUFFLE_STEPS 5  // blocks of 8 floats in flight per thread in that cast
#endif

// One object segment of a launch. For a put/move the user address is the
// source; for a get it is the destination. Bit 63 of nbytes_flags asks for
// the fp32 -> bf16 cast (get only).
struct SegDesc {
    uint64_t user;
    uint64_t nbytes_flags;
    uint32_t start;       // first granule of this segment in the launch byte space
    uint32_t page_begin;  // first entry of its pages in the launch's page array
};
static_assert(sizeof(SegDesc) == 24, "SegDesc layout");
constexpr uint64_t kCastFlag = uint64_t(1) << 63;
// The segment's pages are consecutive in the pool: its page list holds the
// first page only, and pieces may cross page boundaries.
constexpr uint64_t kRunFlag = uint64_t(1) << 62;
constexpr uint64_t kSegBytesMask = ~(kCastFlag | kRunFlag);

struct LaunchHeader {
    uint64_t pool;            // pool base address (device)
    uint64_t work;            // device address of the launch's WorkCounter; 0 = equal static shares
    uint32_t n_seg;
    uint32_t n_granules;      // size of the launch byte space in granules
    uint32_t page_shift;
    uint32_t piece_bytes;     // min(U, page size)
    uint32_t pages_offset;    // byte offset of the uint32 page array in blob
    uint32_t chunk_granules;  // granules a CTA takes at a time from the counter
    uint32_t flags;           // kPrefetchSources, or 0
    uint32_t prefetch_ctas;   // CTAs 0 .. prefetch_ctas-1 prefetch their shares (kPrefetchSources)
};
static_assert(sizeof(LaunchHeader) == 48, "LaunchHeader layout");
// Every source byte of the launch is device memory: a CTA with an equal
// static share may ask L2 for its source bytes before the previous grid on
// the stream has completed (prefetch_share).
constexpr uint32_t kPrefetchSources = 1u;
#ifndef T2I_TUNE_PREFETCH
#define T2I_TUNE_PREFETCH 1
#endif
constexpr bool kPrefetch = T2I_TUNE_PREFETCH != 0;

// The chunk counter of one stream of a store. Zero between launches: the
// last CTA of every launch that used it puts both fields back to zero, and
// the next launch on the same stream reads it only after that launch has
// completed (griddepcontrol.wait, or plain stream order).
struct WorkCounter {
    unsigned int next;  // chunks handed out
    unsigned int done;  // CTAs finished
    unsigned int pad[6];
};
static_assert(sizeof(WorkCounter) == 32, "WorkCounter layout");
#ifndef T2I_TUNE_CHUNK_GRANULES
#define T2I_TUNE_CHUNK_GRANULES 1024
#endif
#ifndef T2I_TUNE_DYN_MIN_CTA_BYTES
#define T2I_TUNE_DYN_MIN_CTA_BYTES (1ull << 20)
#endif
// 32 KiB chunks (a sweep: 16 and 64 KiB were slower on large launches)
constexpr uint32_t kChunkGranules = T2I_TUNE_CHUNK_GRANULES;
// Launches with fewer bytes per resident CTA than this use equal static
// shares: there the barrier each chunk costs more than the imbalance it
// removes (a sweep: a B=8 handoff request, 395 KiB per CTA, and 256-object
// adapter gets lost up to 5% with chunks; 0.7-3 GiB launches gained 6-12%).
constexpr uint64_t kDynMinCtaBytes = T2I_TUNE_DYN_MIN_CTA_BYTES;

template <int BLOB>
struct LaunchParams {
    LaunchHeader h;
    alignas(16) unsigned char blob[BLOB];  // SegDesc[n_seg], then uint32 pages[]
};

// Parameter-space tiers: a launch copies only its tier's bytes of
// parameters, and smaller parameters launch faster (a 256-byte tier for a
// B=1 handoff request, 124 bytes of descriptors, ran the 4-stream B=1 step
// 4% faster than the 1 KiB tier).
constexpr int kBlobTiny = 256;
// Largest segment (bytes) of one launch: 2^31 granules, so that granule
// offsets of a launch (32-bit) never wrap.
constexpr uint64_t kMaxSegBytes = uint64_t(1) << 36;
constexpr int kBlobSmall = 1024;
constexpr int kBlobMid = 8192;
constexpr int kBlobLarge = 31 * 1024;  // header + blob stays below the 32,764-byte parameter limit

// GetCopy: a get whose launch has no cast segment (a leaner kernel).
enum class Mode { Put, Get, Move, GetCopy };

#ifdef __CUDACC__

__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }

// ---------------------------------------------------------------- loads/stores
#if T2I_TUNE_CACHE == 0
__device__ __forceinline__ uint4 ld_stream(const uint4* p) { return __ldcs(p); }
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) { __stcs(p, v); }
#elif T2I_TUNE_CACHE == 1
__device__ __forceinline__ uint4 ld_stream(const uint4* p) { return *p; }
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) { *p = v; }
#else
__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) { __stcs(p, v); }
#endif

// fp32 -> bf16, round to nearest even, on bit patterns: add just under half
// an ulp of bf16, plus one when the kept part is odd, and drop 16 bits (the
// classic bias-and-truncate method); NaN (exponent all ones, mantissa not
// zero) becomes a quiet NaN with its sign.
__device__ __forceinline__ uint32_t bf16_rne_bits(uint32_t u) {
    const bool nan = (u & 0x7FFFFFFFu) > 0x7F800000u;
    const uint32_t r = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
    return nan ? (0x7FC0u | ((u >> 16) & 0x8000u)) : r;
}

// Two of them packed (a in the low half). By default the hardware's
// round-to-nearest-even conversion (cvt.rn.bf16x2.f32, which keeps
// subnormals and rounds overflow to infinity like the bit arithmetic above),
// with NaN results replaced by the quiet NaN with the input's sign; a sweep
// on GB300 over 1 GiB of fp32: casts into 2-byte-aligned destinations 5.83 ->
// 6.50 TB/s (the shuffle cast was bound by its arithmetic), into aligned ones
// 6.45 -> 6.67; handoff gets unchanged. T2I_TUNE_CVT=0 packs two
// bf16_rne_bits instead. Both are compared with the oracle over all 2^32
// inputs by the GPU tests.
#ifndef T2I_TUNE_CVT
#define T2I_TUNE_CVT 1
#endif
__device__ __forceinline__ uint32_t pack_bf16x2(uint32_t a, uint32_t b) {
#if T2I_TUNE_CVT
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(__uint_as_float(b)), "f"(__uint_as_float(a)));
    if ((a & 0x7FFFFFFFu) > 0x7F800000u) r = (r & 0xFFFF0000u) | 0x7FC0u | ((a >> 16) & 0x8000u);
    if ((b & 0x7FFFFFFFu) > 0x7F800000u) r = (r & 0x0000FFFFu) | ((0x7FC0u | ((b >> 16) & 0x8000u)) << 16);
    return r;
#else
    return bf16_rne_bits(a) | (bf16_rne_bits(b) << 16);
#endif
}

// Bytes [sm, sm + 16) of the 32-byte little-endian concatenation lo|hi,
// sm = 4 * Q + r with r in 0..3.
template <int Q>
__device__ __forceinline__ uint4 shift_pick(uint4 lo, uint4 hi, uint32_t r) {
    const uint32_t s = 8u * r;
    const uint32_t w0 = Q == 0 ? lo.x : Q == 1 ? lo.y : Q == 2 ? lo.z : lo.w;
    const uint32_t w1 = Q == 0 ? lo.y : Q == 1 ? lo.z : Q == 2 ? lo.w : hi.x;
    const uint32_t w2 = Q == 0 ? lo.z : Q == 1 ? lo.w : Q == 2 ? hi.x : hi.y;
    const uint32_t w3 = Q == 0 ? lo.w : Q == 1 ? hi.x : Q == 2 ? hi.y : hi.z;
    const uint32_t w4 = Q == 0 ? hi.x : Q == 1 ? hi.y : Q == 2 ? hi.z : hi.w;
    uint4 o;
    o.x = __funnelshift_r(w0, w1, s);
    o.y = __funnelshift_r(w1, w2, s);
    o.z = __funnelshift_r(w2, w3, s);
    o.w = __funnelshift_r(w3, w4, s);
    return o;
}

// CTA-wide copy of len <= U bytes. The aligned case (both sides 16-byte
// aligned: every page, every piece of an aligned tensor) is one round of
// kVecPerThread independent 16-byte loads, then the stores.
template <int V = kVecPerThread>
__device__ __forceinline__ void cta_copy_aligned(unsigned char* __restrict__ dst,
                                                 const unsigned char* __restrict__ src, uint32_t len) {
    const uint32_t nvec = len >> 4;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll 1
    for (uint32_t base = 0; base < nvec; base += kThreads * V) {
        uint4 r[V];
#pragma unroll
        for (int j = 0; j < V; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) r[j] = ld_stream(s + v);
        }
#pragma unroll
        for (int j = 0; j < V; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) st_stream(d + v, r[j]);
        }
    }
    const uint32_t tail = len & 15u;
    if (threadIdx.x < tail) dst[(nvec << 4) + threadIdx.x] = src[(nvec << 4) + threadIdx.x];
}

// CTA-wide copy of one full round (kThreads x V 16-byte vectors, contiguous
// in a segment's bytes from off) when pages are smaller than a round: each
// vector looks up its own page (a warp's 512 bytes lie in one or two pages,
// so the page list is read as a broadcast). Both sides 16-byte aligned. Not
// inlined: its addresses would otherwise take registers from the large-page
// path of every kernel.
template <Mode M, int V>
__device__ __noinline__ void cta_copy_pages(unsigned char* __restrict__ user, unsigned char* __restrict__ pool,
                                               const uint32_t* __restrict__ pages, uint64_t off, uint32_t pshift) {
    constexpr bool kToUser = M == Mode::Get || M == Mode::GetCopy;
    const uint64_t pmask = (uint64_t(1) << pshift) - 1;
    uint4 r[V];
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const uint64_t o = off + (uint64_t(j * kThreads + threadIdx.x) << 4);
        const unsigned char* src =
            kToUser ? pool + (uint64_t(pages[o >> pshift]) << pshift) + (o & pmask) : user + o;
        r[j] = ld_stream(reinterpret_cast<const uint4*>(src));
    }
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const uint64_t o = off + (uint64_t(j * kThreads + threadIdx.x) << 4);
        unsigned char* dst = kToUser ? user + o : pool + (uint64_t(pages[o >> pshift]) << pshift) + (o & pmask);
        st_stream(reinterpret_cast<uint4*>(dst), r[j]);
    }
}

// fp32 (pool, aligned) -> bf16 (user, 16-byte aligned). len = source
// bytes, a multiple of 4: 8 floats (two 16-byte loads) -> 8 bf16 (one
// 16-byte store) per thread step, the last < 8 elements one by one.
template <int V = kVecPerThread>
__device__ __forceinline__ void cta_cast_aligned(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                                 uint32_t len) {
    const uint32_t nf = len >> 2;
    const uint32_t n8 = nf >> 3;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
    constexpr int kSteps = V / 2;
#pragma unroll 1
    for (uint32_t base = 0; base < n8; base += kThreads * kSteps) {
        uint4 a[kSteps], b[kSteps];
#pragma unroll
        for (int j = 0; j < kSteps; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < n8) {
                a[j] = ld_stream(s + 2 * v);
                b[j] = ld_stream(s + 2 * v + 1);
            }
        }
#pragma unroll
        for (int j = 0; j < kSteps; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < n8) {
                uint4 o;
                o.x = pack_bf16x2(a[j].x, a[j].y);
                o.y = pack_bf16x2(a[j].z, a[j].w);
                o.z = pack_bf16x2(b[j].x, b[j].y);
                o.w = pack_bf16x2(b[j].z, b[j].w);
                st_stream(d + v, o);
            }
        }
    }
    const uint32_t done = n8 << 3;
    if (threadIdx.x < nf - done) {
        const uint32_t u = reinterpret_cast<const uint32_t*>(src)[done + threadIdx.x];
        reinterpret_cast<uint16_t*>(dst)[done + threadIdx.x] = (uint16_t)bf16_rne_bits(u);
    }
}

// ------------------------------------------------ any alignment: staged copies
// The any-alignment kernels stage each piece in shared memory: the aligned
// 16-byte window that covers the piece's source bytes is loaded with
// independent aligned 16-byte loads (kVecPerThread per thread, all issued
// before the first is used), then every aligned 16-byte output vector is
// cut out of the staged window (two staged vectors and funnel shifts), so
// every global access is one aligned 16-byte vector and the loads in flight
// per SM are those of the aligned kernels. Each aligned load holds at least
// one byte of the source range, so no access leaves the source allocation.
// A piece is at most U bytes, so its window (up to 15 bytes of misalignment
// in front) is at most U/16 + 1 vectors: one round of kVecPerThread loads
// per thread, plus one more vector.
constexpr uint32_t kStageVecs = kPieceBytes / 16 + 1;
static_assert(kThreads * kVecPerThread * 16 == kPieceBytes, "one round of loads per piece");
// The stage of a CTA of the any-alignment kernels (only they reference it).
__shared__ uint4 g_stage[kStageVecs];

// Loads the nw <= kStageVecs aligned vectors at a into stage, then a CTA
// barrier (every thread sees the whole window).
__device__ __forceinline__ void stage_window(uint4* __restrict__ stage, const uint4* __restrict__ a, uint32_t nw) {
    constexpr uint32_t kRound = kThreads * kVecPerThread;
    uint4 r[kVecPerThread];
#pragma unroll
    for (int j = 0; j < kVecPerThread; ++j) {
        const uint32_t v = j * kThreads + threadIdx.x;
        if (v < nw) r[j] = ld_stream(a + v);
    }
    const bool extra = kRound + threadIdx.x < nw;  // the window's last vector, past one round
    uint4 x;
    if (extra) x = ld_stream(a + kRound + threadIdx.x);
#pragma unroll
    for (int j = 0; j < kVecPerThread; ++j) {
        const uint32_t v = j * kThreads + threadIdx.x;
        if (v < nw) stage[v] = r[j];
    }
    if (extra) stage[kRound + threadIdx.x] = x;
    __syncthreads();
}

// Output vectors d[v] = bytes [16 v + 4 Q + r, ... + 16) of the staged
// window w (r in 0..3; Q = r = 0 is a plain copy).
template <int Q>
__device__ __forceinline__ void emit_shifted(uint4* __restrict__ d, const uint4* __restrict__ w, uint32_t nvec,
                                             uint32_t r) {
#pragma unroll 4
    for (uint32_t v = threadIdx.x; v < nvec; v += kThreads) {
        if (Q == 0 && r == 0)
            st_stream(d + v, w[v]);
        else
            st_stream(d + v, shift_pick<Q>(w[v], w[v + 1], r));
    }
}

// CTA-wide copy of len <= U bytes, any alignment on either
// side: stage the source window, then the destination's head bytes (up to
// its 16-byte boundary) one per thread, its aligned vectors, and the tail
// bytes one per thread.
__device__ __noinline__ void cta_copy_staged(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                             uint32_t len) {
    uint4* stage = g_stage;
    const uint32_t s0 = (uint32_t)(reinterpret_cast<uintptr_t>(src) & 15u);
    stage_window(stage, reinterpret_cast<const uint4*>(src - s0), (s0 + len + 15) >> 4);
    const unsigned char* wb = reinterpret_cast<const unsigned char*>(stage);
    const uint32_t head = umin(len, (16u - (uint32_t)(reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u);
    if (threadIdx.x < head) dst[threadIdx.x] = wb[s0 + threadIdx.x];
    const uint32_t s = s0 + head;  // window offset of the first aligned output vector (< 32)
    const uint32_t nvec = (len - head) >> 4;
    uint4* d = reinterpret_cast<uint4*>(dst + head);
    const uint4* w = stage + (s >> 4);
    const uint32_t r = s & 3u;
    switch ((s >> 2) & 3u) {
        case 0: emit_shifted<0>(d, w, nvec, r); break;
        case 1: emit_shifted<1>(d, w, nvec, r); break;
        case 2: emit_shifted<2>(d, w, nvec, r); break;
        default: emit_shifted<3>(d, w, nvec, r); break;
    }
    const uint32_t done = head + (nvec << 4);
    if (threadIdx.x < len - done) dst[done + threadIdx.x] = wb[s0 + done + threadIdx.x];
    __syncthreads();  // the stage is free for the next piece
}

// Blocks of 8 staged floats starting Q (0..3) words past the staged vectors
// a[2v]: each is cut out of a[2v], a[2v+1] and (Q > 0) a[2v+2], cast, and
// stored as one 16-byte vector d[v].
template <int Q>
__device__ __forceinline__ void emit_cast_blocks(uint4* __restrict__ d, const uint4* __restrict__ a, uint32_t n8) {
#pragma unroll 1
    for (uint32_t v = threadIdx.x; v < n8; v += kThreads) {
        const uint4 x = a[2 * v], y = a[2 * v + 1];
        const uint4 z = Q > 0 ? a[2 * v + 2] : make_uint4(0u, 0u, 0u, 0u);
        const uint32_t w[12] = {x.x, x.y, x.z, x.w, y.x, y.y, y.z, y.w, z.x, z.y, z.z, z.w};
        uint4 o;
        o.x = pack_bf16x2(w[Q + 0], w[Q + 1]);
        o.y = pack_bf16x2(w[Q + 2], w[Q + 3]);
        o.z = pack_bf16x2(w[Q + 4], w[Q + 5]);
        o.w = pack_bf16x2(w[Q + 6], w[Q + 7]);
        st_stream(d + v, o);
    }
}

// fp32 (pool, 16-byte aligned) -> bf16 into a destination that is 2-byte
// aligned, len <= U source bytes (a multiple of 4): stage
// the source, then the first h < 8 elements one per thread (they bring the
// destination to a 16-byte boundary), blocks of 8 as 16-byte stores, and
// the last < 8 elements one per thread.
__device__ __noinline__ void cta_cast_staged(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                             uint32_t len) {
    uint4* stage = g_stage;
    stage_window(stage, reinterpret_cast<const uint4*>(src), (len + 15) >> 4);
    const uint32_t* ws = reinterpret_cast<const uint32_t*>(stage);
    const uint32_t nf = len >> 2;
    uint16_t* d16 = reinterpret_cast<uint16_t*>(dst);
    const uint32_t h = umin(((16u - (uint32_t)(reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u) >> 1, nf);
    if (threadIdx.x < h) d16[threadIdx.x] = (uint16_t)bf16_rne_bits(ws[threadIdx.x]);
    const uint32_t n8 = (nf - h) >> 3;
    uint4* d = reinterpret_cast<uint4*>(dst + 2 * h);
    const uint4* a = stage + (h >> 2);
    switch (h & 3u) {
        case 0: emit_cast_blocks<0>(d, a, n8); break;
        case 1: emit_cast_blocks<1>(d, a, n8); break;
        case 2: emit_cast_blocks<2>(d, a, n8); break;
        default: emit_cast_blocks<3>(d, a, n8); break;
    }
    const uint32_t done = h + (n8 << 3);
    if (threadIdx.x < nf - done) d16[done + threadIdx.x] = (uint16_t)bf16_rne_bits(ws[done + threadIdx.x]);
    __syncthreads();  // the stage is free for the next piece
}

// fp32 (pool, 16-byte aligned) -> bf16 into a destination 2, 4, ..., 14
// bytes past a 16-byte boundary, len <= U source bytes (a multiple of 4),
// without shared memory. With h (1..7) elements before the destination's
// first 16-byte boundary, aligned output vector k holds elements
// [h + 8k, h + 8k + 8): the last 8 - h elements of source block k (floats
// 8k .. 8k + 7) and the first h of block k + 1. Lane l of a warp loads and
// casts block 31q + l, takes block 31q + l + 1 from lane l + 1 by a
// shuffle, and lanes 0..30 store output vector 31q + l (the 32nd block is
// loaded again by the next step: 1/31 more L2 reads, no more DRAM traffic).
// The thread of block 0 also stores the h head elements, and the thread of
// vector n8 (one past the last whole vector) the last < 8 elements, so
// every load of a piece is issued before its first store. S steps of loads
// per thread cover a whole piece in one round (8 warps x S x 31 vectors).
// Source vectors past the piece's bytes are not read (each loaded vector
// holds a source byte; a partial last vector lies in the same page).
template <int Q, int S>
__device__ __forceinline__ void emit_cast_shuffled(unsigned char* __restrict__ dst, const uint4* __restrict__ s,
                                                   uint32_t h, uint32_t n8, uint32_t tail, uint32_t nvs,
                                                   uint32_t r) {
    constexpr uint32_t kWarps = kThreads / 32;
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    uint16_t* d16 = reinterpret_cast<uint16_t*>(dst);
    uint4* d = reinterpret_cast<uint4*>(dst + 2 * h);
#pragma unroll 1
    for (uint32_t q0 = 0; q0 * 31u <= n8; q0 += kWarps * S) {
        uint4 a[S], b[S];
#pragma unroll
        for (int j = 0; j < S; ++j) {
            const uint32_t blk = (q0 + warp * S + j) * 31u + lane;
            a[j] = 2 * blk < nvs ? ld_stream(s + 2 * blk) : make_uint4(0u, 0u, 0u, 0u);
            b[j] = 2 * blk + 1 < nvs ? ld_stream(s + 2 * blk + 1) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int j = 0; j < S; ++j) {
            const uint32_t blk = (q0 + warp * S + j) * 31u + lane;
            uint4 o;
            o.x = pack_bf16x2(a[j].x, a[j].y);
            o.y = pack_bf16x2(a[j].z, a[j].w);
            o.z = pack_bf16x2(b[j].x, b[j].y);
            o.w = pack_bf16x2(b[j].z, b[j].w);
            uint4 nx;
            nx.x = __shfl_down_sync(0xFFFFFFFFu, o.x, 1);
            nx.y = __shfl_down_sync(0xFFFFFFFFu, o.y, 1);
            nx.z = __shfl_down_sync(0xFFFFFFFFu, o.z, 1);
            nx.w = __shfl_down_sync(0xFFFFFFFFu, o.w, 1);
            if (lane < 31u) {
                if (blk < n8) {
                    st_stream(d + blk, shift_pick<Q>(o, nx, r));
                } else if (blk == n8 && tail) {
                    const uint4 v = shift_pick<Q>(o, nx, r);
                    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
                    uint16_t* t = reinterpret_cast<uint16_t*>(d + blk);
#pragma unroll
                    for (uint32_t e = 0; e < 7; ++e)
                        if (e < tail) t[e] = (uint16_t)(w[e >> 1] >> (16 * (e & 1)));
                }
            }
            if (blk == 0) {
                const uint32_t w[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
                for (uint32_t e = 0; e < 7; ++e)
                    if (e < h) d16[e] = (uint16_t)(w[e >> 1] >> (16 * (e & 1)));
            }
        }
    }
}

__device__ __noinline__ void cta_cast_shuffled(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                               uint32_t len) {
    constexpr int S = T2I_TUNE_CAST_SHUFFLE_STEPS;
    static_assert((kThreads / 32) * S * 31 >= kPieceBytes / 32 + 1, "one round covers a piece");
    const uint32_t nf = len >> 2;
    const uint32_t h = umin(((16u - (uint32_t)(reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u) >> 1, nf);
    const uint32_t n8 = (nf - h) >> 3;
    const uint32_t tail = nf - h - (n8 << 3);
    const uint32_t nvs = (len + 15) >> 4;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    // output halfword e of vector k is halfword h + e of blocks k, k + 1:
    // a shift of 2h bytes = 4Q + r bytes
    const uint32_t r = (h & 1u) * 2u;
    switch (h >> 1) {
        case 0: emit_cast_shuffled<0, S>(dst, s, h, n8, tail, nvs, r); break;
        case 1: emit_cast_shuffled<1, S>(dst, s, h, n8, tail, nvs, r); break;
        case 2: emit_cast_shuffled<2, S>(dst, s, h, n8, tail, nvs, r); break;
        default: emit_cast_shuffled<3, S>(dst, s, h, n8, tail, nvs, r); break;
    }
}

// Largest segment index whose first granule is <= g (segments are non-empty
// and ordered by start). All threads search the same g: uniform loads.
__device__ __forceinline__ uint32_t find_segment(const SegDesc* segs, uint32_t n, uint32_t g) {
    uint32_t lo = 0, hi = n - 1;
    while (lo < hi) {
        const uint32_t mid = (lo + hi + 1) >> 1;
        if (segs[mid].start <= g)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// Asks L2 for the first source bytes of this CTA's equal static share (the
// first contiguous source range, at most kPrefetchMax bytes), one 128-byte
// line per thread, before the CTA waits for the previous grid on the stream.
// A CTA of the next launch becomes resident as soon as a CTA of the draining
// one exits, so its first HBM reads overlap that drain instead of following
// it. A prefetch is only a cache hint: it changes no value that a load
// returns (L2 serves every SM's loads), so a source that the previous grid
// is still writing is read correctly after the wait. Sources are device
// memory (the host sets kPrefetchSources only then), and every line holds a
// source byte, so no prefetch leaves the source allocation.
// A sweep on GB300 (handoff B=8 request per launch; 256-object adapter
// gets): one round (32 KiB) by every CTA lifted one-stream puts by 2.8%,
// one-stream gets by 3.5% and adapter gets by 2.1%, and left the 4-stream
// handoff unchanged (+0.1%); the whole 64 KiB share cost the 4-stream put
// 2.2% and adapter gets 2%, and prefetching in the first wave of CTAs only
// gained less. A single bulk prefetch (cp.async.bulk.prefetch) per range
// cost the copy loop ~200 bytes of register spills, so the lines are
// prefetched one per thread.
#ifndef T2I_TUNE_PREFETCH_BYTES
#define T2I_TUNE_PREFETCH_BYTES (32 * 1024)
#endif
#ifndef T2I_TUNE_PREFETCH_WAVE
#define T2I_TUNE_PREFETCH_WAVE 0
#endif
constexpr uint64_t kPrefetchMax = T2I_TUNE_PREFETCH_BYTES;
// 1: only the first wave of CTAs (those resident at launch) prefetches
constexpr bool kPrefetchFirstWave = T2I_TUNE_PREFETCH_WAVE != 0;

template <Mode M, int BLOB>
__device__ __forceinline__ void prefetch_share(const LaunchParams<BLOB>& p) {
    if (!kPrefetch || p.h.work != 0 || !(p.h.flags & kPrefetchSources) || blockIdx.x >= p.h.prefetch_ctas) return;
    constexpr bool kFromPool = M == Mode::Get || M == Mode::GetCopy;  // else the user address is the source
    const SegDesc* segs = reinterpret_cast<const SegDesc*>(p.blob);
    const uint32_t* pages = reinterpret_cast<const uint32_t*>(p.blob + p.h.pages_offset);
    const uint32_t pshift = p.h.page_shift;
    const uint64_t pmask = (uint64_t(1) << pshift) - 1;
    const uint64_t g0 = uint64_t(p.h.n_granules) * blockIdx.x / gridDim.x;
    const uint64_t g1 = uint64_t(p.h.n_granules) * (blockIdx.x + 1) / gridDim.x;
    const SegDesc s = segs[find_segment(segs, p.h.n_seg, uint32_t(g0))];
    const uint64_t off = g0 * kGranule - uint64_t(s.start) * kGranule;
    const uint64_t nbytes = s.nbytes_flags & kSegBytesMask;
    if (g0 == g1 || off >= nbytes) return;
    uint64_t len = umin64(umin64((g1 - g0) * kGranule, nbytes - off), kPrefetchMax);
    uint64_t a;
    if (!kFromPool) {
        a = s.user + off;
    } else if (s.nbytes_flags & kRunFlag) {
        a = p.h.pool + (uint64_t(pages[s.page_begin]) << pshift) + off;
    } else {
        len = umin64(len, pmask + 1 - (off & pmask));
        a = p.h.pool + (uint64_t(pages[s.page_begin + (off >> pshift)]) << pshift) + (off & pmask);
    }
    // lines [a & ~127, a + len): each holds at least one source byte
    const uint64_t first = a & ~uint64_t(127);
    const uint32_t n_lines = uint32_t((a + len - first + 127) >> 7);
#pragma unroll 1
    for (uint32_t k = threadIdx.x; k < n_lines; k += kThreads)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(first + (uint64_t(k) << 7)));
}

// Programmatic dependent launch: wait until the previous grid in the stream
// has completed and its memory is visible (returns at once when this launch
// has no such dependency), then let the next launch begin its set-up.
__device__ __forceinline__ void pdl_wait_then_release() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The piece loop. GENERAL = false: every user address of the launch is
// 16-byte aligned (the host sorts segments into aligned and other launches),
// so the pieces are plain vector copies. GENERAL = true: user addresses of
// any alignment; every piece is staged in shared memory and realigned there.
template <Mode M, bool GENERAL, int BLOB>
__device__ __forceinline__ void run_range(const LaunchParams<BLOB>& p, uint64_t g0, uint64_t g1);

// This CTA's part of the launch: chunks from the counter, or an equal share.
template <Mode M, bool GENERAL, int BLOB>
__device__ __forceinline__ void run_share(const LaunchParams<BLOB>& p) {
    if (p.h.work == 0) {
        const uint64_t g0 = uint64_t(p.h.n_granules) * blockIdx.x / gridDim.x;
        const uint64_t g1 = uint64_t(p.h.n_granules) * (blockIdx.x + 1) / gridDim.x;
        run_range<M, GENERAL, BLOB>(p, g0, g1);
        return;
    }
    // (the counter's address and the sizes are re-read from the parameters
    // where needed: they take no registers across the copy)
    // Two ticket slots: the ticket for chunk k+1 is written into the slot
    // not read in round k, so one barrier per chunk suffices.
    __shared__ uint32_t s_next[2];
    if (threadIdx.x == 0) s_next[0] = atomicAdd(&reinterpret_cast<WorkCounter*>(p.h.work)->next, 1u);
    __syncthreads();
    uint32_t c = s_next[0];
    uint32_t k = 0;
#pragma unroll 1
    while (uint64_t(c) * p.h.chunk_granules < p.h.n_granules) {
        // the next chunk is fetched while this one is copied
        uint32_t t = 0;
        if (threadIdx.x == 0) t = atomicAdd(&reinterpret_cast<WorkCounter*>(p.h.work)->next, 1u);
        const uint64_t g0 = uint64_t(c) * p.h.chunk_granules;
        run_range<M, GENERAL, BLOB>(p, g0, umin64(g0 + p.h.chunk_granules, p.h.n_granules));
        k ^= 1u;
        if (threadIdx.x == 0) s_next[k] = t;
        __syncthreads();
        c = s_next[k];
    }
    // the last CTA out leaves the counter at zero for the next launch
    if (threadIdx.x == 0) {
        WorkCounter* wc = reinterpret_cast<WorkCounter*>(p.h.work);
        __threadfence();
        if (atomicAdd(&wc->done, 1u) == gridDim.x - 1) {
            wc->next = 0;
            wc->done = 0;
            __threadfence();
        }
    }
}

// Copies granules [g0, g1) of the launch byte space.
template <Mode M, bool GENERAL, int BLOB>
__device__ __forceinline__ void run_range(const LaunchParams<BLOB>& p, uint64_t g0, uint64_t g1) {
    constexpr int kV = kVecPerThread;
    const SegDesc* segs = reinterpret_cast<const SegDesc*>(p.blob);
    const uint32_t* pages = reinterpret_cast<const uint32_t*>(p.blob + p.h.pages_offset);
    unsigned char* pool = reinterpret_cast<unsigned char*>(p.h.pool);
    const uint32_t pshift = p.h.page_shift;
    const uint64_t pmask = (uint64_t(1) << pshift) - 1;
    const uint64_t piece = p.h.piece_bytes;
    if (g0 == g1) return;
    uint64_t pos = g0 * kGranule;
    const uint64_t end = g1 * kGranule;
    uint32_t i = find_segment(segs, p.h.n_seg, uint32_t(g0));
    // the current segment and page stay in registers until the walk leaves them
    SegDesc s = segs[i];
    uint64_t lo = uint64_t(s.start) * kGranule;
    uint64_t nbytes = s.nbytes_flags & kSegBytesMask;
    uint64_t page_idx = ~uint64_t(0);
    unsigned char* page_base = nullptr;
#pragma unroll 1
    while (pos < end) {
        if (pos >= lo + nbytes) {  // past this segment (its padding): next one
            if (++i >= p.h.n_seg) break;
            s = segs[i];
            lo = uint64_t(s.start) * kGranule;  // segments are ordered: this is >= pos
            nbytes = s.nbytes_flags & kSegBytesMask;
            page_idx = ~uint64_t(0);
            pos = lo;
            continue;
        }
        const uint64_t off = pos - lo;  // a multiple of kGranule
        // pages smaller than a round: a full round spans several pages of
        // this segment, each vector finding its own page, instead of
        // stopping at every page end (+2% on a handoff in 16 and 64 KiB pages)
        constexpr uint64_t kRound = uint64_t(kThreads) * kV * 16;
        if (!GENERAL && pmask + 1 < kRound && off + kRound <= nbytes && pos + kRound <= end &&
            !(s.nbytes_flags & (kCastFlag | kRunFlag))) {
            cta_copy_pages<M, kV>(reinterpret_cast<unsigned char*>(s.user), pool, pages + s.page_begin, off, pshift);
            pos += kRound;
            continue;
        }
        uint32_t len;
        unsigned char* paddr;
        if (s.nbytes_flags & kRunFlag) {
            // consecutive pages: one contiguous stretch of the pool
            paddr = pool + (uint64_t(pages[s.page_begin]) << pshift) + off;
            len = (uint32_t)umin64(umin64(end - pos, nbytes - off), kPieceBytes);
        } else {
            const uint64_t in_page = off & pmask;
            if ((off >> pshift) != page_idx) {
                page_idx = off >> pshift;
                page_base = pool + (uint64_t(pages[s.page_begin + page_idx]) << pshift);
            }
            len = (uint32_t)umin64(umin64(end - pos, nbytes - off), umin64(piece, pmask + 1 - in_page));
            paddr = page_base + in_page;
        }
        unsigned char* uaddr = reinterpret_cast<unsigned char*>(s.user);
        if (M == Mode::Get || M == Mode::GetCopy) {
            if (M == Mode::Get && (s.nbytes_flags & kCastFlag)) {
                if (GENERAL && T2I_TUNE_CAST_SHUFFLE)
                    cta_cast_shuffled(uaddr + (off >> 1), paddr, len);
                else if (GENERAL)
                    cta_cast_staged(uaddr + (off >> 1), paddr, len);
                else
                    cta_cast_aligned<kV>(uaddr + (off >> 1), paddr, len);
            } else if (GENERAL) {
                cta_copy_staged(uaddr + off, paddr, len);
            } else {
                cta_copy_aligned<kV>(uaddr + off, paddr, len);
            }
        } else {
            if (GENERAL)
                cta_copy_staged(paddr, uaddr + off, len);
            else
                cta_copy_aligned<kV>(paddr, uaddr + off, len);
        }
        pos += len;
    }
}

// Named entry points (one per operation, so that profiles name them).
template <int BLOB, bool GENERAL>
__global__ void __launch_bounds__(kThreads, GENERAL ? kMinBlocksGeneral : kMinBlocks)
    scatter_put_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    prefetch_share<Mode::Put, BLOB>(p);
    pdl_wait_then_release();
    run_share<Mode::Put, GENERAL, BLOB>(p);
}
template <int BLOB, bool GENERAL>
__global__ void __launch_bounds__(kThreads, GENERAL ? kMinBlocksGeneralGet : kMinBlocksGet)
    gather_get_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    prefetch_share<Mode::Get, BLOB>(p);
    pdl_wait_then_release();
    run_share<Mode::Get, GENERAL, BLOB>(p);
}
// A get launch without casts: the copy path alone fits the register budget
// of kMinBlocks resident CTAs, like the put (the cast's registers left out).
template <int BLOB, bool GENERAL>
__global__ void __launch_bounds__(kThreads, GENERAL ? kMinBlocksGeneral : kMinBlocks)
    gather_copy_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    prefetch_share<Mode::GetCopy, BLOB>(p);
    pdl_wait_then_release();
    run_share<Mode::GetCopy, GENERAL, BLOB>(p);
}
template <int BLOB>
__global__ void __launch_bounds__(kThreads, kMinBlocks) compact_move_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    prefetch_share<Mode::Move, BLOB>(p);
    pdl_wait_then_release();
    run_share<Mode::Move, false, BLOB>(p);
}

#endif  // __CUDACC__

}  // namespace t2i
