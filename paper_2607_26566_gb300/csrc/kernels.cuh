// Device code of the paged tensor store: the batched page-table scatter
// (put), gather (get), gather with a fused fp32 -> bf16 round-to-nearest-even
// cast, and live-page moves (compaction). All four are one copy engine over
// "units": a unit is up to U = 2^unit_shift bytes of one object that lie in
// one page. A launch carries its descriptors in its own parameter space
// (up to ~31 KiB): no device scratch memory, no host->device descriptor copy.
//
// HBM-bound by construction (2 bytes of traffic per payload byte, 1.5 for the
// cast): the design goals are fully coalesced 16-byte accesses, enough bytes
// in flight per SM (4 independent 16-byte loads per thread before the first
// store, 6 resident CTAs of 256 threads per SM) and a persistent grid sized
// from the SM count and the occupancy.
#pragma once

#include <cstdint>

namespace t2i {

constexpr int kThreads = 256;     // threads per CTA
constexpr int kVecPerThread = 4;  // 16-byte vectors per thread per unit
constexpr int kMinBlocks = 6;     // resident CTAs per SM the register budget must allow
constexpr int kMinBlocksGet = 5;      // same, gather (its cast path needs a few more registers)
constexpr int kMinBlocksGeneral = 2;  // same, kernels that handle any alignment
constexpr uint32_t kUnitShiftMax = 14;  // U = 16 KiB = kThreads * kVecPerThread * 16

// One object segment of a launch. For a put/move the user address is the
// source; for a get it is the destination. Bit 63 of nbytes_flags asks for
// the fp32 -> bf16 cast (get only).
struct SegDesc {
    uint64_t user;
    uint64_t nbytes_flags;
    uint32_t unit_begin;  // first unit of this segment within the launch
    uint32_t page_begin;  // first entry of its pages in the launch's page array
};
static_assert(sizeof(SegDesc) == 24, "SegDesc layout");
constexpr uint64_t kCastFlag = uint64_t(1) << 63;

struct LaunchHeader {
    uint64_t pool;        // pool base address (device)
    uint32_t n_seg;
    uint32_t n_units;
    uint32_t page_shift;
    uint32_t unit_shift;
    uint32_t pages_offset;  // byte offset of the uint32 page array in blob
    uint32_t pad;
};
static_assert(sizeof(LaunchHeader) == 32, "LaunchHeader layout");

template <int BLOB>
struct LaunchParams {
    LaunchHeader h;
    alignas(16) unsigned char blob[BLOB];  // SegDesc[n_seg], then uint32 pages[]
};

constexpr int kBlobSmall = 1024;
constexpr int kBlobMid = 8192;
constexpr int kBlobLarge = 31 * 1024;  // header + blob stays below the 32,764-byte parameter limit

enum class Mode { Put, Get, Move };

#ifdef __CUDACC__

__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }

// ---------------------------------------------------------------- loads/stores
__device__ __forceinline__ uint4 ld_stream(const uint4* p) { return __ldcs(p); }
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) { __stcs(p, v); }

// fp32 -> bf16, round to nearest even, on bit patterns: add just under half
// an ulp of bf16, plus one when the kept part is odd, and drop 16 bits (the
// classic bias-and-truncate method); NaN becomes a quiet NaN with its sign.
__device__ __forceinline__ uint32_t bf16_rne_bits(uint32_t u) {
    const bool nan = (u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0u;
    const uint32_t r = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
    return nan ? (0x7FC0u | ((u >> 16) & 0x8000u)) : r;
}

__device__ __forceinline__ uint32_t pack_bf16x2(uint32_t a, uint32_t b) {
    return bf16_rne_bits(a) | (bf16_rne_bits(b) << 16);
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
// aligned: every page, every unit of an aligned tensor) is one round of
// kVecPerThread independent 16-byte loads, then the stores.
__device__ __forceinline__ void cta_copy_aligned(unsigned char* __restrict__ dst,
                                                 const unsigned char* __restrict__ src, uint32_t len) {
    const uint32_t nvec = len >> 4;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll 1
    for (uint32_t base = 0; base < nvec; base += kThreads * kVecPerThread) {
        uint4 r[kVecPerThread];
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) r[j] = ld_stream(s + v);
        }
#pragma unroll
        for (int j = 0; j < kVecPerThread; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) st_stream(d + v, r[j]);
        }
    }
    const uint32_t tail = len & 15u;
    if (threadIdx.x < tail) dst[(nvec << 4) + threadIdx.x] = src[(nvec << 4) + threadIdx.x];
}

// dst 16-byte aligned, src misaligned by sm (1..15): each output vector is
// cut out of the two aligned source vectors that cover it. Both aligned
// loads hold at least one byte of the source range, so no access leaves the
// source allocation.
template <int Q>
__device__ __forceinline__ void cta_copy_shifted_q(uint4* __restrict__ d, const uint4* __restrict__ a,
                                                   uint32_t nvec, uint32_t r) {
    // two aligned loads per output vector: half the vectors per round of the
    // aligned path keeps the same loads in flight within the register budget
    constexpr int kV = kVecPerThread / 2;
#pragma unroll 1
    for (uint32_t base = 0; base < nvec; base += kThreads * kV) {
        uint4 lo[kV], hi[kV];
#pragma unroll
        for (int j = 0; j < kV; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) {
                lo[j] = ld_stream(a + v);
                hi[j] = ld_stream(a + v + 1);
            }
        }
#pragma unroll
        for (int j = 0; j < kV; ++j) {
            const uint32_t v = base + j * kThreads + threadIdx.x;
            if (v < nvec) st_stream(d + v, shift_pick<Q>(lo[j], hi[j], r));
        }
    }
}

__device__ __forceinline__ void cta_copy_unaligned(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                                uint32_t len) {
    // head bytes up to dst's 16-byte boundary
    const uint32_t head = umin(len, (16u - (uint32_t)(reinterpret_cast<uintptr_t>(dst) & 15u)) & 15u);
    if (threadIdx.x < head) dst[threadIdx.x] = src[threadIdx.x];
    dst += head;
    src += head;
    len -= head;
    const uint32_t nvec = len >> 4;
    const uint32_t sm = (uint32_t)(reinterpret_cast<uintptr_t>(src) & 15u);
    if (sm == 0) {
        cta_copy_aligned(dst, src, len);
        return;
    }
    uint4* d = reinterpret_cast<uint4*>(dst);
    const uint4* a = reinterpret_cast<const uint4*>(src - sm);
    const uint32_t r = sm & 3u;
    switch (sm >> 2) {
        case 0: cta_copy_shifted_q<0>(d, a, nvec, r); break;
        case 1: cta_copy_shifted_q<1>(d, a, nvec, r); break;
        case 2: cta_copy_shifted_q<2>(d, a, nvec, r); break;
        default: cta_copy_shifted_q<3>(d, a, nvec, r); break;
    }
    const uint32_t tail = len & 15u;
    if (threadIdx.x < tail) dst[(nvec << 4) + threadIdx.x] = src[(nvec << 4) + threadIdx.x];
}

// fp32 (pool, aligned) -> bf16 (user, 16-byte aligned). len = source
// bytes, a multiple of 4: 8 floats (two 16-byte loads) -> 8 bf16 (one
// 16-byte store) per thread step, the last < 8 elements one by one.
__device__ __forceinline__ void cta_cast_aligned(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                                 uint32_t len) {
    const uint32_t nf = len >> 2;
    const uint32_t n8 = nf >> 3;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
    constexpr int kSteps = kVecPerThread / 2;
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

// Same cast into a destination that is only 2-byte aligned: one element per
// thread step.
__device__ __forceinline__ void cta_cast_scalar(unsigned char* __restrict__ dst, const unsigned char* __restrict__ src,
                                                uint32_t len) {
    const uint32_t nf = len >> 2;
    const uint32_t* s = reinterpret_cast<const uint32_t*>(src);
    uint16_t* d = reinterpret_cast<uint16_t*>(dst);
#pragma unroll 1
    for (uint32_t i = threadIdx.x; i < nf; i += kThreads) d[i] = (uint16_t)bf16_rne_bits(s[i]);
}

// Largest segment index whose first unit is <= u (segments are non-empty
// and ordered by unit_begin). All threads search the same u: uniform loads.
__device__ __forceinline__ uint32_t find_segment(const SegDesc* segs, uint32_t n, uint32_t u) {
    uint32_t lo = 0, hi = n - 1;
    while (lo < hi) {
        const uint32_t mid = (lo + hi + 1) >> 1;
        if (segs[mid].unit_begin <= u)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// The unit loop. GENERAL = false: every user address of the launch is
// 16-byte aligned (the host sorts segments into aligned and other launches),
// so only the vector paths are compiled in and the register budget stays
// small enough for kMinBlocks resident CTAs per SM. GENERAL = true adds the
// shifted copies and the element-wise cast for any alignment.
template <Mode M, bool GENERAL, int BLOB>
__device__ __forceinline__ void run_units(const LaunchParams<BLOB>& p) {
    const SegDesc* segs = reinterpret_cast<const SegDesc*>(p.blob);
    const uint32_t* pages = reinterpret_cast<const uint32_t*>(p.blob + p.h.pages_offset);
    unsigned char* pool = reinterpret_cast<unsigned char*>(p.h.pool);
    const uint32_t ushift = p.h.unit_shift;
    const uint32_t pshift = p.h.page_shift;
    const uint64_t pmask = (uint64_t(1) << pshift) - 1;
#pragma unroll 1
    for (uint32_t u = blockIdx.x; u < p.h.n_units; u += gridDim.x) {
        const uint32_t i = find_segment(segs, p.h.n_seg, u);
        const SegDesc s = segs[i];
        const uint64_t nbytes = s.nbytes_flags & ~kCastFlag;
        const uint32_t k = u - s.unit_begin;
        const uint64_t off = uint64_t(k) << ushift;
        const uint32_t len = (uint32_t)umin64(uint64_t(1) << ushift, nbytes - off);
        const uint32_t page = pages[s.page_begin + (k >> (pshift - ushift))];
        unsigned char* paddr = pool + (uint64_t(page) << pshift) + (off & pmask);
        unsigned char* uaddr = reinterpret_cast<unsigned char*>(s.user);
        if (M == Mode::Get) {
            if (s.nbytes_flags & kCastFlag) {
                if (!GENERAL || (reinterpret_cast<uintptr_t>(uaddr) & 15u) == 0)
                    cta_cast_aligned(uaddr + (off >> 1), paddr, len);
                else
                    cta_cast_scalar(uaddr + (off >> 1), paddr, len);
            } else if (!GENERAL || (reinterpret_cast<uintptr_t>(uaddr) & 15u) == 0) {
                cta_copy_aligned(uaddr + off, paddr, len);
            } else {
                cta_copy_unaligned(uaddr + off, paddr, len);
            }
        } else {
            if (!GENERAL || (reinterpret_cast<uintptr_t>(uaddr) & 15u) == 0)
                cta_copy_aligned(paddr, uaddr + off, len);
            else
                cta_copy_unaligned(paddr, uaddr + off, len);
        }
    }
}

// Named entry points (one per operation, so that profiles name them).
template <int BLOB, bool GENERAL>
__global__ void __launch_bounds__(kThreads, GENERAL ? kMinBlocksGeneral : kMinBlocks)
    scatter_put_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    run_units<Mode::Put, GENERAL, BLOB>(p);
}
template <int BLOB, bool GENERAL>
__global__ void __launch_bounds__(kThreads, GENERAL ? kMinBlocksGeneral : kMinBlocksGet)
    gather_get_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    run_units<Mode::Get, GENERAL, BLOB>(p);
}
template <int BLOB>
__global__ void __launch_bounds__(kThreads, kMinBlocks) compact_move_kernel(const __grid_constant__ LaunchParams<BLOB> p) {
    run_units<Mode::Move, false, BLOB>(p);
}

#endif  // __CUDACC__

}  // namespace t2i
