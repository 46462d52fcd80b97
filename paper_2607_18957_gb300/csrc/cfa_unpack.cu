/*
 * Unpack kernels: the "InGPU -> Loaded" transition of InstantInfer section 4.2 (dependency (ii):
 * once a chunk is in GPU memory, its bytes are copied and assembled into every tensor it
 * carries).  One launch handles every work item of one chunk, or of a run of chunks that sit
 * contiguously in device memory.
 *
 * The work is pure data movement plus integer arithmetic, so it is bound by HBM bandwidth:
 * every source byte is read once from the staging buffer and every destination byte written
 * once.  Design points:
 *   - block-per-slab: a slab (tens of KiB of one piece) is copied by a whole CTA with 16-byte
 *     vector loads and stores, several in flight per thread;
 *   - warp-per-descriptor: pieces below the tiny threshold are handled by one warp each, eight
 *     per CTA, so the ~200k small tensors of an MoE checkpoint do not each pay for a CTA;
 *   - a persistent grid (a few CTAs per SM) walks the work list, so the launch cost does not
 *     grow with the number of work items;
 *   - source and destination offsets that differ modulo 16 are realigned in registers (two
 *     aligned loads and a funnel shift per 16-byte store), so stores stay 16 bytes wide;
 *   - dtype conversions (fp32 -> bf16 / fp16, fp16 -> bf16 with round-to-nearest-even;
 *     bf16 / fp16 -> fp32 exactly) work on bit patterns with integer operations;
 *   - checksums are sums modulo 2^64 of the destination element bit patterns, reduced inside the
 *     CTA or warp and added with one 64-bit atomic per (CTA, run of same-tensor slabs) or per
 *     tiny piece; integer addition is associative, so the result does not depend on the order.
 */
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "cfa_device.cuh"
#include "cfa_internal.h"

namespace {

using cfa_dev::vsum;
using cfa_dev::warp_sum;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;
constexpr int kMinBlocks = 4;     /* conversion classes: 64 registers per thread at most */
constexpr int kCopyMinBlocks = 3; /* 2-8-byte copy classes: 80 registers, room for the
                                     realigning path; the 1-byte class keeps 4 CTAs (its byte-wise
                                     checksum wants the warps: 0.96 vs 0.92 of the roofline) */
/* Rounds of 32-vector loads in flight per warp on the realigning path: four for slabs (with
 * three CTAs per SM the copy kernels hold them without spilling; two for the 1-byte class at
 * four CTAs), two for column-slice rows. */
constexpr int kRealignRounds = 4;

constexpr int kRealignRoundsRows = 2;

struct UnpackArgs {
    const cfa_work *slabs;
    const cfa_work *tiny;
    uint32_t n_slabs;
    uint32_t n_tiny;
    uint64_t src_base;   /* device address of blob byte 0 for this launch */
    uint64_t src_period; /* 0, or P: blob byte o sits at src_base + (o mod P) */
    uint64_t src_lo;     /* blob bytes [src_lo, src_hi) are readable in this launch */
    uint64_t src_hi;
    unsigned long long *ck;
    int *status;
    uint32_t dev_src;    /* 1: the source is device memory (staging slots or a device blob) */
};

/* ---- memory operations ------------------------------------------------------------------ */

/* Streaming 16-byte load of staging data: read once, never by L1. */
__device__ __forceinline__ uint4 ld_stream(const void *p)
{
    uint4 v;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
        : "l"(p));
    return v;
}

/* 16-byte load that may be shared with the neighbouring thread (realignment path). */
__device__ __forceinline__ uint4 ld_shared_line(const void *p)
{
    uint4 v;
    asm("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
        : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
        : "l"(p));
    return v;
}

/* Streaming 16-byte store: written once, not read again by this kernel. */
__device__ __forceinline__ void st_stream(void *p, uint4 v)
{
    asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
}

template <int ES> struct Elem;
template <> struct Elem<1> { typedef uint8_t T; };
template <> struct Elem<2> { typedef uint16_t T; };
template <> struct Elem<4> { typedef uint32_t T; };
template <> struct Elem<8> { typedef unsigned long long T; };

/* Sum of the ES-byte little-endian integers in a 16-byte vector. */
/* Bytes k .. k+15 of the 32-byte concatenation a:b (little-endian), 0 < k < 16. */
__device__ __forceinline__ uint4 funnel16(uint4 a, uint4 b, uint32_t k)
{
    const uint32_t s = (k & 3u) * 8u;
    uint32_t w0, w1, w2, w3, w4;
    switch (k >> 2) {
    case 0: w0 = a.x; w1 = a.y; w2 = a.z; w3 = a.w; w4 = b.x; break;
    case 1: w0 = a.y; w1 = a.z; w2 = a.w; w3 = b.x; w4 = b.y; break;
    case 2: w0 = a.z; w1 = a.w; w2 = b.x; w3 = b.y; w4 = b.z; break;
    default: w0 = a.w; w1 = b.x; w2 = b.y; w3 = b.z; w4 = b.w; break;
    }
    uint4 o;
    o.x = __funnelshift_r(w0, w1, s);
    o.y = __funnelshift_r(w1, w2, s);
    o.z = __funnelshift_r(w2, w3, s);
    o.w = __funnelshift_r(w3, w4, s);
    return o;
}

/* fp32 bit pattern -> bf16 bit pattern, round to nearest, ties to even.  Adding 0x7FFF plus the
 * lowest kept bit carries into bit 16 exactly when the dropped half is above one half ulp, or
 * equal to it with an odd kept part.  NaNs become the quiet NaN 0x7FC0. */
__device__ __forceinline__ uint32_t bf16_rne(uint32_t u)
{
    const uint32_t rounded = (u + 0x7FFFu + ((u >> 16) & 1u)) >> 16;
    return ((u & 0x7FFFFFFFu) > 0x7F800000u) ? 0x7FC0u : rounded;
}

/* fp32 bit pattern -> fp16 bit pattern, round to nearest, ties to even.  Magnitudes from
 * 65520 (the largest half, 65504, plus half its ulp) up become infinity; below 2^-14 the result
 * is the subnormal m * 2^-24 with m the 24-bit significand shifted right with the same
 * rounding; NaNs become sign | 0x7E00. */
__device__ __forceinline__ uint32_t f16_rne(uint32_t u)
{
    const uint32_t sign = (u >> 16) & 0x8000u;
    const uint32_t a = u & 0x7FFFFFFFu;
    if (a > 0x7F800000u) return sign | 0x7E00u;
    if (a >= 0x477FF000u) return sign | 0x7C00u;
    if (a >= 0x38800000u) /* normal: rebias the exponent by 112, keep 10 mantissa bits */
        return sign | ((a - 0x38000000u + 0xFFFu + ((a >> 13) & 1u)) >> 13);
    const uint32_t e = a >> 23;
    if (e < 102) return sign; /* below 2^-25: rounds to zero */
    const uint32_t sig = (a & 0x7FFFFFu) | 0x800000u;
    const uint32_t sh = 126u - e; /* 14 .. 24 */
    const uint32_t q = sig >> sh, rem = sig & ((1u << sh) - 1u), half = 1u << (sh - 1u);
    return sign | (q + ((rem > half) || (rem == half && (q & 1u)) ? 1u : 0u));
}

/* fp16 bit pattern -> fp32 bit pattern, exact (subnormals normalised, NaN payloads kept). */
__device__ __forceinline__ uint32_t f16_to_f32(uint32_t h)
{
    const uint32_t sign = (h & 0x8000u) << 16;
    const uint32_t e = (h >> 10) & 0x1Fu, m = h & 0x3FFu;
    if (e == 0x1Fu) return sign | 0x7F800000u | (m << 13);
    if (e != 0) return sign | ((e + 112u) << 23) | (m << 13);
    if (m == 0) return sign;
    const uint32_t p = 31u - __clz(m); /* highest set bit, 0 .. 9 */
    return sign | ((p + 103u) << 23) | ((m << (23u - p)) & 0x7FFFFFu);
}

template <int CONV> __device__ __forceinline__ uint32_t convert1(uint32_t x)
{
    if constexpr (CONV == CFA_CONV_F32_BF16) return bf16_rne(x);
    else if constexpr (CONV == CFA_CONV_F32_F16) return f16_rne(x);
    else if constexpr (CONV == CFA_CONV_F16_BF16) return bf16_rne(f16_to_f32(x));
    else if constexpr (CONV == CFA_CONV_BF16_F32) return x << 16;
    else return f16_to_f32(x);
}

/* Source element size, destination element size and conversion of a work class. */
template <int CLS> struct ClassOf {
    static constexpr int conv = CLS >= 4 ? CLS - 3 : 0;
    static constexpr int ses = conv == 0 ? (1 << CLS)
                               : (conv == CFA_CONV_F32_BF16 || conv == CFA_CONV_F32_F16) ? 4 : 2;
    static constexpr int des = conv == 0 ? (1 << CLS)
                               : (conv == CFA_CONV_BF16_F32 || conv == CFA_CONV_F16_F32) ? 4 : 2;
    static constexpr int log2(int x) { return x == 1 ? 0 : x == 2 ? 1 : x == 4 ? 2 : 3; }
    static constexpr uint32_t mode = CFA_MODE(log2(ses), log2(des), conv);
};

/* ---- copy of one contiguous run --------------------------------------------------------- */

template <int ES>
__device__ __forceinline__ uint64_t copy_elems(const uint8_t *src, uint8_t *dst, uint32_t n,
                                               uint32_t tid, uint32_t nthr)
{
    typedef typename Elem<ES>::T T;
    uint64_t acc = 0;
    for (uint32_t e = tid; e < n; e += nthr) {
        const T v = reinterpret_cast<const T *>(src)[e];
        reinterpret_cast<T *>(dst)[e] = v;
        acc += (uint64_t)v;
    }
    return acc;
}

/* Copies nbytes (a multiple of ES) from src to dst; thread tid of nthr.  Returns this thread's
 * share of the checksum. */
template <int ES, int U, int UR, int W = 32>
__device__ uint64_t copy_run(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst,
                             uint64_t nbytes, uint32_t tid, uint32_t nthr)
{
    uint64_t acc = 0;
    /* head: elements until the destination is 16-byte aligned */
    uint32_t head = (uint32_t)((16u - ((uintptr_t)dst & 15u)) & 15u);
    if (head > nbytes) head = (uint32_t)nbytes;
    acc += copy_elems<ES>(src, dst, head / ES, tid, nthr);
    src += head;
    dst += head;
    nbytes -= head;

    /* runs hold at most 2^32 elements of at most 8 bytes, so vector indices fit 32 bits */
    const uint32_t nvec = (uint32_t)(nbytes >> 4);
    const uint32_t k = (uint32_t)((uintptr_t)src & 15u);
    uint4 *d = reinterpret_cast<uint4 *>(dst);
    if (k == 0) {
        const uint4 *s = reinterpret_cast<const uint4 *>(src);
        const uint32_t step = nthr * U;
        for (uint32_t base = 0; base < nvec; base += step) {
            uint4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const uint32_t i = base + u * nthr + tid;
                if (i < nvec) v[u] = ld_stream(s + i);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const uint32_t i = base + u * nthr + tid;
                if (i < nvec) {
                    st_stream(d + i, v[u]);
                    acc += vsum<ES>(v[u]);
                }
            }
        }
    } else {
        /* source off by k bytes: every 16-byte store takes bytes k..k+15 of two aligned
         * vectors s[i] and s[i + 1], both of which hold needed bytes, so nothing outside the
         * run is read.  A group of W lanes (a warp, W = 32, or an 8-lane segment of one on the
         * sub-warp path for tiny pieces, W = 8) takes UR * W consecutive vectors at a time
         * (lane l, round u: vector w0 + W u + l) and loads each once; s[i + 1] comes by shuffle
         * from the next lane, or for the group's last lane from lane 0 of the next round.  The
         * one vector per group that has no loaded neighbour (the last lane's last one, or the
         * run's last vector) is loaded by its lane in the same round of loads.  Every shuffle
         * stays inside the group. */
        const uint4 *s = reinterpret_cast<const uint4 *>(src - k);
        const uint32_t lane = tid & (W - 1u), wid = tid / W;
        const uint32_t mask =
            W == 32 ? 0xFFFFFFFFu : (((1u << W) - 1u) << (threadIdx.x & 31u & ~(W - 1u)));
        const uint32_t step = nthr * UR;
        for (uint32_t base = 0; base < nvec; base += step) {
            const uint32_t w0 = base + wid * W * UR;
            uint4 a[UR];
            int own = -1; /* the round whose neighbour this lane loads itself */
#pragma unroll
            for (int u = 0; u < UR; ++u) {
                const uint32_t i = w0 + W * u + lane;
                a[u] = make_uint4(0u, 0u, 0u, 0u);
                if (i < nvec) {
                    a[u] = ld_shared_line(s + i);
                    if (i + 1 == nvec || (lane == W - 1u && u == UR - 1)) own = u;
                }
            }
            uint4 c = make_uint4(0u, 0u, 0u, 0u);
            if (own >= 0) c = ld_shared_line(s + w0 + W * own + lane + 1);
#pragma unroll
            for (int u = 0; u < UR; ++u) {
                const uint32_t i = w0 + W * u + lane;
                uint4 b, n0;
                b.x = __shfl_down_sync(mask, a[u].x, 1, W);
                b.y = __shfl_down_sync(mask, a[u].y, 1, W);
                b.z = __shfl_down_sync(mask, a[u].z, 1, W);
                b.w = __shfl_down_sync(mask, a[u].w, 1, W);
                if (u + 1 < UR) {
                    n0.x = __shfl_sync(mask, a[u + 1].x, 0, W);
                    n0.y = __shfl_sync(mask, a[u + 1].y, 0, W);
                    n0.z = __shfl_sync(mask, a[u + 1].z, 0, W);
                    n0.w = __shfl_sync(mask, a[u + 1].w, 0, W);
                    if (lane == W - 1u) b = n0;
                }
                if (i < nvec) {
                    if (own == u) b = c;
                    const uint4 o = funnel16(a[u], b, k);
                    st_stream(d + i, o);
                    acc += vsum<ES>(o);
                }
            }
        }
    }
    /* tail */
    const uint64_t body = (uint64_t)nvec << 4;
    acc += copy_elems<ES>(src + body, dst + body, (uint32_t)((nbytes - body) / ES), tid, nthr);
    return acc;
}

/* n elements of SES bytes at src -> n converted elements of DES bytes at dst.  Destination
 * stores are 16 bytes wide; eight elements form a group (32 or 16 source bytes, 16 or 32
 * destination bytes), loaded as 16-byte vectors when the source is aligned, else one by one. */
template <int SES, int DES, int CONV, int U>
__device__ uint64_t convert_run(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst,
                                uint64_t n, uint32_t tid, uint32_t nthr)
{
    typedef typename Elem<SES>::T ST;
    typedef typename Elem<DES>::T DT;
    uint64_t acc = 0;
    uint32_t h = (uint32_t)(((16u - ((uintptr_t)dst & 15u)) & 15u) / DES);
    if (h > n) h = (uint32_t)n;
    for (uint32_t e = tid; e < h; e += nthr) {
        const uint32_t y = convert1<CONV>(reinterpret_cast<const ST *>(src)[e]);
        reinterpret_cast<DT *>(dst)[e] = (DT)y;
        acc += y;
    }
    src += (uint64_t)SES * h;
    dst += (uint64_t)DES * h;
    n -= h;

    const uint32_t ng = (uint32_t)(n >> 3);
    uint4 *d = reinterpret_cast<uint4 *>(dst);
    const bool vec = ((uintptr_t)src & 15u) == 0;
    const uint32_t step = nthr * U;
    for (uint32_t base = 0; base < ng; base += step) {
        uint32_t x[U][8];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t g = base + u * nthr + tid;
            if (g >= ng) continue;
            if (vec && SES == 4) {
                const uint4 a = ld_stream(src + 32ull * g), b = ld_stream(src + 32ull * g + 16);
                x[u][0] = a.x; x[u][1] = a.y; x[u][2] = a.z; x[u][3] = a.w;
                x[u][4] = b.x; x[u][5] = b.y; x[u][6] = b.z; x[u][7] = b.w;
            } else if (vec && SES == 2) {
                const uint4 a = ld_stream(src + 16ull * g);
                x[u][0] = a.x & 0xFFFFu; x[u][1] = a.x >> 16; x[u][2] = a.y & 0xFFFFu;
                x[u][3] = a.y >> 16; x[u][4] = a.z & 0xFFFFu; x[u][5] = a.z >> 16;
                x[u][6] = a.w & 0xFFFFu; x[u][7] = a.w >> 16;
            } else if (SES == 4 && ((uintptr_t)src & 7u) == 0) {
                /* 8-byte aligned: four 8-byte loads instead of eight 4-byte ones */
                const uint2 *s2 = reinterpret_cast<const uint2 *>(src + 32ull * g);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint2 v = __ldg(s2 + q);
                    x[u][2 * q] = v.x;
                    x[u][2 * q + 1] = v.y;
                }
            } else if (SES == 4) {
                /* 4 mod 8: the first and last elements alone, the six between as 8-byte pairs */
                const uint32_t *s1 = reinterpret_cast<const uint32_t *>(src + 32ull * g);
                const uint2 *s2 = reinterpret_cast<const uint2 *>(s1 + 1);
                x[u][0] = __ldg(s1);
#pragma unroll
                for (int q = 0; q < 3; ++q) {
                    const uint2 v = __ldg(s2 + q);
                    x[u][1 + 2 * q] = v.x;
                    x[u][2 + 2 * q] = v.y;
                }
                x[u][7] = __ldg(s1 + 7);
            } else {
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    x[u][q] = reinterpret_cast<const ST *>(src)[8ull * g + q];
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t g = base + u * nthr + tid;
            if (g >= ng) continue;
            uint32_t r[8];
            uint64_t sum = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                r[q] = convert1<CONV>(x[u][q]);
                sum += r[q];
            }
            if constexpr (DES == 2) {
                st_stream(d + g, make_uint4(r[0] | (r[1] << 16), r[2] | (r[3] << 16),
                                            r[4] | (r[5] << 16), r[6] | (r[7] << 16)));
            } else {
                st_stream(d + 2ull * g, make_uint4(r[0], r[1], r[2], r[3]));
                st_stream(d + 2ull * g + 1, make_uint4(r[4], r[5], r[6], r[7]));
            }
            acc += sum;
        }
    }
    const uint64_t body = (uint64_t)ng << 3;
    for (uint64_t e = body + tid; e < n; e += nthr) {
        const uint32_t y = convert1<CONV>(reinterpret_cast<const ST *>(src)[e]);
        reinterpret_cast<DT *>(dst)[e] = (DT)y;
        acc += y;
    }
    return acc;
}

/* Checks a work item against the launch's readable source range and its kernel's class. */
template <int CLS>
__device__ __forceinline__ bool item_ok(const cfa_work &w, const UnpackArgs &a)
{
    const uint32_t sl = w.mode & 3u;
    const uint64_t src_bytes = (uint64_t)w.n << sl;
    const uint32_t want_mode = ClassOf<CLS>::mode;
    const uint32_t dl = (w.mode >> 2) & 3u;
    return w.mode == want_mode && w.n != 0 && w.src >= a.src_lo && w.src <= a.src_hi &&
           src_bytes <= a.src_hi - w.src && (w.src & ((1ull << sl) - 1)) == 0 &&
           (w.dst & ((1ull << dl) - 1)) == 0;
}

/* One work item: U 16-byte vectors per thread in flight on the aligned path, UR rounds of W
 * vectors per lane group on the realigning path (default: four for slabs of the 2-8-byte copy
 * classes, two for the 1-byte class). */
template <int CLS, int U, int W = 32, int UR = (U > 1 ? (CLS >= 1 ? kRealignRounds : 2) : 1)>
__device__ __forceinline__ uint64_t run_item(const cfa_work &w, const UnpackArgs &a, uint32_t tid,
                                             uint32_t nthr)
{
    const uint64_t off = a.src_period ? w.src % a.src_period : w.src;
    const uint8_t *src = reinterpret_cast<const uint8_t *>(a.src_base + off);
    uint8_t *dst = reinterpret_cast<uint8_t *>(w.dst);
    typedef ClassOf<CLS> C;
    if constexpr (C::conv != CFA_CONV_NONE)
        return convert_run<C::ses, C::des, C::conv, (U > 2 ? 2 : U)>(src, dst, w.n, tid, nthr);
    else
        return copy_run<(1 << CLS), U, UR, W>(src, dst, (uint64_t)w.n << CLS, tid, nthr);
}

/* Adds the CTA's accumulated checksum to slot ck; every thread of the CTA must call it. */
__device__ __forceinline__ void block_flush(uint64_t &acc, uint32_t ck, unsigned long long *out,
                                            unsigned long long *red)
{
    const uint64_t v = warp_sum(acc);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long t = 0;
#pragma unroll
        for (int q = 0; q < kWarps; ++q) t += red[q];
        atomicAdd(out + ck, t);
    }
    __syncthreads();
    acc = 0;
}

/* One launch: the block-level items (slabs) and the warp-level items (tiny pieces, in groups of
 * one per warp) of one class.  The groups are spread evenly among the slabs: a tiny piece is
 * bound by memory latency, a slab by bandwidth, so a CTA working on tiny pieces overlaps with
 * its SM neighbours streaming slabs instead of all of them running at the end of the launch.
 * Item i of the first n_groups * (q + 1) items (q = n_slabs / n_groups) is group i / (q + 1)
 * when i mod (q + 1) == q, else slab (i / (q + 1)) * q + i mod (q + 1); the items after those
 * are the remaining slabs in order. */
/* Tiny pieces: a group is kSegs pieces per warp.  When every piece of a warp's share has at most
 * kSegMaxBytes destination bytes, each 8-lane segment copies one piece on its own (four pieces in
 * flight per warp); otherwise the whole warp copies the pieces one after the other.  The plan
 * puts the small pieces of each (class, chunk) first, so most warps see one kind. */
constexpr int kSegLanes = 8;
constexpr int kSegs = 32 / kSegLanes;
constexpr uint32_t kSegMaxBytes = CFA_TINY_SEG_BYTES;
constexpr uint32_t kTinyPerGroup = kWarps * kSegs;

template <int CLS, int U = 1, int UR = 1>
__device__ __forceinline__ void run_tiny(const UnpackArgs &a, uint32_t group, uint32_t warp,
                                         uint32_t lane)
{
    const uint32_t seg = lane / kSegLanes, sub = lane % kSegLanes;
    const uint32_t t = (group * kWarps + warp) * kSegs + seg;
    cfa_work w{};
    bool ok = false;
    uint32_t bytes = 0;
    if (t < a.n_tiny) {
        w = a.tiny[t]; /* the same 32 bytes for the segment's lanes */
        ok = item_ok<CLS>(w, a);
        if (!ok && sub == 0) atomicCAS(a.status, 0, 1);
        if (ok) bytes = w.n << ((w.mode >> 2) & 3u);
    }
    if (!__any_sync(0xFFFFFFFFu, bytes > kSegMaxBytes)) {
        if (ok) {
            const uint32_t mask = 0xFFu << (seg * kSegLanes);
            uint64_t v = run_item<CLS, U, kSegLanes, UR>(w, a, sub, kSegLanes);
#pragma unroll
            for (int o = kSegLanes / 2; o > 0; o >>= 1) v += __shfl_down_sync(mask, v, o, kSegLanes);
            if (sub == 0 && w.ck != CFA_NO_CK) atomicAdd(a.ck + w.ck, v);
        }
        return;
    }
    for (int k = 0; k < kSegs; ++k) {
        const int src_lane = k * kSegLanes;
        if (!__shfl_sync(0xFFFFFFFFu, (int)ok, src_lane)) continue;
        cfa_work wk;
        wk.src = __shfl_sync(0xFFFFFFFFu, (unsigned long long)w.src, src_lane);
        wk.dst = __shfl_sync(0xFFFFFFFFu, (unsigned long long)w.dst, src_lane);
        wk.n = __shfl_sync(0xFFFFFFFFu, w.n, src_lane);
        wk.ck = __shfl_sync(0xFFFFFFFFu, w.ck, src_lane);
        wk.mode = __shfl_sync(0xFFFFFFFFu, w.mode, src_lane);
        wk.pad = __shfl_sync(0xFFFFFFFFu, w.pad, src_lane);
        const uint64_t v = warp_sum(run_item<CLS, U, 32, UR>(wk, a, lane, 32u));
        if (lane == 0 && wk.ck != CFA_NO_CK) atomicAdd(a.ck + wk.ck, v);
    }
}

template <int CLS>
__global__ void __launch_bounds__(kThreads, (CLS >= 1 && CLS < 4 ? kCopyMinBlocks : kMinBlocks))
    cfa_unpack_kernel(const UnpackArgs a)
{
    __shared__ unsigned long long red[kWarps];
    const uint32_t n_groups = (a.n_tiny + kTinyPerGroup - 1) / kTinyPerGroup;
    const uint32_t n_items = a.n_slabs + n_groups;
    const uint32_t q = n_groups ? a.n_slabs / n_groups : 0;
    const uint32_t mixed = n_groups * (q + 1); /* items in the interleaved prefix */
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    uint64_t acc = 0;
    uint32_t acc_ck = CFA_NO_CK;

    for (uint32_t item = blockIdx.x; item < n_items; item += gridDim.x) {
        uint32_t slab, group;
        bool is_slab;
        if (item < mixed) {
            const uint32_t p = item / (q + 1), r = item - p * (q + 1);
            is_slab = r != q;
            slab = p * q + r;
            group = p;
        } else {
            is_slab = true;
            slab = n_groups * q + (item - mixed);
            group = 0;
        }
        if (is_slab) {
            const cfa_work w = a.slabs[slab]; /* the same 32 bytes for every thread */
            if (!item_ok<CLS>(w, a)) {
                if (threadIdx.x == 0) atomicCAS(a.status, 0, 1);
                continue;
            }
            if (w.ck != acc_ck) {
                if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
                acc = 0;
                acc_ck = w.ck;
            }
            acc += run_item<CLS, kUnroll>(w, a, threadIdx.x, kThreads);
        } else {
            if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
            acc_ck = CFA_NO_CK;
            run_tiny<CLS>(a, group, warp, lane);
        }
    }
    if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
}

/* A launch of tiny pieces only (no block-level items).  A tiny piece is bound by latency, not
 * bandwidth: the combined kernel's one vector per lane kept about 2 MB in flight on the whole
 * GPU, a third of what HBM needs at its latency.  Here every piece is copied by one 8-lane
 * segment with kUnroll vectors per lane in flight: a piece whose source and destination share
 * their 16-byte phase (checkpoints packed at 16-byte or wider alignment) in one round trip of up
 * to 512 bytes, head and tail included (copy_same_phase); other copies and conversions through
 * run_item with one realigning round.  Each segment fetches the descriptor of its next piece
 * before copying the current one, so the descriptor load is off the critical path.  Its own
 * kernel keeps these registers out of the combined kernel's budget. */
constexpr int kTinyRounds = 1;

/* Bytes [lo, hi) of a 16-byte vector kept, the others zeroed. */
__device__ __forceinline__ uint4 keep_bytes(uint4 v, uint32_t lo, uint32_t hi)
{
    uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int h = min(max((int)hi - 4 * q, 0), 4), l = min(max((int)lo - 4 * q, 0), 4);
        const uint32_t below_hi = h >= 4 ? 0xFFFFFFFFu : (1u << (8 * h)) - 1u;
        const uint32_t below_lo = l >= 4 ? 0xFFFFFFFFu : (1u << (8 * l)) - 1u;
        w[q] &= below_hi & ~below_lo;
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

/* Stores the ES-byte elements of v at byte offsets [lo, hi) of the 16-byte block at dst16. */
template <int ES>
__device__ __forceinline__ void store_part(uint8_t *dst16, uint4 v, uint32_t lo, uint32_t hi)
{
    typedef typename Elem<ES>::T T;
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 16 / ES; ++q) {
        const uint32_t b = (uint32_t)(q * ES);
        if (b >= lo && b < hi) {
            T e;
            if constexpr (ES == 8)
                e = ((unsigned long long)w[b / 4 + 1] << 32) | w[b / 4];
            else
                e = (T)(w[b / 4] >> (8 * (b % 4)));
            reinterpret_cast<T *>(dst16)[q] = e;
        }
    }
}

/* A tiny piece whose source and destination share their offset within 16 bytes, on W lanes:
 * the whole 16-byte vectors in rounds of W x U (no branch per vector), and the partial first
 * and last vectors (at most one each) by lanes 0 and 1, loaded whole in the same round (an
 * aligned 16-byte block holding bytes of the piece lies in the same page and allocation) and
 * stored element by element.  A piece of up to W * U * 16 bytes is one round trip, and the
 * element-wise code runs once per piece instead of in every vector slot. */
template <int ES, int U, int W>
__device__ __forceinline__ uint64_t copy_same_phase(const uint8_t *src, uint8_t *dst,
                                                    uint32_t nbytes, uint32_t lane)
{
    const uint32_t p = (uint32_t)((uintptr_t)src & 15u);
    const uint4 *s = reinterpret_cast<const uint4 *>(src - p);
    uint8_t *d = dst - p;
    const uint32_t end = p + nbytes; /* in bytes from s */
    const uint32_t nv = (end + 15u) >> 4;
    /* vector 0 is partial if the piece starts inside it or ends inside it */
    const bool part0 = nv > 0 && (p != 0 || (nv == 1 && (end & 15u) != 0));
    const bool part1 = nv > 1 && (end & 15u) != 0; /* the last vector, when not vector 0 */
    const uint32_t f0 = part0 ? 1u : 0u, f1 = part1 ? nv - 1u : (nv > f0 ? nv : f0);
    /* the partial vectors: lane 0 takes vector 0, lane 1 the last; their loads go first */
    uint4 pv = make_uint4(0u, 0u, 0u, 0u);
    const bool mine = (lane == 0 && part0) || (lane == 1 && part1);
    if (mine) pv = ld_stream(s + (lane == 0 ? 0u : nv - 1u));
    uint64_t acc = 0;
    for (uint32_t base = f0; base < f1; base += W * U) {
        uint4 v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t i = base + u * W + lane;
            if (i < f1) v[u] = ld_stream(s + i);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t i = base + u * W + lane;
            if (i < f1) {
                st_stream(d + 16u * i, v[u]);
                acc += vsum<ES>(v[u]);
            }
        }
    }
    if (mine) { /* bounds recomputed here rather than held across the loop */
        const uint32_t pi = lane == 0 ? 0u : nv - 1u;
        const uint32_t plo = pi == 0 ? p : 0u;
        const uint32_t phi = end - 16u * pi < 16u ? end - 16u * pi : 16u;
        store_part<ES>(d + 16u * pi, pv, plo, phi);
        acc += vsum<ES>(keep_bytes(pv, plo, phi));
    }
    return acc;
}

/* A tiny piece whose source and destination differ in their offset within 16 bytes, on W lanes:
 * every 16-byte destination vector takes bytes k .. k+15 of the two aligned source vectors
 * under it (k the phase difference); each source vector is loaded once and passed to the lane
 * that needs it as its second by shuffle, as on copy_run's realigning path; the partial first
 * and last destination vectors go to lanes 0 and 1 as in copy_same_phase.  Only source vectors that hold bytes of the piece are loaded, so every load
 * stays in the piece's pages.  One round trip for up to W * U * 16 bytes. */
template <int ES, int U, int W>
__device__ __forceinline__ uint64_t copy_diff_phase(const uint8_t *src, uint8_t *dst,
                                                    uint32_t nbytes, uint32_t lane)
{
    const uint32_t dp = (uint32_t)((uintptr_t)dst & 15u);
    uint8_t *d = dst - dp;
    const uint8_t *A = src - dp; /* source byte of destination vector 0's byte 0 */
    const uint32_t k = (uint32_t)((uintptr_t)A & 15u);
    const uint4 *s = reinterpret_cast<const uint4 *>(A - k);
    const uint32_t end = dp + nbytes;
    const uint32_t nv = (end + 15u) >> 4;
    const bool part0 = nv > 0 && (dp != 0 || (nv == 1 && (end & 15u) != 0));
    const bool part1 = nv > 1 && (end & 15u) != 0;
    const uint32_t f0 = part0 ? 1u : 0u, f1 = part1 ? nv - 1u : (nv > f0 ? nv : f0);
    /* destination byte j of vector i comes from source vector i when j < 16 - k, else i + 1 */
    const uint32_t split = 16u - k;
    uint4 pa = make_uint4(0u, 0u, 0u, 0u), pb = pa;
    const bool mine = (lane == 0 && part0) || (lane == 1 && part1);
    if (mine) {
        const uint32_t pi = lane == 0 ? 0u : nv - 1u;
        const uint32_t plo = pi == 0 ? dp : 0u;
        const uint32_t phi = end - 16u * pi < 16u ? end - 16u * pi : 16u;
        if (plo < split) pa = ld_shared_line(s + pi);
        if (phi > split) pb = ld_shared_line(s + pi + 1u);
    }
    uint64_t acc = 0;
    const uint32_t mask =
        W == 32 ? 0xFFFFFFFFu : (((1u << W) - 1u) << (threadIdx.x & 31u & ~(W - 1u)));
    for (uint32_t base = f0; base < f1; base += W * U) {
        /* lane l, round u holds source vector i = base + W u + l; vector i + 1 comes from the
         * next lane, or for the last lane from lane 0 of the next round; the lane whose
         * neighbour holds nothing (i + 1 == f1, or the last lane's last round) loads it */
        uint4 va[U];
        int own = -1;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t i = base + u * W + lane;
            va[u] = make_uint4(0u, 0u, 0u, 0u);
            if (i < f1) {
                va[u] = ld_shared_line(s + i);
                if (i + 1u == f1 || (lane == W - 1u && u == U - 1)) own = u;
            }
        }
        uint4 c = make_uint4(0u, 0u, 0u, 0u);
        if (own >= 0) c = ld_shared_line(s + base + W * own + lane + 1u);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t i = base + u * W + lane;
            uint4 b, n0;
            b.x = __shfl_down_sync(mask, va[u].x, 1, W);
            b.y = __shfl_down_sync(mask, va[u].y, 1, W);
            b.z = __shfl_down_sync(mask, va[u].z, 1, W);
            b.w = __shfl_down_sync(mask, va[u].w, 1, W);
            if (u + 1 < U) {
                n0.x = __shfl_sync(mask, va[u + 1].x, 0, W);
                n0.y = __shfl_sync(mask, va[u + 1].y, 0, W);
                n0.z = __shfl_sync(mask, va[u + 1].z, 0, W);
                n0.w = __shfl_sync(mask, va[u + 1].w, 0, W);
                if (lane == W - 1u) b = n0;
            }
            if (i < f1) {
                if (own == u) b = c;
                const uint4 o = funnel16(va[u], b, k);
                st_stream(d + 16u * i, o);
                acc += vsum<ES>(o);
            }
        }
    }
    if (mine) {
        const uint32_t pi = lane == 0 ? 0u : nv - 1u;
        const uint32_t plo = pi == 0 ? dp : 0u;
        const uint32_t phi = end - 16u * pi < 16u ? end - 16u * pi : 16u;
        const uint4 o = funnel16(pa, pb, k);
        store_part<ES>(d + 16u * pi, o, plo, phi);
        acc += vsum<ES>(keep_bytes(o, plo, phi));
    }
    return acc;
}

/* A work descriptor read with volatile loads: issued where it is written (the top of the
 * tiny kernel's loop, one piece ahead), so the compiler cannot move the load down to its use
 * and put a second memory round trip into every piece. */
__device__ __forceinline__ cfa_work ld_work_now(const cfa_work *p)
{
    uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
                 : "l"(p));
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(b0), "=r"(b1), "=r"(b2), "=r"(b3)
                 : "l"(reinterpret_cast<const uint8_t *>(p) + 16));
    cfa_work w;
    w.src = ((uint64_t)a1 << 32) | a0;
    w.dst = ((uint64_t)a3 << 32) | a2;
    w.n = b0;
    w.ck = b1;
    w.mode = b2;
    w.pad = b3;
    return w;
}

/* ---- tiny copies staged through shared memory with cp.async ----------------------------- */

/* Aligned 16-byte source vectors per warp-level item in shared memory: an item of at most
 * CFA_TINY_SEG_BYTES bytes spans at most CFA_TINY_SEG_BYTES / 16 + 1 of them, plus one that the
 * realigning read may touch (its bytes are never used). */
constexpr int kSlotVecs = CFA_TINY_SEG_BYTES / 16 + 2;

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem)
{
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

/* One item of the segment's pipeline: its descriptor, whether it is to be copied, and its source
 * address (the item's aligned vectors start at src - phase). */
struct TinyItem {
    cfa_work w;
    bool live;
};

template <int CLS>
__device__ __forceinline__ TinyItem tiny_fetch(const UnpackArgs &a, uint32_t group,
                                               uint32_t n_groups, uint32_t slot,
                                               uint32_t per_group)
{
    TinyItem it;
    it.live = false;
    it.w = cfa_work{};
    const uint32_t t = group * per_group + slot;
    if (group < n_groups && t < a.n_tiny) {
        it.w = ld_work_now(a.tiny + t);
        it.live = true;
    }
    return it;
}

/* Issues the cp.async copies of an item's aligned source vectors into `stage` (lanes sub, sub +
 * 8, ...).  Items that fail the kernel's checks, or exceed CFA_TINY_SEG_BYTES, are flagged in
 * the status word and dropped. */
template <int CLS, int L>
__device__ __forceinline__ void tiny_issue(const UnpackArgs &a, TinyItem &it, uint4 *stage,
                                           uint32_t sub)
{
    if (!it.live) return;
    const uint32_t bytes = it.w.n << CLS;
    if (!item_ok<CLS>(it.w, a) || bytes > CFA_TINY_SEG_BYTES) {
        if (sub == 0) atomicCAS(a.status, 0, 1);
        it.live = false;
        return;
    }
    const uint64_t off = a.src_period ? it.w.src % a.src_period : it.w.src;
    const uint64_t src = a.src_base + off;
    const uint32_t ps = (uint32_t)(src & 15u);
    const uint32_t nv = (ps + bytes + 15u) >> 4;
    const uint4 *s = reinterpret_cast<const uint4 *>(src - ps);
    for (uint32_t v = sub; v < nv; v += L) cp_async16(stage + v, s + v);
}

/* Writes a staged item to its destination: destination vector i (aligned) holds staged bytes
 * [16 i + delta, 16 i + delta + 16), delta = source phase - destination phase, so with
 * delta = 16 j0 + k it is staged vector i + j0 (k = 0) or bytes k .. of vectors i + j0 and
 * i + j0 + 1.  The whole vectors go in a tight loop over the segment's lanes; the partial first
 * and last ones (when the item covers them only in part) go to lanes 0 and 1, element by
 * element.  Returns this lane's checksum share. */
template <int CLS, int L>
__device__ __forceinline__ uint64_t tiny_store(const UnpackArgs &a, const TinyItem &it,
                                               const uint4 *stage, uint32_t sub)
{
    constexpr int ES = 1 << CLS;
    if (!it.live) return 0;
    const uint32_t bytes = it.w.n << CLS;
    const uint64_t off = a.src_period ? it.w.src % a.src_period : it.w.src;
    const uint32_t ps = (uint32_t)((a.src_base + off) & 15u);
    const uint32_t dp = (uint32_t)(it.w.dst & 15u);
    uint4 *d = reinterpret_cast<uint4 *>(it.w.dst - dp);
    const uint32_t end = dp + bytes;
    const uint32_t nv = (end + 15u) >> 4;
    const int delta = (int)ps - (int)dp;
    const int j0 = delta >> 4; /* -1 or 0 */
    const uint32_t k = (uint32_t)delta & 15u;
    const bool part0 = dp != 0 || (nv == 1 && (end & 15u) != 0);
    const bool part1 = nv > 1 && (end & 15u) != 0;
    const uint32_t f0 = part0 ? 1u : 0u, f1 = part1 ? nv - 1u : (nv > f0 ? nv : f0);
    uint64_t acc = 0;
    if (k == 0) {
        for (uint32_t i = f0 + sub; i < f1; i += L) {
            const uint4 v = stage[i]; /* k == 0 means delta == 0 */
            st_stream(d + i, v);
            acc += vsum<ES>(v);
        }
    } else {
        for (uint32_t i = f0 + sub; i < f1; i += L) {
            const int j = (int)i + j0; /* >= 0: i >= 1 here when j0 = -1 (part0 is then set) */
            const uint4 v = funnel16(stage[j], stage[j + 1], k);
            st_stream(d + i, v);
            acc += vsum<ES>(v);
        }
    }
    if ((sub == 0 && part0) || (sub == 1 && part1)) {
        const uint32_t i = sub == 0 ? 0u : nv - 1u;
        const int j = (int)i + j0;
        const uint4 lo_v = stage[j < 0 ? 0 : j];
        const uint4 v = k ? funnel16(lo_v, stage[j + 1], k) : lo_v;
        const uint32_t lo = i == 0 ? dp : 0u;
        const uint32_t hi = end - 16u * i < 16u ? end - 16u * i : 16u;
        store_part<ES>(reinterpret_cast<uint8_t *>(d + i), v, lo, hi);
        acc += vsum<ES>(keep_bytes(v, lo, hi));
    }
    return acc;
}

/* The copy classes' tiny kernel body: each group of kStagedLanes lanes runs a two-deep pipeline
 * over its items (one per group of the CTA's groups of items): the cp.async copies of item k + 1
 * are in flight while item k is written out, and the descriptor of item k + 2 is fetched
 * meanwhile.  The source bytes wait in shared memory (dynamic: two slots per lane group), not
 * in registers, so memory-level parallelism does not cost occupancy; with four lanes per item a
 * warp carries eight items at once, so the per-item work (descriptor, checks, checksum
 * reduction) takes half the warp instructions it would with eight lanes. */
constexpr int kStagedLanes = 4;
constexpr int kStagedPerWarp = 32 / kStagedLanes;
constexpr uint32_t kStagedPerGroup = kWarps * kStagedPerWarp;
constexpr uint32_t kStagedSmem = kStagedPerGroup * 2 * kSlotVecs * sizeof(uint4);

template <int CLS>
__device__ __forceinline__ void tiny_staged(const UnpackArgs &a)
{
    constexpr int L = kStagedLanes;
    extern __shared__ __align__(16) uint4 tiny_stage[];
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    const uint32_t seg = lane / L, sub = lane % L;
    const uint32_t mask = ((1u << L) - 1u) << (seg * L);
    const uint32_t n_groups = (a.n_tiny + kStagedPerGroup - 1) / kStagedPerGroup;
    const uint32_t slot = warp * kStagedPerWarp + seg;
    uint4 *buf0 = tiny_stage + (size_t)slot * 2 * kSlotVecs, *buf1 = buf0 + kSlotVecs;
    uint32_t group = blockIdx.x;
    TinyItem cur = tiny_fetch<CLS>(a, group, n_groups, slot, kStagedPerGroup);
    TinyItem nxt = tiny_fetch<CLS>(a, group + gridDim.x, n_groups, slot, kStagedPerGroup);
    tiny_issue<CLS, L>(a, cur, buf0, sub);
    cp_async_commit();
    for (uint32_t k = 0; group < n_groups; ++k, group += gridDim.x) {
        const TinyItem after =
            tiny_fetch<CLS>(a, group + 2 * gridDim.x, n_groups, slot, kStagedPerGroup);
        tiny_issue<CLS, L>(a, nxt, (k & 1) ? buf0 : buf1, sub);
        cp_async_commit();
        cp_async_wait_1(); /* this lane's copies of item k have landed */
        __syncwarp(mask);  /* and the other lanes' of the group */
        uint64_t v = tiny_store<CLS, L>(a, cur, (k & 1) ? buf1 : buf0, sub);
#pragma unroll
        for (int q = L / 2; q > 0; q >>= 1) v += __shfl_down_sync(mask, v, q, L);
        if (sub == 0 && cur.live && cur.w.ck != CFA_NO_CK) atomicAdd(a.ck + cur.w.ck, v);
        __syncwarp(mask);  /* the slot of item k is read; item k + 2 may be copied into it */
        cur = nxt;
        nxt = after;
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
}

template <int CLS>
__global__ void __launch_bounds__(kThreads, (CLS < 4 ? kCopyMinBlocks : kMinBlocks))
    cfa_tiny_kernel(const UnpackArgs a)
{
    if constexpr (CLS < 4) {
        /* device-memory sources take the shared-memory pipeline; host memory read in place over
         * the link keeps plain loads */
        if (a.dev_src) {
            tiny_staged<CLS>(a);
            return;
        }
    }
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    const uint32_t seg = lane / kSegLanes, sub = lane % kSegLanes;
    const uint32_t mask = 0xFFu << (seg * kSegLanes);
    const uint32_t n_groups = (a.n_tiny + kTinyPerGroup - 1) / kTinyPerGroup;
    const uint32_t slot = warp * kSegs + seg; /* this segment's piece within a group */
    uint32_t group = blockIdx.x;
    cfa_work w{};
    if (group < n_groups && group * kTinyPerGroup + slot < a.n_tiny)
        w = ld_work_now(a.tiny + group * kTinyPerGroup + slot);
    while (group < n_groups) {
        const uint32_t t = group * kTinyPerGroup + slot;
        const uint32_t next = group + gridDim.x;
        cfa_work wn{};
        if (next < n_groups && next * kTinyPerGroup + slot < a.n_tiny)
            wn = ld_work_now(a.tiny + next * kTinyPerGroup + slot);
        if (t < a.n_tiny) {
            if (item_ok<CLS>(w, a)) {
                uint64_t v;
                const uint64_t off = a.src_period ? w.src % a.src_period : w.src;
                const uint8_t *src = reinterpret_cast<const uint8_t *>(a.src_base + off);
                uint8_t *dst = reinterpret_cast<uint8_t *>(w.dst);
                constexpr int ES = CLS < 4 ? (1 << CLS) : 1;
                if (CLS >= 4)
                    v = run_item<CLS, kUnroll, kSegLanes, kTinyRounds>(w, a, sub, kSegLanes);
                else if ((((uintptr_t)src ^ (uintptr_t)dst) & 15u) == 0)
                    v = copy_same_phase<ES, kUnroll, kSegLanes>(src, dst, w.n * ES, sub);
                else
                    v = copy_diff_phase<ES, 2, kSegLanes>(src, dst, w.n * ES, sub);
#pragma unroll
                for (int o = kSegLanes / 2; o > 0; o >>= 1)
                    v += __shfl_down_sync(mask, v, o, kSegLanes);
                if (sub == 0 && w.ck != CFA_NO_CK) atomicAdd(a.ck + w.ck, v);
            } else if (sub == 0) {
                atomicCAS(a.status, 0, 1);
            }
        }
        w = wn;
        group = next;
    }
}

/* ---- host -> device pull over the host link --------------------------------------------- */

/* Copies bytes [0, n) from src (host memory the device reads over NVLink-C2C: page-locked, or any
 * memory on devices that read pageable memory) to dst (device memory), which share their offset
 * within 16 bytes: head and tail bytes one by one, the body in 16-byte vectors, four in flight
 * per thread.  The staged pipeline's second transfer path beside the copy engine. */
__global__ void __launch_bounds__(kThreads) cfa_pull_kernel(const uint8_t *__restrict__ src,
                                                            uint8_t *__restrict__ dst, uint64_t n)
{
    const uint64_t tid = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const uint64_t nthr = (uint64_t)gridDim.x * blockDim.x;
    uint64_t head = (16u - ((uintptr_t)dst & 15u)) & 15u;
    if (head > n) head = n;
    for (uint64_t e = tid; e < head; e += nthr) dst[e] = src[e];
    const uint4 *s = reinterpret_cast<const uint4 *>(src + head);
    uint4 *d = reinterpret_cast<uint4 *>(dst + head);
    const uint64_t nv = (n - head) >> 4;
    uint64_t i = tid;
    for (; i + 3 * nthr < nv; i += 4 * nthr) {
        const uint4 a = ld_stream(s + i), b = ld_stream(s + i + nthr);
        const uint4 c = ld_stream(s + i + 2 * nthr), e = ld_stream(s + i + 3 * nthr);
        st_stream(d + i, a);
        st_stream(d + i + nthr, b);
        st_stream(d + i + 2 * nthr, c);
        st_stream(d + i + 3 * nthr, e);
    }
    for (; i < nv; i += nthr) st_stream(d + i, ld_stream(s + i));
    for (uint64_t e = head + (nv << 4) + tid; e < n; e += nthr) dst[e] = src[e];
}

/* ---- column slices: blocks of strided rows -------------------------------------------- */

struct StridedArgs {
    const cfa_swork *items;
    uint32_t n_items;
    uint32_t pad;
    uint64_t src_base;
    uint64_t src_period;
    uint64_t src_lo, src_hi;
    unsigned long long *ck;
    int *status;
};

template <int CLS>
__device__ __forceinline__ bool sitem_ok(const cfa_swork &w, const StridedArgs &a)
{
    const uint32_t want_mode = ClassOf<CLS>::mode;
    if (w.mode != want_mode || w.rows == 0 || w.cols == 0 || w.stride < w.cols) return false;
    const uint32_t sl = w.mode & 3u, dl = (w.mode >> 2) & 3u;
    const uint64_t extent = ((uint64_t)(w.rows - 1) * w.stride + w.cols) << sl;
    return w.src >= a.src_lo && w.src <= a.src_hi && extent <= a.src_hi - w.src &&
           (w.src & ((1ull << sl) - 1)) == 0 && (w.dst & ((1ull << dl) - 1)) == 0;
}

/* Each CTA takes blocks of rows; its warps take the rows of a block in turn and copy each row
 * like a contiguous run (16-byte vectors, realigned when source and destination disagree mod
 * 16, four vectors in flight per lane). */
template <int CLS>
__global__ void __launch_bounds__(kThreads, (CLS < 4 ? kCopyMinBlocks : kMinBlocks))
    cfa_strided_kernel(const StridedArgs a)
{
    typedef ClassOf<CLS> C;
    constexpr int SES = C::ses;
    constexpr int DES = C::des;
    __shared__ unsigned long long red[kWarps];
    const uint32_t lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    uint64_t acc = 0;
    uint32_t acc_ck = CFA_NO_CK;
    for (uint32_t item = blockIdx.x; item < a.n_items; item += gridDim.x) {
        const cfa_swork w = a.items[item];
        if (!sitem_ok<CLS>(w, a)) {
            if (threadIdx.x == 0) atomicCAS(a.status, 0, 1);
            continue;
        }
        if (w.ck != acc_ck) {
            if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
            acc = 0;
            acc_ck = w.ck;
        }
        const uint64_t off = a.src_period ? w.src % a.src_period : w.src;
        const uint8_t *src = reinterpret_cast<const uint8_t *>(a.src_base + off);
        uint8_t *dst = reinterpret_cast<uint8_t *>(w.dst);
        for (uint32_t r = warp; r < w.rows; r += kWarps) {
            const uint8_t *s = src + (uint64_t)r * w.stride * SES;
            uint8_t *d = dst + (uint64_t)r * w.cols * DES;
            if constexpr (C::conv != CFA_CONV_NONE)
                acc += convert_run<SES, DES, C::conv, 2>(s, d, w.cols, lane, 32u);
            else
                acc += copy_run<DES, kUnroll, kRealignRoundsRows>(s, d, (uint64_t)w.cols * DES,
                                                                  lane, 32u);
        }
    }
    if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
}

typedef void (*strided_fn)(const StridedArgs);
const strided_fn kStrided[CFA_N_CLASSES] = {
    cfa_strided_kernel<0>, cfa_strided_kernel<1>, cfa_strided_kernel<2>,
    cfa_strided_kernel<3>, cfa_strided_kernel<4>, cfa_strided_kernel<5>,
    cfa_strided_kernel<6>, cfa_strided_kernel<7>, cfa_strided_kernel<8>};

typedef void (*kernel_fn)(const UnpackArgs);
const kernel_fn kKernels[CFA_N_CLASSES] = {
    cfa_unpack_kernel<0>, cfa_unpack_kernel<1>, cfa_unpack_kernel<2>,
    cfa_unpack_kernel<3>, cfa_unpack_kernel<4>, cfa_unpack_kernel<5>,
    cfa_unpack_kernel<6>, cfa_unpack_kernel<7>, cfa_unpack_kernel<8>};
const kernel_fn kTiny[CFA_N_CLASSES] = {
    cfa_tiny_kernel<0>, cfa_tiny_kernel<1>, cfa_tiny_kernel<2>,
    cfa_tiny_kernel<3>, cfa_tiny_kernel<4>, cfa_tiny_kernel<5>,
    cfa_tiny_kernel<6>, cfa_tiny_kernel<7>, cfa_tiny_kernel<8>};

/* Lets the tiny kernel of copy class cls use kStagedSmem bytes of dynamic shared memory on the
 * current device (over the 48 KiB default), once per device and class. */
cudaError_t tiny_smem_ready(int cls)
{
    static std::atomic<unsigned char> done[64][4];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || cls < 0 || cls >= 4) return cudaErrorInvalidValue;
    if (done[dev][cls].load(std::memory_order_acquire)) return cudaSuccess;
    e = cudaFuncSetAttribute(kTiny[cls], cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kStagedSmem);
    if (e == cudaSuccess) done[dev][cls].store(1, std::memory_order_release);
    return e;
}

} // namespace

/* Resident CTAs per SM of the class-cls kernel (0 if it cannot run). */
extern "C" int cfa_unpack_blocks_per_sm(int cls)
{
    if (cls < 0 || cls >= CFA_N_CLASSES) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kKernels[cls], kThreads, 0) !=
        cudaSuccess)
        return 0;
    return n;
}

/* Launches the class-cls unpack over the given work items; grid_cap bounds the persistent grid.
 * Blob byte o is read at src_base + o, or at src_base + (o mod src_period) for a periodic
 * source (a work item never straddles a period: periods are whole chunks). */
extern "C" cudaError_t cfa_launch_unpack(int cls, const cfa_work *slabs, uint32_t n_slabs,
                                         const cfa_work *tiny, uint32_t n_tiny,
                                         uint64_t src_base, uint64_t src_period,
                                         uint64_t src_lo, uint64_t src_hi,
                                         unsigned long long *ck, int *status, int grid_cap,
                                         int dev_src, cudaStream_t stream)
{
    if (cls < 0 || cls >= CFA_N_CLASSES || grid_cap <= 0) return cudaErrorInvalidValue;
    const uint64_t items = (uint64_t)n_slabs + (n_tiny + kTinyPerGroup - 1) / kTinyPerGroup;
    if (items == 0) return cudaSuccess;
    UnpackArgs a;
    a.slabs = slabs;
    a.tiny = tiny;
    a.n_slabs = n_slabs;
    a.n_tiny = n_tiny;
    a.src_base = src_base;
    a.src_period = src_period;
    a.src_lo = src_lo;
    a.src_hi = src_hi;
    a.ck = ck;
    a.status = status;
    a.dev_src = dev_src ? 1u : 0u;
    const uint64_t grid = items < (uint64_t)grid_cap ? items : (uint64_t)grid_cap;
    /* tiny pieces alone take the tiny kernel (same occupancy class as the combined one, so the
     * same grid cap holds); its copy classes stage device-memory sources in dynamic shared
     * memory */
    if (n_slabs == 0) {
        const bool staged = cls < 4 && dev_src;
        if (staged) {
            cudaError_t e = tiny_smem_ready(cls);
            if (e != cudaSuccess) return e;
        }
        kTiny[cls]<<<(unsigned)grid, kThreads, staged ? kStagedSmem : 0, stream>>>(a);
    } else {
        kKernels[cls]<<<(unsigned)grid, kThreads, 0, stream>>>(a);
    }
    return cudaGetLastError();
}

/* Pulls `bytes` from host memory at src into device memory at dst (same offset within 16
 * bytes) on `stream` with a grid of `grid` CTAs. */
extern "C" cudaError_t cfa_launch_pull(const void *src, void *dst, uint64_t bytes, int grid,
                                       cudaStream_t stream)
{
    if (!bytes) return cudaSuccess;
    if (!src || !dst || grid <= 0 || (((uintptr_t)src ^ (uintptr_t)dst) & 15u))
        return cudaErrorInvalidValue;
    cfa_pull_kernel<<<grid, kThreads, 0, stream>>>(static_cast<const uint8_t *>(src),
                                                   static_cast<uint8_t *>(dst), bytes);
    return cudaGetLastError();
}

/* Resident CTAs per SM of the class-cls strided kernel (0 if it cannot run). */
extern "C" int cfa_strided_blocks_per_sm(int cls)
{
    if (cls < 0 || cls >= CFA_N_CLASSES) return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kStrided[cls], kThreads, 0) !=
        cudaSuccess)
        return 0;
    return n;
}

/* Launches the class-cls unpack of strided row blocks (column slices of checkpoint tensors). */
extern "C" cudaError_t cfa_launch_strided(int cls, const cfa_swork *items, uint32_t n_items,
                                          uint64_t src_base, uint64_t src_period,
                                          uint64_t src_lo, uint64_t src_hi,
                                          unsigned long long *ck, int *status, int grid_cap,
                                          cudaStream_t stream)
{
    if (cls < 0 || cls >= CFA_N_CLASSES || grid_cap <= 0) return cudaErrorInvalidValue;
    if (n_items == 0) return cudaSuccess;
    StridedArgs a;
    a.items = items;
    a.n_items = n_items;
    a.pad = 0;
    a.src_base = src_base;
    a.src_period = src_period;
    a.src_lo = src_lo;
    a.src_hi = src_hi;
    a.ck = ck;
    a.status = status;
    const uint32_t grid = n_items < (uint32_t)grid_cap ? n_items : (uint32_t)grid_cap;
    kStrided[cls]<<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}
