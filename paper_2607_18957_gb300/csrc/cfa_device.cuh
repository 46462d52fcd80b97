/*
 * Device helpers shared by the unpack kernels (cfa_unpack.cu) and the TMA kernel (cfa_bulk.cu):
 * the per-vector checksum term and the warp reduction of checksums.  A checksum is the sum,
 * modulo 2^64, of a tensor's destination elements read as unsigned integers of the element size.
 */
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace cfa_dev {

/* Sum of the elements of one 16-byte vector of ES-byte unsigned elements. */
template <int ES> __device__ __forceinline__ uint64_t vsum(uint4 v);
template <> __device__ __forceinline__ uint64_t vsum<1>(uint4 v)
{
    return (uint64_t)(__vsadu4(v.x, 0u) + __vsadu4(v.y, 0u) + __vsadu4(v.z, 0u) +
                      __vsadu4(v.w, 0u));
}
template <> __device__ __forceinline__ uint64_t vsum<2>(uint4 v)
{
    const uint32_t lo = (v.x & 0xFFFFu) + (v.y & 0xFFFFu) + (v.z & 0xFFFFu) + (v.w & 0xFFFFu);
    const uint32_t hi = (v.x >> 16) + (v.y >> 16) + (v.z >> 16) + (v.w >> 16);
    return (uint64_t)lo + hi;
}
template <> __device__ __forceinline__ uint64_t vsum<4>(uint4 v)
{
    return (uint64_t)v.x + v.y + v.z + v.w;
}
template <> __device__ __forceinline__ uint64_t vsum<8>(uint4 v)
{
    return (((uint64_t)v.y << 32) | v.x) + (((uint64_t)v.w << 32) | v.z);
}

/* Sum over the 32 lanes of a warp; lane 0 holds the total. */
__device__ __forceinline__ uint64_t warp_sum(uint64_t v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, o);
    return v;
}

} // namespace cfa_dev
