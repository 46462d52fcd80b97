/*
 * TMA bulk-copy unpack: the "InGPU -> Loaded" copy of InstantInfer section 4.2 for large
 * contiguous runs that need no cast and whose source, destination and length are multiples of
 * 16 bytes.  Instead of every thread moving 16-byte vectors through registers, one thread per
 * CTA drives the Tensor Memory Accelerator with non-tensor bulk copies:
 *
 *     global (staging) --cp.async.bulk--> shared stage --cp.async.bulk--> global (destination)
 *
 * through a ring of shared-memory stages.  Loads run kStages - 1 sub-blocks ahead of the
 * stores; completion of a load is signalled on the stage's mbarrier (complete_tx); a stage is
 * reloaded only after the bulk store that read it has finished reading (bulk_group wait).  The
 * other threads only sum the stage for the per-tensor checksum while the store drains it.  Plain
 * cp.async.bulk only: no tensor maps, no multicast, one CTA's own shared memory.
 *
 * Every wait is bounded: a wait that runs out sets the status word, the CTA waits (again
 * bounded) for its own copies still in flight, and returns.
 */
#include <cuda_runtime.h>
#include <stdint.h>

#include "cfa_internal.h"

namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kStages = 4;
constexpr uint32_t kStageBytes = 24 * 1024;
constexpr uint32_t kSmemBytes = kStages * kStageBytes; /* 96 KiB: two CTAs per SM */
constexpr uint32_t kSpinLimit = 1u << 20;              /* try_wait polls before giving up */

struct BulkArgs {
    const cfa_work *items;
    uint32_t n_items;
    uint32_t pad;
    uint64_t src_base;
    uint64_t src_period; /* 0, or P: blob byte o sits at src_base + (o mod P) */
    uint64_t src_lo, src_hi;
    unsigned long long *ck;
    int *status;
};

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t done;
    asm volatile("{\n\t.reg .pred p;\n\t"
                 "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(done)
                 : "r"(smem_addr(bar)), "r"(parity)
                 : "memory");
    return done != 0;
}

/* Waits for phase `parity` of the barrier to complete; false if the spin limit ran out. */
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity)
{
    for (uint32_t k = 0; k < kSpinLimit; ++k)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

__device__ __forceinline__ void bulk_load(void *smem, const void *gsrc, uint32_t bytes,
                                          uint64_t *bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
                 "[%0], [%1], %2, [%3];" ::"r"(smem_addr(smem)),
                 "l"(gsrc), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}

__device__ __forceinline__ void bulk_store(void *gdst, const void *smem, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst),
                 "r"(smem_addr(smem)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

__device__ __forceinline__ void bulk_wait_read_all_but_one()
{
    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}

__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

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

__device__ __forceinline__ uint64_t warp_sum(uint64_t v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, o);
    return v;
}

__device__ __forceinline__ void block_flush(uint64_t &acc, uint32_t ck, unsigned long long *out,
                                            unsigned long long *red)
{
    const uint64_t v = warp_sum(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
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

/* A bulk item is sound if its source lies inside the launch's readable range and source,
 * destination and length are multiples of 16 bytes. */
template <int LOG2ES>
__device__ __forceinline__ bool bulk_item_ok(const cfa_work &w, const BulkArgs &a)
{
    const uint64_t bytes = (uint64_t)w.n << LOG2ES;
    return w.n != 0 && w.mode == CFA_MODE(LOG2ES, LOG2ES, 0) && w.src >= a.src_lo &&
           w.src <= a.src_hi && bytes <= a.src_hi - w.src && bytes < (1ull << 31) &&
           ((w.src | w.dst | bytes | a.src_base | a.src_period) & 15u) == 0;
}

/* Walks the sub-blocks of this CTA's items (items blockIdx.x, + gridDim.x, ...), each at most
 * kStageBytes long. */
struct Cursor {
    uint32_t item, off, count;
    __device__ Cursor() : item(blockIdx.x), off(0), count(0) {}
    __device__ void advance(uint32_t len, uint32_t total)
    {
        off += len;
        ++count;
        if (off >= total) {
            off = 0;
            item += gridDim.x;
        }
    }
};

template <int LOG2ES>
__global__ void __launch_bounds__(kThreads) cfa_bulk_kernel(const BulkArgs a)
{
    extern __shared__ __align__(128) uint8_t stage[];
    __shared__ __align__(8) uint64_t full[kStages];
    __shared__ unsigned long long red[kWarps];
    __shared__ int aborted;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        aborted = 0;
    }
    __syncthreads();

    /* producer (thread 0): issues the load of the next sub-block, if any */
    Cursor prod;
    auto issue = [&]() {
        while (prod.item < a.n_items && !bulk_item_ok<LOG2ES>(a.items[prod.item], a))
            prod.item += gridDim.x;
        if (prod.item >= a.n_items) return;
        const cfa_work w = a.items[prod.item];
        const uint32_t total = w.n << LOG2ES;
        const uint32_t len = min(kStageBytes, total - prod.off);
        const int s = prod.count % kStages;
        mbar_expect_tx(&full[s], len);
        const uint64_t off = a.src_period ? w.src % a.src_period : w.src;
        bulk_load(stage + s * kStageBytes,
                  reinterpret_cast<const uint8_t *>(a.src_base + off) + prod.off, len, &full[s]);
        prod.advance(len, total);
    };
    if (threadIdx.x == 0)
        for (int k = 0; k < kStages - 1; ++k) issue();

    uint64_t acc = 0;
    uint32_t acc_ck = CFA_NO_CK;
    Cursor cons;
    while (cons.item < a.n_items) {
        const cfa_work w = a.items[cons.item];
        if (!bulk_item_ok<LOG2ES>(w, a)) { /* skipped by the producer too */
            if (threadIdx.x == 0) atomicCAS(a.status, 0, 1);
            cons.item += gridDim.x;
            continue;
        }
        const uint32_t total = w.n << LOG2ES;
        const uint32_t len = min(kStageBytes, total - cons.off);
        const int s = cons.count % kStages;
        if (!mbar_wait(&full[s], (cons.count / kStages) & 1u)) aborted = 1;
        __syncthreads();
        if (aborted) break;
        if (w.ck != acc_ck) {
            if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
            acc_ck = w.ck;
        }
        if (w.ck != CFA_NO_CK) {
            const uint4 *v = reinterpret_cast<const uint4 *>(stage + s * kStageBytes);
            for (uint32_t i = threadIdx.x; i < (len >> 4); i += kThreads) acc += vsum<1 << LOG2ES>(v[i]);
        }
        if (threadIdx.x == 0) {
            bulk_store(reinterpret_cast<uint8_t *>(w.dst) + cons.off, stage + s * kStageBytes,
                       len);
            bulk_commit();
            /* the stage loaded next is the one the previous store read from */
            bulk_wait_read_all_but_one();
        }
        /* every thread has finished reading stage s (checksum) before it can be reloaded */
        __syncthreads();
        if (threadIdx.x == 0) issue();
        cons.advance(len, total);
    }
    if (aborted) {
        if (threadIdx.x == 0) {
            atomicCAS(a.status, 0, 2);
            /* loads issued but not consumed: wait for them (bounded) before shared memory goes */
            for (uint32_t c = cons.count; c < prod.count; ++c)
                mbar_wait(&full[c % kStages], (c / kStages) & 1u);
            bulk_wait_all();
        }
        return;
    }
    if (acc_ck != CFA_NO_CK) block_flush(acc, acc_ck, a.ck, red);
    if (threadIdx.x == 0) bulk_wait_all();
}

typedef void (*bulk_fn)(const BulkArgs);
const bulk_fn kBulk[4] = {cfa_bulk_kernel<0>, cfa_bulk_kernel<1>, cfa_bulk_kernel<2>,
                          cfa_bulk_kernel<3>};

} // namespace

/* Resident CTAs per SM of the bulk kernel for element size 2^log2es (0 if it cannot run). */
extern "C" int cfa_bulk_blocks_per_sm(int log2es)
{
    if (log2es < 0 || log2es > 3) return 0;
    if (cudaFuncSetAttribute(kBulk[log2es], cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemBytes) != cudaSuccess)
        return 0;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kBulk[log2es], kThreads, kSmemBytes) !=
        cudaSuccess)
        return 0;
    return n;
}

/* Launches the bulk unpack over items whose source, destination and byte length are multiples
 * of 16; grid_cap bounds the persistent grid. */
extern "C" cudaError_t cfa_launch_bulk(int log2es, const cfa_work *items, uint32_t n_items,
                                       uint64_t src_base, uint64_t src_period,
                                       uint64_t src_lo, uint64_t src_hi,
                                       unsigned long long *ck, int *status, int grid_cap,
                                       cudaStream_t stream)
{
    if (log2es < 0 || log2es > 3 || grid_cap <= 0) return cudaErrorInvalidValue;
    if (n_items == 0) return cudaSuccess;
    BulkArgs a;
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
    kBulk[log2es]<<<grid, kThreads, kSmemBytes, stream>>>(a);
    return cudaGetLastError();
}
