/*
 * TMA bulk-copy unpack: the "InGPU -> Loaded" copy of InstantInfer section 4.2 for large
 * contiguous runs that need no cast and whose source, destination and length are multiples of
 * 16 bytes.  Instead of every thread moving 16-byte vectors through registers, the Tensor
 * Memory Accelerator moves the bytes with non-tensor bulk copies:
 *
 *     global (staging) --cp.async.bulk--> shared stage --cp.async.bulk--> global (destination)
 *
 * Each CTA is two warps over a ring of two 32 KiB stages, three CTAs per SM:
 *   - warp 0 (one lane) loads: it waits until a stage is empty, then issues the bulk load of the
 *     next sub-block into it, completing on the stage's `full` mbarrier (complete_tx);
 *   - warp 1 consumes: it waits on `full`, sums the stage for the per-tensor checksum (all 32
 *     lanes), and one lane issues the bulk store; once the store of the previous sub-block has
 *     finished reading its stage (bulk_group read wait), that stage is released on its `empty`
 *     mbarrier.
 * No block-wide barrier runs inside the loop.  Plain cp.async.bulk only: no tensor maps, no
 * multicast, one CTA's own shared memory.
 *
 * Every wait is bounded: a wait that runs out ends both loops; the CTA then waits (again
 * bounded) for the loads it issued but did not consume, and for its stores, and returns with
 * status word 2, or 3 if that drain ran out as well (a load may then still be in flight into
 * shared memory the CTA no longer owns).
 */
#include <cuda_runtime.h>
#include <stdint.h>

#include "cfa_device.cuh"
#include "cfa_internal.h"

namespace {

using cfa_dev::vsum;
using cfa_dev::warp_sum;

constexpr int kThreads = 64; /* warp 0 loads, warp 1 checksums and stores */
constexpr int kStages = 2;
constexpr uint32_t kStageBytes = 32 * 1024;
constexpr uint32_t kSmemBytes = kStages * kStageBytes; /* 64 KiB: three CTAs per SM */
constexpr uint32_t kSpinLimit = 1u << 20;              /* try_wait polls before giving up */
constexpr uint32_t kLoseLoads = 1u << 31;              /* self-test: the loader issues nothing */

struct BulkArgs {
    const cfa_work *items;
    uint32_t n_items;
    uint32_t spin_limit; /* try_wait polls before a wait gives up; the self-test sets a short one
                            and tells the loader to issue nothing (spin_limit | kLoseLoads) */
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
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, uint32_t limit)
{
    for (uint32_t k = 0; k < limit; ++k)
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

/* Adds the consumer warp's checksum to slot ck; all 32 lanes call it. */
__device__ __forceinline__ void warp_flush(uint64_t &acc, uint32_t ck, unsigned long long *out)
{
    const uint64_t v = warp_sum(acc);
    if ((threadIdx.x & 31) == 0) atomicAdd(out + ck, v);
    acc = 0;
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
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

/* What the consumer needs of a staged sub-block; written by the producer before the load is
 * issued, published to the consumer by the stage's `full` barrier.  len == 0 ends the stream. */
struct StageMeta {
    uint64_t dst;
    uint32_t len;
    uint32_t ck;
};

template <int LOG2ES>
__global__ void __launch_bounds__(kThreads) cfa_bulk_kernel(const BulkArgs a)
{
    extern __shared__ __align__(128) uint8_t stage[];
    __shared__ __align__(8) uint64_t full[kStages];
    __shared__ __align__(8) uint64_t empty[kStages];
    __shared__ StageMeta meta[kStages];
    __shared__ volatile int aborted;
    __shared__ uint32_t n_issued, n_consumed;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        aborted = 0;
        n_issued = 0;
        n_consumed = 0;
    }
    __syncthreads();
    const uint32_t lane = threadIdx.x & 31u;
    const uint32_t limit = a.spin_limit & ~kLoseLoads;

    if (threadIdx.x < 32) {
        /* producer: sub-block p goes to stage p mod kStages once sub-block p - kStages, the
         * stage's previous tenant, has been released.  The next item's descriptor is fetched
         * while the current item's sub-blocks are issued. */
        if (lane == 0) {
            /* item `it` is being issued from w; item it + gridDim.x is in flight into nxt */
            uint32_t it = blockIdx.x, p = 0, off = 0;
            bool have = it < a.n_items;
            cfa_work w{}, nxt{};
            if (have) w = a.items[it];
            uint32_t it_n = it + gridDim.x;
            if (it_n < a.n_items) nxt = a.items[it_n];
            auto step = [&]() { /* move to the next item of this CTA */
                it = it_n;
                have = it < a.n_items;
                if (have) {
                    w = nxt;
                    it_n = it + gridDim.x;
                    if (it_n < a.n_items) nxt = a.items[it_n];
                }
            };
            auto settle = [&]() { /* skip items that fail the checks */
                while (have && !bulk_item_ok<LOG2ES>(w, a)) {
                    atomicCAS(a.status, 0, 1);
                    step();
                }
            };
            settle();
            for (;;) {
                const int s = p % kStages;
                if (a.spin_limit & kLoseLoads) break; /* self-test: nothing arrives on full */
                if (p >= kStages && !mbar_wait(&empty[s], ((p / kStages) - 1u) & 1u, limit)) {
                    aborted = 1;
                    break;
                }
                if (!have || aborted) { /* end marker: a plain arrive completes the phase */
                    meta[s].len = 0;
                    mbar_arrive(&full[s]);
                    break;
                }
                const uint32_t total = w.n << LOG2ES;
                const uint32_t len = min(kStageBytes, total - off);
                meta[s].dst = w.dst + off;
                meta[s].len = len;
                meta[s].ck = w.ck;
                mbar_expect_tx(&full[s], len);
                const uint64_t so = a.src_period ? w.src % a.src_period : w.src;
                bulk_load(stage + s * kStageBytes,
                          reinterpret_cast<const uint8_t *>(a.src_base + so) + off, len,
                          &full[s]);
                ++p;
                n_issued = p;
                off += len;
                if (off >= total) {
                    off = 0;
                    step();
                    settle();
                }
            }
        }
    } else {
        /* consumer: checksum and store sub-block c, then release the stage of c - 1 */
        uint64_t acc = 0;
        uint32_t acc_ck = CFA_NO_CK;
        uint32_t c = 0;
        for (;; ++c) {
            const int s = c % kStages;
            const bool ok = mbar_wait(&full[s], (c / kStages) & 1u, limit);
            if (__any_sync(0xFFFFFFFFu, !ok)) {
                if (lane == 0) aborted = 1;
                break;
            }
            const StageMeta m = meta[s];
            if (m.len == 0) break;
            if (m.ck != acc_ck) {
                if (acc_ck != CFA_NO_CK) warp_flush(acc, acc_ck, a.ck);
                acc_ck = m.ck;
            }
            if (m.ck != CFA_NO_CK) {
                /* eight independent shared loads per lane in flight, then the ragged rest */
                const uint4 *v = reinterpret_cast<const uint4 *>(stage + s * kStageBytes);
                const uint32_t nv = m.len >> 4;
                uint32_t i = lane;
                for (; i + 7 * 32 < nv; i += 8 * 32) {
                    uint4 x[8];
#pragma unroll
                    for (int u = 0; u < 8; ++u) x[u] = v[i + u * 32];
#pragma unroll
                    for (int u = 0; u < 8; ++u) acc += vsum<1 << LOG2ES>(x[u]);
                }
                for (; i < nv; i += 32) acc += vsum<1 << LOG2ES>(v[i]);
            }
            if (lane == 0) {
                bulk_store(reinterpret_cast<uint8_t *>(m.dst), stage + s * kStageBytes, m.len);
                bulk_commit();
                /* the store of c - 1 has read its stage, and every lane finished summing it
                 * before the __syncwarp that ended iteration c - 1 */
                bulk_wait_read_all_but_one();
                if (c >= 1) mbar_arrive(&empty[(c - 1) % kStages]);
            }
            __syncwarp();
        }
        if (acc_ck != CFA_NO_CK) warp_flush(acc, acc_ck, a.ck);
        if (lane == 0) {
            bulk_wait_all();
            n_consumed = c;
        }
    }
    __syncthreads();
    if (aborted && threadIdx.x == 0) {
        /* loads issued but not consumed: wait for them (bounded) before shared memory goes.  If
         * one of these waits runs out too, the CTA leaves with a bulk load that may still write
         * into shared memory it no longer owns: status 3 (over 1 and 2) tells the host that the
         * context is suspect, not merely that a wait timed out */
        bool drained = true;
        for (uint32_t k = n_consumed; k < n_issued && drained; ++k)
            drained = mbar_wait(&full[k % kStages], (k / kStages) & 1u, limit);
        if (drained) atomicCAS(a.status, 0, 2);
        else atomicMax(a.status, 3);
    }
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
    a.spin_limit = kSpinLimit;
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

/* Self-test of the bounded waits: one CTA of the TMA kernel over one valid 16-byte item, with a
 * short wait limit and its loader told to issue nothing, so the consumer's first wait on `full`
 * runs out.  The kernel must flag the status word (2) and return; the context stays usable. */
extern "C" cudaError_t cfa_bulk_selftest_timeout(int *status_host)
{
    cfa_work *d_item = nullptr;
    uint8_t *d_buf = nullptr;
    unsigned long long *d_ck = nullptr;
    int *d_status = nullptr;
    cudaError_t e = cudaSuccess;
    if (!status_host) return cudaErrorInvalidValue;
    *status_host = -1;
    if ((e = cudaFuncSetAttribute(kBulk[1], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kSmemBytes)) != cudaSuccess)
        return e;
    if ((e = cudaMalloc(&d_item, sizeof(cfa_work))) != cudaSuccess) goto out;
    if ((e = cudaMalloc(&d_buf, 512)) != cudaSuccess) goto out;
    if ((e = cudaMalloc(&d_ck, sizeof(unsigned long long))) != cudaSuccess) goto out;
    if ((e = cudaMalloc(&d_status, sizeof(int))) != cudaSuccess) goto out;
    {
        cfa_work w{};
        w.src = 0;
        w.dst = (uint64_t)(uintptr_t)(d_buf + 256);
        w.n = 8; /* 16 bytes of 16-bit elements */
        w.ck = 0;
        w.mode = CFA_MODE(1, 1, 0);
        if ((e = cudaMemcpy(d_item, &w, sizeof w, cudaMemcpyHostToDevice)) != cudaSuccess) goto out;
        if ((e = cudaMemset(d_status, 0, sizeof(int))) != cudaSuccess) goto out;
        if ((e = cudaMemset(d_ck, 0, sizeof(unsigned long long))) != cudaSuccess) goto out;
        BulkArgs a;
        a.items = d_item;
        a.n_items = 1;
        a.spin_limit = 256u | kLoseLoads;
        a.src_base = (uint64_t)(uintptr_t)d_buf;
        a.src_period = 0;
        a.src_lo = 0;
        a.src_hi = 256;
        a.ck = d_ck;
        a.status = d_status;
        kBulk[1]<<<1, kThreads, kSmemBytes>>>(a);
        if ((e = cudaGetLastError()) != cudaSuccess) goto out;
        if ((e = cudaDeviceSynchronize()) != cudaSuccess) goto out;
        e = cudaMemcpy(status_host, d_status, sizeof(int), cudaMemcpyDeviceToHost);
    }
out:
    if (d_item) cudaFree(d_item);
    if (d_buf) cudaFree(d_buf);
    if (d_ck) cudaFree(d_ck);
    if (d_status) cudaFree(d_status);
    return e;
}
