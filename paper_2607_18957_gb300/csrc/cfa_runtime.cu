/*
 * Runtime of the loader: the C ABI of cfa.h on top of the host plan (cfa_plan.c) and the unpack
 * kernels (cfa_unpack.cu).
 *
 * InstantInfer section 4.2 runs each chunk through InDisk -> InMem -> InGPU -> Destroyed with
 *   (i)   (C_i, InMem) -> (C_{i+1}, InDisk) and (C_i, InGPU) -> (C_{i+1}, InMem): one chunk at a
 *         time per data path, the paths overlapping (a two-stage pipeline);
 *   (ii)  (C_i, InGPU) -> (T_j, Alloc): a chunk on the GPU lets its tensors be assembled;
 *   (iii) (T_j, Loaded) -> (C_i, InGPU): a chunk is destroyed once all its tensors are loaded.
 * Here every state transition is a CUDA stream operation and every dependency a CUDA event, all
 * enqueued at once by cfa_load_async, so the host never blocks inside a load:
 *
 *   fill stream   wait(host slot free) -> host function: copy chunk c into pinned slot c mod H
 *                 (pageable or callback sources only) -> record(filled)
 *   copy stream   wait(filled) -> wait(device slot free) -> cudaMemcpyAsync H2D into device slot
 *                 c mod D -> record(host slot free) -> record(h2d done)
 *   caller stream wait(h2d done) -> unpack kernel for chunk c -> record(device slot free)
 *                 -> record(layer l ready) for each readiness group whose last chunk is c
 *
 * Each stream runs one chunk at a time (dependency (i)); the three streams overlap; the slot
 * events carry dependencies (ii) and (iii).  A device source skips staging: its chunks already
 * sit in device memory, and contiguous chunks are unpacked by one launch.
 */
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h> /* header-only; ranges show in profilers that attach to NVTX */

#include <algorithm>
#include <atomic>
#include <chrono>
#include <condition_variable>
#include <cstdarg>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <functional>
#include <memory>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "cfa_internal.h"
#include "cfa_pool.h"

extern "C" int cfa_unpack_blocks_per_sm(int cls);
extern "C" int cfa_bulk_blocks_per_sm(int log2es);
extern "C" int cfa_strided_blocks_per_sm(int cls);
extern "C" cudaError_t cfa_launch_strided(int cls, const cfa_swork *items, uint32_t n_items,
                                          uint64_t src_base, uint64_t src_period,
                                          uint64_t src_lo, uint64_t src_hi,
                                          unsigned long long *ck, int *status, int grid_cap,
                                          cudaStream_t stream);
extern "C" cudaError_t cfa_launch_bulk(int log2es, const cfa_work *items, uint32_t n_items,
                                       uint64_t src_base, uint64_t src_period,
                                       uint64_t src_lo, uint64_t src_hi,
                                       unsigned long long *ck, int *status, int grid_cap,
                                       cudaStream_t stream);
extern "C" cudaError_t cfa_bulk_selftest_timeout(int *status_host);
extern "C" cudaError_t cfa_launch_pull(const void *src, void *dst, uint64_t bytes, int grid,
                                       cudaStream_t stream);
extern "C" cudaError_t cfa_launch_unpack(int cls, const cfa_work *slabs, uint32_t n_slabs,
                                         const cfa_work *tiny, uint32_t n_tiny,
                                         uint64_t src_base, uint64_t src_period,
                                         uint64_t src_lo, uint64_t src_hi,
                                         unsigned long long *ck, int *status, int grid_cap,
                                         int dev_src, cudaStream_t stream);

namespace {

thread_local char g_create_err[512];

struct LoadCtx;

struct FillJob {
    LoadCtx *ctx;
    uint32_t chunk;
    int host_slot;
    std::vector<std::pair<uint64_t, uint64_t>> ranges; /* built by the first fill */
};

struct LoadCtx {
    cfa_plan *plan;
    cfa_source src;
    std::atomic<int> error{0};
    std::vector<FillJob> jobs;
};

struct DeviceGuard {
    int prev = -1;
    bool ok = false;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard()
    {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

/* Bytes of one half of the checksum buffer: a word per entry (at least one) and the status
 * word after them, so that one clear resets both. */
inline size_t ck_clear_bytes(size_t n_entries)
{
    return ((n_entries ? n_entries : 1) + 1) * sizeof(unsigned long long);
}

} // namespace

/* Kernels of one launch group beyond the first run on up to this many side streams. */
constexpr int kSideStreams = 2;

struct cfa_plan {
    cfa_host_plan hp{};
    bool host_only = false;
    int device = 0;
    int pageable_access = 0; /* the device can read pageable host memory in place */
    int grid_cap[CFA_N_CLASSES] = {0};
    int bulk_grid_cap[4] = {0};
    int strided_grid_cap[CFA_N_CLASSES] = {0};
    cfa_work *d_slabs = nullptr, *d_tiny = nullptr, *d_bulk = nullptr;
    cfa_swork *d_strided = nullptr;
    /* Two halves of checksums + status word: a load accumulates into the half cleared before
     * it began and clears the other half, its predecessor's, on ck_stream beside its own work,
     * so no clear sits between a load's start and its first kernel.  d_ck / d_status point into
     * the half of the last load (or of cfa_unpack_chunks_async and cfa_reset_checksums). */
    unsigned long long *d_ck_mem = nullptr;
    size_t ck_half_words = 0;
    int ck_half = 0;
    unsigned long long *d_ck = nullptr;
    int *d_status = nullptr;
    cudaStream_t ck_stream = nullptr;
    cudaEvent_t ev_ck_clear = nullptr;
    uint8_t *d_slots = nullptr;
    bool own_slots = false;
    uint64_t slot_bytes = 0;
    int n_dev_slots = 0;
    uint8_t *h_slots = nullptr;
    int n_host_slots = 0;
    cudaStream_t fill_stream = nullptr, copy_stream = nullptr, aux_stream = nullptr;
    /* side streams that run a launch group's other kernels beside the caller's stream */
    cudaStream_t side_stream[kSideStreams] = {nullptr};
    cudaEvent_t ev_fork = nullptr, ev_join[kSideStreams] = {nullptr};
    /* pinned sources: column slices read in place over the host link, beside the copy ring */
    cudaStream_t direct_stream = nullptr;
    cudaEvent_t ev_direct = nullptr;
    /* segmented plans: the gather callback's stream, and per device slot the event after which
     * the slot holds the whole chunk (the chunk's Gathered state) */
    bool segmented = false;
    cudaStream_t gather_stream = nullptr;
    std::vector<cudaEvent_t> ev_gathered;
    /* staged loads with pull_percent > 0: the SM pull kernel's stream, and per device slot the
     * event after which the pulled part of the chunk is in the slot */
    cudaStream_t pull_stream = nullptr;
    std::vector<cudaEvent_t> ev_pulled;
    int n_sms = 0;
    std::vector<cudaEvent_t> ev_dev_free, ev_h2d, ev_host_free, ev_filled, ev_layer;
    cudaEvent_t ev_begin = nullptr, ev_all = nullptr;
    std::vector<cudaEvent_t> t_h2d0, t_h2d1, t_k0, t_k1;
    std::vector<uint32_t> t_k_c0, t_k_c1; /* chunk range of each timed launch */
    std::vector<std::vector<uint32_t>> layers_ending; /* per chunk */
    /* per chunk: some piece reads it.  A staged load skips the other chunks (no fill, copy,
     * slot or launch), so that a rank's plan, which leaves whole chunks of other ranks'
     * experts unread, keeps its copy stream busy instead of cycling slots through them. */
    std::vector<uint8_t> chunk_busy;
    std::vector<uint32_t> layers_empty;
    std::unique_ptr<cfa::Pool> pool;
    std::vector<std::unique_ptr<LoadCtx>> loads;
    LoadCtx *last = nullptr;
    std::mutex mu;
    char err[512] = {0};
    uint64_t n_loads = 0;
    uint64_t last_launches = 0;
    uint32_t last_h2d = 0;
    double plan_ms = 0;
};

namespace {

/* CFA_LOG=1 in the environment: one line per plan, per load and per error on stderr. */
bool log_on()
{
    static const bool on = [] {
        const char *v = std::getenv("CFA_LOG");
        return v && *v && std::strcmp(v, "0") != 0;
    }();
    return on;
}

void logf(const char *fmt, ...)
{
    if (!log_on()) return;
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    std::fprintf(stderr, "cfa: %s\n", buf);
}

void set_err(cfa_plan *p, const char *fmt, ...)
{
    char *buf = p ? p->err : g_create_err;
    size_t n = p ? sizeof(p->err) : sizeof(g_create_err);
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, n, fmt, ap);
    va_end(ap);
    logf("error: %s", buf);
}

#define CK(p, call)                                                                        \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess) {                                                           \
            set_err((p), "%s failed: %s", #call, cudaGetErrorString(e_));                  \
            return CFA_ERR_CUDA;                                                           \
        }                                                                                  \
    } while (0)

/* NVTX range for the lifetime of a scope. */
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

/* InDisk -> InMem for one chunk: puts the byte ranges the chunk's pieces read (its copy
 * segments; the rest of the slot is never read) into pinned slot `host_slot`, split over the
 * plan's fill threads in parts of at most 1 MiB. */
void CUDART_CB fill_host_fn(void *arg)
{
    FillJob *j = static_cast<FillJob *>(arg);
    LoadCtx *ctx = j->ctx;
    cfa_plan *p = ctx->plan;
    if (ctx->error.load()) return;
    NvtxRange range("cfa fill chunk (InDisk -> InMem)");
    const cfa_host_plan &hp = p->hp;
    const uint64_t S = hp.chunk_bytes;
    const uint64_t off = (uint64_t)j->chunk * S;
    uint8_t *dst = p->h_slots + (uint64_t)j->host_slot * S;
    const cfa_source &src = ctx->src;
    /* the byte ranges, as (offset in chunk, length): a 2-D segment gives one per row, and
     * long ranges are cut into 1 MiB pieces so that every fill thread gets a share even when a
     * chunk holds only a few of them (a tensor-parallel shard) */
    std::vector<std::pair<uint64_t, uint64_t>> &ranges = j->ranges;
    if (ranges.empty()) {
        const uint64_t part = 1ull << 20;
        for (uint32_t k = hp.copy_first[j->chunk]; k < hp.copy_first[j->chunk + 1]; ++k) {
            const cfa_copy &cp = hp.copies[k];
            for (uint64_t r = 0; r < cp.rows; ++r)
                for (uint64_t a = 0; a < cp.width; a += part)
                    ranges.emplace_back(cp.src - off + r * cp.pitch + a,
                                        std::min<uint64_t>(part, cp.width - a));
        }
    }
    const int nparts = (int)std::min<size_t>(ranges.size(), 4096);
    const size_t per = (ranges.size() + (size_t)nparts - 1) / (size_t)(nparts ? nparts : 1);
    p->pool->run(nparts, [&](int k) {
        for (size_t q = (size_t)k * per; q < ranges.size() && q < (size_t)(k + 1) * per; ++q) {
            const uint64_t a = ranges[q].first, len = ranges[q].second;
            if (src.kind == CFA_SRC_HOST) {
                const uint64_t so = src.period_bytes ? (off % src.period_bytes) : off;
                std::memcpy(dst + a, static_cast<const uint8_t *>(src.base) + so + a, len);
            } else if (src.fill(src.user, off + a, dst + a, len) != 0) {
                int zero = 0;
                ctx->error.compare_exchange_strong(zero, CFA_ERR_SOURCE);
                return;
            }
        }
    });
}

/* Unpacks chunks [c0, c1), whose blob byte o sits at device address src_base + o (or
 * src_base + (o mod period) for a periodic source): per work class present in those chunks
 * (normally one), a TMA bulk launch for its aligned cast-free slabs, a launch for its column
 * slices and a vector launch for everything else.  The kernels of one group write disjoint
 * destination bytes and add their checksums atomically, so they are independent: the first
 * runs on `s`, the others on side streams forked from `s` and joined back into it, so that
 * one kernel's last CTAs overlap the next kernel's first instead of the GPU draining between
 * them.  With tma = false (a source in host memory, read over the host link) the aligned slabs
 * planned for the TMA kernel are copied by the vector kernel instead: bulk copies are for
 * device memory.  grid_div > 1 divides every kernel's grid cap by it. */
enum { LAUNCH_CONTIG = 1, LAUNCH_STRIDED = 2, LAUNCH_ALL = 3 };

cfa_status launch(cfa_plan *p, uint32_t c0, uint32_t c1, uint64_t src_base, uint64_t period,
                  cudaStream_t s, bool tma = true, int what = LAUNCH_ALL, int grid_div = 1)
{
    auto cap = [grid_div](int c) { return std::max(1, c / grid_div); };
    const cfa_host_plan &hp = p->hp;
    const uint64_t lo = (uint64_t)c0 * hp.chunk_bytes;
    const uint64_t hi = std::min<uint64_t>(hp.blob_bytes, (uint64_t)c1 * hp.chunk_bytes);
    const size_t row = (size_t)hp.n_chunks + 1;
    const bool timing_on = (hp.opts.flags & CFA_OPT_TIMING) != 0;
    enum { BULK, BULK_AS_VECTOR, STRIDED, VECTOR };
    struct Job {
        int type, k;
        uint32_t a0, a1, b0, b1;
    };
    Job jobs[3 * CFA_N_CLASSES];
    int n = 0;
    for (int k = 0; k < CFA_N_CLASSES && hp.n_bulk && (what & LAUNCH_CONTIG); ++k) {
        const uint32_t b0 = hp.bulk_first[k * row + c0], b1 = hp.bulk_first[k * row + c1];
        if (b1 != b0) jobs[n++] = Job{tma ? BULK : BULK_AS_VECTOR, k, b0, b1, 0, 0};
    }
    for (int k = 0; k < CFA_N_CLASSES && hp.n_strided && (what & LAUNCH_STRIDED); ++k) {
        const uint32_t r0 = hp.strided_first[k * row + c0], r1 = hp.strided_first[k * row + c1];
        if (r1 != r0) jobs[n++] = Job{STRIDED, k, r0, r1, 0, 0};
    }
    for (int k = 0; k < CFA_N_CLASSES && (what & LAUNCH_CONTIG); ++k) {
        const uint32_t s0 = hp.slab_first[k * row + c0], s1 = hp.slab_first[k * row + c1];
        const uint32_t t0 = hp.tiny_first[k * row + c0], t1 = hp.tiny_first[k * row + c1];
        if (s1 != s0 || t1 != t0) jobs[n++] = Job{VECTOR, k, s0, s1, t0, t1};
    }
    const int n_side = std::min(n - 1, kSideStreams);
    if (n_side > 0) {
        CK(p, cudaEventRecord(p->ev_fork, s));
        for (int j = 0; j < n_side; ++j) CK(p, cudaStreamWaitEvent(p->side_stream[j], p->ev_fork, 0));
    }
    for (int i = 0; i < n; ++i) {
        const Job &J = jobs[i];
        const int k = J.k;
        cudaStream_t ls = i == 0 ? s : p->side_stream[(i - 1) % kSideStreams];
        const bool timing = timing_on && p->last_launches < p->t_k0.size();
        if (timing) {
            CK(p, cudaEventRecord(p->t_k0[p->last_launches], ls));
            p->t_k_c0[p->last_launches] = c0;
            p->t_k_c1[p->last_launches] = c1;
        }
        if (J.type == BULK)
            CK(p, cfa_launch_bulk(k, p->d_bulk + J.a0, J.a1 - J.a0, src_base, period, lo, hi,
                                  p->d_ck, p->d_status, cap(p->bulk_grid_cap[k]), ls));
        else if (J.type == BULK_AS_VECTOR) /* bulk items are copy-class slabs of class k */
            CK(p, cfa_launch_unpack(k, p->d_bulk + J.a0, J.a1 - J.a0, nullptr, 0, src_base,
                                    period, lo, hi, p->d_ck, p->d_status, cap(p->grid_cap[k]),
                                    tma, ls));
        else if (J.type == STRIDED)
            CK(p, cfa_launch_strided(k, p->d_strided + J.a0, J.a1 - J.a0, src_base, period, lo,
                                     hi, p->d_ck, p->d_status, cap(p->strided_grid_cap[k]), ls));
        else
            CK(p, cfa_launch_unpack(k, p->d_slabs + J.a0, J.a1 - J.a0, p->d_tiny + J.b0,
                                    J.b1 - J.b0, src_base, period, lo, hi, p->d_ck, p->d_status,
                                    cap(p->grid_cap[k]), tma, ls));
        if (timing) CK(p, cudaEventRecord(p->t_k1[p->last_launches], ls));
        p->last_launches++;
    }
    for (int j = 0; j < n_side; ++j) {
        CK(p, cudaEventRecord(p->ev_join[j], p->side_stream[j]));
        CK(p, cudaStreamWaitEvent(s, p->ev_join[j], 0));
    }
    return CFA_OK;
}

cfa_status record_layers(cfa_plan *p, uint32_t c0, uint32_t c1, cudaStream_t s)
{
    for (uint32_t c = c0; c < c1; ++c)
        for (uint32_t l : p->layers_ending[c]) CK(p, cudaEventRecord(p->ev_layer[l], s));
    return CFA_OK;
}

cfa_status make_event(cfa_plan *p, cudaEvent_t *ev, bool timing)
{
    CK(p, cudaEventCreateWithFlags(ev, timing ? cudaEventDefault : cudaEventDisableTiming));
    return CFA_OK;
}

/* Points d_ck / d_status at half h of the checksum buffer. */
void use_ck_half(cfa_plan *p, int h)
{
    p->ck_half = h;
    p->d_ck = p->d_ck_mem + (size_t)h * p->ck_half_words;
    p->d_status = reinterpret_cast<int *>(p->d_ck + (p->ck_half_words - 1));
}

void release(cfa_plan *p)
{
    if (!p) return;
    if (!p->host_only) {
        DeviceGuard g(p->device);
        if (p->fill_stream) cudaStreamSynchronize(p->fill_stream);
        if (p->copy_stream) cudaStreamSynchronize(p->copy_stream);
        if (p->ev_all) cudaEventSynchronize(p->ev_all);
        if (p->aux_stream) cudaStreamSynchronize(p->aux_stream);
        if (p->ck_stream) cudaStreamSynchronize(p->ck_stream);
        auto kill = [](std::vector<cudaEvent_t> &v) {
            for (cudaEvent_t e : v)
                if (e) cudaEventDestroy(e);
            v.clear();
        };
        if (p->gather_stream) cudaStreamSynchronize(p->gather_stream);
        if (p->pull_stream) cudaStreamSynchronize(p->pull_stream);
        kill(p->ev_pulled);
        kill(p->ev_dev_free);
        kill(p->ev_h2d);
        kill(p->ev_gathered);
        kill(p->ev_host_free);
        kill(p->ev_filled);
        kill(p->ev_layer);
        kill(p->t_h2d0);
        kill(p->t_h2d1);
        kill(p->t_k0);
        kill(p->t_k1);
        if (p->ev_begin) cudaEventDestroy(p->ev_begin);
        if (p->ev_all) cudaEventDestroy(p->ev_all);
        if (p->ev_fork) cudaEventDestroy(p->ev_fork);
        if (p->ev_ck_clear) cudaEventDestroy(p->ev_ck_clear);
        if (p->ck_stream) cudaStreamDestroy(p->ck_stream);
        if (p->direct_stream) cudaStreamSynchronize(p->direct_stream);
        if (p->ev_direct) cudaEventDestroy(p->ev_direct);
        if (p->direct_stream) cudaStreamDestroy(p->direct_stream);
        for (int j = 0; j < kSideStreams; ++j) {
            if (p->side_stream[j]) cudaStreamSynchronize(p->side_stream[j]);
            if (p->ev_join[j]) cudaEventDestroy(p->ev_join[j]);
            if (p->side_stream[j]) cudaStreamDestroy(p->side_stream[j]);
        }
        if (p->fill_stream) cudaStreamDestroy(p->fill_stream);
        if (p->copy_stream) cudaStreamDestroy(p->copy_stream);
        if (p->gather_stream) cudaStreamDestroy(p->gather_stream);
        if (p->pull_stream) cudaStreamDestroy(p->pull_stream);
        if (p->aux_stream) cudaStreamDestroy(p->aux_stream);
        if (p->d_slabs) cudaFree(p->d_slabs);
        if (p->d_tiny) cudaFree(p->d_tiny);
        if (p->d_bulk) cudaFree(p->d_bulk);
        if (p->d_strided) cudaFree(p->d_strided);
        if (p->d_ck_mem) cudaFree(p->d_ck_mem);
        if (p->own_slots && p->d_slots) cudaFree(p->d_slots);
        if (p->h_slots) cudaFreeHost(p->h_slots);
    }
    p->pool.reset();
    cfa_host_plan_free(&p->hp);
    delete p;
}

cfa_status setup_device(cfa_plan *p)
{
    cfa_host_plan &hp = p->hp;
    const cfa_plan_opts &o = hp.opts;
    if (o.device >= 0) p->device = o.device;
    else CK(nullptr, cudaGetDevice(&p->device));
    DeviceGuard g(p->device);
    if (!g.ok) {
        set_err(nullptr, "cannot select CUDA device %d", p->device);
        return CFA_ERR_CUDA;
    }
    int sms = 0;
    CK(nullptr, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, p->device));
    p->n_sms = sms;
    CK(nullptr, cudaDeviceGetAttribute(&p->pageable_access, cudaDevAttrPageableMemoryAccess,
                                       p->device));
    for (int k = 0; k < CFA_N_CLASSES; ++k) {
        const int per_sm = cfa_unpack_blocks_per_sm(k);
        if (sms <= 0 || per_sm <= 0) {
            set_err(nullptr, "unpack kernel %d cannot run on device %d (sm=%d, blocks/sm=%d)", k,
                    p->device, sms, per_sm);
            return CFA_ERR_CUDA;
        }
        p->grid_cap[k] = sms * per_sm;
    }
    for (int k = 0; k < CFA_N_CLASSES && hp.n_strided; ++k) {
        const int per_sm = cfa_strided_blocks_per_sm(k);
        if (per_sm <= 0) {
            set_err(nullptr, "strided kernel %d cannot run on device %d", k, p->device);
            return CFA_ERR_CUDA;
        }
        p->strided_grid_cap[k] = sms * per_sm;
    }
    if (hp.n_bulk) {
        for (int k = 0; k < 4; ++k) {
            const int per_sm = cfa_bulk_blocks_per_sm(k);
            if (per_sm <= 0) {
                set_err(nullptr, "bulk kernel %d cannot run on device %d", k, p->device);
                return CFA_ERR_CUDA;
            }
            p->bulk_grid_cap[k] = sms * per_sm;
        }
    }

    auto upload = [&](cfa_work **d, const cfa_work *h, size_t n) -> cfa_status {
        const size_t bytes = (n ? n : 1) * sizeof(cfa_work);
        if (cudaMalloc(d, bytes) != cudaSuccess) {
            set_err(nullptr, "cudaMalloc of %zu descriptor bytes failed", bytes);
            return CFA_ERR_NOMEM;
        }
        if (n) CK(nullptr, cudaMemcpy(*d, h, n * sizeof(cfa_work), cudaMemcpyHostToDevice));
        return CFA_OK;
    };
    cfa_status st = upload(&p->d_slabs, hp.slabs, hp.n_slabs);
    if (st) return st;
    st = upload(&p->d_tiny, hp.tiny, hp.n_tiny);
    if (st) return st;
    st = upload(&p->d_bulk, hp.bulk, hp.n_bulk);
    if (st) return st;
    {
        const size_t bytes = (hp.n_strided ? hp.n_strided : 1) * sizeof(cfa_swork);
        if (cudaMalloc(&p->d_strided, bytes) != cudaSuccess) {
            set_err(nullptr, "cudaMalloc of %zu descriptor bytes failed", bytes);
            return CFA_ERR_NOMEM;
        }
        if (hp.n_strided)
            CK(nullptr, cudaMemcpy(p->d_strided, hp.strided, hp.n_strided * sizeof(cfa_swork),
                                   cudaMemcpyHostToDevice));
    }
    /* two halves of checksums with the status word after them: one clear resets both */
    const size_t ck_bytes = ck_clear_bytes(hp.n_entries);
    p->ck_half_words = ck_bytes / sizeof(unsigned long long);
    if (cudaMalloc(&p->d_ck_mem, 2 * ck_bytes) != cudaSuccess) {
        set_err(nullptr, "cudaMalloc of the checksum buffer failed");
        return CFA_ERR_NOMEM;
    }
    CK(nullptr, cudaMemset(p->d_ck_mem, 0, 2 * ck_bytes));
    use_ck_half(p, 0);

    p->n_dev_slots = o.dev_slots;
    p->n_host_slots = o.host_slots;
    /* a segmented plan's gather fills all seg_world segments of the slot, chunk_bytes in all,
     * even for a blob shorter than one chunk */
    p->slot_bytes = p->segmented ? hp.chunk_bytes
                                 : std::min<uint64_t>(hp.chunk_bytes,
                                                      (hp.blob_bytes + 255) / 256 * 256);
    if (p->n_dev_slots > 0 && p->slot_bytes > 0) {
        if (o.workspace) {
            p->d_slots = static_cast<uint8_t *>(o.workspace);
        } else {
            if (cudaMalloc(&p->d_slots, (uint64_t)p->n_dev_slots * p->slot_bytes) !=
                cudaSuccess) {
                cudaGetLastError();
                set_err(nullptr, "cudaMalloc of %d staging slots of %llu bytes failed",
                        p->n_dev_slots, (unsigned long long)p->slot_bytes);
                return CFA_ERR_NOMEM;
            }
            p->own_slots = true;
        }
    }
    CK(nullptr, cudaStreamCreateWithFlags(&p->fill_stream, cudaStreamNonBlocking));
    CK(nullptr, cudaStreamCreateWithFlags(&p->copy_stream, cudaStreamNonBlocking));
    CK(nullptr, cudaStreamCreateWithFlags(&p->aux_stream, cudaStreamNonBlocking));
    CK(nullptr, cudaStreamCreateWithFlags(&p->ck_stream, cudaStreamNonBlocking));
    if ((st = make_event(nullptr, &p->ev_ck_clear, false))) return st;
    for (int j = 0; j < kSideStreams; ++j) {
        CK(nullptr, cudaStreamCreateWithFlags(&p->side_stream[j], cudaStreamNonBlocking));
        if ((st = make_event(nullptr, &p->ev_join[j], false))) return st;
    }
    if ((st = make_event(nullptr, &p->ev_fork, false))) return st;
    CK(nullptr, cudaStreamCreateWithFlags(&p->direct_stream, cudaStreamNonBlocking));
    if ((st = make_event(nullptr, &p->ev_direct, false))) return st;
    const bool timing = (o.flags & CFA_OPT_TIMING) != 0;
    auto events = [&](std::vector<cudaEvent_t> &v, size_t n, bool t) -> cfa_status {
        v.assign(n, nullptr);
        for (auto &e : v) {
            cfa_status s = make_event(nullptr, &e, t);
            if (s) return s;
        }
        return CFA_OK;
    };
    if ((st = events(p->ev_dev_free, p->n_dev_slots, false))) return st;
    if ((st = events(p->ev_h2d, p->n_dev_slots, false))) return st;
    if (p->segmented) {
        CK(nullptr, cudaStreamCreateWithFlags(&p->gather_stream, cudaStreamNonBlocking));
        if ((st = events(p->ev_gathered, p->n_dev_slots, false))) return st;
    }
    if (o.pull_percent > 0 && !p->segmented && p->n_dev_slots > 0) {
        CK(nullptr, cudaStreamCreateWithFlags(&p->pull_stream, cudaStreamNonBlocking));
        if ((st = events(p->ev_pulled, p->n_dev_slots, false))) return st;
    }
    if ((st = events(p->ev_host_free, p->n_host_slots, false))) return st;
    if ((st = events(p->ev_filled, p->n_host_slots, false))) return st;
    if ((st = events(p->ev_layer, hp.n_layers, timing))) return st;
    if ((st = make_event(nullptr, &p->ev_begin, timing))) return st;
    if ((st = make_event(nullptr, &p->ev_all, timing))) return st;
    if (timing) {
        if ((st = events(p->t_h2d0, hp.n_chunks, true))) return st;
        if ((st = events(p->t_h2d1, hp.n_chunks, true))) return st;
        const size_t nk = 3 * CFA_N_CLASSES * ((size_t)hp.n_chunks + 1);
        if ((st = events(p->t_k0, nk, true))) return st;
        if ((st = events(p->t_k1, nk, true))) return st;
        p->t_k_c0.assign(nk, 0);
        p->t_k_c1.assign(nk, 0);
    }
    if (o.fill_threads > 1) p->pool.reset(new cfa::Pool(o.fill_threads - 1));
    else p->pool.reset(new cfa::Pool(0));
    return CFA_OK;
}

cfa_status check_status_word(cfa_plan *p)
{
    int h = 0;
    CK(p, cudaStreamWaitEvent(p->aux_stream, p->ev_all, 0));
    CK(p, cudaMemcpyAsync(&h, p->d_status, sizeof(int), cudaMemcpyDeviceToHost, p->aux_stream));
    CK(p, cudaStreamSynchronize(p->aux_stream));
    if (h == 3) {
        set_err(p, "a TMA bulk-copy wait ran out and so did the wait for the CTA's own loads in "
                   "flight (status word 3): treat the CUDA context as suspect");
        return CFA_ERR_SUSPECT;
    }
    if (h) {
        set_err(p, h == 2 ? "a TMA bulk-copy wait ran out (status word 2)"
                          : "the unpack kernel rejected a work item outside its chunk or of the "
                            "wrong class (status word %d)",
                h);
        return CFA_ERR_DEVICE;
    }
    return CFA_OK;
}

/* Polls `ev` from the host, sleeping between queries, until it completes or timeout_ns passes
 * (timeout_ns < 0: no limit).  The sleep doubles from 2 us up to kPollSleepMaxUs, so a load is
 * noticed within about that much (plus the thread's timer slack) of its end: a 1 ms cap cost
 * the end-to-end figure of a 76 ms load a whole millisecond. */
constexpr int64_t kPollSleepMaxUs = 50;

cfa_status wait_event_host(cfa_plan *p, cudaEvent_t ev, int64_t timeout_ns)
{
    const auto t0 = std::chrono::steady_clock::now();
    int64_t sleep_us = 2;
    for (;;) {
        const cudaError_t q = cudaEventQuery(ev);
        if (q == cudaSuccess) return CFA_OK;
        if (q != cudaErrorNotReady) {
            set_err(p, "cudaEventQuery failed: %s", cudaGetErrorString(q));
            return CFA_ERR_CUDA;
        }
        if (timeout_ns >= 0) {
            const int64_t el = std::chrono::duration_cast<std::chrono::nanoseconds>(
                                   std::chrono::steady_clock::now() - t0)
                                   .count();
            if (el >= timeout_ns) {
                set_err(p, "wait timed out after %lld ns", (long long)timeout_ns);
                return CFA_ERR_TIMEOUT;
            }
        }
        std::this_thread::sleep_for(std::chrono::microseconds(sleep_us));
        sleep_us = std::min<int64_t>(sleep_us * 2, kPollSleepMaxUs);
    }
}

} // namespace

extern "C" {

cfa_status cfa_plan_create(const cfa_tensor_entry *entries, size_t n_entries,
                           const cfa_dst *dsts, size_t n_dsts, uint64_t blob_bytes,
                           const cfa_plan_opts *opts, cfa_plan **out)
{
    if (!out) {
        set_err(nullptr, "out is NULL");
        return CFA_ERR_INVAL;
    }
    *out = nullptr;
    NvtxRange range("cfa plan create");
    const auto t0 = std::chrono::steady_clock::now();
    cfa_plan *p = new (std::nothrow) cfa_plan();
    if (!p) {
        set_err(nullptr, "out of host memory");
        return CFA_ERR_NOMEM;
    }
    cfa_status st = cfa_host_plan_build(entries, n_entries, dsts, n_dsts, blob_bytes, opts,
                                        &p->hp, g_create_err, sizeof(g_create_err));
    if (st) {
        logf("error: %s", g_create_err);
        delete p;
        return st;
    }
    const cfa_host_plan &hp = p->hp;
    p->host_only = (hp.opts.flags & CFA_OPT_HOST_ONLY) != 0;
    p->layers_ending.assign(hp.n_chunks, {});
    for (uint32_t l = 0; l < hp.n_layers; ++l) {
        if (hp.layer_last_chunk[l] < 0) p->layers_empty.push_back(l);
        else p->layers_ending[(size_t)hp.layer_last_chunk[l]].push_back(l);
    }
    p->segmented = hp.opts.seg_world > 1;
    /* a segmented load takes every chunk: each rank must issue the same gathers */
    p->chunk_busy.assign(hp.n_chunks, p->segmented ? 1 : 0);
    for (size_t i = 0; i < hp.n_pieces; ++i) p->chunk_busy[hp.pieces[i].chunk] = 1;
    if (!p->host_only) {
        st = setup_device(p);
        if (st) {
            char keep[sizeof(g_create_err)];
            std::memcpy(keep, g_create_err, sizeof keep);
            release(p);
            std::memcpy(g_create_err, keep, sizeof keep);
            return st;
        }
    }
    p->plan_ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0)
                     .count();
    logf("plan: %zu entries, %zu destinations, %llu blob bytes in %u chunks of %llu; pieces %zu, "
         "TMA items %zu, vector slabs %zu, tiny %zu, column blocks %zu; staged bytes %llu; "
         "%.1f ms",
         hp.n_entries, hp.n_dsts, (unsigned long long)hp.blob_bytes, hp.n_chunks,
         (unsigned long long)hp.chunk_bytes, hp.n_pieces, hp.n_bulk, hp.n_slabs, hp.n_tiny,
         hp.n_strided, (unsigned long long)hp.staged_bytes, p->plan_ms);
    *out = p;
    return CFA_OK;
}

cfa_status cfa_load_async(cfa_plan *p, const cfa_source *src, cfa_stream stream_)
{
    if (!p || !src) return CFA_ERR_INVAL;
    NvtxRange range("cfa enqueue load");
    if (p->host_only) {
        set_err(p, "host-only plan cannot load");
        return CFA_ERR_INVAL;
    }
    std::unique_lock<std::mutex> lk(p->mu, std::try_to_lock);
    if (!lk.owns_lock()) {
        set_err(p, "plan in use by another thread");
        return CFA_ERR_BUSY;
    }
    const cfa_host_plan &hp = p->hp;
    const uint64_t S = hp.chunk_bytes;
    const int kind = src->kind;
    if (kind < CFA_SRC_HOST || kind > CFA_SRC_HOST_DIRECT || src->reserved) {
        set_err(p, "unknown source kind %d", kind);
        return CFA_ERR_INVAL;
    }
    if (src->period_bytes && (src->period_bytes % S != 0 || kind == CFA_SRC_CALLBACK)) {
        set_err(p, "period_bytes must be a multiple of chunk_bytes (not for callbacks)");
        return CFA_ERR_INVAL;
    }
    if (kind == CFA_SRC_CALLBACK ? !src->fill : (!src->base && hp.blob_bytes)) {
        set_err(p, "source has no base pointer or fill function");
        return CFA_ERR_INVAL;
    }
    if (kind != CFA_SRC_CALLBACK && src->size_bytes) {
        const uint64_t need = src->period_bytes ? std::min(src->period_bytes, hp.blob_bytes)
                                                : hp.blob_bytes;
        if (need > src->size_bytes) {
            set_err(p, "the plan reads %llu bytes of the source, which holds %llu",
                    (unsigned long long)need, (unsigned long long)src->size_bytes);
            return CFA_ERR_INVAL;
        }
    }
    if (kind == CFA_SRC_HOST_DIRECT && ((uintptr_t)src->base & 7u)) {
        set_err(p, "direct host sources must be 8-byte aligned");
        return CFA_ERR_ALIGN;
    }
    if ((kind == CFA_SRC_PINNED || kind == CFA_SRC_DEVICE) && ((uintptr_t)src->base & 255u)) {
        set_err(p, "pinned and device sources must be 256-byte aligned");
        return CFA_ERR_ALIGN;
    }
    /* a pageable source on a device that reads pageable memory, with the pull path on: the pull
     * kernel reads it straight into the device slots (no fill threads, no pinned host slots,
     * no host memcpy); the copy engine cannot read pageable memory without blocking the call,
     * so it takes no share, and column slices are read in place by their kernel */
    const bool host_pull = kind == CFA_SRC_HOST && p->pull_stream && hp.opts.pull_percent > 0 &&
                           p->pageable_access && ((uintptr_t)src->base & 15u) == 0;
    const bool staged = (kind == CFA_SRC_HOST && !host_pull) || kind == CFA_SRC_CALLBACK;
    const bool in_place = kind == CFA_SRC_DEVICE || kind == CFA_SRC_HOST_DIRECT;
    if (p->segmented && in_place) {
        set_err(p, "a segmented plan loads from HOST, PINNED or CALLBACK sources only");
        return CFA_ERR_INVAL;
    }
    if (kind == CFA_SRC_HOST_DIRECT && hp.blob_bytes) {
        /* page-locked memory is mapped for the device; pageable memory is readable in place
         * only where the device shares the host's page tables */
        cudaPointerAttributes at;
        std::memset(&at, 0, sizeof at);
        if (cudaPointerGetAttributes(&at, src->base) != cudaSuccess) {
            cudaGetLastError();
            at.type = cudaMemoryTypeUnregistered;
        }
        const bool mapped = at.type == cudaMemoryTypeHost || at.type == cudaMemoryTypeManaged;
        if (!mapped && !p->pageable_access) {
            set_err(p, "this device cannot read pageable host memory in place; use a HOST "
                       "source or page-locked memory");
            return CFA_ERR_INVAL;
        }
    }
    if (!in_place && hp.n_chunks && (p->n_dev_slots == 0 || !p->d_slots)) {
        set_err(p, "plan has no device staging slots (dev_slots = 0)");
        return CFA_ERR_INVAL;
    }
    if (staged && hp.n_chunks && p->n_host_slots == 0) {
        set_err(p, "plan has no pinned host slots (host_slots = 0)");
        return CFA_ERR_INVAL;
    }
    DeviceGuard g(p->device);
    cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream_);

    /* contexts of loads that have fully completed are no longer referenced by host functions */
    if (!p->loads.empty() && cudaEventQuery(p->ev_all) == cudaSuccess &&
        cudaStreamQuery(p->fill_stream) == cudaSuccess)
        p->loads.clear();
    if (staged && hp.n_chunks && !p->h_slots) {
        if (cudaHostAlloc(&p->h_slots, (uint64_t)p->n_host_slots * S, cudaHostAllocDefault) !=
            cudaSuccess) {
            cudaGetLastError();
            p->h_slots = nullptr;
            set_err(p, "cudaHostAlloc of %d pinned slots of %llu bytes failed", p->n_host_slots,
                    (unsigned long long)S);
            return CFA_ERR_NOMEM;
        }
    }
    std::unique_ptr<LoadCtx> ctx(new (std::nothrow) LoadCtx());
    if (!ctx) return CFA_ERR_NOMEM;
    ctx->plan = p;
    ctx->src = *src;
    if (staged) {
        ctx->jobs.resize(hp.n_chunks);
        uint32_t k = 0; /* busy chunks take the pinned slots in turn */
        for (uint32_t c = 0; c < hp.n_chunks; ++c)
            ctx->jobs[c] = FillJob{ctx.get(), c,
                                   p->chunk_busy[c] ? (int)(k++ % (uint32_t)p->n_host_slots) : -1,
                                   {}};
    }
    LoadCtx *cx = ctx.get();
    p->loads.push_back(std::move(ctx));
    p->last = cx;
    p->n_loads++;
    p->last_launches = 0;
    p->last_h2d = 0;
    const bool timing = (hp.opts.flags & CFA_OPT_TIMING) != 0;

    /* the load starts after the previous load of this plan, after prior work on cs and after
     * the clear of the checksum half it takes; it clears the other half for the next load */
    CK(p, cudaStreamWaitEvent(cs, p->ev_all, 0));
    CK(p, cudaStreamWaitEvent(cs, p->ev_ck_clear, 0));
    CK(p, cudaEventRecord(p->ev_begin, cs));
    CK(p, cudaStreamWaitEvent(p->fill_stream, p->ev_begin, 0));
    CK(p, cudaStreamWaitEvent(p->copy_stream, p->ev_begin, 0));
    {
        /* the half the previous load used is cleared for the next load; this load switches to
         * the other one only once that clear is enqueued, so a load that fails here leaves the
         * clean half for the next */
        unsigned long long *prev = p->d_ck;
        CK(p, cudaStreamWaitEvent(p->ck_stream, p->ev_begin, 0));
        if (hp.any_cksum)
            CK(p, cudaMemsetAsync(prev, 0, ck_clear_bytes(hp.n_entries), p->ck_stream));
        else
            CK(p, cudaMemsetAsync(prev + (p->ck_half_words - 1), 0, sizeof(int), p->ck_stream));
        CK(p, cudaEventRecord(p->ev_ck_clear, p->ck_stream));
        use_ck_half(p, p->ck_half ^ 1);
    }
    for (uint32_t l : p->layers_empty) CK(p, cudaEventRecord(p->ev_layer[l], cs));

    if (in_place) {
        /* the kernel reads the blob where it is: device memory (one launch over all chunks per
         * work class, or one per chunk with CFA_OPT_NO_MERGE) or host memory over the host link
         * (one launch per chunk, so readiness events follow the stream of chunks) */
        const uint64_t base = (uint64_t)(uintptr_t)src->base;
        const uint32_t per_run =
            (kind == CFA_SRC_HOST_DIRECT || (hp.opts.flags & CFA_OPT_NO_MERGE)) ? 1u
                                                                                 : hp.n_chunks;
        for (uint32_t c0 = 0; c0 < hp.n_chunks;) {
            const uint32_t c1 = std::min<uint32_t>(hp.n_chunks, c0 + per_run);
            cfa_status st =
                launch(p, c0, c1, base, src->period_bytes, cs, kind == CFA_SRC_DEVICE);
            if (st) return st;
            if ((st = record_layers(p, c0, c1, cs))) return st;
            c0 = c1;
        }
    } else {
        /* A pinned source is readable by the GPU in place, so its column slices need not go
         * through the slots as strided 2-D copies (slower than plain copies on the copy engine):
         * the column-slice kernels read them over the host link on the direct stream, in chunk
         * order and ahead of the copy ring, and each chunk's readiness also waits for them. */
        const bool slices_in_place =
            ((kind == CFA_SRC_PINNED && !(hp.opts.flags & CFA_OPT_STAGE_SLICES)) || host_pull) &&
            hp.n_strided && !p->segmented;
        const uint64_t seg_bytes = p->segmented ? S / (uint64_t)hp.opts.seg_world : 0;
        cfa_status gather_failed = CFA_OK;
        const size_t row = (size_t)hp.n_chunks + 1;
        auto has_slices = [&](uint32_t c) {
            for (int k = 0; k < CFA_N_CLASSES; ++k)
                if (hp.strided_first[k * row + c + 1] != hp.strided_first[k * row + c])
                    return true;
            return false;
        };
        if (slices_in_place) CK(p, cudaStreamWaitEvent(p->direct_stream, p->ev_begin, 0));
        /* the SM pull path: a share of each contiguous range goes to the pull kernel on the
         * pull stream, the rest to the copy engine; the device must be able to read the host
         * memory the chunk comes from (page-locked memory, or any memory with pageable access) */
        bool pull_on = p->pull_stream != nullptr && hp.opts.pull_percent > 0;
        if (pull_on && kind == CFA_SRC_PINNED && !p->pageable_access) {
            cudaPointerAttributes at;
            std::memset(&at, 0, sizeof at);
            if (cudaPointerGetAttributes(&at, src->base) != cudaSuccess) {
                cudaGetLastError();
                at.type = cudaMemoryTypeUnregistered;
            }
            pull_on = at.type == cudaMemoryTypeHost;
        }
        if (pull_on) CK(p, cudaStreamWaitEvent(p->pull_stream, p->ev_begin, 0));
        constexpr uint64_t kMinPull = 64u << 10; /* smaller shares stay with the copy engine */
        /* A staged chunk's unpack runs beside the next chunk's transfer: at a quarter of the
         * grid it still outruns the host link many times over, and it leaves most SMs to the
         * pull kernel, whose CTAs would otherwise wait for a full-grid unpack to end before
         * they start (the link idle meanwhile).  The last chunk, which nothing follows, takes
         * the whole grid. */
        constexpr int kStagedGridDiv = 4;
        uint32_t last_busy = 0;
        for (uint32_t c = 0; c < hp.n_chunks; ++c)
            if (p->chunk_busy[c]) last_busy = c;
        uint32_t k = 0; /* busy chunks so far: they take the slots in turn */
        cudaEvent_t prev_h2d_end = nullptr; /* CFA_OPT_TIMING: the last transfer's end event */
        for (uint32_t c = 0; c < hp.n_chunks; ++c) {
            if (!p->chunk_busy[c] || gather_failed) {
                cfa_status st = record_layers(p, c, c + 1, cs);
                if (st) return st;
                continue;
            }
            const int ds = (int)(k % (uint32_t)p->n_dev_slots);
            const uint64_t off = (uint64_t)c * S;
            const void *hsrc;
            int hs = -1;
            if (staged) {
                hs = cx->jobs[c].host_slot;
                CK(p, cudaStreamWaitEvent(p->fill_stream, p->ev_host_free[hs], 0));
                CK(p, cudaLaunchHostFunc(p->fill_stream, fill_host_fn, &cx->jobs[c]));
                CK(p, cudaEventRecord(p->ev_filled[hs], p->fill_stream));
                CK(p, cudaStreamWaitEvent(p->copy_stream, p->ev_filled[hs], 0));
                hsrc = p->h_slots + (uint64_t)hs * S;
            } else {
                const uint64_t so = src->period_bytes ? off % src->period_bytes : off;
                hsrc = static_cast<const uint8_t *>(src->base) + so;
            }
            uint8_t *dslot = p->d_slots + (uint64_t)ds * p->slot_bytes;
            CK(p, cudaStreamWaitEvent(p->copy_stream, p->ev_dev_free[ds], 0));
            if (timing) {
                /* with CFA_OPT_TIMING a chunk's transfer (copy engine and pull) begins after the
                 * previous chunk's has ended, so that each interval is that chunk's alone */
                if (prev_h2d_end) CK(p, cudaStreamWaitEvent(p->copy_stream, prev_h2d_end, 0));
                CK(p, cudaEventRecord(p->t_h2d0[c], p->copy_stream));
            }
            bool pulled = false;
            /* InMem -> InGPU: only the ranges the chunk's pieces read */
            for (uint32_t k = hp.copy_first[c]; k < hp.copy_first[c + 1]; ++k) {
                const cfa_copy &cp = hp.copies[k];
                const uint64_t at = cp.src - off;
                if (slices_in_place && cp.rows > 1) continue; /* read in place instead */
                if (cp.rows == 1) {
                    /* bytes [at, at + ce) by the copy engine, the rest by the pull kernel; the
                     * cut sits on a 16-byte boundary of the slot */
                    uint64_t ce = cp.width;
                    if (host_pull) {
                        ce = 0;
                    } else if (pull_on) {
                        const uint64_t want = cp.width - cp.width * hp.opts.pull_percent / 100;
                        const uint64_t cut = (at + want + 15) / 16 * 16 - at;
                        if (cut < cp.width && cp.width - cut >= kMinPull) ce = cut;
                    }
                    if (ce)
                        CK(p, cudaMemcpyAsync(dslot + at,
                                              static_cast<const uint8_t *>(hsrc) + at, ce,
                                              cudaMemcpyHostToDevice, p->copy_stream));
                    if (ce < cp.width) {
                        if (!pulled) {
                            CK(p, cudaStreamWaitEvent(p->pull_stream, p->ev_dev_free[ds], 0));
                            if (staged)
                                CK(p, cudaStreamWaitEvent(p->pull_stream, p->ev_filled[hs], 0));
                            if (timing)
                                CK(p, cudaStreamWaitEvent(p->pull_stream, p->t_h2d0[c], 0));
                            pulled = true;
                        }
                        CK(p, cfa_launch_pull(static_cast<const uint8_t *>(hsrc) + at + ce,
                                              dslot + at + ce, cp.width - ce, p->n_sms,
                                              p->pull_stream));
                    }
                } else
                    CK(p, cudaMemcpy2DAsync(dslot + at, cp.pitch,
                                            static_cast<const uint8_t *>(hsrc) + at, cp.pitch,
                                            cp.width, cp.rows, cudaMemcpyHostToDevice,
                                            p->copy_stream));
            }
            if (timing && !pulled) {
                CK(p, cudaEventRecord(p->t_h2d1[c], p->copy_stream));
                prev_h2d_end = p->t_h2d1[c];
            }
            p->last_h2d++;
            ++k;
            CK(p, cudaEventRecord(p->ev_h2d[ds], p->copy_stream));
            if (pulled) {
                /* both transfers must be done before the unpack, and before the pinned host
                 * slot is refilled: the caller's stream waits for both and marks the slot free */
                CK(p, cudaEventRecord(p->ev_pulled[ds], p->pull_stream));
                if (timing) {
                    /* the transfer ends when both paths have: its end event follows both,
                     * and the unpack waits for that event */
                    CK(p, cudaStreamWaitEvent(p->pull_stream, p->ev_h2d[ds], 0));
                    CK(p, cudaEventRecord(p->t_h2d1[c], p->pull_stream));
                    CK(p, cudaStreamWaitEvent(cs, p->t_h2d1[c], 0));
                    prev_h2d_end = p->t_h2d1[c];
                } else {
                    CK(p, cudaStreamWaitEvent(cs, p->ev_pulled[ds], 0));
                    CK(p, cudaStreamWaitEvent(cs, p->ev_h2d[ds], 0));
                }
                if (staged) CK(p, cudaEventRecord(p->ev_host_free[hs], cs));
            } else if (staged) {
                CK(p, cudaEventRecord(p->ev_host_free[hs], p->copy_stream));
            }
            cudaEvent_t ready = p->ev_h2d[ds];
            if (p->segmented) {
                /* InGPU for this rank's segment -> Gathered: the caller's collective fills the
                 * other segments of the slot on the gather stream */
                CK(p, cudaStreamWaitEvent(p->gather_stream, p->ev_h2d[ds], 0));
                const int r = hp.opts.gather(hp.opts.gather_user, dslot, seg_bytes,
                                             hp.opts.seg_world, hp.opts.seg_rank, c,
                                             reinterpret_cast<cfa_stream>(p->gather_stream));
                if (r != 0) {
                    /* the chunks before this one stay enqueued; the rest of the load is not,
                     * but its events are still recorded so that waits end */
                    set_err(p, "the gather callback failed on chunk %u (returned %d)", c, r);
                    gather_failed = CFA_ERR_GATHER;
                    cx->error.store(CFA_ERR_GATHER);
                    p->last_h2d = 0; /* no per-chunk copy times for a cut-short load */
                    cfa_status st = record_layers(p, c, c + 1, cs);
                    if (st) return st;
                    continue;
                }
                CK(p, cudaEventRecord(p->ev_gathered[ds], p->gather_stream));
                ready = p->ev_gathered[ds];
            }
            const bool direct_c = slices_in_place && has_slices(c);
            if (direct_c) {
                cfa_status st = launch(p, c, c + 1, (uint64_t)(uintptr_t)src->base,
                                       src->period_bytes, p->direct_stream, false, LAUNCH_STRIDED);
                if (st) return st;
                CK(p, cudaEventRecord(p->ev_direct, p->direct_stream));
            }
            CK(p, cudaStreamWaitEvent(cs, ready, 0));
            cfa_status st = launch(p, c, c + 1, (uint64_t)(uintptr_t)dslot - off, 0, cs, true,
                                   slices_in_place ? LAUNCH_CONTIG : LAUNCH_ALL,
                                   c == last_busy ? 1 : kStagedGridDiv);
            if (st) return st;
            CK(p, cudaEventRecord(p->ev_dev_free[ds], cs));
            if (direct_c) CK(p, cudaStreamWaitEvent(cs, p->ev_direct, 0));
            if ((st = record_layers(p, c, c + 1, cs))) return st;
        }
    }
    CK(p, cudaEventRecord(p->ev_all, cs));
    logf("load %llu enqueued: source kind %d, %llu kernel launches, %u staged chunks",
         (unsigned long long)p->n_loads, kind, (unsigned long long)p->last_launches, p->last_h2d);
    return cx->error.load() == CFA_ERR_GATHER ? CFA_ERR_GATHER : CFA_OK;
}

cfa_status cfa_wait_layer(cfa_plan *p, int32_t layer, cfa_stream consumer, int64_t timeout_ns)
{
    if (!p || p->host_only) return CFA_ERR_INVAL;
    if (!p->last) {
        set_err(p, "no load has been enqueued");
        return CFA_ERR_INVAL;
    }
    cudaEvent_t ev;
    if (layer == CFA_ALL) ev = p->ev_all;
    else if (layer >= 0 && (uint32_t)layer < p->hp.n_layers) ev = p->ev_layer[layer];
    else {
        set_err(p, "unknown readiness group %d", layer);
        return CFA_ERR_INVAL;
    }
    DeviceGuard g(p->device);
    if (consumer) {
        CK(p, cudaStreamWaitEvent(reinterpret_cast<cudaStream_t>(consumer), ev, 0));
        const int e = p->last->error.load();
        return e ? e : CFA_OK;
    }
    cfa_status st = wait_event_host(p, ev, timeout_ns);
    if (st) return st;
    const int e = p->last->error.load();
    if (e) {
        if (e != CFA_ERR_GATHER) set_err(p, "the source callback failed");
        return e;
    }
    if (layer == CFA_ALL) return check_status_word(p);
    return CFA_OK;
}

cfa_status cfa_get_checksums(cfa_plan *p, uint64_t *host_out, size_t n)
{
    if (!p || p->host_only || (n && !host_out) || n > p->hp.n_entries) return CFA_ERR_INVAL;
    if (!p->last) {
        set_err(p, "no load has been enqueued");
        return CFA_ERR_INVAL;
    }
    cfa_status st = cfa_wait_layer(p, CFA_ALL, nullptr, -1);
    if (st) return st;
    if (!n) return CFA_OK;
    DeviceGuard g(p->device);
    CK(p, cudaStreamWaitEvent(p->aux_stream, p->ev_all, 0));
    CK(p, cudaMemcpyAsync(host_out, p->d_ck, n * sizeof(uint64_t), cudaMemcpyDeviceToHost,
                          p->aux_stream));
    CK(p, cudaStreamSynchronize(p->aux_stream));
    return CFA_OK;
}

cfa_status cfa_get_stats(cfa_plan *p, cfa_stats *s)
{
    if (!p || !s) return CFA_ERR_INVAL;
    const cfa_host_plan &hp = p->hp;
    std::memset(s, 0, sizeof *s);
    s->blob_bytes = hp.blob_bytes;
    s->n_entries = hp.n_entries;
    s->n_dsts = hp.n_dsts;
    s->n_chunks = hp.n_chunks;
    s->n_layers = hp.n_layers;
    s->n_pieces = hp.n_pieces;
    s->n_slabs = hp.n_slabs;
    s->n_bulk = hp.n_bulk;
    s->n_tiny = hp.n_tiny;
    s->n_strided = hp.n_strided;
    s->bytes_read = hp.bytes_read;
    s->bytes_written = hp.bytes_written;
    s->descriptor_bytes = (hp.n_slabs + hp.n_bulk + hp.n_tiny) * sizeof(cfa_work) +
                          hp.n_strided * sizeof(cfa_swork);
    s->staged_bytes = hp.staged_bytes;
    s->loads = p->n_loads;
    s->kernel_launches = p->last_launches;
    s->plan_ms = p->plan_ms;
    if ((hp.opts.flags & CFA_OPT_TIMING) && p->last && !p->host_only) {
        DeviceGuard g(p->device);
        CK(p, cudaEventSynchronize(p->ev_all));
        float ms = 0;
        CK(p, cudaEventElapsedTime(&ms, p->ev_begin, p->ev_all));
        s->load_ms = ms;
        for (uint32_t c = 0; p->last_h2d && c < p->t_h2d0.size(); ++c) {
            if (!p->chunk_busy[c]) continue;
            CK(p, cudaEventElapsedTime(&ms, p->t_h2d0[c], p->t_h2d1[c]));
            s->h2d_ms += ms;
        }
        for (uint64_t k = 0; k < p->last_launches && k < p->t_k0.size(); ++k) {
            CK(p, cudaEventElapsedTime(&ms, p->t_k0[k], p->t_k1[k]));
            s->unpack_ms += ms;
        }
    }
    return CFA_OK;
}

cfa_status cfa_get_layer_times(cfa_plan *p, float *ms_out, size_t n)
{
    if (!p || p->host_only || (n && !ms_out) || n > p->hp.n_layers) return CFA_ERR_INVAL;
    if (!(p->hp.opts.flags & CFA_OPT_TIMING) || !p->last) {
        set_err(p, "layer times need a CFA_OPT_TIMING plan and a load");
        return CFA_ERR_INVAL;
    }
    DeviceGuard g(p->device);
    CK(p, cudaEventSynchronize(p->ev_all));
    for (size_t l = 0; l < n; ++l)
        CK(p, cudaEventElapsedTime(&ms_out[l], p->ev_begin, p->ev_layer[l]));
    return CFA_OK;
}

cfa_status cfa_get_timeline(cfa_plan *p, cfa_chunk_times *out, size_t n)
{
    if (!p || p->host_only || (n && !out) || n > p->hp.n_chunks) return CFA_ERR_INVAL;
    if (!(p->hp.opts.flags & CFA_OPT_TIMING) || !p->last) {
        set_err(p, "the timeline needs a CFA_OPT_TIMING plan and a load");
        return CFA_ERR_INVAL;
    }
    DeviceGuard g(p->device);
    CK(p, cudaEventSynchronize(p->ev_all));
    for (size_t c = 0; c < n; ++c) out[c] = cfa_chunk_times{-1.f, -1.f, -1.f, -1.f};
    for (uint32_t c = 0; p->last_h2d && c < n && c < p->t_h2d0.size(); ++c) {
        if (!p->chunk_busy[c]) continue; /* not staged */
        CK(p, cudaEventElapsedTime(&out[c].h2d_begin_ms, p->ev_begin, p->t_h2d0[c]));
        CK(p, cudaEventElapsedTime(&out[c].h2d_end_ms, p->ev_begin, p->t_h2d1[c]));
    }
    for (uint64_t k = 0; k < p->last_launches && k < p->t_k0.size(); ++k) {
        float b = 0, e = 0;
        CK(p, cudaEventElapsedTime(&b, p->ev_begin, p->t_k0[k]));
        CK(p, cudaEventElapsedTime(&e, p->ev_begin, p->t_k1[k]));
        for (uint32_t c = p->t_k_c0[k]; c < p->t_k_c1[k] && c < n; ++c) {
            if (out[c].unpack_begin_ms < 0 || b < out[c].unpack_begin_ms)
                out[c].unpack_begin_ms = b;
            if (e > out[c].unpack_end_ms) out[c].unpack_end_ms = e;
        }
    }
    return CFA_OK;
}

cfa_status cfa_plan_info(const cfa_plan *p, uint64_t *n_layers, uint64_t *n_pieces,
                         uint64_t *n_chunks)
{
    if (!p) return CFA_ERR_INVAL;
    if (n_layers) *n_layers = p->hp.n_layers;
    if (n_pieces) *n_pieces = p->hp.n_pieces;
    if (n_chunks) *n_chunks = p->hp.n_chunks;
    return CFA_OK;
}

cfa_status cfa_plan_get_pieces(const cfa_plan *p, cfa_piece *out, size_t cap, size_t *n_out)
{
    if (!p || (cap && !out)) return CFA_ERR_INVAL;
    const size_t n = std::min(cap, p->hp.n_pieces);
    if (n) std::memcpy(out, p->hp.pieces, n * sizeof(cfa_piece));
    if (n_out) *n_out = n;
    return CFA_OK;
}

cfa_status cfa_unpack_chunks_async(cfa_plan *p, uint32_t chunk_begin, uint32_t chunk_end,
                                   const void *chunk_src, cfa_stream stream)
{
    if (!p || p->host_only || chunk_begin > chunk_end || chunk_end > p->hp.n_chunks ||
        (!chunk_src && chunk_end > chunk_begin)) {
        if (p) set_err(p, "bad chunk range or source");
        return CFA_ERR_INVAL;
    }
    if ((uintptr_t)chunk_src & 255u) {
        set_err(p, "chunk_src must be 256-byte aligned");
        return CFA_ERR_ALIGN;
    }
    std::unique_lock<std::mutex> lk(p->mu, std::try_to_lock);
    if (!lk.owns_lock()) return CFA_ERR_BUSY;
    DeviceGuard g(p->device);
    const uint64_t base =
        (uint64_t)(uintptr_t)chunk_src - (uint64_t)chunk_begin * p->hp.chunk_bytes;
    const uint64_t saved = p->last_launches;
    p->last_launches = p->t_k0.size(); /* no timing events for direct launches */
    cfa_status st =
        launch(p, chunk_begin, chunk_end, base, 0, reinterpret_cast<cudaStream_t>(stream));
    p->last_launches = saved;
    return st;
}

cfa_status cfa_reset_checksums(cfa_plan *p, cfa_stream stream)
{
    if (!p || p->host_only) return CFA_ERR_INVAL;
    DeviceGuard g(p->device);
    CK(p, cudaMemsetAsync(p->d_ck, 0, ck_clear_bytes(p->hp.n_entries),
                          reinterpret_cast<cudaStream_t>(stream)));
    return CFA_OK;
}

cfa_status cfa_plan_destroy(cfa_plan *p)
{
    release(p);
    return CFA_OK;
}

const char *cfa_last_error(const cfa_plan *p) { return p ? p->err : g_create_err; }

void cfa_internal_set_error(const char *msg)
{
    std::snprintf(g_create_err, sizeof g_create_err, "%s", msg ? msg : "");
}

const char *cfa_status_name(cfa_status st)
{
    switch (st) {
    case CFA_OK: return "CFA_OK";
    case CFA_ERR_INVAL: return "CFA_ERR_INVAL";
    case CFA_ERR_OVERLAP: return "CFA_ERR_OVERLAP";
    case CFA_ERR_OOB: return "CFA_ERR_OOB";
    case CFA_ERR_COVERAGE: return "CFA_ERR_COVERAGE";
    case CFA_ERR_CUDA: return "CFA_ERR_CUDA";
    case CFA_ERR_SOURCE: return "CFA_ERR_SOURCE";
    case CFA_ERR_TIMEOUT: return "CFA_ERR_TIMEOUT";
    case CFA_ERR_BUSY: return "CFA_ERR_BUSY";
    case CFA_ERR_NOMEM: return "CFA_ERR_NOMEM";
    case CFA_ERR_DTYPE: return "CFA_ERR_DTYPE";
    case CFA_ERR_ALIGN: return "CFA_ERR_ALIGN";
    case CFA_ERR_DEVICE: return "CFA_ERR_DEVICE";
    case CFA_ERR_SHAPE: return "CFA_ERR_SHAPE";
    case CFA_ERR_SUSPECT: return "CFA_ERR_SUSPECT";
    case CFA_ERR_GATHER: return "CFA_ERR_GATHER";
    default: return "CFA_ERR_UNKNOWN";
    }
}

size_t cfa_abi_sizeof(const char *type_name)
{
    if (!type_name) return 0;
    if (!std::strcmp(type_name, "cfa_tensor_entry")) return sizeof(cfa_tensor_entry);
    if (!std::strcmp(type_name, "cfa_dst")) return sizeof(cfa_dst);
    if (!std::strcmp(type_name, "cfa_plan_opts")) return sizeof(cfa_plan_opts);
    if (!std::strcmp(type_name, "cfa_source")) return sizeof(cfa_source);
    if (!std::strcmp(type_name, "cfa_stats")) return sizeof(cfa_stats);
    if (!std::strcmp(type_name, "cfa_piece")) return sizeof(cfa_piece);
    if (!std::strcmp(type_name, "cfa_st_tensor")) return sizeof(cfa_st_tensor);
    if (!std::strcmp(type_name, "cfa_chunk_times")) return sizeof(cfa_chunk_times);
    return 0;
}

cfa_status cfa_selftest_wait_timeout(int device, int *status_word)
{
    if (!status_word) return CFA_ERR_INVAL;
    int prev = 0;
    CK(nullptr, cudaGetDevice(&prev));
    if (device >= 0) CK(nullptr, cudaSetDevice(device));
    const cudaError_t e = cfa_bulk_selftest_timeout(status_word);
    if (device >= 0) cudaSetDevice(prev);
    if (e != cudaSuccess) {
        set_err(nullptr, "TMA wait self-test failed: %s", cudaGetErrorString(e));
        return CFA_ERR_CUDA;
    }
    return CFA_OK;
}

} /* extern "C" */
