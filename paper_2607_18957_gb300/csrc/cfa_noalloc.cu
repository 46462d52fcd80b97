/*
 * cfa_unpack_noalloc: the unpack of a device-resident checkpoint for callers that must not
 * allocate.  The paper has no counterpart; this is a library convenience.
 *
 * Who needs it: code that runs where allocating is not allowed or not possible -- inside a
 * serving engine whose memory pool already owns the whole device and forbids side allocations,
 * on a latency-critical path that cannot afford cudaFree's implicit device-wide
 * synchronisation, or in a restricted runtime that has no allocator at hand.  cfa_plan_create allocates a device descriptor table,
 * a checksum buffer and staging slots; this entry point allocates nothing at all, on the device
 * or on the host.  Its scratch (the work descriptors and a status word) lives in a file-scope
 * device array of fixed size; the host side builds the descriptors in a file-scope host array.
 *
 * Set-up: the first call on a device looks up the device address of the scratch array with
 * cudaGetSymbolAddress (in host code the array's name is only a stand-in, not a device
 * address) and caches it for that device; make the first call on each device before any stream
 * capture.  The cached address belongs to the device's current context: after a
 * cudaDeviceReset the library must not be used again in the process.
 *
 * Blocking: the descriptors go up with a copy from pageable host memory, which returns only
 * once the bytes have been copied, so the call blocks the host until the work already queued
 * on the stream has run and the copy is done; the unpack kernels themselves run after it
 * returns.
 *
 * Sharing: every call on a device uses the same scratch array, which keeps the last call's
 * contents.  Calls are serialised on the host by a mutex, but two calls whose GPU work overlaps
 * (different streams, no ordering between them) race on the scratch: order them on one stream
 * or with events.
 */
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "cfa_internal.h"

extern "C" int cfa_unpack_blocks_per_sm(int cls);
extern "C" cudaError_t cfa_launch_unpack(int cls, const cfa_work *slabs, uint32_t n_slabs,
                                         const cfa_work *tiny, uint32_t n_tiny,
                                         uint64_t src_base, uint64_t src_period,
                                         uint64_t src_lo, uint64_t src_hi,
                                         unsigned long long *ck, int *status, int grid_cap,
                                         int dev_src, cudaStream_t stream);

namespace {

constexpr int kMaxDevices = 64;
constexpr uint64_t kSlabBytes = 2ull << 20; /* destination bytes per block-level item */
constexpr uint64_t kTinyBytes = 8192;      /* below this, one warp per tensor */

/* Device scratch: CFA_NOALLOC_MAX_ITEMS descriptors, then the status word. */
struct NoallocScratch {
    cfa_work items[CFA_NOALLOC_MAX_ITEMS];
    int status;
};
static __device__ __align__(256) NoallocScratch g_noalloc_scratch;

/* Host twin of the descriptors, filled before each upload (guarded by g_mutex). */
static cfa_work g_host_items[CFA_NOALLOC_MAX_ITEMS];

std::mutex g_mutex;
NoallocScratch *g_scratch_dev[kMaxDevices];
int g_grid_cap[kMaxDevices][CFA_N_CLASSES];

/* The caller's message buffer for the current call (may be NULL). */
thread_local char *g_err = nullptr;
thread_local size_t g_err_len = 0;

void say(const char *fmt, ...)
{
    if (!g_err || !g_err_len) return;
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, g_err_len, fmt, ap);
    va_end(ap);
}

int dtype_size(int32_t dt)
{
    switch (dt) {
    case CFA_DTYPE_U8: return 1;
    case CFA_DTYPE_BF16:
    case CFA_DTYPE_F16:
    case CFA_DTYPE_I16: return 2;
    case CFA_DTYPE_F32:
    case CFA_DTYPE_I32: return 4;
    case CFA_DTYPE_I64:
    case CFA_DTYPE_F64: return 8;
    default: return 0;
    }
}

int log2_es(int es) { return es == 1 ? 0 : es == 2 ? 1 : es == 4 ? 2 : 3; }

/* a * b into *out; false when the product does not fit in 64 bits */
bool mul_fits(uint64_t a, uint64_t b, uint64_t *out)
{
    if (a != 0 && b > UINT64_MAX / a) return false;
    *out = a * b;
    return true;
}

/* Warp-level items of a tiny entry of nb > 0 destination bytes at dst0: one per
 * CFA_TINY_SEG_BYTES-aligned block of destination addresses it touches. */
uint64_t tiny_items(uint64_t dst0, uint64_t nb)
{
    return (dst0 + nb - 1) / CFA_TINY_SEG_BYTES - dst0 / CFA_TINY_SEG_BYTES + 1;
}

cfa_status fail(cfa_status st, const char *msg, size_t i)
{
    say("cfa_unpack_noalloc: %s (entry %zu)", msg, i);
    return st;
}

/* Placement of one entry: element count, element sizes and destination byte offset. */
cfa_status place(const cfa_tensor_entry &e, const cfa_dst *dsts, size_t n_dsts,
                 uint64_t blob_bytes, size_t i, uint64_t *n_out, int *es_s, int *es_d,
                 uint64_t *dst_off, int *conv)
{
    *es_s = dtype_size(e.src_dtype);
    if (!*es_s || e.ndim < 0 || e.ndim > CFA_MAX_DIMS || e.dst_index < 0 ||
        (size_t)e.dst_index >= n_dsts || e.src_row_stride ||
        (e.flags & ~(CFA_ENTRY_CAST_BF16 | CFA_ENTRY_CKSUM | CFA_ENTRY_CONVERT)))
        return fail(CFA_ERR_INVAL,
                    "bad dtype, ndim, flags or destination index, or a strided entry (strided "
                    "entries need cfa_plan_create)", i);
    const cfa_dst &d = dsts[e.dst_index];
    const int es_dst = dtype_size(d.dtype);
    if (!es_dst || d.ndim < 0 || d.ndim > CFA_MAX_DIMS)
        return fail(CFA_ERR_INVAL, "bad destination dtype or ndim", i);
    const bool converts = (e.flags & (CFA_ENTRY_CAST_BF16 | CFA_ENTRY_CONVERT)) != 0;
    *conv = converts ? cfa_conversion(e.src_dtype, d.dtype) : CFA_CONV_NONE;
    if (converts ? (*conv == CFA_CONV_NONE ||
                    ((e.flags & CFA_ENTRY_CAST_BF16) && *conv != CFA_CONV_F32_BF16))
                 : (e.src_dtype != d.dtype))
        return fail(CFA_ERR_DTYPE, "dtype does not match the destination", i);
    *es_d = es_dst;
    /* every product is checked: a shape whose size wraps around 64 bits would pass the bounds
     * checks below with a wrong size */
    uint64_t n = 1, d_numel = 1, src_len = 0, d_bytes = 0;
    for (int k = 0; k < e.ndim; ++k) {
        if (e.shape[k] < 0 || !mul_fits(n, (uint64_t)e.shape[k], &n))
            return fail(CFA_ERR_INVAL, "negative or overflowing dimension", i);
    }
    for (int k = 0; k < d.ndim; ++k) {
        if (d.shape[k] < 0 || !mul_fits(d_numel, (uint64_t)d.shape[k], &d_numel))
            return fail(CFA_ERR_INVAL, "negative or overflowing destination dimension", i);
    }
    if (!mul_fits(d_numel, (uint64_t)es_dst, &d_bytes) || !mul_fits(n, (uint64_t)*es_s, &src_len))
        return fail(CFA_ERR_INVAL, "tensor or destination too large", i);
    uint64_t row = 1;
    if (d.ndim >= 2) {
        row = (uint64_t)d.shape[d.ndim - 1];
        if (n && (e.ndim == 0 || (uint64_t)e.shape[e.ndim - 1] != row))
            return fail(CFA_ERR_SHAPE, "last dimension differs from the destination row", i);
    }
    uint64_t first = 0;
    if (e.dst_row_offset < 0 || !mul_fits((uint64_t)e.dst_row_offset, row, &first) ||
        first > d_numel || n > d_numel - first)
        return fail(CFA_ERR_OOB, "rows fall outside the destination", i);
    if (e.blob_offset % (uint64_t)*es_s)
        return fail(CFA_ERR_ALIGN, "blob offset not a multiple of the element size", i);
    if (e.blob_offset > blob_bytes || src_len > blob_bytes - e.blob_offset)
        return fail(CFA_ERR_OOB, "reads past the end of the blob", i);
    if (n && ((uintptr_t)d.dev_ptr % (uintptr_t)*es_d || !d.dev_ptr))
        return fail(CFA_ERR_ALIGN, "destination pointer NULL or misaligned", i);
    *n_out = n;
    *dst_off = first * (uint64_t)*es_d;
    return CFA_OK;
}

/* Once per device, with that device current: device address of the scratch array, and the
 * persistent grid size of each kernel class. */
cfa_status setup(int dev, NoallocScratch **scratch)
{
    if (dev < 0 || dev >= kMaxDevices) {
        say("cfa_unpack_noalloc: device %d out of range", dev);
        return CFA_ERR_INVAL;
    }
    if (g_scratch_dev[dev]) {
        *scratch = g_scratch_dev[dev];
        return CFA_OK;
    }
    void *ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || !ptr) {
        say("cfa_unpack_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
        return CFA_ERR_CUDA;
    }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess || sms <= 0) {
        say("cfa_unpack_noalloc: cannot query the SM count: %s", cudaGetErrorString(e));
        return CFA_ERR_CUDA;
    }
    for (int k = 0; k < CFA_N_CLASSES; ++k) {
        const int per_sm = cfa_unpack_blocks_per_sm(k);
        if (per_sm <= 0) {
            say("cfa_unpack_noalloc: an unpack kernel cannot run on device %d", dev);
            return CFA_ERR_CUDA;
        }
        g_grid_cap[dev][k] = sms * per_sm;
    }
    g_scratch_dev[dev] = static_cast<NoallocScratch *>(ptr);
    *scratch = g_scratch_dev[dev];
    return CFA_OK;
}

} // namespace

extern "C" cfa_status cfa_unpack_noalloc(const cfa_tensor_entry *entries, size_t n_entries,
                                         const cfa_dst *dsts, size_t n_dsts,
                                         const void *blob_dev, uint64_t blob_bytes,
                                         uint64_t *cksum_dev, int *status_dev,
                                         cfa_stream stream_, char *err, size_t err_len)
{
    g_err = err;
    g_err_len = err ? err_len : 0;
    if (g_err_len) g_err[0] = 0;
    if ((n_entries && !entries) || (n_dsts && !dsts) || (blob_bytes && !blob_dev)) {
        say("cfa_unpack_noalloc: NULL argument");
        return CFA_ERR_INVAL;
    }
    if ((uintptr_t)status_dev & 3u) {
        say("cfa_unpack_noalloc: status_dev must be 4-byte aligned");
        return CFA_ERR_ALIGN;
    }
    if ((uintptr_t)blob_dev & 255u) {
        say("cfa_unpack_noalloc: the blob must be 256-byte aligned");
        return CFA_ERR_ALIGN;
    }
    if (n_entries >= (size_t)CFA_NO_CK) return fail(CFA_ERR_INVAL, "too many entries", 0);
    cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
    std::lock_guard<std::mutex> lock(g_mutex);

    /* validate every entry and count the work items, per class, without storing anything */
    uint32_t count[CFA_N_CLASSES][2] = {};
    for (size_t i = 0; i < n_entries; ++i) {
        uint64_t n, off;
        int es_s, es_d, conv;
        cfa_status st =
            place(entries[i], dsts, n_dsts, blob_bytes, i, &n, &es_s, &es_d, &off, &conv);
        if (st) return st;
        if (!n) continue;
        const int cls = conv ? CFA_CLASS_OF_CONV(conv) : log2_es(es_s);
        const uint64_t nb = n * (uint64_t)es_d;
        const uint64_t dst0 = (uint64_t)(uintptr_t)dsts[entries[i].dst_index].dev_ptr + off;
        const uint64_t items = nb < kTinyBytes ? tiny_items(dst0, nb)
                                               : (nb + kSlabBytes - 1) / kSlabBytes;
        uint64_t total = items;
        for (int k = 0; k < CFA_N_CLASSES; ++k) total += count[k][0] + count[k][1];
        if (total > CFA_NOALLOC_MAX_ITEMS) {
            say("cfa_unpack_noalloc: the manifest needs more than the %d work items of the "
                "fixed scratch (one per 2 MiB of destination, one per 512 bytes of a tensor "
                "under 8 KiB); use cfa_plan_create", CFA_NOALLOC_MAX_ITEMS);
            return CFA_ERR_INVAL;
        }
        count[cls][nb < kTinyBytes ? 1 : 0] += (uint32_t)items;
    }

    /* lay the items out as [class 0 slabs][class 0 tiny][class 1 slabs] ... */
    uint32_t base[CFA_N_CLASSES][2], cursor[CFA_N_CLASSES][2];
    uint32_t total = 0;
    for (int k = 0; k < CFA_N_CLASSES; ++k)
        for (int t = 0; t < 2; ++t) {
            base[k][t] = cursor[k][t] = total;
            total += count[k][t];
        }
    for (size_t i = 0; i < n_entries; ++i) {
        uint64_t n, off;
        int es_s, es_d, conv;
        place(entries[i], dsts, n_dsts, blob_bytes, i, &n, &es_s, &es_d, &off, &conv);
        if (!n) continue;
        const int cls = conv ? CFA_CLASS_OF_CONV(conv) : log2_es(es_s);
        cfa_work w;
        w.ck = (cksum_dev && (entries[i].flags & CFA_ENTRY_CKSUM)) ? (uint32_t)i : CFA_NO_CK;
        w.mode = CFA_MODE(log2_es(es_s), log2_es(es_d), conv);
        w.pad = (uint32_t)cls;
        const uint64_t dst0 = (uint64_t)(uintptr_t)dsts[entries[i].dst_index].dev_ptr + off;
        const uint64_t nb = n * (uint64_t)es_d;
        if (nb < kTinyBytes) {
            /* warp-level items of at most CFA_TINY_SEG_BYTES, cut at destination addresses
             * that are multiples of it (the tiny kernel's unit, as in the planned path) */
            for (uint64_t pos = dst0; pos < dst0 + nb;) {
                uint64_t next = (pos / CFA_TINY_SEG_BYTES + 1) * CFA_TINY_SEG_BYTES;
                if (next > dst0 + nb) next = dst0 + nb;
                w.src = entries[i].blob_offset + (pos - dst0) / (uint64_t)es_d * (uint64_t)es_s;
                w.dst = pos;
                w.n = (uint32_t)((next - pos) / (uint64_t)es_d);
                g_host_items[cursor[cls][1]++] = w;
                pos = next;
            }
            continue;
        }
        const uint64_t per = kSlabBytes / (uint64_t)es_d; /* elements per item */
        for (uint64_t e0 = 0; e0 < n; e0 += per) {
            const uint64_t k = n - e0 < per ? n - e0 : per;
            w.src = entries[i].blob_offset + e0 * (uint64_t)es_s;
            w.dst = dst0 + e0 * (uint64_t)es_d;
            w.n = (uint32_t)k;
            g_host_items[cursor[cls][0]++] = w;
        }
    }

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        say("cfa_unpack_noalloc: cudaGetDevice failed: %s", cudaGetErrorString(e));
        return CFA_ERR_CUDA;
    }
    NoallocScratch *scratch = nullptr;
    cfa_status st = setup(dev, &scratch);
    if (st) return st;

    /* the kernels' status word (the caller's, or the scratch's own) and the checksums start at
     * zero; the descriptors are uploaded from the host array (a pageable copy: the call returns
     * once the bytes are on the device, after the work queued before it on the stream) */
    int *status = status_dev ? status_dev : &scratch->status;
    e = cudaMemsetAsync(status, 0, sizeof(int), stream);
    if (e == cudaSuccess && cksum_dev && n_entries)
        e = cudaMemsetAsync(cksum_dev, 0, n_entries * sizeof(uint64_t), stream);
    if (e == cudaSuccess && total)
        e = cudaMemcpyAsync(scratch->items, g_host_items, (size_t)total * sizeof(cfa_work),
                            cudaMemcpyHostToDevice, stream);
    for (int k = 0; e == cudaSuccess && k < CFA_N_CLASSES; ++k) {
        if (!count[k][0] && !count[k][1]) continue;
        e = cfa_launch_unpack(k, scratch->items + base[k][0], count[k][0],
                              scratch->items + base[k][1], count[k][1],
                              (uint64_t)(uintptr_t)blob_dev, 0, 0, blob_bytes,
                              reinterpret_cast<unsigned long long *>(cksum_dev), status,
                              g_grid_cap[dev][k], 1, stream);
    }
    if (e != cudaSuccess) {
        say("cfa_unpack_noalloc: CUDA error %s", cudaGetErrorString(e));
        return CFA_ERR_CUDA;
    }
    return CFA_OK;
}
