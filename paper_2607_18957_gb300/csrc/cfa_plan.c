/*
 * Host plan builder: validates a manifest and precomputes the chunk <-> tensor mapping of
 * InstantInfer section 4.2 (refined CFA model: "tensor.chunks" / "chunk.tensors"), cut down to
 * the GPU's units of work.  Pure host C; makes no CUDA call, so it runs (and is tested) on
 * machines without a GPU.
 *
 *   1. validate options, destinations and entries;
 *   2. place every entry inside its destination (row offset -> byte offset) and check that the
 *      destinations are covered without overlap (exactly once in strict mode);
 *   3. cut the blob into chunks of S bytes (the last one partial) and intersect every entry's
 *      source range with them: one piece per (tensor, chunk) pair;
 *   4. turn pieces into work items: pieces below `tiny_bytes` destination bytes become
 *      warp-level items of at most CFA_TINY_SEG_BYTES each; larger ones are split into
 *      block-level slabs whose cuts fall on destination addresses that are multiples of
 *      `slab_bytes`, so only a piece's first and last slab can start or end off a 16-byte
 *      boundary;
 *   5. record, per readiness group, the last chunk that carries one of its bytes.
 */
#define _GNU_SOURCE /* sched_getaffinity, CPU_COUNT */
#include <sched.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "cfa_internal.h"

/* The TMA bulk kernel takes cast-free slabs whose source, destination and length are all
 * multiples of 16 bytes. */
#ifndef CFA_BULK_READY
#define CFA_BULK_READY 1
#endif

int cfa_dtype_size(int32_t dt)
{
    switch (dt) {
    case CFA_DTYPE_U8: return 1;
    case CFA_DTYPE_BF16: return 2;
    case CFA_DTYPE_F16: return 2;
    case CFA_DTYPE_F32: return 4;
    case CFA_DTYPE_I32: return 4;
    case CFA_DTYPE_I64: return 8;
    case CFA_DTYPE_F64: return 8;
    case CFA_DTYPE_I16: return 2;
    default: return 0;
    }
}

static int log2_small(int x) { return x == 1 ? 0 : x == 2 ? 1 : x == 4 ? 2 : 3; }

/* Fill threads by default: one per CPU the process may run on, at most 32.  On the GB300 machine
 * (16 cores) the pageable ring's rate rises with the thread count up to the core count (4: 51,
 * 8: 85, 16: 106 GB/s) and stays there with more threads (32-64: 104-105 GB/s), where it equals
 * the cores' multi-threaded memcpy rate. */
static int cfa_default_fill_threads(void)
{
    cpu_set_t set;
    int n = 0;
    if (sched_getaffinity(0, sizeof set, &set) == 0) n = CPU_COUNT(&set);
    if (n <= 0) n = 8;
    return n > 32 ? 32 : n;
}

/* Slab size when the caller leaves it to the plan: about 4096 block-level items over the load
 * (the persistent grids hold 456-608 CTAs), as a power of two in [32 KiB, 256 KiB].  Loads of a
 * gigabyte and more get 256 KiB (the size a sweep of 64 KiB - 1 MiB picked on the 8B, 70B,
 * Mixtral and fp32 checkpoints); a 125 MiB load of 1,000 tensors gets 32 KiB, where 256 KiB left
 * one slab per CTA and a launch of 0.073 ms instead of 0.054. */
static uint32_t cfa_auto_slab(uint64_t dst_bytes)
{
    uint64_t s = 32u << 10;
    while (s < (256u << 10) && s * 2 * 4096 <= dst_bytes) s *= 2;
    return (uint32_t)s;
}

void cfa_plan_opts_default(cfa_plan_opts *o)
{
    if (!o) return;
    memset(o, 0, sizeof *o);
    o->chunk_bytes = 512ull << 20;
    o->host_slots = 2;
    o->dev_slots = 3;
    o->fill_threads = cfa_default_fill_threads();
    o->device = -1;
    o->slab_bytes = 0; /* chosen from the load's size: cfa_auto_slab */
    o->tiny_bytes = 8192;
    o->flags = CFA_OPT_STRICT_COVERAGE | CFA_OPT_BULK;
    o->seg_world = 1;
    o->pull_percent = 100;
}

/* Rank `rank`'s segment of chunk `chunk` (section 4.2, distributed loading): the chunk is cut
 * into `world` equal segments of S / world bytes; the part inside the blob. */
cfa_status cfa_segment_range(uint64_t blob_bytes, uint64_t chunk_bytes, int32_t world,
                             int32_t rank, uint32_t chunk, uint64_t *blob_offset,
                             uint64_t *bytes)
{
    if (!blob_offset || !bytes || world < 1 || rank < 0 || rank >= world || chunk_bytes == 0 ||
        chunk_bytes % (256ull * (uint64_t)world) != 0)
        return CFA_ERR_INVAL;
    const uint64_t n_chunks = blob_bytes / chunk_bytes + (blob_bytes % chunk_bytes != 0);
    if ((uint64_t)chunk >= n_chunks) return CFA_ERR_INVAL;
    const uint64_t seg = chunk_bytes / (uint64_t)world;
    const uint64_t lo = (uint64_t)chunk * chunk_bytes + (uint64_t)rank * seg;
    *blob_offset = lo;
    *bytes = lo >= blob_bytes ? 0 : (blob_bytes - lo < seg ? blob_bytes - lo : seg);
    return CFA_OK;
}

static void fail(char *err, size_t n, const char *fmt, ...)
{
    if (!err || !n) return;
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(err, n, fmt, ap);
    va_end(ap);
}

static const char *ename(const cfa_tensor_entry *e) { return e->name ? e->name : "(unnamed)"; }

static char *dup_str(const char *s)
{
    const size_t n = strlen(s) + 1;
    char *d = (char *)malloc(n);
    if (d) memcpy(d, s, n);
    return d;
}

/* ------------------------------------------------------------------------------------------ */
/* growable arrays                                                                            */

typedef struct {
    void *p;
    size_t n, cap, elem;
} vec;

static int vec_push(vec *v, const void *x)
{
    if (v->n == v->cap) {
        size_t cap = v->cap ? 2 * v->cap : 256;
        void *q = realloc(v->p, cap * v->elem);
        if (!q) return -1;
        v->p = q;
        v->cap = cap;
    }
    memcpy((char *)v->p + v->n * v->elem, x, v->elem);
    v->n++;
    return 0;
}

/* ------------------------------------------------------------------------------------------ */
/* stable ordering by a 64-bit key                                                              */

/* Reorders the n records of `elem` bytes at `base` by key[i] (the key of record i), stably:
 * records with equal keys keep their order.  A least-significant-digit radix sort on 11-bit
 * digits, with only as many passes as the largest key needs, so a few hundred thousand pieces
 * take a few milliseconds instead of a comparison sort's tens; records already in order are left
 * alone.  Returns 0, or -1 when out of memory. */
static int sort_by_key(void *base, size_t n, size_t elem, const uint64_t *key)
{
    enum { BITS = 11, RADIX = 1 << BITS };
    uint64_t maxk = 0;
    int sorted = 1;
    for (size_t i = 0; i < n; ++i) {
        if (key[i] > maxk) maxk = key[i];
        if (i && key[i] < key[i - 1]) sorted = 0;
    }
    if (sorted) return 0;
    size_t *idx = (size_t *)malloc(n * sizeof(size_t)), *idx2 = (size_t *)malloc(n * sizeof(size_t));
    uint64_t *k1 = (uint64_t *)malloc(n * sizeof(uint64_t)), *k2 = (uint64_t *)malloc(n * sizeof(uint64_t));
    size_t *count = (size_t *)malloc((RADIX + 1) * sizeof(size_t));
    char *tmp = (char *)malloc(n * elem);
    int rc = -1;
    if (!idx || !idx2 || !k1 || !k2 || !count || !tmp) goto out;
    for (size_t i = 0; i < n; ++i) {
        idx[i] = i;
        k1[i] = key[i];
    }
    for (int shift = 0; shift < 64 && (maxk >> shift); shift += BITS) {
        memset(count, 0, (RADIX + 1) * sizeof(size_t));
        for (size_t i = 0; i < n; ++i) count[((k1[i] >> shift) & (RADIX - 1)) + 1]++;
        for (int d = 0; d < RADIX; ++d) count[d + 1] += count[d];
        for (size_t i = 0; i < n; ++i) {
            const size_t to = count[(k1[i] >> shift) & (RADIX - 1)]++;
            idx2[to] = idx[i];
            k2[to] = k1[i];
        }
        size_t *ti = idx;
        idx = idx2;
        idx2 = ti;
        uint64_t *tk = k1;
        k1 = k2;
        k2 = tk;
    }
    for (size_t i = 0; i < n; ++i) memcpy(tmp + i * elem, (const char *)base + idx[i] * elem, elem);
    memcpy(base, tmp, n * elem);
    rc = 0;
out:
    free(idx);
    free(idx2);
    free(k1);
    free(k2);
    free(count);
    free(tmp);
    return rc;
}

static int bit_width(uint64_t x)
{
    int b = 0;
    while (x) {
        b++;
        x >>= 1;
    }
    return b;
}

/* ------------------------------------------------------------------------------------------ */

typedef struct {
    uint64_t n;       /* elements */
    int es_s, es_d;   /* element sizes */
    int conv;         /* CFA_CONV_* */
    uint64_t dst_off; /* byte offset inside the destination */
    uint64_t cols;    /* elements per row (the last dimension) */
    uint64_t stride;  /* source elements between row starts; == cols when contiguous */
    uint64_t extent;  /* source bytes from the first to the last element */
} ent_info;

typedef struct {
    uint32_t dst;
    uint32_t entry;
    uint64_t off, len;
} span;

static int cmp_span(const void *a, const void *b)
{
    const span *x = (const span *)a, *y = (const span *)b;
    if (x->dst != y->dst) return x->dst < y->dst ? -1 : 1;
    if (x->off != y->off) return x->off < y->off ? -1 : 1;
    return (x->entry > y->entry) - (x->entry < y->entry);
}

typedef struct {
    uint64_t ptr, len;
    uint32_t idx;
} dspan;

static int mul_overflows(uint64_t a, uint64_t b, uint64_t *out)
{
    if (a != 0 && b > UINT64_MAX / a) return 1;
    *out = a * b;
    return 0;
}

/* Class and source blob offset of an item of either descriptor kind. */
static void item_key(const vec *v, size_t q, uint32_t *cls, uint64_t *src)
{
    if (v->elem == sizeof(cfa_swork)) {
        const cfa_swork *w = (const cfa_swork *)v->p + q;
        *cls = w->cls;
        *src = w->src;
    } else {
        const cfa_work *w = (const cfa_work *)v->p + q;
        *cls = w->pad;
        *src = w->src;
    }
}

/* Reorders the items of v (in chunk order) by (class, chunk), stably, and fills
 * first[class * (n_chunks + 1) + chunk] with each group's start. */
static cfa_status partition_by_class(vec *v, uint32_t *first, uint32_t n_chunks, uint64_t S,
                                     char *err, size_t errlen)
{
    if (v->n >= UINT32_MAX) {
        fail(err, errlen, "too many work items; raise slab_bytes");
        return CFA_ERR_INVAL;
    }
    const size_t row = (size_t)n_chunks + 1, nf = (size_t)CFA_N_CLASSES * row;
    for (size_t q = 0; q < v->n; ++q) {
        uint32_t k;
        uint64_t src;
        item_key(v, q, &k, &src);
        first[(size_t)k * row + (size_t)(src / S) + 1]++;
    }
    uint32_t run = 0;
    for (size_t idx = 0; idx < nf; ++idx) {
        if (idx % row == 0) {
            first[idx] = run;
        } else {
            run += first[idx];
            first[idx] = run;
        }
    }
    char *sorted = (char *)malloc((v->n ? v->n : 1) * v->elem);
    uint32_t *cursor = (uint32_t *)malloc(nf * sizeof(uint32_t));
    if (!sorted || !cursor) {
        free(sorted);
        free(cursor);
        return CFA_ERR_NOMEM;
    }
    memcpy(cursor, first, nf * sizeof(uint32_t));
    for (size_t q = 0; q < v->n; ++q) {
        uint32_t k;
        uint64_t src;
        item_key(v, q, &k, &src);
        const uint32_t to = cursor[(size_t)k * row + (size_t)(src / S)]++;
        memcpy(sorted + (size_t)to * v->elem, (const char *)v->p + q * v->elem, v->elem);
    }
    free(cursor);
    free(v->p);
    v->p = sorted;
    return CFA_OK;
}

/* Within each (class, chunk) range of tiny items, the pieces of at most CFA_TINY_SEG_BYTES
 * destination bytes first (stable), so the kernel's warps mostly get pieces of one kind. */
static cfa_status order_tiny(vec *v, const uint32_t *first, uint32_t n_chunks)
{
    if (v->n == 0) return CFA_OK;
    cfa_work *w = (cfa_work *)v->p;
    cfa_work *tmp = (cfa_work *)malloc(v->n * sizeof(cfa_work));
    if (!tmp) return CFA_ERR_NOMEM;
    const size_t row = (size_t)n_chunks + 1;
    for (size_t k = 0; k < CFA_N_CLASSES; ++k) {
        for (size_t c = 0; c < n_chunks; ++c) {
            const uint32_t a = first[k * row + c], b = first[k * row + c + 1];
            size_t o = a;
            for (int pass = 0; pass < 2; ++pass)
                for (uint32_t q = a; q < b; ++q) {
                    const uint64_t bytes = (uint64_t)w[q].n << ((w[q].mode >> 2) & 3u);
                    if ((bytes <= CFA_TINY_SEG_BYTES) == (pass == 0)) tmp[o++] = w[q];
                }
        }
    }
    memcpy(w, tmp, v->n * sizeof(cfa_work));
    free(tmp);
    return CFA_OK;
}

void cfa_host_plan_free(cfa_host_plan *hp)
{
    if (!hp) return;
    if (hp->names) {
        for (size_t i = 0; i < hp->n_entries; ++i) free(hp->names[i]);
    }
    free(hp->names);
    free(hp->entries);
    free(hp->dsts);
    free(hp->pieces);
    free(hp->slabs);
    free(hp->slab_first);
    free(hp->bulk);
    free(hp->bulk_first);
    free(hp->tiny);
    free(hp->tiny_first);
    free(hp->strided);
    free(hp->strided_first);
    free(hp->copies);
    free(hp->copy_first);
    free(hp->layer_last_chunk);
    memset(hp, 0, sizeof *hp);
}

cfa_status cfa_host_plan_build(const cfa_tensor_entry *entries, size_t n_entries,
                               const cfa_dst *dsts, size_t n_dsts, uint64_t blob_bytes,
                               const cfa_plan_opts *opts, cfa_host_plan *out, char *err,
                               size_t errlen)
{
    cfa_status st = CFA_OK;
    ent_info *info = NULL;
    span *spans = NULL;
    dspan *ds = NULL;
    uint64_t *dst_bytes = NULL;
    vec slabs = {0}, bulk = {0}, tiny = {0}, strided = {0};
    if (!out) return CFA_ERR_INVAL;
    memset(out, 0, sizeof *out);
    slabs.elem = bulk.elem = tiny.elem = sizeof(cfa_work);
    strided.elem = sizeof(cfa_swork);

    /* 1. options */
    cfa_plan_opts o;
    if (opts) o = *opts;
    else cfa_plan_opts_default(&o);
    if ((n_entries && !entries) || (n_dsts && !dsts)) {
        fail(err, errlen, "NULL entry or destination array");
        return CFA_ERR_INVAL;
    }
    if (o.chunk_bytes == 0 || o.chunk_bytes % 256 != 0) {
        fail(err, errlen, "chunk_bytes must be a positive multiple of 256 (got %llu)",
             (unsigned long long)o.chunk_bytes);
        return CFA_ERR_INVAL;
    }
    if (o.slab_bytes != 0 &&
        (o.slab_bytes < 4096 || o.slab_bytes % 4096 != 0 || o.slab_bytes > (64u << 20))) {
        fail(err, errlen, "slab_bytes must be 0 or a multiple of 4096 in [4096, 64 MiB]");
        return CFA_ERR_INVAL;
    }
    if (o.tiny_bytes > (1u << 20)) {
        fail(err, errlen, "tiny_bytes must be at most 1 MiB");
        return CFA_ERR_INVAL;
    }
    if (o.host_slots < 0 || o.dev_slots < 0 || o.fill_threads < 0 || o.fill_threads > 256 ||
        o.pull_percent > 100 || o.device < -1) {
        fail(err, errlen, "bad slot, thread or device option");
        return CFA_ERR_INVAL;
    }
    if (o.workspace && o.dev_slots > 0 &&
        o.workspace_bytes / (uint64_t)o.dev_slots < o.chunk_bytes) {
        fail(err, errlen, "workspace too small for %d slots of %llu bytes", o.dev_slots,
             (unsigned long long)o.chunk_bytes);
        return CFA_ERR_INVAL;
    }
    if (o.seg_world == 0) o.seg_world = 1;
    if (o.seg_world < 0 || o.seg_world > 4096 || o.seg_rank < 0 || o.seg_rank >= o.seg_world) {
        fail(err, errlen, "seg_rank %d outside [0, seg_world = %d)", o.seg_rank, o.seg_world);
        return CFA_ERR_INVAL;
    }
    if (o.seg_world > 1 &&
        (!o.gather || o.chunk_bytes % (256ull * (uint64_t)o.seg_world) != 0)) {
        fail(err, errlen, "a segmented plan (seg_world %d) needs a gather function and "
             "chunk_bytes a multiple of 256 * seg_world", o.seg_world);
        return CFA_ERR_INVAL;
    }
    if (o.workspace && ((uintptr_t)o.workspace & 255u)) {
        fail(err, errlen, "workspace must be 256-byte aligned");
        return CFA_ERR_ALIGN;
    }
    if (n_entries >= (size_t)CFA_NO_CK || n_dsts >= (size_t)INT32_MAX) {
        fail(err, errlen, "too many entries or destinations");
        return CFA_ERR_INVAL;
    }
    const uint64_t S = o.chunk_bytes;
    const uint64_t n_chunks64 = blob_bytes / S + (blob_bytes % S != 0);
    if (n_chunks64 >= UINT32_MAX) {
        fail(err, errlen, "blob has too many chunks");
        return CFA_ERR_INVAL;
    }

    /* 1b. destinations */
    dst_bytes = (uint64_t *)calloc(n_dsts ? n_dsts : 1, sizeof(uint64_t));
    ds = (dspan *)calloc(n_dsts ? n_dsts : 1, sizeof(dspan));
    if (!dst_bytes || !ds) { st = CFA_ERR_NOMEM; goto done; }
    for (size_t j = 0; j < n_dsts; ++j) {
        const cfa_dst *d = &dsts[j];
        const int es = cfa_dtype_size(d->dtype);
        if (!es || d->ndim < 0 || d->ndim > CFA_MAX_DIMS) {
            fail(err, errlen, "destination %zu: bad dtype or ndim", j);
            st = CFA_ERR_INVAL;
            goto done;
        }
        uint64_t numel = 1;
        for (int k = 0; k < d->ndim; ++k) {
            if (d->shape[k] < 0 || mul_overflows(numel, (uint64_t)d->shape[k], &numel)) {
                fail(err, errlen, "destination %zu: bad shape", j);
                st = CFA_ERR_INVAL;
                goto done;
            }
        }
        if (mul_overflows(numel, (uint64_t)es, &dst_bytes[j])) {
            fail(err, errlen, "destination %zu: too large", j);
            st = CFA_ERR_INVAL;
            goto done;
        }
        if (dst_bytes[j] && !d->dev_ptr) {
            fail(err, errlen, "destination %zu: NULL pointer", j);
            st = CFA_ERR_INVAL;
            goto done;
        }
        if ((uintptr_t)d->dev_ptr % (uintptr_t)es) {
            fail(err, errlen, "destination %zu: pointer not aligned to its element size", j);
            st = CFA_ERR_ALIGN;
            goto done;
        }
        ds[j].ptr = (uint64_t)(uintptr_t)d->dev_ptr;
        ds[j].len = dst_bytes[j];
        ds[j].idx = (uint32_t)j;
    }
    /* by address; ds[j].idx == j, so the stable order breaks ties by index */
    {
        uint64_t *key = (uint64_t *)calloc(n_dsts ? n_dsts : 1, sizeof(uint64_t));
        if (!key) { st = CFA_ERR_NOMEM; goto done; }
        for (size_t j = 0; j < n_dsts; ++j) key[j] = ds[j].ptr;
        const int r = sort_by_key(ds, n_dsts, sizeof(dspan), key);
        free(key);
        if (r) { st = CFA_ERR_NOMEM; goto done; }
    }
    for (size_t j = 1; j < n_dsts; ++j) {
        const dspan *p = &ds[j - 1], *q = &ds[j];
        if (p->len && q->len && q->ptr < p->ptr + p->len) {
            fail(err, errlen, "destinations %u and %u overlap in memory", p->idx, q->idx);
            st = CFA_ERR_OVERLAP;
            goto done;
        }
    }

    /* 1c. entries */
    info = (ent_info *)calloc(n_entries ? n_entries : 1, sizeof(ent_info));
    if (!info) { st = CFA_ERR_NOMEM; goto done; }
    uint32_t n_layers = 0;
    for (size_t i = 0; i < n_entries; ++i) {
        const cfa_tensor_entry *e = &entries[i];
        const int es_s = cfa_dtype_size(e->src_dtype);
        if (!es_s || e->ndim < 0 || e->ndim > CFA_MAX_DIMS ||
            (e->flags & ~(CFA_ENTRY_CAST_BF16 | CFA_ENTRY_CKSUM | CFA_ENTRY_CONVERT))) {
            fail(err, errlen, "entry %zu (%s): bad dtype, ndim or flags", i, ename(e));
            st = CFA_ERR_INVAL;
            goto done;
        }
        if (e->layer < 0 || e->layer >= CFA_MAX_LAYERS) {
            fail(err, errlen, "entry %zu (%s): layer out of range", i, ename(e));
            st = CFA_ERR_INVAL;
            goto done;
        }
        if ((uint32_t)e->layer + 1 > n_layers) n_layers = (uint32_t)e->layer + 1;
        if (e->dst_index < 0 || (size_t)e->dst_index >= n_dsts) {
            fail(err, errlen, "entry %zu (%s): destination index out of range", i, ename(e));
            st = CFA_ERR_INVAL;
            goto done;
        }
        const cfa_dst *d = &dsts[e->dst_index];
        const int converts = (e->flags & (CFA_ENTRY_CAST_BF16 | CFA_ENTRY_CONVERT)) != 0;
        const int conv = converts ? cfa_conversion(e->src_dtype, d->dtype) : CFA_CONV_NONE;
        if (converts ? (conv == CFA_CONV_NONE ||
                        ((e->flags & CFA_ENTRY_CAST_BF16) && conv != CFA_CONV_F32_BF16))
                     : (e->src_dtype != d->dtype)) {
            fail(err, errlen, "entry %zu (%s): dtype does not match its destination", i,
                 ename(e));
            st = CFA_ERR_DTYPE;
            goto done;
        }
        const int es_d = cfa_dtype_size(d->dtype);
        uint64_t n = 1;
        for (int k = 0; k < e->ndim; ++k) {
            if (e->shape[k] < 0 || mul_overflows(n, (uint64_t)e->shape[k], &n)) {
                fail(err, errlen, "entry %zu (%s): bad shape", i, ename(e));
                st = CFA_ERR_INVAL;
                goto done;
            }
        }
        /* row of the destination */
        uint64_t row = 1;
        if (d->ndim >= 2) {
            row = (uint64_t)d->shape[d->ndim - 1];
            if (n && (e->ndim == 0 || (uint64_t)e->shape[e->ndim - 1] != row)) {
                fail(err, errlen, "entry %zu (%s): last dimension differs from the destination "
                     "row (%llu)", i, ename(e), (unsigned long long)row);
                st = CFA_ERR_SHAPE;
                goto done;
            }
        }
        uint64_t first = 0, src_len = 0, dst_len = 0;
        const uint64_t d_numel = dst_bytes[e->dst_index] / (uint64_t)es_d;
        if (e->dst_row_offset < 0 || mul_overflows((uint64_t)e->dst_row_offset, row, &first) ||
            first > d_numel || n > d_numel - first) {
            fail(err, errlen, "entry %zu (%s): rows fall outside the destination", i, ename(e));
            st = CFA_ERR_OOB;
            goto done;
        }
        if (e->blob_offset % (uint64_t)es_s) {
            fail(err, errlen, "entry %zu (%s): blob offset not a multiple of the element size",
                 i, ename(e));
            st = CFA_ERR_ALIGN;
            goto done;
        }
        /* source layout: rows of `cols` elements, `stride` elements apart */
        const uint64_t cols = e->ndim >= 1 ? (uint64_t)e->shape[e->ndim - 1] : 1;
        if (e->src_row_stride && (e->ndim < 1 || e->src_row_stride < cols)) {
            fail(err, errlen, "entry %zu (%s): source row stride below the row length", i,
                 ename(e));
            st = CFA_ERR_INVAL;
            goto done;
        }
        const uint64_t stride = e->src_row_stride ? e->src_row_stride : cols;
        uint64_t extent_elems = 0;
        if (n && mul_overflows(n / cols - 1, stride, &extent_elems)) extent_elems = UINT64_MAX;
        if (n) extent_elems = extent_elems > UINT64_MAX - cols ? UINT64_MAX : extent_elems + cols;
        if (mul_overflows(extent_elems, (uint64_t)es_s, &src_len) || e->blob_offset > blob_bytes ||
            src_len > blob_bytes - e->blob_offset) {
            fail(err, errlen, "entry %zu (%s): reads past the end of the blob", i, ename(e));
            st = CFA_ERR_OOB;
            goto done;
        }
        dst_len = n * (uint64_t)es_d;
        info[i].n = n;
        info[i].es_s = es_s;
        info[i].es_d = es_d;
        info[i].conv = conv;
        info[i].dst_off = first * (uint64_t)es_d;
        info[i].cols = cols;
        info[i].stride = stride;
        info[i].extent = src_len;
        (void)dst_len;
    }

    /* 2. coverage of every destination */
    spans = (span *)malloc((n_entries ? n_entries : 1) * sizeof(span));
    if (!spans) { st = CFA_ERR_NOMEM; goto done; }
    size_t n_spans = 0;
    for (size_t i = 0; i < n_entries; ++i) {
        if (!info[i].n) continue;
        spans[n_spans].dst = (uint32_t)entries[i].dst_index;
        spans[n_spans].entry = (uint32_t)i;
        spans[n_spans].off = info[i].dst_off;
        spans[n_spans].len = info[i].n * (uint64_t)info[i].es_d;
        n_spans++;
    }
    /* by (destination, offset); spans are in entry order, so the stable order breaks ties by
     * entry.  Both fields go into one key when they fit in 64 bits together. */
    {
        uint64_t max_off = 0;
        for (size_t k = 0; k < n_spans; ++k)
            if (spans[k].off > max_off) max_off = spans[k].off;
        const int ob = bit_width(max_off);
        if (ob + bit_width((uint64_t)n_dsts) <= 64) {
            uint64_t *key = (uint64_t *)calloc(n_spans ? n_spans : 1, sizeof(uint64_t));
            if (!key) { st = CFA_ERR_NOMEM; goto done; }
            for (size_t k = 0; k < n_spans; ++k)
                key[k] = ob == 64 ? spans[k].off : ((uint64_t)spans[k].dst << ob) | spans[k].off;
            const int r = sort_by_key(spans, n_spans, sizeof(span), key);
            free(key);
            if (r) { st = CFA_ERR_NOMEM; goto done; }
        } else {
            qsort(spans, n_spans, sizeof(span), cmp_span);
        }
    }
    {
        size_t k = 0;
        for (size_t j = 0; j < n_dsts; ++j) {
            uint64_t covered = 0; /* bytes [0, covered) are written, without gaps so far */
            int gap = 0;
            for (; k < n_spans && spans[k].dst == j; ++k) {
                if (k > 0 && spans[k - 1].dst == j &&
                    spans[k].off < spans[k - 1].off + spans[k - 1].len) {
                    fail(err, errlen, "entries %u (%s) and %u (%s) overlap in destination %zu",
                         spans[k - 1].entry, ename(&entries[spans[k - 1].entry]),
                         spans[k].entry, ename(&entries[spans[k].entry]), j);
                    st = CFA_ERR_OVERLAP;
                    goto done;
                }
                if (spans[k].off != covered) gap = 1;
                covered = spans[k].off + spans[k].len;
            }
            if ((o.flags & CFA_OPT_STRICT_COVERAGE) && (gap || covered != dst_bytes[j])) {
                fail(err, errlen, "destination %zu is not fully covered", j);
                st = CFA_ERR_COVERAGE;
                goto done;
            }
        }
    }

    /* 3. pieces = tensor x chunk.  A contiguous tensor gives one piece per chunk it touches.
     * A column slice gives one strided piece per run of whole rows inside a chunk, and its rows
     * that cross a chunk boundary are cut into contiguous pieces at the boundary. */
    {
        vec pv = {0};
        pv.elem = sizeof(cfa_piece);
        for (size_t i = 0; i < n_entries; ++i) {
            const ent_info *in = &info[i];
            if (!in->n) continue;
            cfa_piece pc;
            memset(&pc, 0, sizeof pc);
            pc.entry = (uint32_t)i;
            pc.dst_index = (uint32_t)entries[i].dst_index;
            pc.conv = (uint32_t)in->conv;
            pc.rows = 1;
            const uint64_t es_s = (uint64_t)in->es_s, es_d = (uint64_t)in->es_d;
            const uint64_t a0 = entries[i].blob_offset;
            /* contiguous runs [lo, hi) of source bytes whose first element is element e0 */
#define CFA_EMIT_RUN(LO, HI, E0)                                                             \
    do {                                                                                     \
        for (uint64_t c_ = (LO) / S; c_ * S < (HI); ++c_) {                                  \
            const uint64_t lo_ = (LO) > c_ * S ? (LO) : c_ * S;                               \
            const uint64_t hi_ = (HI) < (c_ + 1) * S ? (HI) : (c_ + 1) * S;                   \
            pc.chunk = (uint32_t)c_;                                                         \
            pc.rows = 1;                                                                     \
            pc.src_row_stride = 0;                                                           \
            pc.src_offset = lo_;                                                             \
            pc.n_elems = (hi_ - lo_) / es_s;                                                 \
            pc.dst_offset = in->dst_off + ((E0) + (lo_ - (LO)) / es_s) * es_d;              \
            if (vec_push(&pv, &pc)) { free(pv.p); st = CFA_ERR_NOMEM; goto done; }           \
        }                                                                                    \
    } while (0)
            if (in->stride == in->cols) {
                CFA_EMIT_RUN(a0, a0 + in->n * es_s, 0);
                continue;
            }
            const uint64_t rows = in->n / in->cols;
            const uint64_t row_bytes = in->cols * es_s, step = in->stride * es_s;
            for (uint64_t r = 0; r < rows;) {
                const uint64_t a = a0 + r * step;
                const uint64_t c = a / S;
                if (a + row_bytes <= (c + 1) * S) {
                    /* rows r .. r+k-1 lie entirely inside chunk c */
                    uint64_t k = 1 + ((c + 1) * S - (a + row_bytes)) / step;
                    if (k > rows - r) k = rows - r;
                    if (k > UINT32_MAX) k = UINT32_MAX;
                    pc.chunk = (uint32_t)c;
                    pc.src_offset = a;
                    pc.rows = (uint32_t)k;
                    pc.src_row_stride = k > 1 ? (uint32_t)in->stride : 0;
                    pc.n_elems = k * in->cols;
                    pc.dst_offset = in->dst_off + r * in->cols * es_d;
                    if (vec_push(&pv, &pc)) { free(pv.p); st = CFA_ERR_NOMEM; goto done; }
                    r += k;
                } else {
                    CFA_EMIT_RUN(a, a + row_bytes, r * in->cols);
                    r += 1;
                }
            }
#undef CFA_EMIT_RUN
        }
        out->pieces = (cfa_piece *)pv.p;
        out->n_pieces = pv.n;
        if (!out->pieces) {
            out->pieces = (cfa_piece *)malloc(sizeof(cfa_piece));
            if (!out->pieces) { st = CFA_ERR_NOMEM; goto done; }
        }
    }
    const size_t n_pieces = out->n_pieces;
    /* by (chunk, blob offset, entry): a piece's chunk is its blob offset / S and the pieces were
     * made in entry order, so a stable order by blob offset is that order */
    {
        uint64_t *key = (uint64_t *)calloc(n_pieces ? n_pieces : 1, sizeof(uint64_t));
        if (!key) { st = CFA_ERR_NOMEM; goto done; }
        for (size_t q = 0; q < n_pieces; ++q) key[q] = out->pieces[q].src_offset;
        const int r = sort_by_key(out->pieces, n_pieces, sizeof(cfa_piece), key);
        free(key);
        if (r) { st = CFA_ERR_NOMEM; goto done; }
    }

    /* 4. work items, ordered by (class, chunk) */
    const uint32_t n_chunks = (uint32_t)n_chunks64;
    const size_t nf = (size_t)CFA_N_CLASSES * ((size_t)n_chunks + 1);
    out->slab_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    out->bulk_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    out->tiny_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    out->strided_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    if (!out->slab_first || !out->bulk_first || !out->tiny_first || !out->strided_first) {
        st = CFA_ERR_NOMEM;
        goto done;
    }
    if (o.slab_bytes == 0) {
        uint64_t dst_total = 0;
        for (size_t i = 0; i < n_entries; ++i) dst_total += info[i].n * (uint64_t)info[i].es_d;
        o.slab_bytes = cfa_auto_slab(dst_total);
    }
    {
        const int use_bulk = CFA_BULK_READY && (o.flags & CFA_OPT_BULK);
        const uint64_t slab = o.slab_bytes;
        /* pass 1: items in chunk order, tagged with their class */
        for (size_t p = 0; p < n_pieces; ++p) {
            const cfa_piece *pc = &out->pieces[p];
            const ent_info *in = &info[pc->entry];
            const cfa_tensor_entry *e = &entries[pc->entry];
            const uint32_t ck = (e->flags & CFA_ENTRY_CKSUM) ? pc->entry : CFA_NO_CK;
            const uint32_t mode = CFA_MODE(log2_small(in->es_s), log2_small(in->es_d), pc->conv);
            const uint32_t cls =
                pc->conv ? CFA_CLASS_OF_CONV(pc->conv) : (uint32_t)log2_small(in->es_s);
            const uint64_t a0 = (uint64_t)(uintptr_t)dsts[pc->dst_index].dev_ptr + pc->dst_offset;
            if (pc->rows > 1) {
                /* blocks of whole rows, about slab_bytes of destination each */
                const uint64_t row_d = in->cols * (uint64_t)in->es_d;
                uint64_t per = row_d ? slab / row_d : 1;
                if (per == 0) per = 1;
                for (uint64_t r = 0; r < pc->rows; r += per) {
                    const uint64_t k = pc->rows - r < per ? pc->rows - r : per;
                    cfa_swork sw;
                    memset(&sw, 0, sizeof sw);
                    sw.src = pc->src_offset + r * in->stride * (uint64_t)in->es_s;
                    sw.dst = a0 + r * row_d;
                    sw.rows = (uint32_t)k;
                    sw.cols = (uint32_t)in->cols;
                    sw.stride = (uint32_t)in->stride;
                    sw.ck = ck;
                    sw.mode = mode;
                    sw.cls = cls;
                    if (vec_push(&strided, &sw)) { st = CFA_ERR_NOMEM; goto done; }
                }
                continue;
            }
            cfa_work w;
            memset(&w, 0, sizeof w);
            w.ck = ck;
            w.mode = mode;
            w.pad = cls;
            const uint64_t nb = pc->n_elems * (uint64_t)in->es_d;
            if (nb < o.tiny_bytes) {
                /* warp-level items of at most CFA_TINY_SEG_BYTES destination bytes, cut at
                 * destination addresses that are multiples of it: each is one 8-lane segment's
                 * single round of loads, where a whole warp would take a larger piece in
                 * several dependent rounds (a piece is bound by latency, not bandwidth) */
                uint64_t pos = a0;
                const uint64_t end = a0 + nb;
                while (pos < end) {
                    uint64_t next = (pos / CFA_TINY_SEG_BYTES + 1) * CFA_TINY_SEG_BYTES;
                    if (next > end) next = end;
                    w.src = pc->src_offset + (pos - a0) / (uint64_t)in->es_d * (uint64_t)in->es_s;
                    w.dst = pos;
                    w.n = (uint32_t)((next - pos) / (uint64_t)in->es_d);
                    if (vec_push(&tiny, &w)) { st = CFA_ERR_NOMEM; goto done; }
                    pos = next;
                }
                continue;
            }
            uint64_t pos = a0;
            const uint64_t end = a0 + nb;
            while (pos < end) {
                uint64_t next = (pos / slab + 1) * slab;
                if (next - pos < slab / 2) next += slab;
                if (next >= end || end - next < slab / 2) next = end;
                w.dst = pos;
                w.src = pc->src_offset + (pos - a0) / (uint64_t)in->es_d * (uint64_t)in->es_s;
                w.n = (uint32_t)((next - pos) / (uint64_t)in->es_d);
                const int aligned = ((w.src | w.dst | (next - pos)) & 15u) == 0;
                if (use_bulk && !pc->conv && aligned) {
                    if (vec_push(&bulk, &w)) { st = CFA_ERR_NOMEM; goto done; }
                } else {
                    if (vec_push(&slabs, &w)) { st = CFA_ERR_NOMEM; goto done; }
                }
                pos = next;
            }
        }
        /* pass 2: stable partition by class (items are in chunk order already) */
        if ((st = partition_by_class(&slabs, out->slab_first, n_chunks, S, err, errlen))) goto done;
        if ((st = partition_by_class(&bulk, out->bulk_first, n_chunks, S, err, errlen))) goto done;
        if ((st = partition_by_class(&tiny, out->tiny_first, n_chunks, S, err, errlen))) goto done;
        if ((st = order_tiny(&tiny, out->tiny_first, n_chunks))) goto done;
        if ((st = partition_by_class(&strided, out->strided_first, n_chunks, S, err, errlen)))
            goto done;
    }

    /* 4b. what each chunk's pieces read: contiguous ranges merged across gaps of at most
     * kCopyGap bytes, and column slices that would move more than twice their bytes as
     * strided 2-D copies.  A segmented plan instead copies this rank's whole segment of every
     * chunk (the other ranks may read any of its bytes). */
    out->copy_first = (uint32_t *)calloc((size_t)n_chunks + 1, sizeof(uint32_t));
    if (!out->copy_first) { st = CFA_ERR_NOMEM; goto done; }
    if (o.seg_world > 1) {
        out->copies = (cfa_copy *)calloc(n_chunks ? n_chunks : 1, sizeof(cfa_copy));
        if (!out->copies) { st = CFA_ERR_NOMEM; goto done; }
        for (uint32_t c = 0; c < n_chunks; ++c) {
            uint64_t lo = 0, len = 0;
            cfa_segment_range(blob_bytes, S, o.seg_world, o.seg_rank, c, &lo, &len);
            out->copy_first[c] = (uint32_t)out->n_copies;
            if (!len) continue;
            cfa_copy *cp = &out->copies[out->n_copies++];
            cp->src = lo;
            cp->width = cp->pitch = len;
            cp->rows = 1;
            out->staged_bytes += len;
        }
        out->copy_first[n_chunks] = (uint32_t)out->n_copies;
    } else {
        const uint64_t kCopyGap = 1ull << 20;
        vec cv = {0};
        cv.elem = sizeof(cfa_copy);
        size_t p = 0;
        for (uint32_t c = 0; c < n_chunks; ++c) {
            out->copy_first[c] = (uint32_t)cv.n;
            cfa_copy open;
            int have = 0;
            for (; p < n_pieces && out->pieces[p].chunk == c; ++p) {
                const cfa_piece *pc = &out->pieces[p];
                const uint64_t es = (uint64_t)info[pc->entry].es_s;
                cfa_copy seg;
                memset(&seg, 0, sizeof seg);
                seg.src = pc->src_offset;
                seg.rows = 1;
                if (pc->rows > 1) {
                    const uint64_t width = pc->n_elems / pc->rows * es;
                    const uint64_t pitch = (uint64_t)pc->src_row_stride * es;
                    if (2 * width < pitch) {
                        seg.width = width;
                        seg.pitch = pitch;
                        seg.rows = pc->rows;
                        if (have && vec_push(&cv, &open)) { free(cv.p); st = CFA_ERR_NOMEM; goto done; }
                        have = 0;
                        if (vec_push(&cv, &seg)) { free(cv.p); st = CFA_ERR_NOMEM; goto done; }
                        continue;
                    }
                    seg.width = (pc->rows - 1) * pitch + width;
                } else {
                    seg.width = pc->n_elems * es;
                }
                seg.pitch = seg.width;
                if (have && seg.src <= open.src + open.width + kCopyGap) {
                    const uint64_t end = seg.src + seg.width > open.src + open.width
                                             ? seg.src + seg.width
                                             : open.src + open.width;
                    open.width = end - open.src;
                    open.pitch = open.width;
                } else {
                    if (have && vec_push(&cv, &open)) { free(cv.p); st = CFA_ERR_NOMEM; goto done; }
                    open = seg;
                    have = 1;
                }
            }
            if (have && vec_push(&cv, &open)) { free(cv.p); st = CFA_ERR_NOMEM; goto done; }
        }
        out->copy_first[n_chunks] = (uint32_t)cv.n;
        out->copies = (cfa_copy *)cv.p;
        out->n_copies = cv.n;
        for (size_t k = 0; k < cv.n; ++k)
            out->staged_bytes += out->copies[k].width * out->copies[k].rows;
    }

    /* 5. readiness groups: last chunk carrying one of their bytes */
    out->layer_last_chunk = (int64_t *)malloc((n_layers ? n_layers : 1) * sizeof(int64_t));
    if (!out->layer_last_chunk) { st = CFA_ERR_NOMEM; goto done; }
    for (uint32_t l = 0; l < n_layers; ++l) out->layer_last_chunk[l] = -1;
    for (size_t i = 0; i < n_entries; ++i) {
        if (!info[i].n) continue;
        const uint64_t last = (entries[i].blob_offset + info[i].extent - 1) / S;
        int64_t *slot = &out->layer_last_chunk[entries[i].layer];
        if ((int64_t)last > *slot) *slot = (int64_t)last;
        out->bytes_read += info[i].n * (uint64_t)info[i].es_s;
        out->bytes_written += info[i].n * (uint64_t)info[i].es_d;
        if (entries[i].flags & CFA_ENTRY_CKSUM) out->any_cksum = 1;
    }

    /* copies the plan keeps */
    out->entries = (cfa_tensor_entry *)malloc((n_entries ? n_entries : 1) * sizeof(cfa_tensor_entry));
    out->names = (char **)calloc(n_entries ? n_entries : 1, sizeof(char *));
    out->dsts = (cfa_dst *)malloc((n_dsts ? n_dsts : 1) * sizeof(cfa_dst));
    if (!out->entries || !out->names || !out->dsts) { st = CFA_ERR_NOMEM; goto done; }
    if (n_entries) memcpy(out->entries, entries, n_entries * sizeof(cfa_tensor_entry));
    if (n_dsts) memcpy(out->dsts, dsts, n_dsts * sizeof(cfa_dst));
    out->n_entries = n_entries; /* set now so that cfa_host_plan_free frees the names */
    for (size_t i = 0; i < n_entries; ++i) {
        if (entries[i].name) {
            out->names[i] = dup_str(entries[i].name);
            if (!out->names[i]) { st = CFA_ERR_NOMEM; goto done; }
        }
        out->entries[i].name = out->names[i];
    }

    out->opts = o;
    out->blob_bytes = blob_bytes;
    out->chunk_bytes = S;
    out->n_chunks = n_chunks;
    out->n_layers = n_layers;
    out->n_dsts = n_dsts;
    out->slabs = (cfa_work *)slabs.p;
    out->n_slabs = slabs.n;
    out->bulk = (cfa_work *)bulk.p;
    out->n_bulk = bulk.n;
    out->tiny = (cfa_work *)tiny.p;
    out->n_tiny = tiny.n;
    out->strided = (cfa_swork *)strided.p;
    out->n_strided = strided.n;
    slabs.p = bulk.p = tiny.p = strided.p = NULL;

done:
    free(info);
    free(spans);
    free(ds);
    free(dst_bytes);
    free(slabs.p);
    free(bulk.p);
    free(tiny.p);
    free(strided.p);
    if (st != CFA_OK) cfa_host_plan_free(out);
    return st;
}
