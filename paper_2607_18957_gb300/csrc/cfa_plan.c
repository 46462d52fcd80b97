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
 *   4. turn pieces into work items: pieces below `tiny_bytes` destination bytes become one
 *      warp-level item each; larger ones are split into block-level slabs whose cuts fall on
 *      destination addresses that are multiples of `slab_bytes`, so only a piece's first and
 *      last slab can start or end off a 16-byte boundary;
 *   5. record, per readiness group, the last chunk that carries one of its bytes.
 */
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
    default: return 0;
    }
}

static int log2_small(int x) { return x == 1 ? 0 : x == 2 ? 1 : x == 4 ? 2 : 3; }

void cfa_plan_opts_default(cfa_plan_opts *o)
{
    if (!o) return;
    memset(o, 0, sizeof *o);
    o->chunk_bytes = 512ull << 20;
    o->host_slots = 2;
    o->dev_slots = 2;
    o->fill_threads = 8;
    o->device = -1;
    o->slab_bytes = 65536;
    o->tiny_bytes = 8192;
    o->flags = CFA_OPT_STRICT_COVERAGE;
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

typedef struct {
    uint64_t n;       /* elements */
    int es_s, es_d;   /* element sizes */
    uint64_t dst_off; /* byte offset inside the destination */
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

static int cmp_dspan(const void *a, const void *b)
{
    const dspan *x = (const dspan *)a, *y = (const dspan *)b;
    if (x->ptr != y->ptr) return x->ptr < y->ptr ? -1 : 1;
    return (x->idx > y->idx) - (x->idx < y->idx);
}

static int cmp_piece(const void *a, const void *b)
{
    const cfa_piece *x = (const cfa_piece *)a, *y = (const cfa_piece *)b;
    if (x->chunk != y->chunk) return x->chunk < y->chunk ? -1 : 1;
    if (x->src_offset != y->src_offset) return x->src_offset < y->src_offset ? -1 : 1;
    return (x->entry > y->entry) - (x->entry < y->entry);
}

static int mul_overflows(uint64_t a, uint64_t b, uint64_t *out)
{
    if (a != 0 && b > UINT64_MAX / a) return 1;
    *out = a * b;
    return 0;
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
    vec slabs = {0}, bulk = {0}, tiny = {0};
    if (!out) return CFA_ERR_INVAL;
    memset(out, 0, sizeof *out);
    slabs.elem = bulk.elem = tiny.elem = sizeof(cfa_work);

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
    if (o.slab_bytes < 4096 || o.slab_bytes % 4096 != 0 || o.slab_bytes > (64u << 20)) {
        fail(err, errlen, "slab_bytes must be a multiple of 4096 in [4096, 64 MiB]");
        return CFA_ERR_INVAL;
    }
    if (o.tiny_bytes > (1u << 20)) {
        fail(err, errlen, "tiny_bytes must be at most 1 MiB");
        return CFA_ERR_INVAL;
    }
    if (o.host_slots < 0 || o.dev_slots < 0 || o.fill_threads < 0 || o.fill_threads > 256 ||
        o.reserved != 0 || o.device < -1) {
        fail(err, errlen, "bad slot, thread or device option");
        return CFA_ERR_INVAL;
    }
    if (o.workspace && o.dev_slots > 0 &&
        o.workspace_bytes / (uint64_t)o.dev_slots < o.chunk_bytes) {
        fail(err, errlen, "workspace too small for %d slots of %llu bytes", o.dev_slots,
             (unsigned long long)o.chunk_bytes);
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
    qsort(ds, n_dsts, sizeof(dspan), cmp_dspan);
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
        if (!es_s || e->ndim < 0 || e->ndim > CFA_MAX_DIMS || e->reserved ||
            (e->flags & ~(CFA_ENTRY_CAST_BF16 | CFA_ENTRY_CKSUM))) {
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
        const int cast = (e->flags & CFA_ENTRY_CAST_BF16) != 0;
        if (cast ? (e->src_dtype != CFA_DTYPE_F32 || d->dtype != CFA_DTYPE_BF16)
                 : (e->src_dtype != d->dtype)) {
            fail(err, errlen, "entry %zu (%s): dtype does not match its destination", i,
                 ename(e));
            st = CFA_ERR_DTYPE;
            goto done;
        }
        const int es_d = cast ? 2 : es_s;
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
        src_len = n * (uint64_t)es_s; /* cannot overflow: n <= d_numel and es_s <= 8 ... */
        dst_len = n * (uint64_t)es_d;
        if (src_len / (uint64_t)es_s != n || e->blob_offset > blob_bytes ||
            src_len > blob_bytes - e->blob_offset) {
            fail(err, errlen, "entry %zu (%s): reads past the end of the blob", i, ename(e));
            st = CFA_ERR_OOB;
            goto done;
        }
        info[i].n = n;
        info[i].es_s = es_s;
        info[i].es_d = es_d;
        info[i].dst_off = first * (uint64_t)es_d;
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
    qsort(spans, n_spans, sizeof(span), cmp_span);
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

    /* 3. pieces = tensor x chunk */
    size_t n_pieces = 0;
    for (size_t i = 0; i < n_entries; ++i) {
        if (!info[i].n) continue;
        const uint64_t a = entries[i].blob_offset;
        const uint64_t b = a + info[i].n * (uint64_t)info[i].es_s;
        n_pieces += (size_t)((b - 1) / S - a / S + 1);
    }
    out->pieces = (cfa_piece *)malloc((n_pieces ? n_pieces : 1) * sizeof(cfa_piece));
    if (!out->pieces) { st = CFA_ERR_NOMEM; goto done; }
    {
        size_t p = 0;
        for (size_t i = 0; i < n_entries; ++i) {
            if (!info[i].n) continue;
            const uint64_t a = entries[i].blob_offset;
            const uint64_t b = a + info[i].n * (uint64_t)info[i].es_s;
            for (uint64_t c = a / S; c * S < b; ++c) {
                const uint64_t lo = a > c * S ? a : c * S;
                const uint64_t hi = b < (c + 1) * S ? b : (c + 1) * S;
                cfa_piece *pc = &out->pieces[p++];
                pc->chunk = (uint32_t)c;
                pc->entry = (uint32_t)i;
                pc->src_offset = lo;
                pc->dst_index = (uint32_t)entries[i].dst_index;
                pc->cast = (entries[i].flags & CFA_ENTRY_CAST_BF16) ? 1u : 0u;
                pc->dst_offset = info[i].dst_off +
                                 (lo - a) / (uint64_t)info[i].es_s * (uint64_t)info[i].es_d;
                pc->n_elems = (hi - lo) / (uint64_t)info[i].es_s;
            }
        }
    }
    qsort(out->pieces, n_pieces, sizeof(cfa_piece), cmp_piece);
    out->n_pieces = n_pieces;

    /* 4. work items, ordered by (class, chunk) */
    const uint32_t n_chunks = (uint32_t)n_chunks64;
    const size_t nf = (size_t)CFA_N_CLASSES * ((size_t)n_chunks + 1);
    out->slab_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    out->bulk_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    out->tiny_first = (uint32_t *)calloc(nf, sizeof(uint32_t));
    if (!out->slab_first || !out->bulk_first || !out->tiny_first) { st = CFA_ERR_NOMEM; goto done; }
    {
        const int use_bulk = CFA_BULK_READY && (o.flags & CFA_OPT_BULK);
        const uint64_t slab = o.slab_bytes;
        /* pass 1: items in chunk order, tagged with their class in `pad` */
        for (size_t p = 0; p < n_pieces; ++p) {
            const cfa_piece *pc = &out->pieces[p];
            const ent_info *in = &info[pc->entry];
            const cfa_tensor_entry *e = &entries[pc->entry];
            cfa_work w;
            memset(&w, 0, sizeof w);
            w.ck = (e->flags & CFA_ENTRY_CKSUM) ? pc->entry : CFA_NO_CK;
            w.mode = CFA_MODE(log2_small(in->es_s), log2_small(in->es_d), pc->cast);
            w.pad = pc->cast ? CFA_CLASS_CAST : (uint32_t)log2_small(in->es_s);
            const uint64_t a0 = (uint64_t)(uintptr_t)dsts[pc->dst_index].dev_ptr + pc->dst_offset;
            const uint64_t nb = pc->n_elems * (uint64_t)in->es_d;
            if (nb < o.tiny_bytes) {
                w.src = pc->src_offset;
                w.dst = a0;
                w.n = (uint32_t)pc->n_elems;
                if (vec_push(&tiny, &w)) { st = CFA_ERR_NOMEM; goto done; }
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
                if (use_bulk && !pc->cast && aligned) {
                    if (vec_push(&bulk, &w)) { st = CFA_ERR_NOMEM; goto done; }
                } else {
                    if (vec_push(&slabs, &w)) { st = CFA_ERR_NOMEM; goto done; }
                }
                pos = next;
            }
        }
        /* pass 2: stable partition by class (items are in chunk order already) */
        vec *lists[3] = {&slabs, &bulk, &tiny};
        uint32_t *firsts[3] = {out->slab_first, out->bulk_first, out->tiny_first};
        for (int li = 0; li < 3; ++li) {
            vec *v = lists[li];
            if (v->n >= UINT32_MAX) {
                fail(err, errlen, "too many work items; raise slab_bytes");
                st = CFA_ERR_INVAL;
                goto done;
            }
            cfa_work *src_items = (cfa_work *)v->p;
            cfa_work *sorted = (cfa_work *)malloc((v->n ? v->n : 1) * sizeof(cfa_work));
            if (!sorted) { st = CFA_ERR_NOMEM; goto done; }
            /* count per (class, chunk) */
            uint32_t *first = firsts[li];
            for (size_t q = 0; q < v->n; ++q) {
                const uint32_t k = src_items[q].pad;
                const uint64_t blob_off = src_items[q].src;
                const uint32_t c = (uint32_t)(blob_off / S);
                first[(size_t)k * (n_chunks + 1) + c + 1]++;
            }
            /* exclusive prefix over the (class, chunk) grid */
            uint32_t run = 0;
            for (size_t k = 0; k < CFA_N_CLASSES; ++k) {
                for (uint32_t c = 0; c <= n_chunks; ++c) {
                    const size_t idx = k * ((size_t)n_chunks + 1) + c;
                    if (c == 0) {
                        first[idx] = run;
                    } else {
                        run += first[idx];
                        first[idx] = run;
                    }
                }
            }
            /* scatter, keeping chunk order inside each class */
            uint32_t *cursor = (uint32_t *)malloc(nf * sizeof(uint32_t));
            if (!cursor) { free(sorted); st = CFA_ERR_NOMEM; goto done; }
            memcpy(cursor, first, nf * sizeof(uint32_t));
            for (size_t q = 0; q < v->n; ++q) {
                const uint32_t k = src_items[q].pad;
                const uint32_t c = (uint32_t)(src_items[q].src / S);
                sorted[cursor[(size_t)k * (n_chunks + 1) + c]++] = src_items[q];
            }
            free(cursor);
            free(v->p);
            v->p = sorted;
        }
    }

    /* 5. readiness groups: last chunk carrying one of their bytes */
    out->layer_last_chunk = (int64_t *)malloc((n_layers ? n_layers : 1) * sizeof(int64_t));
    if (!out->layer_last_chunk) { st = CFA_ERR_NOMEM; goto done; }
    for (uint32_t l = 0; l < n_layers; ++l) out->layer_last_chunk[l] = -1;
    for (size_t i = 0; i < n_entries; ++i) {
        if (!info[i].n) continue;
        const uint64_t last =
            (entries[i].blob_offset + info[i].n * (uint64_t)info[i].es_s - 1) / S;
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
    slabs.p = bulk.p = tiny.p = NULL;

done:
    free(info);
    free(spans);
    free(ds);
    free(dst_bytes);
    free(slabs.p);
    free(bulk.p);
    free(tiny.p);
    if (st != CFA_OK) cfa_host_plan_free(out);
    return st;
}
