/* Replays manifests through the host plan builder (paper_2607_18957_gb300/csrc/cfa_plan.c) built
 * with AddressSanitizer and UBSan, so that an out-of-bounds access, a leak or undefined behaviour
 * aborts the run.  Every accepted plan is checked against its own inputs:
 *   - each piece lies inside its chunk and the blob, and inside its destination, and the pieces
 *     are ordered by (chunk, blob offset, entry);
 *   - each work item reads inside the blob and writes inside exactly one destination;
 *   - each class/chunk range table is monotone and ends at the item count.
 * Input file: records of
 *   [u64 n_entries][u64 n_dsts][u64 blob_bytes][u64 chunk_bytes][u32 slab][u32 tiny][u32 flags]
 *   [u32 0][n_entries x cfa_tensor_entry (name = 0)][n_dsts x cfa_dst]
 * Exit status 0 when every record is handled and both outcomes occur. */
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "cfa_internal.h"

void cfa_internal_set_error(const char *msg) { (void)msg; }

static const cfa_dst *g_dsts;
static size_t g_n_dsts;

/* Destination j holding bytes [a, a + len), or -1. */
static long owner(uint64_t a, uint64_t len)
{
    for (size_t j = 0; j < g_n_dsts; ++j) {
        const uint64_t base = (uint64_t)(uintptr_t)g_dsts[j].dev_ptr;
        uint64_t bytes = (uint64_t)cfa_dtype_size(g_dsts[j].dtype);
        for (int k = 0; k < g_dsts[j].ndim; ++k) bytes *= (uint64_t)g_dsts[j].shape[k];
        if (a >= base && len <= bytes && a - base <= bytes - len) return (long)j;
    }
    return -1;
}

static int check_items(const cfa_work *w, size_t n, const uint32_t *first, uint32_t n_chunks,
                       uint64_t blob)
{
    for (size_t q = 0; q < n; ++q) {
        const uint64_t es_s = 1ull << (w[q].mode & 3u), es_d = 1ull << ((w[q].mode >> 2) & 3u);
        if (w[q].src > blob || (uint64_t)w[q].n * es_s > blob - w[q].src) return 10;
        if (w[q].n && owner(w[q].dst, (uint64_t)w[q].n * es_d) < 0) return 11;
    }
    const size_t row = (size_t)n_chunks + 1;
    for (size_t k = 0; k < CFA_N_CLASSES; ++k)
        for (size_t c = 0; c < n_chunks; ++c)
            if (first[k * row + c] > first[k * row + c + 1]) return 12;
    if (first[(CFA_N_CLASSES - 1) * row + n_chunks] != n) return 13;
    return 0;
}

static int check_plan(const cfa_host_plan *hp)
{
    const uint64_t S = hp->chunk_bytes, blob = hp->blob_bytes;
    for (size_t i = 0; i < hp->n_pieces; ++i) {
        const cfa_piece *p = &hp->pieces[i];
        const cfa_tensor_entry *e = &hp->entries[p->entry];
        const uint64_t es_s = (uint64_t)cfa_dtype_size(e->src_dtype);
        const uint64_t es_d = (uint64_t)cfa_dtype_size(hp->dsts[p->dst_index].dtype);
        const uint64_t rows = p->rows ? p->rows : 1, cols = p->n_elems / rows;
        const uint64_t step = rows > 1 ? (uint64_t)p->src_row_stride : cols;
        const uint64_t end = p->src_offset + ((rows - 1) * step + cols) * es_s;
        if (p->chunk >= hp->n_chunks || p->src_offset / S != p->chunk) return 20;
        if (end > blob || (end - 1) / S != p->chunk) return 21;
        const uint64_t base = (uint64_t)(uintptr_t)hp->dsts[p->dst_index].dev_ptr;
        if (owner(base + p->dst_offset, p->n_elems * es_d) != (long)p->dst_index) return 22;
        if (i) { /* ordered by (chunk, blob offset, entry), as the copy ranges are walked */
            const cfa_piece *q = p - 1;
            if (q->chunk > p->chunk ||
                (q->chunk == p->chunk && (q->src_offset > p->src_offset ||
                                          (q->src_offset == p->src_offset && q->entry >= p->entry))))
                return 23;
        }
    }
    int r;
    if ((r = check_items(hp->slabs, hp->n_slabs, hp->slab_first, hp->n_chunks, blob))) return r;
    if ((r = check_items(hp->bulk, hp->n_bulk, hp->bulk_first, hp->n_chunks, blob))) return r;
    if ((r = check_items(hp->tiny, hp->n_tiny, hp->tiny_first, hp->n_chunks, blob))) return r;
    for (size_t q = 0; q < hp->n_strided; ++q) {
        const cfa_swork *w = &hp->strided[q];
        const uint64_t es_s = 1ull << (w->mode & 3u), es_d = 1ull << ((w->mode >> 2) & 3u);
        const uint64_t end = w->src + ((uint64_t)(w->rows - 1) * w->stride + w->cols) * es_s;
        if (!w->rows || end > blob) return 30;
        if (owner(w->dst, (uint64_t)w->rows * w->cols * es_d) < 0) return 31;
    }
    return 0;
}

int main(int argc, char **argv)
{
    if (argc < 2) return 2;
    FILE *f = fopen(argv[1], "rb");
    if (!f) return 2;
    unsigned long accepted = 0, rejected = 0;
    for (;;) {
        uint64_t hdr[4];
        uint32_t o32[4];
        if (fread(hdr, 8, 4, f) != 4 || fread(o32, 4, 4, f) != 4) break;
        const size_t ne = (size_t)hdr[0], nd = (size_t)hdr[1];
        /* exact-size allocations, so that ASan sees any read past the arrays */
        cfa_tensor_entry *e = (cfa_tensor_entry *)malloc(ne ? ne * sizeof *e : 1);
        cfa_dst *d = (cfa_dst *)malloc(nd ? nd * sizeof *d : 1);
        if (!e || !d || fread(e, sizeof *e, ne, f) != ne || fread(d, sizeof *d, nd, f) != nd)
            return 2;
        cfa_plan_opts o;
        cfa_plan_opts_default(&o);
        o.chunk_bytes = hdr[3];
        o.slab_bytes = o32[0];
        o.tiny_bytes = o32[1];
        o.flags = o32[2] | CFA_OPT_HOST_ONLY;
        cfa_host_plan hp;
        char err[256];
        const cfa_status st =
            cfa_host_plan_build(ne ? e : NULL, ne, nd ? d : NULL, nd, hdr[2], &o, &hp, err,
                                sizeof err);
        if (st == CFA_OK) {
            g_dsts = d;
            g_n_dsts = nd;
            const int r = check_plan(&hp);
            cfa_host_plan_free(&hp);
            if (r) {
                fprintf(stderr, "record %lu: check %d failed\n", accepted + rejected, r);
                free(e);
                free(d);
                fclose(f);
                return r;
            }
            accepted++;
        } else {
            rejected++;
        }
        free(e);
        free(d);
    }
    fclose(f);
    printf("accepted %lu rejected %lu\n", accepted, rejected);
    return accepted && rejected ? 0 : 5;
}
