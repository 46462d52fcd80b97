/* A plain C program that uses the loader through include/cfa.h only, linked against libcfa.so:
 * the header must compile as strict C, the library's struct sizes must agree with this
 * compiler's, and a host-only plan (no CUDA call) must give the pieces worked out by hand
 * below.  Exit status 0 on success, else the number of the failed check. */
#include <stdio.h>
#include <string.h>

#include "cfa.h"

#define CHECK(n, cond)                                                                        \
    do {                                                                                      \
        if (!(cond)) {                                                                        \
            fprintf(stderr, "check %d failed: %s (%s)\n", n, #cond, cfa_last_error(NULL));    \
            return n;                                                                         \
        }                                                                                     \
    } while (0)

static cfa_tensor_entry entry(const char *name, int64_t rows, uint64_t off, int64_t row_off)
{
    cfa_tensor_entry e;
    memset(&e, 0, sizeof e);
    e.name = name;
    e.src_dtype = CFA_DTYPE_BF16;
    e.ndim = 2;
    e.shape[0] = rows;
    e.shape[1] = 8;
    e.blob_offset = off;
    e.dst_index = 0;
    e.dst_row_offset = row_off;
    e.flags = CFA_ENTRY_CKSUM;
    e.layer = 1;
    return e;
}

/* A host-only plan never loads, so its gather step is never called. */
static int gather_never_called(void *user, void *chunk_dev, uint64_t segment_bytes, int32_t world,
                               int32_t rank, uint32_t chunk, cfa_stream stream)
{
    (void)user;
    (void)chunk_dev;
    (void)segment_bytes;
    (void)world;
    (void)rank;
    (void)chunk;
    (void)stream;
    return 1;
}

int main(void)
{
    CHECK(1, cfa_abi_sizeof("cfa_tensor_entry") == sizeof(cfa_tensor_entry));
    CHECK(2, cfa_abi_sizeof("cfa_dst") == sizeof(cfa_dst));
    CHECK(3, cfa_abi_sizeof("cfa_plan_opts") == sizeof(cfa_plan_opts));
    CHECK(4, cfa_abi_sizeof("cfa_source") == sizeof(cfa_source));
    CHECK(5, cfa_abi_sizeof("cfa_piece") == sizeof(cfa_piece));
    CHECK(6, cfa_abi_sizeof("cfa_stats") == sizeof(cfa_stats));

    /* q [8, 8], k [2, 8], v [2, 8] (bf16) into one fused qkv [12, 8]; q starts at blob byte
     * 200, so with 256-byte chunks it is cut at byte 256 into 28 + 36 elements */
    cfa_tensor_entry e[3];
    e[0] = entry("q", 8, 200, 0);
    e[1] = entry("k", 2, 328, 8);
    e[2] = entry("v", 2, 360, 10);
    cfa_dst d;
    memset(&d, 0, sizeof d);
    d.dev_ptr = (void *)(uintptr_t)0x100000; /* never dereferenced by a host-only plan */
    d.dtype = CFA_DTYPE_BF16;
    d.ndim = 2;
    d.shape[0] = 12;
    d.shape[1] = 8;
    cfa_plan_opts o;
    cfa_plan_opts_default(&o);
    o.chunk_bytes = 256;
    o.flags |= CFA_OPT_HOST_ONLY;
    cfa_plan *plan = NULL;
    CHECK(10, cfa_plan_create(e, 3, &d, 1, 392, &o, &plan) == CFA_OK && plan);
    uint64_t n_layers = 0, n_pieces = 0, n_chunks = 0;
    CHECK(11, cfa_plan_info(plan, &n_layers, &n_pieces, &n_chunks) == CFA_OK);
    CHECK(12, n_layers == 2 && n_pieces == 4 && n_chunks == 2);
    cfa_piece p[8];
    size_t got = 0;
    CHECK(13, cfa_plan_get_pieces(plan, p, 8, &got) == CFA_OK && got == 4);
    /* (chunk, entry, blob offset, destination byte offset, elements), by chunk then offset */
    static const uint64_t want[4][5] = {
        {0, 0, 200, 0, 28}, {1, 0, 256, 56, 36}, {1, 1, 328, 128, 16}, {1, 2, 360, 160, 16}};
    for (int i = 0; i < 4; ++i) {
        CHECK(20 + i, p[i].chunk == want[i][0] && p[i].entry == want[i][1] &&
                          p[i].src_offset == want[i][2] && p[i].dst_index == 0 &&
                          p[i].dst_offset == want[i][3] && p[i].n_elems == want[i][4] &&
                          p[i].conv == 0 && p[i].rows == 1);
    }
    cfa_stats s;
    CHECK(30, cfa_get_stats(plan, &s) == CFA_OK);
    CHECK(31, s.bytes_read == 192 && s.bytes_written == 192 && s.n_entries == 3);
    cfa_source src;
    memset(&src, 0, sizeof src);
    src.kind = CFA_SRC_DEVICE;
    src.base = (const void *)(uintptr_t)0x200000;
    CHECK(32, cfa_load_async(plan, &src, NULL) == CFA_ERR_INVAL); /* host-only: no loads */
    CHECK(33, cfa_plan_destroy(plan) == CFA_OK);
    CHECK(34, cfa_plan_destroy(NULL) == CFA_OK);

    /* k written over the last row of q: refused, with a message */
    e[1] = entry("k", 2, 328, 7);
    plan = NULL;
    CHECK(40, cfa_plan_create(e, 3, &d, 1, 392, &o, &plan) == CFA_ERR_OVERLAP && !plan);
    CHECK(41, strstr(cfa_last_error(NULL), "overlap") != NULL);
    CHECK(42, strcmp(cfa_status_name(CFA_ERR_OVERLAP), "CFA_ERR_OVERLAP") == 0);

    /* segmented loading: 2 ranks, one 512-byte chunk holding the 392-byte blob; rank 0's
     * segment is bytes 0 .. 255, rank 1's 256 .. 391 (136 bytes), and a segmented host-only plan
     * stages exactly its segment; chunks must be multiples of 256 x ranks, and a segmented plan
     * without a gather step is refused */
    uint64_t so = 0, sn = 0;
    CHECK(50, cfa_segment_range(392, 512, 2, 1, 0, &so, &sn) == CFA_OK && so == 256 && sn == 136);
    CHECK(51, cfa_segment_range(392, 512, 2, 0, 0, &so, &sn) == CFA_OK && so == 0 && sn == 256);
    CHECK(52, cfa_segment_range(392, 256, 2, 0, 0, &so, &sn) == CFA_ERR_INVAL);
    CHECK(57, cfa_segment_range(392, 512, 2, 0, 1, &so, &sn) == CFA_ERR_INVAL);
    e[1] = entry("k", 2, 328, 8);
    o.chunk_bytes = 512;
    o.seg_world = 2;
    o.seg_rank = 1;
    plan = NULL;
    CHECK(53, cfa_plan_create(e, 3, &d, 1, 392, &o, &plan) == CFA_ERR_INVAL && !plan);
    o.gather = gather_never_called;
    CHECK(54, cfa_plan_create(e, 3, &d, 1, 392, &o, &plan) == CFA_OK && plan);
    cfa_stats sst;
    CHECK(55, cfa_get_stats(plan, &sst) == CFA_OK && sst.staged_bytes == 136);
    CHECK(56, cfa_plan_destroy(plan) == CFA_OK);
    o.seg_world = 1;
    o.seg_rank = 0;
    o.gather = NULL;
    o.chunk_bytes = 256;

    /* a safetensors header in memory */
    static const char hdr[] = "{\"__metadata__\":{\"format\":\"pt\"},"
                              "\"w\":{\"dtype\":\"BF16\",\"shape\":[2,3],\"data_offsets\":[0,12]}}";
    const uint64_t n_hdr = sizeof hdr - 1;
    cfa_safetensors *st = NULL;
    CHECK(50, cfa_safetensors_parse(hdr, n_hdr, 8 + n_hdr + 12, &st) == CFA_OK);
    size_t n_t = 0;
    uint64_t data_offset = 0, data_bytes = 0;
    CHECK(51, cfa_safetensors_info(st, &n_t, &data_offset, &data_bytes) == CFA_OK);
    CHECK(52, n_t == 1 && data_offset == 8 + n_hdr && data_bytes == 12);
    cfa_st_tensor t;
    CHECK(53, cfa_safetensors_tensor(st, 0, &t) == CFA_OK);
    CHECK(54, !strcmp(t.name, "w") && t.dtype == CFA_DTYPE_BF16 && t.ndim == 2 &&
                  t.shape[0] == 2 && t.shape[1] == 3 && t.blob_offset == 0 && t.nbytes == 12);
    cfa_st_tensor all[2];
    CHECK(57, cfa_safetensors_tensors(st, 0, 1, all) == CFA_OK &&
                  !memcmp(&all[0], &t, sizeof t));
    CHECK(58, cfa_safetensors_tensors(st, 0, 2, all) == CFA_ERR_INVAL &&
                  cfa_safetensors_tensors(st, 2, 0, all) == CFA_ERR_INVAL &&
                  cfa_safetensors_tensors(st, 1, 0, NULL) == CFA_OK);
    uint64_t name_bytes = 0;
    char names[4] = {'x', 'x', 'x', 'x'};
    CHECK(59, cfa_safetensors_names(st, NULL, 0, &name_bytes) == CFA_OK && name_bytes == 2);
    CHECK(60, cfa_safetensors_names(st, names, 1, &name_bytes) == CFA_ERR_INVAL &&
                  names[0] == 'x');
    CHECK(61, cfa_safetensors_names(st, names, 4, &name_bytes) == CFA_OK &&
                  !memcmp(names, "w\0xx", 4));
    CHECK(55, cfa_safetensors_close(st) == CFA_OK);
    CHECK(56, cfa_safetensors_parse(hdr, n_hdr, 8 + n_hdr + 11, &st) == CFA_ERR_INVAL);
    printf("ok\n");
    return 0;
}
