/*
 * Internal structures shared by the host plan builder (cfa_plan.c), the kernels
 * (cfa_unpack.cu) and the runtime (cfa_runtime.cu).  Not part of the C ABI.
 */
#ifndef CFA_INTERNAL_H
#define CFA_INTERNAL_H

#include <stddef.h>
#include <stdint.h>

#include "cfa.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * One unit of GPU work: a contiguous run of elements of one piece (tensor x chunk).
 * 32 bytes, read once per work item.
 *   src   blob byte offset of the first source element (the launch adds its source base)
 *   dst   device address of the first destination element
 *   n     element count
 *   ck    checksum slot (the entry index), or CFA_NO_CK
 *   mode  bits 0-1: log2 of the source element size; bits 2-3: log2 of the destination element
 *         size; bit 4: fp32 -> bf16 round-to-nearest-even cast
 */
typedef struct cfa_work {
    uint64_t src;
    uint64_t dst;
    uint32_t n;
    uint32_t ck;
    uint32_t mode;
    uint32_t pad;
} cfa_work;

/*
 * A block of rows of a strided piece (a column slice of a larger checkpoint tensor): row k
 * starts at source blob offset src + k * stride * (source element size) and lands at
 * dst + k * cols * (destination element size).  40 bytes.
 */
/* Warp-level work items hold at most this many destination bytes (the plan cuts tiny pieces at
 * destination addresses that are multiples of it): one 8-lane warp segment copies one item. */
#define CFA_TINY_SEG_BYTES 512u

typedef struct cfa_swork {
    uint64_t src;
    uint64_t dst;
    uint32_t rows;
    uint32_t cols;   /* elements per row */
    uint32_t stride; /* source elements between row starts */
    uint32_t ck;
    uint32_t mode;
    uint32_t cls;    /* work class, used while the plan is built */
} cfa_swork;

/*
 * A host->device copy of one chunk: `rows` runs of `width` bytes, `pitch` bytes apart, the first
 * at blob offset `src`; it lands at the same offset inside the chunk's device slot.
 */
typedef struct cfa_copy {
    uint64_t src;
    uint64_t width;
    uint64_t pitch;
    uint64_t rows;
} cfa_copy;

#define CFA_NO_CK 0xFFFFFFFFu

/* Element conversions (cfa_work.mode bits 4-7, cfa_piece.conv). */
#define CFA_CONV_NONE 0
#define CFA_CONV_F32_BF16 1
#define CFA_CONV_F32_F16 2
#define CFA_CONV_F16_BF16 3
#define CFA_CONV_BF16_F32 4
#define CFA_CONV_F16_F32 5
#define CFA_N_CONV 6

/* Work classes: one specialised kernel each.  0..3 = plain copy of 1, 2, 4, 8-byte elements;
 * 3 + conv = conversion `conv`. */
#define CFA_N_CLASSES 9
#define CFA_CLASS_OF_CONV(conv) (3 + (conv))
#define CFA_MODE(src_log2, dst_log2, conv) \
    ((uint32_t)(src_log2) | ((uint32_t)(dst_log2) << 2) | ((uint32_t)(conv) << 4))
#define CFA_MODE_CONV(mode) (((mode) >> 4) & 15u)

/* Conversion for a (source, destination) dtype pair, 0 if the pair has none. */
static inline int cfa_conversion(int32_t src, int32_t dst)
{
    if (src == CFA_DTYPE_F32 && dst == CFA_DTYPE_BF16) return CFA_CONV_F32_BF16;
    if (src == CFA_DTYPE_F32 && dst == CFA_DTYPE_F16) return CFA_CONV_F32_F16;
    if (src == CFA_DTYPE_F16 && dst == CFA_DTYPE_BF16) return CFA_CONV_F16_BF16;
    if (src == CFA_DTYPE_BF16 && dst == CFA_DTYPE_F32) return CFA_CONV_BF16_F32;
    if (src == CFA_DTYPE_F16 && dst == CFA_DTYPE_F32) return CFA_CONV_F16_F32;
    return CFA_CONV_NONE;
}

/* Host side of a plan: everything cfa_plan_create computes before touching the GPU. */
typedef struct cfa_host_plan {
    cfa_plan_opts opts;
    uint64_t blob_bytes;
    uint64_t chunk_bytes;
    uint32_t n_chunks;
    uint32_t n_layers;
    size_t n_entries, n_dsts;
    cfa_tensor_entry *entries; /* copies; names point into `names` */
    char **names;
    cfa_dst *dsts;
    cfa_piece *pieces; /* sorted by (chunk, src offset) */
    size_t n_pieces;
    /* work items ordered by (class, chunk): class k of chunk c owns
     * [first[k * (n_chunks + 1) + c], first[k * (n_chunks + 1) + c + 1]) of each array, so the
     * items of one class over a run of chunks are contiguous */
    cfa_work *slabs; /* block-level, LSU vector path */
    size_t n_slabs;
    uint32_t *slab_first;
    cfa_work *bulk;  /* block-level, TMA bulk path (cast-free, 16-byte aligned) */
    size_t n_bulk;
    uint32_t *bulk_first;
    cfa_work *tiny;  /* warp-level */
    size_t n_tiny;
    uint32_t *tiny_first;
    cfa_swork *strided; /* block-level, rows of column slices */
    size_t n_strided;
    uint32_t *strided_first;
    int64_t *layer_last_chunk; /* n_layers; -1 = the group has no bytes */
    cfa_copy *copies;          /* what each chunk's pieces read: chunk c owns
                                  [copy_first[c], copy_first[c + 1]) */
    size_t n_copies;
    uint32_t *copy_first;
    uint64_t staged_bytes;
    uint64_t bytes_read, bytes_written;
    int any_cksum;
} cfa_host_plan;

/* Sets the calling thread's detail string returned by cfa_last_error(NULL). */
void cfa_internal_set_error(const char *msg);

cfa_status cfa_host_plan_build(const cfa_tensor_entry *entries, size_t n_entries,
                               const cfa_dst *dsts, size_t n_dsts, uint64_t blob_bytes,
                               const cfa_plan_opts *opts, cfa_host_plan *out, char *err,
                               size_t errlen);
void cfa_host_plan_free(cfa_host_plan *hp);
int cfa_dtype_size(int32_t dtype);

#ifdef __cplusplus
}
#endif

#endif /* CFA_INTERNAL_H */
