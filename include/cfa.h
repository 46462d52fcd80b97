/*
 * cfa.h -- C ABI of the chunked tensor-materialization loader.
 *
 * The loader brings a model checkpoint ("the blob": one contiguous byte stream holding every
 * tensor of the model) from host memory into a serving engine's final per-parameter layout on
 * one GPU.  It follows the refined tensor-materialization automaton of InstantInfer
 * (arXiv 2607.18957, section 4.2 "Tensor Materialization", refined CFA model):
 *
 *   - the blob is cut into equal-length chunks, the last one possibly partial;
 *   - the tensor <-> chunk association (tensor.chunks / chunk.tensors) is precomputed once,
 *     here by cfa_plan_create;
 *   - each chunk moves InDisk -> InMem -> InGPU -> Destroyed through a two-stage pipeline
 *     (section 4.2, dependency (i)): host staging into a pinned slot, then a host->device copy
 *     into a device staging slot;
 *   - once a chunk is InGPU, one batched launch group copies and assembles every tensor piece
 *     that lies in it into its destination (dependency (ii)), which moves those tensors from
 *     Alloc to Loaded: a TMA bulk-copy kernel for 16-byte-aligned runs, 16-byte vector kernels
 *     for the rest (realigning unaligned runs in registers), and a kernel for column slices;
 *   - the chunk's staging slot is released once all its pieces are written (dependency (iii)).
 *
 * Beyond what the paper states, the kernels also fuse the serving engine's layout transforms
 * (several checkpoint tensors written at row offsets of one fused destination, e.g. q/k/v into
 * one qkv weight; tensor- and expert-parallel shards), optional dtype conversions (fp32 -> bf16
 * and fp32 -> fp16 with round-to-nearest-even, fp16 -> bf16, bf16 / fp16 -> fp32), and an
 * optional per-tensor 64-bit additive checksum of the destination element bits.
 *
 * Conventions for every function below:
 *   - The return value is a cfa_status: CFA_OK (0) on success, a negative CFA_ERR_* code
 *     otherwise.  No function aborts, throws, traps the GPU or spins without a bound.
 *   - cfa_last_error(plan) gives a human-readable detail of the last failure on that plan;
 *     cfa_last_error(NULL) gives the detail of the last failure of cfa_plan_create or of the
 *     checkpoint-file functions on the calling thread.
 *   - "device pointer" means an address in the global memory of the plan's CUDA device;
 *     "host pointer" means ordinary process memory.
 *   - Streams are CUDA runtime streams (cudaStream_t); NULL is the legacy default stream.
 *   - All integers are little-endian, as on both the host and the GPU.
 */
#ifndef CFA_H
#define CFA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t, declared here so that this header needs no CUDA header. */
typedef struct CUstream_st *cfa_stream;

typedef int cfa_status;

#define CFA_OK            0
#define CFA_ERR_INVAL    (-1)  /* bad argument, bad option, or malformed manifest entry */
#define CFA_ERR_OVERLAP  (-2)  /* two pieces (or two destinations) write the same bytes */
#define CFA_ERR_OOB      (-3)  /* an entry reads past the blob or writes past its destination */
#define CFA_ERR_COVERAGE (-4)  /* strict mode: some destination byte is written by no entry */
#define CFA_ERR_CUDA     (-5)  /* a CUDA runtime call failed; detail in cfa_last_error */
#define CFA_ERR_SOURCE   (-6)  /* the source callback reported an error */
#define CFA_ERR_TIMEOUT  (-7)  /* a host wait reached its deadline; nothing was cancelled */
#define CFA_ERR_BUSY     (-8)  /* the plan is in use by another thread */
#define CFA_ERR_NOMEM    (-9)  /* a host or device allocation failed */
#define CFA_ERR_DTYPE    (-10) /* source and destination dtypes do not match the entry's cast */
#define CFA_ERR_ALIGN    (-11) /* an offset, pointer or size breaks an alignment rule */
#define CFA_ERR_DEVICE   (-12) /* the unpack kernel's own descriptor check failed */
#define CFA_ERR_SHAPE    (-13) /* an entry's last dimension differs from its destination's row */
#define CFA_ERR_SUSPECT  (-14) /* a TMA kernel's wait ran out and so did the wait for its own
                                  loads in flight: a bulk load may have outlived its CTA, so the
                                  CUDA context (and the destinations) must be treated as suspect;
                                  destroy the plan and reset the context before further work */
#define CFA_ERR_GATHER   (-15) /* the gather callback of a segmented load reported an error */

/* Element types.  Only the element size matters for plain copies; 1-byte types cover int8,
 * uint8 and the fp8 formats. */
#define CFA_DTYPE_U8    1
#define CFA_DTYPE_BF16  2
#define CFA_DTYPE_F16   3
#define CFA_DTYPE_F32   4
#define CFA_DTYPE_I32   5
#define CFA_DTYPE_I64   6
#define CFA_DTYPE_F64   7
#define CFA_DTYPE_I16   8

#define CFA_MAX_DIMS    8
#define CFA_MAX_LAYERS  65536

/* cfa_tensor_entry.flags */
#define CFA_ENTRY_CAST_BF16 0x1u /* source fp32, destination bf16, round to nearest even */
#define CFA_ENTRY_CKSUM     0x2u /* accumulate this entry's checksum (see cfa_get_checksums) */
#define CFA_ENTRY_CONVERT   0x4u /* convert to the destination dtype; supported pairs:
                                    f32 -> bf16, f32 -> f16, f16 -> bf16 (round to nearest,
                                    ties to even; NaN -> 0x7FC0 for bf16, sign | 0x7E00 for
                                    f16; overflow -> infinity), bf16 -> f32 and f16 -> f32
                                    (exact, NaN payloads kept) */

/* Passed as `layer` to cfa_wait_layer / cfa_get_layer_times: the whole load. */
#define CFA_ALL (-1)

/*
 * One checkpoint tensor (one tensor component of section 4.2).
 *
 *   name            optional, copied by cfa_plan_create; used only in error messages.
 *   src_dtype       CFA_DTYPE_* of the elements in the blob.
 *   ndim, shape     logical shape, row-major; ndim 0 is a scalar.  Zero-element tensors are
 *                   valid and load nothing.
 *   blob_offset     byte offset of element 0 in the blob; a multiple of the source element size.
 *   dst_index       index into the cfa_dst array.
 *   layer           readiness group, 0 <= layer < CFA_MAX_LAYERS (cfa_wait_layer).
 *   dst_row_offset  where the tensor starts inside its destination, in destination rows.
 *                   For a destination of ndim >= 2, a row is its last dimension R = shape[-1]:
 *                   the entry's last dimension must equal R and the entry fills
 *                   numel / R consecutive rows starting at dst_row_offset.  For a destination
 *                   of ndim <= 1 a row is one element.  This is how fused layouts are written:
 *                   q, k, v at rows 0, Hq, Hq + Hkv of qkv; gate, up at rows 0, I of gate_up;
 *                   expert e's w1, w3 at rows 2Ie, 2Ie + I of the [E*2I, H] view of w13.
 *   flags           CFA_ENTRY_*.  Without CFA_ENTRY_CAST_BF16 or CFA_ENTRY_CONVERT the
 *                   destination dtype must equal src_dtype; with CFA_ENTRY_CAST_BF16, src_dtype
 *                   must be F32 and the destination BF16; with CFA_ENTRY_CONVERT the pair must
 *                   be one CFA_ENTRY_CONVERT lists.
 *   src_row_stride  0 when the tensor's elements are contiguous in the blob.  Otherwise the
 *                   tensor is read as numel / shape[-1] rows of shape[-1] elements whose first
 *                   elements lie src_row_stride source elements apart (>= shape[-1]): a column
 *                   slice of a larger row-major checkpoint tensor.  This is how a
 *                   tensor-parallel rank reads its shard of a row-parallel weight (columns
 *                   [r K / R, (r + 1) K / R) of o_proj, down_proj, w2); column-parallel shards
 *                   (row ranges) are contiguous and need no stride.
 */
typedef struct cfa_tensor_entry {
    const char *name;
    int32_t src_dtype;
    int32_t ndim;
    int64_t shape[CFA_MAX_DIMS];
    uint64_t blob_offset;
    int32_t dst_index;
    int32_t layer;
    int64_t dst_row_offset;
    uint32_t flags;
    uint32_t src_row_stride;
} cfa_tensor_entry;

/*
 * One destination parameter of the serving engine (a Loaded tensor of section 4.2).
 * dev_ptr is a device pointer owned by the caller, aligned to its element size (16-byte
 * alignment of destination and source lets whole slabs take the TMA kernel), and it must stay
 * valid for every load that uses the plan.  Destinations must not overlap one another in memory.
 */
typedef struct cfa_dst {
    void *dev_ptr;
    int32_t dtype;
    int32_t ndim;
    int64_t shape[CFA_MAX_DIMS];
} cfa_dst;

/* cfa_plan_opts.flags */
#define CFA_OPT_STRICT_COVERAGE 0x1u  /* every destination byte must be written exactly once */
#define CFA_OPT_HOST_ONLY       0x2u  /* build and validate on the host only: no CUDA call is made,
                                         cfa_plan_get_pieces works, loads return CFA_ERR_INVAL */
#define CFA_OPT_TIMING          0x4u  /* record per-chunk timing events (cfa_get_stats, timeline);
                                         a staged chunk's transfer then begins after the previous
                                         chunk's has ended on both transfer paths */
#define CFA_OPT_BULK            0x8u  /* copy cast-free slabs whose source, destination and
                                         length are multiples of 16 bytes with the TMA bulk-copy
                                         kernel; without it every slab takes the 16-byte vector
                                         kernel.  Set by cfa_plan_opts_default: the bulk kernel
                                         is 1-4 % faster on GB300 */
#define CFA_OPT_NO_MERGE        0x10u /* DEVICE sources: one launch per chunk instead of one
                                         launch per contiguous run of chunks */
#define CFA_OPT_STAGE_SLICES    0x20u /* PINNED sources: copy column slices through the device
                                         slots as strided 2-D copies; without it (the default)
                                         the column-slice kernel reads them in place from the
                                         pinned memory over the host link, beside the copy ring */

/*
 * Gather step of a segmented (multi-path) load: section 4.2, "Optimization of Distributed
 * Loading".  With W ranks cooperating, every chunk is cut into W equal segments of
 * segment_bytes = chunk_bytes / W; this rank has copied its own segment into
 * chunk_dev + rank * segment_bytes, and the callback must enqueue on `stream` the collective
 * that fills the whole device slot chunk_dev[0, W * segment_bytes) with every rank's segment
 * (an AllGather with send buffer chunk_dev + rank * segment_bytes and receive buffer chunk_dev,
 * in place).  Once that work completes on `stream` the chunk is Gathered and its unpack runs.
 * Bytes of segments past the end of the blob are never read, whatever they hold.
 *
 * It is called on the thread that calls cfa_load_async, once per chunk, for chunks 0, 1, 2 ...
 * in order and for every chunk of the blob (so every rank issues the same sequence of
 * collectives); it must only enqueue work and return (not wait for the GPU), and it returns 0,
 * or non-zero on failure (the load then stops enqueueing and reports CFA_ERR_GATHER).  Every
 * rank's plan must have the same blob_bytes, chunk_bytes and seg_world.
 */
typedef int (*cfa_gather_fn)(void *user, void *chunk_dev, uint64_t segment_bytes, int32_t world,
                             int32_t rank, uint32_t chunk, cfa_stream stream);

typedef struct cfa_plan_opts {
    uint64_t chunk_bytes;     /* chunk length S, a multiple of 256; default 512 MiB */
    int32_t host_slots;       /* pinned host staging slots of S bytes, allocated by the first HOST
                                 or CALLBACK load (0 = none); default 2 */
    int32_t dev_slots;        /* device staging slots of S bytes, allocated by cfa_plan_create
                                 (0 = none: DEVICE sources only); default 3, so that a chunk's
                                 unpack has two transfers' time before its slot is needed */
    int32_t fill_threads;     /* host threads copying pageable sources into pinned slots; default:
                                 the CPUs the process may run on, at most 32 */
    int32_t device;           /* CUDA device ordinal; -1 = the current device */
    uint32_t slab_bytes;      /* destination bytes per block-level work item, a multiple of 4096
                                 in [4096, 64 MiB], or 0 (the default): chosen by the plan for
                                 about 4096 items per load, a power of two in [32 KiB, 256 KiB]
                                 (256 KiB from 1 GiB of destinations up) */
    uint32_t tiny_bytes;      /* pieces with fewer destination bytes become warp-level items of
                                 at most 512 destination bytes, each copied by four or eight
                                 lanes of a warp; default 8192 */
    uint32_t flags;           /* CFA_OPT_*; default CFA_OPT_STRICT_COVERAGE | CFA_OPT_BULK */
    uint32_t pull_percent;    /* staged loads: the share, in percent (0-100), of each chunk's
                                 contiguous byte ranges that the plan's pull kernel copies into
                                 the device slot with SM loads over the host link, beside the
                                 copy engine's copies of the rest (0 = copy engine only).  On
                                 GB300 the SMs read page-locked memory at the link rate even
                                 from buffers the copy engine reads at half of it; the price is
                                 one CTA per SM for the length of the transfer.  Default 100
                                 (all of it pulled); no effect on segmented plans and strided
                                 2-D copies */
    void *workspace;          /* optional device memory for the staging slots (NULL = plan allocates) */
    uint64_t workspace_bytes; /* must be >= dev_slots * chunk_bytes when workspace is given */
    /* Segmented (multi-path) loading, section 4.2 "Optimization of Distributed Loading":
     * seg_world > 1 ranks load every chunk together, each copying only its segment (one
     * seg_world-th of the chunk) from its own source into its own device slot, and `gather`
     * (above) assembles the chunk in every rank's slot before the unpack.  chunk_bytes must be
     * a multiple of 256 * seg_world; the device slots are then chunk_bytes long even for a blob
     * shorter than one chunk.  Loads of such a plan take HOST, PINNED and CALLBACK sources,
     * never skip a chunk, and stage the rank's whole segments (cfa_stats.staged_bytes), not
     * only the byte ranges its own pieces read: the other ranks may need any of them.
     * Default seg_world = 1 (0 and 1 are off), seg_rank = 0, gather = NULL. */
    int32_t seg_world;
    int32_t seg_rank;         /* this rank, 0 <= seg_rank < seg_world */
    cfa_gather_fn gather;     /* required when seg_world > 1 */
    void *gather_user;        /* passed to gather */
} cfa_plan_opts;

/* Fills *opts with the defaults listed above. */
void cfa_plan_opts_default(cfa_plan_opts *opts);

/* Source kinds (cfa_source.kind). */
#define CFA_SRC_HOST     1 /* pageable host memory; copied into pinned slots by host threads */
#define CFA_SRC_PINNED   2 /* page-locked host memory; copied straight to the device slots */
#define CFA_SRC_CALLBACK 3 /* fill(user, blob_offset, dst, len) writes the bytes into a pinned slot */
#define CFA_SRC_DEVICE   4 /* device memory already holding the blob; no staging, no copies */
#define CFA_SRC_HOST_DIRECT 5 /* host memory that the unpack kernel reads in place over the host
                                 link, one launch per chunk: no staging slots, no copy engine.
                                 Page-locked memory always qualifies; pageable memory needs a
                                 device that can access it (cudaDevAttrPageableMemoryAccess:
                                 Grace-Blackwell and Grace-Hopper over NVLink-C2C), otherwise
                                 the load is refused with CFA_ERR_INVAL before any GPU work.
                                 Host memory is read by the vector kernel only: the TMA bulk
                                 path is kept for device memory */

/* Writes blob bytes [blob_offset, blob_offset + len) to host memory dst and returns 0, or
 * returns non-zero on failure.  It is called from the plan's fill threads, several at once for
 * disjoint ranges, so it must be thread-safe; it must not call CUDA. */
typedef int (*cfa_fill_fn)(void *user, uint64_t blob_offset, void *dst, uint64_t len);

/*
 * Where the blob's bytes come from.  With period_bytes == 0, blob byte o is base[o].  With
 * period_bytes > 0 (a multiple of chunk_bytes), the blob is periodic and byte o is
 * base[o % period_bytes]; this streams a blob larger than memory from a smaller pool.  base must
 * be 256-byte aligned for PINNED and DEVICE sources and 8-byte aligned for HOST_DIRECT ones (the
 * vector kernels that read host memory take any 16-byte phase; 8 keeps every element aligned).
 * size_bytes, when not 0, is how many bytes can be read at base: a load whose plan would read
 * past them (blob_bytes, or period_bytes for a periodic source) is refused with CFA_ERR_INVAL
 * before any GPU work.  The source must stay valid until the load has completed
 * (cfa_wait_layer(CFA_ALL) returned).
 */
typedef struct cfa_source {
    int32_t kind;
    int32_t reserved;
    const void *base;
    uint64_t period_bytes;
    cfa_fill_fn fill;
    void *user;
    uint64_t size_bytes; /* 0: not stated */
} cfa_source;

typedef struct cfa_plan cfa_plan;

typedef struct cfa_stats {
    uint64_t blob_bytes;
    uint64_t n_entries, n_dsts, n_chunks, n_layers;
    uint64_t n_pieces;        /* tensor x chunk intersections */
    uint64_t n_slabs;         /* block-level work items (vector path) */
    uint64_t n_bulk;          /* block-level work items (TMA bulk path) */
    uint64_t n_tiny;          /* warp-level work items */
    uint64_t n_strided;       /* block-level work items over rows of column slices */
    uint64_t bytes_read;      /* algorithmic bytes one load reads from staging */
    uint64_t bytes_written;   /* algorithmic bytes one load writes into destinations */
    uint64_t descriptor_bytes;
    uint64_t staged_bytes;    /* blob bytes one staged load copies to the device: the byte
                                 ranges the chunks' pieces read, not whole chunks */
    uint64_t loads;           /* loads enqueued on this plan */
    uint64_t kernel_launches; /* unpack kernel launches enqueued by the last load */
    double plan_ms;           /* host time spent in cfa_plan_create */
    /* CFA_OPT_TIMING only, valid once the last load has completed: */
    double load_ms;           /* first enqueued operation to last unpack, device clock */
    double h2d_ms;            /* sum over chunks of the host->device copy time */
    double unpack_ms;         /* sum over launches of the unpack kernel time */
} cfa_stats;

/* A piece (tensor x chunk) as the plan builder cut it; for inspection and tests.  A piece is
 * `rows` runs of n_elems / rows elements each; run k starts at source byte
 * src_offset + k * src_row_stride * (source element size) and fills the destination
 * contiguously from dst_offset on.  Contiguous pieces have rows = 1. */
typedef struct cfa_piece {
    uint32_t chunk;
    uint32_t entry;
    uint64_t src_offset;      /* byte offset in the blob */
    uint32_t dst_index;
    uint32_t conv;            /* 0 = copy; 1 f32->bf16, 2 f32->f16, 3 f16->bf16, 4 bf16->f32,
                                 5 f16->f32 */
    uint64_t dst_offset;      /* byte offset inside the destination */
    uint64_t n_elems;
    uint32_t rows;
    uint32_t src_row_stride;  /* source elements between run starts (rows > 1) */
} cfa_piece;

/*
 * Validates the manifest, precomputes the chunk <-> tensor mapping (section 4.2) and cuts
 * every tensor into pieces, then, unless CFA_OPT_HOST_ONLY is set, uploads the descriptor table
 * to the device and allocates the staging slots, the streams and the events.
 *
 *   entries, n_entries  the checkpoint's tensors (host memory; copied, may be freed on return).
 *   dsts, n_dsts        the destinations (host array; copied; dev_ptr stays caller-owned).
 *   blob_bytes          length of the blob; every entry must lie inside it.
 *   opts                NULL for the defaults.
 *   out                 receives the plan; set to NULL on failure.
 *
 * Errors: CFA_ERR_INVAL, CFA_ERR_DTYPE, CFA_ERR_ALIGN, CFA_ERR_OOB, CFA_ERR_OVERLAP,
 * CFA_ERR_COVERAGE (strict mode), CFA_ERR_NOMEM, CFA_ERR_CUDA.  Nothing is left allocated.
 */
cfa_status cfa_plan_create(const cfa_tensor_entry *entries, size_t n_entries,
                           const cfa_dst *dsts, size_t n_dsts, uint64_t blob_bytes,
                           const cfa_plan_opts *opts, cfa_plan **out);

/*
 * Enqueues one complete load of the blob into the destinations and returns without waiting.
 * Every chunk goes through: host staging (HOST without pageable access, or with pull_percent
 * 0: copied by the plan's fill threads; CALLBACK: written by src->fill; PINNED, DEVICE and
 * HOST_DIRECT: none), a host->device transfer into a device slot (none for DEVICE and
 * HOST_DIRECT): the plan's pull kernel on a stream of the plan for pull_percent of each
 * contiguous range, the copy engine on the plan's copy stream for the rest and for strided 2-D
 * copies; and the unpack kernels on `stream` that write all pieces of the chunk (DEVICE sources
 * merge all chunks into one launch per work class; a staged chunk's unpack, beside the next
 * transfer, runs on a quarter of the grid, the last chunk's on all of it).  Staging and copies move only the byte ranges the chunk's pieces read (strided 2-D
 * copies for column slices), so a tensor-parallel rank moves about its share of the
 * checkpoint; cfa_stats.staged_bytes gives the total.  A chunk no piece reads (an
 * expert-parallel rank's view of other ranks' experts) is skipped altogether: no fill, no copy,
 * no launch, and it takes no staging slot.  The load is ordered after
 * all work enqueued on `stream` before this call, and work enqueued on `stream` after this
 * call sees every destination written.  Per-layer readiness is published through
 * cfa_wait_layer.  Loads on one plan run in the order they were enqueued; the checksums and
 * layer events always refer to the most recently enqueued load.
 *
 * With seg_world > 1 (segmented plans) each chunk's H2D copy moves only this rank's segment,
 * then opts.gather assembles the chunk in the device slot on a stream of the plan (the chunk's
 * Gathered state), and the unpack waits for that instead of the copy.
 *
 * Errors: CFA_ERR_INVAL (bad source, host-only plan, or a staging kind the plan has no slots
 * for; DEVICE and HOST_DIRECT sources on a segmented plan), CFA_ERR_ALIGN, CFA_ERR_CUDA,
 * CFA_ERR_GATHER (the gather callback failed: the chunks before it were enqueued, the rest of
 * the load was not; the load's events are still recorded, so waits end, and they report
 * CFA_ERR_GATHER).  Failures that happen later (the fill callback, a CUDA error) are latched
 * and returned by cfa_wait_layer / cfa_get_checksums for that load.
 */
cfa_status cfa_load_async(cfa_plan *plan, const cfa_source *src, cfa_stream stream);

/*
 * Waits until readiness group `layer` of the last load is Loaded (all its tensors written), or
 * the whole load with layer == CFA_ALL.
 *   consumer != NULL: makes that stream wait on the GPU (no host blocking) and returns.
 *   consumer == NULL: blocks the host, polling without spinning on the GPU, until the group is
 *                     ready or timeout_ns (< 0: no limit) has passed; then CFA_ERR_TIMEOUT.
 * Errors: CFA_ERR_INVAL (unknown layer, no load yet), CFA_ERR_TIMEOUT, CFA_ERR_SOURCE,
 * CFA_ERR_GATHER, CFA_ERR_CUDA, CFA_ERR_DEVICE (status word 1 or 2: a descriptor rejected by
 * the kernel, or a TMA wait that ran out and ended cleanly), CFA_ERR_SUSPECT (status word 3).
 */
cfa_status cfa_wait_layer(cfa_plan *plan, int32_t layer, cfa_stream consumer, int64_t timeout_ns);

/*
 * Copies the per-entry checksums of the last load to host_out[0 .. n) (n <= n_entries), in entry
 * order.  An entry's checksum is the sum, modulo 2^64, of its destination elements' bit patterns
 * read as unsigned integers of the destination element size (after the cast).  Entries without
 * CFA_ENTRY_CKSUM read 0.  Blocks until the load has completed.
 */
cfa_status cfa_get_checksums(cfa_plan *plan, uint64_t *host_out, size_t n);

/* Fills *out.  Blocks until the last load has completed if CFA_OPT_TIMING is set. */
cfa_status cfa_get_stats(cfa_plan *plan, cfa_stats *out);

/*
 * Milliseconds from the first operation of the last load to the moment each readiness group was
 * Loaded, for groups 0 .. n-1 (CFA_OPT_TIMING plans; blocks until the load completes).
 */
cfa_status cfa_get_layer_times(cfa_plan *plan, float *ms_out, size_t n);

/* One chunk of the last load on the timeline, in milliseconds from its first operation; -1 where
 * the step did not run (no host->device copy for in-place sources, nothing for a chunk no piece
 * reads).  A merged launch over several
 * chunks gives each of them the launch's interval. */
typedef struct cfa_chunk_times {
    float h2d_begin_ms, h2d_end_ms;       /* the chunk's copies into its device slot */
    float unpack_begin_ms, unpack_end_ms; /* first start and last end of the kernels reading it */
} cfa_chunk_times;

/* Per-chunk timeline of the last load, chunks 0 .. n-1 (n <= n_chunks; CFA_OPT_TIMING plans;
 * blocks until the load completes).  Errors: CFA_ERR_INVAL (no timing, no load, n too large). */
cfa_status cfa_get_timeline(cfa_plan *plan, cfa_chunk_times *out, size_t n);

/*
 * Number of readiness groups and pieces of the plan; then the pieces themselves, in chunk order
 * (at most cap of them into out).  Host-only; works on CFA_OPT_HOST_ONLY plans.
 */
cfa_status cfa_plan_info(const cfa_plan *plan, uint64_t *n_layers, uint64_t *n_pieces,
                         uint64_t *n_chunks);
cfa_status cfa_plan_get_pieces(const cfa_plan *plan, cfa_piece *out, size_t cap, size_t *n_out);

/*
 * Unpacks chunks [chunk_begin, chunk_end) that the caller has already placed in device memory:
 * blob byte o of those chunks is at chunk_src + (o - chunk_begin * chunk_bytes).  chunk_src is a
 * device pointer, 256-byte aligned.  One kernel launch on `stream`; checksums accumulate into
 * the plan's checksum buffer (cleared by cfa_load_async, or by cfa_reset_checksums).  This is the
 * bare "InGPU -> Loaded" transition of section 4.2 for callers that manage their own staging.
 */
cfa_status cfa_unpack_chunks_async(cfa_plan *plan, uint32_t chunk_begin, uint32_t chunk_end,
                                   const void *chunk_src, cfa_stream stream);

/*
 * Unpacks a blob that already sits in device memory into its destinations WITHOUT ALLOCATING
 * ANYTHING -- no cudaMalloc, no cudaFree, no host heap.  The paper has no counterpart: it is for
 * callers that cannot allocate, such as a serving engine whose memory pool already owns the
 * device, a latency-critical path that cannot afford cudaFree's implicit device-wide
 * synchronisation, or a restricted runtime with no allocator.  It is cfa_plan_create +
 * cfa_load_async(DEVICE source) + cfa_get_checksums' buffer in one call, with these
 * differences:
 *   - no plan: every entry is validated on its own (dtype, shape, bounds, alignment), but the
 *     coverage and overlap checks of cfa_plan_create are not made; destinations must not
 *     overlap one another and entries must not write the same bytes;
 *   - the work descriptors live in a fixed device array inside this library of
 *     CFA_NOALLOC_MAX_ITEMS entries (16384 x 32 bytes = 512 KiB, plus a status word), held by
 *     every GPU that loads the library until the process exits.  A tensor needs one work item
 *     per 2 MiB of destination bytes, and below 8 KiB one per 512-byte-aligned block of
 *     destination addresses it touches; a manifest that needs more is rejected with
 *     CFA_ERR_INVAL before any GPU work, and `err` says so;
 *   - all calls on a device share that array: calls serialise on the host, but calls whose GPU
 *     work may overlap (different streams, no ordering between them) race on it;
 *   - the first call on a device does a one-time set-up (it looks up the array's device address
 *     and the kernels' occupancy); make it before any stream capture.  That address belongs to
 *     the device's context: do not call this again in a process after cudaDeviceReset;
 *   - the call blocks the host: the descriptors go up as a copy from pageable host memory,
 *     which CUDA completes before returning, and which first waits for the work already
 *     queued on `stream`.  The unpack kernels are enqueued behind it and run after the call
 *     returns.
 *
 *   entries, n_entries, dsts, n_dsts   as for cfa_plan_create (host arrays, read during the call)
 *   blob_dev, blob_bytes   the blob in device memory (256-byte aligned); must stay valid and
 *                          unchanged until the unpack has run on `stream`
 *   cksum_dev              device array of n_entries uint64 receiving the checksums
 *                          (cleared by the call), or NULL for none
 *   status_dev             optional device int (4-byte aligned) receiving the kernels' own
 *                          status word: the call sets it to 0 on `stream`, and a kernel that
 *                          rejects a work item (its source outside the blob, a misaligned
 *                          address, a wrong work class) sets it to 1 and leaves that item's
 *                          bytes unwritten.  The host validation above makes this unreachable
 *                          for any accepted manifest; read it once `stream` has run the unpack
 *                          to confirm.  NULL: the status goes to the scratch array's own word
 *   stream                 all GPU work is enqueued here
 *   err, err_len           optional buffer for a message on failure (NULL for none)
 * Errors: CFA_ERR_INVAL (NULL argument, bad entry, too many work items), CFA_ERR_DTYPE,
 * CFA_ERR_SHAPE, CFA_ERR_OOB, CFA_ERR_ALIGN, CFA_ERR_CUDA.
 */
#define CFA_NOALLOC_MAX_ITEMS 16384
cfa_status cfa_unpack_noalloc(const cfa_tensor_entry *entries, size_t n_entries,
                              const cfa_dst *dsts, size_t n_dsts, const void *blob_dev,
                              uint64_t blob_bytes, uint64_t *cksum_dev, int *status_dev,
                              cfa_stream stream, char *err, size_t err_len);

/* ---- checkpoint files (the InDisk end of section 4.2's chunk automaton) ------------------- */

/*
 * A parsed safetensors header.  The file is an 8-byte little-endian length N, N bytes of JSON
 * mapping each tensor name to {"dtype", "shape", "data_offsets": [begin, end]} (plus an
 * optional "__metadata__" object), then the data section, which is the loader's blob:
 * data_offsets are blob offsets.  The paper loads checkpoints of this format (section 5).
 */
typedef struct cfa_safetensors cfa_safetensors;

typedef struct cfa_st_tensor {
    const char *name;      /* owned by the cfa_safetensors handle */
    int32_t dtype;         /* CFA_DTYPE_* (int8, uint8, bool and fp8 read as U8, uint16 as I16,
                              uint32 as I32, uint64 as I64) */
    int32_t ndim;
    int64_t shape[CFA_MAX_DIMS];
    uint64_t blob_offset;  /* byte offset of the tensor in the data section */
    uint64_t nbytes;
} cfa_st_tensor;

/* Reads and validates the header of `path` (not the data).  Every tensor's data_offsets must
 * match its shape and dtype and lie inside the file.  Errors: CFA_ERR_INVAL (malformed header,
 * unknown dtype, more than 8 dimensions), CFA_ERR_SOURCE (cannot read), CFA_ERR_NOMEM. */
cfa_status cfa_safetensors_open(const char *path, cfa_safetensors **out);

/* The same from a header already in memory (the N JSON bytes); file_bytes is the file's size. */
cfa_status cfa_safetensors_parse(const void *header, uint64_t header_len, uint64_t file_bytes,
                                 cfa_safetensors **out);

/* Tensor count, file offset of the data section (8 + N) and its length. */
cfa_status cfa_safetensors_info(const cfa_safetensors *st, size_t *n_tensors,
                                uint64_t *data_offset, uint64_t *data_bytes);

/* Tensor i (header order), 0 <= i < n_tensors. */
cfa_status cfa_safetensors_tensor(const cfa_safetensors *st, size_t i, cfa_st_tensor *out);

/* Tensors first .. first + count - 1 (header order) into out[0 .. count - 1], in one call (a
 * header of 10^5 tensors is read in milliseconds instead of one call per tensor).  The names
 * stay owned by the handle.  CFA_ERR_INVAL if the range is not inside [0, n_tensors). */
cfa_status cfa_safetensors_tensors(const cfa_safetensors *st, size_t first, size_t count,
                                   cfa_st_tensor *out);

/* Every tensor name in header order, each followed by a NUL byte, into buf (cap bytes); *bytes
 * receives the length this takes.  buf = NULL only reports the length.  Names hold no NUL byte
 * (the parser refuses \u0000).  CFA_ERR_INVAL if cap is smaller than the length. */
cfa_status cfa_safetensors_names(const cfa_safetensors *st, char *buf, uint64_t cap,
                                 uint64_t *bytes);

/* Frees the handle (and the names it owns).  Accepts NULL. */
cfa_status cfa_safetensors_close(cfa_safetensors *st);

/* cfa_file_source_open flags. */
#define CFA_FILE_DIRECT 0x1u /* O_DIRECT reads that bypass the page cache (storage bandwidth) */
#define CFA_FILE_MMAP   0x2u /* map the file read-only and fill with memcpy from the mapping:
                                 no system call per range (page-cache-resident files: 1.2x on
                                 large ranges, 2-5x on the rows of column slices, on Grace).
                                 The file must not shrink while mapped: reading a page past its
                                 end raises SIGBUS instead of CFA_ERR_SOURCE.  Not combinable
                                 with CFA_FILE_DIRECT. */
#define CFA_FILE_MMAP_IN_PLACE 0x4u /* map the file read-only, populated, and give a HOST_DIRECT
                                 source over the mapping: the unpack kernels read the file's
                                 page-cache pages in place over the host link, with no fill
                                 threads, pinned slots or copies (devices with pageable memory
                                 access, such as Grace-based GB300: 2x the pread and copy modes
                                 for a page-cache-resident file).  base = mapping + data_offset,
                                 so data_offset must be a multiple of 8 (a safetensors data
                                 section is); size_bytes = file size - data_offset.  The file
                                 must not shrink or be rewritten while mapped: on the GPU a page
                                 that cannot be read is a device memory fault that ends the CUDA
                                 context, not an error code.  Not combinable with the other
                                 flags. */

/*
 * Fills *out with a CALLBACK source that reads blob byte o from file byte data_offset + o with
 * pread (several fill threads may read at once).  With CFA_FILE_DIRECT the file is opened with
 * O_DIRECT: reads move whole 4 KiB blocks; where a destination range and its file range start
 * at the same offset within a block (data_offset a multiple of 4 KiB and a chunk length that is
 * too) the middle blocks land in the pinned slot directly, the rest passes through 4 MiB
 * bounce buffers owned by the source.  With CFA_FILE_MMAP_IN_PLACE *out is a HOST_DIRECT
 * source instead (its fill pointer is set only to mark it as a file source for
 * cfa_file_source_close; HOST_DIRECT loads never call it).  The file stays open until
 * cfa_file_source_close(out), which must come after every load using it has completed.
 * Errors: CFA_ERR_SOURCE (cannot open or map; for CFA_FILE_DIRECT also a file system without
 * O_DIRECT; data_offset past the end of the file), CFA_ERR_ALIGN (CFA_FILE_MMAP_IN_PLACE with
 * data_offset not a multiple of 8), CFA_ERR_INVAL (unknown flag or combination), CFA_ERR_NOMEM.
 */
cfa_status cfa_file_source_open(const char *path, uint64_t data_offset, uint32_t flags,
                                cfa_source *out);
cfa_status cfa_file_source_close(cfa_source *src);

/*
 * Where rank `rank` of `world` finds its segment of chunk `chunk` in a segmented load (see
 * cfa_plan_opts.seg_world): *blob_offset receives chunk * chunk_bytes + rank * segment_bytes
 * and *bytes the part of [*blob_offset, *blob_offset + segment_bytes) inside the blob (0 for a
 * segment wholly past its end), with segment_bytes = chunk_bytes / world.  Host-only, no CUDA
 * call.  Errors: CFA_ERR_INVAL (NULL output, world < 1, rank outside [0, world), chunk_bytes not
 * a positive multiple of 256 * world, chunk past the end of the blob).
 */
cfa_status cfa_segment_range(uint64_t blob_bytes, uint64_t chunk_bytes, int32_t world,
                             int32_t rank, uint32_t chunk, uint64_t *blob_offset,
                             uint64_t *bytes);

/* Zeroes the plan's checksum buffer on `stream`. */
cfa_status cfa_reset_checksums(cfa_plan *plan, cfa_stream stream);

/*
 * Waits for all work of the plan to finish, then frees everything the plan owns (descriptor
 * table, staging slots, pinned slots, streams, events, checksum buffer, threads).  The
 * destinations stay allocated.  Accepts NULL.
 */
cfa_status cfa_plan_destroy(cfa_plan *plan);

/*
 * Self-test of the loader's only device-side waits, the TMA kernel's bounded mbarrier waits
 * (no counterpart in the paper): on `device` (-1 = current) one CTA of the TMA kernel is given a
 * valid 16-byte item, a short wait limit and a loader that issues nothing, so its first wait for
 * a staged sub-block runs out.  *status_word receives the status word the kernel left: 2 when
 * the expired wait ended the kernel cleanly.  The CUDA context stays usable.  Allocates and
 * frees a few hundred bytes of device memory; synchronizes the device.
 * Errors: CFA_ERR_INVAL (status_word NULL), CFA_ERR_CUDA.
 */
cfa_status cfa_selftest_wait_timeout(int device, int *status_word);

/* Detail of the last failure (see the conventions above).  Never NULL. */
const char *cfa_last_error(const cfa_plan *plan);

/* Name of a status code, e.g. "CFA_ERR_OVERLAP". */
const char *cfa_status_name(cfa_status st);

/* sizeof of the ABI struct with this name ("cfa_tensor_entry", "cfa_dst", "cfa_plan_opts",
 * "cfa_source", "cfa_stats", "cfa_piece", "cfa_st_tensor", "cfa_chunk_times"), or 0 for an
 * unknown name; lets a binding check its
 * own copies of the layouts.  Host-only. */
size_t cfa_abi_sizeof(const char *type_name);

#ifdef __cplusplus
}
#endif

#endif /* CFA_H */
