/*
 * ORACLE -- plain, slow CPU restatement of what tensor materialization computes.
 *
 * Test infrastructure only: the test suite, the smoke check and the benchmark's CPU-baseline
 * leg use it; the loader library never does, and this file shares no code, header or table with
 * it.
 *
 * What it computes (InstantInfer, section 4.2, refined CFA model, and Theorem 2): the chunked,
 * pipelined loader must leave every tensor in exactly the state the naive loader leaves it in:
 * the naive loader takes the tensors one by one and writes each tensor's elements into its
 * destination.  This file is that naive loader, element by element, in the order the definition
 * states:
 *
 *   for each entry t:
 *     D      = destination t.dst
 *     es_s   = element size of t's source dtype;  es_d = element size of D's dtype
 *              (equal to the source dtype unless t converts: f32 -> bf16, f32 -> f16,
 *              f16 -> bf16, bf16 -> f32, f16 -> f32)
 *     n      = product of t.shape
 *     row    = D's last dimension R when D has >= 2 dimensions (t.shape[-1] must equal R),
 *              one element when D has <= 1 dimension
 *     base   = t.row_offset * (elements per row) * es_d     (bytes into D)
 *     C      = t.shape[-1];  stride = t.src_row_stride, or C when it is 0 (contiguous)
 *     for i in 0 .. n-1:
 *         src_i = (i / C) * stride + (i mod C)     (element i of row i / C of a column slice)
 *         x = little-endian es_s-byte integer at blob[t.blob_offset + src_i * es_s]
 *         y = converts ? convert(x) : x
 *         write y as es_d little-endian bytes at D[base + i * es_d]
 *         cover[D][each written byte] += 1
 *         if t checksums: ck[t] = (ck[t] + y) mod 2^64
 *
 * and, in strict mode, every byte of every destination must end with cover == 1.
 *
 * rne_bf16 (round to nearest, ties to even, on the bit pattern; IEEE 754-2008 roundTiesToEven
 * applied to dropping the low 16 bits of a binary32): NaN -> 0x7FC0; otherwise add 0x7FFF plus
 * the lowest kept bit, then drop the low 16 bits.  Inf stays Inf, values past the largest finite
 * bf16 round to Inf, subnormals round like any other value, signed zeros keep their sign.
 *
 * The other conversions follow the IEEE 754 binary16 definition (1 sign, 5 exponent bits with
 * bias 15, 10 fraction bits; subnormals m * 2^-24): f16 -> f32 is exact (the value as a double,
 * then as a float, which holds every binary16 value; NaN keeps its payload in the top fraction
 * bits); f32 -> f16 takes the exact value and rounds it to the nearest binary16 with ties to
 * even (nearbyint in the default rounding mode), overflowing to infinity from 65520 up, NaN ->
 * sign | 0x7E00; f16 -> bf16 is f16 -> f32 then rne_bf16; bf16 -> f32 appends 16 zero bits.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#include <string.h>

/* The oracle's own dtype codes (its Python wrapper maps dtype names onto these). */
enum { ORC_U8 = 1, ORC_BF16 = 2, ORC_F16 = 3, ORC_F32 = 4, ORC_I32 = 5, ORC_I64 = 6, ORC_F64 = 7,
       ORC_I16 = 8 };

/* Entry flags as the wrapper passes them. */
enum { ORC_CONVERT = 1, ORC_CKSUM = 2 };

/* Conversions, by (source, destination) dtype. */
enum { ORC_NONE = 0, ORC_F32_BF16, ORC_F32_F16, ORC_F16_BF16, ORC_BF16_F32, ORC_F16_F32 };

static int orc_conversion(int32_t s, int32_t d)
{
    if (s == ORC_F32 && d == ORC_BF16) return ORC_F32_BF16;
    if (s == ORC_F32 && d == ORC_F16) return ORC_F32_F16;
    if (s == ORC_F16 && d == ORC_BF16) return ORC_F16_BF16;
    if (s == ORC_BF16 && d == ORC_F32) return ORC_BF16_F32;
    if (s == ORC_F16 && d == ORC_F32) return ORC_F16_F32;
    return ORC_NONE;
}

/* Result codes. */
enum {
    ORC_OK = 0,
    ORC_E_INVAL = 1,    /* unknown dtype, bad dimension count, negative size or offset */
    ORC_E_DTYPE = 2,    /* source / destination dtypes do not fit the entry's cast flag */
    ORC_E_ALIGN = 3,    /* blob offset not a multiple of the source element size */
    ORC_E_OOB = 4,      /* reads outside the blob or writes outside the destination */
    ORC_E_SHAPE = 5,    /* last dimension differs from the destination row */
    ORC_E_OVERLAP = 6,  /* some destination byte written more than once */
    ORC_E_COVERAGE = 7, /* some destination byte never written */
};

static int orc_elem_size(int32_t dt)
{
    switch (dt) {
    case ORC_U8: return 1;
    case ORC_BF16: return 2;
    case ORC_F16: return 2;
    case ORC_I16: return 2;
    case ORC_F32: return 4;
    case ORC_I32: return 4;
    case ORC_I64: return 8;
    case ORC_F64: return 8;
    default: return 0;
    }
}

uint16_t oracle_rne_bf16(uint32_t u)
{
    const uint32_t exponent = u & 0x7F800000u;
    const uint32_t mantissa = u & 0x007FFFFFu;
    if (exponent == 0x7F800000u && mantissa != 0u) return 0x7FC0u; /* any NaN */
    const uint32_t lowest_kept_bit = (u >> 16) & 1u;
    return (uint16_t)((u + 0x7FFFu + lowest_kept_bit) >> 16);
}

void oracle_rne_bf16_array(const uint32_t *in, uint16_t *out, uint64_t n)
{
    for (uint64_t i = 0; i < n; ++i) out[i] = oracle_rne_bf16(in[i]);
}

uint32_t oracle_f16_to_f32(uint16_t h)
{
    const uint32_t s = h >> 15, e = (h >> 10) & 31u, m = h & 1023u;
    if (e == 31u) return (s << 31) | 0x7F800000u | (m << 13); /* infinity or NaN */
    const double v = e == 0 ? ldexp((double)m, -24) : ldexp(1024.0 + (double)m, (int)e - 25);
    const float f = (float)(s ? -v : v);
    uint32_t u;
    memcpy(&u, &f, 4);
    return u;
}

uint16_t oracle_f32_to_f16(uint32_t u)
{
    const uint16_t sign = (uint16_t)((u >> 16) & 0x8000u);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return sign | 0x7E00u;
    float f;
    memcpy(&f, &u, 4);
    const double v = fabs((double)f);
    if (isinf(v) || v >= 65520.0) return sign | 0x7C00u; /* 65504 + half an ulp (16) */
    if (v < ldexp(1.0, -14)) {                           /* subnormal: m * 2^-24 */
        const double m = nearbyint(ldexp(v, 24));         /* may round up to 1024 = 2^-14 */
        return sign | (uint16_t)m;
    }
    int e2;
    frexp(v, &e2);          /* v = fr * 2^e2, 0.5 <= fr < 1 */
    int E = e2 - 1;         /* 2^E <= v < 2^(E+1) */
    double m = nearbyint(ldexp(v, 10 - E)); /* 1024 <= m <= 2048 */
    if (m == 2048.0) {
        m = 1024.0;
        E += 1;
    }
    if (E > 15) return sign | 0x7C00u;
    return sign | (uint16_t)((E + 15) << 10) | (uint16_t)(m - 1024.0);
}

uint32_t oracle_bf16_to_f32(uint16_t b) { return (uint32_t)b << 16; }

uint16_t oracle_f16_to_bf16(uint16_t h) { return oracle_rne_bf16(oracle_f16_to_f32(h)); }

static uint64_t orc_convert(int conv, uint64_t x)
{
    switch (conv) {
    case ORC_F32_BF16: return oracle_rne_bf16((uint32_t)x);
    case ORC_F32_F16: return oracle_f32_to_f16((uint32_t)x);
    case ORC_F16_BF16: return oracle_f16_to_bf16((uint16_t)x);
    case ORC_BF16_F32: return oracle_bf16_to_f32((uint16_t)x);
    case ORC_F16_F32: return oracle_f16_to_f32((uint16_t)x);
    default: return x;
    }
}

/* Array forms for the pins (one conversion over n elements). */
void oracle_convert_array(int conv, const void *in, void *out, uint64_t n)
{
    const int in16 = conv == ORC_F16_BF16 || conv == ORC_BF16_F32 || conv == ORC_F16_F32;
    const int out16 = conv == ORC_F32_BF16 || conv == ORC_F32_F16 || conv == ORC_F16_BF16;
    for (uint64_t i = 0; i < n; ++i) {
        const uint64_t x = in16 ? ((const uint16_t *)in)[i] : ((const uint32_t *)in)[i];
        const uint64_t y = orc_convert(conv, x);
        if (out16) ((uint16_t *)out)[i] = (uint16_t)y;
        else ((uint32_t *)out)[i] = (uint32_t)y;
    }
}

static uint64_t read_le(const uint8_t *p, int nbytes)
{
    uint64_t x = 0;
    for (int k = 0; k < nbytes; ++k) x |= (uint64_t)p[k] << (8 * k);
    return x;
}

static void write_le(uint8_t *p, uint64_t y, int nbytes)
{
    for (int k = 0; k < nbytes; ++k) p[k] = (uint8_t)(y >> (8 * k));
}

/*
 * Unpacks every entry whose destination buffer is given.
 *
 *   e_*            entry columns (n_entries); e_shape is n_entries x 8, row-major;
 *                  e_stride may be NULL (every entry contiguous).
 *   d_*            destination columns (n_dsts); d_shape is n_dsts x 8.
 *   d_buf[j]       host buffer of destination j (its full byte size), or NULL: entries into a
 *                  NULL destination are still validated but not executed.
 *   d_cover[j]     optional per-byte write counters of destination j (NULL to skip).
 *   blob           holds blob bytes [blob_begin, blob_end).
 *   blob_bytes     length of the whole blob (for the bounds rule).
 *   cksum          n_entries accumulators, added to (the caller zeroes them).
 *   bad_entry      receives the first failing entry, or -1.
 * Returns ORC_OK or the first failure's code.  An entry whose bytes lie outside
 * [blob_begin, blob_end) but inside the blob is skipped like a NULL destination.
 */
int oracle_unpack(uint64_t n_entries, const int32_t *e_dtype, const int32_t *e_ndim,
                  const int64_t *e_shape, const uint64_t *e_offset, const int32_t *e_dst,
                  const int64_t *e_row, const uint32_t *e_flags, const uint32_t *e_stride,
                  uint64_t n_dsts, const int32_t *d_dtype, const int32_t *d_ndim,
                  const int64_t *d_shape, uint8_t *const *d_buf, uint32_t *const *d_cover,
                  const uint8_t *blob, uint64_t blob_begin, uint64_t blob_end,
                  uint64_t blob_bytes, uint64_t *cksum, int64_t *bad_entry)
{
    *bad_entry = -1;
    for (uint64_t t = 0; t < n_entries; ++t) {
        const int es_s = orc_elem_size(e_dtype[t]);
        if (es_s == 0 || e_ndim[t] < 0 || e_ndim[t] > 8) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
        if (e_dst[t] < 0 || (uint64_t)e_dst[t] >= n_dsts) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
        const uint64_t j = (uint64_t)e_dst[t];
        const int es_dt = orc_elem_size(d_dtype[j]);
        if (es_dt == 0 || d_ndim[j] < 0 || d_ndim[j] > 8) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
        const int converts = (e_flags[t] & ORC_CONVERT) != 0;

        /* dtypes */
        const int conv = converts ? orc_conversion(e_dtype[t], d_dtype[j]) : ORC_NONE;
        if (converts ? conv == ORC_NONE : e_dtype[t] != d_dtype[j]) {
            *bad_entry = (int64_t)t;
            return ORC_E_DTYPE;
        }
        const int es_d = es_dt;

        /* element counts */
        uint64_t n = 1;
        for (int k = 0; k < e_ndim[t]; ++k) {
            if (e_shape[8 * t + k] < 0) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
            n *= (uint64_t)e_shape[8 * t + k];
        }
        uint64_t d_numel = 1;
        for (int k = 0; k < d_ndim[j]; ++k) {
            if (d_shape[8 * j + k] < 0) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
            d_numel *= (uint64_t)d_shape[8 * j + k];
        }

        /* placement inside the destination */
        if (e_row[t] < 0) { *bad_entry = (int64_t)t; return ORC_E_OOB; }
        uint64_t row_elems;
        if (d_ndim[j] >= 2) {
            row_elems = (uint64_t)d_shape[8 * j + d_ndim[j] - 1];
            if (n > 0) {
                if (e_ndim[t] < 1 || (uint64_t)e_shape[8 * t + e_ndim[t] - 1] != row_elems) {
                    *bad_entry = (int64_t)t;
                    return ORC_E_SHAPE;
                }
            }
        } else {
            row_elems = 1;
        }
        const uint64_t base_elem = (uint64_t)e_row[t] * row_elems;
        if (base_elem + n > d_numel) { *bad_entry = (int64_t)t; return ORC_E_OOB; }
        const uint64_t base = base_elem * (uint64_t)es_d;

        /* source layout: rows of C elements, `stride` elements apart */
        const uint64_t C = e_ndim[t] >= 1 ? (uint64_t)e_shape[8 * t + e_ndim[t] - 1] : 1;
        const uint64_t given = e_stride ? (uint64_t)e_stride[t] : 0;
        if (given != 0 && (e_ndim[t] < 1 || given < C)) { *bad_entry = (int64_t)t; return ORC_E_INVAL; }
        const uint64_t stride = given ? given : C;
        /* elements the entry spans in the blob, from its first to its last element */
        const uint64_t extent = n == 0 ? 0 : (n / C - 1) * stride + C;

        /* source range */
        if (e_offset[t] % (uint64_t)es_s != 0) { *bad_entry = (int64_t)t; return ORC_E_ALIGN; }
        if (e_offset[t] + extent * (uint64_t)es_s > blob_bytes) { *bad_entry = (int64_t)t; return ORC_E_OOB; }

        if (d_buf[j] == NULL || n == 0) continue;
        if (e_offset[t] < blob_begin || e_offset[t] + extent * (uint64_t)es_s > blob_end) continue;

        const uint8_t *src = blob + (e_offset[t] - blob_begin);
        uint8_t *dst = d_buf[j] + base;
        uint32_t *cover = d_cover ? d_cover[j] : NULL;
        uint64_t ck = 0;
        for (uint64_t i = 0; i < n; ++i) {
            const uint64_t src_i = (i / C) * stride + (i % C);
            const uint64_t x = read_le(src + src_i * (uint64_t)es_s, es_s);
            const uint64_t y = converts ? orc_convert(conv, x) : x;
            write_le(dst + i * (uint64_t)es_d, y, es_d);
            if (cover)
                for (int k = 0; k < es_d; ++k) cover[base + i * (uint64_t)es_d + (uint64_t)k] += 1u;
            ck += y;
        }
        if (e_flags[t] & ORC_CKSUM) cksum[t] += ck;
    }
    return ORC_OK;
}

/* Strict-mode rule: every byte of every checked destination covered exactly once.  Returns
 * ORC_OK, ORC_E_OVERLAP or ORC_E_COVERAGE and the failing destination in *bad_dst. */
int oracle_check_cover(uint64_t n_dsts, const uint64_t *d_nbytes, uint32_t *const *d_cover,
                       int64_t *bad_dst)
{
    *bad_dst = -1;
    for (uint64_t j = 0; j < n_dsts; ++j) {
        if (d_cover[j] == NULL) continue;
        for (uint64_t b = 0; b < d_nbytes[j]; ++b) {
            if (d_cover[j][b] > 1u) { *bad_dst = (int64_t)j; return ORC_E_OVERLAP; }
            if (d_cover[j][b] == 0u) { *bad_dst = (int64_t)j; return ORC_E_COVERAGE; }
        }
    }
    return ORC_OK;
}
