/*
 * Checkpoint files: the InDisk end of InstantInfer's tensor-materialization automaton
 * (section 4.2: chunks move InDisk -> InMem before InGPU).
 *
 *   - safetensors headers: the file is an 8-byte little-endian header length N, N bytes of JSON
 *     mapping each tensor name to {"dtype", "shape", "data_offsets": [begin, end]} (plus an
 *     optional "__metadata__" object of strings), then the data section.  The data section is
 *     the loader's blob; data_offsets are blob offsets.  The parser below reads only the header.
 *   - a file source: a CALLBACK source whose fill reads blob bytes with pread from the data
 *     section, safe to call from several fill threads at once.
 *
 * Host-only C; no CUDA.
 */
#define _GNU_SOURCE
#include <errno.h>
#include <fcntl.h>
#include <pthread.h>
#include <stdarg.h>
#include <stddef.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <unistd.h>

#include "cfa_internal.h"

#define ST_MAX_HEADER (100ull << 20) /* the format's own limit on the header */

struct cfa_safetensors {
    size_t n;
    cfa_st_tensor *t;
    char **names;
    uint64_t data_offset; /* 8 + N */
    uint64_t data_bytes;  /* file size - data_offset */
};

/* The first failure detail of the current call (reported through cfa_last_error(NULL)). */
static _Thread_local char g_files_err[256];

static void ferr(const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_files_err, sizeof g_files_err, fmt, ap);
    va_end(ap);
    cfa_internal_set_error(g_files_err);
}

/* ---- a small JSON reader, enough for safetensors headers ------------------------------- */

typedef struct {
    const char *p, *end;
    int depth;
} jrd;

static void jws(jrd *r)
{
    while (r->p < r->end && (*r->p == ' ' || *r->p == '\t' || *r->p == '\n' || *r->p == '\r'))
        r->p++;
}

static int jlit(jrd *r, char c)
{
    jws(r);
    if (r->p < r->end && *r->p == c) {
        r->p++;
        return 1;
    }
    return 0;
}

static void put_utf8(char **o, unsigned cp)
{
    char *q = *o;
    if (cp < 0x80) {
        *q++ = (char)cp;
    } else if (cp < 0x800) {
        *q++ = (char)(0xC0 | (cp >> 6));
        *q++ = (char)(0x80 | (cp & 0x3F));
    } else if (cp < 0x10000) {
        *q++ = (char)(0xE0 | (cp >> 12));
        *q++ = (char)(0x80 | ((cp >> 6) & 0x3F));
        *q++ = (char)(0x80 | (cp & 0x3F));
    } else {
        *q++ = (char)(0xF0 | (cp >> 18));
        *q++ = (char)(0x80 | ((cp >> 12) & 0x3F));
        *q++ = (char)(0x80 | ((cp >> 6) & 0x3F));
        *q++ = (char)(0x80 | (cp & 0x3F));
    }
    *o = q;
}

static int hex4(const char *s, unsigned *v)
{
    *v = 0;
    for (int k = 0; k < 4; ++k) {
        const char c = s[k];
        unsigned d;
        if (c >= '0' && c <= '9') d = (unsigned)(c - '0');
        else if (c >= 'a' && c <= 'f') d = (unsigned)(c - 'a' + 10);
        else if (c >= 'A' && c <= 'F') d = (unsigned)(c - 'A' + 10);
        else return 0;
        *v = (*v << 4) | d;
    }
    return 1;
}

/* Length of the well-formed UTF-8 sequence starting at s (at most `left` bytes), 0 if it is
 * not one: the ranges of the Unicode standard's table of well-formed byte sequences, which
 * exclude overlong forms, UTF-16 surrogates and code points above U+10FFFF. */
static int utf8_len(const unsigned char *s, ptrdiff_t left)
{
    const unsigned c = s[0];
    int n;
    unsigned lo = 0x80, hi = 0xBF; /* range of the second byte */
    if (c < 0x80) return 1;
    if (c >= 0xC2 && c <= 0xDF) n = 2;
    else if (c >= 0xE0 && c <= 0xEF) {
        n = 3;
        if (c == 0xE0) lo = 0xA0;
        if (c == 0xED) hi = 0x9F;
    } else if (c >= 0xF0 && c <= 0xF4) {
        n = 4;
        if (c == 0xF0) lo = 0x90;
        if (c == 0xF4) hi = 0x8F;
    } else {
        return 0;
    }
    if (left < n || s[1] < lo || s[1] > hi) return 0;
    for (int k = 2; k < n; ++k)
        if (s[k] < 0x80 || s[k] > 0xBF) return 0;
    return n;
}

/* Reads a string; returns a malloc'd, NUL-terminated UTF-8 copy (NULL on error, including
 * control characters and bytes that are not well-formed UTF-8). */
static char *jstr(jrd *r)
{
    jws(r);
    if (r->p >= r->end || *r->p != '"') return NULL;
    r->p++;
    const char *s = r->p;
    size_t n = 0;
    while (s + n < r->end && s[n] != '"') n += (s[n] == '\\') ? 2 : 1;
    if (s + n >= r->end) return NULL;
    char *out = (char *)malloc(n + 1), *o = out;
    if (!out) return NULL;
    while (r->p < r->end && *r->p != '"') {
        if ((unsigned char)*r->p >= 0x80) {
            const int len = utf8_len((const unsigned char *)r->p, r->end - r->p);
            if (!len) goto bad;
            memcpy(o, r->p, (size_t)len);
            o += len;
            r->p += len;
            continue;
        }
        char c = *r->p++;
        if ((unsigned char)c < 0x20) goto bad;
        if (c != '\\') {
            *o++ = c;
            continue;
        }
        if (r->p >= r->end) goto bad;
        c = *r->p++;
        switch (c) {
        case '"': *o++ = '"'; break;
        case '\\': *o++ = '\\'; break;
        case '/': *o++ = '/'; break;
        case 'b': *o++ = '\b'; break;
        case 'f': *o++ = '\f'; break;
        case 'n': *o++ = '\n'; break;
        case 'r': *o++ = '\r'; break;
        case 't': *o++ = '\t'; break;
        case 'u': {
            unsigned cp;
            if (r->end - r->p < 4 || !hex4(r->p, &cp)) goto bad;
            r->p += 4;
            if (cp >= 0xD800 && cp < 0xDC00) { /* surrogate pair */
                unsigned lo;
                if (r->end - r->p < 6 || r->p[0] != '\\' || r->p[1] != 'u' || !hex4(r->p + 2, &lo) ||
                    lo < 0xDC00 || lo >= 0xE000)
                    goto bad;
                r->p += 6;
                cp = 0x10000 + ((cp - 0xD800) << 10) + (lo - 0xDC00);
            } else if ((cp >= 0xDC00 && cp < 0xE000) || cp == 0) {
                goto bad; /* a lone low surrogate, or U+0000, which a C string cannot hold */
            }
            put_utf8(&o, cp);
            break;
        }
        default: goto bad;
        }
    }
    if (r->p >= r->end) goto bad;
    r->p++; /* closing quote */
    *o = 0;
    return out;
bad:
    free(out);
    return NULL;
}

/* Reads a non-negative integer (no sign, fraction or exponent). */
static int juint(jrd *r, uint64_t *v)
{
    jws(r);
    const char *s = r->p;
    uint64_t x = 0;
    while (r->p < r->end && *r->p >= '0' && *r->p <= '9') {
        const uint64_t d = (uint64_t)(*r->p - '0');
        if (x > (UINT64_MAX - d) / 10) return 0;
        x = x * 10 + d;
        r->p++;
    }
    if (r->p == s || (*s == '0' && r->p - s > 1)) return 0; /* JSON allows no leading zero */
    if (r->p < r->end && (*r->p == '.' || *r->p == 'e' || *r->p == 'E')) return 0;
    *v = x;
    return 1;
}

static int jdigits(jrd *r)
{
    const char *s = r->p;
    while (r->p < r->end && *r->p >= '0' && *r->p <= '9') r->p++;
    return r->p > s;
}

/* Skips a number of the JSON grammar: -? (0 | [1-9][0-9]*) (. [0-9]+)? ([eE] [+-]? [0-9]+)? */
static int jnumber(jrd *r)
{
    if (r->p < r->end && *r->p == '-') r->p++;
    if (r->p < r->end && *r->p == '0') r->p++;
    else if (!jdigits(r)) return 0;
    if (r->p < r->end && *r->p == '.') {
        r->p++;
        if (!jdigits(r)) return 0;
    }
    if (r->p < r->end && (*r->p == 'e' || *r->p == 'E')) {
        r->p++;
        if (r->p < r->end && (*r->p == '+' || *r->p == '-')) r->p++;
        if (!jdigits(r)) return 0;
    }
    return 1;
}

/* Skips any JSON value (used for unknown keys and __metadata__). */
static int jskip(jrd *r)
{
    jws(r);
    if (r->p >= r->end || ++r->depth > 64) return 0;
    int ok = 1;
    const char c = *r->p;
    if (c == '"') {
        char *s = jstr(r);
        ok = s != NULL;
        free(s);
    } else if (c == '{' || c == '[') {
        const char close = c == '{' ? '}' : ']';
        r->p++;
        if (!jlit(r, close)) {
            do {
                if (c == '{') {
                    char *k = jstr(r);
                    if (!k) { ok = 0; break; }
                    free(k);
                    if (!jlit(r, ':')) { ok = 0; break; }
                }
                if (!jskip(r)) { ok = 0; break; }
            } while (jlit(r, ','));
            if (ok && !jlit(r, close)) ok = 0;
        }
    } else if (c == '-' || (c >= '0' && c <= '9')) {
        ok = jnumber(r);
    } else if (r->end - r->p >= 4 && !memcmp(r->p, "true", 4)) {
        r->p += 4;
    } else if (r->end - r->p >= 5 && !memcmp(r->p, "false", 5)) {
        r->p += 5;
    } else if (r->end - r->p >= 4 && !memcmp(r->p, "null", 4)) {
        r->p += 4;
    } else {
        ok = 0;
    }
    r->depth--;
    return ok;
}

static int st_dtype(const char *s, int *es)
{
    static const struct { const char *name; int dt, es; } map[] = {
        {"BOOL", CFA_DTYPE_U8, 1},  {"U8", CFA_DTYPE_U8, 1},       {"I8", CFA_DTYPE_U8, 1},
        {"F8_E4M3", CFA_DTYPE_U8, 1}, {"F8_E5M2", CFA_DTYPE_U8, 1}, {"I16", CFA_DTYPE_I16, 2},
        {"U16", CFA_DTYPE_I16, 2},  {"F16", CFA_DTYPE_F16, 2},     {"BF16", CFA_DTYPE_BF16, 2},
        {"I32", CFA_DTYPE_I32, 4},  {"U32", CFA_DTYPE_I32, 4},     {"F32", CFA_DTYPE_F32, 4},
        {"I64", CFA_DTYPE_I64, 8},  {"U64", CFA_DTYPE_I64, 8},     {"F64", CFA_DTYPE_F64, 8},
    };
    for (size_t k = 0; k < sizeof map / sizeof map[0]; ++k)
        if (!strcmp(s, map[k].name)) {
            *es = map[k].es;
            return map[k].dt;
        }
    return 0;
}

/* One tensor object: {"dtype": ..., "shape": [...], "data_offsets": [b, e]} in any order. */
static int st_tensor(jrd *r, cfa_st_tensor *t, uint64_t *b, uint64_t *e, int *es)
{
    int have_dt = 0, have_shape = 0, have_off = 0;
    if (!jlit(r, '{')) return 0;
    if (jlit(r, '}')) return 0;
    do {
        char *key = jstr(r);
        if (!key || !jlit(r, ':')) {
            free(key);
            return 0;
        }
        if (!strcmp(key, "dtype")) {
            char *v = jstr(r);
            if (!v) {
                free(key);
                return 0;
            }
            t->dtype = st_dtype(v, es);
            free(v);
            have_dt = 1;
            if (!t->dtype) {
                ferr("unsupported safetensors dtype");
                free(key);
                return 0;
            }
        } else if (!strcmp(key, "shape")) {
            if (!jlit(r, '[')) { free(key); return 0; }
            t->ndim = 0;
            if (!jlit(r, ']')) {
                do {
                    uint64_t d;
                    if (t->ndim >= CFA_MAX_DIMS || !juint(r, &d) || d > (uint64_t)INT64_MAX) {
                        free(key);
                        return 0;
                    }
                    t->shape[t->ndim++] = (int64_t)d;
                } while (jlit(r, ','));
                if (!jlit(r, ']')) { free(key); return 0; }
            }
            have_shape = 1;
        } else if (!strcmp(key, "data_offsets")) {
            if (!jlit(r, '[') || !juint(r, b) || !jlit(r, ',') || !juint(r, e) || !jlit(r, ']')) {
                free(key);
                return 0;
            }
            have_off = 1;
        } else if (!jskip(r)) {
            free(key);
            return 0;
        }
        free(key);
    } while (jlit(r, ','));
    return jlit(r, '}') && have_dt && have_shape && have_off;
}

static void st_free(cfa_safetensors *st)
{
    if (!st) return;
    if (st->names)
        for (size_t i = 0; i < st->n; ++i) free(st->names[i]);
    free(st->names);
    free(st->t);
    free(st);
}

/* Parses a header held in memory; file_bytes is the size of the whole file. */
cfa_status cfa_safetensors_parse(const void *header, uint64_t header_len, uint64_t file_bytes,
                                 cfa_safetensors **out)
{
    if (!out || (!header && header_len)) return CFA_ERR_INVAL;
    g_files_err[0] = 0;
    *out = NULL;
    cfa_safetensors *st = (cfa_safetensors *)calloc(1, sizeof *st);
    if (!st) return CFA_ERR_NOMEM;
    st->data_offset = 8 + header_len;
    if (file_bytes < st->data_offset) {
        ferr("file shorter than its header");
        st_free(st);
        return CFA_ERR_INVAL;
    }
    st->data_bytes = file_bytes - st->data_offset;
    jrd r = {(const char *)header, (const char *)header + header_len, 0};
    size_t cap = 0;
    int ok = jlit(&r, '{');
    if (ok && !jlit(&r, '}')) {
        do {
            char *name = jstr(&r);
            if (!name || !jlit(&r, ':')) {
                free(name);
                ok = 0;
                break;
            }
            if (!strcmp(name, "__metadata__")) {
                free(name);
                if (!jskip(&r)) { ok = 0; break; }
                continue;
            }
            if (st->n == cap) {
                cap = cap ? 2 * cap : 256;
                cfa_st_tensor *t = (cfa_st_tensor *)realloc(st->t, cap * sizeof *t);
                char **nm = (char **)realloc(st->names, cap * sizeof *nm);
                if (t) st->t = t;
                if (nm) st->names = nm;
                if (!t || !nm) {
                    free(name);
                    st_free(st);
                    return CFA_ERR_NOMEM;
                }
            }
            cfa_st_tensor *t = &st->t[st->n];
            memset(t, 0, sizeof *t);
            st->names[st->n] = name;
            st->n++;
            t->name = name;
            uint64_t b = 0, e = 0;
            int es = 0;
            if (!st_tensor(&r, t, &b, &e, &es)) {
                if (!g_files_err[0]) ferr("malformed entry for tensor %s", name);
                ok = 0;
                break;
            }
            /* the product of the non-zero dimensions must fit in 64 bits, whatever their order */
            uint64_t numel = 1;
            int zero = 0;
            for (int k = 0; k < t->ndim; ++k) {
                const uint64_t d = (uint64_t)t->shape[k];
                if (!d) {
                    zero = 1;
                    continue;
                }
                if (numel > UINT64_MAX / d) { ok = 0; break; }
                numel *= d;
            }
            if (zero) numel = 0;
            if (!ok || e < b || e > st->data_bytes || (e - b) / (uint64_t)es != numel ||
                (e - b) % (uint64_t)es) {
                ferr("tensor %s: data_offsets [%llu, %llu) do not fit its shape and dtype or the "
                     "file", name, (unsigned long long)b, (unsigned long long)e);
                ok = 0;
                break;
            }
            t->blob_offset = b;
            t->nbytes = e - b;
        } while (jlit(&r, ','));
        if (ok && !jlit(&r, '}')) ok = 0;
    }
    jws(&r);
    if (ok && r.p != r.end) ok = 0;
    if (!ok) {
        if (!g_files_err[0]) ferr("malformed safetensors header");
        st_free(st);
        return CFA_ERR_INVAL;
    }
    *out = st;
    return CFA_OK;
}

cfa_status cfa_safetensors_open(const char *path, cfa_safetensors **out)
{
    g_files_err[0] = 0;
    if (!path || !out) return CFA_ERR_INVAL;
    *out = NULL;
    const int fd = open(path, O_RDONLY | O_CLOEXEC);
    if (fd < 0) {
        ferr("cannot open %s: %s", path, strerror(errno));
        return CFA_ERR_SOURCE;
    }
    struct stat sb;
    unsigned char len8[8];
    cfa_status stc = CFA_OK;
    char *hdr = NULL;
    if (fstat(fd, &sb) != 0 || pread(fd, len8, 8, 0) != 8) {
        ferr("cannot read the header length of %s", path);
        stc = CFA_ERR_SOURCE;
        goto out;
    }
    uint64_t n = 0;
    for (int k = 7; k >= 0; --k) n = (n << 8) | len8[k];
    if (n > ST_MAX_HEADER || n + 8 > (uint64_t)sb.st_size) {
        ferr("header length %llu is not plausible for %s", (unsigned long long)n, path);
        stc = CFA_ERR_INVAL;
        goto out;
    }
    hdr = (char *)malloc(n ? n : 1);
    if (!hdr) {
        stc = CFA_ERR_NOMEM;
        goto out;
    }
    for (uint64_t got = 0; got < n;) {
        const ssize_t k = pread(fd, hdr + got, n - got, (off_t)(8 + got));
        if (k < 0 && errno == EINTR) continue;
        if (k <= 0) {
            ferr("short read of the header of %s", path);
            stc = CFA_ERR_SOURCE;
            goto out;
        }
        got += (uint64_t)k;
    }
    stc = cfa_safetensors_parse(hdr, n, (uint64_t)sb.st_size, out);
    if (stc != CFA_OK && !g_files_err[0]) ferr("%s: malformed safetensors header", path);
out:
    free(hdr);
    close(fd);
    return stc;
}

cfa_status cfa_safetensors_info(const cfa_safetensors *st, size_t *n_tensors,
                                uint64_t *data_offset, uint64_t *data_bytes)
{
    if (!st) return CFA_ERR_INVAL;
    if (n_tensors) *n_tensors = st->n;
    if (data_offset) *data_offset = st->data_offset;
    if (data_bytes) *data_bytes = st->data_bytes;
    return CFA_OK;
}

cfa_status cfa_safetensors_tensor(const cfa_safetensors *st, size_t i, cfa_st_tensor *out)
{
    if (!st || !out || i >= st->n) return CFA_ERR_INVAL;
    *out = st->t[i];
    return CFA_OK;
}

cfa_status cfa_safetensors_names(const cfa_safetensors *st, char *buf, uint64_t cap,
                                 uint64_t *bytes)
{
    if (!st || !bytes || (cap && !buf)) return CFA_ERR_INVAL;
    uint64_t need = 0;
    for (size_t i = 0; i < st->n; ++i) need += strlen(st->t[i].name) + 1;
    *bytes = need;
    if (!buf) return CFA_OK;
    if (cap < need) return CFA_ERR_INVAL;
    char *o = buf;
    for (size_t i = 0; i < st->n; ++i) {
        const size_t k = strlen(st->t[i].name) + 1;
        memcpy(o, st->t[i].name, k);
        o += k;
    }
    return CFA_OK;
}

cfa_status cfa_safetensors_tensors(const cfa_safetensors *st, size_t first, size_t count,
                                   cfa_st_tensor *out)
{
    if (!st || (count && !out) || first > st->n || count > st->n - first) return CFA_ERR_INVAL;
    if (count) memcpy(out, st->t + first, count * sizeof *out);
    return CFA_OK;
}

cfa_status cfa_safetensors_close(cfa_safetensors *st)
{
    st_free(st);
    return CFA_OK;
}

/* ---- a file source --------------------------------------------------------------------- */

/* Direct reads: file offsets, lengths and buffer addresses in multiples of this. */
#define FD_BLOCK 4096u
/* Bounce buffer size of one direct read. */
#define FD_BOUNCE (4u << 20)

typedef struct bounce {
    struct bounce *next;
    uint8_t *buf; /* FD_BOUNCE bytes, FD_BLOCK-aligned */
} bounce;

typedef struct {
    int fd;
    int direct;
    const uint8_t *map; /* CFA_FILE_MMAP(_IN_PLACE): the whole file, mapped read-only */
    uint64_t data_offset;
    uint64_t file_bytes;
    pthread_mutex_t mu; /* guards `free_list` */
    bounce *free_list;  /* bounce buffers not in use (direct reads only) */
} file_src;

/* Reads exactly len bytes at file offset fo into d (buffered, or direct when every one of d,
 * fo and len is a multiple of FD_BLOCK, except that a direct read may end at end of file). */
static int read_full(int fd, uint8_t *d, uint64_t len, uint64_t fo)
{
    for (uint64_t got = 0; got < len;) {
        const ssize_t k = pread(fd, d + got, len - got, (off_t)(fo + got));
        if (k < 0 && errno == EINTR) continue;
        if (k <= 0) return 2;
        got += (uint64_t)k;
    }
    return 0;
}

static bounce *take_bounce(file_src *f)
{
    pthread_mutex_lock(&f->mu);
    bounce *b = f->free_list;
    if (b) f->free_list = b->next;
    pthread_mutex_unlock(&f->mu);
    if (b) return b;
    b = (bounce *)calloc(1, sizeof *b);
    if (!b) return NULL;
    if (posix_memalign((void **)&b->buf, FD_BLOCK, FD_BOUNCE) != 0) {
        free(b);
        return NULL;
    }
    return b;
}

static void give_bounce(file_src *f, bounce *b)
{
    pthread_mutex_lock(&f->mu);
    b->next = f->free_list;
    f->free_list = b;
    pthread_mutex_unlock(&f->mu);
}

/* Direct read of file bytes [fo, fo + len) into d through a bounce buffer: whole blocks are
 * read into the buffer (the last one may stop at end of file) and the wanted bytes copied out. */
static int bounce_read(file_src *f, uint8_t *d, uint64_t len, uint64_t fo)
{
    bounce *b = take_bounce(f);
    if (!b) return 3;
    int rc = 0;
    while (len && !rc) {
        const uint64_t a = fo & ~(uint64_t)(FD_BLOCK - 1);
        const uint64_t head = fo - a;
        uint64_t want = head + len;
        if (want > FD_BOUNCE) want = FD_BOUNCE;
        uint64_t span = (want + FD_BLOCK - 1) & ~(uint64_t)(FD_BLOCK - 1);
        if (a + span > f->file_bytes) { /* the file's last block: read up to its end */
            const uint64_t tail = f->file_bytes - a;
            span = (tail + FD_BLOCK - 1) & ~(uint64_t)(FD_BLOCK - 1);
            if (want > tail) want = tail;
        }
        uint64_t got = 0;
        while (got < want) {
            const ssize_t k = pread(f->fd, b->buf + got, span - got, (off_t)(a + got));
            if (k < 0 && errno == EINTR) continue;
            if (k <= 0) break;
            got += (uint64_t)k;
        }
        if (got < want || want <= head) {
            rc = 2;
            break;
        }
        const uint64_t n = want - head;
        memcpy(d, b->buf + head, n);
        d += n;
        fo += n;
        len -= n;
    }
    give_bounce(f, b);
    return rc;
}

/* O_DIRECT fill: when the destination and the file offset share their position within a
 * block, the whole blocks in the middle are read straight into the destination and only the
 * partial first and last blocks go through a bounce buffer; otherwise everything bounces. */
static int direct_fill(file_src *f, uint8_t *d, uint64_t len, uint64_t fo)
{
    const uint64_t B = FD_BLOCK;
    if (((uintptr_t)d & (B - 1)) == (fo & (B - 1))) {
        const uint64_t lo = (fo + B - 1) & ~(B - 1);
        const uint64_t hi = (fo + len) & ~(B - 1);
        if (hi > lo) {
            int rc = 0;
            if (lo > fo) rc = bounce_read(f, d, lo - fo, fo);
            if (!rc) rc = read_full(f->fd, d + (lo - fo), hi - lo, lo);
            if (!rc && fo + len > hi) rc = bounce_read(f, d + (hi - fo), fo + len - hi, hi);
            return rc;
        }
    }
    return bounce_read(f, d, len, fo);
}

static int file_fill(void *user, uint64_t off, void *dst, uint64_t len)
{
    file_src *f = (file_src *)user;
    const uint64_t fo = f->data_offset + off; /* file offset; every sum checked for wrap-around */
    if (fo < off || fo + len < fo || fo + len > f->file_bytes) return 1;
    if (!len) return 0;
    if (f->map) {
        memcpy(dst, f->map + fo, len);
        return 0;
    }
    if (f->direct) return direct_fill(f, (uint8_t *)dst, len, fo);
    return read_full(f->fd, (uint8_t *)dst, len, fo);
}

cfa_status cfa_file_source_open(const char *path, uint64_t data_offset, uint32_t flags,
                                cfa_source *out)
{
    g_files_err[0] = 0;
    const uint32_t modes = flags & (CFA_FILE_DIRECT | CFA_FILE_MMAP | CFA_FILE_MMAP_IN_PLACE);
    if (!path || !out || modes != flags || (modes & (modes - 1)))
        return CFA_ERR_INVAL; /* an unknown flag, or more than one mode */
    const int in_place = (flags & CFA_FILE_MMAP_IN_PLACE) != 0;
    if (in_place && (data_offset & 7u)) {
        ferr("in-place reads need the data section at a multiple of 8 bytes in the file (data "
             "offset %llu)", (unsigned long long)data_offset);
        return CFA_ERR_ALIGN;
    }
    memset(out, 0, sizeof *out);
    file_src *f = (file_src *)calloc(1, sizeof *f);
    if (!f) return CFA_ERR_NOMEM;
    f->direct = (flags & CFA_FILE_DIRECT) != 0;
    f->fd = open(path, O_RDONLY | O_CLOEXEC | (f->direct ? O_DIRECT : 0));
    struct stat sb;
    if (f->fd < 0 || fstat(f->fd, &sb) != 0) {
        if (f->direct && errno == EINVAL)
            ferr("cannot open %s for direct reads: the file system does not support O_DIRECT",
                 path);
        else
            ferr("cannot open %s: %s", path, strerror(errno));
        if (f->fd >= 0) close(f->fd);
        free(f);
        return CFA_ERR_SOURCE;
    }
    if (!f->direct) posix_fadvise(f->fd, 0, 0, POSIX_FADV_SEQUENTIAL);
    pthread_mutex_init(&f->mu, NULL);
    f->data_offset = data_offset;
    f->file_bytes = (uint64_t)sb.st_size;
    if (data_offset > f->file_bytes) {
        ferr("data offset %llu is past the end of %s (%llu bytes)",
             (unsigned long long)data_offset, path, (unsigned long long)f->file_bytes);
        pthread_mutex_destroy(&f->mu);
        close(f->fd);
        free(f);
        return CFA_ERR_SOURCE;
    }
    if ((flags & (CFA_FILE_MMAP | CFA_FILE_MMAP_IN_PLACE)) && f->file_bytes) {
        /* in place, the pages are mapped up front (read into the page cache if they are not
         * there yet), so the kernels' first reads do not wait on page faults */
        void *m = mmap(NULL, (size_t)f->file_bytes, PROT_READ,
                       MAP_SHARED | (in_place ? MAP_POPULATE : 0), f->fd, 0);
        if (m == MAP_FAILED) {
            ferr("cannot map %s: %s", path, strerror(errno));
            pthread_mutex_destroy(&f->mu);
            close(f->fd);
            free(f);
            return CFA_ERR_SOURCE;
        }
        f->map = (const uint8_t *)m;
    }
    out->fill = file_fill; /* for a HOST_DIRECT source only a mark: such loads never fill */
    out->user = f;
    if (in_place) {
        out->kind = CFA_SRC_HOST_DIRECT;
        out->base = f->map ? f->map + data_offset : NULL;
        out->size_bytes = f->file_bytes - data_offset;
    } else {
        out->kind = CFA_SRC_CALLBACK;
    }
    return CFA_OK;
}

cfa_status cfa_file_source_close(cfa_source *src)
{
    if (!src) return CFA_ERR_INVAL;
    if ((src->kind == CFA_SRC_CALLBACK || src->kind == CFA_SRC_HOST_DIRECT) &&
        src->fill == file_fill && src->user) {
        file_src *f = (file_src *)src->user;
        if (f->map) munmap((void *)f->map, (size_t)f->file_bytes);
        close(f->fd);
        for (bounce *b = f->free_list; b;) {
            bounce *n = b->next;
            free(b->buf);
            free(b);
            b = n;
        }
        pthread_mutex_destroy(&f->mu);
        free(f);
        src->user = NULL;
        return CFA_OK;
    }
    return CFA_ERR_INVAL;
}
