/*
 * Seeded, counter-based generator of synthetic checkpoint bytes ("blobs").
 *
 * Input infrastructure shared by the tests, the benchmark, the oracle side and the GPU side.
 * It holds none of the loader's arithmetic: it only produces the bytes a checkpoint file would
 * hold.  Because every 8-byte word is a pure function of (seed, word index), any byte range can
 * be regenerated on its own, in any order and on any number of threads, with identical bytes.
 *
 * Word stream: word w of seed s is output number w (counting from 0) of SplitMix64 seeded with s
 * (Steele, Lea, Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014; the
 * 64-bit finaliser constants are the ones Vigna publishes for splitmix64.c):
 *     state_w = s + (w + 1) * 0x9E3779B97F4A7C15
 *     z = (state_w ^ (state_w >> 30)) * 0xBF58476D1CE4E5B9
 *     z = (z ^ (z >> 27)) * 0x94D049BB133111EB
 *     word = z ^ (z >> 31)
 *
 * Kinds:
 *   bits   : blob byte o is byte (o mod 8) of word (o div 8), little-endian.  Used for bf16
 *            checkpoints, where a copy is bit-exact whatever the bits are.
 *   f32mix : 4-byte little-endian fp32 elements; element j (blob byte 4j) draws from words
 *            4p .. 4p+3 with p = j div 2.  Mostly normal(0, 0.02) values (Box-Muller on two
 *            53-bit uniforms, computed in double and rounded to float), plus per element, from
 *            16 selector bits c: c < 328 -> a tie pattern (upper half of the normal value,
 *            low half 0x8000); 328 <= c < 656 -> an fp32 subnormal (random sign, random
 *            non-zero 23-bit mantissa, a quarter of them with low half 0x8000);
 *            656 <= c < 660 -> a signed zero.  That is about 0.5 % ties, 0.5 % subnormals and
 *            a few zeros, and never NaN or Inf.
 *   f16fin : 2-byte little-endian binary16 patterns that are always finite: element j (blob byte
 *            2j) takes 16 bits of word j div 4; its exponent field, 5 bits that would be 31 for
 *            infinities and NaNs, is replaced by those bits mod 31 (so 0, subnormals, .. 30).
 */
#define _POSIX_C_SOURCE 200809L
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <time.h>

static inline uint64_t wl_word(uint64_t seed, uint64_t w)
{
    uint64_t z = seed + (w + 1u) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t wl_splitmix64_word(uint64_t seed, uint64_t w) { return wl_word(seed, w); }

/* Blob bytes [off, off + len) of kind "bits" into out. */
void wl_fill_bits(uint64_t seed, uint64_t off, uint64_t len, uint8_t *out)
{
    uint64_t o = off, end = off + len;
    /* leading bytes up to a word boundary */
    while (o < end && (o & 7u)) {
        uint64_t v = wl_word(seed, o >> 3);
        *out++ = (uint8_t)(v >> (8u * (o & 7u)));
        ++o;
    }
    /* whole words */
    while (o + 8 <= end) {
        uint64_t v = wl_word(seed, o >> 3);
        for (int k = 0; k < 8; ++k) out[k] = (uint8_t)(v >> (8 * k));
        out += 8;
        o += 8;
    }
    /* trailing bytes */
    while (o < end) {
        uint64_t v = wl_word(seed, o >> 3);
        *out++ = (uint8_t)(v >> (8u * (o & 7u)));
        ++o;
    }
}

static inline uint32_t wl_f32_bits(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    return u;
}

/* fp32 element j of kind "f32mix" as a bit pattern. */
static uint32_t wl_f32mix_elem(uint64_t seed, uint64_t j)
{
    const uint64_t p = j >> 1;
    const unsigned half = (unsigned)(j & 1u);
    const uint64_t ua = wl_word(seed, 4 * p + 0);
    const uint64_t ub = wl_word(seed, 4 * p + 1);
    const uint64_t uc = wl_word(seed, 4 * p + 2);
    const uint64_t ud = wl_word(seed, 4 * p + 3);

    const double u1 = ((double)(ua >> 11) + 1.0) * 0x1.0p-53; /* (0, 1] */
    const double u2 = (double)(ub >> 11) * 0x1.0p-53;         /* [0, 1) */
    const double r = sqrt(-2.0 * log(u1));
    const double two_pi = 6.283185307179586476925286766559;
    const double z = half ? r * sin(two_pi * u2) : r * cos(two_pi * u2);
    const uint32_t normal_bits = wl_f32_bits((float)(0.02 * z));

    const uint32_t sel = (uint32_t)(uc >> (half ? 16 : 0)) & 0xFFFFu;
    const uint32_t extra = (uint32_t)(ud >> (half ? 32 : 0)); /* 32 fresh bits */
    if (sel < 328u)
        return (normal_bits & 0xFFFF0000u) | 0x8000u;
    if (sel < 656u) {
        const uint32_t sign = (extra & 1u) << 31;
        uint32_t mant = (extra >> 1) & 0x7FFFFFu;
        if (((extra >> 24) & 3u) == 0u) mant = (mant & 0x7F0000u) | 0x8000u;
        if (mant == 0u) mant = 1u;
        return sign | mant;
    }
    if (sel < 660u) return (extra & 1u) << 31;
    return normal_bits;
}

/* Blob bytes [off, off + len) of kind "f32mix" into out; off and len multiples of 4. */
int wl_fill_f32mix(uint64_t seed, uint64_t off, uint64_t len, uint8_t *out)
{
    if ((off & 3u) || (len & 3u)) return -1;
    const uint64_t j0 = off >> 2, n = len >> 2;
    for (uint64_t i = 0; i < n; ++i) {
        const uint32_t v = wl_f32mix_elem(seed, j0 + i);
        out[4 * i + 0] = (uint8_t)v;
        out[4 * i + 1] = (uint8_t)(v >> 8);
        out[4 * i + 2] = (uint8_t)(v >> 16);
        out[4 * i + 3] = (uint8_t)(v >> 24);
    }
    return 0;
}

/* Blob bytes [off, off + len) of kind "f16fin" into out; off and len multiples of 2. */
int wl_fill_f16fin(uint64_t seed, uint64_t off, uint64_t len, uint8_t *out)
{
    if ((off & 1u) || (len & 1u)) return -1;
    const uint64_t j0 = off >> 1, n = len >> 1;
    for (uint64_t i = 0; i < n; ++i) {
        const uint64_t j = j0 + i;
        const uint32_t bits = (uint32_t)(wl_word(seed, j >> 2) >> (16 * (j & 3u))) & 0xFFFFu;
        const uint32_t e = ((bits >> 10) & 31u) % 31u;
        const uint32_t v = (bits & 0x83FFu) | (e << 10);
        out[2 * i] = (uint8_t)v;
        out[2 * i + 1] = (uint8_t)(v >> 8);
    }
    return 0;
}

/*
 * A fill callback with the loader's source signature, so that tests and the benchmark can
 * stream a blob that exists only as its generator definition.  `user` points to a
 * wl_cb_source.  Optional fault injection on the host: fail_from (return an error for ranges
 * reaching that blob offset) and delay_us (sleep before every call).
 */
typedef struct wl_cb_source {
    int32_t kind; /* 0 = bits, 1 = f32mix, 2 = f16fin */
    int32_t reserved;
    uint64_t seed;
    uint64_t period;    /* 0 = none */
    uint64_t fail_from; /* UINT64_MAX = never */
    uint64_t delay_us;
} wl_cb_source;

int wl_fill_cb(void *user, uint64_t off, void *dst, uint64_t len)
{
    const wl_cb_source *s = (const wl_cb_source *)user;
    if (s->delay_us) {
        struct timespec ts;
        ts.tv_sec = (time_t)(s->delay_us / 1000000u);
        ts.tv_nsec = (long)(s->delay_us % 1000000u) * 1000L;
        nanosleep(&ts, NULL);
    }
    if (off + len > s->fail_from) return 1;
    uint8_t *out = (uint8_t *)dst;
    while (len) {
        uint64_t o = s->period ? off % s->period : off;
        uint64_t take = s->period ? s->period - o : len;
        if (take > len) take = len;
        if (s->kind == 0) wl_fill_bits(s->seed, o, take, out);
        else if (s->kind == 1 ? wl_fill_f32mix(s->seed, o, take, out) != 0
                              : wl_fill_f16fin(s->seed, o, take, out) != 0)
            return 2;
        out += take;
        off += take;
        len -= take;
    }
    return 0;
}
