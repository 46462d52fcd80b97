/* Concurrent fills from a checkpoint file source (paper_2607_18957_gb300/csrc/cfa_files.c), the
 * way a load's fill threads call it: several threads read random ranges at random destination
 * alignments, in every read mode (pread, mapped copy, O_DIRECT where the file system allows it),
 * and every byte is compared with the file.  Requests past the data section, including ones
 * whose end wraps around 64 bits, must fail without touching memory.  Built with ThreadSanitizer
 * or AddressSanitizer by the test.  Usage: file_fill_stress <file> <data_offset>. */
#include <pthread.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "cfa.h"

void cfa_internal_set_error(const char *msg) { (void)msg; }

#define THREADS 8
#define FILLS 300
#define MAX_LEN (3u << 20)

static uint8_t *g_file;
static uint64_t g_data_offset, g_data_bytes;

typedef struct {
    const cfa_source *src;
    unsigned seed;
    int bad;
} worker;

static uint64_t rnd(unsigned *s)
{
    *s = *s * 1103515245u + 12345u;
    const uint64_t hi = (*s >> 8) & 0xFFFFFF;
    *s = *s * 1103515245u + 12345u;
    return (hi << 24) | ((*s >> 8) & 0xFFFFFF);
}

static void *run(void *arg)
{
    worker *w = (worker *)arg;
    uint8_t *buf = (uint8_t *)malloc(MAX_LEN + 4096);
    if (!buf) {
        w->bad = 1;
        return NULL;
    }
    for (int i = 0; i < FILLS && !w->bad; ++i) {
        uint64_t len = rnd(&w->seed) % (rnd(&w->seed) % 4 == 0 ? MAX_LEN : 9000);
        if (len > g_data_bytes) len = g_data_bytes;
        const uint64_t off = g_data_bytes - len ? rnd(&w->seed) % (g_data_bytes - len + 1) : 0;
        uint8_t *d = buf + rnd(&w->seed) % 4096;
        if (w->src->fill(w->src->user, off, d, len) != 0 ||
            memcmp(d, g_file + g_data_offset + off, len) != 0)
            w->bad = 2;
    }
    /* past the end, and ends that wrap around */
    if (w->src->fill(w->src->user, g_data_bytes, buf, 1) == 0) w->bad = 3;
    if (w->src->fill(w->src->user, 1, buf, g_data_bytes) == 0) w->bad = 4;
    if (w->src->fill(w->src->user, UINT64_MAX - 8, buf, 16) == 0) w->bad = 5;
    if (w->src->fill(w->src->user, 16, buf, UINT64_MAX - 8) == 0) w->bad = 6;
    /* offset + length fits, but adding the data section's file offset wraps around */
    if (w->src->fill(w->src->user, UINT64_MAX - g_data_offset - 3, buf, 16) == 0) w->bad = 7;
    free(buf);
    return NULL;
}

int main(int argc, char **argv)
{
    if (argc < 3) return 2;
    FILE *f = fopen(argv[1], "rb");
    if (!f) return 2;
    fseek(f, 0, SEEK_END);
    const long size = ftell(f);
    fseek(f, 0, SEEK_SET);
    g_file = (uint8_t *)malloc((size_t)size);
    if (!g_file || fread(g_file, 1, (size_t)size, f) != (size_t)size) return 2;
    fclose(f);
    g_data_offset = strtoull(argv[2], NULL, 10);
    g_data_bytes = (uint64_t)size - g_data_offset;
    const uint32_t modes[3] = {0, CFA_FILE_MMAP, CFA_FILE_DIRECT};
    for (int m = 0; m < 3; ++m) {
        cfa_source src;
        const cfa_status st = cfa_file_source_open(argv[1], g_data_offset, modes[m], &src);
        if (st == CFA_ERR_SOURCE && modes[m] == CFA_FILE_DIRECT) {
            printf("mode %u: no O_DIRECT here\n", modes[m]);
            continue;
        }
        if (st != CFA_OK) return 10 + m;
        pthread_t t[THREADS];
        worker w[THREADS];
        for (int k = 0; k < THREADS; ++k) {
            w[k].src = &src;
            w[k].seed = 77u + 1000u * (unsigned)m + (unsigned)k;
            w[k].bad = 0;
            pthread_create(&t[k], NULL, run, &w[k]);
        }
        for (int k = 0; k < THREADS; ++k) pthread_join(t[k], NULL);
        for (int k = 0; k < THREADS; ++k)
            if (w[k].bad) {
                fprintf(stderr, "mode %u thread %d: failure %d\n", modes[m], k, w[k].bad);
                return 20 + w[k].bad;
            }
        if (cfa_file_source_close(&src) != CFA_OK) return 30;
        printf("mode %u: ok\n", modes[m]);
    }
    /* a data section that starts past the end of the file is refused at open */
    cfa_source src;
    if (cfa_file_source_open(argv[1], (uint64_t)size + 1, CFA_FILE_MMAP, &src) != CFA_ERR_SOURCE)
        return 40;
    free(g_file);
    return 0;
}
