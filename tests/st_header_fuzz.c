/* Replays safetensors headers through the header parser (paper_2607_18957_gb300/csrc/cfa_files.c)
 * built with AddressSanitizer and UBSan, so that a read past a header's end or any undefined
 * behaviour aborts the run.  Input file: records of [u32 header length][u64 file size][header].
 * Accepted headers must give tensors that lie inside the data section with nbytes = the size
 * their shape and dtype give. */
#include <stdio.h>
#include <stdlib.h>

#include "cfa_internal.h"

void cfa_internal_set_error(const char *msg) { (void)msg; }

int main(int argc, char **argv)
{
    if (argc < 2) return 2;
    FILE *f = fopen(argv[1], "rb");
    if (!f) return 2;
    unsigned long ok = 0, rejected = 0;
    for (;;) {
        unsigned len;
        unsigned long long file_bytes;
        if (fread(&len, 4, 1, f) != 1 || fread(&file_bytes, 8, 1, f) != 1) break;
        char *h = (char *)malloc(len ? len : 1); /* exactly len bytes: ASan sees any overread */
        if (!h || (len && fread(h, 1, len, f) != len)) return 2;
        cfa_safetensors *st = NULL;
        if (cfa_safetensors_parse(h, len, file_bytes, &st) == CFA_OK) {
            size_t n = 0;
            uint64_t data_offset = 0, data_bytes = 0;
            if (cfa_safetensors_info(st, &n, &data_offset, &data_bytes) != CFA_OK) return 3;
            for (size_t i = 0; i < n; ++i) {
                cfa_st_tensor t;
                if (cfa_safetensors_tensor(st, i, &t) != CFA_OK) return 3;
                if (t.blob_offset > data_bytes || t.nbytes > data_bytes - t.blob_offset) return 4;
            }
            cfa_safetensors_close(st);
            ok++;
        } else {
            rejected++;
        }
        free(h);
    }
    fclose(f);
    printf("accepted %lu rejected %lu\n", ok, rejected);
    return ok && rejected ? 0 : 5;
}
