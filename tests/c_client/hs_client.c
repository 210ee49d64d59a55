/* A plain C11 client of libhs: the public headers compile as C, and the host-only
 * calls (version, status strings, strict-prefix alignment, checkpoint counts, argument
 * checks that return before any CUDA call) link and behave from C.  Prints one line per
 * check and exits non-zero on the first mismatch. */
#include <stdio.h>
#include <string.h>

#include "hs.h"
#include "hs_test.h"

static int fails = 0;

static void check(int ok, const char *what)
{
    printf("%s %s\n", ok ? "ok" : "FAIL", what);
    if (!ok)
        ++fails;
}

int main(void)
{
    check(hs_version() >= 100, "hs_version");
    check(strncmp(hs_status_string(HS_ERR_MISALIGNED), "HS_", 3) == 0, "hs_status_string");

    /* Table 4 of the paper at C = 1792: a complete hit of 3584 tokens credits 1792,
     * never the whole prompt; one of 3585 tokens credits 3584 */
    const int64_t avail[] = {1792, 3584, 5376};
    int64_t c = -1, pages = -1, tail = -1;
    check(hs_align_prefix(3584, 3584, avail, 3, 16, &c, &pages, &tail) == HS_OK && c == 1792 &&
              pages == 112 && tail == 1792,
          "align 3584 -> 1792");
    check(hs_align_prefix(3585, 3585, avail, 3, 16, &c, &pages, &tail) == HS_OK && c == 3584 &&
              tail == 1,
          "align 3585 -> 3584");
    check(hs_align_prefix(10, 11, avail, 3, 16, &c, &pages, &tail) == HS_ERR_INVALID_ARG,
          "align hit > N rejected");

    /* checkpoints at the multiples of 256 in (pos0, pos0 + n] */
    const int64_t pos0[] = {768, 0};
    const int32_t n[] = {532, 255};
    int64_t total = -1;
    check(hs_linattn_num_checkpoints(2, pos0, n, 256, &total) == HS_OK && total == 2,
          "checkpoint count");

    /* argument errors come back before any CUDA call */
    check(hs_restore_kv_pages(NULL, NULL, 1, NULL, 4, 4096, 16, NULL, 0) == HS_ERR_INVALID_ARG,
          "restore_kv_pages NULL arrays");
    hs_linattn_shape shp = {1, 2, 96, 96, 8, HS_LINATTN_AUTO, 0};
    check(hs_linattn_prefill_from_state(&shp, NULL, NULL, NULL, NULL, NULL, NULL, pos0, n, 0,
                                        NULL, NULL, 0) == HS_ERR_UNSUPPORTED,
          "prefill d = 96 unsupported");
    shp.d_k = shp.d_v = 128;
    check(hs_test_prefill_stalled(&shp, NULL, NULL, NULL, NULL, NULL, NULL, pos0, n, 0, NULL,
                                  NULL, 0) == HS_ERR_UNSUPPORTED,
          "stall hook needs the tensor-core kernel");

    /* the segment-parallel prefill: its workspace, and the allocation-free variant's limit */
    hs_linattn_shape one = {1, 16, 128, 128, 1024, HS_LINATTN_AUTO, 0};
    const int64_t at[] = {4096};
    const int32_t len[] = {512};
    int64_t ws = -1;
    check(hs_linattn_scan_workspace_bytes(&one, at, len, &ws) == HS_OK &&
              ws == (int64_t)HS_NOALLOC_SCRATCH_BYTES,
          "scan workspace of a 512-token tail of 16 heads = the fixed workspace");
    check(hs_linattn_prefill_scan(&one, NULL, NULL, NULL, NULL, NULL, NULL, at, len, 512, NULL,
                                  NULL, 0, NULL, 0) == HS_ERR_INVALID_ARG,
          "scan prefill without a workspace");
    const int32_t longer[] = {513};
    check(hs_linattn_prefill_scan_noalloc(&one, NULL, NULL, NULL, NULL, NULL, NULL, at, longer, 512,
                                          NULL, NULL, 0) == HS_ERR_TOO_LARGE &&
              strncmp(hs_status_string(HS_ERR_TOO_LARGE), "HS_ERR_TOO_LARGE", 16) == 0,
          "allocation-free prefill refuses a call beyond its workspace");
    return fails == 0 ? 0 : 1;
}
