/*
 * A plain C99 caller of the C ABI (include/frac.h), compiled and run by tests/test_abi.py on
 * the CPU: it includes the header as C, links against libfrac.so, and checks the calls that
 * need no GPU (workspace queries, status strings, argument rejection before anything is
 * enqueued).  Prints "ok" and exits 0 when every check holds; otherwise names the first
 * failure and exits 1.
 */
#include <stdio.h>
#include <string.h>

#include "frac.h"

static int fails = 0;

#define CHECK(cond)                                                            \
    do {                                                                       \
        if (!(cond)) {                                                         \
            fprintf(stderr, "abi_check: %s (line %d)\n", #cond, __LINE__);     \
            ++fails;                                                           \
        }                                                                      \
    } while (0)

static frac_dims dims_of(int64_t b, int64_t l, int64_t h, int64_t p, int64_t g, int64_t n,
                         int64_t k, int32_t dtype) {
    frac_dims d;
    memset(&d, 0, sizeof d);
    d.batch = b;
    d.seqlen = l;
    d.nheads = h;
    d.headdim = p;
    d.ngroups = g;
    d.dstate = n;
    d.nmodes = k;
    d.chunk = 0;
    d.dtype = dtype;
    d.flags = 0;
    return d;
}

int main(void) {
    /* every status has a readable name */
    const frac_status all[] = {FRAC_OK, FRAC_ERR_INVALID_ARGUMENT, FRAC_ERR_UNSUPPORTED,
                               FRAC_ERR_CUDA, FRAC_ERR_TIMEOUT};
    for (size_t i = 0; i < sizeof all / sizeof all[0]; ++i) {
        const char *s = frac_status_string(all[i]);
        CHECK(s != NULL && s[0] != '\0');
    }

    /* workspace queries: positive, whole 256-byte units, larger for a longer sequence */
    frac_dims d = dims_of(2, 300, 4, 64, 1, 128, 8, FRAC_DTYPE_BF16);
    size_t fwd = 0, bwd = 0, fwd_long = 0;
    CHECK(frac_scan_fwd_workspace_size(&d, &fwd) == FRAC_OK);
    CHECK(frac_scan_bwd_workspace_size(&d, &bwd) == FRAC_OK);
    CHECK(fwd > 0 && fwd % 256 == 0);
    CHECK(bwd >= fwd && bwd % 256 == 0);
    frac_dims dl = d;
    dl.seqlen = 3000;
    CHECK(frac_scan_fwd_workspace_size(&dl, &fwd_long) == FRAC_OK);
    CHECK(fwd_long > fwd);

    /* rejected before anything is enqueued, with a reason for this thread */
    size_t dummy = 0;
    CHECK(frac_scan_fwd_workspace_size(NULL, &dummy) == FRAC_ERR_INVALID_ARGUMENT);
    frac_dims bad = d;
    bad.nmodes = 0;
    CHECK(frac_scan_fwd_workspace_size(&bad, &dummy) == FRAC_ERR_INVALID_ARGUMENT);
    CHECK(strlen(frac_last_error()) > 0);
    bad = d;
    bad.nheads = 6;
    bad.ngroups = 4; /* H % G != 0 */
    CHECK(frac_scan_bwd_workspace_size(&bad, &dummy) == FRAC_ERR_INVALID_ARGUMENT);

    /* a forward with a NULL input and a decode step without a state are refused */
    float f = 0.f;
    void *p = &f; /* never dereferenced: validation fails first */
    CHECK(frac_scan_fwd(&d, NULL, &f, &f, &f, &f, p, p, p, p, &f, NULL, p, NULL, p, fwd, NULL) ==
          FRAC_ERR_INVALID_ARGUMENT);
    CHECK(frac_decode_step(&d, p, &f, &f, &f, &f, p, p, p, p, &f, NULL, p, NULL) ==
          FRAC_ERR_INVALID_ARGUMENT);

    if (fails) return 1;
    printf("ok\n");
    return 0;
}
