/* A plain C99 caller of the VBQ library: the header must compile as C and the
 * library must answer host-side argument errors without touching a GPU.
 * Prints one line per check and exits 0 when every check holds. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "vbq.h"

static int failures = 0;

static void expect(const char* what, vbq_status_t got, vbq_status_t want) {
    const int ok = got == want;
    printf("%s %s: %s (%s)\n", ok ? "ok" : "FAIL", what, vbq_status_string(got), vbq_last_error());
    if (!ok) ++failures;
}

int main(void) {
    static uint8_t buf[256] __attribute__((aligned(16)));
    vbq_layout* layout = (vbq_layout*)buf;          /* never dereferenced: the calls below fail first */
    vbq_chain* chain = NULL;
    expect("status string", strcmp(vbq_status_string(VBQ_ERR_SHAPE), "VBQ_ERR_SHAPE") == 0 ? VBQ_OK : VBQ_ERR_ARG,
           VBQ_OK);
    expect("pack: out NULL", vbq_pack(buf, buf, (const uint16_t*)buf, 1, 64, 0, NULL, NULL), VBQ_ERR_ARG);
    expect("pack: K not a multiple of 64", vbq_pack(buf, buf, (const uint16_t*)buf, 4, 65, 0, NULL, &layout),
           VBQ_ERR_SHAPE);
    expect("pack: output cleared on error", layout == NULL ? VBQ_OK : VBQ_ERR_ARG, VBQ_OK);
    expect("gemv: NULL layout", vbq_gemv(NULL, (const uint16_t*)buf, (float*)buf, NULL), VBQ_ERR_ARG);
    expect("quantize: K not a multiple of 64",
           vbq_quantize((const float*)buf, buf, 2, 96, buf, (uint16_t*)buf, NULL), VBQ_ERR_SHAPE);
    expect("soft_quant: tau 0", vbq_soft_quant((const float*)buf, (const float*)buf, NULL, 0.0f, 1, 64,
                                               (float*)buf, NULL, NULL, NULL), VBQ_ERR_ARG);
    expect("soft_quant: tau NaN", vbq_soft_quant((const float*)buf, (const float*)buf, NULL, NAN, 1, 64,
                                                 (float*)buf, NULL, NULL, NULL), VBQ_ERR_ARG);
    expect("chain: empty", vbq_chain_create(NULL, NULL, NULL, NULL, 0, &chain), VBQ_ERR_ARG);
    expect("chain: free NULL", vbq_chain_free(NULL), VBQ_OK);
    expect("free NULL", vbq_free(NULL), VBQ_OK);
    expect("self-test: bad limit", vbq_selftest_timeout(0, NULL), VBQ_ERR_ARG);
    printf("%s\n", failures ? "FAILED" : "ALL OK");
    return failures ? 1 : 0;
}
