/*
 * A plain C99 caller of the library's C ABI (no CUDA or C++ headers): checks
 * that include/adapld.h compiles as C and that the host-side entry points
 * answer as declared.  Every call here fails argument validation or needs no
 * device, so the program runs without a GPU.
 */
#include <stdio.h>
#include <string.h>

#include "adapld.h"

static int failures = 0;

static void expect(int got, int want, const char *what) {
    if (got != want) {
        fprintf(stderr, "%s: got %d, want %d\n", what, got, want);
        ++failures;
    }
}

int main(void) {
    adapld_params p;
    memset(&p, 0, sizeof p);
    p.n_max = 5;
    p.k = 32;
    p.branch_width = 4;
    p.draft_len = 16;
    p.succ_len = 1;
    p.tau = 0.1f;
    expect(adapld_tree_nodes(&p), 1 + 16 + 4 * 2, "adapld_tree_nodes");
    expect(adapld_workspace_bytes(8, 131072, 8192, &p) > 0, 1, "adapld_workspace_bytes");
    expect((int)adapld_workspace_bytes(0, 16, 8, &p), 0, "adapld_workspace_bytes(B=0)");
    expect(strcmp(adapld_status_string(ADAPLD_OK), "unknown status") != 0, 1, "status OK");
    expect(strcmp(adapld_status_string(-999), "unknown status"), 0, "status unknown");

    /* argument errors, reported before anything is enqueued */
    int32_t dummy[4];
    expect(adapld_lexical_match(NULL, 64, dummy, 2, 3, 8, dummy, dummy, dummy, dummy, dummy,
                                1 << 20, NULL),
           ADAPLD_ERR_NULL, "lexical null tokens");
    expect(adapld_lexical_match(dummy, 64, dummy, 0, 3, 8, dummy, dummy, dummy, dummy, dummy,
                                1 << 20, NULL),
           ADAPLD_ERR_BATCH, "lexical B=0");
    expect(adapld_accept_greedy(NULL, 64, dummy, dummy, dummy, 1, 4, dummy, dummy, dummy, NULL, 0,
                                NULL, NULL, NULL, 0, NULL, NULL, dummy, 1 << 20, NULL),
           ADAPLD_ERR_NULL, "accept null logits");
    p.k = 0;
    expect(adapld_step(dummy, 64, dummy, (const uint16_t *)dummy, 16, (const uint16_t *)dummy,
                       NULL, 0, 2, &p, NULL, dummy, 1 << 20, NULL),
           ADAPLD_ERR_NULL, "step null outputs");
    if (failures == 0) printf("c-abi ok\n");
    return failures == 0 ? 0 : 1;
}
