/* Plain C11 user of the library's headers: checks that include/cm.h and
 * include/cm_testing.h are valid C and that a C program links against libcm.so.
 * Run without a GPU it exercises only argument validation. */
#include <stdio.h>
#include <string.h>

#include "cm.h"
#include "cm_testing.h"

int main(void) {
    if (cm_abi_version() != CM_ABI_VERSION) return 1;
    cm_context *ctx = NULL;
    if (cm_context_create(0, -1.0, -1, 0, &ctx) != CM_ERR_INVALID_ARG) return 2;
    if (strcmp(cm_status_string(CM_ERR_CAPACITY), "CM_ERR_CAPACITY") != 0) return 3;
    cm_fragment f;
    memset(&f, 0, sizeof f);
    cm_id id;
    if (cm_fragment_id_static(&f, -1, NULL, &id, NULL) != CM_ERR_INVALID_ARG) return 4;
    cm_paged_cache pc;
    memset(&pc, 0, sizeof pc);
    if (cm_render_paged(NULL, &pc, NULL, NULL, NULL) != CM_ERR_INVALID_ARG) return 5;
    if (cm_testing_render_withheld_load(NULL, NULL, NULL, 0, NULL) != CM_ERR_INVALID_ARG) return 6;
    /* the calls over several sets: zero items is a no-op, a NULL set is refused */
    if (cm_render_many(NULL, 0, NULL, NULL) != CM_OK) return 7;
    if (cm_ingest_many(NULL, NULL, 0, NULL, NULL, NULL) != CM_OK) return 8;
    cm_render_job job;
    memset(&job, 0, sizeof job);
    if (cm_render_many(&job, 1, NULL, NULL) != CM_ERR_INVALID_ARG) return 9;
    cm_set *no_set = NULL;
    if (cm_ingest_many(&no_set, &f, 1, NULL, NULL, NULL) != CM_ERR_INVALID_ARG) return 10;
    uint8_t present = 0;
    int32_t leq = 0;
    if (cm_set_contains(NULL, &id, 1, &present) != CM_ERR_INVALID_ARG) return 11;
    if (cm_set_leq(NULL, NULL, &leq) != CM_ERR_INVALID_ARG) return 12;
    if (cm_measure_int_alu(0, NULL, NULL) != CM_ERR_INVALID_ARG) return 13;
    if (cm_context_set_render_warps(NULL, 8) != CM_ERR_INVALID_ARG) return 14;
    if (cm_context_set_dedup_by_bytes(NULL, 1) != CM_ERR_INVALID_ARG) return 15;
    printf("ok %s\n", cm_last_error_message());
    return 0;
}
