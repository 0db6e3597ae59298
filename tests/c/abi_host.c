/* A C99 client of include/acrl.h: the calls that need no GPU.  Struct layouts
 * seen by a C compiler match the library's, the version and status strings
 * are exported, and arguments the host can see are wrong are rejected with
 * ACRL_ERR_INVALID_ARG before anything touches the device.  Prints "ok". */
#include <stdio.h>
#include <string.h>

#include "acrl.h"

static int fails = 0;
#define CHECK(c)                                                            \
    do {                                                                    \
        if (!(c)) {                                                         \
            fprintf(stderr, "FAIL %s:%d: %s\n", __FILE__, __LINE__, #c);    \
            ++fails;                                                        \
        }                                                                   \
    } while (0)

int main(void) {
    acrl_params p;
    acrl_controller_state st;
    int32_t ids[4] = {0, 1, 2, 3};
    float out[4];

    CHECK(acrl_abi_version() == ACRL_ABI_VERSION);
    CHECK(acrl_struct_size(0) == (int64_t)sizeof(acrl_params));
    CHECK(acrl_struct_size(1) == (int64_t)sizeof(acrl_controller_state));
    CHECK(acrl_struct_size(2) == (int64_t)sizeof(acrl_seq_stats));
    CHECK(acrl_struct_size(3) == (int64_t)sizeof(acrl_group_stats));
    CHECK(acrl_struct_size(4) == (int64_t)sizeof(acrl_batch_stats));
    CHECK(strcmp(acrl_status_string(ACRL_OK), "ok") == 0);
    CHECK(strlen(acrl_status_string(ACRL_ERR_INVALID_ARG)) > 0);

    /* sizes and strides the host can see */
    CHECK(acrl_token_stats(NULL, -1, 8, 8, ids, NULL, out, out, out, NULL, NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_token_stats(NULL, 4, 0, 8, ids, NULL, out, out, out, NULL, NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_token_stats(NULL, 4, 16, 8, ids, NULL, out, out, out, NULL, NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_token_stats(NULL, 4, 10, 12, ids, NULL, out, out, out, NULL, NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_loss_grad_logits(NULL, -1, 8, 8, ids, NULL, NULL, NULL, out, NULL, NULL, 0.2f, NULL, out, out, NULL,
                                NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_reduce_loss(out, -1, out, NULL) == ACRL_ERR_INVALID_ARG);
    CHECK(acrl_check_flags(NULL, NULL) == ACRL_ERR_INVALID_ARG);

    /* hyper-parameters out of range */
    memset(&p, 0, sizeof p);
    p.gamma = 0.65f;
    p.C = 3.0f;
    p.clip_eps = 0.2f;
    p.adv_eps = 1e-6f;
    p.kappa = 1.0f;
    p.mode = ACRL_MODE_ACRL;
    p.adv_ddof = 1;
    p.calib_steps = 1;
    CHECK(acrl_controller_init(NULL, &p, NULL) == ACRL_ERR_INVALID_ARG);
    p.kappa = 0.0f;
    CHECK(acrl_controller_init(&st, &p, NULL) == ACRL_ERR_INVALID_ARG);

    /* workspace size of the LM-head path: one 16-byte state per (row, 256-column tile) */
    CHECK(acrl_lmhead_workspace_bytes(4, 300) == 2 * 4 * 16);
    CHECK(acrl_lmhead_workspace_bytes(-1, 300) == -1);

    if (fails) return 1;
    printf("ok\n");
    return 0;
}
