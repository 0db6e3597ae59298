/* A C99 client of the host-buffer pipeline: one prompt of two responses in
 * page-locked host memory (cudaHostAlloc), two overlapping steps through
 * acrl_host_pipeline_step, and the same two steps through the device calls
 * on device copies of the inputs; the gradients and losses must agree bit
 * for bit and the two controller states byte for byte.  Prints "ok". */
#include <stdio.h>
#include <string.h>

#include <cuda_runtime.h>

#include "acrl.h"

enum { T = 9, V = 37, LD = 40, S = 2, GN = 1, CHUNKS = 3 };

#define CHECK(call)                                                          \
    do {                                                                     \
        const acrl_status st_ = (call);                                      \
        if (st_ != ACRL_OK) {                                                \
            fprintf(stderr, "%s: %s\n", #call, acrl_status_string(st_));     \
            return 1;                                                        \
        }                                                                    \
    } while (0)

static acrl_bf16 to_bf16(float x) { /* exact for the values used here */
    uint32_t u;
    memcpy(&u, &x, sizeof u);
    return (acrl_bf16)(u >> 16);
}

static void* host(size_t n) {
    void* p = NULL;
    return cudaHostAlloc(&p, n, cudaHostAllocDefault) == cudaSuccess ? p : NULL;
}

static void* dev(size_t n) {
    void* p = NULL;
    return cudaMalloc(&p, n) == cudaSuccess ? p : NULL;
}

int main(void) {
    const int32_t ids[T] = {0, 7, 36, 3, 11, 5, 20, 21, 2};
    const uint8_t mask[T] = {1, 1, 1, 1, 1, 1, 1, 1, 0};
    const int64_t so[S + 1] = {0, 4, 9};
    const int32_t go[GN + 1] = {0, 2};
    const float rewards[S] = {1.0f, 0.0f};
    acrl_bf16 *h_logits = host(T * LD * 2), *h_grad[2] = {host(T * LD * 2), host(T * LD * 2)};
    int32_t* h_ids = host(sizeof ids);
    uint8_t* h_mask = host(sizeof mask);
    float *h_mu = host(T * 4), *h_rewards = host(sizeof rewards), *h_loss = host(2 * 4);
    int64_t* h_so = host(sizeof so);
    int32_t* h_go = host(sizeof go);
    acrl_bf16 *d_logits = dev(T * LD * 2), *d_grad = dev(T * LD * 2);
    int32_t *d_ids = dev(sizeof ids), *d_go = dev(sizeof go), *d_flags = dev(4), *d_flags2 = dev(4);
    uint8_t* d_mask = dev(sizeof mask);
    int64_t* d_so = dev(sizeof so);
    float *d_mu = dev(T * 4), *d_rewards = dev(sizeof rewards), *d_lse = dev(T * 4), *d_logp = dev(T * 4);
    float *d_ent = dev(T * 4), *d_lr = dev(T * 4), *d_d = dev(T * 4), *d_w = dev(T * 4), *d_coef = dev(T * 4);
    float *d_adv = dev(S * 4), *d_alpha = dev(S * 4), *d_tl = dev(T * 4), *d_loss = dev(4);
    acrl_seq_stats* d_seq = dev(S * sizeof(acrl_seq_stats));
    acrl_group_stats* d_grp = dev(GN * sizeof(acrl_group_stats));
    acrl_batch_stats* d_batch = dev(sizeof(acrl_batch_stats));
    acrl_controller_state *d_state = dev(sizeof(acrl_controller_state)), *d_state2 = dev(sizeof(acrl_controller_state));
    acrl_controller_state s1, s2;
    acrl_host_pipeline* pl = NULL;
    acrl_params p;
    void* ws;
    int64_t ws_bytes;
    static acrl_bf16 ref_grad[T * LD];
    float ref_loss;
    int t, j, k;

    if (!h_logits || !h_grad[0] || !h_grad[1] || !h_loss || !d_logits || !d_state2) {
        fprintf(stderr, "allocation failed\n");
        return 2;
    }
    for (t = 0; t < T; ++t)
        for (j = 0; j < LD; ++j)
            h_logits[t * LD + j] = to_bf16(j < V ? (float)(((t + 5) * (j + 2)) % 19 - 9) / 4.0f : 0.0f);
    memcpy(h_ids, ids, sizeof ids);
    memcpy(h_mask, mask, sizeof mask);
    memcpy(h_so, so, sizeof so);
    memcpy(h_go, go, sizeof go);
    memcpy(h_rewards, rewards, sizeof rewards);
    for (t = 0; t < T; ++t) h_mu[t] = -3.0f - 0.125f * (float)(t % 5); /* rollout log-probs */
    cudaMemcpy(d_logits, h_logits, T * LD * 2, cudaMemcpyHostToDevice);
    cudaMemcpy(d_ids, ids, sizeof ids, cudaMemcpyHostToDevice);
    cudaMemcpy(d_mask, mask, sizeof mask, cudaMemcpyHostToDevice);
    cudaMemcpy(d_so, so, sizeof so, cudaMemcpyHostToDevice);
    cudaMemcpy(d_go, go, sizeof go, cudaMemcpyHostToDevice);
    cudaMemcpy(d_rewards, rewards, sizeof rewards, cudaMemcpyHostToDevice);
    cudaMemcpy(d_mu, h_mu, T * 4, cudaMemcpyHostToDevice);
    cudaMemset(d_flags, 0, 4);
    cudaMemset(d_flags2, 0, 4);

    memset(&p, 0, sizeof p);
    p.gamma = 0.65f;
    p.C = 3.0f;
    p.clip_eps = 0.2f;
    p.adv_eps = 1e-6f;
    p.kappa = 1.0f;
    p.mode = ACRL_MODE_ACRL;
    p.adv_ddof = 1;
    p.calib_steps = 1;
    p.X_init = 0.0; /* calibrate on the first step */

    ws_bytes = acrl_host_pipeline_workspace_bytes(T, LD, S, GN, CHUNKS);
    ws = dev((size_t)ws_bytes);
    if (ws_bytes <= 0 || !ws) return 2;
    CHECK(acrl_host_pipeline_create(&pl, T, V, LD, S, GN, CHUNKS, ws, ws_bytes));
    CHECK(acrl_controller_init(d_state, &p, NULL));
    CHECK(acrl_controller_init(d_state2, &p, NULL));
    for (k = 0; k < 2; ++k) /* two steps enqueued back to back */
        CHECK(acrl_host_pipeline_step(pl, &p, d_state, h_logits, h_ids, h_mask, h_mu, h_rewards, h_so, h_go,
                                      h_grad[k], h_loss + k, d_flags, NULL));
    if (cudaDeviceSynchronize() != cudaSuccess) return 1;

    for (k = 0; k < 2; ++k) {
        CHECK(acrl_token_stats(d_logits, T, V, LD, d_ids, d_mask, d_lse, d_logp, d_ent, d_flags2, NULL));
        CHECK(acrl_seq_discrepancy(d_logp, d_mu, d_mask, T, d_so, S, d_go, GN, d_ent, d_lr, d_d, d_seq, d_grp,
                                   d_batch, d_flags2, NULL));
        CHECK(acrl_grpo_advantage(d_rewards, d_go, GN, S, &p, d_adv, d_flags2, NULL));
        CHECK(acrl_controller_step(d_state2, &p, d_lr, d_mask, T, d_so, S, d_go, GN, d_seq, d_grp, d_batch, d_adv,
                                   d_w, d_coef, d_alpha, NULL, d_flags2, NULL));
        CHECK(acrl_loss_grad_logits(d_logits, T, V, LD, d_ids, d_mask, d_lse, NULL, d_coef, NULL, NULL, p.clip_eps,
                                    d_grad, d_tl, d_loss, d_flags2, NULL));
        cudaMemcpy(ref_grad, d_grad, sizeof ref_grad, cudaMemcpyDeviceToHost);
        cudaMemcpy(&ref_loss, d_loss, 4, cudaMemcpyDeviceToHost);
        for (t = 0; t < T; ++t)
            if (memcmp(h_grad[k] + t * LD, ref_grad + t * LD, V * 2) != 0) {
                fprintf(stderr, "step %d: gradient row %d differs\n", k, t);
                return 1;
            }
        if (memcmp(&h_loss[k], &ref_loss, 4) != 0) {
            fprintf(stderr, "step %d: loss %.9g against %.9g\n", k, h_loss[k], ref_loss);
            return 1;
        }
    }
    CHECK(acrl_check_flags(d_flags, NULL));
    CHECK(acrl_controller_save(d_state, &s1, NULL));
    CHECK(acrl_controller_save(d_state2, &s2, NULL));
    if (memcmp(&s1, &s2, sizeof s1) != 0 || s1.calibrated != 1 || s1.step != 2) {
        fprintf(stderr, "controller states differ\n");
        return 1;
    }
    CHECK(acrl_host_pipeline_destroy(pl));
    printf("ok\n");
    return 0;
}
