/* A C99 client of include/acrl.h that runs the whole on-policy pass on the
 * GPU through the C ABI alone: token statistics, discrepancy statistics, GRPO
 * advantages, the controller and the loss gradient, for one prompt with two
 * responses (3 and 3 rows, the last row masked).  The rollout log-probs are
 * the policy's own (mu = pi), so every log-ratio and distance is 0 and every
 * ACRL weight is 1; the advantages of rewards (1, 0) are +-0.5 / (sqrt(0.5) +
 * adv_eps), the loss coefficients A_i / (Q G n_i), and the gradient
 * coef (p - onehot), all checked against double-precision values computed
 * here; the controller state is saved to the host and restored.  Prints
 * "ok". */
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <cuda_runtime.h>

#include "acrl.h"

enum { T = 6, V = 21, LD = 24, S = 2, GN = 1 };

static acrl_bf16 to_bf16(float x) { /* exact for the values used here */
    uint32_t u;
    memcpy(&u, &x, sizeof u);
    return (acrl_bf16)(u >> 16);
}

static double from_bf16(acrl_bf16 h) {
    const uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

#define CHECK(call)                                                          \
    do {                                                                     \
        const acrl_status st_ = (call);                                      \
        if (st_ != ACRL_OK) {                                                \
            fprintf(stderr, "%s: %s\n", #call, acrl_status_string(st_));     \
            return 1;                                                        \
        }                                                                    \
    } while (0)

static int close_to(double got, double want, double rel, double abs_tol) {
    return fabs(got - want) <= rel * fabs(want) + abs_tol;
}

int main(void) {
    static float z[T][V];
    static acrl_bf16 h_logits[T * LD], h_grad[T * LD];
    const int32_t h_ids[T] = {0, 7, 20, 3, 11, 5};
    const uint8_t h_mask[T] = {1, 1, 1, 1, 1, 0};
    const int64_t h_so[S + 1] = {0, 3, 6};
    const int32_t h_go[GN + 1] = {0, 2};
    const float h_R[S] = {1.0f, 0.0f};
    float h_lse[T], h_coef[T], h_w[T], h_tl[T], h_adv[S], h_loss = 0.0f;
    acrl_seq_stats h_seq[S];
    acrl_batch_stats h_batch;
    acrl_params p;
    void *d_logits, *d_grad, *d_ids, *d_mask, *d_so, *d_go, *d_R, *d_lse, *d_logp, *d_ent, *d_mu, *d_lr, *d_d;
    void *d_seq, *d_grp, *d_batch, *d_state, *d_adv, *d_w, *d_coef, *d_alpha, *d_tl, *d_loss, *d_flags;
    void** bufs[] = {&d_logits, &d_grad, &d_ids, &d_mask, &d_so, &d_go, &d_R, &d_lse, &d_logp, &d_ent, &d_mu,
                     &d_lr, &d_d, &d_seq, &d_grp, &d_batch, &d_state, &d_adv, &d_w, &d_coef, &d_alpha, &d_tl,
                     &d_loss, &d_flags};
    const size_t sizes[] = {sizeof h_logits, sizeof h_grad, sizeof h_ids, sizeof h_mask, sizeof h_so, sizeof h_go,
                            sizeof h_R, T * 4, T * 4, T * 4, T * 4, T * 4, T * 4, sizeof h_seq,
                            GN * sizeof(acrl_group_stats), sizeof h_batch, sizeof(acrl_controller_state), S * 4,
                            T * 4, T * 4, S * 4, T * 4, 4, 4};
    const size_t nbuf = sizeof sizes / sizeof sizes[0];
    const double A0 = 0.5 / (sqrt(0.5) + 1e-6);
    size_t b;
    int t, j, fails = 0;

    memset(h_logits, 0, sizeof h_logits);
    for (t = 0; t < T; ++t)
        for (j = 0; j < V; ++j) {
            z[t][j] = (float)(((t + 2) * (j + 3)) % 23 - 11) / 8.0f;
            h_logits[t * LD + j] = to_bf16(z[t][j]);
        }
    for (b = 0; b < nbuf; ++b)
        if (cudaMalloc(bufs[b], sizes[b]) != cudaSuccess) {
            fprintf(stderr, "cudaMalloc failed\n");
            return 2;
        }
    cudaMemcpy(d_logits, h_logits, sizeof h_logits, cudaMemcpyHostToDevice);
    cudaMemcpy(d_ids, h_ids, sizeof h_ids, cudaMemcpyHostToDevice);
    cudaMemcpy(d_mask, h_mask, sizeof h_mask, cudaMemcpyHostToDevice);
    cudaMemcpy(d_so, h_so, sizeof h_so, cudaMemcpyHostToDevice);
    cudaMemcpy(d_go, h_go, sizeof h_go, cudaMemcpyHostToDevice);
    cudaMemcpy(d_R, h_R, sizeof h_R, cudaMemcpyHostToDevice);
    cudaMemset(d_flags, 0, 4);
    cudaMemset(d_grad, 0, sizeof h_grad);

    memset(&p, 0, sizeof p);
    p.gamma = 0.65f;
    p.C = 3.0f;
    p.clip_eps = 0.2f;
    p.adv_eps = 1e-6f;
    p.kappa = 1.0f;
    p.mode = ACRL_MODE_ACRL;
    p.y_gran = ACRL_Y_GROUP;
    p.agg = ACRL_AGG_SEQ_MEAN_TOKEN_MEAN;
    p.adv_ddof = 1;
    p.singleton_rule = ACRL_SINGLETON_MEAN0_STD1;
    p.calib_steps = 1;
    p.X_init = 0.013; /* the 3B setting's X (Sec. 5.1) */

    CHECK(acrl_token_stats(d_logits, T, V, LD, d_ids, d_mask, d_lse, d_logp, d_ent, d_flags, NULL));
    cudaMemcpy(d_mu, d_logp, T * 4, cudaMemcpyDeviceToDevice); /* mu = pi */
    CHECK(acrl_seq_discrepancy(d_logp, d_mu, d_mask, T, d_so, S, d_go, GN, d_ent, d_lr, d_d, d_seq, d_grp, d_batch,
                               d_flags, NULL));
    CHECK(acrl_grpo_advantage(d_R, d_go, GN, S, &p, d_adv, d_flags, NULL));
    CHECK(acrl_controller_init(d_state, &p, NULL));
    CHECK(acrl_controller_step(d_state, &p, d_lr, d_mask, T, d_so, S, d_go, GN, d_seq, d_grp, d_batch, d_adv, d_w,
                               d_coef, d_alpha, NULL, d_flags, NULL));
    CHECK(acrl_loss_grad_logits(d_logits, T, V, LD, d_ids, d_mask, d_lse, NULL, d_coef, NULL, NULL, p.clip_eps, d_grad,
                                d_tl, d_loss, d_flags, NULL));
    CHECK(acrl_check_flags(d_flags, NULL));
    {   /* checkpoint the controller and restore it into a fresh device state */
        acrl_controller_state saved, again;
        void* d_state2 = NULL;
        CHECK(acrl_controller_save(d_state, &saved, NULL));
        if (cudaMalloc(&d_state2, sizeof saved) != cudaSuccess) return 2;
        CHECK(acrl_controller_load(d_state2, &saved, NULL));
        CHECK(acrl_controller_save(d_state2, &again, NULL));
        cudaFree(d_state2);
        if (saved.X != 0.013 || saved.calibrated != 1 || saved.step != 1 || memcmp(&saved, &again, sizeof saved)) {
            fprintf(stderr, "controller checkpoint off\n");
            return 1;
        }
    }

    cudaMemcpy(h_lse, d_lse, sizeof h_lse, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_coef, d_coef, sizeof h_coef, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_w, d_w, sizeof h_w, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_tl, d_tl, sizeof h_tl, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_adv, d_adv, sizeof h_adv, cudaMemcpyDeviceToHost);
    cudaMemcpy(&h_loss, d_loss, 4, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_seq, d_seq, sizeof h_seq, cudaMemcpyDeviceToHost);
    cudaMemcpy(&h_batch, d_batch, sizeof h_batch, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_grad, d_grad, sizeof h_grad, cudaMemcpyDeviceToHost);

    if (h_seq[0].n != 3 || h_seq[1].n != 2 || h_batch.n_tokens != 5 || h_batch.n_groups_valid != 1 ||
        h_batch.d_max != 0.0 || h_batch.X != 0.013) {
        fprintf(stderr, "counts or statistics off\n");
        ++fails;
    }
    if (!close_to(h_adv[0], A0, 1e-6, 0.0) || !close_to(h_adv[1], -A0, 1e-6, 0.0)) {
        fprintf(stderr, "adv %.8f %.8f, want +-%.8f\n", h_adv[0], h_adv[1], A0);
        ++fails;
    }
    {
        double loss = 0.0;
        for (t = 0; t < T; ++t) {
            const int i = t < 3 ? 0 : 1;
            const double coef = h_mask[t] ? (i == 0 ? A0 : -A0) / (1.0 * 2.0 * h_seq[i].n) : 0.0;
            double m = z[t][0], s = 0.0;
            if (h_w[t] != (h_mask[t] ? 1.0f : 0.0f) || !close_to(h_coef[t], coef, 1e-6, 0.0) ||
                !close_to(h_tl[t], -coef, 1e-6, 0.0)) {
                fprintf(stderr, "row %d: w %g coef %.8f/%.8f token loss %.8f\n", t, h_w[t], h_coef[t], coef, h_tl[t]);
                ++fails;
            }
            loss += -coef;
            for (j = 1; j < V; ++j) m = z[t][j] > m ? z[t][j] : m;
            for (j = 0; j < V; ++j) s += exp((double)z[t][j] - m);
            for (j = 0; j < V; ++j) {
                const double pj = exp((double)z[t][j] - m) / s;
                const double want = coef * (pj - (j == h_ids[t] ? 1.0 : 0.0));
                const double got = from_bf16(h_grad[t * LD + j]);
                if (!close_to(got, want, 1e-2, 1e-6 * fabs(coef))) {
                    fprintf(stderr, "grad[%d][%d] %.8g, want %.8g\n", t, j, got, want);
                    ++fails;
                }
            }
            if (h_mask[t] && !close_to(h_lse[t], m + log(s), 0.0, 1e-5)) {
                fprintf(stderr, "lse[%d] %.7f, want %.7f\n", t, h_lse[t], m + log(s));
                ++fails;
            }
        }
        if (!close_to(h_loss, loss, 1e-5, 1e-7)) {
            fprintf(stderr, "loss %.8f, want %.8f\n", h_loss, loss);
            ++fails;
        }
    }
    for (b = 0; b < nbuf; ++b) cudaFree(*bufs[b]);
    if (fails) return 1;
    printf("ok\n");
    return 0;
}
