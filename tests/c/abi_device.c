/* A C99 client of include/acrl.h on the GPU: device buffers from the CUDA
 * runtime, one acrl_token_stats call on three rows of an odd-width
 * vocabulary (ld > V), the flags word read back with acrl_read_flags, and the
 * results compared with a double-precision log-softmax written here.  The
 * logits are multiples of 1/8, exact in bf16.  Prints "ok". */
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <cuda_runtime.h>

#include "acrl.h"

enum { T = 3, V = 37, LD = 40 };

static acrl_bf16 to_bf16(float x) { /* exact for the values used here */
    uint32_t u;
    memcpy(&u, &x, sizeof u);
    return (acrl_bf16)(u >> 16);
}

int main(void) {
    static float z[T][V];
    static acrl_bf16 h_logits[T * LD];
    int32_t h_ids[T] = {0, 17, 36};
    float h_lse[T], h_logp[T], h_ent[T];
    acrl_bf16* d_logits = NULL;
    int32_t *d_ids = NULL, *d_flags = NULL, flags = -1;
    float *d_lse = NULL, *d_logp = NULL, *d_ent = NULL;
    int t, j, fails = 0;

    memset(h_logits, 0, sizeof h_logits);
    for (t = 0; t < T; ++t)
        for (j = 0; j < V; ++j) {
            z[t][j] = (float)(((t + 3) * (j + 5)) % 29 - 14) / 8.0f;
            h_logits[t * LD + j] = to_bf16(z[t][j]);
        }
    if (cudaMalloc((void**)&d_logits, sizeof h_logits) != cudaSuccess ||
        cudaMalloc((void**)&d_ids, sizeof h_ids) != cudaSuccess ||
        cudaMalloc((void**)&d_flags, sizeof flags) != cudaSuccess ||
        cudaMalloc((void**)&d_lse, sizeof h_lse) != cudaSuccess ||
        cudaMalloc((void**)&d_logp, sizeof h_logp) != cudaSuccess ||
        cudaMalloc((void**)&d_ent, sizeof h_ent) != cudaSuccess) {
        fprintf(stderr, "cudaMalloc failed\n");
        return 2;
    }
    cudaMemcpy(d_logits, h_logits, sizeof h_logits, cudaMemcpyHostToDevice);
    cudaMemcpy(d_ids, h_ids, sizeof h_ids, cudaMemcpyHostToDevice);
    cudaMemset(d_flags, 0, sizeof flags);
    if (acrl_token_stats(d_logits, T, V, LD, d_ids, NULL, d_lse, d_logp, d_ent, d_flags, NULL) != ACRL_OK) {
        fprintf(stderr, "acrl_token_stats failed\n");
        return 1;
    }
    if (acrl_check_flags(d_flags, NULL) != ACRL_OK || acrl_read_flags(d_flags, &flags, NULL) != ACRL_OK || flags != 0) {
        fprintf(stderr, "flags %d\n", flags);
        return 1;
    }
    cudaMemcpy(h_lse, d_lse, sizeof h_lse, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_logp, d_logp, sizeof h_logp, cudaMemcpyDeviceToHost);
    cudaMemcpy(h_ent, d_ent, sizeof h_ent, cudaMemcpyDeviceToHost);
    for (t = 0; t < T; ++t) {
        double m = z[t][0], s = 0.0, sz = 0.0, lse, H;
        for (j = 1; j < V; ++j) m = z[t][j] > m ? z[t][j] : m;
        for (j = 0; j < V; ++j) {
            const double e = exp((double)z[t][j] - m);
            s += e;
            sz += e * z[t][j];
        }
        lse = m + log(s);
        H = lse - sz / s;
        if (fabs(h_lse[t] - lse) > 1e-5 || fabs(h_logp[t] - (z[t][h_ids[t]] - lse)) > 1e-5 ||
            fabs(h_ent[t] - H) > 1e-5 * (1.0 + H)) {
            fprintf(stderr, "row %d: lse %.7f/%.7f logp %.7f/%.7f H %.7f/%.7f\n", t, h_lse[t], lse, h_logp[t],
                    z[t][h_ids[t]] - lse, h_ent[t], H);
            ++fails;
        }
    }
    cudaFree(d_logits);
    cudaFree(d_ids);
    cudaFree(d_flags);
    cudaFree(d_lse);
    cudaFree(d_logp);
    cudaFree(d_ent);
    if (fails) return 1;
    printf("ok\n");
    return 0;
}
