// The O(T) part of the path: per-token log-ratio and distance, masked
// per-response / per-prompt / batch aggregates, GRPO advantages and the
// adaptive controller with its importance weights.
//
// One CTA per response does the segmented reductions; single-CTA kernels
// finalise prompts and the batch.  Every reduction has a fixed order (strided
// per-thread partials, then a fixed warp butterfly and warp-order sum) and no
// floating-point atomics, so the results are bit-reproducible.
#include <cmath>

#include "acrl_device.cuh"
#include "acrl_host.h"

namespace acrl {
namespace {

constexpr int kSeqThreads = 256;
constexpr int kFinThreads = 512;

__device__ __forceinline__ bool seq_range(const int64_t* so, int i, int64_t T, int64_t& lo, int64_t& hi) {
    lo = so[i];
    hi = so[i + 1];
    return lo >= 0 && lo <= hi && hi <= T;
}

// Index g with goff[g] <= i < goff[g+1], or -1.
__device__ __forceinline__ int group_of(const int32_t* goff, int Gn, int i) {
    int lo = 0, hi = Gn;  // invariant: answer in [lo, hi)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (goff[mid] <= i) lo = mid; else hi = mid;
    }
    return (Gn > 0 && goff[lo] <= i && i < goff[lo + 1]) ? lo : -1;
}

// |exp(a) - exp(b)| without cancellation when a and b are close.
__device__ __forceinline__ float prob_distance(float a, float b) {
    const float l = a - b;
    return fabsf(l) < 0.5f ? expf(b) * fabsf(expm1f(l)) : fabsf(expf(a) - expf(b));
}

// K2a: per-token lr and d, per-response sums.  One CTA per response.
__global__ void __launch_bounds__(kSeqThreads) seq_stats_kernel(
    const float* __restrict__ logp_pi, const float* __restrict__ logp_mu, const uint8_t* __restrict__ mask,
    int64_t T, const int64_t* __restrict__ so, int S, const int32_t* __restrict__ goff, int Gn,
    const float* __restrict__ entropy, float* __restrict__ lr, float* __restrict__ d, acrl_seq_stats* seq,
    int32_t* flags) {
    constexpr int NW = kSeqThreads / 32;
    __shared__ double sh[NW * 6];
    const int i = blockIdx.x;
    int64_t lo, hi;
    if (!seq_range(so, i, T, lo, hi)) {
        if (threadIdx.x == 0) raise_flag(flags, ACRL_FLAG_BAD_OFFSETS);
        lo = hi = 0;
    }
    int n = 0;
    double sd = 0.0, sd2 = 0.0, slr = 0.0, sH = 0.0;
    float mxd = 0.f;
    bool nan_lr = false;
    for (int64_t t = lo + threadIdx.x; t < hi; t += kSeqThreads) {
        const bool m = mask ? mask[t] != 0 : true;
        float l = 0.f, dd = 0.f;
        if (m) {
            const float a = logp_pi[t], b = logp_mu[t];
            l = a - b;
            nan_lr |= isnan(l);  // a NaN log-prob on either side
            dd = prob_distance(a, b);
            ++n;
            sd += dd;
            sd2 += double(dd) * dd;
            slr += l;
            if (entropy) sH += entropy[t];
            mxd = fmaxf(mxd, dd);
        }
        lr[t] = l;
        d[t] = dd;
    }
    if (nan_lr) raise_flag(flags, ACRL_FLAG_NONFINITE);
    double v[5] = {double(n), sd, sd2, slr, sH}, mx = mxd;
    block_sums_max0<NW, 5>(v, mx, sh);
    n = int(v[0]);
    sd = v[1];
    sd2 = v[2];
    slr = v[3];
    sH = v[4];
    mxd = float(mx);
    if (threadIdx.x == 0) {
        acrl_seq_stats s;
        s.n = n;
        s.group = group_of(goff, Gn, i);
        s.mean_d = n ? float(sd / n) : 0.f;
        s.max_d = mxd;
        s.sum_d = sd;
        s.sum_d2 = sd2;
        s.sum_lr = slr;
        s.sum_H = sH;
        s.sum_w = 0.0;
        s.n_trunc = 0;
        s.alpha = 0.f;
        seq[i] = s;
    }
}

// K2b: prompt statistics and batch statistics; also checks the offsets.
__global__ void __launch_bounds__(kFinThreads) seq_finalize_kernel(
    int64_t T, const int64_t* __restrict__ so, int S, const int32_t* __restrict__ goff, int Gn,
    const acrl_seq_stats* __restrict__ seq, acrl_group_stats* grp, acrl_batch_stats* batch, int32_t* flags) {
    constexpr int NW = kFinThreads / 32;
    __shared__ double sh[NW * 9];
    bool bad = false;
    for (int i = threadIdx.x; i < S; i += kFinThreads) bad |= so[i] > so[i + 1];
    for (int g = threadIdx.x; g < Gn; g += kFinThreads) bad |= goff[g] > goff[g + 1];
    if (threadIdx.x == 0) bad |= so[0] != 0 || so[S] != T || (Gn > 0 ? (goff[0] != 0 || goff[Gn] != S) : S != 0);
    if (bad) raise_flag(flags, ACRL_FLAG_BAD_OFFSETS);

    int qv = 0;
    double ysum = 0.0;
    for (int g = threadIdx.x; g < Gn; g += kFinThreads) {
        int b = goff[g], e = goff[g + 1];
        b = b < 0 ? 0 : (b > S ? S : b);
        e = e < b ? b : (e > S ? S : e);
        int G = 0;
        long long ntok = 0;
        double y = 0.0;
        for (int i = b; i < e; ++i) {
            const int n = seq[i].n;
            ntok += n;
            if (n > 0) {
                ++G;
                y += seq[i].sum_d / n;
            }
        }
        acrl_group_stats gs;
        gs.n_valid_seqs = G;
        gs.n_seqs = e - b;
        gs.n_tokens = ntok;
        gs.Y = G ? y / G : 0.0;
        grp[g] = gs;
        if (G) {
            ++qv;
            ysum += gs.Y;
        }
    }
    long long N = 0;
    int sv = 0;
    double sd = 0.0, sd2 = 0.0, sH = 0.0, slr = 0.0, dmax = 0.0;
    for (int i = threadIdx.x; i < S; i += kFinThreads) {
        const acrl_seq_stats s = seq[i];
        N += s.n;
        sv += s.n > 0;
        sd += s.sum_d;
        sd2 += s.sum_d2;
        sH += s.sum_H;
        slr += s.sum_lr;
        dmax = fmax(dmax, double(s.max_d));
    }
    // counts travel as doubles: exact below 2^53
    double v[8] = {double(qv), ysum, double(N), double(sv), sd, sd2, sH, slr};
    block_sums_max0<NW, 8>(v, dmax, sh);
    qv = int(v[0]);
    ysum = v[1];
    N = (long long)v[2];
    sv = int(v[3]);
    sd = v[4];
    sd2 = v[5];
    sH = v[6];
    slr = v[7];
    if (threadIdx.x == 0) {
        acrl_batch_stats b = *batch;
        b.n_tokens = N;
        b.n_seqs_valid = sv;
        b.n_groups_valid = qv;
        const double inv = N ? 1.0 / double(N) : 0.0;
        b.d_mean = sd * inv;
        b.d_max = dmax;
        const double var = sd2 * inv - b.d_mean * b.d_mean;
        b.d_std = var > 0.0 ? sqrt(var) : 0.0;
        b.Y_sum = ysum;
        b.Y_mean = qv ? ysum / qv : 0.0;
        b.H_mean = sH * inv;
        b.lr_mean = slr * inv;
        b.X = 0.0;
        b.trunc_frac = 0.0;
        b.w_mean = 0.0;
        b.alpha_mean = 0.0;
        *batch = b;
    }
}

// K3: GRPO advantages, one thread per prompt.
__global__ void grpo_kernel(const float* __restrict__ R, const int32_t* __restrict__ goff, int Gn, int S, float adv_eps,
                            int ddof, int singleton_rule, float* __restrict__ adv, int32_t* flags) {
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= Gn) return;
    const int b = goff[g], e = goff[g + 1];
    if (b < 0 || b > e || e > S) {
        raise_flag(flags, ACRL_FLAG_BAD_OFFSETS);
        return;
    }
    const int G = e - b;
    if (G == 0) return;
    if (G == 1) {
        adv[b] = singleton_rule == ACRL_SINGLETON_MEAN0_STD1 ? R[b] : 0.f;
        return;
    }
    double sum = 0.0;
    for (int i = b; i < e; ++i) sum += R[i];
    const double mean = sum / G;
    double ss = 0.0;
    for (int i = b; i < e; ++i) {
        const double c = R[i] - mean;
        ss += c * c;
    }
    const double var = G > ddof ? ss / (G - ddof) : 0.0;
    const double den = sqrt(var) + double(adv_eps);
    for (int i = b; i < e; ++i) {
        const double c = R[i] - mean;
        adv[i] = den > 0.0 ? float(c / den) : 0.f;
    }
}

__global__ void controller_init_kernel(acrl_controller_state* st, double X_init) {
    acrl_controller_state s;
    s.X = X_init > 0.0 ? X_init : 0.0;
    s.calib_sum = 0.0;
    s.calib_count = 0;
    s.step = 0;
    s.calib_done = 0;
    s.calibrated = X_init > 0.0 ? 1 : 0;
    s.flags = 0;
    s.reserved = 0;
    *st = s;
}

// K4a: state update (calibration of X) and alpha per response.
__global__ void __launch_bounds__(kFinThreads) controller_alpha_kernel(
    acrl_controller_state* st, acrl_params p, int S, int Gn, acrl_seq_stats* seq,
    const acrl_group_stats* __restrict__ grp, acrl_batch_stats* batch, const float* __restrict__ adv,
    float* alpha_out, int32_t* flags) {
    __shared__ double sh_X;
    __shared__ int sh_apply;
    if (threadIdx.x == 0) {
        // Y_mean from the (possibly all-reduced across ranks) sum and prompt count
        batch->Y_mean = batch->n_groups_valid > 0 ? batch->Y_sum / double(batch->n_groups_valid) : 0.0;
        acrl_controller_state s = *st;
        const bool was_calibrated = s.calibrated != 0;
        int apply = 1;
        if (!s.calibrated) {
            s.calib_sum += batch->Y_sum;
            s.calib_count += batch->n_groups_valid;
            s.calib_done += 1;
            if (s.calib_done >= p.calib_steps) {
                s.X = s.calib_count > 0 ? s.calib_sum / double(s.calib_count) : 0.0;
                s.calibrated = 1;
            } else {
                apply = 0;
            }
        }
        s.step += 1;
        const bool uses_x = p.mode == ACRL_MODE_ACRL || p.mode == ACRL_MODE_ACRL_FALLBACK;
        if (uses_x && apply && !(s.X > 0.0)) {
            raise_flag(flags, ACRL_FLAG_X_NONPOS);
            s.flags |= ACRL_FLAG_X_NONPOS;
        }
        const double X_use = s.X;
        // moving-average X (off by default): this step uses X_use, the next one the update
        if (was_calibrated && p.x_ema > 0.f) s.X = (1.0 - double(p.x_ema)) * s.X + double(p.x_ema) * batch->Y_mean;
        *st = s;
        batch->X = apply ? X_use : 0.0;
        sh_X = X_use;
        sh_apply = apply;
    }
    __syncthreads();
    const double X = sh_X;
    const bool apply = sh_apply != 0;
    const double Ybatch = batch->Y_mean;  // written by thread 0 above, before the barrier
    for (int i = threadIdx.x; i < S; i += kFinThreads) {
        float a = 0.f;
        const float A = adv[i];
        const float sgnf = A > 0.f ? 1.f : (A < 0.f ? -1.f : 0.f);
        if (p.mode == ACRL_MODE_TIS || p.mode == ACRL_MODE_MIS) {
            a = 1.f;
        } else if (p.mode == ACRL_MODE_ACRL_CONTINUOUS) {
            a = seq[i].n > 0 ? -p.kappa * sgnf : 0.f;
        } else if ((p.mode == ACRL_MODE_ACRL || p.mode == ACRL_MODE_ACRL_FALLBACK) && apply && X > 0.0 &&
                   seq[i].n > 0) {
            double Y;
            if (p.y_gran == ACRL_Y_SEQUENCE) {
                Y = seq[i].sum_d / seq[i].n;
            } else if (p.y_gran == ACRL_Y_BATCH) {
                Y = Ybatch;
            } else {
                const int g = seq[i].group;
                Y = (g >= 0 && g < Gn) ? grp[g].Y : 0.0;
            }
            a = float(double(p.gamma) * double(sgnf) * (1.0 - Y / X));
            if (p.mode == ACRL_MODE_ACRL_FALLBACK && !(Y > X)) a = 0.f;
        }
        seq[i].alpha = a;
        if (alpha_out) alpha_out[i] = a;
    }
}

// K4b: per-token weights and loss coefficients; one CTA per response.
__global__ void __launch_bounds__(kSeqThreads) controller_weights_kernel(
    acrl_params p, const float* __restrict__ lr, const uint8_t* __restrict__ mask, int64_t T,
    const int64_t* __restrict__ so, int Gn, acrl_seq_stats* seq, const acrl_group_stats* __restrict__ grp,
    const acrl_batch_stats* __restrict__ batch, const float* __restrict__ adv, float* __restrict__ weight,
    float* __restrict__ coef, float* __restrict__ ent_coef) {
    constexpr int NW = kSeqThreads / 32;
    __shared__ double sh[NW * 3];
    const int i = blockIdx.x;
    int64_t lo, hi;
    if (!seq_range(so, i, T, lo, hi)) lo = hi = 0;
    const acrl_seq_stats s = seq[i];
    const float logC = logf(p.C);
    double norm;
    if (p.agg == ACRL_AGG_TOKEN_MEAN) {
        norm = double(batch->n_tokens);
    } else {
        const int G = (s.group >= 0 && s.group < Gn) ? grp[s.group].n_valid_seqs : 0;
        norm = double(batch->n_groups_valid) * double(G) * double(s.n);
    }
    const float scale = norm > 0.0 ? float(double(adv[i]) / norm) : 0.f;
    const float escale = norm > 0.0 ? float(double(p.entropy_coeff) / norm) : 0.f;
    const float Si = float(s.sum_lr);
    const bool mis_cut = Si > logC;
    const float w_mis = (mis_cut || isnan(Si)) ? 0.f : expf(Si);
    int nt = 0;
    double sw = 0.0;
    for (int64_t t = lo + threadIdx.x; t < hi; t += kSeqThreads) {
        const bool m = mask ? mask[t] != 0 : true;
        float w = 0.f;
        if (m) {
            if (p.mode == ACRL_MODE_NONE) {
                w = 1.f;
            } else if (p.mode == ACRL_MODE_MIS) {
                w = w_mis;
                nt += mis_cut;
            } else {
                // rho^0 = 1 even where the log-ratio is infinite (mu = 0); a NaN log-ratio gets weight 0
                const float lrho = s.alpha == 0.f ? 0.f : s.alpha * lr[t];
                w = isnan(lrho) ? 0.f : expf(fminf(lrho, logC));
                nt += lrho > logC;
            }
            sw += w;
        }
        weight[t] = w;
        coef[t] = w * scale;
        if (ent_coef) ent_coef[t] = m ? escale : 0.f;
    }
    double v[2] = {double(nt), sw}, unused = 0.0;
    block_sums_max0<NW, 2>(v, unused, sh);
    nt = int(v[0]);
    sw = v[1];
    if (threadIdx.x == 0) {
        seq[i].n_trunc = nt;
        seq[i].sum_w = sw;
    }
}

// K4c: batch metrics of the controller.
__global__ void __launch_bounds__(kFinThreads) controller_finalize_kernel(int S, const acrl_seq_stats* __restrict__ seq,
                                                                          acrl_batch_stats* batch) {
    constexpr int NW = kFinThreads / 32;
    __shared__ double sh[NW * 4];
    long long nt = 0;
    double sw = 0.0, sa = 0.0;
    for (int i = threadIdx.x; i < S; i += kFinThreads) {
        nt += seq[i].n_trunc;
        sw += seq[i].sum_w;
        if (seq[i].n > 0) sa += seq[i].alpha;
    }
    double v[3] = {double(nt), sw, sa}, unused = 0.0;
    block_sums_max0<NW, 3>(v, unused, sh);
    nt = (long long)v[0];
    sw = v[1];
    sa = v[2];
    if (threadIdx.x == 0) {
        const double N = double(batch->n_tokens);
        batch->trunc_frac = N > 0 ? double(nt) / N : 0.0;
        batch->w_mean = N > 0 ? sw / N : 0.0;
        batch->alpha_mean = batch->n_seqs_valid > 0 ? sa / batch->n_seqs_valid : 0.0;
    }
}

}  // namespace
}  // namespace acrl

using namespace acrl;

extern "C" acrl_status acrl_seq_discrepancy(const float* logp_pi, const float* logp_mu, const uint8_t* mask, int64_t T,
                                            const int64_t* seq_offsets, int32_t S, const int32_t* group_offsets,
                                            int32_t Gn, const float* entropy, float* lr, float* d,
                                            acrl_seq_stats* seq, acrl_group_stats* grp, acrl_batch_stats* batch,
                                            int32_t* dev_flags, acrl_stream stream) {
    if (T < 0 || S < 0 || Gn < 0) return ACRL_ERR_INVALID_ARG;
    if (!seq_offsets || !group_offsets || !batch || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!logp_pi || !logp_mu || !lr || !d)) return ACRL_ERR_INVALID_ARG;
    if ((S > 0 && !seq) || (Gn > 0 && !grp)) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (S > 0)
        seq_stats_kernel<<<S, kSeqThreads, 0, s>>>(logp_pi, logp_mu, mask, T, seq_offsets, S, group_offsets, Gn,
                                                   entropy, lr, d, seq, dev_flags);
    seq_finalize_kernel<<<1, kFinThreads, 0, s>>>(T, seq_offsets, S, group_offsets, Gn, seq, grp, batch, dev_flags);
    return launch_status();
}

extern "C" acrl_status acrl_grpo_advantage(const float* rewards, const int32_t* group_offsets, int32_t Gn, int32_t S,
                                           const acrl_params* p, float* adv, int32_t* dev_flags, acrl_stream stream) {
    if (Gn < 0 || S < 0 || !params_ok(p) || !group_offsets || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if (S > 0 && (!rewards || !adv)) return ACRL_ERR_INVALID_ARG;
    if (Gn == 0) return ACRL_OK;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int threads = 128;
    grpo_kernel<<<(Gn + threads - 1) / threads, threads, 0, s>>>(rewards, group_offsets, Gn, S, p->adv_eps,
                                                                 p->adv_ddof, p->singleton_rule, adv, dev_flags);
    return launch_status();
}

extern "C" acrl_status acrl_controller_init(acrl_controller_state* state, const acrl_params* p, acrl_stream stream) {
    if (!state || !params_ok(p)) return ACRL_ERR_INVALID_ARG;
    controller_init_kernel<<<1, 1, 0, reinterpret_cast<cudaStream_t>(stream)>>>(state, p->X_init);
    return launch_status();
}

extern "C" acrl_status acrl_controller_save(const acrl_controller_state* state, acrl_controller_state* host_state,
                                            acrl_stream stream) {
    if (!state || !host_state) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(host_state, state, sizeof(acrl_controller_state), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return ACRL_ERR_CUDA;
    return cudaStreamSynchronize(s) == cudaSuccess ? ACRL_OK : ACRL_ERR_CUDA;
}

extern "C" acrl_status acrl_controller_load(acrl_controller_state* state, const acrl_controller_state* host_state,
                                            acrl_stream stream) {
    if (!state || !host_state) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(state, host_state, sizeof(acrl_controller_state), cudaMemcpyHostToDevice, s) != cudaSuccess)
        return ACRL_ERR_CUDA;
    return cudaStreamSynchronize(s) == cudaSuccess ? ACRL_OK : ACRL_ERR_CUDA;
}

extern "C" acrl_status acrl_controller_step(acrl_controller_state* state, const acrl_params* p, const float* lr,
                                            const uint8_t* mask, int64_t T, const int64_t* seq_offsets, int32_t S,
                                            const int32_t* group_offsets, int32_t Gn, acrl_seq_stats* seq,
                                            const acrl_group_stats* grp, acrl_batch_stats* batch, const float* adv,
                                            float* weight, float* coef, float* alpha, float* ent_coef,
                                            int32_t* dev_flags, acrl_stream stream) {
    if (!state || !params_ok(p) || T < 0 || S < 0 || Gn < 0) return ACRL_ERR_INVALID_ARG;
    if (!seq_offsets || !group_offsets || !batch || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!lr || !weight || !coef)) return ACRL_ERR_INVALID_ARG;
    if ((S > 0 && (!seq || !adv)) || (Gn > 0 && !grp)) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    controller_alpha_kernel<<<1, kFinThreads, 0, s>>>(state, *p, S, Gn, seq, grp, batch, adv, alpha, dev_flags);
    if (S > 0)
        controller_weights_kernel<<<S, kSeqThreads, 0, s>>>(*p, lr, mask, T, seq_offsets, Gn, seq, grp, batch, adv,
                                                            weight, coef, ent_coef);
    controller_finalize_kernel<<<1, kFinThreads, 0, s>>>(S, seq, batch);
    return launch_status();
}

extern "C" acrl_status acrl_read_flags(const int32_t* dev_flags, int32_t* host_flags, acrl_stream stream) {
    if (!dev_flags || !host_flags) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(host_flags, dev_flags, sizeof(int32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return ACRL_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return ACRL_ERR_CUDA;
    return ACRL_OK;
}

extern "C" acrl_status acrl_check_flags(const int32_t* dev_flags, acrl_stream stream) {
    int32_t host = 0;
    const acrl_status st = acrl_read_flags(dev_flags, &host, stream);
    if (st != ACRL_OK) return st;
    return host != 0 ? ACRL_ERR_DEVICE_FLAGS : ACRL_OK;
}

extern "C" const char* acrl_status_string(acrl_status st) {
    switch (st) {
        case ACRL_OK: return "ok";
        case ACRL_ERR_INVALID_ARG: return "invalid argument";
        case ACRL_ERR_CUDA: return "CUDA launch or runtime error";
        case ACRL_ERR_NOT_IMPLEMENTED: return "not implemented";
        case ACRL_ERR_DEVICE_FLAGS: return "device flags raised";
        case ACRL_ERR_SCRATCH_TOO_SMALL: return "problem larger than the library's fixed scratch array";
    }
    return "unknown status";
}

extern "C" int32_t acrl_abi_version(void) { return ACRL_ABI_VERSION; }

extern "C" int64_t acrl_struct_size(int32_t which) {
    switch (which) {
        case 0: return sizeof(acrl_params);
        case 1: return sizeof(acrl_controller_state);
        case 2: return sizeof(acrl_seq_stats);
        case 3: return sizeof(acrl_group_stats);
        case 4: return sizeof(acrl_batch_stats);
    }
    return -1;
}
