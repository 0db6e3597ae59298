// acrl_loss_grad_logits: the loss of Eq. ACRL and its gradient with respect
// to pi's logits, written in bf16 without ever storing the probabilities.
//
//     grad[t, j] = coef_t g_t r_t (p_tj - 1[j = a_t]),  p_tj = exp(z_tj - lse_t)
//
// One streaming pass per live row: read 2 bytes and write 2 bytes per element.
// The row's factor is folded into the exponent, |c| p = 2^(z log2e - (lse log2e
// - log2|c|)), so each element costs one FMA and one SFU exp2; the sign is
// applied to the packed bf16 pair with one XOR.  The target column is written
// as c * expm1(logp) so that p_a - 1 keeps its accuracy when p_a is near 1.
// Rows that carry no gradient (masked, zero coefficient, clipped) are written
// as zeros without reading their logits.  With lse == NULL the row's
// log-sum-exp is first recomputed by a sweep over the same row.
#include "acrl_device.cuh"
#include "acrl_host.h"
#include "row_lse.cuh"

namespace acrl {
namespace {

constexpr uint32_t kSignPair = 0x80008000u;

struct RowPlan {
    float B;        // lse log2e - log2|c|
    uint32_t sgn;   // kSignPair when c < 0
    float target;   // gradient at the sampled column, sign included
    int a;          // sampled column
};

__device__ __forceinline__ uint4 grad_vec(const uint4 v, const RowPlan& rp, int rel) {
    float e[8];
    e[0] = ex2(fmaf(bf16_lo(v.x), kLog2e, -rp.B));
    e[1] = ex2(fmaf(bf16_hi(v.x), kLog2e, -rp.B));
    e[2] = ex2(fmaf(bf16_lo(v.y), kLog2e, -rp.B));
    e[3] = ex2(fmaf(bf16_hi(v.y), kLog2e, -rp.B));
    e[4] = ex2(fmaf(bf16_lo(v.z), kLog2e, -rp.B));
    e[5] = ex2(fmaf(bf16_hi(v.z), kLog2e, -rp.B));
    e[6] = ex2(fmaf(bf16_lo(v.w), kLog2e, -rp.B));
    e[7] = ex2(fmaf(bf16_hi(v.w), kLog2e, -rp.B));
    uint4 o;
    if (static_cast<unsigned>(rel) < 8u) {  // the vector holding the sampled column
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float val = rp.sgn ? -e[j] : e[j];
            e[j] = (j == rel) ? rp.target : val;
        }
        o.x = pack_bf16x2(e[0], e[1]);
        o.y = pack_bf16x2(e[2], e[3]);
        o.z = pack_bf16x2(e[4], e[5]);
        o.w = pack_bf16x2(e[6], e[7]);
        return o;
    }
    o.x = pack_bf16x2(e[0], e[1]) ^ rp.sgn;
    o.y = pack_bf16x2(e[2], e[3]) ^ rp.sgn;
    o.z = pack_bf16x2(e[4], e[5]) ^ rp.sgn;
    o.w = pack_bf16x2(e[6], e[7]) ^ rp.sgn;
    return o;
}

template <int TEAM, int UNROLL>
__device__ __forceinline__ void stream_grad_row(const acrl_bf16* __restrict__ row, acrl_bf16* __restrict__ grow, int V,
                                                int tid, const RowPlan& rp) {
    const int nvec = V >> 3;
    const uint4* src = reinterpret_cast<const uint4*>(row);
    uint4* dst = reinterpret_cast<uint4*>(grow);
    int v = tid;
    for (; v + (UNROLL - 1) * TEAM < nvec; v += UNROLL * TEAM) {
        uint4 buf[UNROLL];
#pragma unroll
        for (int k = 0; k < UNROLL; ++k) buf[k] = ld_stream(src + v + k * TEAM);
#pragma unroll
        for (int k = 0; k < UNROLL; ++k) {
            const int vi = v + k * TEAM;
            st_stream(dst + vi, grad_vec(buf[k], rp, rp.a - (vi << 3)));
        }
    }
    for (; v < nvec; v += TEAM) st_stream(dst + v, grad_vec(ld_stream(src + v), rp, rp.a - (v << 3)));
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) {
        float val = ex2(fmaf(bf16_to_float(row[j]), kLog2e, -rp.B));
        if (rp.sgn) val = -val;
        if (j == rp.a) val = rp.target;
        grow[j] = static_cast<acrl_bf16>(pack_bf16x2(val, 0.f) & 0xffffu);
    }
}

template <int TEAM>
__device__ __forceinline__ void zero_row(acrl_bf16* __restrict__ grow, int V, int tid) {
    const int nvec = V >> 3;
    uint4* dst = reinterpret_cast<uint4*>(grow);
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (int v = tid; v < nvec; v += TEAM) st_stream(dst + v, z);
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) grow[j] = 0;
}

struct RowCoef {
    float c;       // coef_t g_t r_t
    float loss;    // token loss
    float lp;      // logp_t
};

// Scalar part of a live row: r, the clip gate, the coefficient and the loss.
__device__ __forceinline__ RowCoef row_coef(float c0, float lp, const float* old_logp, int64_t t, float eps) {
    float r = 1.f;
    if (old_logp) r = expf(lp - old_logp[t]);
    const float rc = fminf(fmaxf(r, 1.f - eps), 1.f + eps);
    const bool gate = c0 >= 0.f ? (r <= 1.f + eps) : (r >= 1.f - eps);
    RowCoef out;
    out.c = gate ? c0 * r : 0.f;
    out.loss = -c0 * (c0 >= 0.f ? fminf(r, rc) : fmaxf(r, rc));
    out.lp = lp;
    return out;
}

__device__ __forceinline__ RowPlan make_plan(float c, float L, float lp, int a) {
    RowPlan rp;
    rp.B = fmaf(L, kLog2e, -log2f(fabsf(c)));
    rp.sgn = c < 0.f ? kSignPair : 0u;
    rp.target = c * expm1f(lp);
    rp.a = a;
    return rp;
}

// A whole CTA per row.
template <int THREADS, int UNROLL, bool RECOMPUTE>
__global__ void __launch_bounds__(THREADS) loss_grad_cta(
    const acrl_bf16* __restrict__ logits, int64_t T, int V, int64_t ld, const int32_t* __restrict__ ids,
    const uint8_t* __restrict__ mask, const float* __restrict__ lse, const float* __restrict__ old_logp,
    const float* __restrict__ coef, float eps, acrl_bf16* __restrict__ grad, float* __restrict__ token_loss,
    int32_t* flags) {
    constexpr int NW = THREADS / 32;
    __shared__ LseAcc part[NW];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        const acrl_bf16* row = logits + t * ld;
        acrl_bf16* grow = grad + t * ld;
        const bool m = mask ? mask[t] != 0 : true;
        const float c0 = coef[t];
        const int a = ids[t];
        const bool bad_id = a < 0 || a >= V;
        if (m && bad_id && threadIdx.x == 0) raise_flag(flags, ACRL_FLAG_BAD_ID);
        const bool live = m && c0 != 0.f && !bad_id;
        RowCoef rc{0.f, 0.f, 0.f};
        float L = 0.f;
        if (live) {
            if (RECOMPUTE) {
                float mx;
                LseAcc acc = row_partial<THREADS, UNROLL>(row, V, threadIdx.x, mx);
                acc = warp_lse(acc);
                if (lane == 0) part[wid] = acc;
                __syncthreads();
                LseAcc r = part[0];
#pragma unroll
                for (int w = 1; w < NW; ++w) r = lse_merge(r, part[w]);
                __syncthreads();
                L = kLn2 * (r.U + log2f(r.s0));
            } else {
                L = lse[t];
            }
            rc = row_coef(c0, bf16_to_float(row[a]) - L, old_logp, t, eps);
        }
        if (threadIdx.x == 0) token_loss[t] = rc.loss;
        if (rc.c == 0.f) {
            zero_row<THREADS>(grow, V, threadIdx.x);
        } else {
            stream_grad_row<THREADS, UNROLL>(row, grow, V, threadIdx.x, make_plan(rc.c, L, rc.lp, a));
        }
    }
}

// One warp per row.
template <int THREADS, int UNROLL, bool RECOMPUTE>
__global__ void __launch_bounds__(THREADS) loss_grad_warp(
    const acrl_bf16* __restrict__ logits, int64_t T, int V, int64_t ld, const int32_t* __restrict__ ids,
    const uint8_t* __restrict__ mask, const float* __restrict__ lse, const float* __restrict__ old_logp,
    const float* __restrict__ coef, float eps, acrl_bf16* __restrict__ grad, float* __restrict__ token_loss,
    int32_t* flags) {
    constexpr int NW = THREADS / 32;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int64_t t = int64_t(blockIdx.x) * NW + wid; t < T; t += int64_t(gridDim.x) * NW) {
        const acrl_bf16* row = logits + t * ld;
        acrl_bf16* grow = grad + t * ld;
        const bool m = mask ? mask[t] != 0 : true;
        const float c0 = coef[t];
        const int a = ids[t];
        const bool bad_id = a < 0 || a >= V;
        if (m && bad_id && lane == 0) raise_flag(flags, ACRL_FLAG_BAD_ID);
        const bool live = m && c0 != 0.f && !bad_id;
        RowCoef rc{0.f, 0.f, 0.f};
        float L = 0.f;
        if (live) {
            if (RECOMPUTE) {
                float mx;
                LseAcc acc = warp_lse(row_partial<32, UNROLL>(row, V, lane, mx));
                L = kLn2 * (acc.U + log2f(acc.s0));
            } else {
                L = lse[t];
            }
            rc = row_coef(c0, bf16_to_float(row[a]) - L, old_logp, t, eps);
        }
        if (lane == 0) token_loss[t] = rc.loss;
        if (rc.c == 0.f) {
            zero_row<32>(grow, V, lane);
        } else {
            stream_grad_row<32, UNROLL>(row, grow, V, lane, make_plan(rc.c, L, rc.lp, a));
        }
    }
}

// Scalar loss: sum of token losses in a fixed order with fp64 accumulation.
constexpr int kSumThreads = 1024;
__global__ void __launch_bounds__(kSumThreads) loss_sum_kernel(const float* __restrict__ tl, int64_t T,
                                                               float* __restrict__ loss) {
    __shared__ double sh[kSumThreads / 32];
    double s = 0.0;
    for (int64_t t = threadIdx.x; t < T; t += kSumThreads) s += tl[t];
    s = block_sum<double, kSumThreads / 32>(s, sh);
    if (threadIdx.x == 0) *loss = float(s);
}

template <bool RECOMPUTE>
void launch_loss_grad(const acrl_bf16* logits, int64_t T, int V, int64_t ld, const int32_t* ids, const uint8_t* mask,
                      const float* lse, const float* old_logp, const float* coef, float eps, acrl_bf16* grad,
                      float* token_loss, int32_t* flags, cudaStream_t s) {
    if (V <= kWarpRowMaxV) {
        constexpr int THREADS = 256;
        loss_grad_warp<THREADS, 4, RECOMPUTE><<<unsigned(grid_for(THREADS / 32, T)), THREADS, 0, s>>>(
            logits, T, V, ld, ids, mask, lse, old_logp, coef, eps, grad, token_loss, flags);
    } else {
        constexpr int THREADS = 512;
        loss_grad_cta<THREADS, 4, RECOMPUTE><<<unsigned(grid_for(1, T)), THREADS, 0, s>>>(
            logits, T, V, ld, ids, mask, lse, old_logp, coef, eps, grad, token_loss, flags);
    }
}

}  // namespace
}  // namespace acrl

using namespace acrl;

extern "C" acrl_status acrl_loss_grad_logits(const acrl_bf16* logits, int64_t T, int64_t V, int64_t ld,
                                             const int32_t* ids, const uint8_t* mask, const float* lse,
                                             const float* old_logp, const float* coef, float clip_eps,
                                             acrl_bf16* grad, float* token_loss, float* loss, int32_t* dev_flags,
                                             acrl_stream stream) {
    if (T < 0 || V < 1 || V > kMaxVocab || ld < V || (ld & 7) != 0) return ACRL_ERR_INVALID_ARG;
    if (!(clip_eps >= 0.f && clip_eps < 1.f)) return ACRL_ERR_INVALID_ARG;
    if (!loss || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!logits || !ids || !coef || !grad || !token_loss)) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!aligned16(logits) || !aligned16(grad))) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (T > 0) {
        if (lse)
            launch_loss_grad<false>(logits, T, int(V), ld, ids, mask, lse, old_logp, coef, clip_eps, grad, token_loss,
                                    dev_flags, s);
        else
            launch_loss_grad<true>(logits, T, int(V), ld, ids, mask, lse, old_logp, coef, clip_eps, grad, token_loss,
                                   dev_flags, s);
    }
    loss_sum_kernel<<<1, kSumThreads, 0, s>>>(token_loss, T, loss);
    return launch_status();
}

extern "C" acrl_status acrl_reduce_loss(const float* token_loss, int64_t T, float* loss, acrl_stream stream) {
    if (T < 0 || !loss || (T > 0 && !token_loss)) return ACRL_ERR_INVALID_ARG;
    loss_sum_kernel<<<1, kSumThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(token_loss, T, loss);
    return launch_status();
}
