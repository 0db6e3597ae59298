// acrl_token_stats: one streaming pass over pi's bf16 logits per token row
// giving the log-sum-exp, the sampled token's log-prob and the entropy.
//
// Each row is read exactly once from HBM with 16-byte non-allocating loads.
// A team of threads (eight lanes for rows of up to 4,096 columns, a warp for
// other short rows, the whole CTA for vocabulary-size rows) owns a row; every
// thread keeps an online base-2 state (max, sum 2^(u-U), sum 2^(u-U)(u-U))
// over its strided share of the row, and the team merges the states with a
// fixed butterfly/tree order, so results are bit-reproducible run to run.
#include "acrl_device.cuh"
#include "acrl_host.h"
#include "row_lse.cuh"

namespace acrl {
namespace {

// A whole CTA per row (vocabulary-size rows).
template <int THREADS, int UNROLL>
__global__ void __launch_bounds__(THREADS) token_stats_cta(const acrl_bf16* __restrict__ logits, int64_t T, int V,
                                                           int64_t ld, const int32_t* __restrict__ ids,
                                                           const uint8_t* __restrict__ mask, float* __restrict__ lse,
                                                           float* __restrict__ logp, float* __restrict__ ent,
                                                           int32_t* flags) {
    constexpr int NW = THREADS / 32;
    __shared__ LseAcc part[NW];
    __shared__ float pmax[NW];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        if (mask && mask[t] == 0) {
            if (threadIdx.x == 0) lse[t] = logp[t] = ent[t] = 0.f;
            continue;
        }
        const acrl_bf16* row = logits + t * ld;
        float mx;
        LseAcc acc = row_partial<THREADS, UNROLL>(row, V, threadIdx.x, mx);
        acc = warp_lse(acc);
        mx = warp_max(mx);
        if (lane == 0) {
            part[wid] = acc;
            pmax[wid] = mx;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            LseAcc r = part[0];
            float m = pmax[0];
#pragma unroll
            for (int w = 1; w < NW; ++w) {
                r = lse_merge(r, part[w]);
                m = fmaxf(m, pmax[w]);
            }
            row_outputs(r, m, row, V, ids[t], lse, logp, ent, t, flags);
        }
        __syncthreads();
    }
}

// One warp per row (short rows); THREADS/32 rows per CTA.
template <int THREADS, int UNROLL>
__global__ void __launch_bounds__(THREADS) token_stats_warp(const acrl_bf16* __restrict__ logits, int64_t T, int V,
                                                            int64_t ld, const int32_t* __restrict__ ids,
                                                            const uint8_t* __restrict__ mask, float* __restrict__ lse,
                                                            float* __restrict__ logp, float* __restrict__ ent,
                                                            int32_t* flags) {
    constexpr int NW = THREADS / 32;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    for (int64_t t = int64_t(blockIdx.x) * NW + wid; t < T; t += int64_t(gridDim.x) * NW) {
        if (mask && mask[t] == 0) {
            if (lane == 0) lse[t] = logp[t] = ent[t] = 0.f;
            continue;
        }
        const acrl_bf16* row = logits + t * ld;
        float mx;
        LseAcc acc = row_partial<32, UNROLL>(row, V, lane, mx);
        acc = warp_lse(acc);
        mx = warp_max(mx);
        if (lane == 0) row_outputs(acc, mx, row, V, ids[t], lse, logp, ent, t, flags);
    }
}

// Short rows (V <= kTeamRowMaxV): LANES lanes per row, 32 / LANES rows per warp
// at a time.  The team merges its states over log2(LANES) shuffle levels
// instead of five, which matters where the merges' exponentials are a large
// share of the row's (V = 2,048: 0.75 -> 0.94 of the copy rate with 8 lanes).
// Every lane takes part in the shuffles, whether its row is masked or not.
template <int LANES>
__device__ __forceinline__ LseAcc team_lse(LseAcc a) {
#pragma unroll
    for (int m = LANES / 2; m >= 1; m >>= 1) a = lse_merge(a, shfl_xor(a, m));
    return a;
}

template <int LANES>
__device__ __forceinline__ float team_max(float v) {
#pragma unroll
    for (int m = LANES / 2; m >= 1; m >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, m));
    return v;
}

template <int THREADS, int UNROLL, int LANES>
__global__ void __launch_bounds__(THREADS) token_stats_team(const acrl_bf16* __restrict__ logits, int64_t T, int V,
                                                            int64_t ld, const int32_t* __restrict__ ids,
                                                            const uint8_t* __restrict__ mask, float* __restrict__ lse,
                                                            float* __restrict__ logp, float* __restrict__ ent,
                                                            int32_t* flags) {
    constexpr int NW = THREADS / 32, RPW = 32 / LANES;
    static_assert(LANES >= 2 && LANES <= 32 && (LANES & (LANES - 1)) == 0, "lanes per row");
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, tl = lane % LANES;
    for (int64_t base = (int64_t(blockIdx.x) * NW + wid) * RPW; base < T; base += int64_t(gridDim.x) * NW * RPW) {
        const int64_t t = base + lane / LANES;
        const bool in = t < T;
        const bool live = in && !(mask && mask[t] == 0);
        const acrl_bf16* row = logits + (in ? t : 0) * ld;
        LseAcc acc = lse_empty();
        float mx = -INFINITY;
        if (live) acc = row_partial<LANES, UNROLL>(row, V, tl, mx);
        acc = team_lse<LANES>(acc);
        mx = team_max<LANES>(mx);
        if (tl == 0 && in) {
            if (live)
                row_outputs(acc, mx, row, V, ids[t], lse, logp, ent, t, flags);
            else
                lse[t] = logp[t] = ent[t] = 0.f;
        }
    }
}

}  // namespace

}  // namespace acrl

using namespace acrl;

// Rows up to this many columns (8 KB) are shared by eight lanes each.
constexpr int64_t kTeamRowMaxV = 4096;

// Rows up to this many columns (128 KB) use two warps each.
constexpr int64_t kMidRowMaxV = 65536;

extern "C" acrl_status acrl_token_stats(const acrl_bf16* logits, int64_t T, int64_t V, int64_t ld,
                                        const int32_t* ids, const uint8_t* mask, float* lse, float* logp,
                                        float* entropy, int32_t* dev_flags, acrl_stream stream) {
    if (T < 0 || V < 1 || V > kMaxVocab || ld < V || (ld & 7) != 0) return ACRL_ERR_INVALID_ARG;
    if (T == 0) return ACRL_OK;
    if (!logits || !ids || !lse || !logp || !entropy || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if (!aligned16(logits)) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int v = int(V);
    if (V <= kTeamRowMaxV) {
        constexpr int THREADS = 256, LANES = 8;
        token_stats_team<THREADS, 4, LANES><<<unsigned(grid_for(THREADS / LANES, T)), THREADS, 0, s>>>(
            logits, T, v, ld, ids, mask, lse, logp, entropy, dev_flags);
    } else if (V <= kWarpRowMaxV) {
        constexpr int THREADS = 256;
        token_stats_warp<THREADS, 4><<<unsigned(grid_for(THREADS / 32, T)), THREADS, 0, s>>>(
            logits, T, v, ld, ids, mask, lse, logp, entropy, dev_flags);
    } else if (V <= kMidRowMaxV) {
        // rows of up to 128 KB: two warps per row (measured 2 % faster than four at V = 32,000)
        constexpr int THREADS = 64;
        token_stats_cta<THREADS, 4><<<unsigned(grid_for(1, T)), THREADS, 0, s>>>(
            logits, T, v, ld, ids, mask, lse, logp, entropy, dev_flags);
    } else {
        // 128 threads per row: many independent rows in flight per SM and a short
        // end-of-row merge (measured best of 64/128/256/512/1024 and a warp per row)
        constexpr int THREADS = 128;
        token_stats_cta<THREADS, 4><<<unsigned(grid_for(1, T)), THREADS, 0, s>>>(
            logits, T, v, ld, ids, mask, lse, logp, entropy, dev_flags);
    }
    return launch_status();
}
