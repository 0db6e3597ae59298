// Host-side helpers shared by the entry points: argument checks and launch
// status.  No state is kept between calls.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "acrl.h"

namespace acrl {

constexpr int64_t kMaxGrid = 2147483647LL;     // gridDim.x limit
constexpr int64_t kMaxVocab = 1LL << 30;       // keeps vector indices in int range
constexpr int64_t kWarpRowMaxV = 16384;        // rows up to this many columns use one warp each

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// CTAs for T rows at rows_per_cta rows each (kernels loop if capped).
inline int64_t grid_for(int64_t rows_per_cta, int64_t T) {
    const int64_t g = (T + rows_per_cta - 1) / rows_per_cta;
    return g < kMaxGrid ? g : kMaxGrid;
}

inline acrl_status launch_status() {
    return cudaGetLastError() == cudaSuccess ? ACRL_OK : ACRL_ERR_CUDA;
}

inline bool params_ok(const acrl_params* p) {
    if (!p) return false;
    if (!(p->gamma > 0.f) || !(p->C > 1.f) || !(p->clip_eps >= 0.f && p->clip_eps < 1.f)) return false;
    if (!(p->adv_eps >= 0.f) || !(p->kappa > 0.f) || !(p->x_ema >= 0.f && p->x_ema <= 1.f)) return false;
    if (!(p->entropy_coeff >= 0.f) || p->reserved != 0.f) return false;
    if (p->mode < ACRL_MODE_NONE || p->mode > ACRL_MODE_ACRL_FALLBACK) return false;
    if (p->y_gran < ACRL_Y_GROUP || p->y_gran > ACRL_Y_BATCH) return false;
    if (p->agg < ACRL_AGG_SEQ_MEAN_TOKEN_MEAN || p->agg > ACRL_AGG_TOKEN_MEAN) return false;
    if (p->adv_ddof < 0 || p->adv_ddof > 1) return false;
    if (p->singleton_rule < ACRL_SINGLETON_MEAN0_STD1 || p->singleton_rule > ACRL_SINGLETON_ZERO) return false;
    if (p->calib_steps < 1) return false;
    return true;
}

}  // namespace acrl
