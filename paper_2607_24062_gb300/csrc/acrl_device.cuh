// Device primitives for the ACRL kernels (sm_103a): streaming 16-byte loads
// and stores with cache hints, bf16 unpacking, the hardware base-2
// exponential, and deterministic warp/CTA reductions.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "acrl.h"

namespace acrl {

constexpr float kLog2e = 1.4426950408889634f;   // 1 / ln 2
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------------------
// memory
// ---------------------------------------------------------------------------

// 16-byte read of data that is used once: not kept in L1, L2 asked to fetch
// the surrounding 256 bytes (the rest of the row segment follows immediately).
__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// L2 cache policies for loads: keep a line (the first of two sweeps over a
// row) or let it go first (the last read of a line).
__device__ __forceinline__ uint64_t policy_evict_last() {
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// 16-byte non-allocating read with an explicit L2 policy.
__device__ __forceinline__ uint4 ld_policy(const uint4* p, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}

// 16-byte write of data that is not read back soon (evict-first).
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) {
    asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf16_to_float(acrl_bf16 h) { return __uint_as_float(uint32_t(h) << 16); }

// Two floats to a bf16x2 word, round to nearest even; `lo` lands in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// 2^x on the SFU (flushes subnormal results to zero).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ void raise_flag(int32_t* flags, int32_t bit) {
    if (flags) atomicOr(flags, bit);
}

// ---------------------------------------------------------------------------
// online log-sum-exp state in base 2
//   u = z * log2(e),  U = running max of u,
//   s0 = sum 2^(u - U),  s1 = sum 2^(u - U) (u - U)
// so that lse = ln2 (U + log2 s0) and entropy = ln2 (log2 s0 - s1 / s0).
// ---------------------------------------------------------------------------

struct LseAcc {
    float U;
    float s0;
    float s1;
};

__device__ __forceinline__ LseAcc lse_empty() { return LseAcc{-INFINITY, 0.f, 0.f}; }

// Merge two partial states.  An empty side (s0 == 0) contributes nothing; the
// selects keep -inf * 0 out of the arithmetic.
__device__ __forceinline__ LseAcc lse_merge(const LseAcc& a, const LseAcc& b) {
    const float U = fmaxf(a.U, b.U);
    LseAcc r;
    r.U = U;
    const float da = a.U - U, db = b.U - U;
    const float fa = a.s0 > 0.f ? ex2(da) : 0.f;
    const float fb = b.s0 > 0.f ? ex2(db) : 0.f;
    r.s0 = fa * a.s0 + fb * b.s0;
    const float ta = a.s0 > 0.f ? fa * fmaf(da, a.s0, a.s1) : 0.f;
    const float tb = b.s0 > 0.f ? fb * fmaf(db, b.s0, b.s1) : 0.f;
    r.s1 = ta + tb;
    return r;
}

__device__ __forceinline__ LseAcc shfl_xor(const LseAcc& a, int m) {
    return LseAcc{__shfl_xor_sync(0xffffffffu, a.U, m), __shfl_xor_sync(0xffffffffu, a.s0, m),
                  __shfl_xor_sync(0xffffffffu, a.s1, m)};
}

// Butterfly over the warp: every lane ends with the same value, and the
// combination order is fixed, so the result is deterministic.
__device__ __forceinline__ LseAcc warp_lse(LseAcc a) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) a = lse_merge(a, shfl_xor(a, m));
    return a;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) v += __shfl_xor_sync(0xffffffffu, v, m);
    return v;
}

template <typename T>
__device__ __forceinline__ T warp_max(T v) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, m));
    return v;
}

// CTA-wide sum in a fixed order; `scratch` holds one slot per warp.  Every
// thread gets the result.  Contains __syncthreads(): call from all threads.
template <typename T, int NWARPS>
__device__ __forceinline__ T block_sum(T v, T* scratch) {
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) scratch[wid] = v;
    __syncthreads();
    T r = T(0);
#pragma unroll
    for (int w = 0; w < NWARPS; ++w) r += scratch[w];
    return r;
}

template <typename T, int NWARPS>
__device__ __forceinline__ T block_max(T v, T* scratch) {
    v = warp_max(v);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) scratch[wid] = v;
    __syncthreads();
    T r = scratch[0];
#pragma unroll
    for (int w = 1; w < NWARPS; ++w) r = max(r, scratch[w]);
    return r;
}

// CTA-wide sums of N doubles and the maximum of one more, in the order of
// block_sum / block_max (a butterfly inside each warp, then the warps in
// order), with a single shared-memory exchange.  The results are valid in
// thread 0 only: the cross-warp pass runs there alone (fp64 is a narrow pipe
// on this part, so the other threads skip it).  `scratch` holds
// NWARPS * (N + 1) doubles.  Contains __syncthreads(): call from all threads.
template <int NWARPS, int N>
__device__ __forceinline__ void block_sums_max0(double (&v)[N], double& mx, double* scratch) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
#pragma unroll
        for (int k = 0; k < N; ++k) v[k] += __shfl_xor_sync(0xffffffffu, v[k], m);
        mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, m));
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
#pragma unroll
        for (int k = 0; k < N; ++k) scratch[wid * (N + 1) + k] = v[k];
        scratch[wid * (N + 1) + N] = mx;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
#pragma unroll
        for (int k = 0; k < N; ++k) v[k] = 0.0;
        mx = scratch[N];
        for (int w = 0; w < NWARPS; ++w) {
#pragma unroll
            for (int k = 0; k < N; ++k) v[k] += scratch[w * (N + 1) + k];
            mx = fmax(mx, scratch[w * (N + 1) + N]);
        }
    }
}

}  // namespace acrl
