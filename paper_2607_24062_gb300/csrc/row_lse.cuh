// Per-row online log-sum-exp over bf16 logits, shared by the statistics
// kernel, the gradient kernel's recompute sweep and the LM-head epilogue.
#pragma once

#include "acrl_device.cuh"

namespace acrl {

// Fold UNROLL 8-element vectors into the thread's running state.
template <int UNROLL>
__device__ __forceinline__ void fold_vectors(LseAcc& acc, float& mx, const uint4 (&v)[UNROLL]) {
    float f[UNROLL][8];
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
        f[k][0] = bf16_lo(v[k].x); f[k][1] = bf16_hi(v[k].x);
        f[k][2] = bf16_lo(v[k].y); f[k][3] = bf16_hi(v[k].y);
        f[k][4] = bf16_lo(v[k].z); f[k][5] = bf16_hi(v[k].z);
        f[k][6] = bf16_lo(v[k].w); f[k][7] = bf16_hi(v[k].w);
    }
    float vm = f[0][0];
#pragma unroll
    for (int k = 0; k < UNROLL; ++k)
#pragma unroll
        for (int j = 0; j < 8; ++j) vm = fmaxf(vm, f[k][j]);
    if (vm > mx) {  // new running maximum: rescale the partial sums
        const float Un = vm * kLog2e;
        if (acc.s0 > 0.f) {
            const float dl = acc.U - Un;
            const float s = ex2(dl);
            acc.s1 = s * fmaf(dl, acc.s0, acc.s1);
            acc.s0 *= s;
        }
        acc.U = Un;
        mx = vm;
    }
    const float U = acc.U;
    float s0a = 0.f, s0b = 0.f, s1a = 0.f, s1b = 0.f;
#pragma unroll
    for (int k = 0; k < UNROLL; ++k)
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
            const float y0 = fmaf(f[k][j], kLog2e, -U);
            const float y1 = fmaf(f[k][j + 1], kLog2e, -U);
            const float e0 = ex2(y0), e1 = ex2(y1);
            s0a += e0;
            s0b += e1;
            s1a = fmaf(e0, y0, s1a);
            s1b = fmaf(e1, y1, s1b);
        }
    acc.s0 += s0a + s0b;
    acc.s1 += s1a + s1b;
}

__device__ __forceinline__ void fold_scalar(LseAcc& acc, float& mx, float z) {
    if (z > mx) {
        const float Un = z * kLog2e;
        if (acc.s0 > 0.f) {
            const float dl = acc.U - Un;
            const float s = ex2(dl);
            acc.s1 = s * fmaf(dl, acc.s0, acc.s1);
            acc.s0 *= s;
        }
        acc.U = Un;
        mx = z;
    }
    const float y = fmaf(z, kLog2e, -acc.U);
    const float e = ex2(y);
    acc.s0 += e;
    acc.s1 = fmaf(e, y, acc.s1);
}

// The thread's partial state over its share of one row (lane `tid` of a team of TEAM threads).
template <int TEAM, int UNROLL>
__device__ __forceinline__ LseAcc row_partial(const acrl_bf16* __restrict__ row, int V, int tid, float& mx) {
    LseAcc acc = lse_empty();
    mx = -INFINITY;
    const int nvec = V >> 3;
    const uint4* vrow = reinterpret_cast<const uint4*>(row);
    int v = tid;
    for (; v + (UNROLL - 1) * TEAM < nvec; v += UNROLL * TEAM) {
        uint4 buf[UNROLL];
#pragma unroll
        for (int k = 0; k < UNROLL; ++k) buf[k] = ld_stream(vrow + v + k * TEAM);
        fold_vectors<UNROLL>(acc, mx, buf);
    }
    for (; v < nvec; v += TEAM) {
        uint4 buf[1] = {ld_stream(vrow + v)};
        fold_vectors<1>(acc, mx, buf);
    }
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) fold_scalar(acc, mx, bf16_to_float(row[j]));
    return acc;
}

// Outputs of one row from its merged state; mx is the row maximum (natural units).
__device__ __forceinline__ void row_outputs(const LseAcc& acc, float mx, const acrl_bf16* row, int V, int a,
                                            float* lse, float* logp, float* ent, int64_t t, int32_t* flags) {
    const float l2s0 = log2f(acc.s0);
    // acc.U is mx*log2(e) rounded; c is that rounding error, exact through the FMA
    const float c = fmaf(mx, kLog2e, -acc.U);
    const float lse_v = fmaf(kLn2, l2s0 - c, mx);
    const float H = kLn2 * (l2s0 - acc.s1 / acc.s0);
    float lp = 0.f;
    if (a >= 0 && a < V) {
        lp = (bf16_to_float(row[a]) - mx) - kLn2 * (l2s0 - c);
    } else {
        raise_flag(flags, ACRL_FLAG_BAD_ID);
    }
    if (!isfinite(lse_v) || !isfinite(H)) {
        raise_flag(flags, ACRL_FLAG_NONFINITE);
        lse[t] = logp[t] = ent[t] = __int_as_float(0x7fc00000);
        return;
    }
    lse[t] = lse_v;
    logp[t] = lp;
    ent[t] = H;
}

}  // namespace acrl
