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
// With an entropy bonus e_t the element becomes p (c + e (z - lse + H)): one
// more FMA and a multiply.  Rows that carry no gradient (masked, zero
// coefficient and no bonus, clipped) are written as zeros without reading
// their logits.  With lse == NULL the row's log-sum-exp is first recomputed
// by a sweep over the same row; the first 16-byte vectors of the row (up to
// 40, 72 or 96 KB, by the CTA's size) stay in the CTA's shared memory and, for
// rows of 65,536 columns or more, the next up to kTmemVecs (128 KB) in its
// tensor memory between the two sweeps, so that only the rest of the row is
// read again, from L2.  The shared-memory part arrives by one bulk copy
// started when the row starts, while the threads load the rest.
#include "acrl_device.cuh"
#include "acrl_host.h"
#include "mbarrier.cuh"
#include "row_lse.cuh"

namespace acrl {
namespace {

constexpr uint32_t kSignPair = 0x80008000u;

// CTA kernel: 512 threads, four 16-byte vectors per thread and step.  Its
// recompute path keeps kKeepVecs vectors of a row in shared memory between the
// sweeps (96 KB, three whole sweep chunks; two 512-thread CTAs per SM).
constexpr int kCtaThreads = 512, kCtaUnroll = 4;
// The streaming path (lse given) takes 768-thread CTAs for rows of more than
// 65,536 columns: 1.02-1.04 of the copy rate there against 0.99-1.02 with 512
// threads (whose last step over such a row is more ragged); 512 stay best for
// shorter rows.
constexpr int kWideThreads = 768;
constexpr int64_t kWideRowMinV = 65537;
constexpr int kChunk = kCtaThreads * kCtaUnroll;   // vectors one sweep step of the CTA covers
constexpr int kKeepVecs = 3 * kChunk;
static_assert(kKeepVecs * 16 <= 100 * 1024, "two CTAs per SM must fit");
// The next chunks of the row (whole chunks only, so that every warp takes part
// in each tensor-memory access) go to tensor memory: each of the two CTAs on an
// SM allocates 256 of its 512 columns, 128 lanes x 256 columns x 4 bytes =
// 128 KB = 4 chunks.  Thread t of warp w keeps its k-th vector of chunk c in
// lane 32 (w mod 4) + t, columns 64 (w / 4) + 16 c + 4 k .. + 3.
constexpr uint32_t kTmemCols = 256;
constexpr int kTmemChunks = 4;
constexpr int kTmemVecs = kTmemChunks * kChunk;
static_assert(kTmemVecs * 16 == 128 * kTmemCols * 4, "tensor-memory share of a CTA");
static_assert(kCtaThreads == 512 && kCtaUnroll == 4, "column layout: 16 warps, 4 vectors per step");
// Tensor memory holds whole chunks only, so rows of fewer than kKeepVecs +
// kChunk vectors (V < 65,536) keep nothing there; they take a kernel instance
// without any tcgen05 code (TM = false).  A resident CTA of a kernel that may
// allocate tensor memory keeps the SM from starting another CTA of that kernel
// until it has given up its allocation permit: measured with ncu, 15.6 warps
// resident per SM against 30.7 for the same work without tcgen05 code.
constexpr int kTmemMinVecs = kKeepVecs + kChunk;
// Longer rows of up to kSmallMaxVecs vectors (V <= 40,967) take 256-thread CTAs in
// the recompute path, each keeping up to 72 KB of its row in shared memory so
// that three fit on an SM (the rest of the row, at most 8 KB, is read again
// from L2): 0.92-0.98 of the copy rate for V = 32,000-40,000 against 0.77-0.85
// with two 512-thread CTAs per SM; from V = 44,000 the 512-thread CTAs, which
// keep 96 KB, are ahead (0.87-0.93 against 0.82-0.87).
constexpr int kSmallThreads = 256;
constexpr int kSmallKeepVecs = 4608;
constexpr int kSmallMaxVecs = 5120;
// Rows of up to kTinyMaxVecs vectors (V <= 24,583) take 128-thread CTAs that
// keep up to 40 KB of the row (five or more CTAs per SM; the rest, at most
// 8 KB, is read again from L2): 0.95-1.04 of the copy rate for V = 8,192-
// 24,576, where one warp per row, reading the whole row again from L2, reached
// 0.70-0.87 (32 rows of 32 KB in flight per SM no longer fit in L2 at
// V = 16,384).  Rows of up to kRecomputeWarpMaxV columns keep one warp per
// row (0.95 against 0.82 at V = 6,144).
constexpr int kTinyThreads = 128;
constexpr int kTinyKeepVecs = 2560;
constexpr int kTinyMaxVecs = 3072;
constexpr int kRecomputeWarpMaxV = 6144;

// Vectors of a row that a recompute CTA of THREADS threads keeps in shared memory.
template <int THREADS>
constexpr int kKeepOf = THREADS == kTinyThreads ? kTinyKeepVecs : THREADS == kSmallThreads ? kSmallKeepVecs : kKeepVecs;

// Where the vectors of a row live between the two sweeps of the recompute
// path: [0, s) in `smem` (filled by a bulk copy that completes on `bar`),
// [s, s + tm_chunks kChunk) in tensor memory from the thread's column base
// `tbase`, the rest in L2.
struct RowKeep {
    uint4* smem;
    int s;
    uint32_t tbase;
    int tm_chunks;
    uint64_t* bar;
};

// Bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned) from
// global to this CTA's shared memory, completing on `bar`, with an L2 policy.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
            "r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint4& v) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint4 tmem_ld4(uint32_t taddr) {
    uint4 v;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(taddr));
    return v;
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Per-row constants of the streaming pass.
struct RowPlan {
    float B;        // policy term only: lse log2e - log2|c|
    uint32_t sgn;   // policy term only: kSignPair when c < 0
    float L2;       // with entropy: lse log2e
    float e;        // with entropy: e_t
    float c2;       // with entropy: c - e (lse - H)
    float target;   // gradient at the sampled column
    int a;          // sampled column
};

template <bool ENT>
__device__ __forceinline__ float grad_elem(float z, const RowPlan& rp) {
    if (ENT) {
        const float p = ex2(fmaf(z, kLog2e, -rp.L2));
        return p * fmaf(rp.e, z, rp.c2);
    }
    return ex2(fmaf(z, kLog2e, -rp.B));  // magnitude; sign applied by the caller
}

template <bool ENT>
__device__ __forceinline__ uint4 grad_vec(const uint4 v, const RowPlan& rp, int rel) {
    float e[8];
    e[0] = grad_elem<ENT>(bf16_lo(v.x), rp);
    e[1] = grad_elem<ENT>(bf16_hi(v.x), rp);
    e[2] = grad_elem<ENT>(bf16_lo(v.y), rp);
    e[3] = grad_elem<ENT>(bf16_hi(v.y), rp);
    e[4] = grad_elem<ENT>(bf16_lo(v.z), rp);
    e[5] = grad_elem<ENT>(bf16_hi(v.z), rp);
    e[6] = grad_elem<ENT>(bf16_lo(v.w), rp);
    e[7] = grad_elem<ENT>(bf16_hi(v.w), rp);
    const uint32_t sgn = ENT ? 0u : rp.sgn;
    uint4 o;
    if (static_cast<unsigned>(rel) < 8u) {  // the vector holding the sampled column
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float val = sgn ? -e[j] : e[j];
            e[j] = (j == rel) ? rp.target : val;
        }
        o.x = pack_bf16x2(e[0], e[1]);
        o.y = pack_bf16x2(e[2], e[3]);
        o.z = pack_bf16x2(e[4], e[5]);
        o.w = pack_bf16x2(e[6], e[7]);
        return o;
    }
    o.x = pack_bf16x2(e[0], e[1]) ^ sgn;
    o.y = pack_bf16x2(e[2], e[3]) ^ sgn;
    o.z = pack_bf16x2(e[4], e[5]) ^ sgn;
    o.w = pack_bf16x2(e[6], e[7]) ^ sgn;
    return o;
}

// First sweep of the recompute path: the thread's partial state over its share
// of the row.  Vectors below `kp.s` (read once from HBM, L2 evict-first: they
// are not read from L2 again) come into shared memory by the bulk copy that
// thread 0 started on `kp.bar` (phase parity `parity`) and are folded last,
// once it has landed; those of the next kp.tm_chunks whole chunks are copied
// to tensor memory; the rest are loaded with the L2 evict-last policy, since
// the second sweep reads them again.  The tensor-memory stores are complete
// when the caller has waited for them (tmem_wait_st).  A copy that has not
// landed after the bounded wait raises ACRL_FLAG_TIMEOUT.
template <int TEAM, int UNROLL, bool TM>
__device__ __forceinline__ LseAcc recompute_partial(const acrl_bf16* __restrict__ row, int V, int tid, float& mx,
                                                    const RowKeep& kp, uint32_t parity, int32_t* flags) {
    LseAcc acc = lse_empty();
    mx = -INFINITY;
    const int nvec = V >> 3;
    const uint4* vrow = reinterpret_cast<const uint4*>(row);
    const uint64_t pol = policy_evict_last(), once = policy_evict_first();
    const int s = kp.s;
    int v = s + tid;
    // whole chunks (s is a multiple of the chunk whenever kp.tm_chunks > 0): every thread takes part
    if constexpr (TM) {
        for (int ch = 0; ch < kp.tm_chunks; ++ch, v += UNROLL * TEAM) {
            uint4 buf[UNROLL];
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) buf[k] = ld_policy(vrow + v + k * TEAM, once);
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) tmem_st4(kp.tbase + uint32_t(16 * ch + 4 * k), buf[k]);
            fold_vectors<UNROLL>(acc, mx, buf);
        }
    }
    for (; v + (UNROLL - 1) * TEAM < nvec; v += UNROLL * TEAM) {
        uint4 buf[UNROLL];
#pragma unroll
        for (int k = 0; k < UNROLL; ++k) buf[k] = ld_policy(vrow + v + k * TEAM, pol);
        fold_vectors<UNROLL>(acc, mx, buf);
    }
    for (; v < nvec; v += TEAM) {
        uint4 buf[1] = {ld_policy(vrow + v, pol)};
        fold_vectors<1>(acc, mx, buf);
    }
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) fold_scalar(acc, mx, bf16_to_float(row[j]));
    if (s > 0) {
        if (!wait_phase(kp.bar, parity, nullptr)) raise_flag(flags, ACRL_FLAG_TIMEOUT);
        for (v = tid; v + (UNROLL - 1) * TEAM < s; v += UNROLL * TEAM) {
            uint4 buf[UNROLL];
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) buf[k] = kp.smem[v + k * TEAM];
            fold_vectors<UNROLL>(acc, mx, buf);
        }
        for (; v < s; v += TEAM) {
            uint4 buf[1] = {kp.smem[v]};
            fold_vectors<1>(acc, mx, buf);
        }
    }
    return acc;
}

// LAST: this is the second sweep over a row after recompute_partial, and the
// last read of its lines (L2 evict-first policy).  It reads the part that
// comes from L2 in the order the first sweep loaded it, so that every line
// waits about as long in L2 as any other, then the chunks in tensor memory,
// then the vectors in shared memory.
template <int TEAM, int UNROLL, bool ENT, bool LAST = false, bool TM = false>
__device__ __forceinline__ void stream_grad_row(const acrl_bf16* __restrict__ row, acrl_bf16* __restrict__ grow, int V,
                                                int tid, const RowPlan& rp,
                                                const RowKeep& kp = RowKeep{nullptr, 0, 0u, 0, nullptr}) {
    const int nvec = V >> 3;
    const uint4* src = reinterpret_cast<const uint4*>(row);
    uint4* dst = reinterpret_cast<uint4*>(grow);
    if (LAST) {
        const uint64_t pol = policy_evict_first();
        const int te = kp.s + kp.tm_chunks * UNROLL * TEAM;   // first vector read from L2
        int v = te + tid;
        for (; v + (UNROLL - 1) * TEAM < nvec; v += UNROLL * TEAM) {
            uint4 buf[UNROLL];
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) buf[k] = ld_policy(src + v + k * TEAM, pol);
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) {
                const int vi = v + k * TEAM;
                st_stream(dst + vi, grad_vec<ENT>(buf[k], rp, rp.a - (vi << 3)));
            }
        }
        for (; v < nvec; v += TEAM) st_stream(dst + v, grad_vec<ENT>(ld_policy(src + v, pol), rp, rp.a - (v << 3)));
        for (int ch = 0; TM && ch < kp.tm_chunks; ++ch) {
            uint4 buf[UNROLL];
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) buf[k] = tmem_ld4(kp.tbase + uint32_t(16 * ch + 4 * k));
            tmem_wait_ld();
            const int v0 = kp.s + ch * UNROLL * TEAM + tid;
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) {
                const int vi = v0 + k * TEAM;
                st_stream(dst + vi, grad_vec<ENT>(buf[k], rp, rp.a - (vi << 3)));
            }
        }
        for (int vi = tid; vi < kp.s; vi += TEAM) st_stream(dst + vi, grad_vec<ENT>(kp.smem[vi], rp, rp.a - (vi << 3)));
    } else {
        int v = tid;
        for (; v + (UNROLL - 1) * TEAM < nvec; v += UNROLL * TEAM) {
            uint4 buf[UNROLL];
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) buf[k] = ld_stream(src + v + k * TEAM);
#pragma unroll
            for (int k = 0; k < UNROLL; ++k) {
                const int vi = v + k * TEAM;
                st_stream(dst + vi, grad_vec<ENT>(buf[k], rp, rp.a - (vi << 3)));
            }
        }
        for (; v < nvec; v += TEAM) st_stream(dst + v, grad_vec<ENT>(ld_stream(src + v), rp, rp.a - (v << 3)));
    }
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) {
        float val = grad_elem<ENT>(bf16_to_float(row[j]), rp);
        if (!ENT && rp.sgn) val = -val;
        if (j == rp.a) val = rp.target;
        grow[j] = static_cast<acrl_bf16>(pack_bf16x2(val, 0.f) & 0xffffu);
    }
}

// A gradient row of one value (`pair` holds it twice, as a bf16x2 word), written
// without reading the logits: 0 for rows that carry no gradient, NaN for rows
// whose surrogate is undefined.
constexpr uint32_t kZeroPair = 0u, kNaNPair = 0x7FC07FC0u;

template <int TEAM>
__device__ __forceinline__ void fill_row(acrl_bf16* __restrict__ grow, int V, int tid, uint32_t pair) {
    const int nvec = V >> 3;
    uint4* dst = reinterpret_cast<uint4*>(grow);
    const uint4 z = make_uint4(pair, pair, pair, pair);
    for (int v = tid; v < nvec; v += TEAM) st_stream(dst + v, z);
    for (int j = (nvec << 3) + tid; j < V; j += TEAM) grow[j] = static_cast<acrl_bf16>(pair & 0xffffu);
}

struct RowCoef {
    float c;       // coef_t g_t r_t
    float loss;    // token loss (policy term)
};

// Scalar part of a live row: r, the clip gate, the coefficient and the loss.
__device__ __forceinline__ RowCoef row_coef(float c0, float lp, const float* old_logp, int64_t t, float eps) {
    float r = 1.f;
    if (old_logp) r = expf(lp - old_logp[t]);
    const float rc = fminf(fmaxf(r, 1.f - eps), 1.f + eps);
    const bool gate = c0 >= 0.f ? (r <= 1.f + eps) : (r >= 1.f - eps);
    RowCoef out;
    out.c = gate ? c0 * r : 0.f;
    out.loss = c0 == 0.f ? 0.f : -c0 * (c0 >= 0.f ? fminf(r, rc) : fmaxf(r, rc));
    return out;
}

template <bool ENT>
__device__ __forceinline__ RowPlan make_plan(float c, float e, float L, float H, float za, float lp, int a) {
    RowPlan rp;
    rp.a = a;
    if (ENT) {
        rp.L2 = L * kLog2e;
        rp.e = e;
        rp.c2 = fmaf(-e, L - H, c);
        rp.B = 0.f;
        rp.sgn = 0u;
        // c (p_a - 1) + e p_a (z_a - lse + H)
        rp.target = fmaf(e * expf(lp), za - L + H, c * expm1f(lp));
    } else {
        rp.B = fmaf(L, kLog2e, -log2f(fabsf(c)));
        rp.sgn = c < 0.f ? kSignPair : 0u;
        rp.L2 = rp.e = rp.c2 = 0.f;
        rp.target = c * expm1f(lp);
    }
    return rp;
}

// lse and logp = z_a - lse of a row from its merged state and maximum, in the
// same form as the statistics kernel (the rounding of max*log2(e) corrected
// exactly through an FMA).
__device__ __forceinline__ void lse_logp(const LseAcc& acc, float mx, float za, float& L, float& lp) {
    const float l2s0 = log2f(acc.s0);
    const float c = fmaf(mx, kLog2e, -acc.U);
    L = fmaf(kLn2, l2s0 - c, mx);
    lp = (za - mx) - kLn2 * (l2s0 - c);
}

// One row handled by a team (a whole CTA, or one warp).  `part`/`part_mx` are
// the CTA's shared scratch for the recompute sweep, two buffers of one slot
// per warp used in turn (`par`, flipped at every row that uses them; unused by
// warp teams); `kp` says where the recompute path keeps the row between its
// two sweeps (nothing on chip for warp teams).  The bulk copy of the row's
// shared-memory part is started by thread 0 once the row is known to be live,
// and completes the phase of kp.bar whose parity is `par`: both flip at every
// live row of a CTA team.
template <int TEAM, int UNROLL, bool RECOMPUTE, bool ENT, bool TM>
__device__ __forceinline__ void grad_row(const acrl_bf16* __restrict__ logits, int64_t t, int V, int64_t ld,
                                         const int32_t* __restrict__ ids, const uint8_t* __restrict__ mask,
                                         const float* __restrict__ lse, const float* __restrict__ old_logp,
                                         const float* __restrict__ coef, const float* __restrict__ entropy,
                                         const float* __restrict__ ent_coef, float eps, acrl_bf16* __restrict__ grad,
                                         float* __restrict__ token_loss, int32_t* flags, int tid, LseAcc* part,
                                         float* part_mx, int& par, const RowKeep& kp) {
    const acrl_bf16* row = logits + t * ld;
    acrl_bf16* grow = grad + t * ld;
    const bool m = mask ? mask[t] != 0 : true;
    const float c0 = coef[t];
    const float e = ENT ? ent_coef[t] : 0.f;
    const int a = ids[t];
    const bool bad_id = a < 0 || a >= V;
    if (m && bad_id && tid == 0) raise_flag(flags, ACRL_FLAG_BAD_ID);
    const bool live = m && !bad_id && (c0 != 0.f || e != 0.f);
    float c = 0.f, loss = 0.f, L = 0.f, H = 0.f, za = 0.f, lp = 0.f;
    bool undefined = false;
    if (live) {
        if (RECOMPUTE && TEAM > 32 && kp.s > 0 && tid == 0) {
            // the threads' reads of the last row's part (before the CTA barrier) come before the copy's writes
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_expect_tx(kp.bar, uint32_t(kp.s) * 16u);
            bulk_load(kp.smem, row, uint32_t(kp.s) * 16u, kp.bar, policy_evict_first());
        }
        za = bf16_to_float(row[a]);
        if (RECOMPUTE) {
            float mx;
            LseAcc acc = warp_lse(recompute_partial<TEAM, UNROLL, TM>(row, V, tid, mx, kp, uint32_t(par), flags));
            if (TM && kp.tm_chunks > 0)
                tmem_wait_st();   // before the barrier: the row's tensor-memory part is written
            mx = warp_max(mx);
            if (TEAM > 32) {
                // Every warp combines the warps' states with the same butterfly, so all threads hold the same
                // result with one barrier.  The next write to this buffer comes two rows later, after the next
                // row's barrier, which every warp reaches only once it has read this one.
                constexpr int NW = TEAM / 32;
                static_assert(!RECOMPUTE || (NW <= 32 && (NW & (NW - 1)) == 0), "warps per team");
                const int lane = tid & 31;
                LseAcc* pp = part + par * NW;
                float* pm = part_mx + par * NW;
                if (lane == 0) {
                    pp[tid >> 5] = acc;
                    pm[tid >> 5] = mx;
                }
                __syncthreads();
                acc = lane < NW ? pp[lane] : lse_empty();
                mx = lane < NW ? pm[lane] : -INFINITY;
#pragma unroll
                for (int o = NW / 2; o >= 1; o >>= 1) {
                    acc = lse_merge(acc, shfl_xor(acc, o));
                    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
                }
                acc = LseAcc{__shfl_sync(0xffffffffu, acc.U, 0), __shfl_sync(0xffffffffu, acc.s0, 0),
                             __shfl_sync(0xffffffffu, acc.s1, 0)};
                mx = __shfl_sync(0xffffffffu, mx, 0);
                par ^= 1;
            }
            lse_logp(acc, mx, za, L, lp);
        } else {
            L = lse[t];
            lp = za - L;
        }
        // a row whose lse or log-prob is not finite (a NaN or an infinity among its logits), or whose old
        // log-prob is NaN, has no defined surrogate: NaN token loss and gradient row, and the flag
        undefined = !isfinite(L) || !isfinite(lp) || (old_logp != nullptr && isnan(old_logp[t]));
        if (undefined && tid == 0) raise_flag(flags, ACRL_FLAG_NONFINITE);
        const RowCoef rc = row_coef(c0, lp, old_logp, t, eps);
        c = rc.c;
        loss = rc.loss;
        if (ENT) {
            H = entropy[t];
            loss -= e * H;
        }
    }
    if (tid == 0) token_loss[t] = undefined ? __int_as_float(0x7fc00000) : loss;
    if (undefined) {
        fill_row<TEAM>(grow, V, tid, kNaNPair);
    } else if (c == 0.f && e == 0.f) {
        fill_row<TEAM>(grow, V, tid, kZeroPair);
    } else {
        stream_grad_row<TEAM, UNROLL, ENT, RECOMPUTE, TM>(row, grow, V, tid, make_plan<ENT>(c, e, L, H, za, lp, a),
                                                          kp);
    }
}

// TM: the recompute instance whose CTAs keep whole chunks of a row in tensor
// memory (512 threads, rows of at least kTmemMinVecs vectors).
template <int THREADS, int UNROLL, bool RECOMPUTE, bool ENT, bool TM = false>
__global__ void __launch_bounds__(THREADS) loss_grad_cta(
    const acrl_bf16* __restrict__ logits, int64_t T, int V, int64_t ld, const int32_t* __restrict__ ids,
    const uint8_t* __restrict__ mask, const float* __restrict__ lse, const float* __restrict__ old_logp,
    const float* __restrict__ coef, const float* __restrict__ entropy, const float* __restrict__ ent_coef, float eps,
    acrl_bf16* __restrict__ grad, float* __restrict__ token_loss, int32_t* flags) {
    __shared__ LseAcc part[2 * (THREADS / 32)];
    __shared__ float part_mx[2 * (THREADS / 32)];
    __shared__ uint32_t tmem_base;
    __shared__ __align__(8) uint64_t keep_bar;
    extern __shared__ uint4 keep[];  // recompute path: min(kKeepOf<THREADS>, V / 8) vectors (dynamic size)
    const int warp = threadIdx.x >> 5;
    static_assert(!TM || (RECOMPUTE && THREADS == kCtaThreads && UNROLL == kCtaUnroll), "tensor-memory layout");
    RowKeep kp{keep, 0, 0u, 0, &keep_bar};
    if (RECOMPUTE) {
        const int nvec = V >> 3;
        kp.s = min(kKeepOf<THREADS>, nvec);
        kp.tm_chunks = TM && nvec > kKeepVecs ? min(kTmemChunks, (nvec - kKeepVecs) / kChunk) : 0;
        if (threadIdx.x == 0) {
            mbar_init(&keep_bar, 1);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        if constexpr (TM) {
            if (warp == 0) {   // kp.tm_chunks is the same for every CTA of the launch
                if (kp.tm_chunks > 0)
                    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                                     static_cast<uint32_t>(__cvta_generic_to_shared(&tmem_base))),
                                 "r"(kTmemCols)
                                 : "memory");
                // at once, allocation or not: the SM may then start the kernel's next CTA
                asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        }
        __syncthreads();
        if constexpr (TM) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            if (kp.tm_chunks > 0)
                kp.tbase = tmem_base + (uint32_t((warp & 3) * 32) << 16) + uint32_t((warp >> 2) * 64);
        }
    }
    int par = 0;
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        // a CTA with a further row refills its shared-memory part only once every thread has read the last one
        if (RECOMPUTE && t != blockIdx.x) __syncthreads();
        grad_row<THREADS, UNROLL, RECOMPUTE, ENT, TM>(logits, t, V, ld, ids, mask, lse, old_logp, coef, entropy,
                                                      ent_coef, eps, grad, token_loss, flags, threadIdx.x, part, part_mx,
                                                      par, kp);
    }
    if constexpr (TM) {
        if (kp.tm_chunks > 0) {   // every tensor-memory read has completed (tmem_wait_ld)
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncthreads();
            if (warp == 0) {
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                             "r"(kTmemCols)
                             : "memory");
            }
        }
    }
}

template <int THREADS, int UNROLL, bool RECOMPUTE, bool ENT>
__global__ void __launch_bounds__(THREADS) loss_grad_warp(
    const acrl_bf16* __restrict__ logits, int64_t T, int V, int64_t ld, const int32_t* __restrict__ ids,
    const uint8_t* __restrict__ mask, const float* __restrict__ lse, const float* __restrict__ old_logp,
    const float* __restrict__ coef, const float* __restrict__ entropy, const float* __restrict__ ent_coef, float eps,
    acrl_bf16* __restrict__ grad, float* __restrict__ token_loss, int32_t* flags) {
    constexpr int NW = THREADS / 32;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    int par = 0;
    for (int64_t t = int64_t(blockIdx.x) * NW + wid; t < T; t += int64_t(gridDim.x) * NW)
        grad_row<32, UNROLL, RECOMPUTE, ENT, false>(logits, t, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps,
                                             grad, token_loss, flags, lane, nullptr, nullptr, par,
                                             RowKeep{nullptr, 0, 0u, 0, nullptr});
}

// Scalar loss: sum of token losses in a fixed order, by one cluster of
// kSumCtas CTAs (no scratch memory: the partial sums meet in distributed
// shared memory).  CTA c sums its contiguous block of the token losses: each
// thread adds float4 groups (four values in fp32) into two alternating fp64
// accumulators, so the loads pipeline and the fp64 adds are a quarter of the
// values; then a fixed CTA tree in fp64 whose cross-warp pass runs in thread 0
// alone; CTA 0 adds the CTAs' sums in rank order.  Eight CTAs keep eight SMs'
// loads in flight where one CTA left the reduction latency-bound (T = 524,288:
// ~75 us on one CTA).
constexpr int kSumThreads = 1024, kSumCtas = 8;

__device__ __forceinline__ void sum_cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ double ld_peer_f64(const double* p, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
    double v;
    asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(v) : "r"(a) : "memory");
    return v;
}

__global__ void __cluster_dims__(kSumCtas, 1, 1) __launch_bounds__(kSumThreads)
    loss_sum_kernel(const float* __restrict__ tl, int64_t T, float* __restrict__ loss) {
    __shared__ double sh[kSumThreads / 32 * 2];
    __shared__ double cta_sum;
    const int64_t c = blockIdx.x;   // the launch is one cluster: the block index is the rank
    double s0 = 0.0, s1 = 0.0;
    if ((reinterpret_cast<uintptr_t>(tl) & 15u) == 0) {
        const int64_t n4 = T / 4;
        const int64_t per = (n4 + kSumCtas - 1) / kSumCtas;
        const int64_t lo = min(n4, c * per), hi = min(n4, lo + per);
        const float4* v = reinterpret_cast<const float4*>(tl);
        int64_t i = lo + threadIdx.x;
#pragma unroll 4
        for (; i + kSumThreads < hi; i += 2 * kSumThreads) {
            const float4 a = v[i], b = v[i + kSumThreads];
            s0 += double((a.x + a.y) + (a.z + a.w));
            s1 += double((b.x + b.y) + (b.z + b.w));
        }
        for (; i < hi; i += kSumThreads) {
            const float4 a = v[i];
            s0 += double((a.x + a.y) + (a.z + a.w));
        }
        if (c == kSumCtas - 1)
            for (int64_t j = 4 * n4 + threadIdx.x; j < T; j += kSumThreads) s1 += tl[j];
    } else {
        const int64_t per = (T + kSumCtas - 1) / kSumCtas;
        const int64_t lo = min(T, c * per), hi = min(T, lo + per);
        for (int64_t j = lo + threadIdx.x; j < hi; j += kSumThreads) s0 += tl[j];
    }
    double total[1] = {s0 + s1}, unused = 0.0;
    block_sums_max0<kSumThreads / 32, 1>(total, unused, sh);
    if (threadIdx.x == 0) cta_sum = total[0];
    sum_cluster_sync();   // every CTA's sum is in its shared memory
    if (c == 0 && threadIdx.x == 0) {
        double r = 0.0;
        for (uint32_t k = 0; k < uint32_t(kSumCtas); ++k) r += ld_peer_f64(&cta_sum, k);
        *loss = float(r);
    }
    sum_cluster_sync();   // no CTA leaves while CTA 0 may still read its shared memory
}

template <bool RECOMPUTE, bool ENT>
acrl_status launch_loss_grad(const acrl_bf16* logits, int64_t T, int V, int64_t ld, const int32_t* ids,
                             const uint8_t* mask, const float* lse, const float* old_logp, const float* coef,
                             const float* entropy, const float* ent_coef, float eps, acrl_bf16* grad,
                             float* token_loss, int32_t* flags, cudaStream_t s) {
    if (V <= (RECOMPUTE ? kRecomputeWarpMaxV : kWarpRowMaxV)) {
        constexpr int THREADS = 256;
        loss_grad_warp<THREADS, 4, RECOMPUTE, ENT><<<unsigned(grid_for(THREADS / 32, T)), THREADS, 0, s>>>(
            logits, T, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps, grad, token_loss, flags);
    } else if (!RECOMPUTE && V >= kWideRowMinV) {
        loss_grad_cta<kWideThreads, kCtaUnroll, false, ENT><<<unsigned(grid_for(1, T)), kWideThreads, 0, s>>>(
            logits, T, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps, grad, token_loss, flags);
    } else if (RECOMPUTE && (V >> 3) <= kTinyMaxVecs) {
        if constexpr (RECOMPUTE) {
            auto kernel = loss_grad_cta<kTinyThreads, kCtaUnroll, true, ENT>;
            const int smem = 16 * min(V >> 3, kTinyKeepVecs);
            if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
                return ACRL_ERR_CUDA;
            kernel<<<unsigned(grid_for(1, T)), kTinyThreads, smem, s>>>(
                logits, T, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps, grad, token_loss, flags);
        }
    } else if (RECOMPUTE && (V >> 3) <= kSmallMaxVecs) {
        if constexpr (RECOMPUTE) {
            auto kernel = loss_grad_cta<kSmallThreads, kCtaUnroll, true, ENT>;
            const int smem = 16 * min(V >> 3, kSmallKeepVecs);
            if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
                return ACRL_ERR_CUDA;
            kernel<<<unsigned(grid_for(1, T)), kSmallThreads, smem, s>>>(
                logits, T, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps, grad, token_loss, flags);
        }
    } else if (RECOMPUTE && (V >> 3) >= kTmemMinVecs) {
        if constexpr (RECOMPUTE) {
            auto kernel = loss_grad_cta<kCtaThreads, kCtaUnroll, true, ENT, true>;
            const int smem = 16 * kKeepVecs;
            if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
                return ACRL_ERR_CUDA;
            kernel<<<unsigned(grid_for(1, T)), kCtaThreads, smem, s>>>(
                logits, T, V, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef, eps, grad, token_loss, flags);
        }
    } else {
        auto kernel = loss_grad_cta<kCtaThreads, kCtaUnroll, RECOMPUTE, ENT>;
        const int smem = RECOMPUTE ? 16 * (V >> 3 < kKeepVecs ? V >> 3 : kKeepVecs) : 0;
        if (smem > 0 && cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
            return ACRL_ERR_CUDA;
        kernel<<<unsigned(grid_for(1, T)), kCtaThreads, smem, s>>>(logits, T, V, ld, ids, mask, lse, old_logp, coef,
                                                                   entropy, ent_coef, eps, grad, token_loss, flags);
    }
    return ACRL_OK;
}

}  // namespace
}  // namespace acrl

using namespace acrl;

extern "C" acrl_status acrl_loss_grad_logits(const acrl_bf16* logits, int64_t T, int64_t V, int64_t ld,
                                             const int32_t* ids, const uint8_t* mask, const float* lse,
                                             const float* old_logp, const float* coef, const float* entropy,
                                             const float* ent_coef, float clip_eps, acrl_bf16* grad,
                                             float* token_loss, float* loss, int32_t* dev_flags, acrl_stream stream) {
    if (T < 0 || V < 1 || V > kMaxVocab || ld < V || (ld & 7) != 0) return ACRL_ERR_INVALID_ARG;
    if (!(clip_eps >= 0.f && clip_eps < 1.f)) return ACRL_ERR_INVALID_ARG;
    if (!loss || !dev_flags) return ACRL_ERR_INVALID_ARG;
    if ((entropy == nullptr) != (ent_coef == nullptr)) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!logits || !ids || !coef || !grad || !token_loss)) return ACRL_ERR_INVALID_ARG;
    if (T > 0 && (!aligned16(logits) || !aligned16(grad))) return ACRL_ERR_INVALID_ARG;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (T > 0) {
        const int v = int(V);
        const bool ent = ent_coef != nullptr;
        acrl_status st;
        if (lse && !ent)
            st = launch_loss_grad<false, false>(logits, T, v, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef,
                                                clip_eps, grad, token_loss, dev_flags, s);
        else if (lse && ent)
            st = launch_loss_grad<false, true>(logits, T, v, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef,
                                               clip_eps, grad, token_loss, dev_flags, s);
        else if (!ent)
            st = launch_loss_grad<true, false>(logits, T, v, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef,
                                               clip_eps, grad, token_loss, dev_flags, s);
        else
            st = launch_loss_grad<true, true>(logits, T, v, ld, ids, mask, lse, old_logp, coef, entropy, ent_coef,
                                              clip_eps, grad, token_loss, dev_flags, s);
        if (st != ACRL_OK) return st;
    }
    loss_sum_kernel<<<kSumCtas, kSumThreads, 0, s>>>(token_loss, T, loss);
    return launch_status();
}

extern "C" acrl_status acrl_reduce_loss(const float* token_loss, int64_t T, float* loss, acrl_stream stream) {
    if (T < 0 || !loss || (T > 0 && !token_loss)) return ACRL_ERR_INVALID_ARG;
    loss_sum_kernel<<<kSumCtas, kSumThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(token_loss, T, loss);
    return launch_status();
}
