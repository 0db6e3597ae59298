// LM-head projection on the tensor cores with the log-softmax statistics in
// the epilogue: logits = H W^T (bf16 inputs, fp32 accumulation, bf16 output),
// and for every (row, 256-column tile) the online state (max, sum 2^(u-U),
// sum 2^(u-U)(u-U)) of the bf16-rounded logits, so that the merge kernel gets
// lse, the sampled token's log-prob and the entropy without reading the logits
// again.
//
// Blackwell path: a persistent kernel of CTA pairs (clusters of two CTAs,
// tcgen05 cta_group::2), one CTA per SM, warp-specialised.  A pair computes a
// 256 x 256 tile of the logits: each CTA stages its own 128 rows of H and its
// 128-row half of the weight tile, and the MMAs of the even CTA read both
// CTAs' shared memory and write each CTA's 128 accumulator rows into that
// CTA's TMEM.  Per SM a K slab is 32 KB (A 128 x 64 + B 128 x 64), so six
// stages fit and the weight half is never staged twice in a pair.
//   warp 0     in each CTA, one thread issues the TMA loads (128B-swizzled)
//              of the CTA's A and B into a 6-stage ring, counted on the even
//              CTA's stage barrier;
//   warp 1     in the even CTA, one thread issues tcgen05.mma (M=256, N=256,
//              K=16, kind::f16) into one of two 256-column accumulators and
//              releases each stage to the producers of both CTAs, one commit
//              per CTA;
//   warps 2-5  in each CTA, the epilogue: tcgen05.ld of its accumulator rows
//              (each thread one row), round to bf16, fold the statistics, and
//              write the logits through shared memory with TMA bulk tensor
//              stores (32 x 32 blocks, two staging buffers per warp).
// Tiles are visited in bands of 32 row tiles (16 pairs) so that the weight
// tiles in flight are shared through L2 by the pairs working on the same band.
// Every CTA loads only from this GPU's memory into its own shared memory (the
// tensor maps are encoded over pointers that the entry points have checked to
// be device memory of the current device), and each load fills that CTA's
// shared memory alone.
// Every wait on an mbarrier is bounded in time; on expiry the kernel raises
// ACRL_FLAG_TIMEOUT, lets the copies it issued land, and exits after freeing
// its TMEM.  The two CTAs meet at a cluster barrier after initialising their
// barriers and again before either frees its TMEM or exits, so neither touches
// a peer that has gone.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <initializer_list>

#include "acrl_device.cuh"
#include "acrl_host.h"
#include "row_lse.cuh"
#include "mbarrier.cuh"

namespace acrl {
namespace {

constexpr int kBM = 128, kBN = 256;   // rows of H per CTA, columns (weight rows) per tile
constexpr int kBK = 64;               // K slab: 64 bf16 = one 128-byte row under the 128-byte swizzle
constexpr int kStages = 6;
constexpr int kHalfBN = kBN / 2;      // weight rows staged by each CTA of a pair
constexpr int kABytes = kBM * kBK * 2;
constexpr int kBBytes = kHalfBN * kBK * 2;
constexpr int kStageBytes = kABytes + kBBytes;   // per CTA; the pair's stage barrier counts twice this
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr int kBandM = 32;            // row tiles per band (16 pairs)
// Output staging: each epilogue warp owns two 32 x 32 bf16 blocks (its 32
// rows x one 32-column chunk of the accumulator), stored 64-byte-swizzled.
constexpr int kOutBlockBytes = 32 * 32 * 2;
constexpr int kOutBytes = 4 * 2 * kOutBlockBytes;
// Instruction descriptor of tcgen05.mma kind::f16: D f32 (bits 4-5 = 1), A and
// B bf16 (bits 7-9, 10-12 = 1), both K-major, N/8 at bit 17, M/16 at bit 24
// (M = 256 across the pair, 128 rows in each CTA's TMEM).
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(kBN >> 3) << 17) |
                            (uint32_t((2 * kBM) >> 4) << 24);
// Barriers:
//   full[s]    even CTA: both CTAs' copies of stage s landed
//   empty[s]   each CTA: the MMAs reading stage s are done
//   tfull[b]   each CTA: accumulator b is complete
//   tempty[b]  even CTA: the eight epilogue warps of the pair drained accumulator b
struct Barriers {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t mma_done;
    uint32_t tmem_base;
    int32_t abort;
};
// The B stages come first, then the A stages, the output staging blocks and
// the barriers, with a margin behind them (every descriptor read stays inside
// the allocation).
constexpr int kMargin = 8192;
constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kOutBytes + int(sizeof(Barriers)) + kMargin;
static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t peer_addr(const void* p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
    return r;
}

__device__ __forceinline__ void remote_arrive(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// Tile load into this CTA's shared memory whose completion is counted on the
// barrier at `bar` (a shared::cluster address: either CTA of the pair).
__device__ __forceinline__ void tma_load_pair(void* dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
        "%3}], [%4];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major bf16 tile written by TMA with
// the 128-byte swizzle: rows of 128 bytes, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
    uint64_t d = uint64_t((addr & 0x3FFFFu) >> 4);  // start address
    d |= uint64_t(1024 >> 4) << 32;                  // stride between 8-row groups
    d |= uint64_t(1) << 46;                          // descriptor version of tcgen05
    d |= uint64_t(2) << 61;                          // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void mma_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            tmem_d),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate));
}

// Arrive once on the barrier at shared::cluster address `bar` when this
// thread's MMAs so far have completed.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
        "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void st_shared16(uint32_t addr, const uint4& v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// Make this thread's shared-memory writes visible to the TMA (async proxy).
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(smem_u32(src))
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Wait until at most N of this thread's bulk stores still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ---------------------------------------------------------------------------
// tile schedule: bands of BAND row-tile pairs, all column tiles of a band in
// turn; the pair of cluster c takes tiles c, c + clusters, ...
// ---------------------------------------------------------------------------

__device__ __forceinline__ void tile_coords(int t, int m_pairs, int n_tiles, int& mp, int& n) {
    constexpr int BAND = kBandM / 2;
    const int per_band = BAND * n_tiles;
    const int band = t / per_band;
    const int r = t - band * per_band;
    const int bm = min(BAND, m_pairs - band * BAND);
    mp = band * BAND + r % bm;
    n = r / bm;
}

__device__ __forceinline__ void give_up(volatile int32_t* abort, int32_t* flags) {
    *abort = 1;
    raise_flag(flags, ACRL_FLAG_TIMEOUT);
}

// ---------------------------------------------------------------------------
// roles
// ---------------------------------------------------------------------------

__device__ void producer(const CUtensorMap* tmA, const CUtensorMap* tmB, uint8_t* sA, uint8_t* sB, Barriers* bars,
                         uint32_t rank, int m_pairs, int n_tiles, int total, int k_iters, int32_t* flags) {
    volatile int32_t* abort = &bars->abort;
    const int cl = int(blockIdx.x >> 1), ncl = int(gridDim.x >> 1);
    int stage = 0;
    uint32_t phase = 0;
    long issued = 0;
    bool ok = true;
    for (int t = cl; t < total && ok; t += ncl) {
        int mp, n;
        tile_coords(t, m_pairs, n_tiles, mp, n);
        const int m = 2 * mp + int(rank);
        for (int kk = 0; kk < k_iters; ++kk) {
            if (!mbar_try_wait(&bars->empty[stage], phase ^ 1u) &&
                !wait_phase(&bars->empty[stage], phase ^ 1u, abort)) {
                give_up(abort, flags);
                ok = false;
                break;
            }
            // the even CTA's barrier counts both CTAs' bytes of this stage
            if (rank == 0) mbar_expect_tx(&bars->full[stage], 2 * kStageBytes);
            const uint32_t full0 = peer_addr(&bars->full[stage], 0);
            tma_load_pair(sA + stage * kABytes, tmA, full0, kk * kBK, m * kBM);
            tma_load_pair(sB + stage * kBBytes, tmB, full0, kk * kBK, n * kBN + int(rank) * kHalfBN);
            ++issued;
            if (++stage == kStages) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
    if (!ok) {
        // let the copies this thread started land before the CTA can exit: the even CTA waits for its
        // barriers (they count both CTAs' copies), the odd one gives its copies time to land
        if (rank == 0) {
            for (long j = issued - 1; j >= 0 && j >= issued - kStages; --j)
                wait_phase(&bars->full[j % kStages], uint32_t((j / kStages) & 1), nullptr);
        } else {
            const uint64_t t0 = global_ns();
            while (global_ns() - t0 < 100000ull) {
            }
        }
    }
}

// The even CTA's MMA thread.
__device__ void mma_issuer(uint8_t* sA, uint8_t* sB, Barriers* bars, uint32_t tmem, int total, int k_iters,
                           int32_t* flags) {
    volatile int32_t* abort = &bars->abort;
    const int cl = int(blockIdx.x >> 1), ncl = int(gridDim.x >> 1);
    // descriptors of stage 0; a descriptor advances by (address offset) / 16
    const uint64_t adesc0 = smem_desc(smem_u32(sA)), bdesc0 = smem_desc(smem_u32(sB));
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int t = cl; t < total && ok; t += ncl) {
        if (!wait_phase(&bars->tempty[acc], acc_phase ^ 1u, abort)) {
            give_up(abort, flags);
            break;
        }
        tc_fence_after();
        const uint32_t d = tmem + uint32_t(acc * kBN);
        for (int kk = 0; kk < k_iters; ++kk) {
            // the common case (the stage has landed) stays inline; the bounded wait is the slow path
            if (!mbar_try_wait(&bars->full[stage], phase) && !wait_phase(&bars->full[stage], phase, abort)) {
                give_up(abort, flags);
                ok = false;
                break;
            }
            tc_fence_after();
            const uint64_t ad = adesc0 + uint64_t((stage * kABytes) >> 4);
            const uint64_t bd = bdesc0 + uint64_t((stage * kBBytes) >> 4);
#pragma unroll
            for (int k16 = 0; k16 < kBK / 16; ++k16)  // 16 columns = 32 bytes = 2 descriptor units
                mma_pair(d, ad + uint64_t(2 * k16), bd + uint64_t(2 * k16), (kk | k16) != 0);
            // release the stage to both producers: one commit for each CTA's barrier
            mma_commit(peer_addr(&bars->empty[stage], 0));
            mma_commit(peer_addr(&bars->empty[stage], 1));
            if (++stage == kStages) {
                stage = 0;
                phase ^= 1u;
            }
        }
        if (!ok) break;
        mma_commit(peer_addr(&bars->tfull[acc], 0));
        mma_commit(peer_addr(&bars->tfull[acc], 1));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
    }
    // every MMA this thread issued has finished before the pair moves on
    mma_commit(peer_addr(&bars->mma_done, 0));
    wait_phase(&bars->mma_done, 0, nullptr);
}

__device__ void epilogue(Barriers* bars, uint32_t tmem, uint32_t rank, const CUtensorMap* tmC, uint8_t* sOut, int M,
                         int N, int m_pairs, int n_tiles, int total, float4* __restrict__ partials, int32_t* flags) {
    volatile int32_t* abort = &bars->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3;  // the TMEM lanes (rows) this warp may read
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    // this warp's two staging blocks; row `lane` at 64 bytes, its 16-byte
    // pieces permuted by the 64-byte swizzle the output tensor map applies
    const uint32_t out0 = smem_u32(sOut + (warp - 2) * 2 * kOutBlockBytes) + uint32_t(lane * 64);
    const uint32_t swz = uint32_t((lane >> 1) & 3);
    const int cl = int(blockIdx.x >> 1), ncl = int(gridDim.x >> 1);
    int buf = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = cl; t < total; t += ncl) {
        int mp, n;
        tile_coords(t, m_pairs, n_tiles, mp, n);
        const int m = 2 * mp + int(rank);
        const bool ready = wait_phase(&bars->tfull[acc], acc_phase, abort);
        if (!__all_sync(0xffffffffu, ready)) {
            give_up(abort, flags);
            break;
        }
        tc_fence_after();
        const int row0 = m * kBM + quarter * 32;
        const int row = row0 + lane;
        LseAcc st = lse_empty();
        float mx = -INFINITY;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
            uint32_t r[32];
            __syncwarp();  // tcgen05.ld is warp-collective: reconverge after the per-lane branches below
            tmem_ld32(tmem + uint32_t(acc * kBN + c * 32) + lane_off, r);
            if (c == kBN / 32 - 1) {  // this CTA's rows are read out: tell the even CTA's MMA thread
                tc_fence_before();
                __syncwarp();
                if (lane == 0) remote_arrive(peer_addr(&bars->tempty[acc], 0));
            }
            const int col0 = n * kBN + c * 32;
            if (col0 >= N) continue;  // the same for the whole warp
            uint4 v[4];
            uint32_t* w = reinterpret_cast<uint32_t*>(v);
#pragma unroll
            for (int j = 0; j < 16; ++j) w[j] = pack_bf16x2(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
            if (row < M) {
                if (col0 + 32 <= N) {
                    fold_vectors<4>(st, mx, v);
                } else {
                    const acrl_bf16* h = reinterpret_cast<const acrl_bf16*>(v);
                    for (int j = 0; j < N - col0; ++j) fold_scalar(st, mx, bf16_to_float(h[j]));
                }
            }
            // stage the block and store it with one TMA copy, which leaves out
            // the rows at or beyond M and the columns at or beyond N
            if (lane == 0) bulk_wait_read<1>();  // the store that last read this buffer is done
            __syncwarp();
            const uint32_t dst = out0 + uint32_t(buf * kOutBlockBytes);
#pragma unroll
            for (int q = 0; q < 4; ++q) st_shared16(dst + ((uint32_t(q) ^ swz) << 4), v[q]);
            fence_async_shared();
            __syncwarp();
            if (lane == 0 && row0 < M)
                tma_store_2d(tmC, sOut + (warp - 2) * 2 * kOutBlockBytes + buf * kOutBlockBytes, col0, row0);
            buf ^= 1;
        }
        if (row < M) partials[int64_t(n) * M + row] = make_float4(mx, st.U, st.s0, st.s1);
        __syncwarp();
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
    }
    if (lane == 0) bulk_wait_all();  // the staging blocks stay valid until every store has completed
    __syncwarp();
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    lmhead_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const __grid_constant__ CUtensorMap tmC, int M, int N, int K, float4* __restrict__ partials,
                  int32_t* flags) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sB = base;
    uint8_t* sA = base + kStages * kBBytes;
    uint8_t* sOut = base + kStages * kStageBytes;
    Barriers* bars = reinterpret_cast<Barriers*>(sOut + kOutBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const int m_tiles = (M + kBM - 1) / kBM, n_tiles = (N + kBN - 1) / kBN;
    const int m_pairs = (m_tiles + 1) / 2;
    const int total = m_pairs * n_tiles;  // tiles of 256 x 256 (a pair of row tiles x one column tile)
    const int k_iters = (K + kBK - 1) / kBK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&bars->full[s], 1);
            mbar_init(&bars->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->tfull[b], 1);
            mbar_init(&bars->tempty[b], 8);
        }
        mbar_init(&bars->mma_done, 1);
        bars->abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmC)) : "memory");
    }
    if (warp == 2) {  // one warp of each CTA of the pair allocates, together
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&bars->tmem_base)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers are initialised before either signals the other
    tc_fence_after();
    const uint32_t tmem = bars->tmem_base;

    if (warp == 0) {
        if (lane == 0) producer(&tmA, &tmB, sA, sB, bars, rank, m_pairs, n_tiles, total, k_iters, flags);
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) mma_issuer(sA, sB, bars, tmem, total, k_iters, flags);
    } else {
        epilogue(bars, tmem, rank, &tmC, sOut, M, N, m_pairs, n_tiles, total, partials, flags);
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // no CTA frees its TMEM or leaves while the pair may still touch it
    if (warp == 2) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

// Merge of the per-tile states of each row: lse, logp and entropy.  Eight
// lanes per row, lane j folding tiles j, j+8, ... in order, then a fixed
// butterfly over the eight (deterministic); partials are [n_tiles][M].
constexpr int kMergeLanes = 8;

__global__ void lmhead_merge_kernel(const float4* __restrict__ partials, const acrl_bf16* __restrict__ logits, int M,
                                    int N, int64_t ldl, int n_tiles, const int32_t* __restrict__ ids,
                                    const uint8_t* __restrict__ mask, float* __restrict__ lse, float* __restrict__ logp,
                                    float* __restrict__ ent, int32_t* flags) {
    const int64_t g = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    const int row = int(g / kMergeLanes), sub = int(g % kMergeLanes);
    if (row >= M) return;  // the row's eight lanes leave together
    if (mask && mask[row] == 0) {
        if (sub == 0) lse[row] = logp[row] = ent[row] = 0.f;
        return;
    }
    LseAcc acc = lse_empty();
    float mx = -INFINITY;
#pragma unroll 1  // tiles
    for (int n = sub; n < n_tiles; n += kMergeLanes) {
        const float4 p = partials[int64_t(n) * M + row];
        acc = lse_merge(acc, LseAcc{p.y, p.z, p.w});
        mx = fmaxf(mx, p.x);
    }
    static_assert(kMergeLanes >= 2 && kMergeLanes <= 16 && (kMergeLanes & (kMergeLanes - 1)) == 0, "lanes per row");
    const unsigned group = ((1u << kMergeLanes) - 1u) << (threadIdx.x & 31 & ~(kMergeLanes - 1));
#pragma unroll
    for (int m = kMergeLanes / 2; m >= 1; m >>= 1) {
        const LseAcc o{__shfl_xor_sync(group, acc.U, m), __shfl_xor_sync(group, acc.s0, m),
                       __shfl_xor_sync(group, acc.s1, m)};
        acc = lse_merge(acc, o);
        mx = fmaxf(mx, __shfl_xor_sync(group, mx, m));
    }
    if (sub == 0) row_outputs(acc, mx, logits + int64_t(row) * ldl, N, ids[row], lse, logp, ent, row, flags);
}

acrl_status launch_merge(const float4* partials, const acrl_bf16* logits, int64_t M, int64_t N, int64_t ldl,
                         const int32_t* ids, const uint8_t* mask, float* lse, float* logp, float* entropy,
                         int32_t* flags, cudaStream_t s) {
    const int threads = 256, rows_per_block = threads / kMergeLanes;
    lmhead_merge_kernel<<<unsigned((M + rows_per_block - 1) / rows_per_block), threads, 0, s>>>(
        partials, logits, int(M), int(N), ldl, int((N + kBN - 1) / kBN), ids, mask, lse, logp, entropy, flags);
    return launch_status();
}

bool encode_map(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols, uint64_t ld, uint32_t box_rows,
                uint32_t box_cols, CUtensorMapSwizzle swizzle) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || fn == nullptr)
        return false;
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {ld * 2};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor maps, shared-memory opt-in and the persistent launch (clusters of two
// CTAs, one CTA per SM, fewer if there are fewer tiles).  Arguments, including
// where the operands live, are checked by the callers.
acrl_status launch_lmhead(const acrl_bf16* hidden, int64_t M, int64_t K, int64_t ldh, const acrl_bf16* weight,
                          int64_t N, int64_t ldw, acrl_bf16* logits, int64_t ldl, float4* partials, int32_t* flags,
                          cudaStream_t s) {
    CUtensorMap tmA, tmB, tmC;
    if (!encode_map(&tmA, hidden, uint64_t(M), uint64_t(K), uint64_t(ldh), kBM, kBK, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_map(&tmB, weight, uint64_t(N), uint64_t(K), uint64_t(ldw), kHalfBN, kBK, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_map(&tmC, logits, uint64_t(M), uint64_t(N), uint64_t(ldl), 32, 32, CU_TENSOR_MAP_SWIZZLE_64B))
        return ACRL_ERR_CUDA;
    if (cudaFuncSetAttribute(lmhead_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) != cudaSuccess)
        return ACRL_ERR_CUDA;
    // 256 x 256 tiles; as many clusters as can be resident at once
    const int64_t total = (((M + kBM - 1) / kBM + 1) / 2) * ((N + kBN - 1) / kBN);
    if (total > kMaxGrid / 2) return ACRL_ERR_INVALID_ARG;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * 1024, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = kSmemBytes;
    cfg.stream = s;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, lmhead_kernel, &cfg) != cudaSuccess || clusters < 1)
        return ACRL_ERR_CUDA;
    const int grid = int(2 * (total < clusters ? total : clusters));
    lmhead_kernel<<<grid, kThreads, kSmemBytes, s>>>(tmA, tmB, tmC, int(M), int(N), int(K), partials, flags);
    return launch_status();
}

// True when every pointer is device memory of the current device: not managed
// memory, not host memory and not a peer GPU's memory.  The GEMM's tensor maps
// are encoded over these pointers, and its TMA copies must stay within this
// GPU's own memory.  A failed query counts as "no" and leaves no error behind
// for a later launch check.
bool operands_on_current_device(std::initializer_list<const void*> ptrs) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    for (const void* p : ptrs) {
        cudaPointerAttributes a{};
        if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
            (void)cudaGetLastError();
            return false;
        }
        if (a.type != cudaMemoryTypeDevice || a.device != dev) return false;
    }
    return true;
}

}  // namespace
}  // namespace acrl

using namespace acrl;

extern "C" int64_t acrl_lmhead_workspace_bytes(int64_t M, int64_t N) {
    if (M < 0 || N < 1) return -1;
    return ((N + kBN - 1) / kBN) * M * int64_t(sizeof(float4));
}

extern "C" acrl_status acrl_lmhead_logits_stats(const acrl_bf16* hidden, int64_t M, int64_t K, int64_t ldh,
                                                const acrl_bf16* weight, int64_t N, int64_t ldw, acrl_bf16* logits,
                                                int64_t ldl, float* partials, int32_t* dev_flags,
                                                acrl_stream stream) {
    if (M < 0 || K < 1 || N < 1 || M > kMaxGrid || N > kMaxGrid || K > kMaxGrid) return ACRL_ERR_INVALID_ARG;
    if (ldh < K || ldw < K || ldl < N || (ldh & 7) || (ldw & 7) || (ldl & 7)) return ACRL_ERR_INVALID_ARG;
    if (!dev_flags) return ACRL_ERR_INVALID_ARG;
    if (M == 0) return ACRL_OK;
    if (!hidden || !weight || !logits || !partials) return ACRL_ERR_INVALID_ARG;
    if (!aligned16(hidden) || !aligned16(weight) || !aligned16(logits) || !aligned16(partials))
        return ACRL_ERR_INVALID_ARG;
    if (!operands_on_current_device({hidden, weight, logits})) return ACRL_ERR_INVALID_ARG;
    return launch_lmhead(hidden, M, K, ldh, weight, N, ldw, logits, ldl, reinterpret_cast<float4*>(partials),
                                 dev_flags, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" acrl_status acrl_lmhead_merge(const float* partials, const acrl_bf16* logits, int64_t M, int64_t N,
                                         int64_t ldl, const int32_t* ids, const uint8_t* mask, float* lse, float* logp,
                                         float* entropy, int32_t* dev_flags, acrl_stream stream) {
    if (M < 0 || N < 1 || N > kMaxVocab || M > kMaxGrid || ldl < N) return ACRL_ERR_INVALID_ARG;
    if (!dev_flags) return ACRL_ERR_INVALID_ARG;
    if (M == 0) return ACRL_OK;
    if (!partials || !logits || !ids || !lse || !logp || !entropy) return ACRL_ERR_INVALID_ARG;
    if (!aligned16(partials)) return ACRL_ERR_INVALID_ARG;
    return launch_merge(reinterpret_cast<const float4*>(partials), logits, M, N, ldl, ids, mask, lse, logp, entropy,
                        dev_flags, reinterpret_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// acrl_lmhead_stats_noalloc: the same GEMM + merge with the per-tile partial
// states kept in a fixed device array of this library instead of a
// caller-provided workspace, for callers that cannot allocate device memory.
// ---------------------------------------------------------------------------

#include <mutex>

namespace acrl {
namespace {

constexpr int64_t kNoallocScratchBytes = ACRL_LMHEAD_NOALLOC_SCRATCH_BYTES;

// Every GPU that loads this library holds this array until the process exits.
// Its contents are whatever the last call left: the GEMM writes every entry
// the merge then reads, so nothing needs clearing between calls.
static __device__ __align__(256) float4 g_noalloc_partials[kNoallocScratchBytes / sizeof(float4)];

constexpr int kNoallocMaxDevices = 64;
std::mutex g_noalloc_mutex;
float4* g_noalloc_ptr[kNoallocMaxDevices] = {};

// Device address of g_noalloc_partials on the current device, looked up once
// per device (host code must not pass the symbol itself to a kernel).
float4* noalloc_scratch(int dev) {
    if (dev < 0 || dev >= kNoallocMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (g_noalloc_ptr[dev] == nullptr) {
        float4* ptr = nullptr;
        if (cudaGetSymbolAddress(reinterpret_cast<void**>(&ptr), g_noalloc_partials) != cudaSuccess) return nullptr;
        g_noalloc_ptr[dev] = ptr;
    }
    return g_noalloc_ptr[dev];
}

}  // namespace
}  // namespace acrl

extern "C" acrl_status acrl_lmhead_stats_noalloc(const acrl_bf16* hidden, int64_t M, int64_t K, int64_t ldh,
                                                 const acrl_bf16* weight, int64_t N, int64_t ldw, acrl_bf16* logits,
                                                 int64_t ldl, const int32_t* ids, const uint8_t* mask, float* lse,
                                                 float* logp, float* entropy, int32_t* dev_flags,
                                                 acrl_stream stream) {
    if (M < 0 || K < 1 || N < 1 || M > kMaxGrid || N > kMaxVocab || K > kMaxGrid) return ACRL_ERR_INVALID_ARG;
    if (ldh < K || ldw < K || ldl < N || (ldh & 7) || (ldw & 7) || (ldl & 7)) return ACRL_ERR_INVALID_ARG;
    if (!dev_flags) return ACRL_ERR_INVALID_ARG;
    if (((N + kBN - 1) / kBN) * M * int64_t(sizeof(float4)) > kNoallocScratchBytes) return ACRL_ERR_SCRATCH_TOO_SMALL;
    if (M == 0) return ACRL_OK;
    if (!hidden || !weight || !logits || !ids || !lse || !logp || !entropy) return ACRL_ERR_INVALID_ARG;
    if (!aligned16(hidden) || !aligned16(weight) || !aligned16(logits)) return ACRL_ERR_INVALID_ARG;
    if (!operands_on_current_device({hidden, weight, logits})) return ACRL_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ACRL_ERR_CUDA;
    float4* partials = noalloc_scratch(dev);
    if (partials == nullptr) return ACRL_ERR_CUDA;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const acrl_status st = launch_lmhead(hidden, M, K, ldh, weight, N, ldw, logits, ldl, partials, dev_flags, s);
    if (st != ACRL_OK) return st;
    return launch_merge(partials, logits, M, N, ldl, ids, mask, lse, logp, entropy, dev_flags, s);
}

