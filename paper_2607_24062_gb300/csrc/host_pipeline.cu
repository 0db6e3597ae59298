// The host-buffer pipeline: one on-policy pass over a batch whose inputs and
// outputs live in host memory, built from the library's own entry points.
// Host code only (copies, events and the calls of the other files); every
// step of the computation runs in those calls' kernels.
//
// Streams: the caller's stream runs the kernels; `up` carries the uploads and
// `down` the downloads.  Events order each reuse of a device buffer:
//   up[c]     logits chunk c has landed          -> statistics of chunk c
//   used[c]   the gradient call has read chunk c -> next step's upload of c
//   small[p]  small inputs of slot p have landed -> the step's first kernel
//   done[p]   the step that used slot p is done  -> upload two steps later
//   grad[c]   gradient chunk c written           -> its download
//   freed[r]  ring slot r downloaded             -> the next gradient into r
//   fin       the step's last download           -> the caller's stream
#include <cstdint>
#include <new>

#include <cuda_runtime.h>

#include "acrl.h"
#include "acrl_host.h"

namespace acrl {
namespace {

constexpr int kMaxChunks = 4096;
constexpr int kRing = 4;  // gradient chunks held on the device at once

int64_t align256(int64_t x) { return (x + 255) & ~int64_t(255); }

// Offsets of every buffer in the workspace; `total` is its size.
struct Layout {
    int64_t logits, ring, lse, logp, ent, lr, d, weight, coef, ent_coef, token_loss, adv, alpha, seq, grp, batch,
        loss, chunk_loss;
    int64_t ids[2], mask[2], mu[2], rewards[2], so[2], go[2];
    int64_t rows_max, total;
};

Layout layout(int64_t T, int64_t ld, int32_t S, int32_t Gn, int32_t chunks) {
    Layout L{};
    int64_t o = 0;
    auto take = [&o](int64_t bytes) {
        const int64_t at = o;
        o += align256(bytes);
        return at;
    };
    L.rows_max = (T + chunks - 1) / chunks;
    const int ring = chunks < kRing ? chunks : kRing;
    L.logits = take(T * ld * 2);
    L.ring = take(int64_t(ring) * L.rows_max * ld * 2);
    L.lse = take(T * 4);
    L.logp = take(T * 4);
    L.ent = take(T * 4);
    L.lr = take(T * 4);
    L.d = take(T * 4);
    L.weight = take(T * 4);
    L.coef = take(T * 4);
    L.ent_coef = take(T * 4);
    L.token_loss = take(T * 4);
    L.adv = take(int64_t(S) * 4);
    L.alpha = take(int64_t(S) * 4);
    L.seq = take(int64_t(S) * int64_t(sizeof(acrl_seq_stats)));
    L.grp = take(int64_t(Gn) * int64_t(sizeof(acrl_group_stats)));
    L.batch = take(sizeof(acrl_batch_stats));
    L.loss = take(4);
    L.chunk_loss = take(4);
    for (int p = 0; p < 2; ++p) {
        L.ids[p] = take(T * 4);
        L.mask[p] = take(T);
        L.mu[p] = take(T * 4);
        L.rewards[p] = take(int64_t(S) * 4);
        L.so[p] = take((int64_t(S) + 1) * 8);
        L.go[p] = take((int64_t(Gn) + 1) * 4);
    }
    L.total = o;
    return L;
}

}  // namespace
}  // namespace acrl

using namespace acrl;

struct acrl_host_pipeline {
    int64_t T, V, ld;
    int32_t S, Gn, chunks, ring;
    int64_t step;
    bool begun;      // begin enqueued, finish not yet
    bool has_mask;   // the begun step's mask was given
    char* ws;
    Layout L;
    cudaStream_t up, down;
    cudaEvent_t* ev;  // up[chunks], used[chunks], grad[chunks], freed[ring], small[2], done[2], fin
    cudaEvent_t* ev_up() { return ev; }
    cudaEvent_t* ev_used() { return ev + chunks; }
    cudaEvent_t* ev_grad() { return ev + 2 * chunks; }
    cudaEvent_t* ev_freed() { return ev + 3 * chunks; }
    cudaEvent_t* ev_small() { return ev + 3 * chunks + ring; }
    cudaEvent_t* ev_done() { return ev + 3 * chunks + ring + 2; }
    cudaEvent_t& ev_fin() { return ev[3 * chunks + ring + 4]; }
    int n_events() const { return 3 * chunks + ring + 5; }
    template <class X>
    X* at(int64_t off) {
        return reinterpret_cast<X*>(ws + off);
    }
    int64_t r0(int c) const { return T * c / chunks; }
};

namespace {

void release(acrl_host_pipeline* pl, int events_made) {
    for (int i = 0; i < events_made; ++i) cudaEventDestroy(pl->ev[i]);
    if (pl->up) cudaStreamDestroy(pl->up);
    if (pl->down) cudaStreamDestroy(pl->down);
    delete[] pl->ev;
    delete pl;
}

}  // namespace

extern "C" int64_t acrl_host_pipeline_workspace_bytes(int64_t T, int64_t ld, int32_t S, int32_t Gn, int32_t chunks) {
    if (T < 1 || ld < 1 || S < 1 || Gn < 1 || chunks < 1 || chunks > kMaxChunks) return -1;
    return layout(T, ld, S, Gn, chunks).total;
}

extern "C" acrl_status acrl_host_pipeline_create(acrl_host_pipeline** pipeline, int64_t T, int64_t V, int64_t ld,
                                                 int32_t S, int32_t Gn, int32_t chunks, void* workspace,
                                                 int64_t workspace_bytes) {
    if (!pipeline) return ACRL_ERR_INVALID_ARG;
    *pipeline = nullptr;
    if (T < 1 || V < 1 || V > kMaxVocab || ld < V || (ld & 7) || S < 1 || Gn < 1 || chunks < 1 ||
        chunks > kMaxChunks || int64_t(chunks) > T)
        return ACRL_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < layout(T, ld, S, Gn, chunks).total)
        return ACRL_ERR_INVALID_ARG;
    acrl_host_pipeline* pl = new (std::nothrow) acrl_host_pipeline{};
    if (!pl) return ACRL_ERR_CUDA;
    pl->T = T;
    pl->V = V;
    pl->ld = ld;
    pl->S = S;
    pl->Gn = Gn;
    pl->chunks = chunks;
    pl->ring = chunks < kRing ? chunks : kRing;
    pl->ws = static_cast<char*>(workspace);
    pl->L = layout(T, ld, S, Gn, chunks);
    pl->ev = new (std::nothrow) cudaEvent_t[pl->n_events()];
    if (!pl->ev) {
        delete pl;
        return ACRL_ERR_CUDA;
    }
    if (cudaStreamCreateWithFlags(&pl->up, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&pl->down, cudaStreamNonBlocking) != cudaSuccess) {
        release(pl, 0);
        return ACRL_ERR_CUDA;
    }
    for (int i = 0; i < pl->n_events(); ++i)
        if (cudaEventCreateWithFlags(&pl->ev[i], cudaEventDisableTiming) != cudaSuccess) {
            release(pl, i);
            return ACRL_ERR_CUDA;
        }
    *pipeline = pl;
    return ACRL_OK;
}

extern "C" acrl_status acrl_host_pipeline_begin(acrl_host_pipeline* pl, const acrl_bf16* logits, const int32_t* ids,
                                                const uint8_t* mask, const float* logp_mu, const float* rewards,
                                                const int64_t* seq_offsets, const int32_t* group_offsets,
                                                int32_t* dev_flags, acrl_stream stream) {
    if (!pl || pl->begun || !logits || !ids || !logp_mu || !rewards || !seq_offsets || !group_offsets || !dev_flags)
        return ACRL_ERR_INVALID_ARG;
    cudaStream_t comp = reinterpret_cast<cudaStream_t>(stream);
    const Layout& L = pl->L;
    const int64_t T = pl->T, ld = pl->ld, row_bytes = ld * 2;
    const int S = pl->S, Gn = pl->Gn, C = pl->chunks, slot = int(pl->step & 1);
    auto ok = [](cudaError_t e) { return e == cudaSuccess; };

    // uploads: the small inputs into this step's slot, then the logits chunk by chunk
    int32_t* d_ids = pl->at<int32_t>(L.ids[slot]);
    uint8_t* d_mask = mask ? pl->at<uint8_t>(L.mask[slot]) : nullptr;
    float* d_mu = pl->at<float>(L.mu[slot]);
    int64_t* d_so = pl->at<int64_t>(L.so[slot]);
    int32_t* d_go = pl->at<int32_t>(L.go[slot]);
    acrl_bf16* d_logits = pl->at<acrl_bf16>(L.logits);
    if (!ok(cudaStreamWaitEvent(pl->up, pl->ev_done()[slot], 0)) ||
        !ok(cudaMemcpyAsync(d_ids, ids, T * 4, cudaMemcpyHostToDevice, pl->up)) ||
        (mask && !ok(cudaMemcpyAsync(d_mask, mask, T, cudaMemcpyHostToDevice, pl->up))) ||
        !ok(cudaMemcpyAsync(d_mu, logp_mu, T * 4, cudaMemcpyHostToDevice, pl->up)) ||
        !ok(cudaMemcpyAsync(pl->at<float>(L.rewards[slot]), rewards, int64_t(S) * 4, cudaMemcpyHostToDevice,
                            pl->up)) ||
        !ok(cudaMemcpyAsync(d_so, seq_offsets, (int64_t(S) + 1) * 8, cudaMemcpyHostToDevice, pl->up)) ||
        !ok(cudaMemcpyAsync(d_go, group_offsets, (int64_t(Gn) + 1) * 4, cudaMemcpyHostToDevice, pl->up)) ||
        !ok(cudaEventRecord(pl->ev_small()[slot], pl->up)))
        return ACRL_ERR_CUDA;
    for (int c = 0; c < C; ++c) {
        const int64_t r0 = pl->r0(c), rows = pl->r0(c + 1) - r0;
        if (!ok(cudaStreamWaitEvent(pl->up, pl->ev_used()[c], 0)) ||
            !ok(cudaMemcpyAsync(d_logits + r0 * ld, logits + r0 * ld, rows * row_bytes, cudaMemcpyHostToDevice,
                                pl->up)) ||
            !ok(cudaEventRecord(pl->ev_up()[c], pl->up)))
            return ACRL_ERR_CUDA;
    }

    // statistics, chunk by chunk as the logits land, then the discrepancy call
    float* lse = pl->at<float>(L.lse);
    float* logp = pl->at<float>(L.logp);
    float* ent = pl->at<float>(L.ent);
    if (!ok(cudaStreamWaitEvent(comp, pl->ev_small()[slot], 0))) return ACRL_ERR_CUDA;
    for (int c = 0; c < C; ++c) {
        const int64_t r0 = pl->r0(c), rows = pl->r0(c + 1) - r0;
        if (!ok(cudaStreamWaitEvent(comp, pl->ev_up()[c], 0))) return ACRL_ERR_CUDA;
        const acrl_status st = acrl_token_stats(d_logits + r0 * ld, rows, pl->V, ld, d_ids + r0,
                                                d_mask ? d_mask + r0 : nullptr, lse + r0, logp + r0, ent + r0,
                                                dev_flags, stream);
        if (st != ACRL_OK) return st;
    }
    const acrl_status st = acrl_seq_discrepancy(logp, d_mu, d_mask, T, d_so, S, d_go, Gn, ent, pl->at<float>(L.lr),
                                                pl->at<float>(L.d), pl->at<acrl_seq_stats>(L.seq),
                                                pl->at<acrl_group_stats>(L.grp), pl->at<acrl_batch_stats>(L.batch),
                                                dev_flags, stream);
    if (st != ACRL_OK) return st;
    pl->begun = true;
    pl->has_mask = mask != nullptr;
    return ACRL_OK;
}

extern "C" acrl_status acrl_host_pipeline_finish(acrl_host_pipeline* pl, const acrl_params* p,
                                                 acrl_controller_state* state, acrl_bf16* grad, float* loss,
                                                 int32_t* dev_flags, acrl_stream stream) {
    if (!pl || !pl->begun || !params_ok(p) || !state || !grad || !loss || !dev_flags) return ACRL_ERR_INVALID_ARG;
    pl->begun = false;
    cudaStream_t comp = reinterpret_cast<cudaStream_t>(stream);
    const Layout& L = pl->L;
    const int64_t T = pl->T, ld = pl->ld, row_bytes = ld * 2;
    const int S = pl->S, Gn = pl->Gn, C = pl->chunks, slot = int(pl->step & 1);
    pl->step += 1;
    auto ok = [](cudaError_t e) { return e == cudaSuccess; };
    int32_t* d_ids = pl->at<int32_t>(L.ids[slot]);
    uint8_t* d_mask = pl->has_mask ? pl->at<uint8_t>(L.mask[slot]) : nullptr;
    int64_t* d_so = pl->at<int64_t>(L.so[slot]);
    int32_t* d_go = pl->at<int32_t>(L.go[slot]);
    acrl_bf16* d_logits = pl->at<acrl_bf16>(L.logits);
    float* lse = pl->at<float>(L.lse);
    float* ent = pl->at<float>(L.ent);

    // advantages and controller
    acrl_seq_stats* seq = pl->at<acrl_seq_stats>(L.seq);
    float* adv = pl->at<float>(L.adv);
    float* coef = pl->at<float>(L.coef);
    float* ent_coef = p->entropy_coeff > 0.f ? pl->at<float>(L.ent_coef) : nullptr;
    acrl_status st = acrl_grpo_advantage(pl->at<float>(L.rewards[slot]), d_go, Gn, S, p, adv, dev_flags, stream);
    if (st == ACRL_OK)
        st = acrl_controller_step(state, p, pl->at<float>(L.lr), d_mask, T, d_so, S, d_go, Gn, seq,
                                  pl->at<acrl_group_stats>(L.grp), pl->at<acrl_batch_stats>(L.batch), adv,
                                  pl->at<float>(L.weight), coef, pl->at<float>(L.alpha), ent_coef, dev_flags, stream);
    if (st != ACRL_OK) return st;

    // gradient, chunk by chunk into the ring, each chunk downloaded as soon as it is written
    float* token_loss = pl->at<float>(L.token_loss);
    acrl_bf16* ring = pl->at<acrl_bf16>(L.ring);
    for (int c = 0; c < C; ++c) {
        const int64_t r0 = pl->r0(c), rows = pl->r0(c + 1) - r0;
        const int r = c % pl->ring;
        acrl_bf16* g = ring + int64_t(r) * L.rows_max * ld;
        if (!ok(cudaStreamWaitEvent(comp, pl->ev_freed()[r], 0))) return ACRL_ERR_CUDA;
        st = acrl_loss_grad_logits(d_logits + r0 * ld, rows, pl->V, ld, d_ids + r0, d_mask ? d_mask + r0 : nullptr,
                                   lse + r0, nullptr, coef + r0, ent_coef ? ent + r0 : nullptr,
                                   ent_coef ? ent_coef + r0 : nullptr, p->clip_eps, g, token_loss + r0,
                                   pl->at<float>(L.chunk_loss), dev_flags, stream);
        if (st != ACRL_OK) return st;
        if (!ok(cudaEventRecord(pl->ev_used()[c], comp)) || !ok(cudaEventRecord(pl->ev_grad()[c], comp)) ||
            !ok(cudaStreamWaitEvent(pl->down, pl->ev_grad()[c], 0)) ||
            !ok(cudaMemcpyAsync(grad + r0 * ld, g, rows * row_bytes, cudaMemcpyDeviceToHost, pl->down)) ||
            !ok(cudaEventRecord(pl->ev_freed()[r], pl->down)))
            return ACRL_ERR_CUDA;
    }

    // the loss, downloaded last; the caller's stream waits for every download of the step
    float* d_loss = pl->at<float>(L.loss);
    st = acrl_reduce_loss(token_loss, T, d_loss, stream);
    if (st != ACRL_OK) return st;
    if (!ok(cudaEventRecord(pl->ev_fin(), comp)) || !ok(cudaStreamWaitEvent(pl->down, pl->ev_fin(), 0)) ||
        !ok(cudaMemcpyAsync(loss, d_loss, 4, cudaMemcpyDeviceToHost, pl->down)) ||
        !ok(cudaEventRecord(pl->ev_fin(), pl->down)) || !ok(cudaStreamWaitEvent(comp, pl->ev_fin(), 0)) ||
        !ok(cudaEventRecord(pl->ev_done()[slot], comp)))
        return ACRL_ERR_CUDA;
    return ACRL_OK;
}

extern "C" acrl_status acrl_host_pipeline_step(acrl_host_pipeline* pl, const acrl_params* p,
                                               acrl_controller_state* state, const acrl_bf16* logits,
                                               const int32_t* ids, const uint8_t* mask, const float* logp_mu,
                                               const float* rewards, const int64_t* seq_offsets,
                                               const int32_t* group_offsets, acrl_bf16* grad, float* loss,
                                               int32_t* dev_flags, acrl_stream stream) {
    if (!pl || pl->begun || !params_ok(p) || !state || !grad || !loss) return ACRL_ERR_INVALID_ARG;
    const acrl_status st =
        acrl_host_pipeline_begin(pl, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, dev_flags, stream);
    if (st != ACRL_OK) return st;
    return acrl_host_pipeline_finish(pl, p, state, grad, loss, dev_flags, stream);
}

extern "C" acrl_batch_stats* acrl_host_pipeline_batch_stats(acrl_host_pipeline* pl) {
    return pl ? pl->at<acrl_batch_stats>(pl->L.batch) : nullptr;
}

extern "C" acrl_status acrl_host_pipeline_destroy(acrl_host_pipeline* pl) {
    if (!pl) return ACRL_ERR_INVALID_ARG;
    const bool synced = cudaStreamSynchronize(pl->up) == cudaSuccess && cudaStreamSynchronize(pl->down) == cudaSuccess;
    release(pl, pl->n_events());
    return synced ? ACRL_OK : ACRL_ERR_CUDA;
}
