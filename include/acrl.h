/*
 * acrl.h -- C ABI of the ACRL vocabulary-wide hot path on one GB300 (sm_103a).
 *
 * ACRL: "Adaptive Control of Training-Inference Discrepancy for Stable
 * Reinforcement Learning" (arXiv 2607.24062).  One RL update step runs, per
 * token row of the training policy pi's logits, a log-softmax with the
 * sampled token's log-prob and the entropy; combines them with the rollout
 * engine's cached log-probs of mu into the discrepancy statistics; turns those
 * into importance weights through the adaptive controller; and produces the
 * gradient of the policy loss with respect to the logits.
 *
 * Conventions shared by every call:
 *   - Pointers documented "device" must be device memory of the current CUDA
 *     device (managed memory is accepted too, except by the LM-head calls,
 *     whose tensor-core copies need plain device memory of the current
 *     device: they check this on the host).  The caller owns every buffer; the library
 *     allocates no device memory and keeps no global state, except the fixed
 *     scratch array of acrl_lmhead_stats_noalloc (documented there).  The
 *     host-buffer pipeline's handle owns two streams and its events, made by
 *     acrl_host_pipeline_create and released by acrl_host_pipeline_destroy.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream) except acrl_read_flags and acrl_check_flags,
 *     which synchronise it.
 *   - Problems visible on the host (null required pointers, negative sizes,
 *     misalignment, hyper-parameters out of range) return
 *     ACRL_ERR_INVALID_ARG before anything is launched.
 *   - Problems that depend on device data (a sampled id outside [0, V), a
 *     non-finite logit, inconsistent offsets, X <= 0) never trap: the kernel
 *     ORs an ACRL_FLAG_* bit into the caller's device word `dev_flags` and
 *     writes the documented defined value.  acrl_read_flags fetches the word;
 *     acrl_check_flags turns it into a status.
 *   - A failed launch returns ACRL_ERR_CUDA.  Nothing is ever printed.
 *   - bf16 arrays are IEEE bfloat16 bit patterns (acrl_bf16), row-major with a
 *     row stride `ld` in elements; the base pointer must be 16-byte aligned
 *     and ld a multiple of 8, so every row starts on a 16-byte boundary.
 *   - Sizes: 1 <= V <= 2^30 (column indices stay in 32-bit range); the row
 *     count T is 64-bit (T and T * ld may exceed 2^32); a response holds
 *     fewer than 2^31 tokens (its count is an int32).  Larger V is
 *     ACRL_ERR_INVALID_ARG.
 *
 * Notation: T token rows, V vocabulary size, S responses (sequences),
 * Gn prompts (groups), m_t in {0,1} the response mask, a_t the sampled id.
 */
#ifndef ACRL_H_
#define ACRL_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ACRL_ABI_VERSION 2

typedef uint16_t acrl_bf16;                 /* IEEE bfloat16 bit pattern */
typedef struct CUstream_st* acrl_stream;    /* identical to cudaStream_t */

typedef enum {
    ACRL_OK = 0,
    ACRL_ERR_INVALID_ARG = 1,
    ACRL_ERR_CUDA = 2,
    ACRL_ERR_NOT_IMPLEMENTED = 3,
    ACRL_ERR_DEVICE_FLAGS = 4,      /* acrl_check_flags: a device flag is set */
    ACRL_ERR_SCRATCH_TOO_SMALL = 5  /* acrl_lmhead_stats_noalloc: the problem needs more
                                       scratch than ACRL_LMHEAD_NOALLOC_SCRATCH_BYTES */
} acrl_status;

/* Bits of the device flags word. */
#define ACRL_FLAG_BAD_ID      0x1   /* a_t < 0 or a_t >= V on a valid row      */
#define ACRL_FLAG_NONFINITE   0x2   /* a valid row held a NaN or an infinity   */
#define ACRL_FLAG_BAD_OFFSETS 0x4   /* seq/group offsets not monotone or not covering */
#define ACRL_FLAG_X_NONPOS    0x8   /* ACRL mode with a reference X <= 0       */
#define ACRL_FLAG_TIMEOUT     0x10  /* a bounded wait inside a kernel (the tensor-core
                                       pipeline, or the bulk copy of the lse-recompute
                                       gradient) gave up after its time limit: that call's
                                       outputs are invalid */

/* Importance-weight mode. */
typedef enum {
    ACRL_MODE_NONE = 0,   /* plain GRPO (Eq. grpo_objective): w = 1             */
    ACRL_MODE_TIS = 1,    /* token-level truncated IS (Eq. TIS): min(pi/mu, C)  */
    ACRL_MODE_MIS = 2,    /* sequence-level masked IS (Eq. MIS): rho_i 1{rho_i<=C} */
    ACRL_MODE_ACRL = 3,   /* Eq. ACRL: min((pi/mu)^alpha, C)                    */
    ACRL_MODE_ACRL_CONTINUOUS = 4, /* Sec. 5.5 ablation, continuous reduction:
                                      alpha = -kappa sign(A), no Y/X comparison   */
    ACRL_MODE_ACRL_FALLBACK = 5    /* Sec. 5.5 ablation, fallback to GRPO: the ACRL
                                      alpha when Y > X, alpha = 0 (w = 1) otherwise */
} acrl_mode;

/* Which discrepancy plays Y in alpha = gamma sign(A) (1 - Y/X) (Sec. 4.1). */
typedef enum {
    ACRL_Y_GROUP = 0,     /* Y_g = (1/G) sum_i D_i over the prompt's responses (the formula) */
    ACRL_Y_SEQUENCE = 1,  /* Y = D_i, the response's own mean distance                       */
    ACRL_Y_BATCH = 2      /* Y = mean over prompts of Y_g (the step discrepancy)            */
} acrl_y_granularity;

typedef enum {
    ACRL_AGG_SEQ_MEAN_TOKEN_MEAN = 0, /* (1/Q)(1/G) sum_i (1/|a_i|) sum_t (Eq. grpo_objective) */
    ACRL_AGG_TOKEN_MEAN = 1           /* (1/N) sum over all valid tokens                      */
} acrl_agg;

typedef enum {
    ACRL_SINGLETON_MEAN0_STD1 = 0,    /* a prompt with one response: A = R */
    ACRL_SINGLETON_ZERO = 1           /* a prompt with one response: A = 0 */
} acrl_singleton_rule;

/* Hyper-parameters (host memory, read at call time).  64 bytes. */
typedef struct acrl_params {
    float   gamma;          /* control strength gamma > 0 (Sec. 4.1; 0.35 / 0.65 in Sec. 5.1) */
    float   C;              /* truncation cap C > 1 (Sec. 4.1; 3, or 5 in Sec. 5.3)           */
    float   clip_eps;       /* clip range eps in [0, 1) of Eq. grpo_objective                 */
    float   adv_eps;        /* added to the GRPO std, >= 0                                    */
    float   kappa;          /* |alpha| > 0 of ACRL_MODE_ACRL_CONTINUOUS (1 or 3 in Sec. 5.5)  */
    float   x_ema;          /* 0: X frozen once calibrated (the paper's method).  In (0, 1]:
                               after every later step X <- (1 - x_ema) X + x_ema Y_mean, the
                               moving-average X the Limitations section suggests           */
    float   entropy_coeff;  /* beta >= 0: entropy bonus -beta H_t / norm_t added to the loss
                               (the actor entropy_coeff of App. A; not part of Eq. ACRL)   */
    float   reserved;       /* must be 0 */
    int32_t mode;           /* acrl_mode                                                      */
    int32_t y_gran;         /* acrl_y_granularity                                             */
    int32_t agg;            /* acrl_agg                                                       */
    int32_t adv_ddof;       /* 0 or 1: degrees of freedom of the GRPO std                     */
    int32_t singleton_rule; /* acrl_singleton_rule                                            */
    int32_t calib_steps;    /* >= 1: batches averaged into X before it is frozen              */
    double  X_init;         /* > 0: use this X (as the paper's printed X); <= 0: calibrate    */
} acrl_params;

/* Controller state (device memory, caller-owned, 48 bytes).  Plain data: it
 * can be copied to the host and back to checkpoint and resume exactly. */
typedef struct acrl_controller_state {
    double  X;              /* reference discrepancy X (Sec. 4.1), valid once calibrated */
    double  calib_sum;      /* sum of Y_g over the prompts of the calibration batches    */
    int64_t calib_count;    /* number of prompts in calib_sum                            */
    int64_t step;           /* controller steps taken                                    */
    int32_t calib_done;     /* calibration batches seen                                  */
    int32_t calibrated;     /* 1 once X is fixed                                         */
    int32_t flags;          /* sticky OR of the flags this controller raised             */
    int32_t reserved;
} acrl_controller_state;

/* Per-response statistics (device memory, 64 bytes each). */
typedef struct acrl_seq_stats {
    int32_t n;              /* |a_i|: valid tokens of response i                          */
    int32_t group;          /* prompt index g(i)                                          */
    float   mean_d;         /* D_i = sum_d / n (0 when n = 0)                             */
    float   max_d;          /* max of d over valid tokens (0 when n = 0)                  */
    double  sum_d;          /* sum_t m_t d_t                                              */
    double  sum_d2;         /* sum_t m_t d_t^2                                            */
    double  sum_lr;         /* S_i = sum_t m_t lr_t = log rho_i of Eq. MIS                */
    double  sum_H;          /* sum_t m_t H_t (0 when no entropy was given)                */
    double  sum_w;          /* written by acrl_controller_step: sum_t m_t w_t             */
    int32_t n_trunc;        /* written by acrl_controller_step: truncated valid tokens    */
    float   alpha;          /* written by acrl_controller_step: alpha_i                   */
} acrl_seq_stats;

/* Per-prompt statistics (device memory, 24 bytes each). */
typedef struct acrl_group_stats {
    int32_t n_valid_seqs;   /* G_g: responses of the prompt with n_i > 0 */
    int32_t n_seqs;         /* all responses of the prompt              */
    int64_t n_tokens;       /* sum_i n_i                                */
    double  Y;              /* Y_g = (1/G_g) sum_i D_i (0 when G_g = 0)  */
} acrl_group_stats;

/* Whole-batch statistics (device memory, one struct, 104 bytes). */
typedef struct acrl_batch_stats {
    int64_t n_tokens;       /* N = sum_t m_t                                         */
    int32_t n_seqs_valid;   /* responses with n_i > 0                                */
    int32_t n_groups_valid; /* Q_eff: prompts with G_g > 0                           */
    double  d_mean;         /* token mean of d (the discrepancy curves of Sec. 5.1)  */
    double  d_max;
    double  d_std;          /* population std of d over valid tokens                 */
    double  Y_sum;          /* sum of Y_g over valid prompts                         */
    double  Y_mean;         /* Y_sum / Q_eff: the step discrepancy of Sec. 5.3       */
    double  H_mean;         /* token mean entropy                                    */
    double  lr_mean;        /* token mean log-ratio                                  */
    /* written by acrl_controller_step */
    double  X;              /* X in force this step (0 while still calibrating)      */
    double  trunc_frac;     /* fraction of valid tokens whose weight hit C (or MIS mask) */
    double  w_mean;         /* token mean weight                                     */
    double  alpha_mean;     /* mean alpha over valid responses                       */
} acrl_batch_stats;

/* ------------------------------------------------------------------------ */

const char* acrl_status_string(acrl_status s);
int32_t     acrl_abi_version(void);
/* sizeof of the ABI structs as compiled into the library, for binding checks:
 * 0 params, 1 controller state, 2 seq stats, 3 group stats, 4 batch stats. */
int64_t     acrl_struct_size(int32_t which);

/*
 * acrl_token_stats -- log-softmax statistics of pi per token row.
 * Defines, for each row t (Sec. 2: pi(a_t | q, a_<t) enters r, rho and d;
 * the entropy is the quantity tracked in Sec. 5.1):
 *     lse_t = log sum_j exp(z_tj),  logp_t = z_{t,a_t} - lse_t,
 *     H_t = -sum_j p_tj log p_tj,   p_tj = exp(z_tj - lse_t).
 *   logits  device bf16 [T, ld], the first V columns of each row are used.
 *   ids     device int32 [T] sampled token ids a_t.
 *   mask    device uint8 [T] response mask m_t, or NULL for all ones.
 *   lse, logp, entropy  device float [T] outputs (0 on rows with m_t = 0,
 *           whose logits are not read; NaN on a row with a non-finite logit,
 *           flag NONFINITE; logp = 0 with flag BAD_ID for an id outside [0,V)).
 *   dev_flags  device int32 word, bits ORed in.
 * Arithmetic: bf16 in, fp32 accumulation, one pass over the logits.
 */
acrl_status acrl_token_stats(const acrl_bf16* logits, int64_t T, int64_t V, int64_t ld,
                             const int32_t* ids, const uint8_t* mask,
                             float* lse, float* logp, float* entropy,
                             int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_seq_discrepancy -- training-inference discrepancy statistics.
 * Per token (Eq. TIS, Eq. distance_metric):
 *     lr_t = logp_pi_t - logp_mu_t,   d_t = |exp(logp_pi_t) - exp(logp_mu_t)|
 * (both 0 where m_t = 0).  Per response i over rows [seq_offsets[i],
 * seq_offsets[i+1]): n_i, D_i = mean d, S_i = sum lr, max d, sum d^2 and the
 * entropy sum.  Per prompt g over responses [group_offsets[g],
 * group_offsets[g+1]): G_g = responses with n_i > 0 and
 * Y_g = (1/G_g) sum_i D_i, the current discrepancy Y of Sec. 4.1.  Batch:
 * token mean/max/std of d, Y_sum, Y_mean, mean entropy and log-ratio.
 *   logp_pi   device float [T] log pi_old(a_t) (e.g. acrl_token_stats' logp).
 *   logp_mu   device float [T] the rollout engine's cached log mu(a_t).
 *   mask      device uint8 [T] or NULL.
 *   seq_offsets   device int64 [S+1], non-decreasing, 0 .. T.
 *   group_offsets device int32 [Gn+1], non-decreasing, 0 .. S.
 *   entropy   device float [T] or NULL.
 *   lr, d     device float [T] outputs.
 *   seq [S], grp [Gn], batch [1]  device outputs (the controller fields of
 *             seq and batch are written later by acrl_controller_step).
 * Offsets that break the rules above raise BAD_OFFSETS; the offending
 * response is treated as empty, and rows that no well-formed response covers
 * are not written (here, nor by acrl_controller_step): their lr, d, weight
 * and coef keep whatever the buffers held, so a caller that sees the flag
 * must discard the step.  Deterministic: fixed reduction order, fp64
 * accumulation.
 */
acrl_status acrl_seq_discrepancy(const float* logp_pi, const float* logp_mu, const uint8_t* mask,
                                 int64_t T, const int64_t* seq_offsets, int32_t S,
                                 const int32_t* group_offsets, int32_t Gn, const float* entropy,
                                 float* lr, float* d, acrl_seq_stats* seq, acrl_group_stats* grp,
                                 acrl_batch_stats* batch, int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_grpo_advantage -- GRPO advantages (Sec. 2, under Eq. grpo_objective):
 *     A_i = (R_i - mean_g R) / (std_g R + adv_eps)
 * over the responses of each prompt, std with p->adv_ddof degrees of freedom;
 * a prompt with a single response follows p->singleton_rule.
 *   rewards  device float [S];  adv  device float [S] output.
 *   group_offsets device int32 [Gn+1] (BAD_OFFSETS if inconsistent).
 */
acrl_status acrl_grpo_advantage(const float* rewards, const int32_t* group_offsets, int32_t Gn, int32_t S,
                                const acrl_params* p, float* adv, int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_controller_init -- set *state (device) for the parameters: X = X_init
 * and calibrated when X_init > 0, otherwise empty calibration sums.
 */
acrl_status acrl_controller_init(acrl_controller_state* state, const acrl_params* p, acrl_stream stream);

/*
 * acrl_controller_save / acrl_controller_load -- copy the controller state
 * between its device location and host memory: a checkpoint of the only
 * state the method carries from step to step (X and its calibration, fixed
 * once calibrated, Sec. 4.1).  Resuming from a saved state is bit-exact.
 *   state       device acrl_controller_state.
 *   host_state  host memory of one acrl_controller_state (any alignment).
 * Both are ordered on `stream` and synchronise it before returning.
 */
acrl_status acrl_controller_save(const acrl_controller_state* state, acrl_controller_state* host_state,
                                 acrl_stream stream);
acrl_status acrl_controller_load(acrl_controller_state* state, const acrl_controller_state* host_state,
                                 acrl_stream stream);

/*
 * acrl_controller_step -- the adaptive controller and the importance weights.
 * Calibration (Sec. 4.1, X fixed before training; Sec. 5.1 takes it from
 * step 0): while not calibrated, Y_sum and Q_eff of `batch` are added to the
 * state; after p->calib_steps batches X = sum / count is frozen.  On earlier
 * calibration batches alpha = 0.  Then per response (Sec. 4.1, after Eq. ACRL)
 *     alpha_i = gamma sign(A_i) (1 - Y / X)      (Y per p->y_gran)
 * and per valid token
 *     ACRL: w = exp(min(alpha_i lr_t, ln C))     = min(rho_t, C)
 *     TIS : w = exp(min(lr_t, ln C))             (Eq. TIS)
 *     MIS : w = exp(S_i) if S_i <= ln C else 0   (Eq. MIS)
 *     NONE: w = 1
 * and the per-token loss coefficient of Eq. ACRL
 *     coef_t = m_t w_t A_i / norm_t,  norm_t = Q_eff G_g n_i  (or N for TOKEN_MEAN).
 * X <= 0 in ACRL mode gives alpha = 0 and raises X_NONPOS.
 * The controller reads n_tokens, n_groups_valid and Y_sum of `batch` (and
 * rewrites Y_mean = Y_sum / n_groups_valid): a data-parallel caller that sums
 * those three fields over its ranks before this call gets one global X and
 * the global loss normalisation on every rank.
 *   state     device, updated in place.
 *   lr, mask, seq_offsets, group_offsets  as for acrl_seq_discrepancy.
 *   seq       device [S] in/out (writes alpha, sum_w, n_trunc).
 *   grp       device [Gn] in;  batch  device [1] in/out (writes X, trunc_frac,
 *             w_mean, alpha_mean).
 *   adv       device float [S] GRPO advantages.
 *   weight    device float [T] output w_t (0 where m_t = 0).
 *   coef      device float [T] output coef_t (0 where m_t = 0).
 *   alpha     device float [S] output, or NULL.
 *   ent_coef  device float [T] output beta m_t / norm_t for the entropy bonus,
 *             or NULL (then p->entropy_coeff is not used).
 * Ablations (Sec. 5.5): ACRL_MODE_ACRL_CONTINUOUS uses alpha = -kappa sign(A_i);
 * ACRL_MODE_ACRL_FALLBACK uses the ACRL alpha when Y > X and 0 otherwise.
 * With p->x_ema > 0, every step after the one that fixed X (or every step, if
 * X_init > 0) ends with X <- (1 - x_ema) X + x_ema Y_mean; batch->X reports
 * the X this step used.
 */
acrl_status acrl_controller_step(acrl_controller_state* state, const acrl_params* p,
                                 const float* lr, const uint8_t* mask, int64_t T,
                                 const int64_t* seq_offsets, int32_t S,
                                 const int32_t* group_offsets, int32_t Gn,
                                 acrl_seq_stats* seq, const acrl_group_stats* grp,
                                 acrl_batch_stats* batch, const float* adv,
                                 float* weight, float* coef, float* alpha, float* ent_coef,
                                 int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_loss_grad_logits -- loss of Eq. ACRL and its gradient w.r.t. the logits.
 * With r_t = exp(logp_t - old_logp_t) (exactly 1 when old_logp is NULL, the
 * one-update-per-rollout setting of App. A) and g_t = 1 on the unclipped
 * branch of min(r A, clip(r, 1-eps, 1+eps) A), 0 otherwise:
 *     grad[t, j]   = coef_t g_t r_t (p_tj - 1[j = a_t])          (bf16)
 *     token_loss_t = -coef_t * (coef_t >= 0 ? min(r, clip(r)) : max(r, clip(r)))
 *     *loss        = sum_t token_loss_t   (fixed order, fp64 accumulation)
 * With an entropy bonus (ent_coef and entropy given, e_t = ent_coef_t):
 *     grad[t, j]  += e_t p_tj (log p_tj + H_t),   token_loss_t += -e_t H_t
 * (H_t = -sum_j p_tj log p_tj; d H / d z_j = -p_j (log p_j + H)).
 * The probabilities are never stored.  Rows with m_t = 0, or with no
 * gradient (coef_t g_t = 0 and no entropy bonus), get a zero gradient row
 * without reading the rest of their logits.  A row that carries a gradient
 * but whose lse (given or recomputed) or log-prob is not finite (a NaN or an
 * infinity among its logits), or whose old_logp is NaN, has no defined
 * surrogate: its gradient row and token_loss_t are NaN (and so is *loss), and
 * the call raises ACRL_FLAG_NONFINITE.
 *   logits  device bf16 [T, ld];  grad  device bf16 [T, ld] output (columns
 *           >= V untouched).  May be called on a chunk of rows: every
 *           per-token pointer then points at the chunk's first row.
 *   ids, mask  as for acrl_token_stats.
 *   lse     device float [T] from acrl_token_stats on the same logits, or
 *           NULL to recompute it here (the cached-old path: a second sweep
 *           over each row; for rows of more than 6,144 columns each CTA
 *           keeps up to 40 KB (rows of up to 24,583 columns), 72 KB (up to
 *           40,967) or 96 KB of its row in shared memory, loaded by one bulk copy per row whose wait
 *           is bounded (ACRL_FLAG_TIMEOUT), and, from 65,536 columns, up to
 *           128 KB in tensor memory between the sweeps: it then allocates 256
 *           of the SM's 512 tensor-memory columns while it runs).
 *   old_logp  device float [T] log pi_old(a_t), or NULL for r = 1.
 *   coef    device float [T]: acrl_controller_step's `coef` output for the
 *           same batch (the same rows, in the same order).  It carries
 *           m_t w_t A_i / norm_t, and its sign is the sign of A_i, which the
 *           clip gate g_t reads (A_i >= 0: r <= 1+eps; A_i < 0: r >= 1-eps);
 *           coef_t = 0 carries no policy gradient, whatever A_i was.
 *   entropy, ent_coef  device float [T] (acrl_token_stats' entropy and
 *           acrl_controller_step's ent_coef), both NULL for no entropy bonus.
 *   clip_eps  the eps of Eq. grpo_objective.
 *   token_loss  device float [T] output;  loss  device float [1] output.
 */
acrl_status acrl_loss_grad_logits(const acrl_bf16* logits, int64_t T, int64_t V, int64_t ld,
                                  const int32_t* ids, const uint8_t* mask, const float* lse,
                                  const float* old_logp, const float* coef,
                                  const float* entropy, const float* ent_coef, float clip_eps,
                                  acrl_bf16* grad, float* token_loss, float* loss,
                                  int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_reduce_loss -- *loss = sum_t token_loss[t] over T entries, in the same
 * fixed order and fp64 accumulation as acrl_loss_grad_logits.  Gives the
 * batch loss when the gradient was produced chunk by chunk (Eq. ACRL's outer
 * sums run over every token of the batch).
 *   token_loss  device float [T];  loss  device float [1] output.
 */
acrl_status acrl_reduce_loss(const float* token_loss, int64_t T, float* loss, acrl_stream stream);

/*
 * Host-buffer pipeline -- the whole on-policy pass (token statistics,
 * discrepancy, advantages, controller, gradient: the calls above, each citing
 * its passage) for a batch whose inputs and outputs live in host memory, e.g.
 * logits computed on or offloaded to the host.  A runtime convenience with no
 * counterpart in the paper.  Per step the logits are uploaded in `chunks` row
 * chunks and the statistics call runs on each chunk as it lands; then the
 * discrepancy, advantage and controller calls; then the gradient call chunk
 * by chunk, each gradient chunk downloaded as soon as it is written, and the
 * loss.  Uploads run on one copy stream of the pipeline and downloads on
 * another, so consecutive steps overlap: step k+1's uploads run while step
 * k's gradient is downloaded.  The results are those of the device calls on
 * the same data, bit for bit.
 *
 * acrl_host_pipeline_workspace_bytes -- device bytes the pipeline needs: the
 *   batch's logits [T, ld], a ring of up to four gradient chunks, the
 *   per-token and per-response vectors and two copies of the small inputs.
 * acrl_host_pipeline_create -- binds a caller-owned device workspace of at
 *   least that size (16-byte aligned; the library allocates no device memory)
 *   and creates the two copy streams and the events that order the chunks.
 *   T >= 1, 1 <= V <= ld (ld a multiple of 8), S >= 1, Gn >= 1,
 *   1 <= chunks <= 4096.  *pipeline receives the handle.
 * acrl_host_pipeline_step -- enqueues one step.  Host arrays, page-locked for
 *   the copies to overlap (ordinary memory works, without overlap):
 *     logits bf16 [T, ld], ids int32 [T], mask uint8 [T] (or NULL: all 1),
 *     logp_mu float [T], rewards float [S], seq_offsets int64 [S+1],
 *     group_offsets int32 [Gn+1]  -- read while the uploads run;
 *     grad bf16 [T, ld] (columns >= V untouched), loss float [1]
 *                                 -- written while the downloads run.
 *   `state` is the device controller state, `p` the parameters (with
 *   p->entropy_coeff > 0 the entropy bonus is included), `dev_flags` the
 *   device flags word.  The kernels run on `stream`, which is made to wait
 *   for the step's downloads: once `stream` has been synchronised, grad and
 *   loss hold the step's results.  Host arrays must stay valid until then.
 *   One host thread at a time per pipeline.
 * acrl_host_pipeline_begin / acrl_host_pipeline_finish -- the same step in
 *   two halves, for data-parallel callers: begin enqueues the uploads, the
 *   statistics and the discrepancy call (the arguments the step reads from
 *   host memory, plus dev_flags and stream); then the caller may combine the
 *   batch statistics across ranks on `stream` (n_tokens, n_groups_valid and
 *   Y_sum of the acrl_batch_stats at acrl_host_pipeline_batch_stats, as for
 *   acrl_controller_step); finish enqueues the advantages, the controller, the
 *   gradient, the downloads and the loss.  step = begin + finish.  Calls out
 *   of that order return ACRL_ERR_INVALID_ARG.
 * acrl_host_pipeline_batch_stats -- device address of the pipeline's
 *   acrl_batch_stats (inside the workspace), or NULL for a NULL handle.
 * acrl_host_pipeline_destroy -- waits for the pipeline's copies, releases its
 *   streams and events (not the workspace) and frees the handle.
 */
typedef struct acrl_host_pipeline acrl_host_pipeline;
int64_t     acrl_host_pipeline_workspace_bytes(int64_t T, int64_t ld, int32_t S, int32_t Gn, int32_t chunks);
acrl_status acrl_host_pipeline_create(acrl_host_pipeline** pipeline, int64_t T, int64_t V, int64_t ld, int32_t S,
                                      int32_t Gn, int32_t chunks, void* workspace, int64_t workspace_bytes);
acrl_status acrl_host_pipeline_step(acrl_host_pipeline* pipeline, const acrl_params* p,
                                    acrl_controller_state* state, const acrl_bf16* logits, const int32_t* ids,
                                    const uint8_t* mask, const float* logp_mu, const float* rewards,
                                    const int64_t* seq_offsets, const int32_t* group_offsets, acrl_bf16* grad,
                                    float* loss, int32_t* dev_flags, acrl_stream stream);
acrl_status acrl_host_pipeline_begin(acrl_host_pipeline* pipeline, const acrl_bf16* logits, const int32_t* ids,
                                     const uint8_t* mask, const float* logp_mu, const float* rewards,
                                     const int64_t* seq_offsets, const int32_t* group_offsets, int32_t* dev_flags,
                                     acrl_stream stream);
acrl_status acrl_host_pipeline_finish(acrl_host_pipeline* pipeline, const acrl_params* p,
                                      acrl_controller_state* state, acrl_bf16* grad, float* loss,
                                      int32_t* dev_flags, acrl_stream stream);
acrl_batch_stats* acrl_host_pipeline_batch_stats(acrl_host_pipeline* pipeline);
acrl_status acrl_host_pipeline_destroy(acrl_host_pipeline* pipeline);

/*
 * acrl_lmhead_logits_stats -- the LM-head projection logits = H W^T fused
 * with the log-softmax statistics of acrl_token_stats (the optional fused
 * path of the logits pass; the paper's policy pi ends in this projection).
 * bf16 inputs, fp32 accumulation on the tensor cores (tcgen05, TMEM), logits
 * rounded to bf16 and stored; for every row and every 256-column tile the
 * epilogue writes the online state (max, U = max log2e, sum 2^(u-U),
 * sum 2^(u-U)(u-U)) of those bf16 logits to `partials`, which
 * acrl_lmhead_merge turns into lse / logp / entropy.
 *   hidden   device bf16 [M, ldh] (K used), weight device bf16 [N, ldw] (K used),
 *            both 16-byte aligned with ldh, ldw multiples of 8.
 *   logits   device bf16 [M, ldl] output (ldl >= N, multiple of 8).
 *   partials device float4 workspace of acrl_lmhead_workspace_bytes(M, N)
 *            bytes, layout [ceil(N/256)][M]; owned by the caller.
 * hidden, weight and logits must be device memory of the current device:
 * managed memory, host memory (page-locked or not) and another GPU's memory
 * are refused with ACRL_ERR_INVALID_ARG (checked with cudaPointerGetAttributes
 * before anything is launched), since the tensor-core copies are encoded over
 * these pointers.
 * Pipeline waits are time-bounded: ACRL_FLAG_TIMEOUT means the outputs of this
 * call are invalid.  Requires an sm_100-family GPU (built for sm_103a).
 */
int64_t     acrl_lmhead_workspace_bytes(int64_t M, int64_t N);
acrl_status acrl_lmhead_logits_stats(const acrl_bf16* hidden, int64_t M, int64_t K, int64_t ldh,
                                     const acrl_bf16* weight, int64_t N, int64_t ldw,
                                     acrl_bf16* logits, int64_t ldl, float* partials,
                                     int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_lmhead_merge -- lse, logp = z[a] - lse and entropy per row from the
 * partial states of acrl_lmhead_logits_stats (the tiles of a row combined in
 * a fixed order, so the result is deterministic); same outputs, masking and
 * flags as acrl_token_stats.  z[a] is read from `logits`.
 */
acrl_status acrl_lmhead_merge(const float* partials, const acrl_bf16* logits, int64_t M, int64_t N,
                              int64_t ldl, const int32_t* ids, const uint8_t* mask,
                              float* lse, float* logp, float* entropy,
                              int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_lmhead_stats_noalloc -- acrl_lmhead_logits_stats followed by
 * acrl_lmhead_merge in one call that allocates nothing and takes no
 * workspace.  The paper has no counterpart: this exists for callers that
 * cannot allocate device memory themselves -- a plugin handed only tensors
 * by a framework whose caching allocator already owns nearly all of HBM, or a
 * step that must not call cudaMalloc/cudaFree (cudaFree synchronises the
 * device).  The per-tile partial states live in one fixed device array of
 * this library, ACRL_LMHEAD_NOALLOC_SCRATCH_BYTES (16 MiB) in size, which
 * every GPU that loads the library holds until the process exits.
 *   Limit: ceil(N / 256) * M * 16 bytes must fit, e.g. M <= 1765 rows at
 *   N = 151,936 or M <= 8388 at N = 32,000; larger problems return
 *   ACRL_ERR_SCRATCH_TOO_SMALL before anything is launched.
 *   The first call on each device looks up the array's device address with
 *   that device current and keeps it for the life of the process; make that
 *   first call before any stream capture.  A device reset (cudaDeviceReset,
 *   or the primary context torn down and made again) invalidates the kept
 *   address: do not call this entry point on a device after resetting it.
 *   All calls share the array: calls that overlap on the GPU (different
 *   streams, or different host threads, on the same device) race on it and
 *   must be ordered by the caller.  Nothing in it needs clearing between calls.
 *   Arguments, outputs and flags are those of the two calls it combines,
 *   including the rule that hidden, weight and logits be device memory of
 *   the current device.
 */
#define ACRL_LMHEAD_NOALLOC_SCRATCH_BYTES (16LL << 20)
acrl_status acrl_lmhead_stats_noalloc(const acrl_bf16* hidden, int64_t M, int64_t K, int64_t ldh,
                                      const acrl_bf16* weight, int64_t N, int64_t ldw,
                                      acrl_bf16* logits, int64_t ldl,
                                      const int32_t* ids, const uint8_t* mask,
                                      float* lse, float* logp, float* entropy,
                                      int32_t* dev_flags, acrl_stream stream);

/*
 * acrl_selftest_wait_timeout -- failure-detection self-test: one warp waits on
 * a shared-memory barrier that nothing arrives on, with the same bounded wait
 * that guards every pipeline wait of acrl_lmhead_logits_stats; after
 * `limit_ns` (at most 2e9) it raises ACRL_FLAG_TIMEOUT in *dev_flags and
 * returns, leaving the context usable.  Not part of the paper's method.
 */
acrl_status acrl_selftest_wait_timeout(int32_t* dev_flags, int64_t limit_ns, acrl_stream stream);

/* Copy the device flags word to *host_flags; synchronises `stream`. */
acrl_status acrl_read_flags(const int32_t* dev_flags, int32_t* host_flags, acrl_stream stream);

/* Synchronise `stream` and report the device flags word as a status:
 * ACRL_ERR_DEVICE_FLAGS if any ACRL_FLAG_* bit is set (acrl_read_flags tells
 * which), ACRL_OK if none.  The word is left as it is. */
acrl_status acrl_check_flags(const int32_t* dev_flags, acrl_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* ACRL_H_ */
