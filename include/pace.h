/*
 * pace.h - C ABI of the PACE hot path on GB300 (sm_103a).
 *
 * PACE (Pool-Aware Control of Effective Staleness) admits completed
 * trajectories of an asynchronous RL pool into the trainer.  This library
 * computes, on one GPU:
 *   (a) per-trajectory staleness scores from per-token policy-version tags
 *       (Lemma 1 / Eq. 2; Eqs. 7-10), the occupancy rejection budget
 *       (Eqs. 3-4) and the deterministic rejection of the top-scored units
 *       (Sec. 3.1 quantile rule; Algorithm 1, trainer side);
 *   (b) for the accepted batch, each token's log-probability under the
 *       current policy through a fused LM head (logits never reach memory)
 *       and the asymmetric, dual-clipped token-mean surrogate of the
 *       unchanged GRPO update (shared training settings of the appendix).
 *
 * Conventions shared by every entry point
 *   - Pointers marked "device" are CUDA device pointers; "host" are host
 *     pointers.  The caller owns every buffer; the library never allocates.
 *   - Every call is asynchronous and ordered on `stream` (a cudaStream_t;
 *     NULL is the legacy default stream).  Nothing is synchronised unless a
 *     comment says so.
 *   - Errors found from the arguments alone are returned at once, before any
 *     launch.  Errors found in the data on the device (a version tag above
 *     its completion version, a target outside the vocabulary, a wait that
 *     ran out) are written to `*status_dev`, an int32 in device memory: the
 *     first error wins (compare-and-swap from 0), so the caller sets it to 0
 *     before the work and reads it after synchronising.  status_dev may be
 *     NULL, in which case device-side errors are not reported.  After a
 *     device-side error the outputs of that call are unspecified.
 *   - `workspace` is caller-owned device scratch of at least the size the
 *     matching *_workspace_size() query returns, 256-byte aligned; its
 *     contents need not be initialised and are clobbered.
 *   - bf16 arrays are passed as raw 16-bit storage (`const void*`).
 */
#ifndef PACE_H_
#define PACE_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define PACE_API __attribute__((visibility("default")))
#else
#define PACE_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  PACE_OK = 0,
  PACE_ERR_INVALID_ARG = 1,       /* bad pointer, size, parameter or CSR offsets */
  PACE_ERR_VERSION_ORDER = 2,     /* v_t > c(tau) or c(tau) > j: Lemma 1's premise fails */
  PACE_ERR_NAN_INPUT = 3,         /* NaN in the prefix-score window or in unit scores */
  PACE_ERR_UNSUPPORTED_SHAPE = 4, /* shape or alignment the kernels do not handle */
  PACE_ERR_WORKSPACE = 5,         /* workspace missing, too small or misaligned */
  PACE_ERR_TIMEOUT = 6,           /* a bounded on-device wait ran out (device-side only) */
  PACE_ERR_CUDA = 7               /* a CUDA runtime call failed (no device, launch error) */
} pace_status;

/* Human-readable name of a status code (static storage). */
PACE_API const char* pace_status_string(pace_status status);

/* Library version, major * 10000 + minor * 100 + patch. */
PACE_API int32_t pace_version(void);

/* ------------------------------------------------------------------------ */
/* (a) Pool scoring                                                          */
/* ------------------------------------------------------------------------ */

/* Trajectory score M(tau; j) of Eq. 7 (Sec. 3.2):
 *   PACE_SCORE_EFF  Effective Staleness, Eq. 8:  K_wait + F * K_gen
 *   PACE_SCORE_RAW  PACE (Raw Staleness):         K_wait + K_gen
 *   PACE_SCORE_GEN  PACE (Generation Staleness):  F * K_gen
 * where F = phi_gamma(q) (Eq. 10) and q is the empirical percentile of the
 * trajectory's prefix forgetting score in the window (Eq. 9). */
typedef enum { PACE_SCORE_EFF = 0, PACE_SCORE_RAW = 1, PACE_SCORE_GEN = 2 } pace_score_mode;

typedef struct {
  int32_t mode;       /* pace_score_mode; default PACE_SCORE_EFF */
  int32_t gamma;      /* integer sharpening exponent of Eq. 10, 1..64; default 4 */
  int32_t min_obs;    /* window size below which F = 1 for all (falls back to Raw); default 32 */
  int32_t group_size; /* G: trajectories g*G .. g*G+G-1 form unit g; default 8 (1 = per trajectory) */
  double f_missing;   /* F of a trajectory without a prefix score (s_pre NaN); default 1.0 */
} PaceScoreParams;

/* Fill `p` with the defaults above (the paper's admission settings). */
PACE_API void pace_score_params_default(PaceScoreParams* p);

/* Score every trajectory of the pool (Lemma 1 / Eq. 2, Eqs. 7-10) and average
 * the scores of each group of G ("mean aggregation within groups").
 *
 *   tags        device int32 [n_tokens], 16-byte aligned: policy version v_t
 *               of each response token (Sec. 2), trajectory-major; -1 marks a
 *               token the policy did not generate (tool output), which is left
 *               out of K_gen.  Versions are below 2^31 - 1.
 *   offsets     device int64 [n_traj+1]: tokens of trajectory i are
 *               tags[offsets[i] .. offsets[i+1]); offsets[0] = 0,
 *               non-decreasing, offsets[n_traj] = n_tokens.
 *   c_version   device int32 [n_traj]: c(tau), the trainer version at which
 *               the trajectory completed (= entered the pool), 0 <= c <= j.
 *   s_pre       device float32 [n_traj]: prefix forgetting score (Eq. 6) or
 *               NaN when no prefix was rescored.  May be NULL for RAW mode.
 *   trainer_version  j, the step that consumes the pool.
 *   window      device float32 [window_len]: W^pre, recent prefix scores
 *               (Eq. 9); 0 <= window_len <= 4096; NaN is an error.  May be
 *               NULL when window_len is 0.
 * Outputs (device float64, may individually be NULL except score):
 *   kgen, kwait, weight (F), score [n_traj]; unit_score [n_traj / G].
 * Values are bit-identical to the fp64 definitions: K_gen = S / T with
 * S = sum (c - v_t) summed exactly in integers (0 when T = 0); q = count of
 * window values <= s_pre (float32 compare) / |W|; integer powers by repeated
 * multiplication; no fused multiply-add anywhere.
 * Launches: the tag stream (one wave, whose blocks also sort the window and
 * tabulate F on pools of 8,192 trajectories and more) and a finalisation
 * launch; from 2^18 trajectories (pace_set_score_fused_min_traj) the stream is
 * a cooperative launch that also finalises, each block waiting (bounded) for
 * the blocks that streamed its groups' tokens.
 * Device-side errors: PACE_ERR_VERSION_ORDER (v_t > c or c > j),
 * PACE_ERR_INVALID_ARG (tag < -1, c < 0, bad offsets), PACE_ERR_NAN_INPUT,
 * PACE_ERR_TIMEOUT (a bounded wait of the cooperative launch ran out).
 * Host errors: PACE_ERR_INVALID_ARG when n_traj is not a multiple of G or a
 * required pointer is NULL. */
PACE_API pace_status pace_score_pool(const int32_t* tags, const int64_t* offsets,
                            const int32_t* c_version, const float* s_pre, int64_t n_traj,
                            int64_t n_tokens, int32_t trainer_version, const float* window,
                            int64_t window_len, const PaceScoreParams* params, double* kgen,
                            double* kwait, double* weight, double* score, double* unit_score,
                            void* workspace, size_t workspace_bytes, int32_t* status_dev,
                            void* stream);

/* Workspace bytes pace_score_pool needs for a pool of n_traj trajectories and
 * a window of window_len values: a 16-byte slot per trajectory for the tag
 * stream's totals, 512 KB of per-warp partial slots, the sorted window, the
 * table of F over every possible ECDF count and a few KB of flags.  Its
 * contents need no initialisation and are overwritten by every call; calls
 * that overlap on the GPU need workspaces of their own. */
PACE_API size_t pace_score_pool_workspace_size(int64_t n_traj, int64_t window_len);

/* ------------------------------------------------------------------------ */
/* (a) Rejection budget and selection                                        */
/* ------------------------------------------------------------------------ */

typedef struct {
  int64_t n_target;  /* N^tar, desired buffer of ready trajectories (Eq. 3) */
  double beta;       /* EMA coefficient of Eq. 4, in [0, 1); default 0 */
  double r_max;      /* maximum rejection budget; default 0.9 (admission settings) */
  double r_hat_prev; /* r-hat_{j-1}, the smoothed rate of the previous step; default 0 */
} PaceBudgetParams;

PACE_API void pace_budget_params_default(PaceBudgetParams* p);

/* Host only, no device work.  Eq. 3 and Eq. 4:
 *   r     = clip((N - N^tar) / max(N, 1), 0, 1)        N = n_traj
 *   r_hat = beta * r_hat_prev + (1 - beta) * r
 *   k     = min(floor(min(r_hat, r_max) * n_units + 1e-9), n_units)
 * The 1e-9 nudge lands the floor on the exact surplus when fp64 rounding of
 * the product falls just below an integer (N = 47, N^tar = 35 gives 12).
 * Outputs are host pointers; r_out may be NULL. */
PACE_API pace_status pace_budget(int64_t n_traj, int64_t n_units, const PaceBudgetParams* p,
                        double* r_out, double* r_hat_out, int64_t* k_units_out);

/* Budget + rejection (Sec. 3.1; Algorithm 1, trainer side).  Computes k on
 * the host with pace_budget (no device synchronisation), then rejects on the
 * device the k units with the largest unit score; equal scores reject the
 * lower unit id first.  This is the quantile rule of Sec. 3.1 with the
 * window taken as the current pool: it rejects exactly floor(r_hat * U)
 * units, and ties are settled deterministically.
 *   unit_score     device float64 [n_units], >= 0 (as pace_score_pool
 *                  writes them); NaN gives PACE_ERR_NAN_INPUT on the device.
 *   group_size     G; unit u is trajectories u*G .. u*G+G-1; n_traj = U*G.
 *   r_hat_out, k_units_out   host outputs: r-hat_j (carry to the next step)
 *                  and k.
 *   accepted_ids   device int32, room for n_units*G entries: the
 *                  (U-k)*G accepted trajectory ids, ascending.
 *   rejected_ids   device int32, room for n_units*G entries (or NULL): the
 *                  k*G rejected ids, ascending.
 *   traj_accepted  device uint8 [n_units*G] or NULL: 1 accepted, 0 rejected. */
PACE_API pace_status pace_select(const double* unit_score, int64_t n_units, int32_t group_size,
                        const PaceBudgetParams* budget, double* r_hat_out,
                        int64_t* k_units_out, int32_t* accepted_ids, int32_t* rejected_ids,
                        uint8_t* traj_accepted, void* workspace, size_t workspace_bytes,
                        int32_t* status_dev, void* stream);

/* Same rejection with k given by the caller (0 <= k_units <= n_units).
 * Pools of at most 131,072 units are selected by one thread-block cluster and
 * touch no workspace (it may be NULL); larger pools need
 * pace_select_workspace_size bytes.  The first call on a device with more than
 * 512 units sets a kernel attribute (its shared-memory size): make it before
 * any stream capture. */
PACE_API pace_status pace_select_k(const double* unit_score, int64_t n_units, int32_t group_size,
                          int64_t k_units, int32_t* accepted_ids, int32_t* rejected_ids,
                          uint8_t* traj_accepted, void* workspace, size_t workspace_bytes,
                          int32_t* status_dev, void* stream);

PACE_API size_t pace_select_workspace_size(int64_t n_units);

/* ---- Sharded rejection: the pool's units partitioned across ranks --------
 * The rule of pace_select_k over the WHOLE pool (Sec. 3.1, Algorithm 1: the
 * k top-scored units are rejected, ties lowest id first), when rank r holds
 * the contiguous units [u0_r, u0_r + n_units_r) and their unit scores, u0
 * increasing with r.  Every rank computes the same k (pace_budget on the
 * whole pool's counts).  The calls run an MSB-first radix select of the
 * order-preserving 64-bit keys of the scores; the caller sums the histograms
 * over the ranks between the calls, with any collective:
 *   for pass in 0..PACE_SHARD_PASSES-1:
 *     pace_select_shard_pass(.., pass, k, hist_sum_prev, hist_mine, ..)
 *     hist_sum = sum over ranks of hist_mine         (all-reduce, uint32 bins)
 *   pace_select_shard_ties(.., hist_sum, &tied_mine, ..)
 *   tied_before = sum of tied_mine over lower ranks  (exclusive scan)
 *   pace_select_shard_write(.., k, tied_before, u0 * G, ..)
 * The union of the ranks' lists is exactly pace_select_k's on the whole pool.
 * Every call is stream-ordered and needs no host synchronisation; the
 * workspace (pace_select_shard_workspace_size, 256-byte aligned) carries the
 * select state from call to call and must not be shared by concurrent calls.
 *   hist_prev, hist_out, hist_last   device uint32 [PACE_SHARD_HIST_BINS];
 *                    hist_prev is the summed histogram of pass - 1 (NULL at
 *                    pass 0); hist_out is this shard's histogram of pass
 *                    (cleared by the call).
 *   n_tied_out       device int64 [1]: this shard's units tied at the pivot.
 *   tied_before      device int64 [1]: units tied at the pivot on lower ranks.
 *   id_base          the global id of this shard's first trajectory (u0 * G);
 *                    ids written are id_base + local ids; traj_accepted is
 *                    indexed locally (n_units * G entries).
 *   n_rejected_out   device int64 [1] or NULL: units rejected on this shard.
 * A shard may hold no units (it still takes part in every pass).  NaN scores
 * report PACE_ERR_NAN_INPUT through status_dev at pass 0. */
#define PACE_SHARD_PASSES 6
#define PACE_SHARD_HIST_BINS 2048

PACE_API size_t pace_select_shard_workspace_size(int64_t n_units);

PACE_API pace_status pace_select_shard_pass(const double* unit_score, int64_t n_units,
                                            int32_t pass, int64_t k_units,
                                            const uint32_t* hist_prev, uint32_t* hist_out,
                                            void* workspace, size_t workspace_bytes,
                                            int32_t* status_dev, void* stream);

PACE_API pace_status pace_select_shard_ties(const double* unit_score, int64_t n_units,
                                            const uint32_t* hist_last, int64_t* n_tied_out,
                                            void* workspace, size_t workspace_bytes,
                                            int32_t* status_dev, void* stream);

PACE_API pace_status pace_select_shard_write(const double* unit_score, int64_t n_units,
                                             int32_t group_size, int64_t k_units,
                                             const int64_t* tied_before, int64_t id_base,
                                             int32_t* accepted_ids, int32_t* rejected_ids,
                                             uint8_t* traj_accepted, int64_t* n_rejected_out,
                                             void* workspace, size_t workspace_bytes,
                                             int32_t* status_dev, void* stream);

/* pace_select_k for callers that cannot allocate device memory.  The paper has
 * no counterpart: this exists for code that must not call cudaMalloc, such as
 * a plugin running inside a host framework whose memory pool owns all device
 * memory, or a latency-critical loop where an allocation could synchronise
 * the device.  Such a caller still passes its inputs and outputs.  Whenever
 * the one-cluster selection does not fit on the device (on GB300: pools above
 * 131,072 units; on a device with a smaller cluster limit, smaller pools too),
 * the radix path's scratch comes from a fixed array of 128 KB inside the
 * library (123,136 bytes are used at the 2^20-unit maximum), which every GPU
 * that loads the library keeps until the process exits.
 *   - n_units must be at most 2^20 (1,048,576); larger pools get
 *     PACE_ERR_UNSUPPORTED_SHAPE and nothing is launched.
 *   - The first call on a device looks up the array's device address (with
 *     that device current) and caches it; make that first call before any
 *     stream capture.  The cached address belongs to the device's context
 *     at that time: after cudaDeviceReset on that device the entry point must
 *     not be called again in the same process.
 *   - All calls on a device share the one array and each call re-initialises
 *     what it needs, so results do not depend on earlier calls; but calls
 *     that overlap on the GPU (different streams, or threads) race on it.
 * Arguments and outputs are those of pace_select_k; no cudaMalloc, cudaFree or
 * other allocating routine is called. */
PACE_API pace_status pace_select_k_noalloc(const double* unit_score, int64_t n_units,
                                           int32_t group_size, int64_t k_units,
                                           int32_t* accepted_ids, int32_t* rejected_ids,
                                           uint8_t* traj_accepted, int32_t* status_dev,
                                           void* stream);

/* ------------------------------------------------------------------------ */
/* (b) Log-probabilities and the clipped surrogate                           */
/* ------------------------------------------------------------------------ */

typedef enum {
  PACE_AGG_TOKEN_MEAN = 0,          /* sum_t m_t L_t / sum_t m_t ("Token mean") */
  PACE_AGG_SEQ_MEAN_TOKEN_MEAN = 1  /* mean over sequences of each one's token mean */
} pace_loss_agg;

typedef struct {
  float eps_low;      /* lower clip width; default 0.20 */
  float eps_high;     /* upper clip width; default 0.28 */
  float dual_clip;    /* dual-clip coefficient c (applies when A < 0); default 10 */
  float adv_eps;      /* epsilon of the group standardisation; default 1e-6 */
  int32_t agg;        /* pace_loss_agg; default PACE_AGG_TOKEN_MEAN */
  int32_t std_unbiased; /* 1: sample std (n - 1), 0: population std; default 1 */
} PaceLossParams;

PACE_API void pace_loss_params_default(PaceLossParams* p);

/* A batch of sequences laid out as rows (one row per token). */
typedef struct {
  const int64_t* seq_offsets;  /* device int64 [n_seq+1]: rows of sequence i are
                                  [seq_offsets[i], seq_offsets[i+1]); 0 .. n_rows */
  const uint8_t* seq_accepted; /* device uint8 [n_seq] or NULL (all accepted) */
  const uint8_t* mask;         /* device uint8 [n_rows] or NULL (all rows): 1 = the
                                  row is a policy token in the loss, 0 = prompt or
                                  tool output (kept in context, masked from the loss) */
  int64_t n_seq;
  int64_t n_rows;
} PaceBatch;

/* The policy-objective inputs of the batch. */
typedef struct {
  const float* behav_lp; /* device float32 [n_rows]: ell^mu_t recorded at rollout */
  const float* reward;   /* device float32 [n_seq] */
  int32_t group_size;    /* G: sequences g*G .. g*G+G-1 are prompt group g; n_seq % G == 0 */
  PaceLossParams params;
  double* loss;          /* device float64 [1]: the loss (output) */
  float* adv;            /* device float32 [n_seq] or NULL: advantages used (output) */
  float* ratio;          /* device float32 [n_rows] or NULL: rho_t of rows in the loss,
                            0 elsewhere (output) */
  double* partial;       /* device float64 [2] or NULL: the aggregate's numerator and
                            denominator before the division (output): sum_t m_t L_t
                            and sum_t m_t (TOKEN_MEAN), or the sum of the sequences'
                            token means and the number of sequences with tokens
                            (SEQ_MEAN_TOKEN_MEAN).  Batches split across ranks by
                            whole prompt groups add these, then divide. */
} PaceLossArgs;

/* GRPO within-group standardisation over the accepted members of each group:
 *   A_i = (R_i - mean_g) / (std_g + adv_eps);  rejected members get 0; a
 *   member whose reward equals the group mean gets 0.
 * reward device float32 [n_seq]; seq_accepted device uint8 [n_seq] or NULL;
 * adv device float32 [n_seq] (output).  Sums in fp64, lowest index first. */
PACE_API pace_status pace_group_advantages(const float* reward, const uint8_t* seq_accepted,
                                  int64_t n_seq, int32_t group_size, float adv_eps,
                                  int32_t std_unbiased, float* adv, void* stream);

/* Fused LM head: for every row r in the loss (mask[r] != 0 and its sequence
 * accepted) compute
 *   z_v     = h_r . W_v              bf16 x bf16, fp32 accumulation (tcgen05/TMEM)
 *   lse_r   = log sum_v exp(z_v / temperature)   (online, over the whole vocabulary)
 *   lp_r    = z_{y_r} / temperature - lse_r
 * without writing any logit to memory.  Rows not in the loss get lp = 0 and
 * lse = 0.  The hidden row r must be the state that predicts targets[r].
 *   hidden     device bf16 [n_rows][hidden_size], row-major, 16-byte aligned.
 *   w_vocab    device bf16 [vocab_size][hidden_size] (the lm_head.weight
 *              layout), 16-byte aligned.
 *   targets    device int32 [n_rows], 0 <= y < vocab_size for rows in the loss
 *              (else PACE_ERR_INVALID_ARG on the device and lp = NaN).
 *   hidden_size  multiple of 64, 64..16384; vocab_size 1..2^24; temperature > 0.
 *   logprob    device float32 [n_rows] (output); lse device float32 [n_rows]
 *              or NULL (output).
 *   loss       NULL, or the surrogate inputs: the call then also computes
 *              advantages (pace_group_advantages), the per-token clipped terms
 *              and the aggregated loss exactly as pace_surrogate_loss does,
 *              fused after the log-probs.
 * Rows in the loss are first compacted into a list of row indices, and the LM
 * head reads their hidden states through it, so the tensor cores only see rows
 * that count; the hidden states are never copied (the workspace holds the
 * index list and per-row partials, not rows: its size does not depend on
 * hidden_size). */
PACE_API pace_status pace_token_logprob(const PaceBatch* batch, const void* hidden, const void* w_vocab,
                               const int32_t* targets, int32_t hidden_size, int32_t vocab_size,
                               float temperature, float* logprob, float* lse,
                               const PaceLossArgs* loss, void* workspace, size_t workspace_bytes,
                               int32_t* status_dev, void* stream);

PACE_API size_t pace_token_logprob_workspace_size(int64_t n_rows, int64_t n_seq, int32_t hidden_size,
                                         int32_t vocab_size);

/* Clipped surrogate on given log-probabilities (shared training settings:
 * asymmetric clip eps_low / eps_high, dual clip c, token-mean aggregation):
 *   rho_t = exp(clamp(lp_t - ell^mu_t, -20, 20))
 *   L_t   = max(-A rho_t, -A clip(rho_t, 1 - eps_low, 1 + eps_high)),
 *           then min(L_t, -c A) when A < 0
 *   loss  = sum_t m_t L_t / sum_t m_t  (TOKEN_MEAN), or the mean over
 *           sequences with tokens of each sequence's token mean.
 * A is the group-standardised advantage of the row's sequence.  Per-token
 * terms in fp32, sums in fp64 in a fixed order (deterministic).  An empty
 * loss is 0.  logprob is device float32 [n_rows]. */
PACE_API pace_status pace_surrogate_loss(const PaceBatch* batch, const float* logprob,
                                const PaceLossArgs* loss, void* workspace,
                                size_t workspace_bytes, int32_t* status_dev, void* stream);

PACE_API size_t pace_surrogate_loss_workspace_size(int64_t n_rows, int64_t n_seq);

/* The loss of a batch split across ranks by whole prompt groups: each rank's
 * pace_token_logprob / pace_surrogate_loss fills PaceLossArgs.partial; the
 * caller sums the two values over the ranks (one all-reduce) and this writes
 * loss = numerator / denominator (0 when the denominator is 0), the division
 * of the unsplit batch's aggregate.  partial: device float64 [2]; loss: device
 * float64 [1]. */
PACE_API pace_status pace_loss_from_partial(const double* partial, double* loss, void* stream);

/* The literal admission rule of Sec. 3.1 and Algorithm 1 (trainer side), kept
 * across steps with a sliding window of recently observed unit scores:
 *   kappa = Quantile_{1 - r}(W^M)  (inverted-CDF: the k-th smallest window
 *           score, k = max(ceil((1 - r) |W| - 1e-9), 1); +inf while the window
 *           holds fewer than min_obs scores),
 * then candidates are drawn in the given order: score > kappa is rejected
 * (decision 0), the rest retained (1) until batch_units are retained, and the
 * candidates after that are not drawn (2; batch_units <= 0 draws all).  Every
 * drawn score then enters the window.
 *   unit_score   device float64 [n_cand], in draw order.
 *   r_hat        host: the budget, min(r-hat_j, r_max) from pace_budget.
 *   window       device float64 [capacity], capacity <= 4096 (the paper uses 512
 *                groups); window_state device int64 [2] = {count, next slot},
 *                zero-initialised by the caller once; both updated in place.
 *   decision     device uint8 [n_cand] (output); kappa device float64 [1] (output).
 * pace_select is the same rule with the window taken as the current pool. */
PACE_API pace_status pace_quantile_admit(const double* unit_score, int64_t n_cand,
                                         double r_hat, int64_t batch_units, int32_t min_obs,
                                         double* window, int64_t capacity,
                                         int64_t* window_state, uint8_t* decision,
                                         double* kappa, int32_t* status_dev, void* stream);

/* ------------------------------------------------------------------------ */
/* Stale-k admission and staleness diagnostics                               */
/* ------------------------------------------------------------------------ */

/* Stale-k admission, the prior-work baseline of Sec. 2 ("Controlled Stale-k
 * Analysis"): trajectory tau is admitted when its token-weighted policy lag
 *   kbar(tau; j) = (1/T) sum_t (j - v_t)                      (Eq. 1)
 * is at most k_max (kbar == k_max is admitted; T = 0 gives kbar = 0).  kbar is
 * computed from exact integer sums with one rounding.  tags / offsets /
 * n_tokens / trainer_version as for pace_score_pool; kbar device float64
 * [n_traj] (output, may be NULL); admitted device uint8 [n_traj] (output).
 * Device-side errors: PACE_ERR_VERSION_ORDER when a tag exceeds j,
 * PACE_ERR_INVALID_ARG for tags below -1 or bad offsets. */
PACE_API pace_status pace_stale_k(const int32_t* tags, const int64_t* offsets, int64_t n_traj,
                                  int64_t n_tokens, int32_t trainer_version, double k_max,
                                  double* kbar, uint8_t* admitted, void* workspace,
                                  size_t workspace_bytes, int32_t* status_dev, void* stream);

PACE_API size_t pace_stale_k_workspace_size(int64_t n_traj);

/* Histograms of a per-unit staleness value (K_wait, K_gen, K_eff, s_pre, ...)
 * for rejected and accepted units, as in the paper's retained-vs-rejected
 * admission analysis.  n_bins (1..4096) equal-width bins over [lo, hi): the bin
 * of x is floor((x - lo) / (hi - lo) * n_bins) in fp64, values below lo count
 * in the first bin and values at or above hi in the last.  hist is device
 * uint32 [2 * n_bins] (output): [0, n_bins) rejected (flag 0), [n_bins,
 * 2 n_bins) accepted; with flags NULL every value counts in the first half.
 * Exact integer counts; NaN values are skipped and reported as
 * PACE_ERR_NAN_INPUT. */
PACE_API pace_status pace_staleness_histogram(const double* values, const uint8_t* flags,
                                              int64_t n, double lo, double hi, int32_t n_bins,
                                              uint32_t* hist, int32_t* status_dev, void* stream);

/* Prefix Forgetting Score (Eq. 6, Sec. 3.2) with the collection rules of the
 * admission settings.  Each sequence of the batch is an interrupted rollout's
 * prefix (prompt plus the response tokens generated before a weight sync),
 * whose hidden states come from a forward pass of the updated rollout policy
 * u.  For each prefix,
 *   s_pre = (1/m) sum |log pi_u(y_t | x, y_<t) - l^mu_t|
 * over its first m = min(#eligible, cap_tokens) eligible rows (row order),
 * with log pi_u from the same fused LM head as pace_token_logprob; s_pre is NaN
 * when fewer than min_tokens rows are eligible (the paper requires 32; its caps
 * are 1,024 response tokens for math and 2,048 for ReTool).
 *   batch      seq_offsets over the prefix rows; mask marks eligible rows (policy
 *              response tokens; prompt and tool rows 0); NULL = every row;
 *              seq_accepted, if given, makes unaccepted prefixes empty.
 *   hidden, w_vocab, targets, hidden_size, vocab_size, temperature: as for
 *              pace_token_logprob, under policy u.
 *   behav_lp   device float32 [n_rows]: recorded behaviour log-probs l^mu_t.
 *   s_pre      device float32 [n_seq] (output), the input pace_score_pool takes.
 *   logprob    device float32 [n_rows] (output: log pi_u of the scored rows, 0
 *              elsewhere) or NULL (kept in the workspace).
 * The mean is an fp64 sum in a fixed order; device-side errors as for
 * pace_token_logprob. */
PACE_API pace_status pace_prefix_score(const PaceBatch* batch, const void* hidden,
                                       const void* w_vocab, const int32_t* targets,
                                       const float* behav_lp, int32_t hidden_size,
                                       int32_t vocab_size, float temperature, int32_t min_tokens,
                                       int32_t cap_tokens, float* s_pre, float* logprob,
                                       void* workspace, size_t workspace_bytes,
                                       int32_t* status_dev, void* stream);

PACE_API size_t pace_prefix_score_workspace_size(int64_t n_rows, int64_t n_seq,
                                                 int32_t hidden_size, int32_t vocab_size);

/* ------------------------------------------------------------------------ */
/* Backward: gradients for the unchanged policy update                       */
/* ------------------------------------------------------------------------ */

/* Derivative of pace_surrogate_loss's loss with respect to each row's
 * log-probability (the policy-gradient signal of the clipped objective):
 *   dL_t/dlp_t = -A rho_t when the unclipped term is the active maximum and the
 *                dual clip is not active; 0 when the clipped term or the dual
 *                clip is active or lp - l^mu is clamped; scaled by 1 / sum m
 *                (TOKEN_MEAN) or 1 / (#sequences * #tokens of the sequence);
 * dlp device float32 [n_rows] (output; 0 outside the loss).  Arguments as for
 * pace_surrogate_loss (loss->loss is not written). */
PACE_API pace_status pace_surrogate_backward(const PaceBatch* batch, const float* logprob,
                                             const PaceLossArgs* loss, float* dlp,
                                             void* workspace, size_t workspace_bytes,
                                             int32_t* status_dev, void* stream);

PACE_API size_t pace_surrogate_backward_workspace_size(int64_t n_rows, int64_t n_seq);

/* Backward of pace_token_logprob through the LM head, without materialising
 * more than one chunk of logits: with p = softmax(z / tau), z = h W^T and
 * g_r = dlp[r],
 *   G_rv = (g_r / tau) (1[v = y_r] - p_rv)
 *   grad_hidden[r] = sum_v G_rv W_v         device float32 [n_rows][H] (output)
 *   grad_w[v]      = sum_r G_rv h_r         device float32 [V][H] (output)
 * over the rows in the loss (rows outside it get 0).  lse is the forward's
 * output for the same rows (device float32 [n_rows]).  Rows are processed in
 * chunks of up to 32,768: logits are recomputed on the tensor cores, G is held
 * in bf16 in the workspace for the chunk (in 64-column blocks), then two
 * tensor-core GEMMs form G W and G^T H.  Chunks past the rows in the loss (a
 * count known only on the device) cost no tensor-core work.  Returns
 * PACE_ERR_UNSUPPORTED_SHAPE when ceil(V / 64) x the chunk's rows exceeds
 * 2^31 - 1 (V above about 4.2M at full chunks).  Other arguments and errors as
 * for pace_token_logprob. */
PACE_API pace_status pace_token_logprob_backward(const PaceBatch* batch, const void* hidden,
                                                 const void* w_vocab, const int32_t* targets,
                                                 int32_t hidden_size, int32_t vocab_size,
                                                 float temperature, const float* lse,
                                                 const float* dlp, float* grad_hidden,
                                                 float* grad_w, void* workspace,
                                                 size_t workspace_bytes, int32_t* status_dev,
                                                 void* stream);

PACE_API size_t pace_token_logprob_backward_workspace_size(int64_t n_rows, int64_t n_seq,
                                                           int32_t hidden_size,
                                                           int32_t vocab_size);

/* ------------------------------------------------------------------------ */
/* Profiling                                                                 */
/* ------------------------------------------------------------------------ */

typedef enum {
  PACE_PROFILE_LMHEAD = 0,     /* the fused LM-head kernel of pace_token_logprob */
  PACE_PROFILE_TAG_REDUCE = 1  /* the tag-stream reduction of pace_score_pool */
} pace_profile_kernel;

/* Not part of the method: a tuning control for the fused LM head
 * (pace_token_logprob, pace_prefix_score).  Its work items are (pair of
 * 128-row blocks, vocabulary split); how many contiguous splits the
 * vocabulary is cut into changes neither results beyond rounding order nor
 * FLOPs, but it changes how many vocabulary streams are in flight at once and
 * so the power, and on GB300 the power-capped clock, of a long launch, in a
 * way that differs from GPU to GPU (2 or 4 splits, either may be 2-10 %
 * faster).  From now on, in this process, batches with enough rows to give
 * every resident cluster at least four items use `splits` (clamped to the
 * number of 256-column vocabulary tiles); smaller batches and splits = 0 use
 * the automatic choice (the first of 4, 2, 3, 6, 8 that keeps rounds of items
 * at least 90 % full; 4 reads the vocabulary from HBM about once per round).
 * Returns PACE_ERR_INVALID_ARG unless 0 <= splits <= 8. */
PACE_API pace_status pace_set_lmhead_splits(int32_t splits);

/* Not part of the method: a tuning control for pace_score_pool.  Pools of at
 * least min_traj trajectories (with groups of at most 256) finalise their
 * scores inside the tag reduction's launch: each block, once its share of the
 * tag stream is done, scores its own slice of the groups after bounded waits
 * for the blocks that streamed those groups' tokens (a cooperative launch, so
 * every block is resident and the waits end); most of the per-trajectory work
 * then hides in the stream's ragged tail.  Smaller pools, and every pool on a
 * device without cooperative launches, finalise in a launch of their own,
 * which is faster on small pools.  Results are identical either way.
 * From now on, in this process, the given threshold applies (0: every pool;
 * the default is pace_score_fused_min_traj_default(), 2^18).  Returns
 * PACE_ERR_INVALID_ARG for a negative min_traj. */
PACE_API pace_status pace_set_score_fused_min_traj(int64_t min_traj);

/* The library's default for pace_set_score_fused_min_traj (2^18 trajectories). */
PACE_API int64_t pace_score_fused_min_traj_default(void);

/* Not part of the method: a measurement aid.  From now on, on the calling
 * host thread, record the CUDA event `begin` (a cudaEvent_t) on the call's
 * stream immediately before each launch of the given kernel and `end`
 * immediately after it, so a caller can time that kernel alone with
 * cudaEventElapsedTime.  NULL events turn it off.  The events stay owned by
 * the caller.  Returns PACE_ERR_INVALID_ARG for an unknown kernel. */
PACE_API pace_status pace_set_profile_events(int32_t kernel, void* begin, void* end);

/* Not part of the method: checks the integer construction of the doubles the
 * scoring writes.  For every i, with T[i] >= 1:
 *   q_int[i]  = S[i] / T[i] as the scoring kernels build it on the integer pipe,
 *   q_fp64[i] = the same quotient from the fp64 pipe, __ll2double_rn(S[i]) then
 *               a correctly rounded division (the rounding the oracle's
 *               (double)S / (double)T performs),
 *   c_int[i], c_fp64[i] = (double)S[i] both ways.
 * The two must agree bit for bit.  All arrays are device arrays of n entries.
 * Returns PACE_ERR_INVALID_ARG for n < 0 or a NULL array when n > 0. */
PACE_API pace_status pace_div_selftest(const int64_t* S, const uint32_t* T, int64_t n,
                                       double* q_int, double* q_fp64, double* c_int,
                                       double* c_fp64, void* stream);

/* Not part of the method: exercises the failure path every tensor-core
 * kernel relies on.  One GPU thread waits, with the same bounded wait the
 * kernels use, on an mbarrier that nothing ever completes; after limit_ns
 * (1 .. 2e9) it gives up, writes PACE_ERR_TIMEOUT to *status_dev (device, the
 * usual first-error-wins word) and the kernel returns normally, leaving the
 * context usable.  Returns PACE_ERR_INVALID_ARG for a NULL status or a limit
 * outside that range. */
PACE_API pace_status pace_wait_timeout_selftest(uint64_t limit_ns, int32_t* status_dev,
                                                void* stream);

/* Not part of the method: the number of CUDA kernels this library has
 * launched from the calling host thread since it was loaded (memsets and
 * copies are not kernels and are not counted). */
PACE_API uint64_t pace_kernel_launches(void);

#ifdef __cplusplus
}
#endif

#endif /* PACE_H_ */
