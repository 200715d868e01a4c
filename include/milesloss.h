/*
 * libmilesloss: the per-token RL loss over the vocabulary, forward and
 * backward, on one GB300 GPU (sm_103a).
 *
 * The trainer side of an RL post-training loop ("Miles v0.1: Production-Level
 * Post-Training", arxiv 2609.08368) computes, for every token a policy sampled,
 * the trainer's log-prob of that token, the importance ratio against the log-
 * prob the rollout engine reported, r = exp(log pi_train - log pi_rollout)
 * (Sec. 3.4), a group-relative advantage (GRPO, Sec. 2 and Sec. 9.1), and a
 * loss whose gradient updates the policy (Sec. 1.1). This library evaluates
 * that loss from the policy's logits over the full vocabulary and writes
 * dLogits, without ever materialising the softmax.
 *
 * Per token t (row t of the logits), with s = z / T:
 *   logp_t = s_y - logsumexp(s),  H_t = -sum_j p_j log p_j      (entropy)
 *   r_t    = exp(logp_t - base_t), base = old log-probs if given, else the
 *            rollout log-probs                                       (Sec. 3.4)
 *   pg_t   = max(-A r, -A clip(r, 1-eps_lo, 1+eps_hi)), then for A < 0 capped
 *            at -A c by the dual clip                               (PPO)
 *   optional TIS / clip-or-pop weight on pg_t                      (Sec. 3.4)
 *   k3_t   = exp(q - logp) - (q - logp) - 1 against reference log-probs q
 *   l_t    = pg_t + kl_coef k3_t - entropy_coef H_t
 *   loss   = sum_t m_t l_t / sum_t m_t  (m = loss mask, Sec. 2.4)
 * A is the GRPO advantage of the token's trajectory: rewards centred (and by
 * default scaled by the sample std, floored) within the trajectory's group;
 * a group whose rewards are all equal gets A = 0 (Sec. 2.2, Table 2). With
 * on-policy distillation, A_t -= opd_coef (rollout_logprob_t -
 * teacher_logprob_t) (Sec. 5.2).
 *
 * Conventions shared by every call below.
 *  - Every array pointer is DEVICE memory owned by the caller. The library
 *    never allocates, frees or synchronises; each call only enqueues work on
 *    `stream` and returns. The library keeps no state between calls except
 *    per-device kernel attributes set once.
 *  - Calls on different streams are safe given distinct workspaces and
 *    outputs. A workspace written by rl_loss_fwd must not be reused before
 *    the matching rl_loss_bwd has run.
 *  - Host-side argument errors return a status before anything is enqueued.
 *  - Data-dependent errors (a target or a top-K candidate id outside
 *    [0, vocab), a group id outside [0, n_groups), cu_seqlens not
 *    non-decreasing from 0 to n_rows, a wait inside a kernel that ran out of
 *    time) never trap: the kernels finish, write zeros for the affected rows,
 *    and record the error in the workspace; read it with
 *    rl_loss_check_device_error after the stream is synchronised. Every wait
 *    inside a kernel is bounded (2 s); a CTA whose wait runs out stops
 *    issuing copies, waits (bounded) for the copies it has in flight, writes
 *    zeros for its remaining rows and returns.
 *  - Outputs are defined for every row, trained or not; rows with mask 0 get
 *    their log-prob and entropy and a zero dLogits row.
 *  - n_rows == 0 is a valid no-op apart from zeroed statistics.
 */
#ifndef MILESLOSS_H
#define MILESLOSS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* rl_stream;

typedef enum {
  RL_OK = 0,
  RL_ERR_INVALID_ARG = 1,         /* a pointer, size or parameter is invalid   */
  RL_ERR_UNSUPPORTED = 2,         /* valid but not implemented (see message)   */
  RL_ERR_WORKSPACE_TOO_SMALL = 3, /* workspace_bytes < rl_loss_workspace_size  */
  RL_ERR_CUDA = 4,                /* a CUDA runtime call failed                */
  RL_ERR_TARGET_OUT_OF_RANGE = 5, /* device: a target id not in [0, vocab)     */
  RL_ERR_GROUP_OUT_OF_RANGE = 6,  /* device: a group id not in [0, n_groups)   */
  RL_ERR_BAD_SEQLENS = 7,         /* device: cu_seqlens not 0 <= ... <= n_rows,
                                     non-decreasing, ending at n_rows          */
  RL_ERR_DEVICE_TIMEOUT = 8,      /* device: a bounded wait gave up            */
  RL_ERR_TOPK_ID_OUT_OF_RANGE = 9 /* device: a top-K OPD candidate id not in
                                     [0, vocab)                                */
} rl_status;

typedef enum { RL_BF16 = 0, RL_F32 = 1 } rl_dtype;

/* Ratio corrections of Sec. 3.4: a constant per-token weight on the
 * policy-gradient term from the train/rollout ratio
 * rc = exp(log pi_train - log pi_rollout), where log pi_train is
 * old_logprobs when given (the PPO ratio is then exp(logp - old)) and else
 * the trainer's own log-prob of the token in this pass (the single-pass
 * step: rc = exp(logp - rollout), held constant, and the PPO ratio is taken
 * against the rollout log-probs too):
 *   RL_CORR_TIS          weight = min(max(rc, corr_lo), corr_hi)
 *   RL_CORR_CLIP_OR_POP  weight = rc if corr_lo <= rc <= corr_hi, else 0 */
typedef enum { RL_CORR_NONE = 0, RL_CORR_TIS = 1, RL_CORR_CLIP_OR_POP = 2 } rl_correction;

/* Advantage estimators of Sec. 3.4.
 *   RL_EST_GRPO                 rewards centred within the trajectory's group and
 *                               divided by max(group std, std_floor) (GRPO)
 *   RL_EST_REINFORCEPP          the outcome reward is every token's return; the
 *                               returns are normalised over all training tokens
 *                               of the call (REINFORCE++)
 *   RL_EST_REINFORCEPP_BASELINE the reward minus its group's mean, then the same
 *                               normalisation (REINFORCE++ baseline-relative)
 *   RL_EST_GSPO                 GRPO advantages with a sequence-level ratio:
 *                               s_i = exp(mean over trajectory i's training tokens
 *                               of logp - base), clipped per trajectory; the
 *                               policy term is the mean over trajectories with
 *                               training tokens (GSPO). Runs as forward sweep,
 *                               per-trajectory pass and gradient sweep (the
 *                               gradient of a token depends on its whole
 *                               trajectory), so it reads the logits twice. */
typedef enum {
  RL_EST_GRPO = 0,
  RL_EST_REINFORCEPP = 1,
  RL_EST_REINFORCEPP_BASELINE = 2,
  RL_EST_GSPO = 3
} rl_estimator;

typedef struct {
  float temperature;   /* T > 0: logits are divided by T before the softmax      */
  float eps_lo;        /* >= 0: lower clip at 1 - eps_lo                          */
  float eps_hi;        /* >= 0: upper clip at 1 + eps_hi                          */
  float dual_clip_c;   /* 0 = off, else > 1: for A < 0 the PG term is capped at -A c */
  float kl_coef;       /* beta >= 0; ref_logprobs must be given when beta > 0     */
  float entropy_coef;  /* gamma >= 0: the token loss gets -gamma * H              */
  float std_floor;     /* > 0: GRPO divides by max(std, std_floor)                */
  int32_t normalize_std; /* 1: divide by the group std (GRPO); 0: centre only   */
  int32_t unbiased_std;  /* 1: sample std (n - 1); 0: population std (n)        */
  int32_t correction;    /* rl_correction                                       */
  float corr_lo;       /* correction interval [corr_lo, corr_hi], default [0, 2] */
  float corr_hi;
  float opd_coef;      /* on-policy distillation coefficient; 0 = off (Sec. 5.2) */
  int32_t estimator;   /* rl_estimator; RL_EST_GSPO does not combine with opd_coef */
  int32_t opd_topk;    /* K >= 1 selects the top-K OPD signal (Sec. 5.2), 0 the
                          one-sample signal from teacher_logprobs; K <= 64     */
  /* Top-K OPD inputs (DEVICE pointers, read by the kernels; used when
   * opd_topk > 0 and opd_coef != 0): for row t, K candidate token ids
   * opd_topk_ids[t*K + k] in [0, vocab) chosen on the serving side (e.g. the
   * student's K most likely tokens) and the teacher's log-probs of them,
   * opd_topk_teacher[t*K + k]. The signal is sum_k w_k (log p_k - teacher_k)
   * with the trainer's probabilities p_k of the candidates renormalised over
   * the set as weights w_k; it is subtracted, times opd_coef, from the token's
   * advantage and is not differentiated. Both arrays are device memory,
   * 4-byte aligned (else RL_ERR_INVALID_ARG); K <= 64. A row with a
   * candidate id outside [0, vocab) gets zeros like a row with a bad target,
   * and the call records RL_ERR_TOPK_ID_OUT_OF_RANGE. */
  const int32_t* opd_topk_ids;
  const float* opd_topk_teacher;
} rl_loss_params;

/* Call-wide statistics, written to DEVICE memory by the stream. Means are
 * over the tokens that train (mask 1); all fields are 0 when there are none.
 * The integers are exact counts. */
typedef struct {
  double loss;                 /* sum m l / N                                      */
  double pg_loss_mean;         /* mean PG term (after any correction weight)       */
  double kl_mean;              /* mean k3 (0 without ref_logprobs)                 */
  double entropy_mean;         /* mean H                                           */
  double ratio_mean;           /* mean r                                           */
  double ratio_absdev_mean;    /* mean |r - 1|                                     */
  double logprob_absdiff_mean; /* mean |logp - rollout logp| (train/rollout divergence, Sec. 9.2) */
  double corr_ratio_mean;      /* mean pre-clamp correction ratio rc (1 without)   */
  double corr_absdev_mean;     /* mean |rc - 1|                                    */
  float ratio_min;
  float ratio_max;
  int64_t n_tokens;            /* N = sum m                                        */
  int64_t n_clip_hi;           /* PPO clip engaged above 1 + eps_hi               */
  int64_t n_clip_lo;           /* PPO clip engaged below 1 - eps_lo               */
  int64_t n_dual_clip;         /* dual clip engaged                                */
  int64_t n_corr_clip;         /* correction weight differs from rc (Sec. 3.4 clipped fraction) */
} rl_loss_stats;

/* A shard's partial statistics (row-sharded calls, below), in DEVICE memory.
 * Combine the shards' copies element by element: `sum` and `count` by
 * addition, `max` by maximum. */
typedef struct {
  double sum[9];   /* over the shard's training tokens: l, pg, k3, H, r, |r - 1|,
                      |logp - rollout logp|, rc, |rc - 1|                        */
  double count[5]; /* training tokens, clip_hi, clip_lo, dual clip, correction
                      clip (exact integers)                                      */
  double max[2];   /* -(minimum r) and maximum r over the shard's training
                      tokens (-inf when it has none)                             */
} rl_loss_partials;

/* Bytes of device workspace that one call with these sizes needs (the same
 * value serves rl_loss_fwd, rl_loss_bwd and rl_loss_fwd_bwd). The workspace
 * is caller-owned, 256-byte aligned, needs no initialisation, and carries the
 * per-row state from rl_loss_fwd to rl_loss_bwd. */
rl_status rl_loss_workspace_size(int64_t n_rows, int32_t n_traj, int32_t n_groups,
                                 size_t* bytes);

/* Forward: log-probs, entropy, advantages, the loss and its statistics.
 *
 *  logits            [n_rows, ld] of `logits_dtype` (bf16 or fp32); row t
 *                    holds the logits that scored targets[t] (already shifted
 *                    by the caller); only the first `vocab` columns are read.
 *                    Rows whose start is 16-byte aligned (ld * element size a
 *                    multiple of 16 and a 16-byte aligned base) take the
 *                    fast bulk-copy path; any other layout is still correct.
 *  targets           [n_rows] int32 sampled token ids, in [0, vocab)
 *  rollout_logprobs  [n_rows] fp32 log-probs the rollout engine reported
 *  ref_logprobs      [n_rows] fp32 reference-policy log-probs, or NULL
 *                    (required when kl_coef > 0)
 *  old_logprobs      [n_rows] fp32 log-probs of the policy before this update,
 *                    or NULL (then the PPO ratio is taken against the rollout
 *                    log-probs, and a correction uses this pass's own
 *                    log-prob as log pi_train)
 *  teacher_logprobs  [n_rows] fp32 teacher log-probs for OPD, or NULL
 *                    (required when opd_coef != 0 and opd_topk == 0)
 *  rewards           [n_traj] fp32, one outcome reward per trajectory
 *  group_id          [n_traj] int32 in [0, n_groups): the prompt of each
 *                    trajectory; members of a group may be anywhere
 *  cu_seqlens        [n_traj + 1] int32 row offsets: trajectory i owns rows
 *                    [cu[i], cu[i+1]); cu[0] = 0, cu[n_traj] = n_rows
 *  loss_mask         [n_rows] uint8, nonzero = the token trains (model-
 *                    generated; tool output and prompts are masked, Sec. 2.4)
 *  params            host pointer, read during the call only
 *  token_logprobs    [n_rows] fp32 out, or NULL
 *  entropy           [n_rows] fp32 out, or NULL
 *  advantages        [n_traj] fp32 out (before OPD shaping), or NULL
 *  group_sizes       [n_groups] int32 out, or NULL
 *  stats             one rl_loss_stats out (device), or NULL
 *  workspace         device, >= rl_loss_workspace_size bytes
 */
rl_status rl_loss_fwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                      int64_t vocab, int64_t ld, const int32_t* targets,
                      const float* rollout_logprobs, const float* ref_logprobs,
                      const float* old_logprobs, const float* teacher_logprobs,
                      const float* rewards, const int32_t* group_id,
                      const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                      const uint8_t* loss_mask, const rl_loss_params* params,
                      float* token_logprobs, float* entropy, float* advantages,
                      int32_t* group_sizes, rl_loss_stats* stats, void* workspace,
                      size_t workspace_bytes, rl_stream stream);

/* Backward from the state rl_loss_fwd left in `workspace`: dLogits of
 * g * loss with g = grad_loss * (*grad_loss_device if non-NULL), i.e.
 *   dZ_tj = g (m_t / N) (1/T) [G_t (1[j = y_t] - p_j) + gamma p_j (log p_j + H_t)]
 * with G_t = d l_t / d logp_t. Re-reads the logits once. The logits, targets,
 * mask and params must be the ones given to rl_loss_fwd.
 *  dlogits  [n_rows, ld_out] of `dlogits_dtype` (bf16 rounded to nearest
 *           even, or fp32); columns >= vocab are not written. */
rl_status rl_loss_bwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                      int64_t vocab, int64_t ld, const int32_t* targets,
                      const uint8_t* loss_mask, const rl_loss_params* params,
                      float grad_loss, const float* grad_loss_device,
                      const void* workspace, size_t workspace_bytes, void* dlogits,
                      rl_dtype dlogits_dtype, int64_t ld_out, rl_stream stream);

/* Forward and backward in one pass that reads each logit row from HBM once:
 * every output of rl_loss_fwd plus dLogits as in rl_loss_bwd. */
rl_status rl_loss_fwd_bwd(const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                          int64_t vocab, int64_t ld, const int32_t* targets,
                          const float* rollout_logprobs, const float* ref_logprobs,
                          const float* old_logprobs, const float* teacher_logprobs,
                          const float* rewards, const int32_t* group_id,
                          const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                          const uint8_t* loss_mask, const rl_loss_params* params,
                          float* token_logprobs, float* entropy, float* advantages,
                          int32_t* group_sizes, rl_loss_stats* stats,
                          float grad_loss, const float* grad_loss_device, void* dlogits,
                          rl_dtype dlogits_dtype, int64_t ld_out, void* workspace,
                          size_t workspace_bytes, rl_stream stream);

/* Phases of rl_loss_fwd_bwd_rows. */
enum {
  RL_PHASE_BEGIN = 1, /* advantages, N and validation over the whole call      */
  RL_PHASE_ROWS = 2,  /* the vocabulary sweep over rows [row_begin, row_end)   */
  RL_PHASE_END = 4,   /* the loss and its statistics over the whole call       */
  RL_PHASE_ALL = 7
};

/* rl_loss_fwd_bwd for logits that exist a block of rows at a time (the usual
 * way to bound the memory of the language-model head): one BEGIN, any number
 * of ROWS calls that together cover the rows once, one END, all on the same
 * workspace and stream (or ordered by the caller across streams). The
 * arguments are those of rl_loss_fwd_bwd for the whole call (n_rows, the
 * per-row inputs and outputs, rewards, groups, cu_seqlens), except:
 *  logits    rows [row_begin, row_end): logits points at row row_begin with
 *            row stride ld (the chunk buffer); NULL outside ROWS
 *  dlogits   the same rows of dLogits, pointing at row row_begin; NULL runs
 *            the chunk forward-only (log-probs, entropy, loss terms; the
 *            per-row state stays in the workspace)
 * rl_loss_fwd_bwd_rows(RL_PHASE_ALL, 0, n_rows, ...) is rl_loss_fwd_bwd.
 * GSPO needs every log-prob before any gradient: with RL_EST_GSPO only that
 * whole call is accepted (RL_ERR_UNSUPPORTED otherwise). */
rl_status rl_loss_fwd_bwd_rows(int32_t phase, int64_t row_begin, int64_t row_end,
                               const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                               int64_t vocab, int64_t ld, const int32_t* targets,
                               const float* rollout_logprobs, const float* ref_logprobs,
                               const float* old_logprobs, const float* teacher_logprobs,
                               const float* rewards, const int32_t* group_id,
                               const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                               const uint8_t* loss_mask, const rl_loss_params* params,
                               float* token_logprobs, float* entropy, float* advantages,
                               int32_t* group_sizes, rl_loss_stats* stats, float grad_loss,
                               const float* grad_loss_device, void* dlogits,
                               rl_dtype dlogits_dtype, int64_t ld_out, void* workspace,
                               size_t workspace_bytes, rl_stream stream);

/* Phases of rl_loss_shard_fwd_bwd. */
enum {
  RL_SHARD_COUNT = 1,  /* this shard's training tokens per trajectory        */
  RL_SHARD_SWEEP = 2,  /* advantages, the sweep over the shard's rows, dLogits
                          and the shard's partial statistics (GSPO: the
                          forward sweep and the per-trajectory sums)          */
  RL_SHARD_FINISH = 4, /* the call's statistics from the combined partials   */
  RL_SHARD_SEQ = 8     /* GSPO only, after SWEEP: the trajectories' terms from
                          the added sums, dLogits, partial statistics        */
};

/* rl_loss_fwd_bwd with the rows of one call spread over several shards (one
 * per GPU or rank: data parallelism, or context parallelism, which splits
 * each long session over ranks, Sec. 9.1). Shard k holds the contiguous rows
 * [row_offset, row_offset + n_rows) of a call of n_rows_total rows; the
 * per-row arrays (logits, targets, log-probs, mask, token_logprobs, entropy,
 * dlogits) cover those rows only, while rewards, group_id and cu_seqlens
 * (row offsets in the whole call's numbering) describe the whole call on
 * every shard. The loss needs two exchanges between the shards, which the
 * caller performs (the library has no collective):
 *   1. RL_SHARD_COUNT writes traj_counts[n_traj] (int32, device): the
 *      training tokens of each trajectory within this shard. The caller sums
 *      the array over the shards (an all-reduce) in place.
 *   2. RL_SHARD_SWEEP, given the summed traj_counts, computes the advantages
 *      (every shard the same), the sweep over its rows with the whole call's
 *      N, dLogits (dlogits NULL: forward only) and writes `partials`. The
 *      caller combines the shards' partials as rl_loss_partials says.
 *   3. RL_SHARD_FINISH writes `stats` from the combined partials.
 * GSPO (a token's gradient needs its whole trajectory's sequence ratio) takes
 * one more exchange: SWEEP runs the forward sweep and writes
 * traj_sums[n_traj][2] (double, device): per trajectory, the sums over this
 * shard's training tokens of (log-prob - base log-prob) and of the
 * correction weight. The caller adds traj_sums over the shards in place;
 * RL_SHARD_SEQ then computes each trajectory's sequence ratio and terms,
 * dLogits and `partials`; FINISH as above.
 * Each shard's outputs for its rows (log-probs, entropies, dLogits) are those
 * of the unsharded call (GSPO: up to the order of the per-trajectory sums);
 * the statistics differ from it only in the order of their floating-point
 * sums. Every phase of a shard uses the same workspace
 * (rl_loss_workspace_size(n_rows, n_traj, n_groups)), in order, on one
 * stream. Arguments a phase does not read may be NULL (COUNT: logits,
 * outputs, dlogits, traj_sums, partials, stats; SWEEP without GSPO:
 * traj_sums; GSPO's SWEEP: dlogits, partials, stats; FINISH: everything but
 * partials, stats and the stream). */
rl_status rl_loss_shard_fwd_bwd(int32_t phase, int64_t row_offset, int64_t n_rows_total,
                                const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                                int64_t vocab, int64_t ld, const int32_t* targets,
                                const float* rollout_logprobs, const float* ref_logprobs,
                                const float* old_logprobs, const float* teacher_logprobs,
                                const float* rewards, const int32_t* group_id,
                                const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                                const uint8_t* loss_mask, const rl_loss_params* params,
                                float* token_logprobs, float* entropy, float* advantages,
                                int32_t* group_sizes, int32_t* traj_counts, double* traj_sums,
                                rl_loss_partials* partials, rl_loss_stats* stats,
                                float grad_loss, const float* grad_loss_device, void* dlogits,
                                rl_dtype dlogits_dtype, int64_t ld_out, void* workspace,
                                size_t workspace_bytes, rl_stream stream);

/* Phases of rl_loss_vocab_shard_fwd_bwd. */
enum {
  RL_VSHARD_COUNT = 1,    /* this shard's training tokens per trajectory        */
  RL_VSHARD_PARTIAL = 2,  /* advantages; the forward sweep over the shard's
                             columns, writing each row's partial sums          */
  RL_VSHARD_SWEEP = 3,    /* merge of the gathered partial sums; dLogits over
                             the shard's columns; the shard's partial statistics */
  RL_VSHARD_FINISH = 4,   /* the call's statistics from the combined partials   */
  RL_VSHARD_SEQ = 5       /* GSPO only, after SWEEP: the trajectories' terms from
                             the added sums, dLogits, partial statistics       */
};

/* rl_loss_fwd_bwd with the VOCABULARY of one call split over shards (tensor
 * parallelism: each rank holds a block of the logits' columns, as the
 * paper's case study trains with TP 2, Sec. 9.1), optionally combined with
 * a split of its rows as in rl_loss_shard_fwd_bwd (context / data
 * parallelism, CP 4 there).
 *
 *  col_starts      HOST array of n_col_shards + 1 vocabulary ids: shard k
 *                  holds columns [col_starts[k], col_starts[k+1]);
 *                  col_starts[0] = 0, strictly increasing (every shard has a
 *                  column), col_starts[n_col_shards] = the vocabulary size
 *                  (<= INT32_MAX). 1 <= n_col_shards <= 64.
 *  col_shard       this shard's index in col_starts.
 *  logits          [n_rows, ld] of logits_dtype: this shard's columns of its
 *                  rows (ld >= its column count); dlogits and ld_out alike.
 *  targets         vocabulary ids in [0, col_starts[n_col_shards]), the same
 *                  on every column shard of a row.
 *  row_offset, n_rows_total, traj_counts, traj_sums, partials, stats: as
 *                  in rl_loss_shard_fwd_bwd (one column shard of the whole
 *                  rows: row_offset 0, n_rows_total = n_rows).
 *  row_partials    [n_rows][8] floats (device, 16-byte aligned), written by
 *                  PARTIAL: per row, m, s, u and zy, with m a reference in
 *                  log2 units (a multiple of k = log2(e)/T of a logit),
 *                  s = sum_j 2^(z_j k - m) and u = sum_j 2^(z_j k - m)
 *                  (z_j k - m) over the shard's columns j, zy the target's
 *                  logit if the target is one of them, else 0; then, with
 *                  top-K OPD, the part of the row's candidates c in the
 *                  shard's columns: mt = max z_c k, sw = sum_c 2^(z_c k - mt),
 *                  acc = sum_c 2^(z_c k - mt) (z_c / T - teacher_c), and 1 if
 *                  a candidate id lies outside the vocabulary (else 0);
 *                  (-inf, 0, 0, 0) without candidates there or without
 *                  top-K. m = NaN marks a row the shard gave up on
 *                  (RL_ERR_DEVICE_TIMEOUT in its workspace): every shard
 *                  then writes zeros for that row.
 *  row_partials_all [n_col_shards][n_rows][8] floats (device, 16-byte
 *                  aligned), read by SWEEP: every column shard's row_partials
 *                  of the same rows, in shard order (an all-gather).
 *
 * Phases, in order, on one stream, with one workspace
 * (rl_loss_workspace_size(n_rows, n_traj, n_groups)) per shard:
 *   1. COUNT writes traj_counts; the caller sums it over the ROW shards.
 *   2. PARTIAL computes the advantages and N from the summed counts (the
 *      same on every shard) and writes row_partials. The caller gathers the
 *      records of the COLUMN shards of its rows into row_partials_all.
 *   3. SWEEP merges each row's records in shard order (every column shard
 *      computes the same bits), writes token_logprobs and entropy (the
 *      same on every column shard), dLogits over the shard's columns
 *      (dlogits NULL: none) and `partials`. Column shards of the same rows
 *      write the same partials: the caller combines them over the ROW
 *      shards only, as rl_loss_partials says.
 *   4. FINISH writes `stats` from the combined partials.
 * GSPO: SWEEP stops after the merge with the shard's per-trajectory sums in
 * traj_sums (as in rl_loss_shard_fwd_bwd); the caller adds them over the ROW
 * shards (column shards of the same rows hold the same sums), then SEQ
 * writes dLogits over the shard's columns and `partials`, and FINISH
 * follows.
 * A shard's log-probs, entropies and dLogits equal the unsharded call's up
 * to the order of the row's floating-point sums (within the library's
 * tolerances, not bit for bit). The logits are read twice (PARTIAL and the
 * gradient in SWEEP or SEQ), as for the split rl_loss_fwd / rl_loss_bwd
 * pair. With top-K OPD the candidate ids and teacher log-probs
 * (rl_loss_params.opd_topk_ids / opd_topk_teacher, [n_rows][K]) are the
 * shard's rows' whole candidate lists, as vocabulary ids, on every column
 * shard. A target outside the vocabulary is reported by SWEEP
 * (RL_ERR_TARGET_OUT_OF_RANGE; the row gets zeros), a candidate id outside
 * it likewise (RL_ERR_TOPK_ID_OUT_OF_RANGE). Arguments a phase does not read may be NULL (COUNT: logits,
 * outputs, dlogits, traj_sums, row_partials*, partials, stats; PARTIAL:
 * outputs other than advantages and group_sizes, traj_sums,
 * row_partials_all, dlogits, partials, stats; SWEEP: row_partials, stats,
 * traj_sums without GSPO, and dlogits and partials with it; SEQ:
 * row_partials*, stats; FINISH: everything but partials, stats and the
 * stream). */
rl_status rl_loss_vocab_shard_fwd_bwd(
    int32_t phase, int32_t col_shard, int32_t n_col_shards, const int64_t* col_starts,
    int64_t row_offset, int64_t n_rows_total, const void* logits, rl_dtype logits_dtype,
    int64_t n_rows, int64_t ld, const int32_t* targets, const float* rollout_logprobs,
    const float* ref_logprobs, const float* old_logprobs, const float* teacher_logprobs,
    const float* rewards, const int32_t* group_id, const int32_t* cu_seqlens, int32_t n_traj,
    int32_t n_groups, const uint8_t* loss_mask, const rl_loss_params* params,
    float* token_logprobs, float* entropy, float* advantages, int32_t* group_sizes,
    int32_t* traj_counts, double* traj_sums, float* row_partials, const float* row_partials_all,
    rl_loss_partials* partials, rl_loss_stats* stats, float grad_loss,
    const float* grad_loss_device, void* dlogits, rl_dtype dlogits_dtype, int64_t ld_out,
    void* workspace, size_t workspace_bytes, rl_stream stream);

/* rl_loss_fwd_bwd for callers that cannot allocate device memory at call
 * time (the paper has no counterpart; this is a deployment convenience).
 * Frameworks that reserve nearly all of HBM for their own pool, plain-C
 * hosts and plugins without access to the process's allocator, and code
 * whose memory footprint must stay fixed after start-up cannot provide a
 * workspace; this call takes every other argument of rl_loss_fwd_bwd and
 * uses an 8 MiB array compiled into the library instead (about 200,000 rows
 * at small trajectory and group counts). Larger calls return
 * RL_ERR_WORKSPACE_TOO_SMALL before anything is enqueued. Each device on
 * which the library's code is loaded keeps the array until the process
 * exits. Every call looks up the array's device address on the current
 * device (cudaGetSymbolAddress, which allocates nothing); the first call on
 * a device also loads the library's device code there, so make it before
 * any stream capture. No call allocates or frees memory. All calls on a
 * device share the array: calls that overlap on the GPU race and must be
 * serialised by the caller; what must start at zero is reset by every
 * call. The data-dependent errors of a call (bad target, group id,
 * cu_seqlens or top-K candidate, a wait that ran out) are recorded in the
 * array as for rl_loss_fwd_bwd and read with
 * rl_loss_noalloc_check_device_error; the affected rows get zeros. */
rl_status rl_loss_fwd_bwd_noalloc(const void* logits, rl_dtype logits_dtype, int64_t n_rows,
                                  int64_t vocab, int64_t ld, const int32_t* targets,
                                  const float* rollout_logprobs, const float* ref_logprobs,
                                  const float* old_logprobs, const float* teacher_logprobs,
                                  const float* rewards, const int32_t* group_id,
                                  const int32_t* cu_seqlens, int32_t n_traj, int32_t n_groups,
                                  const uint8_t* loss_mask, const rl_loss_params* params,
                                  float* token_logprobs, float* entropy, float* advantages,
                                  int32_t* group_sizes, rl_loss_stats* stats, float grad_loss,
                                  const float* grad_loss_device, void* dlogits,
                                  rl_dtype dlogits_dtype, int64_t ld_out, rl_stream stream);

/* The device-side error of the last rl_loss_fwd_bwd_noalloc call on the
 * current device, read after its stream has been synchronised: RL_OK or the
 * lowest recorded code, as rl_loss_check_device_error. Reads four bytes of
 * the array with one blocking copy (cudaMemcpyFromSymbol, no allocation).
 * A later no-alloc call on the device overwrites the value. */
rl_status rl_loss_noalloc_check_device_error(void);

/* After the stream that ran a call on `workspace` has been synchronised:
 * RL_OK, or the data-dependent error the kernels recorded (when several
 * kinds occurred, the lowest code). Performs one small blocking
 * device-to-host copy on the legacy default stream. */
rl_status rl_loss_check_device_error(const void* workspace);

/* Static text for a status code; never NULL. */
const char* rl_status_string(rl_status status);

/* Launch-plan overrides: measurement aids and a test hook, not needed for
 * normal use. The library picks every launch shape itself (the sweep kernel
 * by row length, the cluster kernel's cluster size, ring depth and block
 * shape, the streaming kernel's ring); these fields force one instead. -1
 * in a field keeps the library's choice; rl_launch_overrides_init sets
 * every field to -1. A forced value outside the compiled shapes makes later
 * calls return RL_ERR_UNSUPPORTED before anything is enqueued.
 *  sweep_kernel         0 = the cluster kernel, 1 = the streaming kernel
 *                       (16-byte aligned rows only)
 *  cluster_size         1, 2, 4 or 8 CTAs per row (cluster kernel)
 *  cluster_stages       1..4 ring stages (cluster kernel)
 *  cluster_threads      256 or 512 threads per CTA (cluster kernel)
 *  cluster_ctas_per_sm  4 or 5 with 256 threads, 2 with 512
 *  stream_chunk_bytes   ring slot size, a multiple of 128 in [1 KB, 128 KB]
 *  stream_slots         ring slots (as many as fit by default)
 *  stream_hold          last chunks of a row pass B reads from shared memory
 *  stream_split_first   1: the ragged chunk first, 0: last
 *  stream_prefetch_bytes bytes of the next row the streaming kernel asks L2
 *                       to fetch once a row's first-pass copies are issued
 *                       (0 = none; a multiple of 16)
 *  stream_ctas_per_sm   streaming kernel: CTAs per SM, 1 (sixteen consumer
 *                       warps per CTA), 2 (eight each, half of the shared
 *                       memory each) or 4 (four each, a quarter)
 *  stream_cluster       streaming kernel, fused calls without top-K (other
 *                       calls ignore it): CTAs per row, 1 (each row on one
 *                       CTA) or 2, 4 or 8 (a cluster of that many CTAs per
 *                       row, each streaming a slice of it; one CTA per SM)
 *  stall_first_wait_ns  TEST HOOK, > 0: in each CTA of the vocabulary sweep,
 *                       the first wait for logits waits instead on a barrier
 *                       that nothing completes, bounded by this many
 *                       nanoseconds. It runs out, the CTA gives up as it
 *                       would on a copy that never arrives (stops issuing
 *                       copies, waits for the ones in flight, writes zeros
 *                       for its rows) and the call records
 *                       RL_ERR_DEVICE_TIMEOUT. Nothing hangs and no fault is
 *                       raised; it exists to test that path.
 * The overrides are process-wide and apply to calls made after the setter
 * returns. */
typedef struct {
  int32_t sweep_kernel;
  int32_t cluster_size;
  int32_t cluster_stages;
  int32_t cluster_threads;
  int32_t cluster_ctas_per_sm;
  int32_t stream_chunk_bytes;
  int32_t stream_slots;
  int32_t stream_hold;
  int32_t stream_split_first;
  int32_t stream_prefetch_bytes;
  int32_t stream_ctas_per_sm;
  int64_t stall_first_wait_ns;
  int32_t stream_cluster;
} rl_launch_overrides;

/* Sets every field of *o to -1 (no override). */
rl_status rl_launch_overrides_init(rl_launch_overrides* o);

/* Installs *o as the process-wide overrides; NULL removes them. Returns
 * RL_ERR_INVALID_ARG for a value outside a field's documented range. */
rl_status rl_set_launch_overrides(const rl_launch_overrides* o);

/* Optional timing hook for the calling host thread: when both are non-NULL,
 * later calls on this thread record `begin` / `end` (cudaEvent_t) on their
 * stream immediately before and after the main vocabulary-sweep kernel.
 * Pass NULLs to turn it off. */
rl_status rl_set_sweep_events(void* begin_event, void* end_event);

/* Version of this interface, e.g. 100 for 1.0. */
int32_t rl_loss_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MILESLOSS_H */
