/*
 * rl_loss.h -- C ABI of the GB300 (sm_103a) policy-loss library.
 *
 * The library computes the token-level, group-relative clipped policy-gradient
 * objective of black-box agent RL (ClawGym II, arXiv 2608.16798) over packed,
 * ragged trajectories, and its gradient with respect to the logits:
 *
 *   - group-relative advantages A_i = (R_i - mu_g) / (sigma_g + eps) with the
 *     population standard deviation (Sec. 2.3.2, GRPO advantage equation;
 *     Sec. 3.2.3 for groups of rollouts; Sec. 3.3 for task-harness groups);
 *   - the masked objective (1/G) sum_i (1 / sum_t M_it) sum_t M_it [min(rho A,
 *     clip(rho, 1-eps, 1+eps) A) - beta KL] (Sec. 2.3.2, GRPO objective; the
 *     mask M_t of Sec. 2.3.1 excludes harness / tool-observation tokens);
 *   - the token-level truncated importance weight w_t = min(exp(log pi_old -
 *     log pi_rollout), c-bar) (Sec. 3.2.4, TIS equation);
 *   - log pi(a_t | s_t) of the sampled token, a log-softmax over the vocabulary
 *     (Sec. 2.3, the policy pi_theta(a_t | s_t)), from logits rows or through a
 *     fused LM head (logits = hidden W^T formed on the tensor cores, never stored);
 *   - PPO's masked GAE, per-token advantages and masked value loss (Sec. 2.3.1,
 *     Sec. 2.3.4);
 *   - rollout-level prefix trees of captured model calls, packed once per shared
 *     prefix, and the advantages and counts of their tokens in any order
 *     (Sec. 3.2.1-3.2.3);
 *   - sequence-level importance weights (Sec. 3.2.4) and batch summaries of the
 *     per-token statistics (entropy, clip fraction; Sec. 4);
 *   - a self-test of the failure path that every bounded device wait shares
 *     (rl_selftest_bounded_wait).
 *
 * Conventions shared by every entry point:
 *   - Array arguments are DEVICE pointers owned by the caller (the one
 *     exception, rl_prefix_tree_build_batch, is a host function on host
 *     pointers). The library never allocates device memory, frees or
 *     synchronises (except rl_query_status, which synchronises the given
 *     stream). All work is enqueued on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream).
 *   - Argument errors that the host can see return a status before anything is
 *     launched; rl_last_error_message() then describes the problem.
 *   - Errors that only the device can see (a token id outside [0, V), a
 *     trajectory index outside [0, n_traj), inconsistent offsets, a bounded
 *     wait that ran out) set bits of a status word kept in the workspace;
 *     kernels never trap. Read it with rl_query_status().
 *   - The loss returned is the NEGATED objective (the paper maximises the
 *     objective; the library gives a loss to minimise and its gradient).
 *   - Logits rows are dense, row-major, row r starting at element r * ld.
 *     bf16 values are IEEE bfloat16 bit patterns.
 */
#ifndef RL_LOSS_H
#define RL_LOSS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t. */
typedef struct CUstream_st* rl_stream_t;

typedef enum rl_status {
  RL_OK = 0,
  RL_ERR_INVALID_ARG = 1,         /* null pointer, negative size, bad enum value, ld < V ... */
  RL_ERR_UNSUPPORTED = 2,         /* a shape the kernels do not handle (e.g. V too large) */
  RL_ERR_ALIGNMENT = 3,           /* a base pointer that must be 16-byte aligned is not */
  RL_ERR_WORKSPACE_TOO_SMALL = 4, /* ws_bytes below rl_workspace_size(...) */
  RL_ERR_CUDA = 5,                /* a CUDA runtime call failed; see rl_last_error_message() */
  RL_ERR_DEVICE_CHECK = 6,        /* rl_query_status: a device-side check failed */
  RL_ERR_TIMEOUT = 7              /* rl_query_status: a bounded device wait ran out */
} rl_status;

typedef enum rl_dtype { RL_BF16 = 0, RL_F32 = 1 } rl_dtype;

/* How per-token terms are weighted into the batch loss (the coefficient c_i of
 * trajectory i, so that loss = sum_t c_{i(t)} M_t l_t). */
typedef enum rl_loss_agg {
  /* c_i = 1 / (N * L_i), N = number of valid trajectories with L_i > 0: the
   * per-trajectory token mean of Sec. 2.3.2, then the mean over trajectories. */
  RL_AGG_SEQ_MEAN_TOKEN_MEAN = 0,
  RL_AGG_TOKEN_MEAN = 1, /* c_i = 1 / sum_valid L_i */
  RL_AGG_TOKEN_SUM = 2   /* c_i = 1 */
} rl_loss_agg;

/* Bits of the device status word. */
enum {
  RL_DEV_BAD_TOKEN = 1,   /* a token id outside [0, V); that row gets no loss and a zero gradient */
  RL_DEV_BAD_TRAJ = 2,    /* token_traj outside [0, n_traj); same treatment */
  RL_DEV_BAD_OFFSETS = 4, /* group / trajectory offsets not non-decreasing within range */
  RL_DEV_TIMEOUT = 8,     /* a bounded wait for an asynchronous copy ran out */
  RL_DEV_BAD_VALUE = 16   /* a non-finite or out-of-range input value (rl_sequence_is_weights) */
};

typedef struct rl_loss_params {
  float clip_eps_low;  /* ratio clipped to [1 - clip_eps_low, 1 + clip_eps_high] */
  float clip_eps_high;
  float kl_coef;       /* beta; used when kl_estimator == 3 and ref_logp != NULL */
  int32_t kl_estimator;/* 0 = no KL term, 3 = k3: exp(r - logp) - (r - logp) - 1 */
  float entropy_coef;  /* alpha >= 0: loss -= alpha * H_t (entropy bonus) */
  float tis_cap;       /* c-bar; <= 0 or rollout_logp == NULL disables the TIS weight */
  float adv_eps;       /* epsilon added to sigma in the advantage denominator */
  int32_t loss_agg;    /* rl_loss_agg */
  int32_t token_level_adv; /* 0: adv is float [n_traj], A_{i(t)} per trajectory (GRPO, Sec. 2.3.2);
                              1: adv is float [rows], one A_t per row, e.g. from rl_masked_gae
                              (PPO, Sec. 2.3.1); coef stays per trajectory */
} rl_loss_params;

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t rl_version(void);

/* Text of the last error returned on this host thread ("" if none). The
 * pointer stays valid until the next call into the library on this thread. */
const char* rl_last_error_message(void);

/* Workspace bytes needed by calls on at most `max_rows` logits rows of
 * vocabulary V (D = hidden size of the fused head, 0 if unused). The
 * workspace holds the device status word and per-row loss contributions; with
 * D > 0 it also holds the fused head's buffers, the largest being the bf16
 * gradient of the logits of ONE chunk of min(max_rows, 4096) tokens
 * (min(max_rows, 4096) * ceil(V / 8) * 8 * 2 bytes: 1.24 GB at V = 151,936).
 * This is the smallest workspace of rl_fused_head_loss_fwd_bwd. */
size_t rl_workspace_size(int64_t max_rows, int64_t V, int64_t D);

/* Workspace bytes with which rl_fused_head_loss_fwd_bwd on up to T tokens keeps the
 * bf16 logits gradient of up to group_tokens tokens at once (rounded up to whole
 * chunks of 4,096 tokens; group_tokens <= 4096 gives rl_workspace_size(T, V, D)).
 * The fused head then runs its dH and dW products once per group instead of once
 * per chunk, which reads and writes the fp32 d_weight fewer times, at the cost of
 * ceil(V / 8) * 8 * 2 bytes per token of the group. Any workspace size between the
 * two works: the group is as many whole chunks as the workspace holds. */
size_t rl_fused_head_workspace_size(int64_t T, int64_t V, int64_t D, int64_t group_tokens);

/* Zero the workspace's 256-byte header: the status word and the finished-block
 * counters of the policy and value losses (which each launch leaves at zero
 * again). Call once after allocating a workspace, and again to clear a reported
 * device error. */
rl_status rl_workspace_init(void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * Self-test of the failure path (no counterpart in the paper): one CTA waits, through the
 * kernels' own bounded waits (the plain and the cluster-scope form), on an mbarrier that
 * nothing arrives at. Each wait gives up after limit_ns nanoseconds of %globaltimer (the
 * kernels use 2e9); the kernel then sets RL_DEV_TIMEOUT in the status word and returns, so
 * rl_query_status reports RL_ERR_TIMEOUT and the context stays usable (rl_workspace_init
 * clears the word). No fault, trap or unbounded wait is involved.
 *
 *   ws, ws_bytes  workspace (its status word is set), at least the 256-byte header
 *   limit_ns      in [1e3, 2e9]
 *   waited_ns     device uint64 (or NULL): receives the longest time the CTA spent waiting
 *                 (max with its previous value)
 */
rl_status rl_selftest_bounded_wait(void* ws, size_t ws_bytes, int64_t limit_ns, uint64_t* waited_ns,
                                   rl_stream_t stream);

/* Synchronise `stream`, then read the device status word into
 * *device_status_out (0 = no error; else RL_DEV_* bits). Returns RL_OK,
 * RL_ERR_DEVICE_CHECK or RL_ERR_TIMEOUT. The word is not cleared. */
rl_status rl_query_status(const void* ws, rl_stream_t stream, int32_t* device_status_out);

/*
 * Group-relative advantages and loss coefficients (Sec. 2.3.2 GRPO advantage
 * and objective; Sec. 3.2.3 rollout groups; Sec. 3.3 task-harness groups;
 * Sec. 3.4 discarded rollouts are left out of advantage estimation and
 * optimisation).
 *
 *   n_traj            number of trajectories n (>= 0)
 *   n_groups          number of groups (>= 0)
 *   group_offsets     int32 [n_groups + 1]: group g owns trajectories
 *                     [group_offsets[g], group_offsets[g+1]); non-decreasing, in [0, n_traj]
 *   rewards           float [n_traj]: R_i
 *   traj_valid        uint8 [n_traj] or NULL (all valid): 0 = discarded rollout
 *   n_tokens          T, length of the packed token stream (>= 0)
 *   traj_offsets      int64 [n_traj + 1]: trajectory i owns tokens
 *                     [traj_offsets[i], traj_offsets[i+1]) of the packed stream
 *   mask              uint8 [T]: M_t (nonzero = trainable, policy-generated token)
 *   params            host pointer; adv_eps and loss_agg are used
 *   adv_out           float [n_traj]: A_i (0 for invalid trajectories, for
 *                     trajectories in no group, and for groups whose valid rewards
 *                     are all equal)
 *   coef_out          float [n_traj]: c_i per loss_agg (0 if invalid or L_i = 0)
 *   n_tok_out         int32 [n_traj]: L_i = sum of M_t over the trajectory (exact)
 *   token_traj_out    int32 [T] or NULL: owner trajectory of each token
 *   ws, ws_bytes      workspace (rl_workspace_size(0, 0, 0) bytes suffice)
 *
 * mu and sigma are taken over the valid members of each group in double
 * precision; outputs are rounded to float.
 */
rl_status rl_group_advantages(int32_t n_traj, int32_t n_groups, const int32_t* group_offsets,
                              const float* rewards, const uint8_t* traj_valid, int64_t n_tokens,
                              const int64_t* traj_offsets, const uint8_t* mask,
                              const rl_loss_params* params, float* adv_out, float* coef_out,
                              int32_t* n_tok_out, int32_t* token_traj_out, void* ws,
                              size_t ws_bytes, rl_stream_t stream);

/*
 * Forward-only log-probabilities of the sampled tokens (the pi_old / pi_ref
 * recompute of Sec. 3.2.4): for every row r,
 *   lse_r = log sum_v exp(z_rv), logp_r = z_{r,a_r} - lse_r, H_r = -sum_v p_rv log p_rv.
 *
 *   logits       [rows x ld] of `dtype`; base 16-byte aligned
 *   rows, V, ld  rows >= 0, 1 <= V <= ld; V at most 819,200 (bf16) or 409,600 (fp32): a
 *                row is spread over at most 16 CTAs of 100 KB (RL_ERR_UNSUPPORTED above)
 *   token_ids    int32 [rows]: a_r (out of range -> logp_r = NaN and RL_DEV_BAD_TOKEN)
 *   logp_out     float [rows]
 *   entropy_out  float [rows] or NULL (entropy work is skipped when NULL)
 *   lse_out      float [rows] or NULL
 * One streaming pass over the logits (online softmax, fp32 accumulation).
 */
rl_status rl_token_logprobs(const void* logits, rl_dtype dtype, int64_t rows, int64_t V, int64_t ld,
                            const int32_t* token_ids, float* logp_out, float* entropy_out,
                            float* lse_out, void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * Masked clipped policy loss over one microbatch of logits rows and its
 * gradient d loss / d logits (Sec. 2.3.1 PPO masked objective; Sec. 2.3.2 GRPO
 * objective with the KL penalty; Sec. 3.2.4 TIS weight).
 *
 * For each row t with M_t != 0 and c_{i(t)} != 0 (i(t) = token_traj[t]):
 *   logp = z_a - lse; rho = exp(logp - old_logp);
 *   surr = min(rho A, clip(rho, 1 - eps_low, 1 + eps_high) A);
 *   w = min(exp(old_logp - rollout_logp), tis_cap) if enabled, else 1 (no gradient);
 *   KL = exp(r - logp) - (r - logp) - 1 with r = ref_logp (k3), if enabled;
 *   l_t = -w surr + beta KL - alpha H;
 *   loss += c_i l_t;
 *   grad_v = c_i [g (delta_{v,a} - p_v) + alpha p_v (log p_v + H)],
 *   g = -w A rho act + beta (1 - exp(r - logp)), act = 0 iff
 *   (A > 0 and rho > 1 + eps_high) or (A < 0 and rho < 1 - eps_low).
 * Every other row gets an exactly-zero gradient row and contributes nothing.
 * Logits at -inf have probability 0 (and a zero gradient); a NaN logit makes its own row's
 * loss term, statistics and gradient NaN (so the loss is NaN) and leaves the other rows alone.
 *
 *   logits        [rows x ld] of `dtype`, base 16-byte aligned
 *   rows, V, ld   rows >= 0, 1 <= V <= ld; V at most 819,200 (bf16) or 409,600 (fp32), as
 *                 for rl_token_logprobs (RL_ERR_UNSUPPORTED above)
 *   token_ids     int32 [rows]
 *   mask          uint8 [rows]: M_t
 *   token_traj    int32 [rows]: trajectory of each row (index into adv / coef)
 *   n_traj        length of adv and coef
 *   adv, coef     float [n_traj]: A_i and c_i for the WHOLE batch (from
 *                 rl_group_advantages), so a trajectory split across
 *                 microbatches keeps its normaliser
 *   old_logp      float [rows]: log pi_old(a_t | s_t)
 *   ref_logp      float [rows] or NULL: log pi_ref(a_t | s_t) for the KL term
 *   rollout_logp  float [rows] or NULL: log pi_rollout(a_t | s_t) for TIS
 *   params        host pointer
 *   grad_out      [rows x ld] of `dtype`, base 16-byte aligned; may equal logits
 *                 (in place); elements v >= V of each row are not written
 *   loss_accum    double [1] on the device: the microbatch loss is ADDED to it
 *                 (deterministic: fixed-order reduction)
 *   token_stats   float [rows x 5] or NULL: (logp, rho, clipped flag, H, KL) for
 *                 active rows, zeros for the others
 *   ws, ws_bytes  workspace of at least rl_workspace_size(rows, V, 0) bytes
 */
rl_status rl_policy_loss_fwd_bwd(const void* logits, rl_dtype dtype, int64_t rows, int64_t V,
                                 int64_t ld, const int32_t* token_ids, const uint8_t* mask,
                                 const int32_t* token_traj, int32_t n_traj, const float* adv,
                                 const float* coef, const float* old_logp, const float* ref_logp,
                                 const float* rollout_logp, const rl_loss_params* params,
                                 void* grad_out, double* loss_accum, float* token_stats, void* ws,
                                 size_t ws_bytes, rl_stream_t stream);

/*
 * Fused LM head: the same objective as rl_policy_loss_fwd_bwd with the logits
 * Z = hidden W^T computed tile by tile on the tensor cores and never written to
 * memory; returns the loss and the gradients with respect to hidden and W
 * (pi_theta(a_t | s_t) of Sec. 2.3 as the softmax of the LM head's output;
 * objective of Sec. 2.3.2 with the TIS weight of Sec. 3.2.4).
 *
 *   hidden        bf16 [T x D], row-major, 16-byte aligned
 *   weight        bf16 [V x D], row-major (row v = output embedding of token v)
 *   T, D, V       T >= 0, D >= 64 and a multiple of 64 (at most 65,536), 1 <= V <= 524,288
 *                 (RL_ERR_UNSUPPORTED otherwise)
 *   token_ids, mask, token_traj, n_traj, adv, coef, old_logp, ref_logp,
 *   rollout_logp, params, loss_accum, token_stats
 *                 as for rl_policy_loss_fwd_bwd, with one row per token
 *   d_hidden      [T x D] of d_hidden_dtype (RL_BF16 or RL_F32): d loss / d hidden
 *                 (overwritten; zero rows for tokens that are not trained on)
 *   d_weight      float [V x D]: d loss / d W is ADDED to it
 *   ws, ws_bytes  workspace of at least rl_workspace_size(T, V, D) bytes; it holds,
 *                 among others, the gradient of the logits (bf16) of one chunk of
 *                 4,096 tokens, or of a group of several chunks when ws_bytes allows
 *                 (rl_fused_head_workspace_size), consumed by the dH and dW products
 * Tokens are processed in chunks of 4,096: per chunk, one tensor-core pass forms the
 * logits tile by tile, folds them into softmax partials and keeps exp(z - tile max)
 * in bf16 with the tile maxima; a per-token merge evaluates the objective; an in-place
 * rescale turns the kept values into the logits' gradient. After the last chunk of
 * each group (each chunk, with the smallest workspace), two tensor-core products give
 * the group's dH and add its dW (fp32, one addition per element and group, in chunk
 * order: deterministic). The groups follow ws_bytes, so the rounding of d_weight and
 * d_hidden (not their values up to rounding) depends on the workspace size; calls with
 * the same ws_bytes give the same bits. The logits of all T tokens are never held at once.
 */
rl_status rl_fused_head_loss_fwd_bwd(const void* hidden, const void* weight, int64_t T, int64_t D, int64_t V,
                                     const int32_t* token_ids, const uint8_t* mask, const int32_t* token_traj,
                                     int32_t n_traj, const float* adv, const float* coef, const float* old_logp,
                                     const float* ref_logp, const float* rollout_logp,
                                     const rl_loss_params* params, void* d_hidden, rl_dtype d_hidden_dtype,
                                     float* d_weight, double* loss_accum, float* token_stats, void* ws,
                                     size_t ws_bytes, rl_stream_t stream);

/*
 * Batch summary of the per-token statistics written by rl_policy_loss_fwd_bwd /
 * rl_fused_head_loss_fwd_bwd (token_stats rows (logp, rho, clipped, H, KL)): over the trained
 * tokens (M_t != 0, owner in range, c_{i(t)} != 0) it ADDS to summary_accum
 *   [0] the number of trained tokens, [1] the number clipped, [2] sum of H_t,
 *   [3] sum of KL_t, [4] sum of rho_t
 * (the clip fraction and the mean policy entropy tracked during training, Sec. 4). Call it
 * once per microbatch with the same accumulator; divide by [0] for the means.
 *
 *   rows, token_stats  float [rows x 5]
 *   mask, token_traj, n_traj, coef   as for rl_policy_loss_fwd_bwd
 *   summary_accum      double [5] on the device
 *   ws, ws_bytes       rl_workspace_size(0, 0, 0) bytes suffice (status word)
 * One launch of one 8-CTA cluster, a fixed assignment of rows to threads and a fixed order of
 * the partial sums, in double precision: deterministic.
 */
rl_status rl_token_stats_summary(int64_t rows, const float* token_stats, const uint8_t* mask,
                                 const int32_t* token_traj, int32_t n_traj, const float* coef,
                                 double* summary_accum, void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * Masked generalised advantage estimation for PPO (Sec. 2.3.1, masked GAE and TD
 * residual; Sec. 2.3.4, PPO with each trajectory backed up on its own), per
 * trajectory of the packed stream:
 *   printed reading (skip_masked = 0):
 *     A_t = sum_l (gamma lambda)^l delta_{t+l} M_{t+l},
 *     delta_t = r_t + gamma V_{t+1} M_{t+1} - V_t   (V past the trajectory's end = 0);
 *   skip reading (skip_masked = 1): the same recursion over the trajectory's
 *     trainable tokens only (masked tokens are stepped over, their rewards ignored,
 *     delta_t bootstraps from the next trainable token's value). With gamma =
 *     lambda = 1 and the reward at the final trainable token it gives
 *     A_t = R_i - V_t, the form Sec. 2.3.4 states; the printed reading does not
 *     when the mask has gaps. Without masked tokens the two agree.
 *   returns G_t = A_t + V_t (the targets of the value loss).
 *
 *   n_traj, traj_offsets  int64 [n_traj + 1]: trajectory i owns tokens
 *                         [traj_offsets[i], traj_offsets[i+1]) (non-decreasing, in [0, n_tokens];
 *                         else RL_DEV_BAD_OFFSETS and that trajectory is skipped)
 *   mask                  uint8 [n_tokens]: M_t
 *   values                float [n_tokens]: V(s_t) of the value model that scored the rollout
 *   token_rewards         float [n_tokens] or NULL: r_t
 *   traj_rewards          float [n_traj] or NULL: R_i, added to r_t at trajectory i's last
 *                         token with M_t = 1 (none if it has no such token)
 *   gamma, gae_lambda     in [0, 1]
 *   adv_out               float [n_tokens]: A_t, 0 at masked tokens
 *   returns_out           float [n_tokens] or NULL: G_t, 0 at masked tokens
 *   ws, ws_bytes          workspace (rl_workspace_size(0, 0, 0) bytes suffice)
 * Tokens outside every trajectory's span are not written. fp32 arithmetic: one CTA per
 * trajectory runs a block-wide suffix scan of the recursion's affine maps.
 */
rl_status rl_masked_gae(int32_t n_traj, const int64_t* traj_offsets, int64_t n_tokens, const uint8_t* mask,
                        const float* values, const float* token_rewards, const float* traj_rewards, float gamma,
                        float gae_lambda, int32_t skip_masked, float* adv_out, float* returns_out, void* ws,
                        size_t ws_bytes, rl_stream_t stream);

/*
 * Masked value loss of PPO (Sec. 2.3.1, masked mean-squared critic loss) over one
 * microbatch of rows:
 *   loss += sum_t c_{i(t)} M_t (V_t - G_t)^2,   d_values_t = 2 c_{i(t)} M_t (V_t - G_t).
 * With coef from rl_group_advantages under RL_AGG_TOKEN_MEAN this is the token mean
 * E_t of the paper. Rows with M_t = 0 or c = 0 get d_values_t = 0.
 *
 *   values, returns   float [rows]: V_t of the current value model, G_t (from rl_masked_gae)
 *   mask, token_traj  uint8 [rows], int32 [rows] (token_traj outside [0, n_traj) on a row
 *                     with M_t != 0 sets RL_DEV_BAD_TRAJ and the row contributes nothing)
 *   coef              float [n_traj]
 *   d_values          float [rows]
 *   loss_accum        double [1] on the device, added to (fixed-order reduction)
 *   ws, ws_bytes      workspace of at least rl_workspace_size(rows, 0, 0) bytes
 */
rl_status rl_value_loss_fwd_bwd(int64_t rows, const float* values, const float* returns, const uint8_t* mask,
                                const int32_t* token_traj, int32_t n_traj, const float* coef, float* d_values,
                                double* loss_accum, void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * rl_group_advantages for tokens in any order (tree-packed batches, Sec. 3.2.3): the owner
 * of every token is given instead of contiguous spans, so a rollout's deduplicated prefix-tree
 * tokens (rl_prefix_tree_build_batch) or an interleaved packing can be used directly. The
 * advantage A_i of rollout i (Sec. 3.2.3, GRPO over the n rollouts of a task) is assigned to
 * all its trainable token nodes, each shared prefix token once; L_i counts those nodes.
 *
 *   n_traj, n_groups, group_offsets, rewards, traj_valid, params, adv_out, coef_out
 *                  as for rl_group_advantages
 *   n_tokens       T
 *   token_traj     int32 [T]: owner of each token (any order); an owner outside [0, n_traj)
 *                  on a token with M_t != 0 sets RL_DEV_BAD_TRAJ and the token is not counted
 *   mask           uint8 [T]
 *   n_tok_out      int32 [n_traj]: L_i (overwritten; exact, independent of token order)
 *   ws, ws_bytes   rl_workspace_size(0, 0, 0) bytes suffice
 */
rl_status rl_group_advantages_by_owner(int32_t n_traj, int32_t n_groups, const int32_t* group_offsets,
                                       const float* rewards, const uint8_t* traj_valid, int64_t n_tokens,
                                       const int32_t* token_traj, const uint8_t* mask, const rl_loss_params* params,
                                       float* adv_out, float* coef_out, int32_t* n_tok_out, void* ws,
                                       size_t ws_bytes, rl_stream_t stream);

/*
 * PPO advantages with gamma = lambda = 1 for tokens in any order (Sec. 2.3.4: every
 * trajectory of a rollout receives R_i at its final token and is backed up on its own, so
 * A_t = R_i - V(s_t); on a prefix shared by several trajectories of a tree all of them give
 * the same value):
 *   A_t = R_{i(t)} - V_t and G_t = R_{i(t)} for M_t != 0, A_t = G_t = 0 otherwise.
 *
 *   n_tokens, token_traj, mask   as for rl_group_advantages_by_owner
 *   values         float [n_tokens]: V(s_t)
 *   rewards        float [n_traj]: R_i
 *   adv_out        float [n_tokens]
 *   returns_out    float [n_tokens] or NULL
 *   ws, ws_bytes   rl_workspace_size(0, 0, 0) bytes suffice
 */
rl_status rl_rollout_value_advantages(int64_t n_tokens, const int32_t* token_traj, const uint8_t* mask,
                                      const float* values, const float* rewards, int32_t n_traj, float* adv_out,
                                      float* returns_out, void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * Sequence-level importance weights (Sec. 3.2.4: the sequence-level importance ratio
 * between the training engine's pi_old and the rollout engine's pi_rollout, the
 * unbiased alternative to the token-level TIS weight), truncated at c-bar:
 *   S_i = sum over tokens t with owner i and M_t = 1 of (log pi_old(a_t) - log pi_rollout(a_t)),
 *   w_i = min(exp(S_i), cap)   (no truncation when cap <= 0).
 * Like the token-level weight, w_i scales the surrogate term only. For a positive weight
 * that is the same as scaling the advantage, so the weights are applied by scaling the
 * advantages handed to rl_policy_loss_fwd_bwd / rl_fused_head_loss_fwd_bwd (in place here,
 * if asked); the loss entry points are unchanged.
 *
 *   n_traj, n_tokens   units (trajectories, or rollouts of a tree-packed batch) and tokens of
 *                      the WHOLE batch (a unit's sum spans microbatches)
 *   token_traj         int32 [n_tokens]: owner of each token, any order (a unit's tokens need
 *                      not be contiguous); an owner outside [0, n_traj) on a token with
 *                      M_t != 0 sets RL_DEV_BAD_TRAJ and the token is skipped
 *   mask               uint8 [n_tokens]
 *   old_logp, rollout_logp  float [n_tokens]; a difference that is not finite or above 2^22
 *                      in magnitude sets RL_DEV_BAD_VALUE (it is clamped, NaN counts as 0)
 *   cap                c-bar
 *   weight_out         float [n_traj]: w_i
 *   log_ratio_out      float [n_traj] or NULL: S_i
 *   traj_adv_inout     float [n_traj] or NULL: A_i, multiplied by w_i in place
 *   token_adv_inout    float [n_tokens] or NULL: A_t (per-token advantages), multiplied by
 *                      w_{owner(t)} in place
 *   ws, ws_bytes       workspace of at least rl_workspace_size(n_traj, 0, 0) bytes
 * Each difference is taken in double and rounded to a multiple of 2^-40; the sums are
 * 64-bit integer additions, so the result is independent of the order in which the GPU
 * adds the tokens (bit-reproducible). |S_i error| <= (tokens of unit i) x 2^-41.
 */
rl_status rl_sequence_is_weights(int32_t n_traj, int64_t n_tokens, const int32_t* token_traj, const uint8_t* mask,
                                 const float* old_logp, const float* rollout_logp, float cap, float* weight_out,
                                 float* log_ratio_out, float* traj_adv_inout, float* token_adv_inout, void* ws,
                                 size_t ws_bytes, rl_stream_t stream);

/*
 * Forward-only log-probabilities through the fused LM head (the pi_old / pi_ref
 * recompute of Sec. 3.2.4 when pi's logits are the LM head's output): for every
 * token t, with z_t = hidden_t W^T formed tile by tile on the tensor cores and
 * never written to memory,
 *   lse_t = log sum_v exp(z_tv), logp_t = z_{t,a_t} - lse_t, H_t = -sum_v p_tv log p_tv.
 *
 *   hidden, weight, T, D, V   as for rl_fused_head_loss_fwd_bwd
 *   token_ids    int32 [T]: a_t (out of range -> logp_t = NaN and RL_DEV_BAD_TOKEN)
 *   logp_out     float [T]
 *   entropy_out  float [T] or NULL (entropy work is skipped when NULL)
 *   lse_out      float [T] or NULL
 *   ws, ws_bytes workspace; rl_workspace_size(T, V, D) bytes always suffice (the
 *                call uses the status word and 32 * ceil(V / 4096) * min(T, 4096)
 *                bytes of softmax partials after it: two per token and 4,096-entry
 *                vocabulary block)
 * One tensor-core pass per chunk of 4,096 tokens, then a per-token merge of the
 * vocabulary blocks' partials in fixed order (deterministic).
 */
rl_status rl_fused_head_token_logprobs(const void* hidden, const void* weight, int64_t T, int64_t D, int64_t V,
                                       const int32_t* token_ids, float* logp_out, float* entropy_out,
                                       float* lse_out, void* ws, size_t ws_bytes, rl_stream_t stream);

/*
 * Allocation-free form of rl_policy_loss_fwd_bwd (no counterpart in the paper:
 * it exists for callers that cannot allocate device memory, e.g. code inside a
 * memory pool that forbids cudaMalloc during a training step, or a plugin that
 * only receives pointers from its host application).
 *
 * Same arguments and results as rl_policy_loss_fwd_bwd, without the workspace:
 * the library uses its own fixed workspace, a 1 MiB + 256 B array in device
 * global memory that every GPU loading the library holds until process exit.
 * The call allocates nothing and calls no allocating routine.
 *
 *   rows           at most 131072; larger microbatches return RL_ERR_UNSUPPORTED
 *                  before anything is launched
 *   device_status  int32 [1] on the device, or NULL: receives the call's device
 *                  status word (0 or RL_DEV_* bits) when the call completes on
 *                  `stream`
 *
 * The first call on a device looks up the array's device address (once per
 * device, with that device current) and the library keeps it for the life of
 * the process; make that first call before any stream capture, and make no call
 * after a cudaDeviceReset of that device (the kept address would be stale).
 * Every call shares the one array. Each call first clears the array's 256-byte
 * header (the status word and the loss kernel's finished-cluster counter), so a
 * call is not affected by what an earlier call left there; calls that overlap on
 * the GPU (for example on two streams at once) race on the array, give wrong
 * losses, and must be serialised by the caller.
 */
rl_status rl_policy_loss_fwd_bwd_noalloc(const void* logits, rl_dtype dtype, int64_t rows, int64_t V,
                                         int64_t ld, const int32_t* token_ids, const uint8_t* mask,
                                         const int32_t* token_traj, int32_t n_traj, const float* adv,
                                         const float* coef, const float* old_logp, const float* ref_logp,
                                         const float* rollout_logp, const rl_loss_params* params,
                                         void* grad_out, double* loss_accum, float* token_stats,
                                         int32_t* device_status, rl_stream_t stream);

/*
 * Rollout-level prefix trees for a batch of rollouts, packed into one deduplicated token
 * stream (HOST function: every pointer here is a host pointer; nothing touches the GPU).
 * Sec. 3.2.1 "Prefix Tree Construction": the captured model calls (x_i, y_i) of a rollout
 * form a tree rooted at the initial task prompt; each call is attached to the existing node
 * whose accumulated history is the longest prefix of x_i (the earliest node on ties), and the
 * part of x_i past that history is the harness content in between (tool outputs, environment
 * feedback). Sec. 3.2.2 "Trajectory Extraction and Filtering": a rollout whose tree has more
 * than max_leaves leaves (max_leaves > 0) is discarded; auxiliary calls (subagent, context
 * compaction) are removed with their subtrees; the root's children are grouped into segments
 * by equal input (a compaction starts a new one) and in each segment only the leaf with the
 * longest history is kept (the others are dead leaves of retries). Sec. 3.2.3: the kept
 * trajectories' nodes are written once each, so shared prefixes count once in the loss.
 *
 *   n_rollouts
 *   prompt_offsets, prompt_tokens  CSR [n_rollouts + 1]: rollout r's task prompt
 *   call_offsets                   int32 [n_rollouts + 1]: rollout r owns calls
 *                                  [call_offsets[r], call_offsets[r+1]) in capture order
 *   x_offsets, x_tokens            CSR [n_calls + 1]: each call's input context
 *   y_offsets, y_tokens            CSR [n_calls + 1]: each call's response
 *   aux                            uint8 [n_calls] or NULL: 1 = auxiliary call
 *   max_leaves                     <= 0: no limit
 *   n_threads                      host threads (<= 1: the calling thread only)
 *   capacity                       length of the per-token outputs
 * Per packed token (rollouts in order, each rollout's kept nodes in depth-first preorder,
 * children in creation order):
 *   tokens_out     int32: token id
 *   mask_out       uint8: 1 for response tokens, 0 for prompt and harness tokens (M_t)
 *   parent_out     int64: position of the previous token on the token's path, -1 for the
 *                  first prompt token (the row whose logits predicted this token)
 *   depth_out      int32 or NULL: index of the token along its path (position id)
 *   owner_out      int32 or NULL: rollout index (token_traj of the loss entry points)
 *   node_call_out  int32 or NULL: global call index of the token's node, -1 for the prompt
 * Per kept leaf (rollouts in order, preorder within a rollout), at most n_calls:
 *   leaf_call_out  int32 or NULL: global call index of the leaf
 *   leaf_end_out   int64 or NULL: position of the leaf's last token (-1 if its path is empty)
 *   leaf_offsets_out int64 [n_rollouts + 1] or NULL
 * Per rollout:
 *   stats_out            rl_tree_stats [n_rollouts] or NULL
 *   rollout_offsets_out  int64 [n_rollouts + 1] or NULL: rollout r's tokens are
 *                        [rollout_offsets[r], rollout_offsets[r+1]) (empty if discarded)
 *   n_tokens_out         total packed tokens (always written)
 * When the packed stream is longer than capacity the call returns
 * RL_ERR_WORKSPACE_TOO_SMALL after writing n_tokens_out, stats and offsets, so that a caller
 * can size the outputs and call again (capacity 0 with NULL outputs is a size query).
 * Offsets must be non-decreasing (RL_ERR_INVALID_ARG otherwise). The function allocates host
 * memory for its temporary trees.
 */
typedef struct rl_tree_stats {
  int32_t valid;          /* 0: discarded for over-branching */
  int32_t n_leaves;       /* leaves of the whole tree (auxiliary calls included) */
  int32_t n_kept_leaves;  /* trajectories kept for training */
  int32_t n_unplaced;     /* calls whose input does not start with the prompt */
  int64_t n_tokens;       /* packed tokens of the rollout */
  int64_t n_trainable;    /* of which responses (M_t = 1) */
} rl_tree_stats;

rl_status rl_prefix_tree_build_batch(int32_t n_rollouts, const int64_t* prompt_offsets, const int32_t* prompt_tokens,
                                     const int32_t* call_offsets, const int64_t* x_offsets, const int32_t* x_tokens,
                                     const int64_t* y_offsets, const int32_t* y_tokens, const uint8_t* aux,
                                     int32_t max_leaves, int32_t n_threads, int64_t capacity, int32_t* tokens_out,
                                     uint8_t* mask_out, int64_t* parent_out, int32_t* depth_out, int32_t* owner_out,
                                     int32_t* node_call_out, int32_t* leaf_call_out, int64_t* leaf_end_out,
                                     int64_t* leaf_offsets_out, rl_tree_stats* stats_out,
                                     int64_t* rollout_offsets_out, int64_t* n_tokens_out);

#ifdef __cplusplus
}
#endif

#endif /* RL_LOSS_H */
