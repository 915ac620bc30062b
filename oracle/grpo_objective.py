"""Float64 CPU statement of the masked, group-relative clipped policy objective.

TEST INFRASTRUCTURE. This module is the oracle that the CUDA library is checked
against. Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import it. The product path
(``paper_2608_16798_gb300`` and its CUDA library) never imports, links or runs
anything here, and this module imports nothing from the product path.

Every function follows one passage of the paper (arXiv 2608.16798, "ClawGym II"):

* ``trajectory_token_counts``  -- the per-trajectory trainable-token count
  sum_t M_{i,t} that normalises each trajectory in the masked GRPO objective
  (Sec. 2.3.2, GRPO objective equation).
* ``group_advantages``         -- group-relative advantage with population
  standard deviation and epsilon added outside the square root (Sec. 2.3.2,
  GRPO advantage equation; restated for rollout groups in Sec. 3.2.3).
  Discarded rollouts are left out of the group statistics (Sec. 3.4,
  "Robust Sandbox Execution and Fault Handling").
* ``loss_coefficients``        -- the 1/G * 1/sum_t M weights of the masked GRPO
  objective (Sec. 2.3.2), extended to a batch of groups.
* ``row_statistics``           -- log pi_theta(a|s) of the sampled token as a
  log-softmax over the vocabulary, plus the policy entropy (Sec. 2.3, pi_theta).
* ``token_terms``              -- importance ratio, clipped surrogate (Sec. 2.3.1,
  PPO objective; Sec. 2.3.2 GRPO objective), k3 reference-KL penalty
  (Sec. 2.3.2), token-level truncated importance weight (Sec. 3.2.4, TIS
  equation) and the entropy bonus.
* ``policy_loss_fwd_bwd``      -- the loss (negated objective) over a packed
  microbatch and its exact gradient with respect to the logits.
* ``token_logprobs``           -- forward-only log-probabilities (the pi_old /
  pi_ref recompute of Sec. 3.2.4).
* ``fused_head_loss_fwd_bwd``  -- the same objective with logits = hidden @ W^T
  and gradients with respect to hidden and W.
* ``fused_head_logprobs``      -- forward-only log-probabilities of logits = hidden @ W^T.
* ``stats_summary``            -- batch sums of the per-token statistics (trained tokens,
  clipped tokens, entropy, KL, ratio): the clip fraction and the mean policy entropy that
  the paper tracks during training (Sec. 4, training dynamics).
* ``sequence_is_weights``      -- the sequence-level importance ratio between the training
  engine's and the rollout engine's policies, truncated at c-bar (Sec. 3.2.4, the
  sequence-level alternative to the token-level TIS weight).

Readings of the paper where it is silent (all documented with the library):

* clip range is asymmetric, [1 - eps_low, 1 + eps_high];
* the objective is maximised in the paper; this module returns the loss
  (negated objective) and its gradient;
* batch aggregation "seq-mean-token-mean": c_i = 1 / (N * L_i) where N counts
  valid trajectories with L_i > 0; alternatives token-mean (c = 1 / sum L) and
  token-sum (c = 1);
* a trajectory with no trainable token, or a discarded one, has c_i = 0 and
  is not counted in N;
* KL is the k3 estimator exp(r - logp) - (r - logp) - 1 on the sampled token,
  added to the loss with coefficient beta;
* the entropy bonus alpha * H (not part of the paper's objective) is
  subtracted from the loss;
* the truncated importance weight w_t scales the surrogate term only and
  carries no gradient;
* at a ratio exactly on a clip bound the surrogate gradient passes;
* the sequence-level ratio multiplies pi_old / pi_rollout over the trainable tokens
  (M_t = 1) of the unit that owns them (a trajectory, or a rollout's deduplicated tree);
  like the token-level weight it scales the surrogate only, which for a positive weight
  is the same as scaling the advantage; c-bar <= 0 leaves it untruncated.

Rows with M_t = 0, or whose trajectory has c_i = 0, contribute nothing to the
loss and get an exactly-zero gradient row.

The arithmetic is plain numpy float64; rows are processed in independent
chunks only to bound memory, which reorders nothing inside a row.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

AGG_SEQ_MEAN_TOKEN_MEAN = 0
AGG_TOKEN_MEAN = 1
AGG_TOKEN_SUM = 2


@dataclass(frozen=True)
class LossParams:
    """Hyper-parameters of the objective (names follow the paper's symbols)."""

    clip_eps_low: float = 0.2      # epsilon below 1 in clip(rho, 1-eps, 1+eps)
    clip_eps_high: float = 0.28    # epsilon above 1
    kl_coef: float = 0.0           # beta
    kl_estimator: int = 0          # 0 = off, 3 = k3 estimator
    entropy_coef: float = 0.0      # alpha, bonus: loss -= alpha * H
    tis_cap: float = 0.0           # c-bar of the TIS weight; <= 0 disables it
    adv_eps: float = 1e-6          # epsilon of the advantage denominator
    loss_agg: int = AGG_SEQ_MEAN_TOKEN_MEAN
    token_level_adv: bool = False  # adv holds one A_t per row (PPO, Sec. 2.3.1), not one per trajectory


# ----------------------------------------------------------------------------
# input decoding (exact): bf16 is carried as uint16 bit patterns
# ----------------------------------------------------------------------------

def decode_logits(raw: np.ndarray, dtype: str) -> np.ndarray:
    """Exact conversion of bf16 (uint16 bit patterns), float32 or float64 values to float64."""
    if dtype == "bf16":
        bits = np.asarray(raw, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
        return bits.view(np.float32).astype(np.float64)
    if dtype == "f32":
        return np.asarray(raw, dtype=np.float32).astype(np.float64)
    if dtype == "f64":
        return np.asarray(raw, dtype=np.float64)
    raise ValueError(f"unknown dtype {dtype!r}")


# ----------------------------------------------------------------------------
# A1: trainable tokens per trajectory (the 1 / sum_t M_{i,t} normaliser)
# ----------------------------------------------------------------------------

def trajectory_token_counts(mask: np.ndarray, traj_offsets: np.ndarray):
    """L_i = sum of M_t over the packed span of trajectory i, and the owner of each token.

    Returns (L int64[n], token_traj int64[T]).
    """
    mask = np.asarray(mask)
    offs = np.asarray(traj_offsets, dtype=np.int64)
    n = len(offs) - 1
    T = int(offs[-1]) if n >= 0 and len(offs) else 0
    L = np.zeros(n, dtype=np.int64)
    token_traj = np.full(T, -1, dtype=np.int64)
    for i in range(n):
        s, e = int(offs[i]), int(offs[i + 1])
        L[i] = int(np.count_nonzero(mask[s:e]))
        token_traj[s:e] = i
    return L, token_traj


# ----------------------------------------------------------------------------
# A2: group-relative advantages
# ----------------------------------------------------------------------------

def group_advantages(rewards, group_offsets, traj_valid=None, adv_eps: float = 1e-6):
    """A_i = (R_i - mu_g) / (sigma_g + eps) over the valid members of each group.

    mu_g is the mean and sigma_g the population standard deviation (1/k inside
    the square root) of the rewards of the k valid trajectories of group g.
    Invalid trajectories get A_i = 0 and are not part of mu or sigma. A group
    whose valid rewards are all bitwise equal gets A = 0 for every member.
    """
    rewards = np.asarray(rewards, dtype=np.float64)
    go = np.asarray(group_offsets, dtype=np.int64)
    n = len(rewards)
    valid = np.ones(n, dtype=bool) if traj_valid is None else np.asarray(traj_valid).astype(bool)
    adv = np.zeros(n, dtype=np.float64)
    for g in range(len(go) - 1):
        members = [i for i in range(int(go[g]), int(go[g + 1])) if valid[i]]
        k = len(members)
        if k == 0:
            continue
        R = [float(rewards[i]) for i in members]
        if all(r == R[0] for r in R):
            continue  # all equal -> zero advantage
        mu = math.fsum(R) / k
        sigma = math.sqrt(math.fsum((r - mu) ** 2 for r in R) / k)
        for i, r in zip(members, R):
            adv[i] = (r - mu) / (sigma + adv_eps)
    return adv


# ----------------------------------------------------------------------------
# A3: per-trajectory loss coefficients
# ----------------------------------------------------------------------------

def loss_coefficients(L, traj_valid=None, loss_agg: int = AGG_SEQ_MEAN_TOKEN_MEAN):
    """c_i such that loss = sum_t c_{i(t)} M_t l_t.

    seq-mean-token-mean: c_i = 1 / (N * L_i), N = #{valid i : L_i > 0}
    token-mean:          c_i = 1 / sum_{valid} L_i
    token-sum:           c_i = 1
    Trajectories that are invalid or have L_i = 0 get c_i = 0.
    """
    L = np.asarray(L, dtype=np.int64)
    n = len(L)
    valid = np.ones(n, dtype=bool) if traj_valid is None else np.asarray(traj_valid).astype(bool)
    counted = valid & (L > 0)
    c = np.zeros(n, dtype=np.float64)
    N = int(np.count_nonzero(counted))
    if N == 0:
        return c
    if loss_agg == AGG_SEQ_MEAN_TOKEN_MEAN:
        c[counted] = 1.0 / (N * L[counted].astype(np.float64))
    elif loss_agg == AGG_TOKEN_MEAN:
        c[counted] = 1.0 / float(L[counted].sum())
    elif loss_agg == AGG_TOKEN_SUM:
        c[counted] = 1.0
    else:
        raise ValueError(f"unknown loss_agg {loss_agg}")
    return c


def advantages_and_coefficients(rewards, group_offsets, traj_offsets, mask,
                                traj_valid=None, params: LossParams = LossParams()):
    """A1 + A2 + A3 together: returns (adv, coef, L, token_traj)."""
    L, token_traj = trajectory_token_counts(mask, traj_offsets)
    adv = group_advantages(rewards, group_offsets, traj_valid, params.adv_eps)
    coef = loss_coefficients(L, traj_valid, params.loss_agg)
    return adv, coef, L, token_traj


# ----------------------------------------------------------------------------
# B1: log-softmax statistics of one logits row (vectorised over a row chunk)
# ----------------------------------------------------------------------------

def row_statistics(z: np.ndarray, a: np.ndarray):
    """For rows z[r, :] (float64) and sampled ids a[r]:

    lse = log sum_v exp(z_v), log p_v = z_v - lse, logp = z_a - lse and the entropy
    H = -sum_v p_v log p_v with 0 log 0 = 0 (entries at -inf have p = 0 and add nothing).
    Returns (lse, logp, H, p, z_a).
    """
    z = np.atleast_2d(z)
    a = np.asarray(a, dtype=np.int64)
    m = z.max(axis=1, keepdims=True)
    s = np.exp(z - m).sum(axis=1, keepdims=True)
    lse = m + np.log(s)
    logp_all = z - lse
    p = np.exp(logp_all)
    rows = np.arange(z.shape[0])
    z_a = z[rows, a]
    logp = z_a - lse[:, 0]
    with np.errstate(invalid="ignore"):  # 0 * (-inf) in the branch that np.where discards
        H = -np.where(p > 0, p * logp_all, 0.0).sum(axis=1)
    return lse[:, 0], logp, H, p, z_a


# ----------------------------------------------------------------------------
# B2: per-token scalar terms
# ----------------------------------------------------------------------------

def token_terms(z_a, lse, H, old_logp, adv, params: LossParams,
                ref_logp=None, rollout_logp=None):
    """Per-token scalars of the objective for arrays of tokens.

    rho = exp(logp - old_logp); surr = min(rho A, clip(rho, 1-el, 1+eh) A);
    w = min(exp(old - rollout), c-bar) (TIS, else 1); KL = exp(r - logp) - (r - logp) - 1;
    l = -w surr + beta KL - alpha H.

    Also returns g = d l / d logp with the entropy part excluded:
    g = -w A rho act + beta (1 - exp(r - logp)), act = 0 iff
    (A > 0 and rho > 1 + eh) or (A < 0 and rho < 1 - el).
    """
    z_a = np.asarray(z_a, dtype=np.float64)
    lse = np.asarray(lse, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    A = np.asarray(adv, dtype=np.float64)
    el, eh = params.clip_eps_low, params.clip_eps_high
    # logp - old with the two large operands differenced first, so that rows
    # whose logits sit near -1e4 keep an accurate ratio
    log_ratio = (z_a - old) - lse
    logp = z_a - lse
    rho = np.exp(log_ratio)
    clipped_rho = np.minimum(np.maximum(rho, 1.0 - el), 1.0 + eh)
    surr = np.minimum(rho * A, clipped_rho * A)
    cut = ((A > 0) & (rho > 1.0 + eh)) | ((A < 0) & (rho < 1.0 - el))
    act = np.where(cut, 0.0, 1.0)
    if params.tis_cap > 0 and rollout_logp is not None:
        w = np.minimum(np.exp(old - np.asarray(rollout_logp, dtype=np.float64)), params.tis_cap)
    else:
        w = np.ones_like(rho)
    beta = params.kl_coef if params.kl_estimator == 3 and ref_logp is not None else 0.0
    if beta != 0.0:
        d = (np.asarray(ref_logp, dtype=np.float64) - z_a) + lse   # r - logp
        ed = np.exp(d)
        kl = ed - d - 1.0
        dkl = 1.0 - ed
    else:
        kl = np.zeros_like(rho)
        dkl = np.zeros_like(rho)
    alpha = params.entropy_coef
    ell = -w * surr + beta * kl - alpha * np.asarray(H, dtype=np.float64)
    g = -w * A * rho * act + beta * dkl
    return dict(logp=logp, rho=rho, surr=surr, act=act, cut=cut, w=w, kl=kl, ell=ell, g=g)


# ----------------------------------------------------------------------------
# B1..B4: loss and its gradient over a microbatch of logits rows
# ----------------------------------------------------------------------------

STAT_LOGP, STAT_RATIO, STAT_CLIPPED, STAT_ENTROPY, STAT_KL = range(5)


def policy_loss_fwd_bwd(logits, dtype, token_ids, mask, token_traj, adv, coef, old_logp,
                        params: LossParams = LossParams(), ref_logp=None, rollout_logp=None,
                        want_grad: bool = True, rows=None, chunk: int = 64):
    """Loss = sum_t c_{i(t)} M_t l_t over the rows of one microbatch and dLoss/dz.

    logits: [n_rows, V] bf16 bit patterns (uint16) or float32. token_traj maps each
    row to its trajectory; adv and coef are per-trajectory (with params.token_level_adv,
    adv holds one A_t per row, as in the PPO objective of Sec. 2.3.1). Returns
    (loss, grad float64 [n_rows, V] or None, stats float64 [n_rows, 5], contrib)
    where contrib[t] = c M l_t and stats hold (logp, rho, clipped, H, KL) for active
    rows (M_t = 1 and c != 0) and zeros elsewhere.  If ``rows`` is given, only
    those row indices are evaluated (grad then has len(rows) rows).
    """
    n_rows = logits.shape[0]
    sel = np.arange(n_rows) if rows is None else np.asarray(rows, dtype=np.int64)
    V = logits.shape[1]
    token_ids = np.asarray(token_ids, dtype=np.int64)
    mask = np.asarray(mask)
    token_traj = np.asarray(token_traj, dtype=np.int64)
    adv = np.asarray(adv, dtype=np.float64)
    coef = np.asarray(coef, dtype=np.float64)
    grad = np.zeros((len(sel), V), dtype=np.float64) if want_grad else None
    stats = np.zeros((len(sel), 5), dtype=np.float64)
    contrib = np.zeros(len(sel), dtype=np.float64)
    c_row = coef[token_traj[sel]]
    A_row = adv[sel] if params.token_level_adv else adv[token_traj[sel]]
    active = (mask[sel] != 0) & (c_row != 0.0)
    idx_active = np.nonzero(active)[0]
    alpha = params.entropy_coef
    for c0 in range(0, len(idx_active), chunk):
        loc = idx_active[c0:c0 + chunk]
        r = sel[loc]
        z = decode_logits(logits[r], dtype)
        a = token_ids[r]
        lse, logp, H, p, z_a = row_statistics(z, a)
        tt = token_terms(z_a, lse, H, np.asarray(old_logp)[r], A_row[loc], params,
                         None if ref_logp is None else np.asarray(ref_logp)[r],
                         None if rollout_logp is None else np.asarray(rollout_logp)[r])
        c = c_row[loc]
        contrib[loc] = c * tt["ell"]
        stats[loc, STAT_LOGP] = tt["logp"]
        stats[loc, STAT_RATIO] = tt["rho"]
        stats[loc, STAT_CLIPPED] = tt["cut"].astype(np.float64)
        stats[loc, STAT_ENTROPY] = H
        stats[loc, STAT_KL] = tt["kl"]
        if want_grad:
            # d l / d z_v = g (delta_{v,a} - p_v) + alpha p_v (z_v - lse + H)
            gz = -tt["g"][:, None] * p
            gz[np.arange(len(r)), a] += tt["g"]
            if alpha != 0.0:
                with np.errstate(invalid="ignore"):  # 0 * (-inf) in the discarded branch
                    gz += np.where(p > 0, alpha * p * (z - lse[:, None] + H[:, None]), 0.0)
            grad[loc] = c[:, None] * gz
    loss = math.fsum(contrib.tolist())
    return loss, grad, stats, contrib


def token_logprobs(logits, dtype, token_ids, chunk: int = 64):
    """Forward-only logp of the sampled ids, entropy and lse for every row."""
    n_rows = logits.shape[0]
    logp = np.zeros(n_rows)
    H = np.zeros(n_rows)
    lse = np.zeros(n_rows)
    token_ids = np.asarray(token_ids, dtype=np.int64)
    for r0 in range(0, n_rows, chunk):
        z = decode_logits(logits[r0:r0 + chunk], dtype)
        l, lp, h, _, _ = row_statistics(z, token_ids[r0:r0 + chunk])
        lse[r0:r0 + chunk] = l
        logp[r0:r0 + chunk] = lp
        H[r0:r0 + chunk] = h
    return logp, H, lse


# ----------------------------------------------------------------------------
# C: fused LM head (logits = hidden @ W^T, never handed to the caller)
# ----------------------------------------------------------------------------

def fused_head_loss_fwd_bwd(hidden_bf16, weight_bf16, token_ids, mask, token_traj, adv, coef,
                            old_logp, params: LossParams = LossParams(), ref_logp=None,
                            rollout_logp=None):
    """Z = H W^T (float64), then the objective on Z; d_hidden = dZ W, d_W = dZ^T H.

    hidden_bf16: uint16 [T, D]; weight_bf16: uint16 [V, D] (row v is the output
    embedding of token v). Returns (loss, d_hidden [T, D], d_weight [V, D], stats).
    """
    Hm = decode_logits(hidden_bf16, "bf16")
    Wm = decode_logits(weight_bf16, "bf16")
    Z = Hm @ Wm.T
    loss, dZ, stats, _ = policy_loss_fwd_bwd(Z, "f64", token_ids, mask, token_traj, adv, coef, old_logp,
                                             params, ref_logp, rollout_logp)
    d_hidden = dZ @ Wm
    d_weight = dZ.T @ Hm
    return loss, d_hidden, d_weight, stats


def fused_head_logprobs(hidden_bf16, weight_bf16, token_ids, chunk: int = 256):
    """Forward-only logp, entropy and lse of the sampled ids for logits Z = H W^T (float64):
    the pi_old / pi_ref recompute of Sec. 3.2.4 on the LM head's output."""
    Hm = decode_logits(hidden_bf16, "bf16")
    Wm = decode_logits(weight_bf16, "bf16")
    T = Hm.shape[0]
    token_ids = np.asarray(token_ids, dtype=np.int64)
    logp, H, lse = np.zeros(T), np.zeros(T), np.zeros(T)
    for r0 in range(0, T, chunk):
        Z = Hm[r0:r0 + chunk] @ Wm.T
        l, lp, h, _, _ = row_statistics(Z, token_ids[r0:r0 + chunk])
        lse[r0:r0 + chunk], logp[r0:r0 + chunk], H[r0:r0 + chunk] = l, lp, h
    return logp, H, lse


# ----------------------------------------------------------------------------
# Sequence-level importance weight (Sec. 3.2.4)
# ----------------------------------------------------------------------------

def sequence_is_weights(token_traj, mask, old_logp, rollout_logp, n_traj: int, cap: float):
    """S_i = sum over the trainable tokens t of unit i of (log pi_old - log pi_rollout);
    w_i = min(exp(S_i), c-bar) (no truncation when c-bar <= 0).

    Returns (w float64 [n_traj], S float64 [n_traj])."""
    tt = np.asarray(token_traj, dtype=np.int64)
    M = np.asarray(mask) != 0
    d = np.asarray(old_logp, dtype=np.float64) - np.asarray(rollout_logp, dtype=np.float64)
    S = np.zeros(n_traj)
    for i in range(n_traj):
        S[i] = math.fsum(d[(tt == i) & M].tolist())
    w = np.exp(S)
    if cap > 0:
        w = np.minimum(w, cap)
    return w, S


# ----------------------------------------------------------------------------
# Batch summaries of the per-token statistics (monitoring)
# ----------------------------------------------------------------------------

def stats_summary(stats, mask, token_traj, coef):
    """Over the trained tokens (M_t != 0 and c_{i(t)} != 0): (count, number clipped, sum of H,
    sum of KL, sum of rho) from per-token stats rows (logp, rho, clipped, H, KL)."""
    st = np.asarray(stats, dtype=np.float64).reshape(-1, 5)
    c = np.asarray(coef, dtype=np.float64)[np.asarray(token_traj, dtype=np.int64)]
    act = (np.asarray(mask) != 0) & (c != 0)
    return np.array([float(act.sum()), math.fsum(st[act, STAT_CLIPPED]), math.fsum(st[act, STAT_ENTROPY]),
                     math.fsum(st[act, STAT_KL]), math.fsum(st[act, STAT_RATIO])])
