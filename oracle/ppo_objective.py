"""Float64 CPU statement of the PPO parts of the method: masked GAE and the masked value loss.

TEST INFRASTRUCTURE. Like ``oracle.grpo_objective`` this module is the oracle
the CUDA library is checked against; only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU legs may import it, and it imports nothing from the
product path.

Every function follows one passage of the paper (arXiv 2608.16798, "ClawGym II"):

* ``final_token_rewards``  -- each trajectory receives its rollout's reward R_i
  at its own final token (Sec. 2.3.4, "Advantage Estimate for PPO").
* ``masked_gae``           -- the masked generalised advantage estimate of
  Sec. 2.3.1: A_t = sum_l (gamma lambda)^l delta_{t+l} M_{t+l} with
  delta_t = r_t + gamma V(s_{t+1}) M_{t+1} - V(s_t), per trajectory.
* ``masked_gae_skip``      -- the same estimate with the recursion stepping over
  masked positions (the reading under which gamma = lambda = 1 gives
  A_t = R_i - V(s_t), the form Sec. 2.3.4 states).
* ``value_loss_fwd_bwd``   -- the masked mean-squared value loss of Sec. 2.3.1,
  E_t[M_t (V(s_t) - G_t)^2], and its gradient with respect to V.

Readings where the paper is silent or at odds with itself:

* "final token" is the trajectory's last trainable token (M_t = 1): with the
  printed estimator a reward on a masked token would be multiplied by M = 0
  and lost;
* the bootstrap value past the end of a trajectory is 0 (trajectories are
  backed up independently, Sec. 2.3.4);
* the printed estimator keeps the discount running across masked positions and
  does not bootstrap into them (the M_{t+1} factor); with gaps in the mask it
  does not reduce to R_i - V(s_t) at gamma = lambda = 1. ``masked_gae_skip``
  is the reading that does: masked positions are stepped over, their rewards
  are ignored and delta_t bootstraps from the next trainable token's value;
* advantages and returns are reported as 0 at masked positions (the objective
  multiplies them by M_t = 0);
* the return is G_t = A_t + V(s_t);
* the value loss carries no 1/2 factor, as printed; its token weights are the
  caller's per-trajectory coefficients c_i (token-mean for the E_t of the paper).
"""

from __future__ import annotations

import math

import numpy as np


def final_token_rewards(traj_offsets, mask, traj_rewards):
    """r_t = R_i at the last token of trajectory i with M_t = 1, zero elsewhere."""
    offs = np.asarray(traj_offsets, dtype=np.int64)
    mask = np.asarray(mask)
    r = np.zeros(int(offs[-1]) if len(offs) else 0, dtype=np.float64)
    for i in range(len(offs) - 1):
        s, e = int(offs[i]), int(offs[i + 1])
        valid = np.nonzero(mask[s:e])[0]
        if len(valid):
            r[s + valid[-1]] += float(traj_rewards[i])
    return r


def masked_gae(traj_offsets, mask, values, rewards, gamma: float, lam: float):
    """Sec. 2.3.1 as printed, trajectory by trajectory, by the backward recursion
    A_t = M_t delta_t + gamma lambda A_{t+1} (A past the end = 0), which is the sum
    sum_l (gamma lambda)^l delta_{t+l} M_{t+l} term by term.

    Returns (adv, returns) float64 [T], both 0 at masked positions."""
    offs = np.asarray(traj_offsets, dtype=np.int64)
    M = np.asarray(mask) != 0
    Vv = np.asarray(values, dtype=np.float64)
    r = np.asarray(rewards, dtype=np.float64)
    adv = np.zeros(len(Vv))
    for i in range(len(offs) - 1):
        s, e = int(offs[i]), int(offs[i + 1])
        nxt = 0.0
        for t in range(e - 1, s - 1, -1):
            boot = Vv[t + 1] if (t + 1 < e and M[t + 1]) else 0.0
            delta = r[t] + gamma * boot - Vv[t]
            cur = (delta if M[t] else 0.0) + gamma * lam * nxt
            adv[t] = cur
            nxt = cur
    adv = np.where(M, adv, 0.0)
    return adv, np.where(M, adv + Vv, 0.0)


def masked_gae_skip(traj_offsets, mask, values, rewards, gamma: float, lam: float):
    """GAE over the trainable tokens of each trajectory only: with p_0 < p_1 < ... its
    positions with M = 1, delta_j = r_{p_j} + gamma V_{p_{j+1}} - V_{p_j} (V past the
    last = 0) and A_{p_j} = delta_j + gamma lambda A_{p_{j+1}}.

    Returns (adv, returns) float64 [T], both 0 at masked positions."""
    offs = np.asarray(traj_offsets, dtype=np.int64)
    M = np.asarray(mask) != 0
    Vv = np.asarray(values, dtype=np.float64)
    r = np.asarray(rewards, dtype=np.float64)
    adv = np.zeros(len(Vv))
    for i in range(len(offs) - 1):
        s, e = int(offs[i]), int(offs[i + 1])
        pos = [t for t in range(s, e) if M[t]]
        nxt_a, nxt_v = 0.0, 0.0
        for t in reversed(pos):
            delta = r[t] + gamma * nxt_v - Vv[t]
            adv[t] = delta + gamma * lam * nxt_a
            nxt_a, nxt_v = adv[t], Vv[t]
    return adv, np.where(M, adv + Vv, 0.0)


def value_loss_fwd_bwd(values, returns, mask, token_traj, coef):
    """loss = sum_t c_{i(t)} M_t (V_t - G_t)^2 and d loss / d V_t = 2 c M (V_t - G_t).

    Returns (loss, grad float64 [rows], contrib float64 [rows])."""
    Vv = np.asarray(values, dtype=np.float64)
    G = np.asarray(returns, dtype=np.float64)
    M = np.asarray(mask) != 0
    c = np.asarray(coef, dtype=np.float64)[np.asarray(token_traj, dtype=np.int64)]
    w = np.where(M, c, 0.0)
    d = Vv - G
    contrib = w * d * d
    return math.fsum(contrib.tolist()), 2.0 * w * d, contrib
