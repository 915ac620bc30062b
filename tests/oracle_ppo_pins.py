"""Pins for the float64 PPO oracle (masked GAE, value loss): brute-force sums of the
printed estimator, closed forms (Monte-Carlo return at lambda = 1, one-step TD at
lambda = 0, R_i - V(s_t) at gamma = lambda = 1), a hand-worked example, invariants and
finite differences. Each pin is ``pin_xxx(P)`` of a PPO oracle module ``P``."""

from __future__ import annotations

import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _close(a, b, rtol=1e-12, atol=1e-12, what=""):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    if a.shape != b.shape or not np.all(np.abs(a - b) <= atol + rtol * np.abs(b)):
        raise AssertionError(f"{what}: {a} != {b}")


def _problem(seed, n=6, masked=0.4, max_len=9):
    rng = np.random.default_rng(seed)
    lengths = rng.integers(0, max_len + 1, size=n)
    offs = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    T = int(offs[-1])
    mask = (rng.random(T) >= masked).astype(np.uint8)
    values = rng.normal(0, 1, size=T)
    rewards = rng.normal(0, 1, size=T)
    return offs, mask, values, rewards


def pin_final_rewards_worked(P):
    """mask [1,1,0 | 0,0 | 1,0,1,0]: R_0 at token 1, none for the all-masked span, R_2 at 7."""
    offs = np.array([0, 3, 5, 9])
    mask = np.array([1, 1, 0, 0, 0, 1, 0, 1, 0], dtype=np.uint8)
    r = P.final_token_rewards(offs, mask, [2.0, 3.0, 5.0])
    _close(r, [0, 2, 0, 0, 0, 0, 0, 5, 0], what="final-token rewards")


def pin_gae_brute_force(P):
    """The printed estimator summed term by term: A_t = sum_l (gl)^l delta_{t+l} M_{t+l}."""
    for seed in range(4):
        offs, mask, V, r = _problem(seed)
        g, lam = 0.9, 0.7
        ref = np.zeros(len(V))
        for i in range(len(offs) - 1):
            s, e = offs[i], offs[i + 1]
            for t in range(s, e):
                if not mask[t]:
                    continue
                acc = 0.0
                for u in range(t, e):
                    nxt = V[u + 1] * mask[u + 1] if u + 1 < e else 0.0
                    acc += (g * lam) ** (u - t) * (r[u] + g * nxt - V[u]) * mask[u]
                ref[t] = acc
        adv, ret = P.masked_gae(offs, mask, V, r, g, lam)
        _close(adv, ref, rtol=1e-12, atol=1e-12, what="printed GAE vs brute force")
        _close(ret, np.where(mask != 0, ref + V, 0.0), rtol=1e-12, atol=1e-12, what="returns")


def pin_gae_skip_brute_force(P):
    """Skip reading, term by term over each trajectory's trainable positions."""
    for seed in range(4):
        offs, mask, V, r = _problem(10 + seed)
        g, lam = 0.8, 0.6
        ref = np.zeros(len(V))
        for i in range(len(offs) - 1):
            pos = [t for t in range(offs[i], offs[i + 1]) if mask[t]]
            for j, t in enumerate(pos):
                acc = 0.0
                for k in range(j, len(pos)):
                    nv = V[pos[k + 1]] if k + 1 < len(pos) else 0.0
                    acc += (g * lam) ** (k - j) * (r[pos[k]] + g * nv - V[pos[k]])
                ref[t] = acc
        adv, _ = P.masked_gae_skip(offs, mask, V, r, g, lam)
        _close(adv, ref, rtol=1e-12, atol=1e-12, what="skip GAE vs brute force")


def pin_gae_degenerate_form(P):
    """gamma = lambda = 1, reward R_i at the final trainable token: A_t = R_i - V(s_t) and
    G_t = R_i on every trainable token (Sec. 2.3.4), for any mask, in the skip reading."""
    offs, mask, V, _ = _problem(21, n=8, masked=0.5, max_len=12)
    R = np.random.default_rng(22).normal(0, 1, size=8)
    r = P.final_token_rewards(offs, mask, R)
    adv, ret = P.masked_gae_skip(offs, mask, V, r, 1.0, 1.0)
    owner = np.repeat(np.arange(8), np.diff(offs))
    M = mask != 0
    _close(adv[M], (R[owner] - V)[M], rtol=1e-12, atol=1e-12, what="A = R - V")
    _close(ret[M], R[owner][M], rtol=1e-12, atol=1e-12, what="G = R")
    assert np.all(adv[~M] == 0) and np.all(ret[~M] == 0)


def pin_gae_monte_carlo(P):
    """Unmasked trajectories, lambda = 1: A_t + V_t is the discounted return sum_l g^l r_{t+l};
    lambda = 0: A_t is the one-step TD residual. Both readings agree without masked tokens."""
    offs, _, V, r = _problem(31, n=5, masked=0.0)
    mask = np.ones(len(V), dtype=np.uint8)
    g = 0.95
    mc = np.zeros(len(V))
    td = np.zeros(len(V))
    for i in range(len(offs) - 1):
        s, e = offs[i], offs[i + 1]
        for t in range(s, e):
            mc[t] = sum(g ** (u - t) * r[u] for u in range(t, e))
            td[t] = r[t] + (g * V[t + 1] if t + 1 < e else 0.0) - V[t]
    for fn in (P.masked_gae, P.masked_gae_skip):
        adv, ret = fn(offs, mask, V, r, g, 1.0)
        _close(ret, mc, rtol=1e-11, atol=1e-12, what=f"{fn.__name__} MC return")
        adv0, _ = fn(offs, mask, V, r, g, 0.0)
        _close(adv0, td, rtol=1e-12, atol=1e-12, what=f"{fn.__name__} TD residual")
    a1, _ = P.masked_gae(offs, mask, V, r, 0.9, 0.8)
    a2, _ = P.masked_gae_skip(offs, mask, V, r, 0.9, 0.8)
    _close(a1, a2, rtol=1e-12, atol=1e-12, what="readings agree unmasked")


def pin_gae_golden(P):
    with open(os.path.join(GOLDEN, "ppo_gae_worked_example.json")) as f:
        ex = json.load(f)
    r = P.final_token_rewards(ex["traj_offsets"], np.array(ex["mask"]), ex["traj_rewards"])
    _close(r, ex["rewards_by_token"], what="golden rewards")
    for key, fn in (("printed", P.masked_gae), ("skip", P.masked_gae_skip)):
        adv, ret = fn(ex["traj_offsets"], np.array(ex["mask"]), ex["values"], r, ex["gamma"], ex["lambda"])
        _close(adv, ex[key]["adv"], what=f"golden {key} adv")
        _close(ret, ex[key]["returns"], what=f"golden {key} returns")


def pin_gae_trajectories_independent(P):
    """Changing one trajectory's inputs leaves every other trajectory's outputs unchanged."""
    offs, mask, V, r = _problem(41, n=6, masked=0.3)
    s, e = offs[2], offs[3]
    V2, r2 = V.copy(), r.copy()
    V2[s:e] += 5.0
    r2[s:e] -= 3.0
    for fn in (P.masked_gae, P.masked_gae_skip):
        a, _ = fn(offs, mask, V, r, 0.9, 0.9)
        b, _ = fn(offs, mask, V2, r2, 0.9, 0.9)
        keep = np.ones(len(V), bool)
        keep[s:e] = False
        assert np.array_equal(a[keep], b[keep]), fn.__name__


def pin_value_loss(P):
    """Closed forms and finite differences of sum_t c M (V - G)^2."""
    loss, g, _ = P.value_loss_fwd_bwd([3.0, 1.0], [1.0, 7.0], [1, 0], [0, 0], [0.5])
    _close([loss], [2.0], what="single token")
    _close(g, [2.0, 0.0], what="single token grad")
    rng = np.random.default_rng(51)
    T = 12
    V = rng.normal(0, 1, T)
    G = rng.normal(0, 1, T)
    mask = (rng.random(T) < 0.7).astype(np.uint8)
    tt = np.sort(rng.integers(0, 3, T))
    coef = np.array([0.1, 0.25, 0.05])
    loss0, g, _ = P.value_loss_fwd_bwd(V, V, mask, tt, coef)
    assert loss0 == 0.0
    loss, g, _ = P.value_loss_fwd_bwd(V, G, mask, tt, coef)
    h = 1e-6
    for t in range(T):
        Vp, Vm = V.copy(), V.copy()
        Vp[t] += h
        Vm[t] -= h
        fd = (P.value_loss_fwd_bwd(Vp, G, mask, tt, coef)[0] - P.value_loss_fwd_bwd(Vm, G, mask, tt, coef)[0]) / (2 * h)
        _close([g[t]], [fd], rtol=1e-6, atol=1e-9, what=f"value grad fd {t}")


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
