"""Pins for the float64 oracle: checks against closed forms, invariants, a library
special case, finite differences and a hand-worked example -- never against the
oracle's own formulas retyped.

Each pin is a function ``pin_xxx(O)`` of an oracle module ``O`` and raises
AssertionError on a mismatch. ``test_oracle_pins.py`` runs them on the real
oracle; ``test_oracle_mutations.py`` runs them on copies of the oracle with a
planted mistake and requires that at least one pin fails for every mistake.
"""

from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _close(a, b, rtol=1e-12, atol=1e-12, what=""):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    if a.shape != b.shape or not np.all(np.abs(a - b) <= atol + rtol * np.abs(b)):
        raise AssertionError(f"{what}: {a} != {b}")


# ---------------------------------------------------------------------------
# A1: trainable-token counts
# ---------------------------------------------------------------------------

def pin_counts_worked(O):
    """Hand count: mask [1,0,1,1,0 | - | 0,0,1], spans [0,5), [5,5), [5,8)."""
    mask = np.array([1, 0, 1, 1, 0, 0, 0, 1], dtype=np.uint8)
    offs = np.array([0, 5, 5, 8])
    L, tt = O.trajectory_token_counts(mask, offs)
    assert list(L) == [3, 0, 1], L
    assert list(tt) == [0, 0, 0, 0, 0, 2, 2, 2], tt


def pin_counts_conservation(O):
    """sum_i L_i = sum_t M_t and token owners are the spans' indices."""
    rng = np.random.default_rng(11)
    lengths = rng.integers(0, 9, size=40)
    offs = np.concatenate([[0], np.cumsum(lengths)])
    mask = (rng.random(offs[-1]) < 0.6).astype(np.uint8)
    L, tt = O.trajectory_token_counts(mask, offs)
    assert int(L.sum()) == int(mask.sum())
    assert np.array_equal(tt, np.repeat(np.arange(40), lengths))


# ---------------------------------------------------------------------------
# A2: group-relative advantages (population std, eps outside the sqrt)
# ---------------------------------------------------------------------------

def pin_adv_binary_closed_form(O):
    """k of G rewards are 1: mu = k/G, sigma = sqrt(mu (1 - mu)),
    A+ = (1 - mu)/(sigma + eps), A- = -mu/(sigma + eps)."""
    eps = 1e-6
    for G in (2, 4, 8, 16):
        for k in range(1, G):
            R = np.array([1.0] * k + [0.0] * (G - k))
            A = O.group_advantages(R, [0, G], None, eps)
            mu = k / G
            sig = math.sqrt(mu * (1 - mu))
            _close(A[:k], [(1 - mu) / (sig + eps)] * k, what=f"A+ G={G} k={k}")
            _close(A[k:], [-mu / (sig + eps)] * (G - k), what=f"A- G={G} k={k}")


def pin_adv_sum_and_square_sum(O):
    """With eps = 0: sum_S A_i = 0 and sum_S A_i^2 = k (population variance)."""
    rng = np.random.default_rng(5)
    for G in (3, 5, 8):
        R = rng.normal(size=G)
        A = O.group_advantages(R, [0, G], None, 0.0)
        assert abs(A.sum()) < 1e-12, A.sum()
        assert abs((A * A).sum() - G) < 1e-10, (A * A).sum()


def pin_adv_affine_invariance(O):
    """With eps = 0, A is unchanged by R -> a R + b (a > 0) and flips sign for a < 0."""
    R = np.array([0.3, 1.7, -2.0, 0.9, 0.0])
    A = O.group_advantages(R, [0, 5], None, 0.0)
    _close(O.group_advantages(3.0 * R + 7.0, [0, 5], None, 0.0), A, rtol=1e-12, atol=1e-12, what="affine")
    _close(O.group_advantages(-2.0 * R, [0, 5], None, 0.0), -A, rtol=1e-12, atol=1e-12, what="negated")


def pin_adv_groups_independent_and_invalid(O):
    """Groups are normalised separately; invalid members leave the statistics and get 0.
    {1, 0 | 1, 0, 100(invalid)} -> +-0.5/(0.5 + eps) in both groups."""
    eps = 1e-6
    R = np.array([1.0, 0.0, 1.0, 0.0, 100.0])
    valid = np.array([1, 1, 1, 1, 0], dtype=np.uint8)
    A = O.group_advantages(R, [0, 2, 5], valid, eps)
    a = 0.5 / (0.5 + eps)
    _close(A, [a, -a, a, -a, 0.0], what="groups/invalid")


def pin_adv_degenerate(O):
    """All-equal rewards, a single valid member and an all-invalid group give A = 0."""
    A = O.group_advantages(np.array([0.7] * 4 + [3.0] + [1.0, 2.0]), [0, 4, 5, 7],
                           np.array([1, 1, 1, 1, 1, 0, 0], np.uint8), 1e-6)
    assert np.all(A == 0.0), A


def pin_adv_golden(O):
    """tests/golden/grpo_advantage_example.json (hand-derived)."""
    with open(os.path.join(GOLDEN, "grpo_advantage_example.json")) as f:
        ex = json.load(f)
    for case in ex["cases"]:
        A = O.group_advantages(np.array(case["rewards"]), case["group_offsets"],
                               case.get("traj_valid"), case["eps"])
        _close(A, case["advantages"], rtol=1e-12, atol=1e-14, what=case["name"])


# ---------------------------------------------------------------------------
# A3: loss coefficients
# ---------------------------------------------------------------------------

def pin_coef_worked(O):
    """L = [2, 3, 0, 4], valid = [1, 1, 1, 0]: counted = {0, 1}, N = 2.
    seq-mean-token-mean: c = [1/4, 1/6, 0, 0]; token-mean: [1/5, 1/5, 0, 0]; token-sum: [1, 1, 0, 0]."""
    L = np.array([2, 3, 0, 4])
    v = np.array([1, 1, 1, 0], np.uint8)
    _close(O.loss_coefficients(L, v, O.AGG_SEQ_MEAN_TOKEN_MEAN), [0.25, 1 / 6, 0, 0], what="smtm")
    _close(O.loss_coefficients(L, v, O.AGG_TOKEN_MEAN), [0.2, 0.2, 0, 0], what="tm")
    _close(O.loss_coefficients(L, v, O.AGG_TOKEN_SUM), [1, 1, 0, 0], what="ts")


def pin_coef_normalisation(O):
    """sum_i c_i L_i = 1 under both mean modes (each counted token-weight sums to one)."""
    rng = np.random.default_rng(3)
    L = rng.integers(0, 50, size=64)
    v = (rng.random(64) < 0.8).astype(np.uint8)
    for agg in (O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN):
        c = O.loss_coefficients(L, v, agg)
        assert abs((c * L).sum() - 1.0) < 1e-12
        assert np.all(c[(v == 0) | (L == 0)] == 0)


# ---------------------------------------------------------------------------
# B1: log-softmax statistics
# ---------------------------------------------------------------------------

def pin_rowstats_uniform(O):
    """Uniform row: logp = -ln V, H = ln V, lse = z0 + ln V."""
    for V in (1, 2, 7, 4096):
        z = np.full((1, V), 1.25)
        lse, logp, H, p, _ = O.row_statistics(z, [V - 1])
        _close(logp, [-math.log(V)], what="uniform logp")
        _close(H, [math.log(V)], atol=1e-12, what="uniform H")
        _close(lse, [1.25 + math.log(V)], what="uniform lse")


def pin_rowstats_two_point(O):
    """z = (0, x): p1 = e^x/(1+e^x), H = ln(1+e^x) - x p1."""
    for x in (-3.0, 0.4, 5.0):
        lse, logp, H, p, _ = O.row_statistics(np.array([[0.0, x]]), [1])
        p1 = math.exp(x) / (1 + math.exp(x))
        _close(logp, [math.log(p1)], what="two-point logp")
        _close(H, [math.log1p(math.exp(x)) - x * p1], what="two-point H")


def pin_rowstats_spike(O):
    """One logit at +40, the rest at 0: logp = -ln(1 + (V-1) e^-40) for the spike."""
    V = 4096
    z = np.zeros((1, V))
    z[0, 17] = 40.0
    lse, logp, H, p, _ = O.row_statistics(z, [17])
    # lse sits next to 40, whose float64 ulp is 2^-47 = 7.1e-15: that bounds the absolute error
    _close(logp, [-math.log1p((V - 1) * math.exp(-40.0))], rtol=0, atol=2 ** -47, what="spike logp")
    q = math.exp(-40.0) / (1 + (V - 1) * math.exp(-40.0))
    Hc = -(1 - (V - 1) * q) * math.log(1 - (V - 1) * q) - (V - 1) * q * math.log(q)
    # the spike's own -p log p term carries the same 2^-47 absolute rounding of log p
    _close(H, [Hc], rtol=1e-6, atol=2 ** -47, what="spike H")


def pin_rowstats_library(O):
    """float64 torch.log_softmax (a library routine) and -sum p log p on random rows."""
    import torch

    rng = np.random.default_rng(0)
    z = rng.normal(0, 3, size=(6, 64))
    z[2, :32] = -1e4
    a = rng.integers(0, 64, size=6)
    a[2] = 40
    lse, logp, H, p, _ = O.row_statistics(z, a)
    ls = torch.log_softmax(torch.from_numpy(z), dim=1).numpy()
    _close(logp, ls[np.arange(6), a], rtol=1e-12, atol=1e-12, what="logp vs torch")
    pt = np.exp(ls)
    Ht = np.array([-math.fsum(pi * li for pi, li in zip(pr, lr) if pi > 0) for pr, lr in zip(pt, ls)])
    _close(H, Ht, rtol=1e-10, atol=1e-12, what="H vs -sum p log p")
    _close(p, pt, rtol=1e-10, atol=1e-300, what="p vs torch")


def pin_rowstats_neg_inf(O):
    """Entries at -inf have probability 0: lse, logp and H equal those of the row without them,
    and the loss gradient is exactly 0 there and equal to the reduced row's elsewhere
    (entropy bonus and KL on)."""
    rng = np.random.default_rng(21)
    V = 12
    z = rng.normal(0, 1.5, size=(3, V))
    drop = [np.array([1, 5, 6]), np.array([0]), np.array([2, 3, 4, 9, 11])]
    a = np.array([0, 4, 10])
    for r, dr in enumerate(drop):
        z[r, dr] = -np.inf
    keep = [np.setdiff1d(np.arange(V), dr) for dr in drop]
    lse, logp, H, _, _ = O.row_statistics(z, a)
    for r in range(3):
        zr = z[r, keep[r]][None, :]
        ar = np.array([int(np.nonzero(keep[r] == a[r])[0][0])])
        l2, lp2, h2, _, _ = O.row_statistics(zr, ar)
        _close([lse[r], logp[r], H[r]], [l2[0], lp2[0], h2[0]], rtol=1e-13, atol=1e-14, what=f"-inf row {r}")
        P = O.LossParams(entropy_coef=0.05, kl_coef=0.1, kl_estimator=3)
        old, ref = np.array([logp[r] + 0.1]), np.array([logp[r] - 0.2])
        _, g, _, _ = O.policy_loss_fwd_bwd(z[r:r + 1], "f64", a[r:r + 1], [1], [0], [1.3], [0.5], old, P, ref)
        _, g2, _, _ = O.policy_loss_fwd_bwd(zr, "f64", ar, [1], [0], [1.3], [0.5], old, P, ref)
        assert np.all(g[0, drop[r]] == 0.0)
        _close(g[0, keep[r]], g2[0], rtol=1e-12, atol=1e-15, what=f"-inf grad {r}")


def pin_rowstats_shift(O):
    """lse(z + c) = lse(z) + c; logp and H unchanged (c = -1e4 and +37)."""
    rng = np.random.default_rng(1)
    z = rng.normal(0, 2, size=(3, 50))
    a = [0, 10, 49]
    l0, lp0, h0, _, _ = O.row_statistics(z, a)
    for c in (-1e4, 37.0):
        l1, lp1, h1, _, _ = O.row_statistics(z + c, a)
        _close(l1, l0 + c, rtol=1e-14, atol=1e-9, what="shift lse")
        _close(lp1, lp0, rtol=0, atol=1e-9, what="shift logp")
        _close(h1, h0, rtol=0, atol=1e-9, what="shift H")


# ---------------------------------------------------------------------------
# B2: per-token terms
# ---------------------------------------------------------------------------

def _terms_at_ratio(O, rho, A, params, **kw):
    # logp = z_a - lse with lse = 0 so that logp = z_a; old chosen so rho = exp(logp - old)
    z_a = np.array([-1.3])
    old = z_a - math.log(rho)
    return O.token_terms(z_a, np.array([0.0]), np.array([0.0]), old, np.array([A]), params, **kw)


def pin_terms_clip_branches(O):
    """eps = (0.2, 0.28): the four clip cases of min(rho A, clip(rho) A)."""
    P = O.LossParams()
    cases = [  # rho, A, surrogate, gradient passes?
        (1.5, 1.0, 1.28, False), (0.5, 1.0, 0.5, True), (1.1, 1.0, 1.1, True),
        (0.5, -1.0, -0.8, False), (1.5, -1.0, -1.5, True), (0.9, -1.0, -0.9, True),
        (1.28 + 1e-9, 2.0, 2.56, False), (0.79, -2.0, -1.6, False),
    ]
    for rho, A, surr, passes in cases:
        t = _terms_at_ratio(O, rho, A, P)
        _close(t["rho"], [rho], rtol=1e-12, what="rho")
        _close(t["surr"], [surr], rtol=1e-9, what=f"surr rho={rho} A={A}")
        _close(t["ell"], [-surr], rtol=1e-9, what="ell")
        g = -A * rho if passes else 0.0
        _close(t["g"], [g], rtol=1e-9, atol=1e-15, what=f"g rho={rho} A={A}")


def pin_terms_bound_passes(O):
    """At rho exactly on the upper bound (A > 0) the gradient passes: g = -A rho."""
    P = O.LossParams(clip_eps_high=0.25)  # 1.25 and ln(1.25) round-trip well
    z_a = np.array([0.0])
    t = O.token_terms(z_a, np.array([0.0]), np.array([0.0]), np.array([0.0]), np.array([1.0]), P)
    _close(t["g"], [-1.0], what="rho=1 passes")
    t = O.token_terms(np.array([1.0]), np.array([1.0]), np.array([0.0]), np.array([0.0]),
                      np.array([1.0]), O.LossParams(clip_eps_high=0.0, clip_eps_low=0.0))
    _close(t["g"], [-1.0], what="rho on both bounds passes")


def pin_terms_kl_k3(O):
    """k3: r - logp = ln 2 -> KL = 1 - ln 2 and dKL/dlogp = -1; r = logp -> KL = 0 and 0 gradient."""
    P = O.LossParams(kl_coef=0.5, kl_estimator=3)
    z_a = np.array([-2.0, -2.0])
    ref = np.array([-2.0 + math.log(2.0), -2.0])
    t = O.token_terms(z_a, np.array([0.0, 0.0]), np.array([0.0, 0.0]), z_a, np.array([0.0, 0.0]),
                      P, ref_logp=ref)
    _close(t["kl"], [1 - math.log(2.0), 0.0], atol=1e-15, what="k3 value")
    _close(t["ell"], [0.5 * (1 - math.log(2.0)), 0.0], atol=1e-15, what="k3 loss")
    _close(t["g"], [0.5 * (1 - 2.0), 0.0], atol=1e-15, what="k3 grad")
    rng = np.random.default_rng(2)
    d = rng.normal(0, 2, size=100)
    t = O.token_terms(np.zeros(100), np.zeros(100), np.zeros(100), np.zeros(100), np.zeros(100), P,
                      ref_logp=d)
    assert np.all(t["kl"] >= 0.0)


def pin_terms_tis(O):
    """w = min(exp(old - rollout), c-bar): ln 3 with c-bar 2 -> 2; ln 1.5 -> 1.5; scales surrogate only."""
    P = O.LossParams(tis_cap=2.0, entropy_coef=0.1)
    old = np.array([-1.0, -1.0])
    roll = old - np.array([math.log(3.0), math.log(1.5)])
    z_a = old.copy()  # rho = 1 with lse = 0
    H = np.array([2.0, 2.0])
    t = O.token_terms(z_a, np.zeros(2), H, old, np.array([1.0, -1.0]), P, rollout_logp=roll)
    _close(t["w"], [2.0, 1.5], what="tis w")
    _close(t["ell"], [-2.0 * 1.0 - 0.1 * 2.0, -1.5 * -1.0 - 0.1 * 2.0], what="tis loss")
    _close(t["g"], [-2.0, 1.5], what="tis grad")


def pin_terms_entropy_sign(O):
    """A = 0, beta = 0: l = -alpha H (a bonus lowers the loss)."""
    P = O.LossParams(entropy_coef=0.25)
    t = O.token_terms(np.array([-1.0]), np.array([0.0]), np.array([3.0]), np.array([-1.0]),
                      np.array([0.0]), P)
    _close(t["ell"], [-0.75], what="entropy bonus")


# ---------------------------------------------------------------------------
# B1..B4: loss and gradient
# ---------------------------------------------------------------------------

def _tiny_problem(seed, V=7, n_traj=4, G=2, agg=2, alpha=0.03, beta=0.05, tis=1.7, masked_frac=0.3):
    rng = np.random.default_rng(seed)
    lengths = rng.integers(1, 5, size=n_traj)
    offs = np.concatenate([[0], np.cumsum(lengths)])
    T = int(offs[-1])
    z = rng.normal(0, 1.5, size=(T, V))
    a = rng.integers(0, V, size=T)
    mask = (rng.random(T) > masked_frac).astype(np.uint8)
    tt = np.repeat(np.arange(n_traj), lengths)
    adv = rng.normal(0, 1, size=n_traj)
    coef = rng.uniform(0.2, 1.0, size=n_traj) if agg != 2 else np.ones(n_traj)
    # ratios spread over [0.5, 2.0], at least 1e-3 from a clip bound in log space
    lr = rng.uniform(-0.7, 0.7, size=T)
    for b in (math.log(0.8), math.log(1.28)):
        lr = np.where(np.abs(lr - b) < 1e-3, lr + 3e-3, lr)
    zmax = z.max(axis=1)
    lse = zmax + np.log(np.exp(z - zmax[:, None]).sum(axis=1))  # only used to place old/ref near logp
    logp = z[np.arange(T), a] - lse
    old = logp - lr
    ref = logp + rng.normal(0, 0.3, size=T)
    roll = old + rng.normal(0, 0.4, size=T)
    P = dict(entropy_coef=alpha, kl_coef=beta, kl_estimator=3 if beta else 0, tis_cap=tis, loss_agg=agg)
    return dict(z=z, a=a, mask=mask, tt=tt, adv=adv, coef=coef, old=old, ref=ref, roll=roll, P=P)


def _loss(O, pr, z, P):
    return O.policy_loss_fwd_bwd(z, "f64", pr["a"], pr["mask"], pr["tt"], pr["adv"], pr["coef"],
                                 pr["old"], P, pr["ref"], pr["roll"])


def pin_grad_finite_differences(O):
    """Central differences (h = 1e-6) of the loss match the analytic gradient (1e-6 relative),
    with clipping, k3-KL, entropy bonus and TIS all on."""
    for seed in (0, 1):
        pr = _tiny_problem(seed)
        P = O.LossParams(**pr["P"])
        loss, grad, _, _ = _loss(O, pr, pr["z"], P)
        h = 1e-6
        fd = np.zeros_like(grad)
        for t in range(grad.shape[0]):
            for v in range(grad.shape[1]):
                zp = pr["z"].copy(); zp[t, v] += h
                zm = pr["z"].copy(); zm[t, v] -= h
                fd[t, v] = (_loss(O, pr, zp, P)[0] - _loss(O, pr, zm, P)[0]) / (2 * h)
        scale = np.abs(fd).max()
        assert np.abs(fd - grad).max() <= 1e-6 * scale + 1e-10, (np.abs(fd - grad).max(), scale)


def pin_grad_structure(O):
    """Each gradient row sums to 0 over v; inactive rows are exactly 0;
    a surrogate-only row is g (onehot_a - p)."""
    pr = _tiny_problem(4, V=9, n_traj=6)
    P = O.LossParams(**pr["P"])
    _, grad, stats, _ = _loss(O, pr, pr["z"], P)
    assert np.abs(grad.sum(axis=1)).max() < 1e-14
    assert np.all(grad[pr["mask"] == 0] == 0.0)
    # surrogate only: rho on the unclipped side, A known
    z = np.array([[0.0, math.log(3.0)]])
    t_old = np.array([math.log(0.75)])  # logp(a=1) = ln(3/4) -> rho = 1
    loss, g, _, _ = O.policy_loss_fwd_bwd(z, "f64", [1], [1], [0], [2.0], [1.0], t_old, O.LossParams())
    # g_t = -A rho = -2; row = g (onehot - p) = -2 ([0,1] - [1/4, 3/4]) = [0.5, -0.5]
    _close(g[0], [0.5, -0.5], what="surrogate row")
    _close(loss, -2.0, what="surrogate loss")


def pin_loss_ratio_one(O):
    """old = logp (rho = 1), no KL/entropy/TIS: loss = -sum_i c_i L_i A_i,
    which is 0 for complete groups under seq-mean-token-mean."""
    rng = np.random.default_rng(9)
    G, ng, V = 4, 3, 11
    n = G * ng
    lengths = rng.integers(2, 6, size=n)
    offs = np.concatenate([[0], np.cumsum(lengths)])
    T = int(offs[-1])
    mask = (rng.random(T) < 0.7).astype(np.uint8)
    for i in range(n):
        mask[offs[i]] = 1  # every trajectory counted
    R = rng.normal(size=n)
    go = np.arange(0, n + 1, G)
    z = rng.normal(0, 1, size=(T, V))
    a = rng.integers(0, V, size=T)
    zmax = z.max(axis=1)
    logp = z[np.arange(T), a] - (zmax + np.log(np.exp(z - zmax[:, None]).sum(axis=1)))
    for agg in (O.AGG_SEQ_MEAN_TOKEN_MEAN, O.AGG_TOKEN_MEAN):
        P = O.LossParams(loss_agg=agg)
        adv, coef, L, tt = O.advantages_and_coefficients(R, go, offs, mask, None, P)
        loss, _, stats, _ = O.policy_loss_fwd_bwd(z, "f64", a, mask, tt, adv, coef, logp, P)
        Lc = np.array([mask[offs[i]:offs[i + 1]].sum() for i in range(n)])
        if agg == O.AGG_SEQ_MEAN_TOKEN_MEAN:
            expect = -adv.sum() / n      # N = n counted trajectories
            assert abs(expect) < 1e-12   # group sums vanish
        else:
            expect = -(Lc * adv).sum() / Lc.sum()
        assert abs(loss - expect) < 1e-12, (loss, expect)
        act = mask == 1
        _close(stats[act, 1], np.ones(act.sum()), rtol=1e-12, what="rho = 1")


def pin_token_level_advantages(O):
    """Per-token advantages (PPO, Sec. 2.3.1): rho = 1 and no other term gives
    loss = -sum_t c M A_t and surrogate rows -c A_t (onehot_a - p); advantages broadcast
    from the trajectories reproduce the per-trajectory call exactly."""
    pr = _tiny_problem(13, n_traj=5, agg=1)
    T = pr["z"].shape[0]
    A_t = np.random.default_rng(14).normal(0, 1, size=T)
    z = pr["z"]
    zmax = z.max(axis=1)
    lse = zmax + np.log(np.exp(z - zmax[:, None]).sum(axis=1))
    logp = z[np.arange(T), pr["a"]] - lse
    P = O.LossParams(loss_agg=1, token_level_adv=True)
    loss, grad, _, _ = O.policy_loss_fwd_bwd(z, "f64", pr["a"], pr["mask"], pr["tt"], A_t, pr["coef"], logp, P)
    c_t = pr["coef"][pr["tt"]] * (pr["mask"] != 0)
    _close(loss, -(c_t * A_t).sum(), rtol=1e-12, atol=1e-14, what="token-level loss at rho = 1")
    p = np.exp(z - lse[:, None])
    onehot = np.zeros_like(p)
    onehot[np.arange(T), pr["a"]] = 1.0
    _close(grad, -(c_t * A_t)[:, None] * (onehot - p), rtol=1e-12, atol=1e-14, what="token-level rows")
    P0 = O.LossParams(**pr["P"])
    P1 = O.LossParams(**pr["P"], token_level_adv=True)
    l0, g0, _, _ = _loss(O, pr, z, P0)
    l1, g1, _, _ = O.policy_loss_fwd_bwd(z, "f64", pr["a"], pr["mask"], pr["tt"], pr["adv"][pr["tt"]], pr["coef"],
                                         pr["old"], P1, pr["ref"], pr["roll"])
    assert l0 == l1 and np.array_equal(g0, g1)


def pin_sequence_is_weights(O):
    """The sequence-level weight is the product of the per-token ratios pi_old / pi_rollout over
    the unit's trainable tokens, truncated at c-bar; equal policies give w = 1; a unit with one
    trainable token gets the token-level TIS weight, and the loss with advantages scaled by w_i
    equals the loss with that token-level weight (both scale the surrogate only)."""
    rng = np.random.default_rng(31)
    T, n = 40, 5
    tt = rng.integers(0, n, T)
    mask = (rng.random(T) < 0.7).astype(np.uint8)
    old = rng.normal(-2, 1, T)
    roll = old + rng.normal(0, 0.05, T)
    w, S = O.sequence_is_weights(tt, mask, old, roll, n, cap=0.0)
    for i in range(n):
        prod = 1.0
        for t in range(T):
            if tt[t] == i and mask[t]:
                prod *= math.exp(old[t]) / math.exp(roll[t])
        _close([w[i]], [prod], rtol=1e-12, what=f"product of ratios {i}")
    wc, _ = O.sequence_is_weights(tt, mask, old, roll, n, cap=1.01)
    _close(wc, np.minimum(w, 1.01), rtol=0, atol=0, what="truncation")
    w1, S1 = O.sequence_is_weights(tt, mask, old, old, n, cap=2.0)
    assert np.all(w1 == 1.0) and np.all(S1 == 0.0)
    # one trainable token per trajectory: sequence weight == token-level TIS weight
    pr = _tiny_problem(17, n_traj=4, agg=2, alpha=0.02, beta=0.03, tis=1.5)
    z = pr["z"]
    Tn = z.shape[0]
    mask1 = np.zeros(Tn, np.uint8)
    for i in range(4):
        mask1[np.nonzero(pr["tt"] == i)[0][0]] = 1
    P_tok = O.LossParams(**pr["P"])
    pr_tok = dict(pr, mask=mask1)
    l_tok, g_tok, _, _ = _loss(O, pr_tok, z, P_tok)
    wseq, _ = O.sequence_is_weights(pr["tt"], mask1, pr["old"], pr["roll"], 4, cap=P_tok.tis_cap)
    P_seq = O.LossParams(**dict(pr["P"], tis_cap=0.0))
    l_seq, g_seq, _, _ = O.policy_loss_fwd_bwd(z, "f64", pr["a"], mask1, pr["tt"], pr["adv"] * wseq, pr["coef"],
                                               pr["old"], P_seq, pr["ref"], None)
    _close([l_seq], [l_tok], rtol=1e-12, atol=1e-15, what="sequence weight vs token weight, loss")
    _close(g_seq, g_tok, rtol=1e-12, atol=1e-15, what="sequence weight vs token weight, grad")


def pin_stats_summary(O):
    """Hand-worked: three trained tokens (one clipped), one masked and one of a zero-coefficient
    trajectory are left out; and the summary of a loss call's stats at rho = 1 counts every
    trained token with ratio 1 and none clipped."""
    stats = np.array([[-1.0, 1.5, 1.0, 2.0, 0.1], [-2.0, 0.9, 0.0, 1.0, 0.2], [-0.5, 1.0, 0.0, 3.0, 0.0],
                      [-9.0, 7.0, 1.0, 9.0, 9.0], [-9.0, 7.0, 1.0, 9.0, 9.0]])
    mask = [1, 1, 1, 0, 1]
    tt = [0, 0, 1, 1, 2]
    coef = [0.5, 0.25, 0.0]
    _close(O.stats_summary(stats, mask, tt, coef), [3.0, 1.0, 6.0, 0.3, 3.4], rtol=1e-15, what="summary")
    pr = _tiny_problem(23, n_traj=5, agg=1, alpha=0.0, beta=0.0, tis=0.0)
    z = pr["z"]
    T = z.shape[0]
    zmax = z.max(axis=1)
    logp = z[np.arange(T), pr["a"]] - (zmax + np.log(np.exp(z - zmax[:, None]).sum(axis=1)))
    P = O.LossParams(**pr["P"])
    _, _, st, _ = O.policy_loss_fwd_bwd(z, "f64", pr["a"], pr["mask"], pr["tt"], pr["adv"], pr["coef"], logp, P)
    sm = O.stats_summary(st, pr["mask"], pr["tt"], pr["coef"])
    n_act = int(((pr["mask"] != 0) & (pr["coef"][pr["tt"]] != 0)).sum())
    _close(sm[[0, 1, 4]], [n_act, 0.0, n_act], rtol=1e-12, what="rho = 1 summary")


def pin_loss_additive_and_permutation(O):
    """The loss of two microbatches adds up to the loss of the whole batch; permuting the
    rows permutes the gradient rows and keeps the loss."""
    pr = _tiny_problem(7, n_traj=8)
    P = O.LossParams(**pr["P"])
    loss, grad, _, _ = _loss(O, pr, pr["z"], P)
    T = pr["z"].shape[0]
    k = T // 2
    parts = 0.0
    for sl in (slice(0, k), slice(k, T)):
        l2, g2, _, _ = O.policy_loss_fwd_bwd(pr["z"][sl], "f64", pr["a"][sl], pr["mask"][sl], pr["tt"][sl],
                                             pr["adv"], pr["coef"], pr["old"][sl], P, pr["ref"][sl],
                                             pr["roll"][sl])
        parts += l2
        _close(g2, grad[sl], rtol=0, atol=0, what="split grad")
    assert abs(parts - loss) <= 1e-14 * max(1.0, abs(loss))
    perm = np.random.default_rng(0).permutation(T)
    l3, g3, _, _ = O.policy_loss_fwd_bwd(pr["z"][perm], "f64", pr["a"][perm], pr["mask"][perm],
                                         pr["tt"][perm], pr["adv"], pr["coef"], pr["old"][perm], P,
                                         pr["ref"][perm], pr["roll"][perm])
    assert abs(l3 - loss) <= 1e-13 * max(1.0, abs(loss))
    _close(g3, grad[perm], rtol=0, atol=0, what="permuted grad")


def pin_loss_golden(O):
    """tests/golden/grpo_loss_worked_example.json: a four-token batch worked by hand."""
    with open(os.path.join(GOLDEN, "grpo_loss_worked_example.json")) as f:
        ex = json.load(f)
    inp = ex["inputs"]
    P = O.LossParams(**ex["params"])
    adv, coef, L, tt = O.advantages_and_coefficients(np.array(inp["rewards"]), inp["group_offsets"],
                                                     inp["traj_offsets"], np.array(inp["mask"], np.uint8),
                                                     None, P)
    exp = ex["expected"]
    _close(adv, exp["advantages"], rtol=1e-12, what="worked adv")
    _close(coef, exp["coef"], rtol=1e-12, what="worked coef")
    z = np.array(inp["logits"], dtype=np.float64)
    loss, grad, stats, _ = O.policy_loss_fwd_bwd(z, "f64", inp["token_ids"], np.array(inp["mask"], np.uint8),
                                                 tt, adv, coef, np.array(inp["old_logp"]), P)
    _close(loss, exp["loss"], rtol=1e-9, atol=1e-15, what="worked loss")
    _close(grad, exp["grad"], rtol=1e-9, atol=1e-15, what="worked grad")
    _close(stats[:, 2], exp["clipped"], what="worked clipped flags")


def pin_logprobs_vs_library(O):
    """token_logprobs matches float64 torch.log_softmax / entropy on bf16-valued rows."""
    import torch

    rng = np.random.default_rng(21)
    f = rng.normal(0, 3, size=(5, 33)).astype(np.float32)
    bits = (f.view(np.uint32) >> 16).astype(np.uint16)       # truncation: any bf16 pattern will do
    zz = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    a = rng.integers(0, 33, size=5)
    logp, H, lse = O.token_logprobs(bits, "bf16", a)
    ls = torch.log_softmax(torch.from_numpy(zz), dim=1).numpy()
    _close(logp, ls[np.arange(5), a], rtol=1e-12, atol=1e-12, what="token_logprobs logp")
    _close(lse, torch.logsumexp(torch.from_numpy(zz), dim=1).numpy(), rtol=1e-13, what="lse")
    _close(H, -(np.exp(ls) * ls).sum(axis=1), rtol=1e-10, what="entropy")


def pin_decode_logits_vs_library(O):
    """decode_logits of bf16 bit patterns equals torch's own bfloat16 -> float64 conversion on
    every class of pattern: zeros of both signs, subnormals, normals, the largest finite values,
    +-inf and NaNs, and a random sample of all 65,536 patterns."""
    import torch

    special = np.array([0x0000, 0x8000, 0x0001, 0x8001, 0x007F, 0x807F, 0x0080, 0x8080, 0x3F80, 0xBF80,
                        0x7F7F, 0xFF7F, 0x7F80, 0xFF80, 0x7FC0, 0xFFC0, 0x7F81, 0xFFFF], dtype=np.uint16)
    rng = np.random.default_rng(31)
    bits = np.concatenate([special, rng.integers(0, 1 << 16, size=4096, dtype=np.uint32).astype(np.uint16)])
    got = O.decode_logits(bits, "bf16")
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    assert got.dtype == np.float64 and got.shape == ref.shape
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan), "NaN patterns"
    assert np.array_equal(got[~nan], ref[~nan]), "decoded values"
    assert np.array_equal(np.signbit(got[~nan]), np.signbit(ref[~nan])), "signs (of zeros too)"
    assert got[2] == 2.0 ** -133 and got[4] == (1 - 2.0 ** -7) * 2.0 ** -126 and got[6] == 2.0 ** -126, "subnormals"
    f32 = rng.normal(0, 100, size=64).astype(np.float32)
    _close(O.decode_logits(f32, "f32"), torch.from_numpy(f32).double().numpy(), rtol=0, atol=0, what="f32 decode")


# ---------------------------------------------------------------------------
# C: fused head
# ---------------------------------------------------------------------------

def _bf16(x):
    u = np.asarray(x, dtype=np.float32).view(np.uint32)
    return ((u + np.uint32(0x7FFF) + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def _unbf16(b):
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def pin_fused_head_finite_differences(O):
    """d_hidden and d_W of the fused head against central differences of its loss
    (square T = D = V = 4 so that a transposed operand changes values, not shapes)."""
    rng = np.random.default_rng(8)
    T = D = V = 4
    h = _bf16(rng.normal(0, 1, size=(T, D)))
    w = _bf16(rng.normal(0, 0.7, size=(V, D)))
    a = rng.integers(0, V, size=T)
    mask = np.array([1, 1, 0, 1], np.uint8)
    tt = np.array([0, 0, 1, 1])
    adv = np.array([0.8, -1.1])
    coef = np.array([1.0, 1.0])
    Hm, Wm = _unbf16(h), _unbf16(w)
    Z = Hm @ Wm.T
    zmax = Z.max(axis=1)
    logp = Z[np.arange(T), a] - (zmax + np.log(np.exp(Z - zmax[:, None]).sum(axis=1)))
    old = logp - np.array([0.3, -0.05, 0.0, 0.1])
    ref = logp + 0.2
    P = O.LossParams(entropy_coef=0.05, kl_coef=0.1, kl_estimator=3, loss_agg=O.AGG_TOKEN_SUM)
    loss, dH, dW, _ = O.fused_head_loss_fwd_bwd(h, w, a, mask, tt, adv, coef, old, P, ref)

    def f(Hx, Wx):
        Zx = Hx @ Wx.T
        return O.policy_loss_fwd_bwd(Zx, "f64", a, mask, tt, adv, coef, old, P, ref, None, want_grad=False)[0]

    eps = 1e-6
    fdH = np.zeros_like(Hm)
    for i in range(T):
        for j in range(D):
            Hp = Hm.copy(); Hp[i, j] += eps
            Hn = Hm.copy(); Hn[i, j] -= eps
            fdH[i, j] = (f(Hp, Wm) - f(Hn, Wm)) / (2 * eps)
    fdW = np.zeros_like(Wm)
    for i in range(V):
        for j in range(D):
            Wp = Wm.copy(); Wp[i, j] += eps
            Wn = Wm.copy(); Wn[i, j] -= eps
            fdW[i, j] = (f(Hm, Wp) - f(Hm, Wn)) / (2 * eps)
    assert abs(f(Hm, Wm) - loss) < 1e-14
    assert np.abs(fdH - dH).max() <= 1e-6 * np.abs(fdH).max(), np.abs(fdH - dH).max()
    assert np.abs(fdW - dW).max() <= 1e-6 * np.abs(fdW).max(), np.abs(fdW - dW).max()


def pin_fused_head_zero_hidden(O):
    """Zero hidden rows give uniform softmax: logp = -ln V, H = ln V, d_W rows from those tokens vanish
    except through dZ; with A = 0 and no regularisers everything is 0."""
    V, D = 6, 3
    h = np.zeros((2, D), np.uint16)
    w = _bf16(np.random.default_rng(1).normal(size=(V, D)))
    loss, dH, dW, stats = O.fused_head_loss_fwd_bwd(h, w, [2, 5], [1, 1], [0, 0], [0.5], [1.0],
                                                    np.array([-math.log(V)] * 2), O.LossParams())
    _close(stats[:, 0], [-math.log(V)] * 2, what="uniform logp")
    _close(stats[:, 3], [math.log(V)] * 2, what="uniform H")
    _close(loss, -2 * 0.5, what="rho = 1 loss")
    assert np.all(dW == 0.0)  # hidden = 0 -> dW = dZ^T H = 0


def pin_fused_head_logprobs_vs_library(O):
    """Forward-only fused-head log-probs against float64 torch.log_softmax(H W^T), and the
    uniform case (zero hidden rows: logp = -ln V, H = ln V)."""
    import torch

    rng = np.random.default_rng(12)
    h = _bf16(rng.normal(0, 1, size=(5, 64)))
    w = _bf16(rng.normal(0, 0.3, size=(40, 64)))
    h[3] = 0
    a = rng.integers(0, 40, size=5)
    logp, H, lse = O.fused_head_logprobs(h, w, a, chunk=2)
    Z = torch.from_numpy(_unbf16(h)) @ torch.from_numpy(_unbf16(w)).T
    ls = torch.log_softmax(Z, dim=1).numpy()
    _close(logp, ls[np.arange(5), a], rtol=1e-12, atol=1e-12, what="fused logp vs torch")
    _close(lse, torch.logsumexp(Z, dim=1).numpy(), rtol=1e-12, atol=1e-12, what="fused lse vs torch")
    _close(H, -(np.exp(ls) * ls).sum(axis=1), rtol=1e-10, atol=1e-12, what="fused entropy")
    _close([logp[3], H[3]], [-math.log(40), math.log(40)], what="zero hidden row")


def pin_gradients_autograd(O):
    """The analytic d loss / d logits against autograd of a separate float64 PyTorch statement of
    the objective (clipped surrogate with both branches present, k3 KL, entropy, TIS as a constant
    weight, coefficient-weighted sum), to float64 rounding."""
    import torch

    rng = np.random.default_rng(41)
    rows, V, n = 40, 29, 5
    z = rng.normal(0.0, 2.0, (rows, V))
    ids = rng.integers(0, V, rows)
    zt = torch.tensor(z, requires_grad=True)
    logp_all = torch.log_softmax(zt, dim=1)
    logp0 = logp_all.detach().numpy()[np.arange(rows), ids]
    delta = rng.uniform(-0.6, 0.6, rows)
    delta = np.where(np.abs(delta - np.log(0.8)) < 2e-4, delta + 5e-4, delta)
    delta = np.where(np.abs(delta - np.log(1.28)) < 2e-4, delta + 5e-4, delta)
    old, ref = logp0 - delta, logp0 + rng.normal(0.0, 0.3, rows)
    roll = old + rng.normal(0.0, 0.4, rows)
    tt = rng.integers(0, n, rows)
    mask = (rng.random(rows) < 0.8).astype(np.uint8)
    adv, coef = rng.normal(0.0, 1.0, n), rng.uniform(0.05, 1.0, n)
    prm = O.LossParams(kl_coef=0.05, kl_estimator=3, entropy_coef=0.03, tis_cap=1.5)
    loss, grad, stats, _ = O.policy_loss_fwd_bwd(z, "f64", ids, mask, tt, adv, coef, old, prm, ref, roll)
    if not 0 < stats[mask != 0, O.STAT_CLIPPED].sum() < (mask != 0).sum():
        raise AssertionError("the case must hold clipped and unclipped tokens")
    T = lambda x: torch.tensor(x, dtype=torch.float64)  # noqa: E731
    logp = logp_all.gather(1, torch.tensor(ids)[:, None])[:, 0]
    p = logp_all.exp()
    H = -(p * logp_all).sum(dim=1)
    A, c = T(adv)[torch.tensor(tt)], T(coef)[torch.tensor(tt)] * T(mask)
    rho = torch.exp(logp - T(old))
    surr = torch.minimum(rho * A, torch.clamp(rho, 0.8, 1.28) * A)
    w = torch.clamp(torch.exp(T(old) - T(roll)), max=1.5)
    d = T(ref) - logp
    ell = -w * surr + 0.05 * (torch.exp(d) - d - 1.0) - 0.03 * H
    (c * ell).sum().backward()
    g = zt.grad.numpy()
    _close([loss], [float((c * ell).sum().detach())], rtol=1e-12, atol=1e-12, what="loss vs autograd")
    _close(grad, g, rtol=0.0, atol=1e-11 * float(np.abs(g).max()), what="gradient vs autograd")


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
