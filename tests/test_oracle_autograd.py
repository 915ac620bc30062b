"""The oracle's hand-derived gradients against automatic differentiation.

A float64 PyTorch statement of the per-token objective (log-softmax, ratio, clipped surrogate,
k3 KL, entropy bonus, truncated importance weight, coefficient-weighted sum), differentiated by
autograd on the CPU, must give the oracle's analytic d loss / d logits, its fused-head products
d hidden = dZ W and d W = dZ^T H, and its value-loss gradient, to float64 rounding. This pins
the backward derivations (the clip rule, the entropy and KL terms, TIS as a constant weight)
exactly, beyond what central differences resolve. Clip boundaries are kept at least 1e-4 away,
where the derivative of min / clip is undefined.
"""

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
import oracle.ppo_objective as P
from paper_2608_16798_gb300 import workloads as W


def torch_loss(z, ids, mask, tt, adv, coef, old, prm: O.LossParams, ref=None, roll=None):
    logp_all = torch.log_softmax(z, dim=1)
    logp = logp_all.gather(1, ids[:, None])[:, 0]
    p = logp_all.exp()
    H = -(p * logp_all).sum(dim=1)
    A = adv if prm.token_level_adv else adv[tt]
    c = coef[tt] * mask
    rho = torch.exp(logp - old)
    surr = torch.minimum(rho * A, torch.clamp(rho, 1.0 - prm.clip_eps_low, 1.0 + prm.clip_eps_high) * A)
    w = torch.ones_like(rho)
    if prm.tis_cap > 0 and roll is not None:
        w = torch.clamp(torch.exp(old - roll), max=prm.tis_cap)  # a constant: no gradient flows into it
    kl = torch.zeros_like(rho)
    if prm.kl_estimator == 3 and prm.kl_coef != 0 and ref is not None:
        d = ref - logp
        kl = torch.exp(d) - d - 1.0
    ell = -w * surr + prm.kl_coef * kl - prm.entropy_coef * H
    return (c * ell).sum()


def make_inputs(seed, rows=60, V=37, n_traj=7, token_level=False):
    rng = np.random.default_rng(seed)
    z = rng.normal(0.0, 2.0, (rows, V))
    ids = rng.integers(0, V, rows)
    lse = np.log(np.exp(z - z.max(1, keepdims=True)).sum(1)) + z.max(1)
    logp = z[np.arange(rows), ids] - lse
    delta = rng.uniform(-0.6, 0.6, rows)
    for b in (np.log(0.8), np.log(1.28)):  # keep rho at least 1e-4 (relative) off the clip bounds
        delta = np.where(np.abs(delta - b) < 2e-4, delta + 5e-4, delta)
    old = logp - delta
    ref = logp + rng.normal(0.0, 0.3, rows)
    roll = old + rng.normal(0.0, 0.4, rows)
    tt = rng.integers(0, n_traj, rows)
    mask = (rng.random(rows) < 0.75).astype(np.uint8)
    adv = rng.normal(0.0, 1.0, rows if token_level else n_traj)
    coef = rng.uniform(0.01, 1.0, n_traj)
    coef[rng.integers(0, n_traj)] = 0.0  # a trajectory that is not trained on
    return dict(z=z, ids=ids, old=old, ref=ref, roll=roll, tt=tt, mask=mask, adv=adv, coef=coef)


def autograd(x, prm, use_ref, use_roll):
    z = torch.tensor(x["z"], dtype=torch.float64, requires_grad=True)
    f = lambda k: torch.tensor(x[k], dtype=torch.float64)  # noqa: E731
    loss = torch_loss(z, torch.tensor(x["ids"]), f("mask"), torch.tensor(x["tt"]), f("adv"), f("coef"), f("old"),
                      prm, f("ref") if use_ref else None, f("roll") if use_roll else None)
    loss.backward()
    return loss.item(), z.grad.numpy()


@pytest.mark.parametrize("kl,ent,tis,token_level,agg_eps", [
    (False, False, False, False, (0.2, 0.28)),
    (True, False, False, False, (0.2, 0.28)),
    (False, True, False, False, (0.1, 0.1)),
    (False, False, True, False, (0.2, 0.28)),
    (True, True, True, False, (0.2, 0.28)),
    (True, True, False, True, (0.15, 0.3)),
])
def test_policy_gradient_matches_autograd(kl, ent, tis, token_level, agg_eps):
    x = make_inputs(11 + 7 * kl + 3 * ent + 5 * tis + 13 * token_level, token_level=token_level)
    prm = O.LossParams(clip_eps_low=agg_eps[0], clip_eps_high=agg_eps[1], kl_coef=0.05 if kl else 0.0,
                       kl_estimator=3 if kl else 0, entropy_coef=0.02 if ent else 0.0, tis_cap=1.5 if tis else 0.0,
                       token_level_adv=token_level)
    loss, grad, stats, _ = O.policy_loss_fwd_bwd(x["z"], "f64", x["ids"], x["mask"], x["tt"], x["adv"], x["coef"],
                                                 x["old"], prm, x["ref"] if kl else None, x["roll"] if tis else None)
    l_ag, g_ag = autograd(x, prm, kl, tis)
    assert abs(loss - l_ag) <= 1e-12 * max(1.0, abs(l_ag))
    scale = np.abs(g_ag).max(axis=1, keepdims=True) + 1e-300
    assert np.all(np.abs(grad - g_ag) <= 1e-11 * scale), np.abs(grad - g_ag).max()
    # clipped and unclipped tokens are both present, and masked / zero-coefficient rows are exactly 0
    active = (x["mask"] != 0) & (x["coef"][x["tt"]] != 0)
    clipped = stats[active, O.STAT_CLIPPED]
    assert 0 < clipped.sum() < active.sum()
    assert np.all(grad[~active] == 0.0)


def test_fused_head_products_match_autograd():
    rng = np.random.default_rng(5)
    T, D, V = 24, 64, 53
    h_bits = W.bf16_bits_from_f32(rng.normal(0, 1, (T, D)).astype(np.float32))
    w_bits = W.bf16_bits_from_f32(rng.normal(0, 0.1, (V, D)).astype(np.float32))
    Hm, Wm = O.decode_logits(h_bits, "bf16"), O.decode_logits(w_bits, "bf16")
    Z = Hm @ Wm.T
    x = make_inputs(21, rows=T, V=V, n_traj=4)
    x["z"] = Z
    lse = np.log(np.exp(Z - Z.max(1, keepdims=True)).sum(1)) + Z.max(1)
    logp = Z[np.arange(T), x["ids"]] - lse
    x["old"] = logp - np.random.default_rng(6).uniform(-0.1, 0.1, T)  # rho well inside the clip range
    prm = O.LossParams(kl_coef=0.05, kl_estimator=3, entropy_coef=0.02)
    loss, dH, dW, _ = O.fused_head_loss_fwd_bwd(h_bits, w_bits, x["ids"], x["mask"], x["tt"], x["adv"], x["coef"],
                                                x["old"], prm, x["ref"], None)
    h = torch.tensor(Hm, requires_grad=True)
    w = torch.tensor(Wm, requires_grad=True)
    f = lambda k: torch.tensor(x[k], dtype=torch.float64)  # noqa: E731
    l_ag = torch_loss(h @ w.T, torch.tensor(x["ids"]), f("mask"), torch.tensor(x["tt"]), f("adv"), f("coef"),
                      f("old"), prm, f("ref"), None)
    l_ag.backward()
    assert abs(loss - l_ag.item()) <= 1e-12 * max(1.0, abs(l_ag.item()))
    for got, ref in ((dH, h.grad.numpy()), (dW, w.grad.numpy())):
        assert np.all(np.abs(got - ref) <= 1e-11 * (np.abs(ref).max() + 1e-300)), np.abs(got - ref).max()


def test_value_loss_gradient_matches_autograd():
    rng = np.random.default_rng(8)
    rows, n_traj = 80, 6
    values, returns = rng.normal(0.3, 0.3, rows), rng.normal(0.5, 0.5, rows)
    mask = (rng.random(rows) < 0.7).astype(np.uint8)
    tt = rng.integers(0, n_traj, rows)
    coef = rng.uniform(0.0, 1.0, n_traj)
    loss, dv, _ = P.value_loss_fwd_bwd(values, returns, mask, tt, coef)
    v = torch.tensor(values, requires_grad=True)
    c = torch.tensor(coef)[torch.tensor(tt)] * torch.tensor(mask, dtype=torch.float64)
    l_ag = (c * (v - torch.tensor(returns)) ** 2).sum()
    l_ag.backward()
    assert abs(loss - l_ag.item()) <= 1e-12 * max(1.0, abs(l_ag.item()))
    assert np.allclose(dv, v.grad.numpy(), rtol=1e-13, atol=1e-15)
