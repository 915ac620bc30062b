"""PPO path on the GPU against the float64 oracle: masked GAE (both readings), the value
loss, and the clipped policy loss with per-token advantages (logits path and fused head).

Tolerances: GAE as in parity_cases.check_gae (a scan-depth multiple of 2^-24 times the sum of
the absolute terms); value loss 1e-4 of sum |c M (V - G)^2| and 4 * 2^-24 |g| + 1e-30 per
element of the gradient (three fp32 roundings); policy loss and gradients with the
logits-path tolerances.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
import oracle.ppo_objective as PO
from parity_cases import (check_gae, check_grad, check_loss, check_stats, cuda_params, gae_error_scale, grad_to_np,
                          logits_to_dev, make_case, to_dev)
from paper_2608_16798_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_16798_gb300 import build

    build.build()
    import paper_2608_16798_gb300.rl_loss as R

    R.lib()
    return R


def gae_inputs(name, seed=0, token_rewards=False):
    w = W.WORKLOADS[name]
    lay = W.make_layout(w, seed)
    T = lay.n_tokens
    V = W.value_predictions(w, seed, T)
    rt = W.token_reward_draws(w, seed, T) if token_rewards else None
    return w, lay, V, rt


def run_gae(R, lay, V, rt, gamma, lam, skip, traj_rewards=True):
    ws = R.new_workspace(0, 0)
    adv, ret = R.rl_masked_gae(to_dev(lay.traj_offsets.astype(np.int64)), to_dev(lay.mask), to_dev(V), ws,
                               gamma=gamma, gae_lambda=lam, skip_masked=skip,
                               token_rewards=None if rt is None else to_dev(rt),
                               traj_rewards=to_dev(lay.rewards.astype(np.float32)) if traj_rewards else None)
    word = R.rl_query_status(ws)[1]
    return adv.cpu().numpy().astype(np.float64), ret.cpu().numpy().astype(np.float64), word


def oracle_gae(lay, V, rt, gamma, lam, skip):
    r = PO.final_token_rewards(lay.traj_offsets, lay.mask, lay.rewards.astype(np.float32))
    if rt is not None:
        r = r + rt.astype(np.float64)
    fn = PO.masked_gae_skip if skip else PO.masked_gae
    adv, ret = fn(lay.traj_offsets, lay.mask, V, r, gamma, lam)
    return adv, ret, r


@pytest.mark.parametrize("name,gamma,lam,skip,trew", [
    ("tiny", 0.99, 0.95, False, True),
    ("tiny", 0.99, 0.95, True, True),
    ("multiturn", 1.0, 1.0, True, False),    # the paper's PPO setting (Sec. 2.3.4)
    ("multiturn", 1.0, 1.0, False, False),   # printed reading at gamma = lambda = 1
    ("multiturn", 0.99, 0.9, False, True),
    ("multiturn", 0.97, 0.0, True, True),    # one-step TD residuals
    ("edge", 0.9, 0.8, True, True),          # 16,384 trajectories of 8 tokens, fully masked ones
])
def test_gae_parity(R, name, gamma, lam, skip, trew):
    w, lay, V, rt = gae_inputs(name, token_rewards=trew)
    adv_d, ret_d, word = run_gae(R, lay, V, rt, gamma, lam, skip)
    assert word == 0
    adv, ret, r = oracle_gae(lay, V, rt, gamma, lam, skip)
    S = gae_error_scale(lay.traj_offsets, lay.mask, V, r, gamma, lam, skip)
    check_gae(adv_d, ret_d, adv, ret, V, S, lay.mask, int(np.diff(lay.traj_offsets).max()),
              f"{name} gamma={gamma} lambda={lam} skip={skip}")


def test_gae_degenerate_form(R):
    """gamma = lambda = 1, skip reading, R_i at the final trainable token: A_t = R_i - V_t and
    G_t = R_i on every trainable token (Sec. 2.3.4)."""
    w, lay, V, _ = gae_inputs("multiturn")
    adv_d, ret_d, word = run_gae(R, lay, V, None, 1.0, 1.0, True)
    assert word == 0
    owner = np.repeat(np.arange(lay.n_traj), np.diff(lay.traj_offsets))
    M = lay.mask != 0
    has = np.zeros(lay.n_traj, bool)
    np.logical_or.at(has, owner, M)
    Rt = lay.rewards.astype(np.float64)[owner]
    S = gae_error_scale(lay.traj_offsets, lay.mask, V, PO.final_token_rewards(lay.traj_offsets, lay.mask, lay.rewards),
                        1.0, 1.0, True)
    u = 2.0 ** -24
    k = 64 + 2 * int(np.ceil(np.diff(lay.traj_offsets).max() / 1024))
    assert np.all(np.abs(adv_d - (Rt - V))[M] <= (k * u * S + u * np.abs(Rt - V) + 1e-30)[M])
    assert np.all(np.abs(ret_d - Rt)[M] <= (k * u * S + 2 * u * (np.abs(Rt) + np.abs(V)) + 1e-30)[M])


def test_gae_spans_and_bad_offsets(R):
    """Tokens outside every span are left untouched; empty spans are fine; a trajectory whose
    span runs past n_tokens sets RL_DEV_BAD_OFFSETS and is skipped while the others are computed."""
    rng = np.random.default_rng(5)
    T = 3000
    mask = (rng.random(T) < 0.6).astype(np.uint8)
    V = rng.normal(0.3, 0.25, T).astype(np.float32)
    offs = np.array([7, 7, 1500, 2990, 5000], dtype=np.int64)  # span 3 ends past T
    R_i = np.array([1.0, 0.0, 1.0, 1.0], np.float32)
    ws = R.new_workspace(0, 0)
    adv = torch.full((T,), float("nan"), device="cuda")
    ret = torch.full((T,), float("nan"), device="cuda")
    R.rl_masked_gae(to_dev(offs), to_dev(mask), to_dev(V), ws, 0.95, 0.9, True, traj_rewards=to_dev(R_i),
                    adv_out=adv, returns_out=ret)
    assert R.rl_query_status(ws)[1] == R.RL_DEV_BAD_OFFSETS
    a, g = adv.cpu().numpy().astype(np.float64), ret.cpu().numpy().astype(np.float64)
    untouched = np.r_[0:7, 2990:T]
    assert np.isnan(a[untouched]).all() and np.isnan(g[untouched]).all()
    for (s, e), Ri in zip(((7, 1500), (1500, 2990)), (R_i[1], R_i[2])):  # the two good non-empty spans
        sub = np.array([0, e - s])
        r = PO.final_token_rewards(sub, mask[s:e], [Ri])
        ra, rr = PO.masked_gae_skip(sub, mask[s:e], V[s:e], r, 0.95, 0.9)
        S = gae_error_scale(sub, mask[s:e], V[s:e], r, 0.95, 0.9, True)
        check_gae(a[s:e], g[s:e], ra, rr, V[s:e], S, mask[s:e], e - s, f"span [{s}, {e})")


def test_value_loss_parity(R):
    w, lay, V, _ = gae_inputs("multiturn")
    adv, ret, _ = oracle_gae(lay, V, None, 1.0, 1.0, True)
    P = O.LossParams(loss_agg=O.AGG_TOKEN_MEAN)
    _, coef, _, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                   lay.traj_valid, P)
    coef32 = coef.astype(np.float32)
    G32 = ret.astype(np.float32)
    Vnew = (V + np.random.default_rng(3).normal(0, 0.1, len(V))).astype(np.float32)  # the updated value model
    lo, hi = W.microbatches(lay, w.microbatch)[1]
    ws = R.new_workspace(hi - lo, 0)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    dV = R.rl_value_loss_fwd_bwd(to_dev(Vnew[lo:hi]), to_dev(G32[lo:hi]), to_dev(lay.mask[lo:hi]),
                                 to_dev(tt[lo:hi].astype(np.int32)), to_dev(coef32), ws, loss)
    assert R.rl_query_status(ws)[1] == 0
    l_ref, g_ref, contrib = PO.value_loss_fwd_bwd(Vnew[lo:hi], G32[lo:hi], lay.mask[lo:hi], tt[lo:hi], coef32)
    check_loss(loss.item(), l_ref, contrib, "value loss")
    g = dV.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(g - g_ref) <= 4 * 2.0 ** -24 * np.abs(g_ref) + 1e-30), np.abs(g - g_ref).max()
    assert np.all(g[lay.mask[lo:hi] == 0] == 0.0)


def _token_adv_case(name, rows, vocab, seed=0, row0=0):
    c = make_case(name, seed=seed, row0=row0, rows=rows, vocab=vocab, loss_agg=O.AGG_TOKEN_MEAN)
    V = W.value_predictions(c.w, seed, c.layout.n_tokens)
    adv_t, _, _ = oracle_gae(c.layout, V, None, 1.0, 1.0, True)
    P = dataclasses.replace(c.P, token_level_adv=True)
    _, coef, _, _ = O.advantages_and_coefficients(c.layout.rewards, c.layout.group_offsets, c.layout.traj_offsets,
                                                  c.layout.mask, c.layout.traj_valid, P)
    return c, adv_t.astype(np.float32), coef.astype(np.float32), P


@pytest.mark.parametrize("name,rows,vocab", [("multiturn", 700, 4096), ("longhorizon", 300, 3000)])
def test_ppo_policy_loss_token_adv(R, name, rows, vocab):
    c, adv32, coef32, P = _token_adv_case(name, rows, vocab, row0=1000)
    sl = c.sl
    loss_ref, g_ref, st_ref, contrib = O.policy_loss_fwd_bwd(c.raw, c.w.dtype, c.ids, c.mask, c.tt,
                                                             adv32[sl].astype(np.float64), coef32.astype(np.float64),
                                                             c.old, P, c.ref, None)
    ws = R.new_workspace(c.rows, vocab)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(c.rows * 5, dtype=torch.float32, device="cuda")
    grad = R.rl_policy_loss_fwd_bwd(logits_to_dev(c), to_dev(c.ids), to_dev(c.mask), to_dev(c.tt.astype(np.int32)),
                                    to_dev(adv32[sl]), to_dev(coef32), to_dev(c.old), cuda_params(R, P), ws, loss,
                                    ref_logp=None if c.ref is None else to_dev(c.ref), token_stats=st)
    assert R.rl_query_status(ws)[1] == 0
    check_loss(loss.item(), loss_ref, contrib, f"{name} ppo loss")
    active = (c.mask != 0) & (coef32[c.tt] != 0)
    check_stats(st.view(-1, 5).cpu().numpy(), st_ref, active, f"{name} ppo stats")
    check_grad(grad_to_np(grad), g_ref, c.w.dtype, f"{name} ppo grad")


def test_ppo_token_adv_microbatch_split(R):
    """Two calls on halves of the rows (adv sliced like old_logp) give the one-call result."""
    c, adv32, coef32, P = _token_adv_case("multiturn", 512, 2048, row0=300)
    sl = c.sl
    lg = logits_to_dev(c)
    args = lambda a, b: (lg[a:b], to_dev(c.ids[a:b]), to_dev(c.mask[a:b]), to_dev(c.tt[a:b].astype(np.int32)),
                         to_dev(adv32[sl][a:b]), to_dev(coef32), to_dev(c.old[a:b]), cuda_params(R, P))
    ws = R.new_workspace(c.rows, 2048)
    l1 = torch.zeros(1, dtype=torch.float64, device="cuda")
    g1 = R.rl_policy_loss_fwd_bwd(*args(0, c.rows), ws, l1, ref_logp=None if c.ref is None else to_dev(c.ref))
    l2 = torch.zeros(1, dtype=torch.float64, device="cuda")
    k = 200
    ga = R.rl_policy_loss_fwd_bwd(*args(0, k), ws, l2, ref_logp=None if c.ref is None else to_dev(c.ref[:k]))
    gb = R.rl_policy_loss_fwd_bwd(*args(k, c.rows), ws, l2, ref_logp=None if c.ref is None else to_dev(c.ref[k:]))
    assert R.rl_query_status(ws)[1] == 0
    assert torch.equal(torch.cat([ga, gb]), g1)
    assert abs(l1.item() - l2.item()) <= 1e-12 * max(1e-30, abs(l1.item()))
