"""Sequence-level importance weights (Sec. 3.2.4) on the GPU against the float64 oracle.

Tolerances: S_i within n_i 2^-41 (each difference is rounded to a multiple of 2^-40) plus
the float32 rounding of the output; w_i within (n_i 2^-40 + 2^-23) w_i. The sums are integer
additions, so any permutation of the tokens gives bit-identical results.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
from parity_cases import check_grad, check_loss, cuda_params, grad_to_np, logits_to_dev, make_case, to_dev
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


def batch(name="multiturn", seed=0):
    w = W.WORKLOADS[name]
    lay = W.make_layout(w, seed)
    _, tt = O.trajectory_token_counts(lay.mask, lay.traj_offsets)
    rng = np.random.default_rng(seed + 40)
    old = rng.normal(-2.0, 1.0, lay.n_tokens).astype(np.float32)
    roll = W.rollout_logp_from(old, seed, std=0.02)
    return lay, tt.astype(np.int32), old, roll


def run(R, tt, mask, old, roll, n, cap, traj_adv=None, token_adv=None):
    ws = R.new_workspace(n, 0)
    w, S = R.rl_sequence_is_weights(to_dev(tt), to_dev(mask), to_dev(old), to_dev(roll), n, ws, cap=cap,
                                    want_log_ratio=True, traj_adv_inout=traj_adv, token_adv_inout=token_adv)
    word = R.rl_query_status(ws)[1]
    return w.cpu().numpy().astype(np.float64), S.cpu().numpy().astype(np.float64), word


def check(w_d, S_d, w_ref, S_ref, n_i, what):
    u = 2.0 ** -24
    assert np.all(np.abs(S_d - S_ref) <= n_i * 2.0 ** -41 + u * np.abs(S_ref) + 1e-30), f"{what}: S"
    assert np.all(np.abs(w_d - w_ref) <= (n_i * 2.0 ** -40 + 2 * u) * w_ref + 1e-30), f"{what}: w"


@pytest.mark.parametrize("name,cap", [("multiturn", 0.0), ("multiturn", 1.02), ("edge", 2.0), ("longhorizon", 5.0)])
def test_sequence_weights_parity(R, name, cap):
    lay, tt, old, roll = batch(name)
    n = lay.n_traj
    w_d, S_d, word = run(R, tt, lay.mask, old, roll, n, cap)
    assert word == 0
    w_ref, S_ref = O.sequence_is_weights(tt, lay.mask, old, roll, n, cap)
    n_i = np.bincount(tt[lay.mask != 0], minlength=n)
    check(w_d, S_d, w_ref, S_ref, n_i, name)
    if cap > 0:
        assert np.all(w_d <= np.float32(cap))


def test_any_token_order_bit_identical(R):
    """Owners in arbitrary order (a tree-packed or shuffled batch): the same bits."""
    lay, tt, old, roll = batch("multiturn")
    perm = np.random.default_rng(1).permutation(lay.n_tokens)
    w1, S1, _ = run(R, tt, lay.mask, old, roll, lay.n_traj, 1.5)
    w2, S2, word = run(R, tt[perm], lay.mask[perm], old[perm], roll[perm], lay.n_traj, 1.5)
    assert word == 0
    assert np.array_equal(w1, w2) and np.array_equal(S1, S2)


def test_advantage_scaling_in_place(R):
    lay, tt, old, roll = batch("multiturn")
    n, T = lay.n_traj, lay.n_tokens
    rng = np.random.default_rng(2)
    a_traj = torch.from_numpy(rng.normal(0, 1, n).astype(np.float32)).cuda()
    a_tok = torch.from_numpy(rng.normal(0, 1, T).astype(np.float32)).cuda()
    a_traj0, a_tok0 = a_traj.clone(), a_tok.clone()
    w_d, _, word = run(R, tt, lay.mask, old, roll, n, 1.2, traj_adv=a_traj, token_adv=a_tok)
    assert word == 0
    w = torch.from_numpy(w_d.astype(np.float32)).cuda()
    assert torch.equal(a_traj, a_traj0 * w)
    assert torch.equal(a_tok, a_tok0 * w[torch.from_numpy(tt).long().cuda()])


def test_bad_owner_and_value(R):
    lay, tt, old, roll = batch("tiny")
    tt2, old2 = tt.copy(), old.copy()
    t_bad = int(np.nonzero(lay.mask)[0][0])
    tt2[t_bad] = lay.n_traj + 3
    w_d, _, word = run(R, tt2, lay.mask, old, roll, lay.n_traj, 0.0)
    assert word == R.RL_DEV_BAD_TRAJ
    keep = np.ones(lay.n_tokens, bool)
    keep[t_bad] = False
    w_ref, _ = O.sequence_is_weights(tt[keep], lay.mask[keep], old[keep], roll[keep], lay.n_traj, 0.0)
    assert np.allclose(w_d, w_ref, rtol=1e-6)
    old2[t_bad] = np.nan
    _, _, word = run(R, tt, lay.mask, old2, roll, lay.n_traj, 0.0)
    assert word == R.RL_DEV_BAD_VALUE


def test_loss_with_sequence_weights(R):
    """End to end: weights from the whole batch scale A_i; the loss and gradient match the
    oracle's objective with w_i on the surrogate (entropy and KL unscaled)."""
    c = make_case("tiny", seed=3, tis=True)  # rollout_logp drawn for TIS; used here at sequence level
    P = dataclasses.replace(c.P, tis_cap=0.0)
    w_ref, _ = O.sequence_is_weights(c.token_traj, c.layout.mask, c.old, c.roll, c.layout.n_traj, 1.3)
    adv32 = c.adv64.astype(np.float32)
    a_dev = to_dev(adv32)
    ws = R.new_workspace(max(c.layout.n_traj, c.rows), c.raw.shape[1])
    R.rl_sequence_is_weights(to_dev(c.token_traj.astype(np.int32)), to_dev(c.layout.mask), to_dev(c.old),
                             to_dev(c.roll), c.layout.n_traj, ws, cap=1.3, traj_adv_inout=a_dev)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    grad = R.rl_policy_loss_fwd_bwd(logits_to_dev(c), to_dev(c.ids), to_dev(c.mask), to_dev(c.tt.astype(np.int32)),
                                    a_dev, to_dev(c.coef64.astype(np.float32)), to_dev(c.old), cuda_params(R, P), ws,
                                    loss)
    assert R.rl_query_status(ws)[1] == 0
    loss_ref, g_ref, _, contrib = O.policy_loss_fwd_bwd(c.raw, c.w.dtype, c.ids, c.mask, c.tt,
                                                        adv32.astype(np.float64) * w_ref,
                                                        c.coef64.astype(np.float32).astype(np.float64), c.old, P)
    check_loss(loss.item(), loss_ref, contrib, "sequence-weighted loss")
    check_grad(grad_to_np(grad), g_ref, c.w.dtype, "sequence-weighted grad")
