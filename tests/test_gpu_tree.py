"""Tree-packed batches on the GPU (Sec. 3.2.1-3.2.3): deduplicated prefix-tree tokens from the
native builder, owners in any order, against the oracle.

Counts by owner are bit-exact; advantages and coefficients within one float32 rounding of the
float64 oracle; the loss and gradient with the logits-path tolerances; A_t = R_i - V_t exactly
(one float32 subtraction)."""

import dataclasses

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
import oracle.prefix_tree as PT
from parity_cases import check_grad, check_loss, cuda_params, grad_to_np, to_dev
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


@pytest.fixture(scope="module")
def packed(R):
    w = dataclasses.replace(W.WORKLOADS["tree"], vocab=4096)
    prompts, calls, aux = W.tree_rollouts(w, seed=2, n_rollouts=32)
    out = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves)
    n = len(prompts)
    rng = np.random.default_rng(3)
    rewards = (rng.random(n) < 0.4).astype(np.float32)
    valid = np.array([s["valid"] for s in out["stats"]], np.uint8)
    return w, out, n, rewards, valid


def _ulp_close(a, b):
    return np.all(np.abs(a - b) <= 2.0 ** -23 * np.abs(b) + 1e-30)


@pytest.mark.parametrize("interleave", [False, True])
def test_group_advantages_by_owner(R, packed, interleave):
    w, out, n, rewards, valid = packed
    owner, mask = out["owner"], out["mask"]
    if interleave:  # any token order: a random permutation of the packed stream
        perm = np.random.default_rng(4).permutation(len(owner))
        owner, mask = owner[perm], mask[perm]
    P = O.LossParams(loss_agg=0)
    go = np.arange(0, n + 1, 8, dtype=np.int32)
    ws = R.new_workspace(0, 0)
    adv, coef, L = R.rl_group_advantages_by_owner(to_dev(go), to_dev(rewards), to_dev(owner), to_dev(mask),
                                                  cuda_params(R, P), ws, traj_valid=to_dev(valid))
    assert R.rl_query_status(ws)[1] == 0
    a_ref, c_ref, L_ref = PT.advantages_and_coefficients_by_owner(rewards, go, owner, mask, n, valid, P)
    assert np.array_equal(L.cpu().numpy(), L_ref)
    assert _ulp_close(adv.cpu().numpy().astype(np.float64), a_ref)
    assert _ulp_close(coef.cpu().numpy().astype(np.float64), c_ref)
    # discarded rollouts own no tokens and get nothing
    assert np.all(L_ref[valid == 0] == 0) and np.all(c_ref[valid == 0] == 0)


def test_policy_loss_on_tree_tokens(R, packed):
    """A microbatch of the packed tree stream through rl_policy_loss_fwd_bwd: rows are the
    deduplicated tokens, token_traj the owning rollout, coefficients from the deduplicated counts."""
    w, out, n, rewards, valid = packed
    P = O.LossParams(loss_agg=0)
    go = np.arange(0, n + 1, 8, dtype=np.int32)
    a_ref, c_ref, _ = PT.advantages_and_coefficients_by_owner(rewards, go, out["owner"], out["mask"], n, valid, P)
    lo, rows = 1000, 2500
    sl = slice(lo, lo + rows)
    raw, vals = W.logits_rows_np(w, 5, lo, rows)
    ids = out["tokens"][sl].astype(np.int32)
    logp, _, _ = O.token_logprobs(raw, "bf16", ids)
    old = W.old_logp_from(logp, w, 5, lo)
    adv32, coef32 = a_ref.astype(np.float32), c_ref.astype(np.float32)
    loss_ref, g_ref, _, contrib = O.policy_loss_fwd_bwd(raw, "bf16", ids, out["mask"][sl], out["owner"][sl],
                                                        adv32.astype(np.float64), coef32.astype(np.float64), old, P)
    ws = R.new_workspace(rows, w.vocab)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    logits = torch.from_numpy(raw.view(np.int16).copy()).view(torch.bfloat16).cuda()
    grad = R.rl_policy_loss_fwd_bwd(logits, to_dev(ids), to_dev(out["mask"][sl]), to_dev(out["owner"][sl]),
                                    to_dev(adv32), to_dev(coef32), to_dev(old), cuda_params(R, P), ws, loss)
    assert R.rl_query_status(ws)[1] == 0
    check_loss(loss.item(), loss_ref, contrib, "tree loss")
    check_grad(grad_to_np(grad), g_ref, "bf16", "tree grad")


def test_rollout_value_advantages(R, packed):
    w, out, n, rewards, valid = packed
    T = len(out["owner"])
    V = W.value_predictions(w, 0, T)
    ws = R.new_workspace(0, 0)
    adv, ret = R.rl_rollout_value_advantages(to_dev(out["owner"]), to_dev(out["mask"]), to_dev(V), to_dev(rewards),
                                             ws)
    assert R.rl_query_status(ws)[1] == 0
    a_ref, g_ref = PT.rollout_value_advantages(out["owner"], out["mask"], V, rewards)
    assert np.array_equal(adv.cpu().numpy(), a_ref.astype(np.float32))  # one float32 subtraction: exact
    assert np.array_equal(ret.cpu().numpy(), g_ref.astype(np.float32))


def test_tree_sequence_weights(R, packed):
    """Sequence-level weights over a rollout's deduplicated tree tokens (owners not contiguous
    after a permutation) match the oracle."""
    w, out, n, rewards, valid = packed
    T = len(out["owner"])
    rng = np.random.default_rng(9)
    old = rng.normal(-2.0, 1.0, T).astype(np.float32)
    roll = W.rollout_logp_from(old, 1, std=0.01)
    perm = rng.permutation(T)
    ws = R.new_workspace(n, 0)
    wt, _ = R.rl_sequence_is_weights(to_dev(out["owner"][perm]), to_dev(out["mask"][perm]), to_dev(old[perm]),
                                     to_dev(roll[perm]), n, ws, cap=3.0)
    assert R.rl_query_status(ws)[1] == 0
    w_ref, _ = O.sequence_is_weights(out["owner"], out["mask"], old, roll, n, 3.0)
    n_i = np.bincount(out["owner"][out["mask"] != 0], minlength=n)
    assert np.all(np.abs(wt.cpu().numpy() - w_ref) <= (n_i * 2.0 ** -40 + 2.0 ** -23) * w_ref + 1e-30)


def test_full_tree_workload_by_owner(R):
    """The benchmark's tree batch (128 rollouts, 652K packed tokens): counts by owner bit-exact
    against the oracle, A_i and c_i within one float32 rounding, sequence weights too."""
    w = W.WORKLOADS["tree"]
    prompts, calls, aux = W.tree_rollouts(w, seed=0)
    out = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves)
    n = len(prompts)
    rewards = (np.random.default_rng(0).random(n) < w.reward_p).astype(np.float32)
    valid = np.array([s["valid"] for s in out["stats"]], np.uint8)
    go = np.arange(0, n + 1, w.group_size, dtype=np.int32)
    P = O.LossParams(loss_agg=0)
    ws = R.new_workspace(n, 0)
    adv, coef, L = R.rl_group_advantages_by_owner(to_dev(go), to_dev(rewards), to_dev(out["owner"]),
                                                  to_dev(out["mask"]), cuda_params(R, P), ws,
                                                  traj_valid=to_dev(valid))
    assert R.rl_query_status(ws)[1] == 0
    L_ref = np.bincount(out["owner"][out["mask"] != 0], minlength=n)  # plain count by owner
    assert np.array_equal(L.cpu().numpy(), L_ref)
    a_ref, c_ref, L2 = PT.advantages_and_coefficients_by_owner(rewards, go, out["owner"], out["mask"], n, valid, P)
    assert np.array_equal(L2, L_ref)
    assert _ulp_close(adv.cpu().numpy().astype(np.float64), a_ref)
    assert _ulp_close(coef.cpu().numpy().astype(np.float64), c_ref)
