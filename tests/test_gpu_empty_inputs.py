"""Empty inputs through every entry point on the GPU: no tokens, no trajectories, trajectories
without tokens. Each call returns RL_OK, leaves the accumulators it would add to unchanged,
and, where trajectories exist without tokens, gives the oracle's per-trajectory values
(no trainable token: L_i = 0 and c_i = 0; the sequence-level weight of an empty sum is
min(exp(0), cap))."""
import numpy as np
import pytest
import torch

import oracle.grpo_objective as O

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


def dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def zeros(n, dt):
    return torch.zeros(n, dtype=dt, device="cuda")


def test_no_trajectories_no_tokens(R):
    ws = R.new_workspace(0, 0)
    p = R.make_params()
    adv, coef, n_tok, tt = R.rl_group_advantages(dev(np.zeros(1, np.int32)), zeros(0, torch.float32),
                                                 dev(np.zeros(1, np.int64)), zeros(0, torch.uint8), p, ws)
    assert adv.numel() == coef.numel() == n_tok.numel() == tt.numel() == 0
    a2, c2, n2 = R.rl_group_advantages_by_owner(dev(np.zeros(1, np.int32)), zeros(0, torch.float32),
                                                zeros(0, torch.int32), zeros(0, torch.uint8), p, ws)
    assert a2.numel() == c2.numel() == n2.numel() == 0
    A, G = R.rl_masked_gae(dev(np.zeros(1, np.int64)), zeros(0, torch.uint8), zeros(0, torch.float32), ws)
    assert A.numel() == 0 and G.numel() == 0
    loss = torch.full((1,), -2.25, dtype=torch.float64, device="cuda")
    dv = R.rl_value_loss_fwd_bwd(zeros(0, torch.float32), zeros(0, torch.float32), zeros(0, torch.uint8),
                                 zeros(0, torch.int32), zeros(0, torch.float32), ws, loss)
    assert dv.numel() == 0
    A2, G2 = R.rl_rollout_value_advantages(zeros(0, torch.int32), zeros(0, torch.uint8), zeros(0, torch.float32),
                                           zeros(0, torch.float32), ws)
    assert A2.numel() == 0 and G2.numel() == 0
    w, lr = R.rl_sequence_is_weights(zeros(0, torch.int32), zeros(0, torch.uint8), zeros(0, torch.float32),
                                     zeros(0, torch.float32), 0, ws, cap=2.0, want_log_ratio=True)
    assert w.numel() == 0 and lr.numel() == 0
    summ = torch.full((5,), 1.5, dtype=torch.float64, device="cuda")
    R.rl_token_stats_summary(zeros(0, torch.float32), zeros(0, torch.uint8), zeros(0, torch.int32),
                             zeros(0, torch.float32), ws, summary_accum=summ)
    torch.cuda.synchronize()
    assert loss.item() == -2.25 and torch.all(summ == 1.5).item()
    assert R.rl_query_status(ws)[1] == 0


def test_trajectories_without_tokens(R):
    """Four trajectories in two groups, none of them with a token: counts and coefficients are
    zero, the advantages are those of the rewards alone (the oracle's), every sequence weight
    is min(1, cap)."""
    rewards = np.array([1.0, 0.0, 0.25, 0.25], np.float32)
    go = np.array([0, 2, 4], np.int32)
    offs = np.zeros(5, np.int64)
    ws = R.new_workspace(4, 0)
    p = R.make_params()
    adv, coef, n_tok, tt = R.rl_group_advantages(dev(go), dev(rewards), dev(offs), zeros(0, torch.uint8), p, ws)
    P = O.LossParams()
    ref_adv, ref_coef, ref_L, _ = O.advantages_and_coefficients(rewards, go, offs, np.zeros(0, np.uint8),
                                                                np.ones(4, np.uint8), P)
    assert np.array_equal(n_tok.cpu().numpy(), ref_L.astype(np.int32)) and np.all(ref_L == 0)
    assert np.array_equal(coef.cpu().numpy(), ref_coef.astype(np.float32)) and np.all(ref_coef == 0)
    np.testing.assert_allclose(adv.cpu().numpy(), ref_adv, rtol=2e-7, atol=1e-7)
    a2, c2, n2 = R.rl_group_advantages_by_owner(dev(go), dev(rewards), zeros(0, torch.int32), zeros(0, torch.uint8),
                                                p, ws)
    assert torch.equal(a2, adv) and torch.equal(c2, coef) and torch.equal(n2, n_tok)
    for cap in (2.0, 0.5):
        w, lr = R.rl_sequence_is_weights(zeros(0, torch.int32), zeros(0, torch.uint8), zeros(0, torch.float32),
                                         zeros(0, torch.float32), 4, ws, cap=cap, want_log_ratio=True)
        ref_w, ref_lr = O.sequence_is_weights(np.zeros(0, np.int64), np.zeros(0, np.uint8), np.zeros(0),
                                              np.zeros(0), 4, cap)
        assert np.array_equal(lr.cpu().numpy(), ref_lr.astype(np.float32)) and np.all(ref_lr == 0)
        assert np.array_equal(w.cpu().numpy(), ref_w.astype(np.float32)) and np.all(ref_w == min(1.0, cap))
    A, G = R.rl_masked_gae(dev(offs), zeros(0, torch.uint8), zeros(0, torch.float32), ws,
                           traj_rewards=dev(rewards))
    assert A.numel() == 0 and G.numel() == 0
    assert R.rl_query_status(ws)[1] == 0


def test_fused_head_without_tokens(R):
    """T = 0 through both fused-head calls: d_weight (added to) and the loss stay as they were."""
    V, D = 1000, 128
    g = torch.Generator(device="cuda").manual_seed(5)
    weight = torch.randn((V, D), generator=g, device="cuda").to(torch.bfloat16)
    hidden = torch.zeros((0, D), dtype=torch.bfloat16, device="cuda")
    ws = R.new_workspace(0, V, D)
    loss = torch.full((1,), 0.75, dtype=torch.float64, device="cuda")
    d_weight = torch.full((V, D), 0.125, dtype=torch.float32, device="cuda")
    dh = R.rl_fused_head_loss_fwd_bwd(hidden, weight, zeros(0, torch.int32), zeros(0, torch.uint8),
                                      zeros(0, torch.int32), zeros(2, torch.float32), zeros(2, torch.float32),
                                      zeros(0, torch.float32), R.make_params(), ws, loss, d_weight)
    logp, H, lse = R.rl_fused_head_token_logprobs(hidden, weight, zeros(0, torch.int32), ws, want_entropy=True,
                                                  want_lse=True)
    torch.cuda.synchronize()
    assert dh.shape == (0, D) and logp.numel() == H.numel() == lse.numel() == 0
    assert loss.item() == 0.75 and torch.all(d_weight == 0.125).item()
    assert R.rl_query_status(ws)[1] == 0


def test_token_logprobs_without_rows(R):
    ws = R.new_workspace(1, 8)
    logp, H, lse = R.rl_token_logprobs(torch.zeros((0, 8), dtype=torch.bfloat16, device="cuda"),
                                       zeros(0, torch.int32), ws, want_entropy=True, want_lse=True)
    assert logp.numel() == H.numel() == lse.numel() == 0
    assert R.rl_query_status(ws)[1] == 0
