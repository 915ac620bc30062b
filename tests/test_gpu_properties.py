"""Properties of the CUDA path that need no oracle (needs a GB300).

Reordering whole groups in the packed batch (each group's trajectories and their tokens move
together) changes nothing a row or a trajectory sees: its own logits, its group's rewards, and
N, S over the batch. So after the reordering every row's gradient and statistics and every
trajectory's advantage, coefficient and count must be the same bits, and the loss the same up
to the order of its sum.
"""

import dataclasses

import numpy as np
import pytest
import torch

from parity_cases import cuda_params, loss_params, to_dev
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


def _reorder_groups(lay, perm):
    """The layout with its groups in the order perm; returns (group offsets, trajectory offsets,
    rewards, validity, mask) of the new packing, the old trajectory of each new one and the old
    token of each new one."""
    go, to = lay.group_offsets, lay.traj_offsets
    traj_order = np.concatenate([np.arange(go[g], go[g + 1]) for g in perm]).astype(np.int64)
    sizes = np.array([go[g + 1] - go[g] for g in perm])
    new_go = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    lens = (to[1:] - to[:-1])[traj_order]
    new_to = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tok_order = np.concatenate([np.arange(to[i], to[i + 1]) for i in traj_order]).astype(np.int64)
    return (new_go, new_to, lay.rewards[traj_order], lay.traj_valid[traj_order], lay.mask[tok_order], traj_order,
            tok_order)


def _step(R, P, go, to, rewards, valid, mask, logits, ids, old):
    T, V = logits.shape
    ws = R.new_workspace(T, V)
    adv, coef, n_tok, tt = R.rl_group_advantages(to_dev(go), to_dev(rewards), to_dev(to), to_dev(mask),
                                                 cuda_params(R, P), ws, traj_valid=to_dev(valid))
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(T * 5, dtype=torch.float32, device="cuda")
    grad = R.rl_policy_loss_fwd_bwd(logits, ids, to_dev(mask), tt, adv, coef, old, cuda_params(R, P), ws, loss,
                                    token_stats=st)
    assert R.rl_query_status(ws)[1] == 0
    return adv, coef, n_tok, grad, st.view(T, 5), loss.item()


@pytest.mark.parametrize("name,vocab", [("multiturn", 4096), ("edge", None)])  # warp-per-row, cluster kernel
def test_reordering_groups_changes_nothing(R, name, vocab):
    w = W.WORKLOADS[name] if vocab is None else dataclasses.replace(W.WORKLOADS[name], vocab=vocab)
    lay = W.make_layout(w, 3)
    T = lay.n_tokens
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    logits = torch.empty((T, w.vocab), dtype=dt, device="cuda")
    W.logits_rows_torch(w, 3, 0, T, logits)
    ids = W.sample_tokens_torch(logits, 3, 0, w)
    logp, _, _ = R.rl_token_logprobs(logits, ids, R.new_workspace(T, w.vocab))
    old = to_dev(W.old_logp_from(logp.cpu().numpy().astype(np.float64), w, 3))
    P = loss_params(w, loss_agg=0)

    a0, c0, n0, g0, s0, l0 = _step(R, P, lay.group_offsets, lay.traj_offsets, lay.rewards, lay.traj_valid, lay.mask,
                                   logits, ids, old)
    perm = np.random.default_rng(4).permutation(len(lay.group_offsets) - 1)
    go, to, rw, va, mk, traj_order, tok_order = _reorder_groups(lay, perm)
    t_ord = torch.from_numpy(tok_order).cuda()
    j_ord = torch.from_numpy(traj_order).cuda()
    a1, c1, n1, g1, s1, l1 = _step(R, P, go, to, rw, va, mk, logits.index_select(0, t_ord).contiguous(),
                                   ids.index_select(0, t_ord).contiguous(), old.index_select(0, t_ord).contiguous())

    assert torch.equal(a1, a0.index_select(0, j_ord)) and torch.equal(c1, c0.index_select(0, j_ord))
    assert torch.equal(n1, n0.index_select(0, j_ord))
    assert torch.equal(s1, s0.index_select(0, t_ord))
    view = torch.int16 if dt == torch.bfloat16 else torch.int32
    assert torch.equal(g1.view(view), g0.index_select(0, t_ord).view(view))
    # the loss terms are the same; only the order of the double-precision sum changes
    assert abs(l1 - l0) <= 1e-9 * max(abs(l0), 1e-30) + 1e-15, (l0, l1)


def test_fused_head_token_order(R):
    """The fused head with its tokens reordered (each with its id, mask, owner and old_logp):
    every token's d_hidden row and statistics are the same bits, the loss the same up to the
    order of its sum, and d_W, a sum over tokens that the products now group differently, the
    same up to float32 rounding of its terms."""
    from test_gpu_fused_head import make_head_case, run_head

    c = make_head_case(4096 + 515, 192, 3000, seed=31, agg=0, ent=True)
    a = run_head(R, c)
    perm = np.random.default_rng(5).permutation(c["T"])
    p = dict(c)
    p["h"] = c["h"][perm]
    for k in ("ids", "mask", "tt", "old", "ref"):
        p[k] = c[k][perm]
    b = run_head(R, p)
    assert a["word"] == 0 and b["word"] == 0
    assert np.array_equal(b["dH"], a["dH"][perm]), "d_hidden rows differ after reordering the tokens"
    assert np.array_equal(b["stats"], a["stats"][perm])
    assert abs(b["loss"] - a["loss"]) <= 1e-9 * max(abs(a["loss"]), 1e-30) + 1e-15
    scale = np.abs(a["dW"]).max()
    assert np.all(np.abs(b["dW"] - a["dW"]) <= 1e-3 * scale + 1e-5 * np.abs(a["dW"])), \
        np.abs(b["dW"] - a["dW"]).max() / scale


@pytest.mark.parametrize("name,vocab", [("multiturn", 4096), ("multiturn", None), ("edge", None)])
def test_statistics_request_changes_no_bit(R, name, vocab):
    """Asking for the per-token statistics selects the kernel form that also sums the entropy;
    with no entropy bonus (alpha = 0) the loss is the same bits and every gradient element the
    same value as without the statistics (the warp-per-row kernel and the cluster kernel, bf16
    and fp32), logits at -inf included. Zeros may differ in sign: in a row whose surrogate
    weight c g is 0 and whose log-sum-exp lies below its entropy (the edge workload's rows at
    -1e4), the entropy form's coefficient is -0 + 0 (H - lse) = +0 where the other's is -0."""
    from parity_cases import make_case, logits_to_dev

    case = make_case(name, seed=41, row0=500, rows=300, vocab=vocab, loss_agg=2)
    raw = case.raw.copy()
    ninf = np.uint16(0xFF80) if case.w.dtype == "bf16" else np.float32(-np.inf)
    for r in range(0, case.rows, 3):  # a few entries at -inf (never the sampled one)
        cols = np.random.default_rng(r).choice(raw.shape[1], size=max(1, raw.shape[1] // 50), replace=False)
        cols = cols[cols != case.ids[r]]
        raw[r, cols] = ninf
    case = dataclasses.replace(case, raw=raw)
    logits = logits_to_dev(case)
    args = (to_dev(case.ids), to_dev(case.mask), to_dev(case.tt.astype(np.int32)),
            to_dev(case.adv64.astype(np.float32)), to_dev(case.coef64.astype(np.float32)), to_dev(case.old),
            cuda_params(R, case.P))
    assert case.P.entropy_coef == 0.0
    outs = []
    for stats in (None, torch.zeros(case.rows * 5, dtype=torch.float32, device="cuda")):
        ws = R.new_workspace(case.rows, raw.shape[1])
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        g = R.rl_policy_loss_fwd_bwd(logits, *args, ws, loss, ref_logp=None if case.ref is None else to_dev(case.ref),
                                     token_stats=stats)
        assert R.rl_query_status(ws)[1] == 0
        outs.append((loss.item(), g))
    assert outs[0][0] == outs[1][0]
    assert torch.equal(outs[0][1], outs[1][1])  # values: -0 == +0


def test_stats_summary_skips_bad_owners(R):
    """Rows whose owner is outside [0, n_traj) set RL_DEV_BAD_TRAJ and are left out of the sums."""
    import oracle.grpo_objective as O

    rng = np.random.default_rng(8)
    rows, n_traj = 20000, 50
    stats = rng.random((rows, 5), dtype=np.float32)
    mask = (rng.random(rows) < 0.7).astype(np.uint8)
    tt = rng.integers(0, n_traj, rows).astype(np.int32)
    bad = rng.choice(rows, size=37, replace=False)
    tt[bad] = np.where(np.arange(37) % 2 == 0, -3, n_traj + 5)
    coef = rng.random(n_traj).astype(np.float32)
    ws = R.new_workspace(0, 0)
    got = R.rl_token_stats_summary(torch.from_numpy(stats.reshape(-1)).cuda(), to_dev(mask), to_dev(tt),
                                   to_dev(coef), ws).cpu().numpy()
    assert R.rl_query_status(ws)[1] & R.RL_DEV_BAD_TRAJ
    keep = np.ones(rows, bool)
    keep[bad] = False
    ref = O.stats_summary(stats[keep].astype(np.float64), mask[keep], tt[keep], coef)
    assert got[0] == ref[0] and got[1] == ref[1] and np.allclose(got[2:], ref[2:], rtol=1e-12, atol=1e-12)
