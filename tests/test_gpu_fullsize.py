"""Full-size parity: whole microbatches of the workloads, in the launch configuration
the benchmark times (same entry points, same shapes).

The oracle computes log-probabilities, entropies and log-sum-exps of EVERY row (a
spawn pool over row ranges); those fix old_logp and ref_logp, every row's loss terms
(through the oracle's own token_terms) and the loss. Gradients are compared row by
row on a sample of rows, for which the oracle runs in full.
"""

import math

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
from oracle.pool import token_logprobs_parallel
from parity_cases import (check_grad, check_loss, check_stats, cuda_params, grad_to_np, logit_error_bound, loss_params,
                          to_dev)
from paper_2608_16798_gb300 import workloads as W

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

BLOCK = 8192  # rows of logits held on the host at a time


@pytest.fixture(scope="module")
def R():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_16798_gb300 import build

    build.build()
    import paper_2608_16798_gb300.rl_loss as R

    R.lib()
    return R


def _host_raw(logits, dtype):
    if dtype == "bf16":
        return logits.view(torch.int16).cpu().numpy().view(np.uint16)
    return logits.cpu().numpy()


@pytest.mark.parametrize("name,mb", [("multiturn", 0), ("multiturn", -1), ("longhorizon", 0), ("longhorizon", 1),
                                     ("longhorizon", -1), ("edge", 0)])
def test_full_microbatch(R, name, mb):
    w = W.WORKLOADS[name]
    seed = 0
    lay = W.make_layout(w, seed)
    lo, hi = W.microbatches(lay, w.microbatch)[mb]
    rows = hi - lo
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    logits = torch.empty((rows, w.vocab), dtype=dt, device="cuda")
    W.logits_rows_torch(w, seed, lo, rows, logits)
    ids = W.sample_tokens_torch(logits, seed, lo, w)
    ids_np = ids.cpu().numpy()

    # oracle over every row, in blocks of rows copied to the host one at a time
    logp, H, lse = np.empty(rows), np.empty(rows), np.empty(rows)
    for b0 in range(0, rows, BLOCK):
        b1 = min(rows, b0 + BLOCK)
        logp[b0:b1], H[b0:b1], lse[b0:b1] = token_logprobs_parallel(_host_raw(logits[b0:b1], w.dtype), w.dtype,
                                                                    ids_np[b0:b1])
    old = W.old_logp_from(logp, w, seed, lo)
    ref = W.ref_logp_from(logp, w, seed, lo) if w.ref_noise_std else None
    P = loss_params(w)
    adv, coef, L, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                     lay.traj_valid, P)
    adv32, coef32 = adv.astype(np.float32), coef.astype(np.float32)
    mask = lay.mask[lo:hi]
    tt_mb = tt[lo:hi]
    z_a = O.decode_logits(_host_raw(logits.gather(1, ids.long()[:, None])[:, 0].contiguous(), w.dtype), w.dtype)
    terms = O.token_terms(z_a, lse, H, old, adv32.astype(np.float64)[tt_mb], P, ref_logp=ref)
    c_row = coef32.astype(np.float64)[tt_mb]
    active = (mask != 0) & (c_row != 0)
    contrib = np.where(active, c_row * terms["ell"], 0.0)
    loss_ref = math.fsum(contrib.tolist())
    stats_ref = np.zeros((rows, 5))
    stats_ref[:, 0] = terms["logp"]
    stats_ref[:, 1] = terms["rho"]
    stats_ref[:, 2] = terms["cut"]
    stats_ref[:, 3] = H
    stats_ref[:, 4] = terms["kl"]
    stats_ref[~active] = 0.0

    # CUDA path, as the benchmark calls it
    ws = R.new_workspace(rows, w.vocab)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(rows * 5, dtype=torch.float32, device="cuda")
    grad = R.rl_policy_loss_fwd_bwd(logits, ids, to_dev(mask), to_dev(tt_mb.astype(np.int32)), to_dev(adv32),
                                    to_dev(coef32), to_dev(old), cuda_params(R, P), ws, loss,
                                    ref_logp=None if ref is None else to_dev(ref), token_stats=st)
    lp_d, H_d, lse_d = R.rl_token_logprobs(logits, ids, ws, want_entropy=True, want_lse=True)
    status, word = R.rl_query_status(ws)
    assert word == 0

    check_loss(loss.item(), loss_ref, contrib, f"{name} mb {mb} loss")
    check_stats(st.view(-1, 5).cpu().numpy(), stats_ref, active, f"{name} mb {mb} stats")
    lp_d, H_d, lse_d = (x.cpu().numpy().astype(np.float64) for x in (lp_d, H_d, lse_d))
    assert np.all(np.abs(lp_d - logp) <= 1e-5 + 2.0 ** -22 * np.abs(logp)), np.abs(lp_d - logp).max()
    assert np.all(np.abs(lse_d - lse) <= 1e-5 + 2.0 ** -22 * np.abs(lse)), np.abs(lse_d - lse).max()
    assert np.all(np.abs(H_d - H) <= 5e-5 + 2e-5 * np.abs(H)), np.abs(H_d - H).max()

    # every inactive row exactly zero (checked on the device), sampled rows element by element
    inactive_idx = torch.from_numpy(np.nonzero(~active)[0]).cuda()
    if inactive_idx.numel():
        assert int(torch.count_nonzero(grad.index_select(0, inactive_idx)).item()) == 0
    rng = np.random.default_rng(123)
    act_idx = np.nonzero(active)[0]
    big = act_idx[np.argsort(-np.abs(c_row[act_idx] * terms["g"][act_idx]))[:4]]
    sample = np.unique(np.concatenate([rng.choice(act_idx, size=min(16, len(act_idx)), replace=False), big,
                                       [0, rows - 1]]))
    sel = torch.from_numpy(sample).cuda()
    raw_s = _host_raw(logits.index_select(0, sel), w.dtype)
    _, g_ref, _, _ = O.policy_loss_fwd_bwd(raw_s, w.dtype, ids_np[sample], mask[sample], tt_mb[sample],
                                           adv32.astype(np.float64), coef32.astype(np.float64), old[sample], P,
                                           None if ref is None else ref[sample], None)
    g_dev = grad_to_np(grad.index_select(0, sel))
    scale = (np.abs(c_row[sample]) * (np.abs(adv32.astype(np.float64)[tt_mb][sample]) * stats_ref[sample, 1]
                                      + P.kl_coef * 2 + P.entropy_coef * (1 + np.abs(H[sample]))))[:, None]
    check_grad(g_dev, g_ref, w.dtype, f"{name} mb {mb} sampled rows", row_scale=scale)


def test_whole_multiturn_batch(R):
    """The benchmark's whole step as bench.py calls it: rl_group_advantages over the 155,959-token
    multi-turn batch, then rl_policy_loss_fwd_bwd on each of its ten 16,384-row microbatches into
    one loss accumulator (V = 151,936 bf16). The oracle computes every row's log-probability,
    entropy and log-sum-exp in float64 and, with its own advantages and coefficients, the batch
    loss. Checked: token counts and owners (bit-exact), advantages and coefficients (one float32
    ulp), the total loss, every row's statistics, every inactive row exactly zero, and gradients
    on sampled rows of every microbatch."""
    w = W.WORKLOADS["multiturn"]
    seed = 0
    lay = W.make_layout(w, seed)
    T = lay.n_tokens
    logits = torch.empty((T, w.vocab), dtype=torch.bfloat16, device="cuda")
    W.logits_rows_torch(w, seed, 0, T, logits)
    ids = W.sample_tokens_torch(logits, seed, 0, w)
    ids_np = ids.cpu().numpy()
    logp, H, lse = np.empty(T), np.empty(T), np.empty(T)
    for b0 in range(0, T, BLOCK):
        b1 = min(T, b0 + BLOCK)
        logp[b0:b1], H[b0:b1], lse[b0:b1] = token_logprobs_parallel(_host_raw(logits[b0:b1], "bf16"), "bf16",
                                                                    ids_np[b0:b1])
    old = W.old_logp_from(logp, w, seed)
    P = loss_params(w)
    adv, coef, L, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                     lay.traj_valid, P)

    # the CUDA path: advantages over the batch, then the microbatches
    ws = R.new_workspace(w.microbatch, w.vocab)
    a_d, c_d, n_d, tt_d = R.rl_group_advantages(to_dev(lay.group_offsets), to_dev(lay.rewards),
                                                to_dev(lay.traj_offsets), to_dev(lay.mask), cuda_params(R, P), ws,
                                                traj_valid=to_dev(lay.traj_valid))
    mbs = W.microbatches(lay, w.microbatch)
    assert len(mbs) == 10
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(T * 5, dtype=torch.float32, device="cuda")
    grad = torch.empty_like(logits)
    mask_d, old_d = to_dev(lay.mask), to_dev(old.astype(np.float32))
    for lo, hi in mbs:
        R.rl_policy_loss_fwd_bwd(logits[lo:hi], ids[lo:hi], mask_d[lo:hi], tt_d[lo:hi], a_d, c_d, old_d[lo:hi],
                                 cuda_params(R, P), ws, loss, grad_out=grad[lo:hi], token_stats=st[lo * 5:hi * 5])
    assert R.rl_query_status(ws)[1] == 0
    assert np.array_equal(n_d.cpu().numpy(), L) and np.array_equal(tt_d.cpu().numpy(), tt)
    a32, c32 = a_d.cpu().numpy().astype(np.float64), c_d.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(a32 - adv) <= 2.0 ** -23 * np.abs(adv)) and np.all(np.abs(c32 - coef) <= 2.0 ** -23 * coef)

    adv_o, coef_o = adv.astype(np.float32).astype(np.float64), coef.astype(np.float32).astype(np.float64)
    z_a = O.decode_logits(_host_raw(logits.gather(1, ids.long()[:, None])[:, 0].contiguous(), "bf16"), "bf16")
    terms = O.token_terms(z_a, lse, H, old, adv_o[tt], P)
    c_row = coef_o[tt]
    active = (lay.mask != 0) & (c_row != 0)
    contrib = np.where(active, c_row * terms["ell"], 0.0)
    check_loss(loss.item(), math.fsum(contrib.tolist()), contrib, "whole multi-turn batch loss")
    stats_ref = np.stack([terms["logp"], terms["rho"], terms["cut"], H, terms["kl"]], axis=1)
    stats_ref[~active] = 0.0
    check_stats(st.view(-1, 5).cpu().numpy(), stats_ref, active, "whole multi-turn batch stats")

    inactive_idx = torch.from_numpy(np.nonzero(~active)[0]).cuda()
    assert int(torch.count_nonzero(grad.index_select(0, inactive_idx)).item()) == 0
    rng = np.random.default_rng(321)
    sample = []
    for lo, hi in mbs:
        act = np.nonzero(active[lo:hi])[0] + lo
        sample.extend(rng.choice(act, size=min(3, len(act)), replace=False).tolist())
    sample = np.array(sorted(sample))
    sel = torch.from_numpy(sample).cuda()
    _, g_ref, _, _ = O.policy_loss_fwd_bwd(_host_raw(logits.index_select(0, sel), "bf16"), "bf16", ids_np[sample],
                                           lay.mask[sample], tt[sample], adv_o, coef_o, old[sample], P)
    scale = (np.abs(c_row[sample]) * np.abs(adv_o[tt][sample]) * stats_ref[sample, 1])[:, None]
    check_grad(grad_to_np(grad.index_select(0, sel)), g_ref, "bf16", "whole batch sampled rows", row_scale=scale)


def test_fused_head_full_size(R):
    """The fused LM head at 32,768 x 4,096 x 151,936 (four chunks), as the benchmark calls it.

    The oracle forms every token's logits row in float64 (host GEMM blocks) for lse and the
    entropy; old_logp follows from them. Loss and statistics are checked for every token,
    d_hidden on sampled tokens, d_weight on sampled vocabulary rows (their column of dZ over
    all tokens), with the bound of test_gpu_fused_head.py."""
    w = W.WORKLOADS["fusedhead"]
    T, D, V, seed = 32768, w.hidden, w.vocab, 0
    hidden = torch.empty((T, D), dtype=torch.bfloat16, device="cuda")
    weight = torch.empty((V, D), dtype=torch.bfloat16, device="cuda")
    W.hidden_and_weight_torch(w, seed, T, hidden, weight)
    Hm = O.decode_logits(_host_raw(hidden, "bf16"), "bf16")
    Wm = O.decode_logits(_host_raw(weight, "bf16"), "bf16")
    rng = np.random.default_rng(17)
    # sampled ids: Gumbel-max over softmax(hidden W^T), drawn on the device (input synthesis)
    ids_d = torch.empty(T, dtype=torch.int32, device="cuda")
    g = torch.Generator(device="cuda")
    for r0 in range(0, T, 1024):
        g.manual_seed(1000 + r0)
        z = torch.matmul(hidden[r0:r0 + 1024], weight.t()).float()
        u = torch.rand(z.shape, generator=g, device="cuda").clamp_(min=1e-30).log_().neg_().log_().neg_()
        ids_d[r0:r0 + 1024] = torch.argmax(z + u, dim=1).to(torch.int32)
        del z, u
    ids = ids_d.cpu().numpy()
    lse, H, z_a = np.empty(T), np.empty(T), np.empty(T)
    for r0 in range(0, T, 1024):
        Z = Hm[r0:r0 + 1024] @ Wm.T
        l, _, h, _, za = O.row_statistics(Z, ids[r0:r0 + 1024])
        lse[r0:r0 + 1024], H[r0:r0 + 1024], z_a[r0:r0 + 1024] = l, h, za
        del Z
    logp = z_a - lse
    lay = W.make_layout(w, seed)
    P = loss_params(w)
    adv, coef, L, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                     lay.traj_valid, P)
    adv32, coef32 = adv.astype(np.float32), coef.astype(np.float32)
    mask, tt_t = lay.mask[:T], tt[:T]
    old = W.old_logp_from(logp, w, seed)

    ws = R.new_workspace(T, V, D)
    # forward-only log-probs (the old / reference policy recompute) on every token
    zerr = logit_error_bound(Hm, Wm)
    f_logp, f_H, f_lse = R.rl_fused_head_token_logprobs(hidden, weight, ids_d, ws, want_entropy=True, want_lse=True)
    assert R.rl_query_status(ws)[1] == 0
    f_logp, f_H, f_lse = (x.cpu().numpy().astype(np.float64) for x in (f_logp, f_H, f_lse))
    assert np.all(np.abs(f_logp - logp) <= 1e-5 + 2.0 ** -22 * np.abs(logp) + zerr), np.abs(f_logp - logp).max()
    assert np.all(np.abs(f_lse - lse) <= 1e-5 + 2.0 ** -22 * np.abs(lse) + zerr), np.abs(f_lse - lse).max()
    assert np.all(np.abs(f_H - H) <= 5e-5 + 2e-5 * np.abs(H) + 2 * zerr), np.abs(f_H - H).max()

    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(T * 5, dtype=torch.float32, device="cuda")
    dW = torch.zeros((V, D), dtype=torch.float32, device="cuda")
    dH = R.rl_fused_head_loss_fwd_bwd(hidden, weight, to_dev(ids), to_dev(mask), to_dev(tt_t.astype(np.int32)),
                                      to_dev(adv32), to_dev(coef32), to_dev(old), cuda_params(R, P), ws, loss, dW,
                                      d_hidden_dtype=torch.float32, token_stats=st)
    assert R.rl_query_status(ws)[1] == 0

    A_t, c_t = adv32.astype(np.float64)[tt_t], coef32.astype(np.float64)[tt_t]
    terms = O.token_terms(z_a, lse, H, old, A_t, P)
    active = (mask != 0) & (c_t != 0)
    contrib = np.where(active, c_t * terms["ell"], 0.0)
    check_loss(loss.item(), math.fsum(contrib.tolist()), contrib, "fused head full-size loss")
    stats_ref = np.stack([terms["logp"], terms["rho"], terms["cut"], H, terms["kl"]], axis=1)
    stats_ref[~active] = 0.0
    check_stats(st.view(-1, 5).cpu().numpy(), stats_ref, active, "fused head full-size stats",
                zerr=logit_error_bound(Hm, Wm))

    # dZ rows of sampled tokens and dZ columns of sampled vocabulary entries, in float64
    g_t = np.where(active, c_t * terms["g"], 0.0)

    def dz_rows(rows):
        Z = Hm[rows] @ Wm.T
        p = np.exp(Z - lse[rows, None])
        dz = -g_t[rows, None] * p
        dz[np.arange(len(rows)), ids[rows]] += g_t[rows]
        return dz

    act_idx = np.nonzero(active)[0]
    rows = np.unique(np.concatenate([rng.choice(act_idx, 24, replace=False), np.nonzero(~active)[0][:4]]))
    dz = dz_rows(rows)
    ref_dH = dz @ Wm
    S_h = np.sqrt((dz ** 2) @ (Wm ** 2))
    got = dH.index_select(0, torch.from_numpy(rows).cuda()).cpu().numpy().astype(np.float64)
    tol = 2.0 ** -6 * S_h + 1e-4 * np.abs(ref_dH) + 1e-6 * np.abs(ref_dH).max() + 1e-30
    assert np.all(np.abs(got - ref_dH) <= tol), np.abs(got - ref_dH).max()

    vs = np.unique(np.concatenate([ids[rng.choice(act_idx, 8, replace=False)], rng.integers(0, V, 24)]))
    Zc = Hm @ Wm[vs].T                                     # [T x |vs|]
    p = np.exp(Zc - lse[:, None])
    dzc = -g_t[:, None] * p + g_t[:, None] * (ids[:, None] == vs[None, :])
    ref_dW = dzc.T @ Hm                                    # [|vs| x D]
    S_w = np.sqrt((dzc.T ** 2) @ (Hm ** 2))
    got = dW.index_select(0, torch.from_numpy(vs).cuda()).cpu().numpy().astype(np.float64)
    tol = 2.0 ** -6 * S_w + 1e-4 * np.abs(ref_dW) + 1e-6 * np.abs(ref_dW).max() + 1e-30
    assert np.all(np.abs(got - ref_dW) <= tol), np.abs(got - ref_dW).max()
