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
from parity_cases import check_grad, check_loss, check_stats, cuda_params, grad_to_np, loss_params, to_dev
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


@pytest.mark.parametrize("name,mb", [("multiturn", 0), ("multiturn", -1), ("longhorizon", 1), ("edge", 0)])
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
