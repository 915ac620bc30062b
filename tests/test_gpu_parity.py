"""CUDA path against the float64 oracle on seeded inputs (needs a GB300).

Sizes here let the oracle finish in seconds while spanning many tiles, all
cluster widths the launcher picks (1, 4, 8 and 16 CTAs per row), ragged
vocabulary tails, unaligned leading dimensions and the degenerate cases.
Full-size workloads are in test_gpu_fullsize.py.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
from parity_cases import (check_grad, check_loss, compare, cuda_params, grad_to_np, logits_to_dev, make_case,
                          oracle_loss, run_loss, to_dev)
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


# ----------------------------------------------------------------------------- A1..A3

@pytest.mark.parametrize("name,n_groups,invalid,agg", [
    ("tiny", None, 0.0, 0), ("multiturn", None, 0.0, 0), ("longhorizon", None, 0.0, 0), ("edge", None, 0.0, 0),
    ("multiturn", None, 0.2, 0), ("edge", 512, 0.1, 1), ("longhorizon", None, 0.1, 2)])
def test_group_advantages_parity(R, name, n_groups, invalid, agg):
    case_w = W.WORKLOADS[name]
    lay = W.make_layout(case_w, 3, n_groups)
    if invalid:
        lay.traj_valid = (np.random.default_rng(5).random(lay.n_traj) >= invalid).astype(np.uint8)
    P = O.LossParams(loss_agg=agg)
    adv, coef, L, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                     lay.traj_valid, P)
    ws = R.new_workspace(0, 0)
    a, c, n_tok, tt_d = R.rl_group_advantages(to_dev(lay.group_offsets), to_dev(lay.rewards), to_dev(lay.traj_offsets),
                                              to_dev(lay.mask), cuda_params(R, P), ws, traj_valid=to_dev(lay.traj_valid))
    st, word = R.rl_query_status(ws)
    assert word == 0
    assert np.array_equal(n_tok.cpu().numpy(), L), "trainable-token counts must be exact"
    assert np.array_equal(tt_d.cpu().numpy(), tt), "token owners must be exact"
    a, c = a.cpu().numpy().astype(np.float64), c.cpu().numpy().astype(np.float64)
    # double-precision statistics rounded once to float32: within one float32 ulp
    assert np.all(np.abs(a - adv) <= 2.0 ** -23 * np.abs(adv)), np.abs(a - adv).max()
    assert np.all(np.abs(c - coef) <= 2.0 ** -23 * np.abs(coef)), np.abs(c - coef).max()
    assert np.all(a[lay.traj_valid == 0] == 0) and np.all(c[lay.traj_valid == 0] == 0)


@pytest.mark.parametrize("scale", [1, 20000])  # a few tokens per trajectory, or tens of thousands
@pytest.mark.parametrize("go", [[2, 5, 8], [0], [0, 10], [0, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10]])
def test_group_advantages_outside_groups_and_one_member_groups(R, go, scale):
    """Trajectories before the first group or after the last keep A = 0 (also with no group at
    all), one-member groups give A = 0, and the coefficients count every trajectory."""
    rng = np.random.default_rng(len(go))
    n = 10
    rewards = rng.random(n).astype(np.float32)
    traj_offsets = np.cumsum([0] + list(rng.integers(0, 6, n) * scale)).astype(np.int64)
    mask = (rng.random(int(traj_offsets[-1])) < 0.7).astype(np.uint8)
    group_offsets = np.array(go, np.int32)
    P = O.LossParams(loss_agg=0)
    adv, coef, L, tt = O.advantages_and_coefficients(rewards, group_offsets, traj_offsets, mask, None, P)
    ws = R.new_workspace(0, 0)
    a, c, n_tok, tt_d = R.rl_group_advantages(to_dev(group_offsets), to_dev(rewards), to_dev(traj_offsets),
                                              to_dev(mask), cuda_params(R, P), ws)
    assert R.rl_query_status(ws)[1] == 0
    assert np.array_equal(n_tok.cpu().numpy(), L) and np.array_equal(tt_d.cpu().numpy(), tt)
    a, c = a.cpu().numpy().astype(np.float64), c.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(a - adv) <= 2.0 ** -23 * np.abs(adv)), (a, adv)
    assert np.all(np.abs(c - coef) <= 2.0 ** -23 * np.abs(coef)), (c, coef)
    inside = np.zeros(n, bool)
    if len(go):
        inside[go[0]:go[-1]] = True
    assert np.all(a[~inside] == 0.0)


def test_group_advantages_bad_offsets_flagged(R):
    go = to_dev(np.array([0, 3, 2], np.int32))   # decreasing
    rw = to_dev(np.zeros(3, np.float32))
    to = to_dev(np.array([0, 1, 2, 3], np.int64))
    mk = to_dev(np.ones(3, np.uint8))
    ws = R.new_workspace(0, 0)
    R.rl_group_advantages(go, rw, to, mk, R.make_params(), ws)
    st, word = R.rl_query_status(ws)
    assert st == 6 and word & R.RL_DEV_BAD_OFFSETS


# ----------------------------------------------------------------------------- B1: token log-probs

@pytest.mark.parametrize("name,row0,rows,vocab,ld_pad", [
    ("tiny", 0, 512, None, 0), ("multiturn", 700, 48, None, 0), ("edge", 0, 1024, None, 0),
    ("multiturn", 0, 16, 1001, 0), ("tiny", 0, 40, 4097, 3), ("edge", 0, 64, 999, 5),
    ("multiturn", 0, 8, 400_000, 0), ("multiturn", 0, 6, 819_200, 0), ("edge", 0, 6, 409_600, 0),
    ("tiny", 0, 7, 1, 0), ("tiny", 0, 9, 3, 8)])
def test_token_logprobs_parity(R, name, row0, rows, vocab, ld_pad):
    case = make_case(name, seed=1, row0=row0, rows=rows, vocab=vocab)
    V = case.raw.shape[1]
    logits = logits_to_dev(case, V + ld_pad)
    ws = R.new_workspace(case.rows, V)
    logp, H, lse = R.rl_token_logprobs(logits, to_dev(case.ids), ws, want_entropy=True, want_lse=True)
    st, word = R.rl_query_status(ws)
    assert word == 0
    lp_ref, H_ref, lse_ref = O.token_logprobs(case.raw, case.w.dtype, case.ids)
    lp, Hd, ls = (x.cpu().numpy().astype(np.float64) for x in (logp, H, lse))
    assert np.all(np.abs(lp - lp_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lp_ref)), np.abs(lp - lp_ref).max()
    assert np.all(np.abs(ls - lse_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lse_ref)), np.abs(ls - lse_ref).max()
    assert np.all(np.abs(Hd - H_ref) <= 5e-5 + 2e-5 * np.abs(H_ref)), np.abs(Hd - H_ref).max()
    # without the entropy output the logp path is the same numbers
    logp2, _, _ = R.rl_token_logprobs(logits, to_dev(case.ids), ws)
    assert np.all(np.abs(logp2.cpu().numpy() - lp_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lp_ref))


def test_token_logprobs_bad_token_flagged(R):
    case = make_case("tiny", rows=4)
    ids = case.ids.copy()
    ids[2] = case.raw.shape[1]
    ws = R.new_workspace(4, case.raw.shape[1])
    logp, _, _ = R.rl_token_logprobs(logits_to_dev(case), to_dev(ids), ws)
    st, word = R.rl_query_status(ws)
    assert word & R.RL_DEV_BAD_TOKEN
    lp = logp.cpu().numpy()
    assert np.isnan(lp[2]) and np.all(np.isfinite(lp[[0, 1, 3]]))


# ----------------------------------------------------------------------------- B1..B4: policy loss

@pytest.mark.parametrize("name,row0,rows,agg,tis", [
    ("tiny", 0, None, 0, False), ("tiny", 0, None, 2, False), ("tiny", 0, None, 2, True),
    ("multiturn", 1500, 96, 0, False), ("multiturn", 1500, 96, 2, False),
    ("longhorizon", 5000, 64, 0, False), ("longhorizon", 5000, 64, 2, True),
    ("edge", 0, 2048, 0, False), ("edge", 4096, 2048, 2, False), ("edge", 0, 2048, 1, True)])
def test_policy_loss_parity(R, name, row0, rows, agg, tis):
    case = make_case(name, seed=2, row0=row0, rows=rows, loss_agg=agg, tis=tis)
    out = run_loss(R, case)
    compare(case, out, f"{name}[{row0}:+{rows}] agg={agg} tis={tis}")


@pytest.mark.parametrize("vocab,ld_pad,dtype_case", [
    (1001, 0, "multiturn"), (4097, 3, "tiny"), (999, 1, "edge"), (400_000, 0, "multiturn"), (3, 5, "tiny"),
    (1, 0, "tiny"), (151_936, 16, "multiturn"),
    (819_200, 0, "multiturn"), (409_600, 8, "edge")])  # the largest rows: 16 CTAs of 100 KB
def test_policy_loss_ragged_shapes(R, vocab, ld_pad, dtype_case):
    case = make_case(dtype_case, seed=4, rows=24, vocab=vocab, loss_agg=2)
    out = run_loss(R, case, ld=vocab + ld_pad)
    compare(case, out, f"V={vocab} ld=V+{ld_pad}")


@pytest.mark.parametrize("name,vocab,ld_pad,rows,agg,tis,ent", [
    ("longhorizon", 4096, 0, 3000, 2, True, None),  # entropy + k3 KL + TIS; many rows per warp
    ("multiturn", 4096, 0, 6000, 0, False, None),   # 40% masked rows, the paper's weighting
    ("edge", 2048, 0, 2000, 2, False, None),        # fp32 at the 8 KB limit
    ("edge", 1536, 4, 800, 2, False, 1e-2),         # fp32 with the entropy term
    ("tiny", 37, 3, 200, 2, False, None),           # four vectors and a ragged tail of five
    ("longhorizon", 4104, 0, 300, 2, False, None),  # bf16 rows just over 8 KB: one CTA per row
    ("edge", 2049, 3, 300, 2, True, None)])         # fp32 rows just over 8 KB, 16-byte aligned
def test_policy_loss_short_rows(R, name, vocab, ld_pad, rows, agg, tis, ent):
    """Rows of at most 8 KB (aligned) take the warp-per-row kernel; rows just over it take the
    cluster kernel with one CTA per row. Both against the oracle, with the workloads' masks."""
    case = make_case(name, seed=21, row0=0, rows=rows, vocab=vocab, loss_agg=agg, tis=tis)
    if ent is not None:
        case = dataclasses.replace(case, P=dataclasses.replace(case.P, entropy_coef=ent))
    out = run_loss(R, case, ld=vocab + ld_pad)
    compare(case, out, f"{name} V={vocab} ld=V+{ld_pad} rows={rows}")


@pytest.mark.parametrize("name,row0,rows", [("tiny", 0, 1), ("multiturn", 100, 1), ("edge", 3, 2), ("multiturn", 0, 3)])
def test_policy_loss_fewest_rows(R, name, row0, rows):
    """One to three rows: a single cluster (or as many as rows), whose last one sums the loss."""
    case = make_case(name, seed=12, row0=row0, rows=rows, loss_agg=2)
    out = run_loss(R, case)
    compare(case, out, f"{name}[{row0}:+{rows}]")
    lp, H, lse = R.rl_token_logprobs(logits_to_dev(case), to_dev(case.ids), R.new_workspace(rows, case.raw.shape[1]),
                                     want_entropy=True, want_lse=True)
    lp_ref, H_ref, _ = O.token_logprobs(case.raw, case.w.dtype, case.ids)
    assert np.all(np.abs(lp.cpu().numpy() - lp_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lp_ref))
    assert np.all(np.abs(H.cpu().numpy() - H_ref) <= 5e-5 + 2e-5 * np.abs(H_ref))


@pytest.mark.parametrize("name,row0,rows", [("multiturn", 300, 64), ("tiny", 0, 512)])
def test_policy_loss_in_place_and_deterministic(R, name, row0, rows):
    case = make_case(name, seed=5, row0=row0, rows=rows, loss_agg=2)
    a = run_loss(R, case)
    b = run_loss(R, case, in_place=True)
    c = run_loss(R, case)
    assert a["loss"] == c["loss"], "loss must be bit-reproducible"
    assert np.array_equal(a["grad"], c["grad"]) and np.array_equal(a["grad"], b["grad"])
    compare(case, b, "in place")


@pytest.mark.parametrize("name,row0,rows,vocab", [("longhorizon", 2000, 80, None), ("longhorizon", 100, 2000, 4096)])
def test_policy_loss_microbatch_split(R, name, row0, rows, vocab):
    case = make_case(name, seed=6, row0=row0, rows=rows, vocab=vocab, loss_agg=0)
    whole = run_loss(R, case)
    parts = []
    cut = rows * 2 // 5 + 1
    for lo, hi in ((0, cut), (cut, rows)):
        sub = make_case(name, seed=6, row0=row0 + lo, rows=hi - lo, vocab=vocab, loss_agg=0)
        # the same rows: the generator is keyed by row, only the noise streams differ -> reuse the parent's
        sub.raw, sub.ids, sub.old = case.raw[lo:hi], case.ids[lo:hi], case.old[lo:hi]
        sub.ref = None if case.ref is None else case.ref[lo:hi]
        parts.append(run_loss(R, sub))
    assert abs(sum(p["loss"] for p in parts) - whole["loss"]) <= 1e-12 * max(1e-30, abs(whole["loss"])) + 1e-15
    assert np.array_equal(np.concatenate([p["grad"] for p in parts]), whole["grad"])


def test_policy_loss_all_masked_and_zero_rows(R):
    case = make_case("tiny", seed=7, rows=64)
    case.layout.mask[:] = 0
    out = run_loss(R, case)
    assert out["loss"] == 0.0 and np.all(out["grad"] == 0.0) and np.all(out["stats"] == 0.0)
    ws = R.new_workspace(1, 8)
    loss = torch.full((1,), 3.5, dtype=torch.float64, device="cuda")
    empty = torch.zeros((0, 8), dtype=torch.bfloat16, device="cuda")
    z32 = torch.zeros(0, dtype=torch.int32, device="cuda")
    R.rl_policy_loss_fwd_bwd(empty, z32, torch.zeros(0, dtype=torch.uint8, device="cuda"), z32,
                             torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda"),
                             torch.zeros(0, device="cuda"), R.make_params(), ws, loss)
    assert loss.item() == 3.5


def test_policy_loss_bad_ids_flagged_and_zeroed(R):
    case = make_case("tiny", seed=8, rows=32, loss_agg=2)
    bad_tok = case.ids.copy()
    bad_tok[3] = -1
    tt = case.tt.astype(np.int32).copy()
    tt[5] = 10_000
    logits = logits_to_dev(case)
    ws = R.new_workspace(case.rows, case.raw.shape[1])
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    g = R.rl_policy_loss_fwd_bwd(logits, to_dev(bad_tok), to_dev(case.mask), to_dev(tt),
                                 to_dev(case.adv64.astype(np.float32)), to_dev(case.coef64.astype(np.float32)),
                                 to_dev(case.old), cuda_params(R, case.P), ws, loss)
    st, word = R.rl_query_status(ws)
    assert word & R.RL_DEV_BAD_TOKEN and word & R.RL_DEV_BAD_TRAJ
    gg = grad_to_np(g)
    assert np.all(gg[[3, 5]] == 0.0) and np.any(gg[0] != 0.0)
    R.rl_workspace_init(ws)
    assert R.rl_query_status(ws)[1] == 0
    # the same workspace (its finished-cluster counter included) serves a clean call next
    clean = make_case("tiny", seed=9, rows=32)
    compare(clean, run_loss(R, clean, ws=ws), "clean call after the flagged one")


def test_end_to_end_advantages_then_loss(R):
    """GPU advantages feed the GPU loss; the oracle runs A and B in float64 end to end."""
    case = make_case("longhorizon", seed=9, row0=12000, rows=48, loss_agg=0)
    lay = case.layout
    ws = R.new_workspace(case.rows, case.raw.shape[1])
    adv, coef, n_tok, tt = R.rl_group_advantages(to_dev(lay.group_offsets), to_dev(lay.rewards),
                                                 to_dev(lay.traj_offsets), to_dev(lay.mask), cuda_params(R, case.P), ws)
    logits = logits_to_dev(case)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    sl = case.sl
    g = R.rl_policy_loss_fwd_bwd(logits, to_dev(case.ids), to_dev(case.mask), tt[sl.start:sl.stop].contiguous(),
                                 adv, coef, to_dev(case.old), cuda_params(R, case.P), ws, loss,
                                 ref_logp=to_dev(case.ref))
    l_ref, g_ref, _, contrib = oracle_loss(case)
    check_loss(loss.item(), l_ref, contrib, "end to end")
    check_grad(grad_to_np(g), g_ref, "bf16", "end to end")


# ----------------------------------------------------------------------------- logits at -inf

def neg_inf_case(name, rows, seed=6, entropy=False, fill="-inf"):
    """Rows with vocabulary entries masked to -inf (never the sampled one): 30% of the entries
    in half the rows, all but three entries in one row. old_logp and ref_logp follow from the
    masked rows' log-probabilities, so the ratio band around the clip bounds still holds.
    fill="max_finite" masks with the most negative finite value instead (exp of it is 0 too;
    x = (z - m) log2(e) overflows there, which the kernels must treat like -inf)."""
    c = make_case(name, seed=seed, rows=rows)
    raw = c.raw.copy()
    V = raw.shape[1]
    rng = np.random.default_rng(seed + 100)
    if fill == "-inf":
        ninf = np.uint16(0xFF80) if c.w.dtype == "bf16" else np.float32(-np.inf)
    else:
        ninf = np.uint16(0xFF7F) if c.w.dtype == "bf16" else np.float32(-np.finfo(np.float32).max)
    for r in range(0, c.rows, 2):
        cols = rng.random(V) < 0.3
        cols[c.ids[r]] = False
        raw[r, cols] = ninf
    r = 1
    cols = np.ones(V, bool)
    cols[[c.ids[r], (c.ids[r] + 1) % V, (c.ids[r] + 7) % V]] = False
    raw[r, cols] = ninf
    logp, _, _ = O.token_logprobs(raw, c.w.dtype, c.ids)
    old = W.old_logp_from(logp, c.w, seed, c.row0)
    ref = W.ref_logp_from(logp, c.w, seed, c.row0) if c.w.ref_noise_std else None
    P = dataclasses.replace(c.P, entropy_coef=1e-2) if entropy else c.P
    return dataclasses.replace(c, raw=raw, old=old, ref=ref, P=P)


@pytest.mark.parametrize("name,entropy,fill", [("longhorizon", False, "-inf"), ("multiturn", True, "-inf"),
                                               ("edge", True, "-inf"), ("multiturn", False, "-inf"),
                                               ("longhorizon", True, "max_finite"), ("edge", True, "max_finite"),
                                               ("tiny", True, "-inf"), ("tiny", False, "max_finite")])
def test_policy_loss_neg_inf_logits(R, name, entropy, fill):
    case = neg_inf_case(name, 64, entropy=entropy, fill=fill)
    out = run_loss(R, case)
    compare(case, out, f"{name} {fill} entries, entropy={entropy}")
    assert np.isfinite(out["grad"]).all()


@pytest.mark.parametrize("name,fill", [("multiturn", "-inf"), ("edge", "-inf"), ("multiturn", "max_finite")])
def test_token_logprobs_neg_inf_logits(R, name, fill):
    case = neg_inf_case(name, 48, fill=fill)
    V = case.raw.shape[1]
    ws = R.new_workspace(case.rows, V)
    logp, H, lse = R.rl_token_logprobs(logits_to_dev(case), to_dev(case.ids), ws, want_entropy=True, want_lse=True)
    assert R.rl_query_status(ws)[1] == 0
    lp_ref, H_ref, lse_ref = O.token_logprobs(case.raw, case.w.dtype, case.ids)
    lp, Hd, ls = (x.cpu().numpy().astype(np.float64) for x in (logp, H, lse))
    assert np.all(np.abs(lp - lp_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lp_ref)), np.abs(lp - lp_ref).max()
    assert np.all(np.abs(ls - lse_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lse_ref)), np.abs(ls - lse_ref).max()
    assert np.all(np.abs(Hd - H_ref) <= 5e-5 + 2e-5 * np.abs(H_ref)), np.abs(Hd - H_ref).max()



# ----------------------------------------------------------------------------- NaN logits, batch summaries

def test_nan_logits_stay_in_their_rows(R):
    """A NaN logit makes its own row's loss term and gradient NaN and nothing else: every other
    row matches the oracle, and the loss (a sum over rows) is NaN."""
    case = make_case("multiturn", seed=8, row0=2000, rows=40)
    raw = case.raw.copy()
    bad = [int(r) for r in np.nonzero((case.mask != 0) & (case.coef64[case.tt] != 0))[0][:3]]
    for r in bad:
        raw[r, (case.ids[r] + 11) % raw.shape[1]] = np.uint16(0x7FC0)  # bf16 NaN
    c2 = dataclasses.replace(case, raw=raw)
    out = run_loss(R, c2)
    assert np.isnan(out["loss"])
    ok = np.ones(case.rows, bool)
    ok[bad] = False
    assert np.isnan(out["grad"][bad]).any(axis=1).all()
    adv32 = case.adv64.astype(np.float32).astype(np.float64)
    coef32 = case.coef64.astype(np.float32).astype(np.float64)
    rows = np.nonzero(ok)[0]
    _, g_ref, st_ref, _ = O.policy_loss_fwd_bwd(case.raw, case.w.dtype, case.ids, case.mask, case.tt, adv32, coef32,
                                                case.old, case.P, case.ref, case.roll, rows=rows)
    check_grad(out["grad"][rows], g_ref, case.w.dtype, "rows without NaN")


@pytest.mark.parametrize("rows", [1, 8191, 8193, 77881, 155959])
def test_stats_summary_sizes(R, rows):
    """The summary over batches that span the cluster's 8,192 threads several times with a
    ragged tail (and the multi-turn batch's size): counts exact, sums within 1e-12 of the float64
    sums of the same float32 values, and the same bits on a second call."""
    rng = np.random.default_rng(rows)
    n_traj = 97
    stats = rng.random((rows, 5), dtype=np.float32)
    stats[:, 2] = (rng.random(rows) < 0.1).astype(np.float32)  # clipped flags
    mask = (rng.random(rows) < 0.6).astype(np.uint8)
    tt = rng.integers(0, n_traj, rows).astype(np.int32)
    coef = rng.random(n_traj).astype(np.float32)
    coef[::7] = 0.0
    ws = R.new_workspace(0, 0)
    args = (torch.from_numpy(stats.reshape(-1)).cuda(), to_dev(mask), to_dev(tt), to_dev(coef), ws)
    a = R.rl_token_stats_summary(*args).cpu().numpy()
    b = R.rl_token_stats_summary(*args).cpu().numpy()
    assert R.rl_query_status(ws)[1] == 0
    ref = O.stats_summary(stats.astype(np.float64), mask, tt, coef)
    assert a[0] == ref[0] and a[1] == ref[1]
    assert np.allclose(a[2:], ref[2:], rtol=1e-12, atol=1e-12)
    assert np.array_equal(a, b)


def test_stats_summary(R):
    """Summaries of the loss call's statistics: counts exact, sums equal the float64 sum of the
    same float32 values (order-independent to 1e-12), and within the statistics' own tolerances
    of the oracle's summary."""
    case = make_case("longhorizon", seed=9, row0=3000, rows=96, tis=True)
    out = run_loss(R, case)
    st_dev = torch.from_numpy(out["stats"].reshape(-1).astype(np.float32)).cuda()
    coef32 = case.coef64.astype(np.float32)
    ws = R.new_workspace(0, 0)
    acc = R.rl_token_stats_summary(st_dev, to_dev(case.mask), to_dev(case.tt.astype(np.int32)), to_dev(coef32), ws)
    acc = R.rl_token_stats_summary(st_dev, to_dev(case.mask), to_dev(case.tt.astype(np.int32)), to_dev(coef32), ws,
                                   summary_accum=acc)  # accumulates
    assert R.rl_query_status(ws)[1] == 0
    got = acc.cpu().numpy() / 2
    mine = O.stats_summary(out["stats"].astype(np.float64), case.mask, case.tt, coef32)
    assert got[0] == mine[0] and got[1] == mine[1]
    assert np.allclose(got[2:], mine[2:], rtol=1e-12, atol=1e-12)
    _, _, st_ref, _ = oracle_loss(case, case.adv64.astype(np.float32).astype(np.float64),
                                  coef32.astype(np.float64), want_grad=False)
    ref = O.stats_summary(st_ref, case.mask, case.tt, coef32)
    assert got[0] == ref[0] and got[1] == ref[1]
    act = (case.mask != 0) & (coef32[case.tt] != 0)
    tolH = float((5e-5 + 2e-5 * np.abs(st_ref[act, 3])).sum())
    assert abs(got[2] - ref[2]) <= tolH and abs(got[4] - ref[4]) <= float((2e-5 * st_ref[act, 1]).sum())
