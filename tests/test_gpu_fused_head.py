"""Fused LM head (logits = hidden @ W^T never materialised) against the float64 oracle.

The library keeps exp(z - m_j) of each 256-wide tile in bf16 between its tensor-core pass
and the formation of dZ, and rounds dZ itself to bf16 before the two products dH = dZ W and
dW = dZ^T H: each term of those products carries two independent roundings of at most 2^-8
relative (bf16's unit roundoff; plus, with the entropy bonus, alpha c p 2^-8 from the
logarithm of the rounded value). Rounding errors of independent terms add like a random
walk (standard deviation about 2^-7 / sqrt(3) of the root of the summed squared terms), so
the bound used is 2^-6 * sqrt(sum of squared terms) (computed exactly in float64), about 3.5
standard deviations, plus 1e-4 of the element and 1e-6 of the largest element for the
float32 parts; a bf16 d_hidden adds its own rounding, 2^-8 of the element. Loss, clip flags
and per-token statistics use the logits-path tolerances.
"""

import dataclasses

import numpy as np
import pytest
import torch

import oracle.grpo_objective as O
from parity_cases import check_loss, check_stats, cuda_params, logit_error_bound, to_dev
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


def _bf16_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def make_head_case(T, D, V, seed=0, masked=0.3, agg=0, ent=False, tis=False, wstd=0.05):
    w = dataclasses.replace(W.WORKLOADS["fusedhead"], weight_std=wstd)
    h_bits, w_bits = W.hidden_and_weight_np(w, seed, T, V, D)
    Z = O.decode_logits(h_bits, "bf16") @ O.decode_logits(w_bits, "bf16").T
    rng = np.random.default_rng(seed + 1)
    gumbel = -np.log(-np.log(rng.random(Z.shape)))
    ids = np.argmax(Z + gumbel, axis=1).astype(np.int32)
    lse, logp, H, _, _ = O.row_statistics(Z, ids)
    n_traj = max(4, (T // 50) // 4 * 4)
    cuts = np.sort(rng.choice(np.arange(1, T), size=n_traj - 1, replace=False))
    offs = np.concatenate([[0], cuts, [T]]).astype(np.int64)
    mask = (rng.random(T) >= masked).astype(np.uint8)
    rewards = (rng.random(n_traj) < 0.4).astype(np.float32)
    go = np.arange(0, n_traj + 1, 4, dtype=np.int32)
    P = O.LossParams(entropy_coef=1e-2 if ent else 0.0, kl_coef=2e-2 if ent else 0.0, kl_estimator=3 if ent else 0,
                     tis_cap=2.0 if tis else 0.0, loss_agg=agg)
    adv, coef, L, tt = O.advantages_and_coefficients(rewards, go, offs, mask, None, P)
    delta = rng.uniform(-0.5, 0.5, size=T)
    for b in (np.log(0.8), np.log(1.28)):
        delta = np.where(np.abs(delta - b) < 1e-3, delta + 3e-3, delta)
    old = (logp - delta).astype(np.float32)
    ref = (logp + rng.normal(0, 0.2, size=T)).astype(np.float32) if ent else None
    roll = (old + rng.normal(0, 0.3, size=T)).astype(np.float32) if tis else None
    return dict(h=h_bits, w=w_bits, ids=ids, mask=mask, tt=tt, adv32=adv.astype(np.float32),
                coef32=coef.astype(np.float32), old=old, ref=ref, roll=roll, P=P, T=T, D=D, V=V)


def run_head(R, c, dh_dtype=torch.float32, group_tokens=0):
    T, D, V = c["T"], c["D"], c["V"]
    ws = R.new_workspace(T, V, D, group_tokens=group_tokens)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    dW = torch.zeros((V, D), dtype=torch.float32, device="cuda")
    st = torch.zeros(T * 5, dtype=torch.float32, device="cuda")
    dH = R.rl_fused_head_loss_fwd_bwd(_bf16_dev(c["h"]), _bf16_dev(c["w"]), to_dev(c["ids"]), to_dev(c["mask"]),
                                      to_dev(c["tt"].astype(np.int32)), to_dev(c["adv32"]), to_dev(c["coef32"]),
                                      to_dev(c["old"]), cuda_params(R, c["P"]), ws, loss, dW,
                                      d_hidden_dtype=dh_dtype,
                                      ref_logp=None if c["ref"] is None else to_dev(c["ref"]),
                                      rollout_logp=None if c["roll"] is None else to_dev(c["roll"]), token_stats=st)
    status, word = R.rl_query_status(ws)
    return dict(loss=loss.item(), dH=dH.float().cpu().numpy().astype(np.float64),
                dW=dW.cpu().numpy().astype(np.float64), stats=st.view(-1, 5).cpu().numpy(), word=word)


def check_product(got, ref, S, what):
    tol = 2.0 ** -6 * S + 1e-4 * np.abs(ref) + 1e-6 * np.abs(ref).max() + 1e-30
    print(f"{what}: max error / bound = {float((np.abs(got - ref) / tol).max()):.3f}")
    bad = np.abs(got - ref) > tol
    if bad.any():
        i, j = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} elements out of tolerance, e.g. [{i},{j}] "
                             f"gpu {got[i, j]} oracle {ref[i, j]} tol {tol[i, j]}")


def compare_head(c, out, dh_bf16=False):
    P = c["P"]
    adv, coef = c["adv32"].astype(np.float64), c["coef32"].astype(np.float64)
    loss, dH, dW, stats = O.fused_head_loss_fwd_bwd(c["h"], c["w"], c["ids"], c["mask"], c["tt"], adv, coef, c["old"],
                                                    P, c["ref"], c["roll"])
    Hm, Wm = O.decode_logits(c["h"], "bf16"), O.decode_logits(c["w"], "bf16")
    Z = Hm @ Wm.T
    _, dZ, _, contrib = O.policy_loss_fwd_bwd(Z, "f64", c["ids"], c["mask"], c["tt"], adv, coef, c["old"], P, c["ref"],
                                              c["roll"])
    check_loss(out["loss"], loss, contrib, "fused head loss")
    active = (c["mask"] != 0) & (coef[c["tt"]] != 0)
    Hm, Wm = O.decode_logits(c["h"], "bf16"), O.decode_logits(c["w"], "bf16")
    check_stats(out["stats"], stats, active, "fused head stats", zerr=logit_error_bound(Hm, Wm))
    S_h = np.sqrt((dZ ** 2) @ (Wm ** 2))
    S_w = np.sqrt((dZ.T ** 2) @ (Hm ** 2))
    if dh_bf16:
        S_h = S_h + np.abs(dH) / 4  # 2^-6 |dH| / 4 = 2^-8 |dH|: the bf16 output's rounding
    check_product(out["dH"], dH, S_h, "d_hidden")
    check_product(out["dW"], dW, S_w, "d_weight")
    assert np.all(out["dH"][~active] == 0.0), "tokens that are not trained on must get zero d_hidden rows"
    assert out["word"] == 0


@pytest.mark.parametrize("T,D,V,agg,ent,tis", [
    (300, 256, 1000, 2, False, False),     # ragged M tile and vocabulary tile
    (256, 128, 8292, 0, False, False),     # three vocabulary blocks
    (200, 192, 700, 2, True, False),       # entropy + k3 KL
    (130, 64, 513, 1, False, True),        # TIS, token-mean, smallest D
    (260, 128, 2000, 0, True, True),       # entropy + k3 KL + TIS together
    (100, 128, 777, 0, True, False),       # one CTA pair whose odd CTA's 128 tokens all lie past T
    (5, 64, 300, 2, False, False),         # a handful of tokens
    (40, 64, 524_288, 2, False, False),    # the largest vocabulary (128 blocks of 4,096)
    (8, 65_536, 256, 0, True, False),      # the largest hidden size (1,024 K slices per tile)
])
def test_fused_head_parity(R, T, D, V, agg, ent, tis):
    c = make_head_case(T, D, V, seed=T + V, agg=agg, ent=ent, tis=tis)
    out = run_head(R, c)
    compare_head(c, out)


@pytest.mark.parametrize("group_tokens", [0, 6000, 3 * 4096])
def test_fused_head_three_chunks_bf16_grad(R, group_tokens):
    """More than 8,192 tokens, bf16 d_hidden. With the smallest workspace each chunk of 4,096 is
    its own group and dW is added three times; with room for two chunks (6,000 tokens round up
    to two) the groups are two chunks and a ragged last one; with room for three the group
    holds them all and dW is added once."""
    c = make_head_case(8192 + 77, 128, 1100, seed=5, agg=2)
    out = run_head(R, c, dh_dtype=torch.bfloat16, group_tokens=group_tokens)
    compare_head(c, out, dh_bf16=True)


@pytest.mark.parametrize("group_tokens", [0, 32768])
def test_fused_head_ten_chunks(R, group_tokens):
    """More than 32,768 tokens: ten chunks, each its own group (the smallest workspace: dW
    added ten times), or a full group of eight and a ragged second group of two (dH stored in
    fp32 over 32,768 tokens, the second group's dW added onto the first's)."""
    c = make_head_case(32768 + 4096 + 50, 64, 600, seed=11, agg=0, ent=True)
    out = run_head(R, c, group_tokens=group_tokens)
    compare_head(c, out)


def test_fused_head_deterministic_and_workspace_independent(R):
    """Two calls give the same bits (dH's split halves and dW's per-chunk additions land in a
    fixed order); the smallest and a grouped workspace give the same loss and statistics bit
    for bit (the products group their sums differently, so those are held to the oracle)."""
    c = make_head_case(4096 + 300, 128, 2000, seed=8, agg=0)
    a = run_head(R, c)
    b = run_head(R, c)
    g = run_head(R, c, group_tokens=8192)
    for k in ("loss", "dH", "dW", "stats"):
        assert np.array_equal(a[k], b[k]), k
    for k in ("loss", "stats"):
        assert np.array_equal(a[k], g[k]), k
    compare_head(c, g)


def test_fused_head_matches_logits_path(R):
    """The fused head's loss equals rl_policy_loss_fwd_bwd on the materialised fp32 logits."""
    c = make_head_case(384, 256, 2048, seed=9, agg=0)
    out = run_head(R, c)
    Z = torch.from_numpy(O.decode_logits(c["h"], "bf16")) @ torch.from_numpy(O.decode_logits(c["w"], "bf16")).T
    z32 = Z.float().cuda()
    ws = R.new_workspace(c["T"], c["V"])
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    R.rl_policy_loss_fwd_bwd(z32, to_dev(c["ids"]), to_dev(c["mask"]), to_dev(c["tt"].astype(np.int32)),
                             to_dev(c["adv32"]), to_dev(c["coef32"]), to_dev(c["old"]), cuda_params(R, c["P"]), ws,
                             loss)
    assert abs(loss.item() - out["loss"]) <= 1e-4 * max(abs(loss.item()), 1e-12)


def test_fused_head_token_level_adv(R):
    """Per-token advantages (PPO, Sec. 2.3.1) through the fused head, token-mean weights."""
    c = make_head_case(300, 128, 1000, seed=21, agg=1)
    c["adv32"] = np.random.default_rng(22).normal(0, 1, c["T"]).astype(np.float32)
    c["P"] = dataclasses.replace(c["P"], token_level_adv=True)
    out = run_head(R, c)
    compare_head(c, out)


def check_logprobs(c, logp, H, lse, what):
    """Forward-only outputs against the oracle, with the logit allowance zerr per token."""
    ref_logp, ref_H, ref_lse = O.fused_head_logprobs(c["h"], c["w"], c["ids"])
    zerr = logit_error_bound(O.decode_logits(c["h"], "bf16"), O.decode_logits(c["w"], "bf16"))
    d = np.abs(logp - ref_logp)
    assert np.all(d <= 1e-5 + 2.0 ** -22 * np.abs(ref_logp) + zerr), f"{what}: logp max diff {d.max()}"
    d = np.abs(lse - ref_lse)
    assert np.all(d <= 1e-5 + 2.0 ** -22 * np.abs(ref_lse) + zerr), f"{what}: lse max diff {d.max()}"
    if H is not None:
        d = np.abs(H - ref_H)
        assert np.all(d <= 5e-5 + 2e-5 * np.abs(ref_H) + 2 * zerr), f"{what}: entropy max diff {d.max()}"


def run_logprobs(R, c, want_entropy=True, ids=None):
    T, V, D = c["T"], c["V"], c["D"]
    ws = R.new_workspace(T, V, D)
    logp, H, lse = R.rl_fused_head_token_logprobs(_bf16_dev(c["h"]), _bf16_dev(c["w"]),
                                                  to_dev(c["ids"] if ids is None else ids), ws,
                                                  want_entropy=want_entropy, want_lse=True)
    word = R.rl_query_status(ws)[1]
    f = lambda x: None if x is None else x.cpu().numpy().astype(np.float64)
    return f(logp), f(H), f(lse), word


@pytest.mark.parametrize("T,D,V", [
    (300, 256, 1000),        # ragged M tile and vocabulary tile
    (256, 128, 8292),        # three vocabulary blocks, ragged last block
    (130, 64, 513),          # smallest D
    (64, 64, 1000),          # the odd CTA of the only pair has no tokens
    (8192 + 77, 128, 1100),  # three chunks
])
def test_fused_head_logprobs_parity(R, T, D, V):
    c = make_head_case(T, D, V, seed=3 * T + V)
    logp, H, lse, word = run_logprobs(R, c)
    assert word == 0
    check_logprobs(c, logp, H, lse, f"fused logprobs {T}x{D}x{V}")


def test_fused_head_logprobs_without_entropy_and_bad_ids(R):
    """entropy_out NULL skips the entropy work and leaves logp and lse unchanged (bit for bit);
    an id outside [0, V) gives NaN for its token only and sets RL_DEV_BAD_TOKEN."""
    c = make_head_case(260, 128, 900, seed=4)
    logp_e, _, lse_e, _ = run_logprobs(R, c, want_entropy=True)
    logp, H, lse, word = run_logprobs(R, c, want_entropy=False)
    assert H is None and word == 0
    assert np.array_equal(logp, logp_e) and np.array_equal(lse, lse_e)
    bad = c["ids"].copy()
    bad[[5, 200]] = [-1, 900]
    logp_b, _, lse_b, word = run_logprobs(R, c, ids=bad)
    assert word == R.RL_DEV_BAD_TOKEN
    assert np.isnan(logp_b[[5, 200]]).all()
    keep = np.ones(260, bool)
    keep[[5, 200]] = False
    assert np.array_equal(logp_b[keep], logp[keep]) and np.array_equal(lse_b, lse)


def test_fused_head_logprobs_match_loss_pass(R):
    """The forward-only call and the loss call's first pass form the same statistics: logp and
    entropy agree bit for bit with token_stats of rl_fused_head_loss_fwd_bwd on trained tokens."""
    c = make_head_case(384, 192, 3000, seed=11, masked=0.3, ent=True)
    out = run_head(R, c)
    logp, H, _, word = run_logprobs(R, c)
    active = (c["mask"] != 0) & (c["coef32"][c["tt"]] != 0)
    st = out["stats"].astype(np.float64)
    assert np.array_equal(st[active, 0], logp[active])
    assert np.array_equal(st[active, 3], H[active])
