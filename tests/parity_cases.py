"""Shared helpers for the GPU parity tests: seeded cases from the workload
generators, the oracle's answers, the CUDA path's answers, and the tolerance
checks.

Inputs flow one way: the generators draw logits, ids, masks, rewards and noise;
the oracle computes its own advantages, coefficients and log-probs (old_logp =
oracle logp - noise); the CUDA path receives the same float32 / bf16 arrays.
No value computed by the CUDA path is ever fed to the oracle.

Tolerances (float32 kernels against the float64 oracle):
  loss       |d| <= 1e-4 * max(|L|, sum_t |c l_t|)
  gradient   |d| <= 2e-3 absolute (paper's weighting; not for token-sum, c = 1), and the tighter
             |d| <= fmt * |g| + 2e-5 * |g| + 2e-5 * s_row, s_row = max(max_v |g_row|,
             the row's coefficient size |c| (w |A| rho + beta |1 - e^(r-logp)| + alpha (1 + |H|)))
             with fmt = 2^-8 for bf16 output (half an ulp of an 8-bit significand)
             and 2^-23 for float32 output
  logp       |d| <= 1e-5 + 2^-22 |logp|   (2^-22: float32 ulp at -1e4 rows)
  ratio      |d| <= 2e-5 * rho
  entropy    |d| <= 5e-5 + 2e-5 |H|
  KL         |d| <= 1e-6 + 1e-4 |KL|
  clipped flag, token owners, counts, masked / inactive rows: bit-exact
  fused head: logits formed on the GPU add a per-token allowance zerr to logp, ratio,
             entropy and KL (logit_error_bound)
"""

from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch

import oracle.grpo_objective as O
from paper_2608_16798_gb300 import workloads as W

GRAD_ABS = 2e-3


def loss_params(w: W.Workload, loss_agg=0, tis_cap=0.0):
    return O.LossParams(clip_eps_low=W.CLIP_EPS_LOW, clip_eps_high=W.CLIP_EPS_HIGH, kl_coef=w.kl_coef,
                        kl_estimator=3 if w.kl_coef else 0, entropy_coef=w.entropy_coef, tis_cap=tis_cap,
                        adv_eps=1e-6, loss_agg=loss_agg)


def cuda_params(R, P: O.LossParams):
    return R.make_params(P.clip_eps_low, P.clip_eps_high, P.kl_coef, P.kl_estimator, P.entropy_coef, P.tis_cap,
                         P.adv_eps, P.loss_agg, int(P.token_level_adv))


def gae_error_scale(offs, mask, values, rewards, gamma, lam, skip):
    """S_t = sum_l (gamma lambda)^l |b_{t+l}| with |b_u| = M_u (|r_u| + gamma |V_next(u)| + |V_u|):
    the size of the terms an fp32 evaluation of the GAE recursion adds up (V_next is the next
    token's value in the printed reading, the next trainable token's in the skip reading).
    A scan of depth k rounds each partial sum at most k times, so |error_t| <= k 2^-24 S_t."""
    M = np.asarray(mask) != 0
    V = np.abs(np.asarray(values, dtype=np.float64))
    r = np.abs(np.asarray(rewards, dtype=np.float64))
    S = np.zeros(len(V))
    gl = gamma * lam
    for i in range(len(offs) - 1):
        s, e = int(offs[i]), int(offs[i + 1])
        acc, vn = 0.0, 0.0
        for t in range(e - 1, s - 1, -1):
            if skip:
                if M[t]:
                    acc = r[t] + gamma * vn + V[t] + gl * acc
                    vn = V[t]
            else:
                nb = V[t + 1] if (t + 1 < e and M[t + 1]) else 0.0
                acc = (r[t] + gamma * nb + V[t] if M[t] else 0.0) + gl * acc
            S[t] = acc
    return np.where(M, S, 0.0)


def check_gae(adv_dev, ret_dev, adv_ref, ret_ref, values, S, mask, max_len, what=""):
    """fp32 scan against the float64 oracle: |d adv| <= k 2^-24 S_t + 2^-24 |A_t| with the scan
    depth k = 64 + 2 ceil(L_max / 1024); returns add the rounding of A + V. Masked tokens: exactly 0."""
    u = 2.0 ** -24
    k = 64 + 2 * math.ceil(max(max_len, 1) / 1024)
    M = np.asarray(mask) != 0
    assert np.all(adv_dev[~M] == 0.0) and np.all(ret_dev[~M] == 0.0), f"{what}: masked tokens not zero"
    tol = k * u * S + u * np.abs(adv_ref) + 1e-30
    d = np.abs(adv_dev - adv_ref)
    if np.any(d > tol):
        t = int(np.argmax(d - tol))
        raise AssertionError(f"{what}: adv token {t} gpu {adv_dev[t]} oracle {adv_ref[t]} tol {tol[t]}")
    tol_r = tol + u * (np.abs(adv_ref) + np.abs(np.asarray(values, dtype=np.float64)))
    d = np.abs(ret_dev - ret_ref)
    if np.any(d > tol_r):
        t = int(np.argmax(d - tol_r))
        raise AssertionError(f"{what}: return token {t} gpu {ret_dev[t]} oracle {ret_ref[t]} tol {tol_r[t]}")
    return float((np.abs(adv_dev - adv_ref) / np.maximum(S, 1e-30))[M].max(initial=0.0))


@dataclasses.dataclass
class Case:
    w: W.Workload
    layout: W.Layout
    row0: int
    raw: np.ndarray          # uint16 (bf16 bits) or float32 [rows, V]
    ids: np.ndarray          # int32 [rows]
    old: np.ndarray          # float32 [rows]
    ref: np.ndarray | None
    roll: np.ndarray | None
    P: O.LossParams
    adv64: np.ndarray        # oracle advantages (float64, whole batch)
    coef64: np.ndarray
    L: np.ndarray
    token_traj: np.ndarray   # oracle owners (whole batch)

    @property
    def rows(self):
        return self.raw.shape[0]

    @property
    def sl(self):
        return slice(self.row0, self.row0 + self.rows)

    @property
    def mask(self):
        return self.layout.mask[self.sl]

    @property
    def tt(self):
        return self.token_traj[self.sl]


def make_case(name, seed=0, row0=0, rows=None, vocab=None, n_groups=None, loss_agg=0, tis=False,
              invalid_frac=0.0, logit_std=None):
    w = W.WORKLOADS[name]
    over = {}
    if vocab is not None:
        over["vocab"] = vocab
    if logit_std is not None:
        over["logit_std"] = logit_std
    if over:
        w = dataclasses.replace(w, **over)
    layout = W.make_layout(w, seed, n_groups)
    if invalid_frac > 0:
        rng = np.random.default_rng(seed + 77)
        layout.traj_valid = (rng.random(layout.n_traj) >= invalid_frac).astype(np.uint8)
    T = layout.n_tokens
    rows = T - row0 if rows is None else min(rows, T - row0)
    raw, vals = W.logits_rows_np(w, seed, row0, rows)
    ids = W.sample_tokens_np(vals, seed, row0, w)
    logp, _, _ = O.token_logprobs(raw, w.dtype, ids)
    old = W.old_logp_from(logp, w, seed, row0)
    ref = W.ref_logp_from(logp, w, seed, row0) if w.ref_noise_std else None
    roll = W.rollout_logp_from(old, seed, row0=row0) if tis else None
    P = loss_params(w, loss_agg, tis_cap=2.0 if tis else 0.0)
    adv, coef, L, tt = O.advantages_and_coefficients(layout.rewards, layout.group_offsets, layout.traj_offsets,
                                                     layout.mask, layout.traj_valid, P)
    return Case(w, layout, row0, raw, ids, old, ref, roll, P, adv, coef, L, tt)


def oracle_loss(case: Case, adv=None, coef=None, rows=None, want_grad=True):
    adv = case.adv64 if adv is None else adv
    coef = case.coef64 if coef is None else coef
    return O.policy_loss_fwd_bwd(case.raw, case.w.dtype, case.ids, case.mask, case.tt, adv, coef, case.old, case.P,
                                 case.ref, case.roll, want_grad=want_grad, rows=rows)


def to_dev(x, dtype=None, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(device)


def logits_to_dev(case: Case, ld=None, device="cuda"):
    V = case.raw.shape[1]
    ld = V if ld is None else ld
    if case.w.dtype == "bf16":
        host = torch.from_numpy(case.raw.view(np.int16).copy()).view(torch.bfloat16)
    else:
        host = torch.from_numpy(case.raw.copy())
    if ld == V:
        return host.to(device)
    full = torch.full((case.rows, ld), float("nan"), dtype=host.dtype, device=device)
    full[:, :V] = host.to(device)
    return full[:, :V]


def grad_to_np(g):
    if g.dtype == torch.bfloat16:
        return g.float().cpu().numpy().astype(np.float64)
    return g.cpu().numpy().astype(np.float64)


def check_grad(g_dev, g_ref, dtype, what="", row_scale=None, absolute=True):
    """absolute=False for token-sum weighting (c = 1), where gradient elements are O(1) and
    the 2e-3 absolute bound is below half a bf16 ulp; the relative bound still applies."""
    d = np.abs(g_dev - g_ref)
    if absolute:
        assert d.max(initial=0.0) <= GRAD_ABS, f"{what}: max |dgrad| {d.max()} above {GRAD_ABS}"
    fmt = 2.0 ** -8 if dtype == "bf16" else 2.0 ** -23
    rs = np.abs(g_ref).max(axis=1, keepdims=True) if g_ref.size else np.zeros((g_ref.shape[0], 1))
    row_scale = rs if row_scale is None else np.maximum(rs, row_scale)
    tol = (fmt + 2e-5) * np.abs(g_ref) + 2e-5 * row_scale + 1e-30
    if g_ref.size:
        # relative to the row's scale (its largest element, or the coefficient size when the
        # exact row is 0, e.g. V = 1)
        rel = d.max(axis=1, keepdims=True) / np.maximum(row_scale, 1e-30)
        print(f"{what}: max per-row relative error {float(rel.max()):.3e}, "
              f"max error / bound {float((d / tol).max()):.3f}")
    bad = d > tol
    if bad.any():
        r, v = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} elements out of tolerance; first row {r} col {v}: "
                             f"gpu {g_dev[r, v]!r} oracle {g_ref[r, v]!r} tol {tol[r, v]!r}")


def check_loss(loss_dev, loss_ref, contrib_ref, what=""):
    scale = max(abs(loss_ref), float(np.abs(contrib_ref).sum()))
    assert abs(loss_dev - loss_ref) <= 1e-4 * scale + 1e-300, f"{what}: loss {loss_dev} vs {loss_ref} (scale {scale})"


def logit_error_bound(hidden_f64, weight_f64):
    """Per-token bound on the error of logits the GPU forms itself (fused head): z = h . w
    accumulated in fp32 over D products has partial sums bounded by |h| |w| (Cauchy-Schwarz)
    and roundings of at most 2^-24 of them that add like a random walk over D terms, so
    |dz| <= 2^-24 sqrt(D) |h_t| max_v |w_v|; logp = z_a - lse carries two such errors."""
    D = hidden_f64.shape[1]
    wmax = np.sqrt((weight_f64 ** 2).sum(axis=1)).max()
    return 2 * 2.0 ** -24 * np.sqrt(D) * np.sqrt((hidden_f64 ** 2).sum(axis=1)) * wmax


def check_stats(st_dev, st_ref, active, what="", zerr=None):
    """zerr (per row, optional): error allowance of logits formed on the GPU (see logit_error_bound)."""
    st_dev = st_dev.astype(np.float64)
    assert np.all(st_dev[~active] == 0.0), f"{what}: stats of inactive rows not zero"
    a, b = st_dev[active], st_ref[active]
    z = np.zeros(len(a)) if zerr is None else np.broadcast_to(zerr, active.shape)[active]
    d = np.abs(a - b)
    assert np.all(d[:, 0] <= 1e-5 + 2.0 ** -22 * np.abs(b[:, 0]) + z), f"{what}: logp max diff {d[:, 0].max()}"
    assert np.all(d[:, 1] <= (2e-5 + z) * np.abs(b[:, 1])), f"{what}: ratio max rel diff {(d[:, 1] / b[:, 1]).max()}"
    assert np.array_equal(a[:, 2], b[:, 2]), f"{what}: clipped flags differ"
    assert np.all(d[:, 3] <= 5e-5 + 2e-5 * np.abs(b[:, 3]) + 2 * z), f"{what}: entropy max diff {d[:, 3].max()}"
    assert np.all(d[:, 4] <= 1e-6 + 1e-4 * np.abs(b[:, 4]) + 2 * z * (1 + np.abs(b[:, 4]))), \
        f"{what}: KL max diff {d[:, 4].max()}"


# ----------------------------------------------------------------------------- the loss call and its comparison

def run_loss(R, case, adv32=None, coef32=None, ld=None, in_place=False, stats=True, ws=None):
    dev = "cuda"
    logits = logits_to_dev(case, ld)
    adv32 = case.adv64.astype(np.float32) if adv32 is None else adv32
    coef32 = case.coef64.astype(np.float32) if coef32 is None else coef32
    ws = R.new_workspace(case.rows, case.raw.shape[1]) if ws is None else ws
    loss = torch.zeros(1, dtype=torch.float64, device=dev)
    st = torch.full((case.rows * 5,), float("nan"), dtype=torch.float32, device=dev) if stats else None
    # the gradient buffer starts as NaN everywhere (padding columns included): an element the
    # library should write and does not stays NaN and fails the comparison
    poison = torch.full_like(logits, float("nan")) if logits.is_contiguous() else None
    if not in_place and poison is None:
        full = torch.full((case.rows, logits.stride(0)), float("nan"), dtype=logits.dtype, device=dev)
        poison = full[:, :logits.shape[1]]
    g = R.rl_policy_loss_fwd_bwd(logits, to_dev(case.ids), to_dev(case.mask), to_dev(case.tt.astype(np.int32)),
                                 to_dev(adv32), to_dev(coef32), to_dev(case.old), cuda_params(R, case.P), ws, loss,
                                 grad_out=logits if in_place else poison,
                                 ref_logp=None if case.ref is None else to_dev(case.ref),
                                 rollout_logp=None if case.roll is None else to_dev(case.roll), token_stats=st)
    status, word = R.rl_query_status(ws)
    if not in_place and not logits.is_contiguous():  # columns past V are never written
        assert torch.isnan(full[:, logits.shape[1]:]).all()
    return dict(loss=float(loss.item()), grad=grad_to_np(g), stats=None if st is None else st.view(-1, 5).cpu().numpy(),
                status=status, word=word)


def grad_scale(case, stats, adv, coef):
    """Per-row size of the gradient's coefficients |c| (w |A| rho + beta |1 - e^(r - logp)| + alpha (1 + |H|)),
    the scale of the float32 rounding in a row (used only as an error floor)."""
    c = np.abs(coef[case.tt])
    A = np.abs(adv[case.tt])
    rho, H, logp = stats[:, 1], stats[:, 3], stats[:, 0]
    w = np.ones_like(rho)
    if case.roll is not None and case.P.tis_cap > 0:
        w = np.minimum(np.exp(case.old.astype(np.float64) - case.roll), case.P.tis_cap)
    kl = 0.0
    if case.ref is not None and case.P.kl_coef:
        kl = case.P.kl_coef * np.abs(1 - np.exp(np.clip(case.ref - logp, -50, 50)))
    return (c * (w * A * rho + kl + case.P.entropy_coef * (1 + np.abs(H))))[:, None]


def compare(case, out, what):
    adv32 = case.adv64.astype(np.float32).astype(np.float64)
    coef32 = case.coef64.astype(np.float32).astype(np.float64)
    loss, grad, stats, contrib = oracle_loss(case, adv32, coef32)
    check_loss(out["loss"], loss, contrib, what)
    check_grad(out["grad"], grad, case.w.dtype, what, row_scale=grad_scale(case, stats, adv32, coef32),
               absolute=case.P.loss_agg != O.AGG_TOKEN_SUM)
    active = (case.mask != 0) & (coef32[case.tt] != 0)
    assert np.all(out["grad"][~active] == 0.0), f"{what}: inactive rows not exactly zero"
    if out["stats"] is not None:
        check_stats(out["stats"], stats, active, what)
    assert out["word"] == 0, f"{what}: device status {out['word']}"
