"""Planted mistakes in the oracle must be caught by the pins.

Each mutant is the oracle's source with one plausible error planted (a dropped
term, a wrong sign, index or bound, a transposed operand, a sample instead of a
population statistic). The mutated module is built on the CPU, in memory, and
every pin of ``oracle_pins.py`` is run against it: at least one must fail.
"""

import inspect
import sys
import types

import pytest

import oracle.grpo_objective as O
from oracle_pins import ALL_PINS

SRC = inspect.getsource(O)

MUTANTS = {
    "sample std": ("math.fsum((r - mu) ** 2 for r in R) / k)", "math.fsum((r - mu) ** 2 for r in R) / (k - 1))"),
    "eps inside sqrt": ("math.sqrt(math.fsum((r - mu) ** 2 for r in R) / k)",
                        "math.sqrt(math.fsum((r - mu) ** 2 for r in R) / k + adv_eps)"),
    "mean over group size": ("mu = math.fsum(R) / k", "mu = math.fsum(R) / (k + 1)"),
    "invalid kept in stats": ("if valid[i]]", "if True]"),
    "empty trajectories counted": ("counted = valid & (L > 0)", "counted = valid"),
    "token-mean over all": ("c[counted] = 1.0 / float(L[counted].sum())", "c[counted] = 1.0 / float(L.sum())"),
    "seq-mean uses n": ("c[counted] = 1.0 / (N * L[counted].astype(np.float64))",
                        "c[counted] = 1.0 / (n * L[counted].astype(np.float64))"),
    "count off by one span": ("L[i] = int(np.count_nonzero(mask[s:e]))", "L[i] = int(np.count_nonzero(mask[s:e + 1]))"),
    "lse without max": ("lse = m + np.log(s)", "lse = np.log(s)"),
    "entropy sign": ("H = -np.where(p > 0, p * logp_all, 0.0).sum(axis=1)",
                     "H = np.where(p > 0, p * logp_all, 0.0).sum(axis=1)"),
    "entropy 0 log 0 not 0": ("H = -np.where(p > 0, p * logp_all, 0.0).sum(axis=1)",
                              "H = -(p * logp_all).sum(axis=1)"),
    "gather wrong index": ("z_a = z[rows, a]", "z_a = z[rows, (a + 1) % z.shape[1]]"),
    "ratio inverted": ("log_ratio = (z_a - old) - lse", "log_ratio = (old - z_a) + lse"),
    "symmetric clip": ("clipped_rho = np.minimum(np.maximum(rho, 1.0 - el), 1.0 + eh)",
                       "clipped_rho = np.minimum(np.maximum(rho, 1.0 - el), 1.0 + el)"),
    "max instead of min": ("surr = np.minimum(rho * A, clipped_rho * A)", "surr = np.maximum(rho * A, clipped_rho * A)"),
    "wrong cut side": ("cut = ((A > 0) & (rho > 1.0 + eh)) | ((A < 0) & (rho < 1.0 - el))",
                       "cut = ((A > 0) & (rho < 1.0 - el)) | ((A < 0) & (rho > 1.0 + eh))"),
    "non-strict cut": ("cut = ((A > 0) & (rho > 1.0 + eh))", "cut = ((A > 0) & (rho >= 1.0 + eh))"),
    "tis max": ("w = np.minimum(np.exp(old - np.asarray(rollout_logp, dtype=np.float64)), params.tis_cap)",
                "w = np.maximum(np.exp(old - np.asarray(rollout_logp, dtype=np.float64)), params.tis_cap)"),
    "tis inverted": ("np.exp(old - np.asarray(rollout_logp, dtype=np.float64))",
                     "np.exp(np.asarray(rollout_logp, dtype=np.float64) - old)"),
    "kl k1 instead of k3": ("kl = ed - d - 1.0", "kl = -d"),
    "kl grad sign": ("dkl = 1.0 - ed", "dkl = ed - 1.0"),
    "entropy bonus sign": ("ell = -w * surr + beta * kl - alpha", "ell = -w * surr + beta * kl + alpha"),
    "objective not negated": ("ell = -w * surr", "ell = w * surr"),
    "grad without tis weight": ("g = -w * A * rho * act", "g = -A * rho * act"),
    "grad without ratio": ("g = -w * A * rho * act", "g = -w * A * act"),
    "dropped entropy grad term": ("gz += np.where(p > 0, alpha * p * (z - lse[:, None] + H[:, None]), 0.0)",
                                  "gz += np.where(p > 0, alpha * p * (z - lse[:, None]), 0.0)"),
    "entropy grad at -inf entries": ("gz += np.where(p > 0, alpha * p * (z - lse[:, None] + H[:, None]), 0.0)",
                                     "gz += alpha * p * (z - lse[:, None] + H[:, None])"),
    "dropped softmax grad term": ('gz = -tt["g"][:, None] * p', 'gz = 0.0 * p'),
    "masked rows kept": ("active = (mask[sel] != 0) & (c_row != 0.0)", "active = (c_row != 0.0)"),
    "loss not weighted": ('contrib[loc] = c * tt["ell"]', 'contrib[loc] = tt["ell"]'),
    "grad not weighted": ("grad[loc] = c[:, None] * gz", "grad[loc] = gz"),
    "head dW transposed": ("d_weight = dZ.T @ Hm", "d_weight = (dZ.T @ Hm).T"),
    "head dH uses W^T": ("d_hidden = dZ @ Wm", "d_hidden = dZ @ Wm.T"),
    "head logits transposed": ("Z = Hm @ Wm.T", "Z = (Hm @ Wm.T).T"),
    "token-level adv ignored": ("A_row = adv[sel] if params.token_level_adv else adv[token_traj[sel]]",
                                "A_row = adv[token_traj[sel]]"),
    "seq weight includes masked tokens": ("S[i] = math.fsum(d[(tt == i) & M].tolist())",
                                          "S[i] = math.fsum(d[tt == i].tolist())"),
    "seq weight inverted ratio": ("d = np.asarray(old_logp, dtype=np.float64) - np.asarray(rollout_logp, dtype=np.float64)",
                                  "d = np.asarray(rollout_logp, dtype=np.float64) - np.asarray(old_logp, dtype=np.float64)"),
    "seq weight cap as max": ("w = np.minimum(w, cap)", "w = np.maximum(w, cap)"),
    "summary counts masked tokens": ("act = (np.asarray(mask) != 0) & (c != 0)", "act = c != 0"),
    "summary sums the wrong column": ("math.fsum(st[act, STAT_ENTROPY])", "math.fsum(st[act, STAT_LOGP])"),
    "head logprobs chunk offset": ("Z = Hm[r0:r0 + chunk] @ Wm.T", "Z = Hm[r0 + 1:r0 + 1 + chunk] @ Wm.T"),
    "bf16 decode shifted by 15": ("<< np.uint32(16)", "<< np.uint32(15)"),
    "bf16 decoded as fp16": ("return bits.view(np.float32).astype(np.float64)",
                             "return np.asarray(raw, dtype=np.uint16).view(np.float16).astype(np.float64)"),
}


def _mutant(old, new):
    assert SRC.count(old) >= 1, f"snippet not in oracle: {old}"
    src = SRC.replace(old, new, 1)
    mod = types.ModuleType("oracle_mutant")
    mod.__file__ = O.__file__
    sys.modules["oracle_mutant"] = mod  # dataclasses resolve their module through sys.modules
    try:
        exec(compile(src, "<oracle mutant>", "exec"), mod.__dict__)
    finally:
        del sys.modules["oracle_mutant"]
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name):
    mod = _mutant(*MUTANTS[name])
    failed = []
    for pin in ALL_PINS:
        try:
            pin(mod)
        except Exception as e:  # an assertion or a crash both count as caught
            failed.append((pin.__name__, type(e).__name__))
    assert failed, f"no pin catches the planted mistake '{name}'"


def test_unmutated_copy_passes_every_pin():
    mod = _mutant("import math", "import math")
    for pin in ALL_PINS:
        pin(mod)
