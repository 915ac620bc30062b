"""Seeded synthetic inputs for the policy-loss path.

This module only draws inputs. It holds none of the objective's arithmetic:
no log-softmax, ratio, clipping, advantage or gradient. The CUDA library, the
float64 oracle, the tests and the benchmark all take their inputs from here, and
nothing here imports either side.

The five workloads follow the shapes of the paper's RL batches (groups of 8 and
16 rollouts per task, 32 x 8 task batches, long multi-turn trajectories with
harness / tool-observation spans excluded from training, Qwen3's 151,936-token
vocabulary):

  tiny       1 group x 8 trajectories x 64 tokens, V = 4,096, bf16 N(0, 3^2)
  multiturn  16 groups x 8, lengths U{256..2048}, V = 151,936, bf16 N(0, 2^2),
             ~40% of tokens masked in spans, R ~ Bernoulli(0.3), 16,384-row microbatches
  longhorizon 32 groups x 16, lengths log-uniform [512, 8192], V = 151,936, bf16,
             4 of 32 groups with all-equal rewards, entropy + k3-KL (1e-3 each),
             32,768-row microbatches
  edge       4,096 groups x 4 x 8 tokens, V = 32,000, fp32 N(0, 2^2) with +40 spikes
             and -1e4 rows, log-ratios spread over both clip bounds,
             fully-masked / fully-unmasked / half-masked trajectories
  fusedhead  hidden bf16 [32,768 x 4,096] ~ N(0, 1), W bf16 [151,936 x 4,096] ~ N(0, 0.02^2),
             masks and rewards of the first 32,768 tokens of a multiturn batch

  tree       16 tasks x 8 rollouts of captured model calls (prompt, turns with tool outputs,
             retries, subagent and compaction calls), packed as deduplicated prefix trees

For the PPO path, value predictions V(s_t) are N(0.3, 0.25^2) per token and the
rollout reward R_i of the layout is placed at each trajectory's last trainable token;
sparse per-token rewards can be added.

Quantities that depend on the current policy's log-probability (old_logp,
ref_logp) are formed as ``logp + noise``; the caller supplies ``logp`` from
whichever side it is preparing inputs for, and this module only adds the
seeded noise. Noise is drawn so that the log-ratio never lands within
``RATIO_BAND`` of ln(1 - eps_low) or ln(1 + eps_high): float32 and float64 then
agree on which side of a clip bound every token falls.

bf16 values are carried as uint16 bit patterns on the host (numpy has no bf16).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

RATIO_BAND = 1e-4
CLIP_EPS_LOW = 0.2
CLIP_EPS_HIGH = 0.28


@dataclass(frozen=True)
class Workload:
    name: str
    n_groups: int
    group_size: int
    vocab: int
    dtype: str                 # "bf16" or "f32"
    logit_std: float
    microbatch: int
    lengths: tuple             # ("fixed", L) | ("uniform", lo, hi) | ("loguniform", lo, hi)
    mask_kind: str             # "none" | "spans" | "edge"
    reward_p: float
    old_noise_std: float       # old_logp = logp + N(0, std^2); 0 -> edge log-ratio law
    ref_noise_std: float = 0.0  # > 0 -> ref_logp = logp + N(0, std^2)
    entropy_coef: float = 0.0
    kl_coef: float = 0.0
    equal_groups: int = 0      # groups forced to all-equal rewards (half 0, half 1)
    hidden: int = 0            # fused head only
    weight_std: float = 0.0    # fused head only
    tree_max_leaves: int = 0   # prefix-tree workload only
    extra: dict = field(default_factory=dict)


WORKLOADS = {
    "tiny": Workload("tiny", 1, 8, 4096, "bf16", 3.0, 512, ("fixed", 64), "none", 0.5, 0.05),
    "multiturn": Workload("multiturn", 16, 8, 151936, "bf16", 2.0, 16384, ("uniform", 256, 2048),
                          "spans", 0.3, 0.1),
    "longhorizon": Workload("longhorizon", 32, 16, 151936, "bf16", 2.0, 32768,
                            ("loguniform", 512, 8192), "spans", 0.3, 0.1, ref_noise_std=0.2,
                            entropy_coef=1e-3, kl_coef=1e-3, equal_groups=4),
    "edge": Workload("edge", 4096, 4, 32000, "f32", 2.0, 131072, ("fixed", 8), "edge", 0.5, 0.0),
    "fusedhead": Workload("fusedhead", 16, 8, 151936, "bf16", 0.0, 32768, ("uniform", 256, 2048),
                          "spans", 0.3, 0.1, hidden=4096, weight_std=0.02),
    "tree": Workload("tree", 16, 8, 151936, "bf16", 2.0, 16384, ("calls", 4, 16), "tree", 0.3, 0.1,
                     tree_max_leaves=12),
}

# the order in which the workloads are listed in the project's configuration
WORKLOAD_ORDER = ["tiny", "multiturn", "longhorizon", "edge", "fusedhead", "tree"]


def _rng(seed: int, *stream) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(seed) & 0xFFFFFFFF, *[int(s) for s in stream]]))


def _name_id(name: str) -> int:
    return WORKLOAD_ORDER.index(name) + 1


# ----------------------------------------------------------------------------
# batch layout: trajectories, groups, masks, rewards
# ----------------------------------------------------------------------------

@dataclass
class Layout:
    traj_offsets: np.ndarray   # int64 [n + 1]
    group_offsets: np.ndarray  # int32 [n_groups + 1]
    rewards: np.ndarray        # float32 [n]
    traj_valid: np.ndarray     # uint8 [n]
    mask: np.ndarray           # uint8 [T]

    @property
    def n_traj(self) -> int:
        return len(self.traj_offsets) - 1

    @property
    def n_tokens(self) -> int:
        return int(self.traj_offsets[-1])

    @property
    def n_groups(self) -> int:
        return len(self.group_offsets) - 1

    def token_owner(self) -> np.ndarray:
        """Trajectory index of each packed token (layout bookkeeping, int32)."""
        lengths = np.diff(self.traj_offsets)
        return np.repeat(np.arange(self.n_traj, dtype=np.int32), lengths)


def _lengths(w: Workload, n: int, rng) -> np.ndarray:
    kind = w.lengths[0]
    if kind == "fixed":
        return np.full(n, w.lengths[1], dtype=np.int64)
    if kind == "uniform":
        return rng.integers(w.lengths[1], w.lengths[2] + 1, size=n).astype(np.int64)
    if kind == "loguniform":
        lo, hi = math.log(w.lengths[1]), math.log(w.lengths[2])
        return np.rint(np.exp(rng.uniform(lo, hi, size=n))).astype(np.int64)
    raise ValueError(kind)


def _span_mask(length: int, rng) -> np.ndarray:
    """Alternating trainable / observation spans, the first span trainable.

    Trainable spans ~ U{64..752}, observation spans ~ U{32..512} tokens, which
    masks about 40% of the tokens.
    """
    m = np.empty(length, dtype=np.uint8)
    pos, trainable = 0, True
    while pos < length:
        span = int(rng.integers(64, 753)) if trainable else int(rng.integers(32, 513))
        m[pos:pos + span] = 1 if trainable else 0
        pos += span
        trainable = not trainable
    return m


def make_layout(w: Workload, seed: int = 0, n_groups: int | None = None) -> Layout:
    ng = w.n_groups if n_groups is None else n_groups
    n = ng * w.group_size
    rng = _rng(seed, _name_id(w.name), 1)
    lengths = _lengths(w, n, rng)
    offs = np.zeros(n + 1, dtype=np.int64)
    np.cumsum(lengths, out=offs[1:])
    go = (np.arange(ng + 1, dtype=np.int64) * w.group_size).astype(np.int32)
    rewards = (rng.random(n) < w.reward_p).astype(np.float32)
    if w.equal_groups:
        eq = rng.choice(ng, size=min(w.equal_groups, ng), replace=False)
        for j, g in enumerate(eq):
            rewards[go[g]:go[g + 1]] = 0.0 if j < len(eq) // 2 else 1.0
    T = int(offs[-1])
    if w.mask_kind == "none":
        mask = np.ones(T, dtype=np.uint8)
    elif w.mask_kind == "spans":
        mask = np.concatenate([_span_mask(int(L), rng) for L in lengths]) if n else np.zeros(0, np.uint8)
    elif w.mask_kind == "edge":
        mask = np.empty(T, dtype=np.uint8)
        kind = rng.random(n)
        for i in range(n):
            s, e = offs[i], offs[i + 1]
            if kind[i] < 0.25:
                mask[s:e] = 0
            elif kind[i] < 0.75:
                mask[s:e] = 1
            else:
                mask[s:e] = (rng.random(e - s) < 0.5).astype(np.uint8)
    else:
        raise ValueError(w.mask_kind)
    valid = np.ones(n, dtype=np.uint8)
    return Layout(offs, go, rewards, valid, mask)


def microbatches(layout: Layout, rows_per_mb: int):
    """Row ranges [start, stop) that cut the packed stream into microbatches."""
    T = layout.n_tokens
    return [(s, min(T, s + rows_per_mb)) for s in range(0, T, rows_per_mb)]


# ----------------------------------------------------------------------------
# logits rows (numpy, host) with the edge workload's special rows
# ----------------------------------------------------------------------------

def bf16_bits_from_f32(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest, ties to even) and return the bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


@dataclass
class EdgeRows:
    spike_rows: np.ndarray      # rows with one +40 logit
    spike_cols: np.ndarray
    neg_rows: np.ndarray        # rows with half of the entries at -1e4
    forced_rows: np.ndarray     # subset of neg_rows whose sampled id is forced onto a -1e4 entry


def edge_rows(w: Workload, n_rows: int, seed: int, row0: int = 0) -> EdgeRows:
    """1% of rows get a +40 spike, 1% get half their entries at -1e4 (edge workload)."""
    rng = _rng(seed, _name_id(w.name), 7, row0)
    k = max(1, n_rows // 100) if n_rows >= 4 else 0
    perm = rng.permutation(n_rows)
    spike = np.sort(perm[:k])
    neg = np.sort(perm[k:2 * k])
    forced = np.sort(rng.choice(neg, size=min(len(neg), max(1, round(10 * n_rows / 131072))),
                                replace=False)) if len(neg) else neg
    return EdgeRows(spike, rng.integers(0, w.vocab, size=len(spike)), neg, forced)


def _neg_cols(w: Workload, seed: int, row: int) -> np.ndarray:
    rng = _rng(seed, _name_id(w.name), 8, row)
    return np.sort(rng.permutation(w.vocab)[: w.vocab // 2])


def logits_rows_np(w: Workload, seed: int, row0: int, n_rows: int, vocab: int | None = None):
    """Host logits for rows [row0, row0 + n_rows): uint16 bf16 bits or float32, and a float32 copy.

    Each row is drawn from its own seeded stream, so any row range reproduces the
    same values. Returns (raw, values_f32).
    """
    V = w.vocab if vocab is None else vocab
    vals = np.empty((n_rows, V), dtype=np.float32)
    for r in range(n_rows):
        rng = _rng(seed, _name_id(w.name), 2, row0 + r)
        vals[r] = rng.standard_normal(V, dtype=np.float32) * np.float32(w.logit_std)
    if w.name == "edge":
        ed = edge_rows(w, n_rows, seed, row0)
        for r, c in zip(ed.spike_rows, ed.spike_cols):
            vals[r, c] = 40.0
        for r in ed.neg_rows:
            vals[r, _neg_cols(w, seed, row0 + r)] = -1e4
    if w.dtype == "bf16":
        raw = bf16_bits_from_f32(vals)
        vals = (raw.astype(np.uint32) << np.uint32(16)).view(np.float32)
        return raw, vals
    return vals.copy(), vals


def sample_tokens_np(values_f32: np.ndarray, seed: int, row0: int, w: Workload) -> np.ndarray:
    """Sampled ids: Gumbel-max draws from softmax(z) (the rollout policy's sampling)."""
    n_rows, V = values_f32.shape
    ids = np.empty(n_rows, dtype=np.int32)
    for r in range(n_rows):
        rng = _rng(seed, _name_id(w.name), 3, row0 + r)
        u = rng.random(V)
        gumbel = -np.log(-np.log(np.clip(u, 1e-300, 1.0)))
        ids[r] = int(np.argmax(values_f32[r].astype(np.float64) + gumbel))
    if w.name == "edge":
        ed = edge_rows(w, n_rows, seed, row0)
        for r in ed.forced_rows:
            cols = _neg_cols(w, seed, row0 + r)
            ids[r] = int(cols[_rng(seed, _name_id(w.name), 9, row0 + r).integers(0, len(cols))])
    return ids


# ----------------------------------------------------------------------------
# log-ratio / reference noise
# ----------------------------------------------------------------------------

def _clip_log_bounds(eps_low=CLIP_EPS_LOW, eps_high=CLIP_EPS_HIGH):
    return (math.log(1.0 - eps_low), math.log(1.0 + eps_high))


def logratio_draws(w: Workload, n: int, seed: int, row0: int = 0, stream: int = 4) -> np.ndarray:
    """delta = logp - old_logp for n tokens, away from the clip bounds by RATIO_BAND.

    Gaussian N(0, std^2) for the Gaussian workloads, U[-0.7, 0.7] for the edge
    workload (ratios between 0.50 and 2.01, both bounds crossed often).
    """
    rng = _rng(seed, _name_id(w.name), stream, row0)
    bounds = _clip_log_bounds()
    out = np.empty(n, dtype=np.float64)
    filled = 0
    while filled < n:
        m = n - filled
        d = rng.uniform(-0.7, 0.7, size=m) if w.old_noise_std == 0.0 else rng.normal(0.0, w.old_noise_std, size=m)
        ok = np.ones(m, dtype=bool)
        for b in bounds:
            ok &= np.abs(d - b) > RATIO_BAND
        d = d[ok]
        out[filled:filled + len(d)] = d
        filled += len(d)
    return out


def old_logp_from(logp: np.ndarray, w: Workload, seed: int, row0: int = 0) -> np.ndarray:
    """old_logp = logp - delta as float32, delta from ``logratio_draws``.

    The subtraction is done in float64 and then rounded; the band around each
    clip bound (1e-4 in log space) is far wider than that rounding.
    """
    d = logratio_draws(w, len(logp), seed, row0)
    return (np.asarray(logp, dtype=np.float64) - d).astype(np.float32)


def ref_logp_from(logp: np.ndarray, w: Workload, seed: int, row0: int = 0) -> np.ndarray:
    rng = _rng(seed, _name_id(w.name), 5, row0)
    noise = rng.normal(0.0, w.ref_noise_std, size=len(logp))
    return (np.asarray(logp, dtype=np.float64) + noise).astype(np.float32)


def rollout_logp_from(old_logp: np.ndarray, seed: int, std: float = 0.05, row0: int = 0) -> np.ndarray:
    """Rollout-engine log-probs for TIS tests: old_logp + N(0, std^2)."""
    rng = _rng(seed, 99, 6, row0)
    return (np.asarray(old_logp, dtype=np.float64) + rng.normal(0.0, std, size=len(old_logp))).astype(np.float32)


def tree_rollouts(w: Workload, seed: int = 0, n_rollouts: int | None = None):
    """Captured model calls of black-box rollouts (Sec. 3.2.1), for the prefix-tree path.

    Per rollout: a task prompt of U{200..800} tokens, then U{lo..hi} main-agent turns (the
    workload's ``lengths`` = ("calls", lo, hi)); every turn after the first appends a tool
    output of U{16..512} tokens to the history, and the model answers with U{16..384} tokens.
    The input of each call is the whole history so far, as a serving proxy sees it. With
    probability 0.1 a turn is first attempted and abandoned (a retry: same input, another
    response that nothing continues); with probability 0.05 an auxiliary subagent call branches
    off (history + an instruction of U{8..32} tokens, a response of U{16..128}); with
    probability 0.06 the context is compacted: an auxiliary summariser call (history + an
    instruction, a summary of U{64..256} tokens) and the history restarts as prompt + summary.
    One rollout in 20 runs away with a retry on nearly every turn (more leaves than
    ``tree_max_leaves``). Token ids are uniform on [0, vocab).

    Returns (prompts, calls, aux): lists per rollout; calls are (x, y) int32 arrays."""
    n = w.n_groups * w.group_size if n_rollouts is None else n_rollouts
    lo, hi = w.lengths[1], w.lengths[2]
    prompts, calls, aux = [], [], []
    for r in range(n):
        rng = _rng(seed, _name_id(w.name), 9, r)
        tok = lambda k: rng.integers(0, w.vocab, int(k)).astype(np.int32)  # noqa: E731
        prompt = tok(rng.integers(200, 801))
        runaway = rng.random() < 0.05
        p_retry = 0.9 if runaway else 0.1
        hist = prompt
        cs, ax = [], []
        for turn in range(int(rng.integers(lo, hi + 1))):
            x = hist if turn == 0 else np.concatenate([hist, tok(rng.integers(16, 513))])
            if rng.random() < p_retry:
                cs.append((x, tok(rng.integers(16, 385))))
                ax.append(0)
            y = tok(rng.integers(16, 385))
            cs.append((x, y))
            ax.append(0)
            hist = np.concatenate([x, y])
            if rng.random() < 0.05:
                cs.append((np.concatenate([hist, tok(rng.integers(8, 33))]), tok(rng.integers(16, 129))))
                ax.append(1)
            if rng.random() < 0.06:
                summary = tok(rng.integers(64, 257))
                cs.append((np.concatenate([hist, tok(rng.integers(8, 33))]), summary))
                ax.append(1)
                hist = np.concatenate([prompt, summary])
        prompts.append(prompt)
        calls.append(cs)
        aux.append(ax)
    return prompts, calls, aux


def value_predictions(w: Workload, seed: int, n_tokens: int, mean: float = 0.3, std: float = 0.25) -> np.ndarray:
    """V(s_t) of a value model for the PPO path: N(mean, std^2) per token as float32 (mean at
    the workloads' reward rate 0.3)."""
    rng = _rng(seed, _name_id(w.name), 7)
    return rng.normal(mean, std, size=n_tokens).astype(np.float32)


def token_reward_draws(w: Workload, seed: int, n_tokens: int, frac: float = 0.05, std: float = 0.1) -> np.ndarray:
    """Sparse per-token rewards r_t (a fraction `frac` of tokens, N(0, std^2)) as float32, to
    exercise the per-token reward input of the GAE next to the final-token reward."""
    rng = _rng(seed, _name_id(w.name), 8)
    r = rng.normal(0.0, std, size=n_tokens)
    r[rng.random(n_tokens) >= frac] = 0.0
    return r.astype(np.float32)


# ----------------------------------------------------------------------------
# device-side generation (torch), for the full-size workloads
# ----------------------------------------------------------------------------

def logits_rows_torch(w: Workload, seed: int, row0: int, n_rows: int, out, chunk: int = 2048):
    """Fill ``out`` ([n_rows, >= V] torch tensor of w's dtype, on a CUDA device) with seeded
    N(0, std^2) logits (the edge workload's special rows included). The stream is torch's
    Philox generator keyed by (seed, workload, row0); values differ from ``logits_rows_np``."""
    import torch

    V = w.vocab
    g = torch.Generator(device=out.device)
    for r0 in range(0, n_rows, chunk):
        r1 = min(n_rows, r0 + chunk)
        g.manual_seed((int(seed) * 1_000_003 + _name_id(w.name) * 7919 + row0 + r0) & 0x7FFFFFFFFFFF)
        x = torch.randn((r1 - r0, V), generator=g, device=out.device, dtype=torch.float32)
        x.mul_(w.logit_std)
        out[r0:r1, :V].copy_(x)
    if w.name == "edge":
        ed = edge_rows(w, n_rows, seed, row0)
        for r, c in zip(ed.spike_rows, ed.spike_cols):
            out[int(r), int(c)] = 40.0
        for r in ed.neg_rows:
            cols = torch.from_numpy(_neg_cols(w, seed, row0 + int(r))).to(out.device)
            out[int(r)].index_fill_(0, cols, -1e4)
    return out


def sample_tokens_torch(logits, seed: int, row0: int, w: Workload, chunk: int = 2048):
    """Gumbel-max sampled ids for device logits rows (int32 tensor on the same device)."""
    import torch

    n_rows = logits.shape[0]
    V = w.vocab
    ids = torch.empty(n_rows, dtype=torch.int32, device=logits.device)
    g = torch.Generator(device=logits.device)
    for r0 in range(0, n_rows, chunk):
        r1 = min(n_rows, r0 + chunk)
        g.manual_seed((int(seed) * 2_000_003 + _name_id(w.name) * 104729 + row0 + r0) & 0x7FFFFFFFFFFF)
        u = torch.rand((r1 - r0, V), generator=g, device=logits.device, dtype=torch.float32)
        u.clamp_(min=1e-30).log_().neg_().log_().neg_()       # Gumbel(0, 1)
        u.add_(logits[r0:r1, :V].float())
        ids[r0:r1] = torch.argmax(u, dim=1).to(torch.int32)
    if w.name == "edge":
        ed = edge_rows(w, n_rows, seed, row0)
        for r in ed.forced_rows:
            cols = _neg_cols(w, seed, row0 + int(r))
            ids[int(r)] = int(cols[_rng(seed, _name_id(w.name), 9, row0 + int(r)).integers(0, len(cols))])
    return ids


def hidden_and_weight_torch(w: Workload, seed: int, T: int, out_hidden, out_weight, chunk: int = 8192):
    """Fused-head inputs: hidden ~ N(0, 1), W ~ N(0, weight_std^2), both bf16, on device."""
    import torch

    g = torch.Generator(device=out_hidden.device)
    for r0 in range(0, T, chunk):
        r1 = min(T, r0 + chunk)
        g.manual_seed((int(seed) * 3_000_017 + 11 + r0) & 0x7FFFFFFFFFFF)
        out_hidden[r0:r1].copy_(torch.randn((r1 - r0, w.hidden), generator=g, device=out_hidden.device))
    for r0 in range(0, w.vocab, chunk):
        r1 = min(w.vocab, r0 + chunk)
        g.manual_seed((int(seed) * 3_000_017 + 13 + r0) & 0x7FFFFFFFFFFF)
        x = torch.randn((r1 - r0, w.hidden), generator=g, device=out_weight.device)
        out_weight[r0:r1].copy_(x.mul_(w.weight_std))


def hidden_and_weight_np(w: Workload, seed: int, T: int, V: int, D: int):
    """Small host fused-head inputs (uint16 bf16 bits): hidden ~ N(0, 1), W ~ N(0, std^2)."""
    rng = _rng(seed, _name_id(w.name), 10, T, V, D)
    h = rng.standard_normal((T, D), dtype=np.float32)
    wt = rng.standard_normal((V, D), dtype=np.float32) * np.float32(w.weight_std or 0.02)
    return bf16_bits_from_f32(h), bf16_bits_from_f32(wt)
