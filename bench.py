"""Throughput of the policy-loss hot path on the multi-turn agent workload.

Workload (the configuration the headline metric is quoted on): 16 groups x 8
trajectories with lengths U{256..2048} (about 147K packed tokens), ~40% of the
tokens masked in spans, rewards Bernoulli(0.3), vocabulary V = 151,936, bf16
logits ~ N(0, 2^2), 16,384-row microbatches. The whole batch's logits and
gradient stay resident in HBM (about 90 GB, far above the 129 MB L2, so no L2
flush is needed between steps).

One step = rl_group_advantages over the batch, then rl_policy_loss_fwd_bwd over
every microbatch (the loss accumulates on the device; its value is read back
once after the timed region).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line. With N > 1 (launched by torchrun) every rank runs its own
replica of the workload; the step time is the maximum over ranks.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import multiprocessing as mp
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_16798_gb300 import workloads as W  # noqa: E402

METRIC = "policy-loss fwd+bwd tokens/s at V=151,936 and % of HBM roofline (1 GB300)"
UNIT = "tokens/s"
WORKLOAD = W.WORKLOADS["multiturn"]
PROFILE = os.path.join(ROOT, "profiles", "rows_kernel_multiturn.md")
KERNEL_SRC = os.path.join(ROOT, "paper_2608_16798_gb300", "csrc", "rl_rows.cu")
FALLBACK_HBM_GBS = 6800.0


def workload_config(T, n_mb):
    w = WORKLOAD
    return {"workload": f"multiturn: {w.n_groups} groups x {w.group_size} trajectories, lengths U{{256..2048}}, "
                        f"~40% masked in spans, V={w.vocab}, bf16 logits N(0,2^2), {w.microbatch}-row microbatches",
            "tokens_per_step": int(T), "microbatches": int(n_mb), "vocab": w.vocab, "logits": "bf16",
            "l2": "no flush: resident inputs (logits + gradient) far larger than L2",
            "parallelism": "replicas", "seed": 0}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def profiled_traffic():
    """Per-launch DRAM bytes of the rows kernel from the committed ncu summary, if it was taken
    on the current kernel source (else None)."""
    if not os.path.exists(PROFILE):
        return None
    txt = open(PROFILE).read()
    m_b = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    m_h = re.search(r"kernel_source_sha256:\s*([0-9a-f]{64})", txt)
    if not m_b or not m_h:
        return None
    cur = hashlib.sha256(open(KERNEL_SRC, "rb").read()).hexdigest()
    return float(m_b.group(1)) if cur == m_h.group(1) else None


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index  # nvidia-smi --id value: the GPU's UUID when torch reports one
        self.proc = None
        self.path = os.path.join("/tmp", f"bench_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.remove(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------- device workload

class DeviceBatch:
    def __init__(self, torch, R, dev, seed=0):
        w = WORKLOAD
        self.lay = W.make_layout(w, seed)
        self.T = self.lay.n_tokens
        self.V = w.vocab
        self.mbs = W.microbatches(self.lay, w.microbatch)
        t = torch
        self.logits = t.empty((self.T, self.V), dtype=t.bfloat16, device=dev)
        W.logits_rows_torch(w, seed, 0, self.T, self.logits)
        self.ids = W.sample_tokens_torch(self.logits, seed, 0, w)
        self.grad = t.empty_like(self.logits)
        d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
        self.mask = d(self.lay.mask)
        self.rewards = d(self.lay.rewards)
        self.group_offsets = d(self.lay.group_offsets)
        self.traj_offsets = d(self.lay.traj_offsets)
        self.valid = d(self.lay.traj_valid)
        self.params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
        self.ws = R.new_workspace(w.microbatch, self.V, device=dev)
        # pi_old as the training engine recomputes it: this library's forward log-probs, plus noise
        logp = t.empty(self.T, dtype=t.float32, device=dev)
        for lo, hi in self.mbs:
            R.rl_token_logprobs(self.logits[lo:hi], self.ids[lo:hi], self.ws, logp_out=logp[lo:hi])
        self.old = d(W.old_logp_from(logp.cpu().numpy(), w, seed))
        self.adv = t.empty(self.lay.n_traj, dtype=t.float32, device=dev)
        self.coef = t.empty_like(self.adv)
        self.n_tok = t.empty(self.lay.n_traj, dtype=t.int32, device=dev)
        self.token_traj = t.empty(self.T, dtype=t.int32, device=dev)
        self.loss = t.zeros(1, dtype=t.float64, device=dev)
        h = hashlib.sha256()
        for a in (self.lay.traj_offsets, self.lay.group_offsets, self.lay.rewards, self.lay.mask,
                  self.ids.cpu().numpy(), self.old.cpu().numpy()):
            h.update(np.ascontiguousarray(a).tobytes())
        for r in (0, self.T // 2, self.T - 1):
            h.update(self.logits[r].view(t.int16).cpu().numpy().tobytes())
        self.inputs_sha256 = h.hexdigest()
        m = self.lay.mask.astype(np.int64)
        es = 2
        # algorithmic bytes per microbatch launch: trainable rows read + write, other rows write only
        self.mb_bytes = [int(((m[lo:hi] + 1) * self.V * es).sum()) for lo, hi in self.mbs]

    def step(self, R, events=None):
        R.rl_group_advantages(self.group_offsets, self.rewards, self.traj_offsets, self.mask, self.params, self.ws,
                              traj_valid=self.valid, adv_out=self.adv, coef_out=self.coef, n_tok_out=self.n_tok,
                              token_traj_out=self.token_traj)
        for k, (lo, hi) in enumerate(self.mbs):
            if events is not None:
                events[k][0].record()
            R.rl_policy_loss_fwd_bwd(self.logits[lo:hi], self.ids[lo:hi], self.mask[lo:hi], self.token_traj[lo:hi],
                                     self.adv, self.coef, self.old[lo:hi], self.params, self.ws, self.loss,
                                     grad_out=self.grad[lo:hi])
            if events is not None:
                events[k][1].record()

    def launches_per_step(self):
        # rl_group_advantages: 2 kernels; rl_policy_loss_fwd_bwd: 1 kernel per microbatch
        return 2 + len(self.mbs)


def time_logits_extras(torch, R, batch, dev, peak, reps=20):
    """Forward-only log-probs over the batch's microbatches (the pi_old / pi_ref recompute; one
    read of each logits row, V x 2 bytes), with and without the entropy, and the advantages
    alone (CUDA-graph replays)."""
    t = torch
    logp = t.empty(batch.T, dtype=t.float32, device=dev)
    ent = t.empty_like(logp)
    out = {}
    for name, want_ent in (("token_logprobs", False), ("token_logprobs_entropy", True)):
        def run():
            for lo, hi in batch.mbs:
                R.rl_token_logprobs(batch.logits[lo:hi], batch.ids[lo:hi], batch.ws, logp_out=logp[lo:hi],
                                    entropy_out=ent[lo:hi] if want_ent else None)
        ms = _time_calls(torch, run, 3, reps)
        gbs = batch.T * batch.V * 2 / (ms * 1e-3) / 1e9
        out[name] = {"ms_per_batch": ms, "tokens_per_s": batch.T / (ms * 1e-3), "achieved_gbs": gbs,
                     "frac": gbs / peak, "frac_of_nominal_8tbs": gbs / 8000.0,
                     "algorithmic_bytes_per_token": batch.V * 2}
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
    ms_adv = _time_graph(torch, lambda: R.rl_group_advantages(batch.group_offsets, batch.rewards, batch.traj_offsets,
                                                              batch.mask, params, batch.ws, traj_valid=batch.valid,
                                                              adv_out=batch.adv, coef_out=batch.coef,
                                                              n_tok_out=batch.n_tok, token_traj_out=batch.token_traj),
                         50)
    out["group_advantages_us"] = ms_adv * 1e3
    return out


def time_other_workloads(torch, R, dev, peak, reps=10, oracle_slices=None):
    """rl_policy_loss_fwd_bwd on the long-horizon workload (bf16, entropy + k3 KL, two resident
    32,768-row microbatches: the first and the middle one) and the edge workload (fp32,
    V = 32,000, the whole 131,072-row batch as one microbatch), timed with CUDA events around
    `reps` launches after two warm-up launches; and rl_group_advantages over each workload's
    whole batch (512 trajectories in 32 groups; 16,384 in 4,096 groups) as CUDA-graph replays. The logits stay resident (20 and 17 GB, far
    above L2); pi_old comes from the library's forward pass plus the workload's noise. With
    `oracle_slices` (a dict), bounded spans of the same device rows are copied to the host for
    the CPU oracle's timing: 4,096 rows at the start of each of the two timed long-horizon
    microbatches and of the last (partial) one, drawn on the device like the others, the whole
    edge batch, the whole tiny batch."""
    t = torch
    out = {}
    # (microbatch, timed): the last long-horizon microbatch is partial (18,951 rows), so only the
    # CPU oracle's sample takes rows from it
    for name, picks in (("longhorizon", (("first", True), ("middle", True), ("last", False))),
                        ("edge", (("first", True),))):
        w = W.WORKLOADS[name]
        lay = W.make_layout(w, 0)
        mbs = W.microbatches(lay, w.microbatch)
        where = {"first": mbs[0], "middle": mbs[len(mbs) // 2], "last": mbs[-1]}
        chosen = [(where[k], timed) for k, timed in picks]
        dt = t.bfloat16 if w.dtype == "bf16" else t.float32
        es = 2 if w.dtype == "bf16" else 4
        d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
        kl = 3 if w.kl_coef else 0
        params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, w.kl_coef, kl, w.entropy_coef, 0.0, 1e-6, 0)
        ws = R.new_workspace(w.microbatch, w.vocab, device=dev)
        go, rw, to, mk, va = (d(lay.group_offsets), d(lay.rewards), d(lay.traj_offsets), d(lay.mask),
                              d(lay.traj_valid))
        adv, coef, n_tok, tt = R.rl_group_advantages(go, rw, to, mk, params, ws, traj_valid=va)
        coef_h, tt_h = coef.cpu().numpy(), tt.cpu().numpy()
        # the advantages over the workload's whole batch, alone (CUDA-graph replays)
        ms_adv = _time_graph(torch, lambda: R.rl_group_advantages(go, rw, to, mk, params, ws, traj_valid=va,
                                                                  adv_out=adv, coef_out=coef, n_tok_out=n_tok,
                                                                  token_traj_out=tt), 20)
        items, nbytes, rows_total = [], 0, 0
        for (lo, hi), timed in chosen:
            if not timed and oracle_slices is None:
                continue
            n = hi - lo if timed else min(hi - lo, ORACLE_ROWS[name])
            logits = t.empty((n, w.vocab), dtype=dt, device=dev)
            W.logits_rows_torch(w, 0, lo, n, logits)
            ids = W.sample_tokens_torch(logits, 0, lo, w)
            logp, _, _ = R.rl_token_logprobs(logits, ids, ws)
            lp = logp.cpu().numpy()
            old = d(W.old_logp_from(lp, w, 0, lo))
            ref = d(W.ref_logp_from(lp, w, 0, lo)) if w.ref_noise_std else None
            if oracle_slices is not None:
                n_or = min(n, ORACLE_ROWS[name])
                oracle_slices.setdefault(name, []).append((lo, logits[:n_or], ids[:n_or]))
            if not timed:
                continue
            grad = t.empty_like(logits)
            trained = (lay.mask[lo:hi] != 0) & (coef_h[tt_h[lo:hi]] != 0)
            nbytes += int((trained.astype(np.int64) + 1).sum()) * w.vocab * es
            rows_total += n
            items.append((logits, ids, d(lay.mask[lo:hi]), tt[lo:hi], old, ref, grad))
        loss = t.zeros(1, dtype=t.float64, device=dev)

        def launch(k):
            lg, ids, m, tk, old, ref, g = items[k % len(items)]
            R.rl_policy_loss_fwd_bwd(lg, ids, m, tk, adv, coef, old, params, ws, loss, grad_out=g, ref_logp=ref)

        for k in range(2):
            launch(k)
        t.cuda.synchronize(dev)
        a, b = t.cuda.Event(enable_timing=True), t.cuda.Event(enable_timing=True)
        a.record()
        for k in range(reps):
            launch(k)
        b.record()
        b.synchronize()
        st, word = R.rl_query_status(ws)
        if word != 0:
            raise RuntimeError(f"device status word {word} after the {name} timing")
        ms = a.elapsed_time(b) / reps
        per_launch_bytes = nbytes / len(items)
        rows_per_launch = rows_total / len(items)
        gbs = per_launch_bytes / (ms * 1e-3) / 1e9
        if oracle_slices is not None:
            oracle_slices[name] = make_oracle_slice(w, oracle_slices[name], ORACLE_PARAMS[name])
        out[name] = {"rows_per_launch": rows_per_launch, "vocab": w.vocab, "dtype": w.dtype,
                     "entropy_coef": w.entropy_coef, "kl_coef": w.kl_coef, "ms_per_launch": ms,
                     "tokens_per_s": rows_per_launch / (ms * 1e-3), "algorithmic_bytes_per_launch": per_launch_bytes,
                     "achieved_gbs": gbs, "frac": gbs / peak, "reps": reps,
                     "group_advantages_us": ms_adv * 1e3, "trajectories": int(lay.n_traj),
                     "groups": int(len(lay.group_offsets) - 1), "batch_tokens": int(lay.n_tokens)}
        del items
        t.cuda.empty_cache()
    out["tiny"] = time_tiny(torch, R, dev, oracle_slices=oracle_slices)
    return out


# rows of each span the CPU oracle is timed on, and the objective's parameters there
ORACLE_ROWS = {"longhorizon": 4096, "edge": 131072, "tiny": 512}
ORACLE_PARAMS = {"longhorizon": {"kl_coef": 1e-3, "kl_estimator": 3, "entropy_coef": 1e-3}, "edge": {}, "tiny": {}}
ORACLE_HEAD_TOKENS = 1024


def time_tiny(torch, R, dev, reps=100, oracle_slices=None):
    """The tiny workload (one group of 8 trajectories x 64 tokens, V = 4,096 bf16): a whole step
    (advantages + the loss over the 512 rows) is 8.4 MB of logits and gradient, resident in the
    129 MB L2, so it is latency-bound and gets no HBM fraction. Timed as CUDA-graph replays (device
    time) and as eager calls (with the host's launch overhead)."""
    t = torch
    w = W.WORKLOADS["tiny"]
    lay = W.make_layout(w, 0)
    d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    T = lay.n_tokens
    logits = t.empty((T, w.vocab), dtype=t.bfloat16, device=dev)
    W.logits_rows_torch(w, 0, 0, T, logits)
    ids = W.sample_tokens_torch(logits, 0, 0, w)
    if oracle_slices is not None:
        oracle_slices["tiny"] = make_oracle_slice(w, [(0, logits, ids)], ORACLE_PARAMS["tiny"])
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
    ws = R.new_workspace(T, w.vocab, device=dev)
    logp, _, _ = R.rl_token_logprobs(logits, ids, ws)
    old = d(W.old_logp_from(logp.cpu().numpy(), w, 0, 0))
    go, rw, to, mask, valid = (d(lay.group_offsets), d(lay.rewards), d(lay.traj_offsets), d(lay.mask),
                               d(lay.traj_valid))
    adv, coef = t.empty(lay.n_traj, device=dev), t.empty(lay.n_traj, device=dev)
    n_tok = t.empty(lay.n_traj, dtype=t.int32, device=dev)
    tt = t.empty(T, dtype=t.int32, device=dev)
    grad, loss = t.empty_like(logits), t.zeros(1, dtype=t.float64, device=dev)

    def step():
        R.rl_group_advantages(go, rw, to, mask, params, ws, traj_valid=valid, adv_out=adv, coef_out=coef,
                              n_tok_out=n_tok, token_traj_out=tt)
        R.rl_policy_loss_fwd_bwd(logits, ids, mask, tt, adv, coef, old, params, ws, loss, grad_out=grad)

    ms_graph = _time_graph(torch, step, reps)
    ms_eager = _time_calls(torch, step, 3, reps)
    st, word = R.rl_query_status(ws)
    if word != 0:
        raise RuntimeError(f"device status word {word} after the tiny timing")
    return {"rows_per_step": T, "vocab": w.vocab, "dtype": w.dtype, "l2_resident": True,
            "bytes_per_step": int(((lay.mask.astype(np.int64) + 1) * w.vocab * 2).sum()),
            "us_per_step_graph": ms_graph * 1e3, "us_per_step_eager": ms_eager * 1e3,
            "tokens_per_s_graph": T / (ms_graph * 1e-3), "tokens_per_s_eager": T / (ms_eager * 1e-3),
            "note": "advantages + loss over the whole batch; resident in L2, so latency-bound: no HBM fraction"}


def time_ppo(torch, R, batch, dev, warmup=3, reps=20):
    """PPO step on the same batch (Sec. 2.3.1, Sec. 2.3.4): token-mean coefficients, masked GAE over
    the whole batch (skip reading, gamma = lambda = 1, R_i at each trajectory's last trainable token,
    value predictions N(0.3, 0.25^2)), then per microbatch the clipped policy loss with per-token
    advantages and the masked value loss."""
    t = torch
    w = WORKLOAD
    d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    values = d(W.value_predictions(w, 0, batch.T))
    v_new = values + 0.05  # the value model being trained
    traj_r = batch.rewards.float()
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 1, token_level_adv=1)
    coef = t.empty_like(batch.coef)
    adv_traj = t.empty_like(batch.adv)
    adv = t.empty(batch.T, dtype=t.float32, device=dev)
    ret = t.empty_like(adv)
    dv = t.empty_like(adv)
    loss = t.zeros(1, dtype=t.float64, device=dev)
    vloss = t.zeros(1, dtype=t.float64, device=dev)

    def gae():
        R.rl_masked_gae(batch.traj_offsets, batch.mask, values, batch.ws, 1.0, 1.0, True, traj_rewards=traj_r,
                        adv_out=adv, returns_out=ret)

    def step():
        R.rl_group_advantages(batch.group_offsets, batch.rewards, batch.traj_offsets, batch.mask, params, batch.ws,
                              traj_valid=batch.valid, adv_out=adv_traj, coef_out=coef, n_tok_out=batch.n_tok,
                              token_traj_out=batch.token_traj)
        gae()
        for lo, hi in batch.mbs:
            R.rl_policy_loss_fwd_bwd(batch.logits[lo:hi], batch.ids[lo:hi], batch.mask[lo:hi],
                                     batch.token_traj[lo:hi], adv[lo:hi], coef, batch.old[lo:hi], params, batch.ws,
                                     loss, grad_out=batch.grad[lo:hi])
            R.rl_value_loss_fwd_bwd(v_new[lo:hi], ret[lo:hi], batch.mask[lo:hi], batch.token_traj[lo:hi], coef,
                                    batch.ws, vloss, d_values=dv[lo:hi])

    lo, hi = batch.mbs[0]
    ms_step = _time_calls(torch, step, warmup, reps)
    # the two small kernels are timed as CUDA-graph replays, so that host launch overhead stays out
    ms_gae = _time_graph(torch, gae, 10 * reps)
    ms_val = _time_graph(torch, lambda: R.rl_value_loss_fwd_bwd(v_new[lo:hi], ret[lo:hi], batch.mask[lo:hi],
                                                                batch.token_traj[lo:hi], coef, batch.ws, vloss,
                                                                d_values=dv[lo:hi]), 10 * reps)
    # sequence-level importance weights over the whole batch (rollout log-probs = old + N(0, 0.02^2))
    roll = d(W.rollout_logp_from(batch.old.cpu().numpy(), 0, std=0.02))
    w_seq = t.empty(batch.lay.n_traj, dtype=t.float32, device=dev)
    ms_seq = _time_graph(torch, lambda: R.rl_sequence_is_weights(batch.token_traj, batch.mask, batch.old, roll,
                                                                 batch.lay.n_traj, batch.ws, cap=2.0,
                                                                 weight_out=w_seq), 10 * reps)
    st, word = R.rl_query_status(batch.ws)
    if word != 0:
        raise RuntimeError(f"device status word {word} after the PPO timing")
    gae_bytes = batch.T * (1 + 4 + 4 + 4) + 8 * (batch.lay.n_traj + 1) + 4 * batch.lay.n_traj
    val_bytes = (hi - lo) * (4 + 4 + 1 + 4 + 4 + 8) + 4 * batch.lay.n_traj
    return {"workload": "multiturn batch: values N(0.3,0.25^2), gamma = lambda = 1, skip reading, token-mean weights",
            "ms_per_step": ms_step, "tokens_per_s": batch.T / (ms_step * 1e-3),
            "gae_us": ms_gae * 1e3, "gae_algorithmic_bytes": gae_bytes,
            "gae_achieved_gbs": gae_bytes / (ms_gae * 1e-3) / 1e9,
            "value_loss_us_per_microbatch": ms_val * 1e3, "value_loss_algorithmic_bytes": val_bytes,
            "sequence_is_us": ms_seq * 1e3, "sequence_is_algorithmic_bytes": batch.T * (4 + 1 + 4 + 4),
            "reps": reps,
            "note": "step = advantages/coefficients + GAE + per microbatch (policy loss with per-token advantages "
                    "+ value loss); GAE and value loss (+ its reduction) timed as CUDA-graph replays; both are "
                    "latency-bound (a few bytes per token)"}


def time_tree(torch, R, dev, reps=3):
    """Tree-packed batches (Sec. 3.2.1-3.2.3): the native prefix-tree builder over the tree
    workload's 128 rollouts on the host cores, then advantages and coefficients by owner and the
    sequence-level weights on the packed stream (CUDA-graph replays)."""
    t = torch
    w = W.WORKLOADS["tree"]
    prompts, calls, aux = W.tree_rollouts(w, seed=0)
    captured = sum(len(x) + len(y) for cs in calls for x, y in cs)
    threads = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves, n_threads=threads)
    t0 = time.perf_counter()
    for _ in range(reps):
        out = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves, n_threads=threads)
    host_s = (time.perf_counter() - t0) / reps
    n = len(prompts)
    d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    owner, mask = d(out["owner"]), d(out["mask"])
    go = d(np.arange(0, n + 1, w.group_size, dtype=np.int32))
    rewards = d((np.random.default_rng(0).random(n) < w.reward_p).astype(np.float32))
    valid = d(np.array([s["valid"] for s in out["stats"]], np.uint8))
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
    ws = R.new_workspace(n, 0, device=dev)
    adv, coef, L = (t.empty(n, dtype=dt, device=dev) for dt in (t.float32, t.float32, t.int32))
    ms_adv = _time_graph(torch, lambda: R.rl_group_advantages_by_owner(go, rewards, owner, mask, params, ws,
                                                                       traj_valid=valid, adv_out=adv, coef_out=coef,
                                                                       n_tok_out=L), 50)
    st, word = R.rl_query_status(ws)
    if word != 0:
        raise RuntimeError(f"device status word {word} after the tree timing")
    T = len(out["tokens"])
    return {"workload": "tree: 16 tasks x 8 rollouts of captured calls (prompt U{200..800}, 4-16 turns, tool "
                        "outputs, 10% retries, subagent and compaction calls, 1 in 20 runaway), max 12 leaves",
            "calls": sum(len(c) for c in calls), "captured_tokens": captured, "packed_tokens": T,
            "trainable_tokens": int(out["mask"].sum()), "rollouts_kept": int(sum(s["valid"] for s in out["stats"])),
            "dedup_ratio": captured / max(T, 1), "host_build_ms": host_s * 1e3, "host_threads": threads,
            "host_captured_tokens_per_s": captured / host_s,
            "advantages_by_owner_us": ms_adv * 1e3,
            "note": "host build = rl_prefix_tree_build_batch (C++, one thread per rollout at a time); "
                    "advantages by owner timed as CUDA-graph replays"}


class StagedPinned:
    """Host memory for the end-to-end leg: a HostStagingBuffer (one mapping with transparent huge
    pages, registered with the CUDA runtime). Once filled, its units are qualified by timing a
    copy from each to the device; units that copy far below the median are replaced and refilled
    before any timed work. On the Grace host of a GB300, a few physical huge pages in some
    processes were measured to copy at 3-72 GB/s against 210 GB/s from the rest, and pages can
    turn slow when first written. Falls back to
    torch's pinned allocator when the mapping or registration is refused."""

    def __init__(self, torch, rows, cols, dtype, dev):
        from paper_2608_16798_gb300.host_staging import HostStagingBuffer

        self.torch, self.dev, self.buf, self.qualified = torch, dev, None, None
        nbytes = rows * cols * torch.empty((), dtype=dtype).element_size()
        cr = torch.cuda.cudart()
        try:
            self.buf = HostStagingBuffer(nbytes, lambda a, n: cr.cudaHostRegister(a, n, 0) == cr.cudaError.success,
                                         lambda a: cr.cudaHostUnregister(a))
            self.tensor = torch.frombuffer(self.buf.buffer(), dtype=dtype).view(rows, cols)
            self.kind = "huge pages, registered, qualified"
        except Exception:
            self.close()
            self.tensor = torch.empty((rows, cols), dtype=dtype, pin_memory=True)
            self.kind = "torch pinned"

    def qualify(self, source):
        """After the fill: time a copy from each unit, replace slow units and refill them from
        `source` (a device tensor whose bytes the buffer holds from its start)."""
        if self.buf is None:
            return
        t = self.torch
        units = t.frombuffer(self.buf.buffer(whole_units=True), dtype=t.uint8)
        src = source.view(-1).view(t.uint8)
        scratch = t.empty(self.buf.unit, dtype=t.uint8, device=self.dev)
        s = t.cuda.Stream(self.dev)

        def probe(off, n):
            a0, a1 = t.cuda.Event(enable_timing=True), t.cuda.Event(enable_timing=True)
            with t.cuda.stream(s):
                a0.record(s)
                scratch[:n].copy_(units[off:off + n], non_blocking=True)
                a1.record(s)
            a1.synchronize()
            return n / a0.elapsed_time(a1) / 1e6

        def refill(off, n):
            n = max(0, min(n, self.buf.nbytes - off, src.numel() - off))
            if n:
                units[off:off + n].copy_(src[off:off + n])

        try:
            self.qualified = self.buf.qualify(probe, refill)
        except OSError as exc:
            self.qualified = {"error": str(exc), "replaced": self.buf.replaced, "unit_bytes": self.buf.unit}
            if self.buf.broken:  # never copy from a range with a hole: torch's pinned memory instead
                rows, cols = self.tensor.shape
                dtype = self.tensor.dtype
                del units
                self.close()
                self.tensor = t.empty((rows, cols), dtype=dtype, pin_memory=True)
                self.tensor.view(-1).copy_(source.view(-1)[:self.tensor.numel()])
                self.kind = "torch pinned (a staging unit could not be replaced)"
        t.cuda.synchronize(self.dev)

    def close(self):
        self.tensor = None
        if self.buf is not None:
            self.buf.close()
            self.buf = None


def host_mem_available() -> int:
    """MemAvailable of /proc/meminfo in bytes (0 if unknown)."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def e2e_run(torch, R, batch, dev, steps, warmup, slots=4, repeats=3):
    """Same step through host buffers: every step copies its inputs from pinned host memory (the
    whole batch's logits, microbatch by microbatch, and the metadata) to the device and reads the
    step's loss back; the gradient stays in HBM (batch.grad), where a training step's backward
    consumes it.

    Logits go through `slots` device buffers on two copy streams: the copy of microbatch k waits
    only for the kernel that last read its slot, so copies run back to back while the kernels
    follow, and a copy from a slow region of host memory overlaps the next one."""
    t = torch
    w = WORKLOAD
    V, mb = batch.V, w.microbatch
    # the whole batch in pinned host memory when every rank on the node fits in 40% of the
    # available host memory; otherwise a ring of two microbatches (the timing is the same)
    ranks_here = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
    whole = batch.T * V * 2 * ranks_here <= 0.4 * host_mem_available()
    # pinned host memory (huge pages, registered), filled by device-to-host copies (host-side
    # CPU writes would leave dirty cache lines that the GPU's reads then have to fetch)
    # one mapping for the whole host source (separate per-microbatch mappings measured 3-73 GB/s
    # from some of them, one mapping 211 GB/s from nearly all of its microbatches)
    if whole:
        pinned = StagedPinned(t, batch.T, V, t.bfloat16, dev)
        for lo, hi in batch.mbs:
            pinned.tensor[lo:hi].copy_(batch.logits[lo:hi])
        pinned.qualify(batch.logits)

        def make_host_views():
            return [pinned.tensor[lo:hi] for lo, hi in batch.mbs]
    else:
        pinned = StagedPinned(t, 2 * mb, V, t.bfloat16, dev)
        for k in range(2):
            lo, hi = batch.mbs[k % len(batch.mbs)]
            pinned.tensor[k * mb:k * mb + hi - lo].copy_(batch.logits[lo:hi])
        if len(batch.mbs) >= 2:  # the ring then holds the batch's first 2 x mb rows, byte for byte
            pinned.qualify(batch.logits)

        def make_host_views():
            return [pinned.tensor[(k % 2) * mb:(k % 2) * mb + hi - lo] for k, (lo, hi) in enumerate(batch.mbs)]
    host_mb = make_host_views()
    src = list(range(len(batch.mbs)))
    meta_host = {n: getattr(batch, n).cpu().pin_memory() for n in
                 ("ids", "mask", "old", "rewards", "group_offsets", "traj_offsets", "valid")}
    meta_dev = {n: t.empty_like(getattr(batch, n)) for n in meta_host}
    dev_logits = [t.empty((mb, V), dtype=t.bfloat16, device=dev) for _ in range(slots)]
    loss_host = t.zeros(1, dtype=t.float64, pin_memory=True)
    copy_streams = [t.cuda.Stream(dev), t.cuda.Stream(dev)]
    copy_in = copy_streams[0]
    comp = t.cuda.current_stream(dev)
    adv, coef = t.empty_like(batch.adv), t.empty_like(batch.coef)
    n_tok, tt = t.empty_like(batch.n_tok), t.empty_like(batch.token_traj)
    loss = t.zeros(1, dtype=t.float64, device=dev)
    h2d = sum(v.numel() * v.element_size() for v in meta_host.values())
    h2d += sum((hi - lo) * V * 2 for lo, hi in batch.mbs)
    d2h = loss_host.numel() * loss_host.element_size()
    read_done = [None] * slots

    def one_step():
        with t.cuda.stream(copy_in):
            for n, h in meta_host.items():
                meta_dev[n].copy_(h, non_blocking=True)
            meta_ready = t.cuda.Event()
            meta_ready.record(copy_in)
        comp.wait_event(meta_ready)
        loss.zero_()
        R.rl_group_advantages(meta_dev["group_offsets"], meta_dev["rewards"], meta_dev["traj_offsets"],
                              meta_dev["mask"], batch.params, batch.ws, traj_valid=meta_dev["valid"], adv_out=adv,
                              coef_out=coef, n_tok_out=n_tok, token_traj_out=tt)
        for k, (lo, hi) in enumerate(batch.mbs):
            s = k % slots
            n = hi - lo
            cs = copy_streams[k & 1]
            with t.cuda.stream(cs):
                if read_done[s] is not None:
                    cs.wait_event(read_done[s])
                dev_logits[s][:n].copy_(host_mb[src[k]][:n], non_blocking=True)
                loaded = t.cuda.Event()
                loaded.record(cs)
            comp.wait_event(loaded)
            R.rl_policy_loss_fwd_bwd(dev_logits[s][:n], meta_dev["ids"][lo:hi], meta_dev["mask"][lo:hi], tt[lo:hi],
                                     adv, coef, meta_dev["old"][lo:hi], batch.params, batch.ws, loss,
                                     grad_out=batch.grad[lo:hi], stream=comp)
            read_done[s] = t.cuda.Event()
            read_done[s].record(comp)
        loss_host.copy_(loss, non_blocking=True)

    def copies_alone():
        # each microbatch's copy timed alone: the host source's bandwidth, which bounds the step
        out = []
        for k, (lo, hi) in enumerate(batch.mbs):
            a0, a1 = t.cuda.Event(enable_timing=True), t.cuda.Event(enable_timing=True)
            with t.cuda.stream(copy_in):
                a0.record(copy_in)
                dev_logits[0][:hi - lo].copy_(host_mb[src[k]][:hi - lo], non_blocking=True)
                a1.record(copy_in)
            a1.synchronize()
            out.append((hi - lo) * V * 2 / a0.elapsed_time(a1) / 1e6)
        return out

    # repetitions of `steps` timed steps; before each, the staging buffer is qualified again
    # (pages of a qualified buffer have been seen to turn slow later in the same process)
    runs = []
    for rep in range(repeats):
        if rep > 0 and (whole or len(batch.mbs) >= 2):
            pinned.qualify(batch.logits)
            host_mb[:] = make_host_views()  # the buffer may have been replaced
        staging = pinned.qualified
        alone = copies_alone()
        t.cuda.synchronize(dev)
        for _ in range(warmup):
            one_step()
        t.cuda.synchronize(dev)
        e0, e1 = t.cuda.Event(enable_timing=True), t.cuda.Event(enable_timing=True)
        e0.record(comp)
        for _ in range(steps):
            one_step()
        e1.record(comp)
        e1.synchronize()
        t.cuda.synchronize(dev)
        ms_run = e0.elapsed_time(e1)
        runs.append({"ms": ms_run, "in_steps_gbs": h2d * steps / (ms_run * 1e-3) / 1e9,
                     "alone_gbs_min": min(alone), "alone_gbs_median": statistics.median(alone),
                     "staging_replaced": None if staging is None else staging["replaced"]})
    check = float(loss_host.item())
    del host_mb
    pinned.close()
    ms = statistics.median(r["ms"] for r in runs)
    copy_gbs = {"in_steps_median": h2d * steps / (ms * 1e-3) / 1e9, "runs": runs,
                "staging_unit_bytes": None if pinned.qualified is None else pinned.qualified["unit_bytes"]}
    return ms, h2d, d2h, check, ("whole batch" if whole else "ring of 2 microbatches") + ", " + pinned.kind, copy_gbs


# ----------------------------------------------------------------------------- oracle (CPU) legs

_W = {}


def _gen_init(shm_name, shape, ids_name):
    from multiprocessing import shared_memory

    sys.path.insert(0, ROOT)
    shm, ids_shm = shared_memory.SharedMemory(name=shm_name), shared_memory.SharedMemory(name=ids_name)
    _W.update(shm=shm, ids_shm=ids_shm, raw=np.ndarray(shape, dtype=np.uint16, buffer=shm.buf),
              ids=np.ndarray((shape[0],), dtype=np.int32, buffer=ids_shm.buf))


def _gen_rows(span):
    """Draw rows [lo, hi) of the workload with the numpy generators (each row its own seeded
    stream, so any split of the rows gives the same values)."""
    lo, hi = span
    raw, vals = W.logits_rows_np(WORKLOAD, 0, lo, hi - lo)
    _W["raw"][lo:hi] = raw
    _W["ids"][lo:hi] = W.sample_tokens_np(vals, 0, lo, WORKLOAD)
    return hi - lo


def _oracle_init(shm_name, shape, dtype, inputs, params):
    from multiprocessing import shared_memory

    sys.path.insert(0, ROOT)
    shm = shared_memory.SharedMemory(name=shm_name)
    raw = np.ndarray(shape, dtype=np.uint16 if dtype == "bf16" else np.float32, buffer=shm.buf)
    _W.update(shm=shm, raw=raw, dtype=dtype, params=params, **inputs)


def _oracle_rows(span):
    import oracle.grpo_objective as O

    lo, hi = span
    ref = None if _W["ref"] is None else _W["ref"][lo:hi]
    O.policy_loss_fwd_bwd(_W["raw"][lo:hi], _W["dtype"], _W["ids"][lo:hi], _W["mask"][lo:hi], _W["tt"][lo:hi],
                          _W["adv"], _W["coef"], _W["old"][lo:hi], O.LossParams(**_W["params"]), ref_logp=ref)
    return hi - lo


def _logp_from_law(w, z_a):
    """Log-probability of the sampled token from the logit law alone (lse ~ ln V + sigma^2 / 2 for
    N(0, sigma^2) logits): places old_logp (and ref_logp) near it without using any output of the
    CUDA library."""
    return z_a - (math.log(w.vocab) + w.logit_std ** 2 / 2)


def _oracle_layout_inputs(w, lay, gidx):
    """Advantages, coefficients and trajectory ids of the whole batch (oracle), and the mask and
    trajectory ids of the rows gidx."""
    import oracle.grpo_objective as O

    P = O.LossParams(loss_agg=0)
    adv, coef, _, tt = O.advantages_and_coefficients(lay.rewards, lay.group_offsets, lay.traj_offsets, lay.mask,
                                                     lay.traj_valid, P)
    return adv, coef, lay.mask[gidx], tt[gidx]


class OracleSample:
    """The first microbatch of the benchmark batch (its first 16,384 packed tokens) in host
    shared memory for the float64 oracle: copied from the device batch (torch-drawn, the rows the
    GPU times) or, without a GPU, drawn by the numpy generators on all host cores (same law)."""

    def __init__(self, rows, device_logits=None, device_ids=None):
        from multiprocessing import shared_memory

        self.layout = W.make_layout(WORKLOAD, 0)
        self.rows = rows
        V = WORKLOAD.vocab
        self.shm = shared_memory.SharedMemory(create=True, size=rows * V * 2)
        self.raw = np.ndarray((rows, V), dtype=np.uint16, buffer=self.shm.buf)
        if device_logits is not None:
            import torch

            torch.from_numpy(self.raw.view(np.int16)).copy_(device_logits[:rows].view(torch.int16))
            self.ids = device_ids[:rows].cpu().numpy().astype(np.int32)
            self.source = "the device batch's torch-drawn logits, copied to the host"
        else:
            ids_shm = shared_memory.SharedMemory(create=True, size=rows * 4)
            try:
                spans = [(i, min(rows, i + 16)) for i in range(0, rows, 16)]
                cores = len(os.sched_getaffinity(0))
                with mp.get_context("spawn").Pool(cores, initializer=_gen_init,
                                                  initargs=(self.shm.name, (rows, V), ids_shm.name)) as pool:
                    pool.map(_gen_rows, spans, chunksize=4)
                self.ids = np.ndarray((rows,), dtype=np.int32, buffer=ids_shm.buf).copy()
            finally:
                ids_shm.close()
                ids_shm.unlink()
            self.source = "numpy-drawn logits of the same law (no GPU used)"

    dtype = "bf16"
    params = {}

    def oracle_inputs(self):
        """Inputs of the oracle for these rows; old_logp from the logit law (_logp_from_law)."""
        w, lay, rows = WORKLOAD, self.layout, self.rows
        z_a = (self.raw[np.arange(rows), self.ids].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        old = W.old_logp_from(_logp_from_law(w, z_a), w, 0)
        adv, coef, mask, tt = _oracle_layout_inputs(w, lay, np.arange(rows))
        return {"ids": self.ids, "mask": mask, "tt": tt, "adv": adv, "coef": coef, "old": old, "ref": None}

    def close(self):
        self.shm.close()
        self.shm.unlink()


class OracleSlice:
    """Spans of rows of a workload's device logits (rows the GPU timed), copied into host shared
    memory for the float64 oracle, with the oracle's own inputs for them: the batch's advantages
    and coefficients from the oracle, old_logp (and ref_logp) from the logit law."""

    def __init__(self, w, pieces, params):
        """pieces: (first global row, device logits [n x V], device ids [n]) per span."""
        from multiprocessing import shared_memory

        import torch

        self.w, self.params, self.dtype = w, params, w.dtype
        self.layout = W.make_layout(w, 0)
        self.rows = sum(int(lg.shape[0]) for _, lg, _ in pieces)
        es = 2 if w.dtype == "bf16" else 4
        self.shm = shared_memory.SharedMemory(create=True, size=self.rows * w.vocab * es)
        self.raw = np.ndarray((self.rows, w.vocab), dtype=np.uint16 if es == 2 else np.float32, buffer=self.shm.buf)
        ids, old, ref, gidx, r = [], [], [], [], 0
        for lo, lg, dids in pieces:
            n = int(lg.shape[0])
            view = torch.from_numpy(self.raw[r:r + n].view(np.int16 if es == 2 else np.int32))
            view.copy_(lg.view(torch.int16 if es == 2 else torch.int32))
            a = dids.cpu().numpy().astype(np.int32)
            z = self.raw[np.arange(r, r + n), a]
            z_a = ((z.astype(np.uint32) << 16).view(np.float32) if es == 2 else z).astype(np.float64)
            lp = _logp_from_law(w, z_a)
            ids.append(a)
            old.append(W.old_logp_from(lp, w, 0, lo))
            ref.append(W.ref_logp_from(lp, w, 0, lo) if w.ref_noise_std else None)
            gidx.append(np.arange(lo, lo + n))
            r += n
        self.ids, self.old = np.concatenate(ids), np.concatenate(old)
        self.ref = None if ref[0] is None else np.concatenate(ref)
        self.gidx = np.concatenate(gidx)
        self.spans = [(lo, lo + int(lg.shape[0])) for lo, lg, _ in pieces]

    def oracle_inputs(self):
        adv, coef, mask, tt = _oracle_layout_inputs(self.w, self.layout, self.gidx)
        return {"ids": self.ids, "mask": mask, "tt": tt, "adv": adv, "coef": coef, "old": self.old, "ref": self.ref}

    def close(self):
        self.shm.close()
        self.shm.unlink()


def make_oracle_slice(w, pieces, params, fallback_rows=32768):
    """An OracleSlice, or the reason it could not be made (host or shared memory short): the
    CPU leg's extra samples never cost the benchmark its line. When the whole span does not fit,
    the first `fallback_rows` rows of the first span are tried instead."""
    try:
        return OracleSlice(w, pieces, params)
    except (OSError, MemoryError) as e:
        if not pieces or int(pieces[0][1].shape[0]) <= fallback_rows:
            return f"{type(e).__name__}: {e}"
        lo, lg, ids = pieces[0]
        try:
            return OracleSlice(w, [(lo, lg[:fallback_rows], ids[:fallback_rows])], params)
        except (OSError, MemoryError) as e2:
            return f"{type(e2).__name__}: {e2}"


class OraclePool:
    """The float64 oracle, as it stands, over a spawn pool of all host cores. Each job is a
    16-row span of the sample; ``run(lo, hi)`` times the oracle over rows [lo, hi) once."""

    CHUNK = 16

    def __init__(self, sample):
        self.cores = len(os.sched_getaffinity(0))
        self.sample = sample
        self.pool = mp.get_context("spawn").Pool(self.cores, initializer=_oracle_init,
                                                 initargs=(sample.shm.name, sample.raw.shape, sample.dtype,
                                                           sample.oracle_inputs(), sample.params))
        # imports and first touch of the workers (untimed)
        self.pool.map(_oracle_rows, [(i * self.CHUNK, (i + 1) * self.CHUNK) for i in range(self.cores)], chunksize=1)

    def run(self, lo, hi):
        """Seconds of wall time for the oracle over rows [lo, hi)."""
        spans = [(i, min(hi, i + self.CHUNK)) for i in range(lo, hi, self.CHUNK)]
        t0 = time.perf_counter()
        n = sum(self.pool.map(_oracle_rows, spans, chunksize=1))
        dt = time.perf_counter() - t0
        assert n == hi - lo
        return dt

    def close(self):
        self.pool.close()
        self.pool.join()


def time_oracle(sample: OracleSample):
    """The oracle over the whole first microbatch, once (about 1.5 s on 16 host cores)."""
    op = OraclePool(sample)
    try:
        dt = op.run(0, sample.rows)
    finally:
        op.close()
    lay = sample.layout
    trained = int(lay.mask[:sample.rows].sum())
    return {"value": sample.rows / dt, "unit": UNIT, "cores": op.cores, "kind": "oracle", "seconds": dt,
            "sample": f"the first microbatch of the batch, all {sample.rows} rows ({trained} trained, the others "
                      f"masked), once, from {sample.source}; float64 numpy oracle on {op.cores} spawn workers"}


def time_oracle_slice(sl):
    """The oracle over every row of a workload's slice, once, on all host cores (or the reason
    the slice is missing)."""
    if isinstance(sl, str):
        return {"unavailable": sl}
    op = OraclePool(sl)
    try:
        dt = op.run(0, sl.rows)
    finally:
        op.close()
    spans = ", ".join(f"[{lo}, {hi})" for lo, hi in sl.spans)
    return {"rows": sl.rows, "seconds": dt, "tokens_per_s": sl.rows / dt, "cores": op.cores,
            "sample": f"rows {spans} of the {sl.w.name} batch ({sl.w.dtype}, V = {sl.w.vocab}), drawn on the "
                      f"device as the GPU's workload draws them, once; float64 numpy oracle on {op.cores} spawn "
                      f"workers"}


# ----------------------------------------------------------------------------- main

def _r(x, nd=4):
    return None if x is None else float(f"{x:.{nd}g}")


def compact_summary(value, ms_step, roofline, extras, head, ppo, tree, cpu, e2e):
    """One short object per workload (time, tokens/s, fraction of the roofline it is held to),
    printed as the last key of the JSON line so that a reader keeping only the line's tail
    still has every workload's numbers."""
    out = {"multiturn_loss": {"ms_per_step": _r(ms_step), "tokens_per_s": _r(value), "frac": _r(roofline["frac"]),
                              "bound": "hbm"}}
    for k in ("longhorizon", "edge"):
        o = (extras.get("other_workloads") or {}).get(k)
        if o:
            out[f"{k}_loss"] = {"ms": _r(o["ms_per_launch"]), "tokens_per_s": _r(o["tokens_per_s"]),
                                "frac": _r(o["frac"]), "bound": "hbm", "adv_us": _r(o["group_advantages_us"])}
    tiny = (extras.get("other_workloads") or {}).get("tiny")
    if tiny:
        out["tiny_step"] = {"us_graph": _r(tiny["us_per_step_graph"]), "tokens_per_s": _r(tiny["tokens_per_s_graph"]),
                            "frac": None, "bound": "latency (L2-resident)"}
    for k in ("token_logprobs", "token_logprobs_entropy"):
        o = extras.get(k)
        if o:
            out[k] = {"ms": _r(o["ms_per_batch"]), "tokens_per_s": _r(o["tokens_per_s"]), "frac": _r(o["frac"]),
                      "bound": "hbm (read only)"}
    if head:
        out["fused_head_loss"] = {"ms": _r(head["ms_per_call"]), "tokens_per_s": _r(head["tokens_per_s"]),
                                  "frac": _r(head["frac"]), "frac_of_sustained": _r(head["frac_of_sustained"]),
                                  "bound": "tensor"}
        f = head["logprobs"]
        out["fused_head_logprobs"] = {"ms": _r(f["ms_per_call"]), "tokens_per_s": _r(f["tokens_per_s"]),
                                      "frac": _r(f["frac"]), "frac_of_sustained": _r(f["frac_of_sustained"]),
                                      "bound": "tensor"}
    if ppo:
        out["ppo_step"] = {"ms": _r(ppo["ms_per_step"]), "tokens_per_s": _r(ppo["tokens_per_s"]), "frac": None,
                           "bound": "hbm (its policy loss)"}
    if "group_advantages_us" in extras:
        out["group_advantages"] = {"us": _r(extras["group_advantages_us"]), "bound": "latency"}
    if tree:
        out["tree_build"] = {"ms": _r(tree["host_build_ms"]), "captured_tokens_per_s": _r(tree["host_captured_tokens_per_s"]),
                             "bound": "host"}
    if cpu:
        out["cpu_oracle"] = {"tokens_per_s": _r(cpu["value"]), "cores": cpu["cores"]}
        for k, o in (cpu.get("workloads") or {}).items():
            out["cpu_oracle"][f"{k}_tokens_per_s"] = _r(o.get("tokens_per_s"))
    if e2e:
        out["e2e"] = {"tokens_per_s": _r(e2e["value"])}
    return out


def max_over_ranks(value, dist, device):
    """Maximum of a per-rank float over all ranks (the step time every rank reports)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank, world, ms_total, steps):
    """Whole-job tokens per second: every rank processes tokens_per_rank per step (replicas)."""
    return tokens_per_rank * world / (ms_total / 1e3 / steps)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return int(os.environ.get("RANK", "0")), ws, int(os.environ.get("LOCAL_RANK", "0"))


def run_reference(args):
    """The oracle timed on the host cores, on the same workload, metric and unit. Each step runs
    the oracle over a span of the first microbatch's rows (the whole microbatch when the run is
    short; fewer rows per step for many steps, so that the run stays within a few minutes), the
    spans following each other through the microbatch; value is rows over the measured seconds
    of the timed steps and ms_per_step their measured median."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    lay = W.make_layout(WORKLOAD, 0)
    n_mb = len(W.microbatches(lay, WORKLOAD.microbatch))
    rows = min(lay.n_tokens, WORKLOAD.microbatch)
    sample = OracleSample(rows)
    op = None
    try:
        op = OraclePool(sample)
        # rows per step: about 120 s of oracle time for the whole run at the first span's rate
        n_probe = min(rows, 4 * op.CHUNK * op.cores)
        rate = n_probe / op.run(0, n_probe)
        steps = args.warmup + args.steps
        per_step = int(min(rows, max(op.CHUNK * op.cores, rate * 120.0 / steps)))
        per_step -= per_step % op.CHUNK
        times, lo = [], 0
        for i in range(steps):
            if lo + per_step > rows:
                lo = 0
            dt = op.run(lo, lo + per_step)
            lo += per_step
            if i >= args.warmup:
                times.append(dt)
        cores = op.cores
    finally:
        if op is not None:
            op.close()
        sample.close()
    v = per_step * len(times) / sum(times)
    ms_step = statistics.median(times) * 1e3
    trained = int(lay.mask[:rows].sum())
    cb = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
          "sample": f"{per_step} rows per step (of the first microbatch's {rows}, {trained} trained), "
                    f"{args.steps} timed steps after {args.warmup} warm-up steps, from {sample.source}; float64 "
                    f"numpy oracle on {cores} spawn workers"}
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "rows_per_step": per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(lay.n_tokens, n_mb), "cpu_baseline": cb,
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


HEAD = W.WORKLOADS["fusedhead"]
HEAD_T = 32768


class HeadBatch:
    """Fused-LM-head workload on the device: hidden bf16 [T x 4096] ~ N(0, 1), W bf16 [151,936 x 4096]
    ~ N(0, 0.02^2); masks and trajectories of the first T packed tokens of a multi-turn batch, advantages
    and coefficients from that whole batch; sampled ids drawn from softmax(hidden W^T) by Gumbel-max
    (the logits for this draw come from a torch matmul in the set-up, not from the library).
    old_logp sits near the sampled token's log-probability: z_a minus the log-sum-exp of V logits
    distributed N(0, |h_t|^2 0.02^2), ln V + |h_t|^2 0.02^2 / 2, minus the workload's log-ratio noise."""

    def __init__(self, torch, R, dev, T=HEAD_T, seed=0):
        t = torch
        w = HEAD
        self.T, self.D, self.V = T, w.hidden, w.vocab
        self.hidden = t.empty((T, self.D), dtype=t.bfloat16, device=dev)
        self.weight = t.empty((self.V, self.D), dtype=t.bfloat16, device=dev)
        W.hidden_and_weight_torch(w, seed, T, self.hidden, self.weight)
        ids = t.empty(T, dtype=t.int32, device=dev)
        za = t.empty(T, dtype=t.float32, device=dev)
        g = t.Generator(device=dev)
        for r0 in range(0, T, 1024):
            r1 = min(T, r0 + 1024)
            z = t.matmul(self.hidden[r0:r1], self.weight.t()).float()
            g.manual_seed(seed * 7_000_003 + r0)
            u = t.rand(z.shape, generator=g, device=dev).clamp_(min=1e-30).log_().neg_().log_().neg_()
            a = t.argmax(z + u, dim=1)
            ids[r0:r1] = a.to(t.int32)
            za[r0:r1] = z.gather(1, a[:, None])[:, 0]
            del z, u
        lay = W.make_layout(w, seed)
        d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
        self.params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
        ws_adv = R.new_workspace(0, 0, device=dev)
        self.adv, self.coef, _, tt = R.rl_group_advantages(d(lay.group_offsets), d(lay.rewards),
                                                           d(lay.traj_offsets), d(lay.mask), self.params, ws_adv)
        self.token_traj = tt[:T].contiguous()
        self.mask = d(lay.mask[:T])
        self.ids = ids
        h2 = self.hidden.float().pow(2).sum(dim=1) * (w.weight_std ** 2)
        logp_hat = (za - (math.log(self.V) + h2 / 2)).cpu().numpy()
        self.old = d(W.old_logp_from(logp_hat, w, seed))
        self.ws = R.new_workspace(T, self.V, self.D, device=dev)
        self.loss = t.zeros(1, dtype=t.float64, device=dev)
        self.dW = t.zeros((self.V, self.D), dtype=t.float32, device=dev)
        self.dH = t.empty((T, self.D), dtype=t.bfloat16, device=dev)
        self.trained = int(lay.mask[:T].sum())
        self.logp = t.empty(T, dtype=t.float32, device=dev)
        self.ent = t.empty(T, dtype=t.float32, device=dev)

    def call(self, R):
        R.rl_fused_head_loss_fwd_bwd(self.hidden, self.weight, self.ids, self.mask, self.token_traj, self.adv,
                                     self.coef, self.old, self.params, self.ws, self.loss, self.dW, d_hidden=self.dH)

    def call_logprobs(self, R):
        R.rl_fused_head_token_logprobs(self.hidden, self.weight, self.ids, self.ws, logp_out=self.logp,
                                       entropy_out=self.ent)


def _time_graph(torch, fn, reps, replays=5):
    """Average device time of one fn() call: reps calls captured in a CUDA graph, replayed."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(3):
            fn()
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for _ in range(reps):
            fn()
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(replays):
        g.replay()
    b.record()
    b.synchronize()
    return a.elapsed_time(b) / (replays * reps)


def _time_calls(torch, fn, warmup, reps):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        fn()
    b.record()
    b.synchronize()
    return a.elapsed_time(b) / reps


class HeadSample:
    """The first tokens of the fused-head workload (hidden rows, the whole W, ids) on the host for
    the CPU oracle; old_logp as the device workload draws it (from a torch matmul of the set-up,
    not from the library), the advantages and coefficients from the oracle."""

    def __init__(self, torch, hb, n):
        t = torch
        self.n = n
        self.hidden = hb.hidden[:n].view(t.int16).cpu().numpy().view(np.uint16)
        self.weight = hb.weight.view(t.int16).cpu().numpy().view(np.uint16)
        self.ids = hb.ids[:n].cpu().numpy()
        self.old = hb.old[:n].cpu().numpy().astype(np.float64)
        self.layout = W.make_layout(HEAD, 0)


def time_oracle_head(hs: HeadSample):
    """The float64 oracle of the fused head (Z = H W^T, the objective, dH = dZ W, dW = dZ^T H)
    over the sample's tokens at the full D and V, once, in this process (numpy's BLAS threads)."""
    import oracle.grpo_objective as O

    adv, coef, mask, tt = _oracle_layout_inputs(HEAD, hs.layout, np.arange(hs.n))
    t0 = time.perf_counter()
    O.fused_head_loss_fwd_bwd(hs.hidden, hs.weight, hs.ids, mask, tt, adv, coef, hs.old, O.LossParams())
    dt = time.perf_counter() - t0
    V, D = hs.weight.shape
    return {"rows": hs.n, "seconds": dt, "tokens_per_s": hs.n / dt, "flops": 6.0 * hs.n * D * V,
            "threads": f"numpy BLAS, {len(os.sched_getaffinity(0))} host cores",
            "sample": f"the first {hs.n} tokens of the fused-head workload at full D = {D} and V = {V} "
                      "(W decoded to float64, Z, the objective, dH and dW in float64), from the device inputs"}


def time_head(torch, R, dev, warmup=2, reps=5, oracle_tokens=0):
    hb = HeadBatch(torch, R, dev)
    hs = HeadSample(torch, hb, oracle_tokens) if oracle_tokens else None
    ms = _time_calls(torch, lambda: hb.call(R), warmup, reps)
    ms_fwd = _time_calls(torch, lambda: hb.call_logprobs(R), warmup, reps)
    st, word = R.rl_query_status(hb.ws)
    if word != 0:
        raise RuntimeError(f"device status word {word} after the fused-head timing")
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    burst, sustained, kind = 1900.0, 1700.0, "fallback"
    if os.path.exists(p):
        with open(p) as f:
            pk = json.load(f)
        burst, sustained, kind = float(pk["bf16_tflops"]), float(pk["bf16_tflops_sustained"]), "measured"
    flops = 6.0 * hb.T * hb.D * hb.V
    tf = flops / (ms * 1e-3) / 1e12
    chunks = (hb.T + 4095) // 4096
    tf_fwd = 2.0 * hb.T * hb.D * hb.V / (ms_fwd * 1e-3) / 1e12
    fwd = {"ms_per_call": ms_fwd, "tokens_per_s": hb.T / (ms_fwd * 1e-3), "achieved": tf_fwd, "frac": tf_fwd / burst,
           "frac_of_sustained": tf_fwd / sustained, "algorithmic_flops_per_call": 2.0 * hb.T * hb.D * hb.V,
           "note": "rl_fused_head_token_logprobs with entropy: one tensor-core pass (2 T D V) and the merge"}
    return {"workload": f"fusedhead: hidden bf16 [{hb.T} x {hb.D}] N(0,1), W bf16 [{hb.V} x {hb.D}] N(0,0.02^2), "
                        f"masks and coefficients of the first {hb.T} multiturn tokens ({hb.trained} trained)",
            "ms_per_call": ms, "tokens_per_s": hb.T / (ms * 1e-3), "bound": "tensor", "achieved": tf,
            "peak": burst, "unit": "TFLOP/s", "frac": tf / burst, "frac_of_sustained": tf / sustained,
            "peak_source": kind, "algorithmic_flops_per_call": flops, "executed_flops_per_call": flops,
            "reps": reps, "chunks_per_call": chunks,
            "note": "6 T D V (Z once, dH, dW), all on hand-written tcgen05 kernels (head_kernel: logits tiles and "
                    "softmax partials; head_grad_kernel: dH and dW in one launch), smallest workspace "
                    f"({hb.ws.numel() / 1e9:.2f} GB: one 4,096-token chunk of the logits gradient)",
            "logprobs": fwd}, hs


def profile_head(T):
    """A small fused-head case for profiler captures: three loss calls, then three forward-only
    log-prob calls, on the first T tokens."""
    import torch

    from paper_2608_16798_gb300 import build as B

    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    dev = torch.device("cuda", 0)
    hb = HeadBatch(torch, R, dev, T=T)
    for _ in range(3):
        hb.call(R)
    for _ in range(3):
        hb.call_logprobs(R)
    st, word = R.rl_query_status(hb.ws)
    print(json.dumps({"profile_head_tokens": T, "status": word, "flops_per_call": 6.0 * T * hb.D * hb.V}))
    return 0 if word == 0 else 1


def profile_case(rows, workload="multiturn"):
    """A small slice of a workload for profiler captures: the first `rows` packed tokens
    (logits resident on the device), then three rl_policy_loss_fwd_bwd launches (with the
    workload's entropy and KL terms) and three rl_token_logprobs launches."""
    import torch

    from paper_2608_16798_gb300 import build as B

    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    dev = torch.device("cuda", 0)
    w = W.WORKLOADS[workload]
    lay = W.make_layout(w, 0)
    rows = min(rows, lay.n_tokens)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    logits = torch.empty((rows, w.vocab), dtype=dt, device=dev)
    W.logits_rows_torch(w, 0, 0, rows, logits)
    ids = W.sample_tokens_torch(logits, 0, 0, w)
    d = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, w.kl_coef, 3 if w.kl_coef else 0, w.entropy_coef,
                           0.0, 1e-6, 0)
    ws = R.new_workspace(rows, w.vocab, device=dev)
    adv, coef, n_tok, tt = R.rl_group_advantages(d(lay.group_offsets), d(lay.rewards), d(lay.traj_offsets),
                                                 d(lay.mask), params, ws, traj_valid=d(lay.traj_valid))
    logp, _, _ = R.rl_token_logprobs(logits, ids, ws)
    lp = logp.cpu().numpy()
    old = d(W.old_logp_from(lp, w, 0))
    ref = d(W.ref_logp_from(lp, w, 0)) if w.ref_noise_std else None
    grad = torch.empty_like(logits)
    loss = torch.zeros(1, dtype=torch.float64, device=dev)
    mask = d(lay.mask[:rows])
    for _ in range(3):
        R.rl_policy_loss_fwd_bwd(logits, ids, mask, tt[:rows], adv, coef, old, params, ws, loss, grad_out=grad,
                                 ref_logp=ref)
    for _ in range(3):
        R.rl_token_logprobs(logits, ids, ws, logp_out=logp)
    st, word = R.rl_query_status(ws)
    m = lay.mask[:rows].astype(np.int64)
    es = 2 if w.dtype == "bf16" else 4
    trained = m * (coef.cpu().numpy()[tt[:rows].cpu().numpy()] != 0)
    print(json.dumps({"profile_case_rows": rows, "workload": workload, "trained_rows": int(trained.sum()),
                      "status": word, "algorithmic_bytes_fwd_bwd": int(((trained + 1) * w.vocab * es).sum()),
                      "algorithmic_bytes_fwd": rows * w.vocab * es}))
    return 0 if word == 0 else 1


def profile_segments(reps=3):
    """The segmented reductions alone, for profiler captures (a few MB on the device): `reps`
    calls of rl_group_advantages (count_adv_kernel, coef_kernel) on the multi-turn batch's layout
    and on the edge workload's (16,384 trajectories in 4,096 groups), then on the tree workload's
    packed stream rl_group_advantages_by_owner (the same kernels, counting by owner),
    rl_sequence_is_weights (owner_logratio_kernel,
    seq_weight_kernel; log-probs N(-2, 1) per token, rollout = old + N(0, 0.02^2)), the same with
    per-token advantages scaled in place (token_scale_kernel) and rl_rollout_value_advantages
    (rollout_adv_kernel; values N(0, 1) per token); and rl_token_stats_summary over the multi-turn
    batch's rows (stats_summary_kernel; per-token statistics uniform on [0, 1))."""
    import torch

    from paper_2608_16798_gb300 import build as B

    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    dev = torch.device("cuda", 0)
    t = torch
    d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    lay = W.make_layout(WORKLOAD, 0)
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 0)
    ws = R.new_workspace(0, 0, device=dev)
    go, rw, to, mask, valid = (d(lay.group_offsets), d(lay.rewards), d(lay.traj_offsets), d(lay.mask),
                               d(lay.traj_valid))
    for _ in range(reps):
        _, coef, _, tt = R.rl_group_advantages(go, rw, to, mask, params, ws, traj_valid=valid)
    el = W.make_layout(W.WORKLOADS["edge"], 0)
    eargs = (d(el.group_offsets), d(el.rewards), d(el.traj_offsets), d(el.mask), params, ws)
    for _ in range(reps):
        R.rl_group_advantages(*eargs, traj_valid=d(el.traj_valid))
    stats = d(np.random.default_rng(2).random(lay.n_tokens * 5, dtype=np.float32))
    for _ in range(reps):
        R.rl_token_stats_summary(stats, mask, tt, coef, ws)
    w = W.WORKLOADS["tree"]
    prompts, calls, aux = W.tree_rollouts(w, seed=0)
    out = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves, n_threads=4)
    n = len(prompts)
    owner, tmask = d(out["owner"]), d(out["mask"])
    T = len(out["tokens"])
    tgo = d(np.arange(0, n + 1, w.group_size, dtype=np.int32))
    trw = d((np.random.default_rng(0).random(n) < w.reward_p).astype(np.float32))
    tvalid = d(np.array([st["valid"] for st in out["stats"]], np.uint8))
    old_h = np.random.default_rng(1).normal(-2.0, 1.0, T).astype(np.float32)
    old, roll = d(old_h), d(W.rollout_logp_from(old_h, 0, std=0.02))
    for _ in range(reps):
        R.rl_group_advantages_by_owner(tgo, trw, owner, tmask, params, ws, traj_valid=tvalid)
    ws_tree = R.new_workspace(n, 0, device=dev)
    for _ in range(reps):
        R.rl_sequence_is_weights(owner, tmask, old, roll, n, ws_tree, cap=2.0)
    tok_adv = d(np.random.default_rng(3).normal(0.0, 1.0, T).astype(np.float32))
    for _ in range(reps):
        R.rl_sequence_is_weights(owner, tmask, old, roll, n, ws_tree, cap=2.0, token_adv_inout=tok_adv)
    values = d(np.random.default_rng(4).normal(0.0, 1.0, T).astype(np.float32))
    for _ in range(reps):
        R.rl_rollout_value_advantages(owner, tmask, values, trw, ws_tree)
    word = R.rl_query_status(ws)[1] | R.rl_query_status(ws_tree)[1]
    print(json.dumps({"profile_segments": reps, "multiturn_tokens": lay.n_tokens, "multiturn_traj": lay.n_traj,
                      "tree_tokens": T, "tree_rollouts": n, "status": word}))
    return 0 if word == 0 else 1


def profile_ppo(steps):
    """The PPO step of the benchmark on the whole multi-turn batch, `steps` times without timing
    (for a profiler's launch list): advantages and coefficients, masked GAE, then per microbatch
    the policy loss with per-token advantages and the value loss; then sequence-level weights."""
    import torch

    from paper_2608_16798_gb300 import build as B

    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    batch = DeviceBatch(torch, R, dev)
    t = torch
    d = lambda x: t.from_numpy(np.ascontiguousarray(x)).to(dev)  # noqa: E731
    values = d(W.value_predictions(WORKLOAD, 0, batch.T))
    v_new = values + 0.05
    params = R.make_params(W.CLIP_EPS_LOW, W.CLIP_EPS_HIGH, 0.0, 0, 0.0, 0.0, 1e-6, 1, token_level_adv=1)
    coef, adv_traj = t.empty_like(batch.coef), t.empty_like(batch.adv)
    adv, ret, dv = (t.empty(batch.T, dtype=t.float32, device=dev) for _ in range(3))
    loss, vloss = t.zeros(1, dtype=t.float64, device=dev), t.zeros(1, dtype=t.float64, device=dev)
    roll = d(W.rollout_logp_from(batch.old.cpu().numpy(), 0, std=0.02))
    w_seq = t.empty(batch.lay.n_traj, dtype=t.float32, device=dev)
    for _ in range(steps):
        R.rl_group_advantages(batch.group_offsets, batch.rewards, batch.traj_offsets, batch.mask, params, batch.ws,
                              traj_valid=batch.valid, adv_out=adv_traj, coef_out=coef, n_tok_out=batch.n_tok,
                              token_traj_out=batch.token_traj)
        R.rl_masked_gae(batch.traj_offsets, batch.mask, values, batch.ws, 1.0, 1.0, True,
                        traj_rewards=batch.rewards.float(), adv_out=adv, returns_out=ret)
        for lo, hi in batch.mbs:
            R.rl_policy_loss_fwd_bwd(batch.logits[lo:hi], batch.ids[lo:hi], batch.mask[lo:hi],
                                     batch.token_traj[lo:hi], adv[lo:hi], coef, batch.old[lo:hi], params, batch.ws,
                                     loss, grad_out=batch.grad[lo:hi])
            R.rl_value_loss_fwd_bwd(v_new[lo:hi], ret[lo:hi], batch.mask[lo:hi], batch.token_traj[lo:hi], coef,
                                    batch.ws, vloss, d_values=dv[lo:hi])
        R.rl_sequence_is_weights(batch.token_traj, batch.mask, batch.old, roll, batch.lay.n_traj, batch.ws, cap=2.0,
                                 weight_out=w_seq)
    st, word = R.rl_query_status(batch.ws)
    print(json.dumps({"profile_ppo_steps": steps, "tokens_per_step": batch.T, "status": word}))
    return 0 if word == 0 else 1


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="cuda", choices=["cuda", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--profile-case", type=int, default=0, metavar="ROWS",
                    help="run a small slice of the workload for a profiler capture and exit")
    ap.add_argument("--profile-workload", default="multiturn", choices=["tiny", "multiturn", "longhorizon", "edge"],
                    help="workload of --profile-case (default: the benchmark's multiturn)")
    ap.add_argument("--profile-head", type=int, default=0, metavar="TOKENS",
                    help="run a small fused-head case for a profiler capture and exit")
    ap.add_argument("--profile-segments", action="store_true",
                    help="run the segmented-reduction kernels alone (a few MB) for a profiler capture and exit")
    ap.add_argument("--profile-ppo", type=int, default=0, metavar="STEPS",
                    help="run the PPO step on the batch STEPS times for a profiler's launch list and exit")
    ap.add_argument("--no-head", action="store_true", help="skip the fused-head measurement")
    ap.add_argument("--no-ppo", action="store_true", help="skip the PPO-step measurement")
    ap.add_argument("--no-tree", action="store_true", help="skip the prefix-tree measurement")
    ap.add_argument("--no-other", action="store_true", help="skip the long-horizon and edge workloads")
    args = ap.parse_args()
    if args.profile_case:
        return profile_case(args.profile_case, args.profile_workload)
    if args.profile_head:
        return profile_head(args.profile_head)
    if args.profile_ppo:
        return profile_ppo(args.profile_ppo)
    if args.profile_segments:
        return profile_segments()
    if args.impl == "reference":
        return run_reference(args)
    args.warmup = max(3, args.warmup)

    import torch
    import torch.distributed as dist

    from paper_2608_16798_gb300 import build as B

    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    rank, world, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    R.lib()

    batch = DeviceBatch(torch, R, dev)
    n_mb = len(batch.mbs)
    for _ in range(args.warmup):
        batch.step(R)
    torch.cuda.synchronize(dev)

    # timed region: K steps, barrier + synchronize on both sides
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_mb)]
           for _ in range(args.steps)]
    props = torch.cuda.get_device_properties(dev)
    uuid = str(getattr(props, "uuid", "") or "")
    sampler = ClockSampler(("GPU-" + uuid) if uuid and not uuid.startswith("GPU-") else (uuid or str(dev.index)))
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    sampler.start()
    time.sleep(0.3)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for k in range(args.steps):
        batch.step(R, evs[k])
    t1.record()
    torch.cuda.synchronize(dev)
    clocks = sampler.stop()
    if world > 1:
        dist.barrier()
    ms = t0.elapsed_time(t1)
    kern_ms = [a.elapsed_time(b) for step in evs for (a, b) in step]
    st, word = R.rl_query_status(batch.ws)
    if word != 0:
        raise RuntimeError(f"device status word {word} after the timed region")
    ms = max_over_ranks(ms, dist if world > 1 else None, dev)
    ms_step = ms / args.steps
    value = job_throughput(batch.T, world, ms, args.steps)

    peak, peak_kind = measured_peaks()
    per_launch_bytes = sum(batch.mb_bytes) / n_mb
    avg_launch_ms = sum(kern_ms) / len(kern_ms)
    achieved = per_launch_bytes / (avg_launch_ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": profiled_traffic(), "peak_source": peak_kind,
                "kernel": "rows_kernel<bf16> via rl_policy_loss_fwd_bwd (one launch; its last cluster sums the loss)",
                "algorithmic_bytes_per_launch": per_launch_bytes, "avg_launch_ms": avg_launch_ms,
                "frac_of_nominal_8tbs": achieved / 8000.0}
    # per microbatch: median and best launch over the timed steps, and each one's GB/s
    per_mb = []
    for k in range(n_mb):
        ts = [kern_ms[s * n_mb + k] for s in range(args.steps)]
        per_mb.append({"rows": batch.mbs[k][1] - batch.mbs[k][0], "median_ms": statistics.median(ts),
                       "best_ms": min(ts), "median_gbs": batch.mb_bytes[k] / (statistics.median(ts) * 1e-3) / 1e9})
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    oracle_slices = {} if want_cpu else None  # host copies of device rows for the CPU oracle
    extras = time_logits_extras(torch, R, batch, dev, peak)
    if not args.no_other:
        extras["other_workloads"] = time_other_workloads(torch, R, dev, peak, oracle_slices=oracle_slices)
    extras["loss_batch_sum_ms"] = sum(m["median_ms"] for m in per_mb)
    extras["loss_microbatch_median_ms"] = [round(m["median_ms"], 4) for m in per_mb]

    e2e = None
    if not args.no_e2e:
        e_ms, h2d, d2h, e_loss, src, copy_gbs = e2e_run(torch, R, batch, dev, args.e2e_steps, 2)
        e2e = {"value": batch.T / (e_ms / 1e3 / args.e2e_steps) * world, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": args.e2e_steps, "repetitions": len(copy_gbs["runs"]),
               "value_of": "median of the repetitions, each `steps` timed steps", "loss": e_loss,
               "host_source": src, "h2d_gbs": copy_gbs,
               "note": "per step: metadata and every microbatch's logits from pinned host memory, loss read "
                       "back; the gradient stays in HBM for the model's backward"}

    ppo = None if args.no_ppo else time_ppo(torch, R, batch, dev)
    tree = None if args.no_tree else time_tree(torch, R, dev)

    head, head_sample = None, None
    if not args.no_head:
        head, head_sample = time_head(torch, R, dev, oracle_tokens=ORACLE_HEAD_TOKENS if want_cpu else 0)

    cpu = None
    if want_cpu:
        # the CPU oracle (float64, as it stands): the benchmark's first microbatch, then bounded
        # samples of the other workloads' device rows
        sample = OracleSample(batch.mbs[0][1] - batch.mbs[0][0], batch.logits, batch.ids)
        try:
            cpu = time_oracle(sample)
            cpu["workloads"] = {name: time_oracle_slice(sl) for name, sl in oracle_slices.items()}
            if head_sample is not None:
                try:
                    cpu["workloads"]["fusedhead"] = time_oracle_head(head_sample)
                except MemoryError as e:
                    cpu["workloads"]["fusedhead"] = {"unavailable": f"MemoryError: {e}"}
        finally:
            sample.close()
            for sl in oracle_slices.values():
                if not isinstance(sl, str):
                    sl.close()

    if rank == 0:
        summary = compact_summary(value, ms_step, roofline, extras, head, ppo, tree, cpu, e2e)
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": workload_config(batch.T, n_mb),
                "inputs_sha256": batch.inputs_sha256, "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks, "logits_path": extras, "fused_head": head, "ppo": ppo, "tree": tree,
                "gpu_launches": batch.launches_per_step() * args.steps,
                "loss_per_step": float(batch.loss.item()) / (args.warmup + args.steps),
                "summary": summary}
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
