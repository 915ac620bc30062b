"""A seeded sweep of loss-call shapes against the float64 oracle (needs a GB300).

Vocabulary sizes are drawn log-uniformly up to the largest rows the loss kernels accept
(819,200 bf16, 409,600 fp32 entries), so the sweep crosses every cluster width the launcher
picks (1 to 16 CTAs per row) and both sides of the 8 KB limit of the warp-per-row kernel;
leading dimensions are padded by 0-8 elements (16-byte aligned or not), rows are taken anywhere
in a workload's packed stream (its masks and owners), and the objective's optional terms
(entropy bonus, k3 KL, TIS) and the three aggregation modes are drawn too. The row count keeps
the oracle's work under about 8 M logits per case.
"""

import dataclasses

import numpy as np
import pytest
import torch

from parity_cases import compare, make_case, run_loss
from paper_2608_16798_gb300 import workloads as W


def _draw(n=40, seed=2026):
    """Cases 0-13: vocabularies log-uniform up to 8,192, mostly with rows on 16-byte boundaries
    (the warp-per-row kernel where a row fits in 8 KB; one-CTA clusters otherwise); cases 14-39: a cluster width C drawn from 1-16 and a
    vocabulary within that width's range (C x 40 KB of bf16 or C x 30 KB of fp32 per row), C = 16
    up to the largest rows accepted."""
    rng = np.random.default_rng(seed)
    cases = []
    for k in range(n):
        fp32 = rng.random() < 0.35
        name = "edge" if fp32 else ["tiny", "multiturn", "longhorizon"][int(rng.integers(0, 3))]
        if k < 14:
            V = int(np.exp(rng.uniform(0.0, np.log(8192))))
        else:
            span = 7680 if fp32 else 20480  # elements per CTA slice at the loss kernel's target
            C = int(rng.integers(1, 17))
            hi = (409_600 if fp32 else 819_200) if C == 16 else C * span
            V = int(rng.integers((C - 1) * span + 1, hi + 1))
        rows = int(max(1, min(48, 8_000_000 // V)))
        epv = 4 if fp32 else 8  # elements per 16 bytes
        if k < 14 and rng.random() < 0.7:  # rows on 16-byte boundaries: the warp-per-row kernel
            ld_pad = (-V) % epv + epv * int(rng.integers(0, 2))
        else:
            ld_pad = int(rng.integers(0, 9))
        agg = int(rng.integers(0, 3))
        tis = bool(rng.random() < 0.3)
        ent = 1e-2 if rng.random() < 0.3 else None
        cases.append((k, name, V, ld_pad, rows, agg, tis, ent, int(rng.integers(0, 1 << 30))))
    return cases


CASES = _draw()


@pytest.fixture(scope="module")
def R():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_16798_gb300 import build

    build.build()
    import paper_2608_16798_gb300.rl_loss as R

    R.lib()
    return R


def test_sweep_spans_the_kernel_shapes():
    """The draw covers short rows and every cluster width the launcher can pick (no GPU needed)."""
    widths = set()
    short = 0
    for _, name, V, ld_pad, *_ in CASES:
        es = 4 if name == "edge" else 2
        if V * es <= 8192 and ((V + ld_pad) * es) % 16 == 0:
            short += 1
            continue
        target = 30 * 1024 if es == 4 else 40 * 1024
        for C in range(1, 17):
            per = -(-V // C)
            slice_b = -(-per // (16 // es)) * 16
            if slice_b <= target or (C == 16 and slice_b <= 100 * 1024):
                widths.add(C)
                break
    assert short >= 5 and len(widths) >= 8, (short, sorted(widths))


@pytest.mark.gpu
@pytest.mark.parametrize("k,name,V,ld_pad,rows,agg,tis,ent,seed", CASES,
                         ids=[f"{c[0]}-{c[1]}-V{c[2]}-ld{c[3]}-r{c[4]}" for c in CASES])
def test_loss_shape_sweep(R, k, name, V, ld_pad, rows, agg, tis, ent, seed):
    n_tokens = W.make_layout(W.WORKLOADS[name], seed % 1000).n_tokens
    row0 = int(np.random.default_rng(seed).integers(0, max(1, n_tokens - rows)))
    case = make_case(name, seed=seed % 1000, row0=row0, rows=rows, vocab=V, loss_agg=agg, tis=tis)
    if ent is not None:
        case = dataclasses.replace(case, P=dataclasses.replace(case.P, entropy_coef=ent))
    out = run_loss(R, case, ld=V + ld_pad)
    compare(case, out, f"case {k}: {name} V={V} ld=V+{ld_pad} rows={rows} agg={agg} tis={tis} ent={ent}")


def _draw_head(n=12, seed=7):
    """Fused-head shapes: tokens 1-5,000 (ragged 128-row tiles, one or two 4,096-token chunks),
    hidden sizes 64-1,024 (multiples of 64), vocabularies up to 20,000 (ragged 256-wide tiles,
    up to five 4,096-wide blocks), with T D V at most 4e9 so the oracle stays quick."""
    rng = np.random.default_rng(seed)
    cases = []
    for k in range(n):
        D = 64 * int(rng.integers(1, 17))
        V = int(rng.integers(1, 20_001))
        T = int(min(rng.integers(1, 5_001), max(1, 4_000_000_000 // (D * V))))
        cases.append((k, T, D, V, int(rng.integers(0, 3)), bool(rng.random() < 0.4), bool(rng.random() < 0.3)))
    return cases


HEAD_CASES = _draw_head()


@pytest.mark.gpu
@pytest.mark.parametrize("k,T,D,V,agg,ent,tis", HEAD_CASES,
                         ids=[f"{c[0]}-T{c[1]}-D{c[2]}-V{c[3]}" for c in HEAD_CASES])
def test_fused_head_shape_sweep(R, k, T, D, V, agg, ent, tis):
    from test_gpu_fused_head import compare_head, make_head_case, run_head

    if T < 8:
        pytest.skip("the case builder cuts at least four trajectories inside the token range")
    c = make_head_case(T, D, V, seed=1000 + k, agg=agg, ent=ent, tis=tis)
    compare_head(c, run_head(R, c))


def _draw_fwd(n=16, seed=11):
    """Forward log-probs shapes: bf16 or fp32 rows up to 400,000 entries, padded leading
    dimensions, with and without the entropy and lse outputs."""
    rng = np.random.default_rng(seed)
    cases = []
    for k in range(n):
        fp32 = rng.random() < 0.4
        V = int(np.exp(rng.uniform(0.0, np.log(400_000))))
        if fp32:  # the edge workload's generator (spikes, half-masked rows) needs two entries
            V = max(V, 2)
        rows = int(max(1, min(64, 8_000_000 // V)))
        cases.append((k, "edge" if fp32 else "multiturn", V, int(rng.integers(0, 9)), rows, bool(rng.random() < 0.5),
                      int(rng.integers(0, 1 << 30))))
    return cases


FWD_CASES = _draw_fwd()


@pytest.mark.gpu
@pytest.mark.parametrize("k,name,V,ld_pad,rows,ent,seed", FWD_CASES,
                         ids=[f"{c[0]}-{c[1]}-V{c[2]}-ld{c[3]}-r{c[4]}" for c in FWD_CASES])
def test_token_logprobs_shape_sweep(R, k, name, V, ld_pad, rows, ent, seed):
    import oracle.grpo_objective as O
    from parity_cases import logits_to_dev, to_dev

    case = make_case(name, seed=seed % 1000, rows=rows, vocab=V)
    ws = R.new_workspace(case.rows, V)
    logp, H, lse = R.rl_token_logprobs(logits_to_dev(case, V + ld_pad), to_dev(case.ids), ws, want_entropy=ent,
                                       want_lse=True)
    assert R.rl_query_status(ws)[1] == 0
    lp_ref, H_ref, lse_ref = O.token_logprobs(case.raw, case.w.dtype, case.ids)
    lp, ls = logp.cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(lp - lp_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lp_ref)), np.abs(lp - lp_ref).max()
    assert np.all(np.abs(ls - lse_ref) <= 1e-5 + 2.0 ** -22 * np.abs(lse_ref)), np.abs(ls - lse_ref).max()
    if ent:
        Hd = H.cpu().numpy().astype(np.float64)
        assert np.all(np.abs(Hd - H_ref) <= 5e-5 + 2e-5 * np.abs(H_ref)), np.abs(Hd - H_ref).max()
