"""The entry points inside CUDA graphs and on concurrent streams.

Every entry point enqueues work on the caller's stream and allocates nothing, so a whole
step (advantages, then the loss over the microbatches; the fused head with its tensor-core
backward products and their work counter) can be captured once and replayed; replays give the eager results bit for bit
(the reductions have a fixed order). Host threads calling the library on their own streams
with their own workspaces get the same bits as serial calls.
"""

import threading

import numpy as np
import pytest
import torch

from parity_cases import cuda_params, logits_to_dev, make_case, to_dev
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


def _step_inputs(R, seed=0):
    case = make_case("multiturn", seed=seed, row0=0, rows=3000, vocab=8192)
    lay = case.layout
    d = {k: to_dev(v) for k, v in dict(go=lay.group_offsets, rw=lay.rewards, to=lay.traj_offsets,
                                       mask=lay.mask[:case.rows], full_mask=lay.mask, ids=case.ids,
                                       old=case.old).items()}
    d["logits"] = logits_to_dev(case)
    return case, d


def _step(R, case, d, ws, out):
    """Advantages over the batch layout, then the loss over three microbatches of the rows, all
    on torch's current stream (the binding's default)."""
    P = cuda_params(R, case.P)
    R.rl_group_advantages(d["go"], d["rw"], d["to"], d["full_mask"], P, ws, adv_out=out["adv"],
                          coef_out=out["coef"], n_tok_out=out["ntok"], token_traj_out=out["tt"])
    out["loss"].zero_()
    for lo, hi in ((0, 1000), (1000, 2100), (2100, case.rows)):
        R.rl_policy_loss_fwd_bwd(d["logits"][lo:hi], d["ids"][lo:hi], d["mask"][lo:hi], out["tt"][lo:hi], out["adv"],
                                 out["coef"], d["old"][lo:hi], P, ws, out["loss"], grad_out=out["grad"][lo:hi])


def _buffers(case, d):
    n, T = case.layout.n_traj, case.layout.n_tokens
    return dict(adv=torch.empty(n, device="cuda"), coef=torch.empty(n, device="cuda"),
                ntok=torch.empty(n, dtype=torch.int32, device="cuda"), tt=torch.empty(T, dtype=torch.int32, device="cuda"),
                loss=torch.zeros(1, dtype=torch.float64, device="cuda"), grad=torch.empty_like(d["logits"]))


def test_graph_capture_of_a_step(R):
    case, d = _step_inputs(R)
    ws = R.new_workspace(case.layout.n_tokens, case.raw.shape[1])
    eager = _buffers(case, d)
    _step(R, case, d, ws, eager)
    torch.cuda.synchronize()
    assert R.rl_query_status(ws)[1] == 0
    graphed = _buffers(case, d)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        _step(R, case, d, ws, graphed)  # warm-up on a side stream before the capture
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        _step(R, case, d, ws, graphed)
    for _ in range(3):
        graphed["grad"].fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert graphed["loss"].item() == eager["loss"].item()
        assert torch.equal(graphed["grad"], eager["grad"])
        assert torch.equal(graphed["adv"], eager["adv"]) and torch.equal(graphed["coef"], eager["coef"])
    assert R.rl_query_status(ws)[1] == 0


def test_graph_capture_of_the_fused_head(R):
    T, D, V = 512, 128, 3000
    rng = np.random.default_rng(4)
    hid = to_dev(W.bf16_bits_from_f32(rng.normal(0, 1, (T, D)).astype(np.float32)).view(np.int16)).view(torch.bfloat16)
    wgt = to_dev(W.bf16_bits_from_f32(rng.normal(0, 0.05, (V, D)).astype(np.float32)).view(np.int16)).view(torch.bfloat16)
    ids = to_dev(rng.integers(0, V, T).astype(np.int32))
    mask = to_dev((rng.random(T) < 0.7).astype(np.uint8))
    tt = to_dev((np.arange(T) // 64).astype(np.int32))
    adv = to_dev(rng.normal(0, 1, 8).astype(np.float32))
    coef = to_dev(np.full(8, 1e-3, np.float32))
    old = to_dev(rng.normal(-8, 0.5, T).astype(np.float32))
    P = R.make_params()
    ws = R.new_workspace(T, V, D)

    def call(loss, dW, dH):
        loss.zero_()
        dW.zero_()
        R.rl_fused_head_loss_fwd_bwd(hid, wgt, ids, mask, tt, adv, coef, old, P, ws, loss, dW, d_hidden=dH)

    e = (torch.zeros(1, dtype=torch.float64, device="cuda"), torch.zeros((V, D), device="cuda"),
         torch.empty((T, D), dtype=torch.bfloat16, device="cuda"))
    call(*e)
    torch.cuda.synchronize()
    gb = (torch.zeros(1, dtype=torch.float64, device="cuda"), torch.zeros((V, D), device="cuda"),
          torch.empty((T, D), dtype=torch.bfloat16, device="cuda"))
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        call(*gb)
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call(*gb)
    g.replay()
    torch.cuda.synchronize()
    assert gb[0].item() == e[0].item()
    assert torch.equal(gb[1], e[1]) and torch.equal(gb[2], e[2])
    assert R.rl_query_status(ws)[1] == 0


def test_concurrent_streams_and_threads(R):
    """Two host threads, each with its own stream and workspace, run steps on different inputs
    at the same time; the results equal the serial ones bit for bit."""
    inputs = [_step_inputs(R, seed) for seed in (1, 2)]
    serial = []
    for case, d in inputs:
        ws = R.new_workspace(case.layout.n_tokens, case.raw.shape[1])
        out = _buffers(case, d)
        _step(R, case, d, ws, out)
        torch.cuda.synchronize()
        serial.append((out["loss"].item(), out["grad"].clone()))
    results, errors = [None, None], []

    def worker(k):
        try:
            case, d = inputs[k]
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.default_stream())
            with torch.cuda.stream(s):
                ws = R.new_workspace(case.layout.n_tokens, case.raw.shape[1])
                out = _buffers(case, d)
                for _ in range(5):
                    _step(R, case, d, ws, out)
                word = R.rl_query_status(ws)[1]
                results[k] = (out["loss"].item(), out["grad"].clone(), word)
        except Exception as exc:  # reported on the main thread
            errors.append(exc)

    threads = [threading.Thread(target=worker, args=(k,)) for k in range(2)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    assert not errors, errors
    for k in range(2):
        loss, grad, word = results[k]
        assert word == 0
        assert loss == serial[k][0]
        assert torch.equal(grad, serial[k][1])
