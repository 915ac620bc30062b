"""The allocation-free loss entry point against the workspace entry point.

rl_policy_loss_fwd_bwd_noalloc serves callers that cannot allocate device
memory (a memory pool that forbids cudaMalloc during a step, a plugin handed
only pointers): it runs the same computation on a built-in device array. Two
calls in a row must each agree with rl_policy_loss_fwd_bwd on the same inputs,
so nothing left in the shared array from one call leaks into the next. Both run
the same kernel on the same inputs, so they must agree bit for bit. This file is
collected last so that a stop-at-first-failure run has run everything else first.
"""

import ctypes

import numpy as np
import pytest
import torch

from parity_cases import check_grad, check_loss, cuda_params, grad_to_np, logits_to_dev, make_case, oracle_loss, to_dev

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


def _inputs(case):
    return dict(token_ids=to_dev(case.ids), mask=to_dev(case.mask), token_traj=to_dev(case.tt.astype(np.int32)),
                adv=to_dev(case.adv64.astype(np.float32)), coef=to_dev(case.coef64.astype(np.float32)),
                old_logp=to_dev(case.old), ref_logp=None if case.ref is None else to_dev(case.ref))


def _with_workspace(R, case, logits, inp):
    ws = R.new_workspace(case.rows, case.raw.shape[1])
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(case.rows * 5, dtype=torch.float32, device="cuda")
    g = R.rl_policy_loss_fwd_bwd(logits, inp["token_ids"], inp["mask"], inp["token_traj"], inp["adv"], inp["coef"],
                                 inp["old_logp"], cuda_params(R, case.P), ws, loss, ref_logp=inp["ref_logp"],
                                 token_stats=st)
    assert R.rl_query_status(ws)[1] == 0
    return loss.item(), grad_to_np(g), st.cpu().numpy()


def _no_alloc(R, case, logits, inp):
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(case.rows * 5, dtype=torch.float32, device="cuda")
    grad = torch.empty_like(logits)
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    R.rl_policy_loss_fwd_bwd_noalloc(logits, inp["token_ids"], inp["mask"], inp["token_traj"], inp["adv"],
                                     inp["coef"], inp["old_logp"], cuda_params(R, case.P), loss, grad,
                                     ref_logp=inp["ref_logp"], token_stats=st, device_status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    return loss.item(), grad_to_np(grad), st.cpu().numpy()


def _same(a, b, what):
    """Both entry points run the same kernel on the same inputs: the results agree bit for bit
    (loss, gradient and per-token statistics)."""
    (l_a, g_a, s_a), (l_b, g_b, s_b) = a, b
    assert l_a == l_b, f"{what}: loss {l_a!r} vs {l_b!r}"
    assert np.array_equal(g_a, g_b), f"{what}: gradients differ"
    assert np.array_equal(s_a, s_b), f"{what}: statistics differ"


def test_no_alloc_matches_workspace_entry_point_twice(R):
    cases = [make_case("longhorizon", seed=11, row0=4000, rows=96, loss_agg=2),
             make_case("tiny", seed=12, rows=300, loss_agg=0)]
    for k, case in enumerate(cases):
        logits = logits_to_dev(case)
        inp = _inputs(case)
        ref = _with_workspace(R, case, logits, inp)
        _same(_no_alloc(R, case, logits, inp), ref, f"call {k}")
        # and both are at parity with the oracle
        l_o, g_o, _, contrib = oracle_loss(case)
        check_loss(ref[0], l_o, contrib, f"call {k}")
        check_grad(ref[1], g_o, case.w.dtype, f"call {k}", absolute=case.P.loss_agg != 2)


def test_no_alloc_at_its_row_limit(R):
    """131,072 rows, the largest microbatch the built-in array holds (small vocabulary)."""
    case = make_case("edge", seed=13, vocab=64, loss_agg=0)
    assert case.rows == 131072
    logits = logits_to_dev(case)
    inp = _inputs(case)
    _same(_no_alloc(R, case, logits, inp), _with_workspace(R, case, logits, inp), "131072 rows")


def test_no_alloc_after_a_flagged_call_and_after_overlapping_calls(R):
    """A call whose status word was set (a token id outside [0, V)) and two calls that overlap on
    two streams (a documented race on the shared array: their losses are not checked) leave
    nothing behind: the next call, on its own, gives the workspace entry point's results and a
    clean status word."""
    case = make_case("tiny", seed=14, rows=512, loss_agg=0)
    logits = logits_to_dev(case)
    inp = _inputs(case)
    ref = _with_workspace(R, case, logits, inp)

    bad = dict(inp)
    ids = case.ids.copy()
    ids[[3, 100]] = [case.raw.shape[1], -1]
    bad["token_ids"] = to_dev(ids)
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    R.rl_policy_loss_fwd_bwd_noalloc(logits, bad["token_ids"], inp["mask"], inp["token_traj"], inp["adv"],
                                     inp["coef"], inp["old_logp"], cuda_params(R, case.P),
                                     torch.zeros(1, dtype=torch.float64, device="cuda"), torch.empty_like(logits),
                                     device_status=status)
    torch.cuda.synchronize()
    assert status.item() == R.RL_DEV_BAD_TOKEN
    _same(_no_alloc(R, case, logits, inp), ref, "after a flagged call")

    big = make_case("edge", seed=15, vocab=256, loss_agg=0)
    big_logits = logits_to_dev(big)
    big_inp = _inputs(big)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    outs = [(torch.zeros(1, dtype=torch.float64, device="cuda"), torch.empty_like(big_logits)) for _ in streams]
    torch.cuda.synchronize()
    for s, (loss, grad) in zip(streams, outs):
        with torch.cuda.stream(s):
            R.rl_policy_loss_fwd_bwd_noalloc(big_logits, big_inp["token_ids"], big_inp["mask"],
                                             big_inp["token_traj"], big_inp["adv"], big_inp["coef"],
                                             big_inp["old_logp"], cuda_params(R, big.P), loss, grad)
    torch.cuda.synchronize()
    _same(_no_alloc(R, case, logits, inp), ref, "after overlapping calls")


def test_no_alloc_rejects_rows_beyond_its_limit(R):
    # returns during argument checks, before any launch or memory access
    st = R.lib().rl_policy_loss_fwd_bwd_noalloc(ctypes.c_void_p(0x10000), R.RL_BF16, 131073, 8, 8,
                                                *([ctypes.c_void_p(0x10000)] * 3), 1,
                                                *([ctypes.c_void_p(0x10000)] * 3), None, None,
                                                ctypes.byref(R.make_params()), ctypes.c_void_p(0x10000),
                                                ctypes.c_void_p(0x10000), None, None, None)
    assert st == 2
    assert "131072" in R.rl_last_error_message()
