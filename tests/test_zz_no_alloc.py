"""The allocation-free loss entry point against the workspace entry point.

rl_policy_loss_fwd_bwd_noalloc serves callers that cannot allocate device
memory (a memory pool that forbids cudaMalloc during a step, a plugin handed
only pointers): it runs the same computation on a built-in device array. Two
calls in a row must each agree with rl_policy_loss_fwd_bwd on the same inputs,
so nothing left in the shared array from one call leaks into the next. This
file is collected last so that a stop-at-first-failure run has run everything
else first.
"""

import ctypes

import numpy as np
import pytest
import torch

from parity_cases import check_grad, cuda_params, grad_to_np, logits_to_dev, make_case, to_dev

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


def test_no_alloc_matches_workspace_entry_point_twice(R):
    cases = [make_case("longhorizon", seed=11, row0=4000, rows=96, loss_agg=2),
             make_case("tiny", seed=12, rows=300, loss_agg=0)]
    for k, case in enumerate(cases):
        logits = logits_to_dev(case)
        inp = _inputs(case)
        l_ws, g_ws, s_ws = _with_workspace(R, case, logits, inp)
        l_na, g_na, s_na = _no_alloc(R, case, logits, inp)
        scale = max(abs(l_ws), 1e-30)
        assert abs(l_na - l_ws) <= 1e-4 * scale, (k, l_na, l_ws)
        check_grad(g_na, g_ws, case.w.dtype, f"call {k}", absolute=case.P.loss_agg != 2)
        assert np.allclose(s_na, s_ws, rtol=1e-6, atol=1e-7)


def test_no_alloc_rejects_rows_beyond_its_limit(R):
    # returns during argument checks, before any launch or memory access
    st = R.lib().rl_policy_loss_fwd_bwd_noalloc(ctypes.c_void_p(0x10000), R.RL_BF16, 131073, 8, 8,
                                                *([ctypes.c_void_p(0x10000)] * 3), 1,
                                                *([ctypes.c_void_p(0x10000)] * 3), None, None,
                                                ctypes.byref(R.make_params()), ctypes.c_void_p(0x10000),
                                                ctypes.c_void_p(0x10000), None, None, None)
    assert st == 2
    assert "131072" in R.rl_last_error_message()
