"""The failure path of the kernels' waits, exercised without a fault: a bounded wait on an
mbarrier that nothing completes runs out after its limit, the status word reports
RL_DEV_TIMEOUT (rl_query_status: RL_ERR_TIMEOUT), and the same context then computes a correct
loss after rl_workspace_init clears the word."""

import time

import pytest
import torch

from parity_cases import make_case
from test_gpu_parity import compare, run_loss

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


def test_bounded_wait_runs_out_and_the_context_survives(R):
    ws = R.new_workspace(512, 4096)
    waited = torch.zeros(1, dtype=torch.int64, device="cuda")
    limit = 50_000_000  # 50 ms per wait, two waits
    t0 = time.perf_counter()
    R.rl_selftest_bounded_wait(ws, limit, waited)
    st, word = R.rl_query_status(ws)
    dt = time.perf_counter() - t0
    assert st == 7 and word & R.RL_DEV_TIMEOUT  # RL_ERR_TIMEOUT
    w = int(waited.item())
    assert 2 * limit <= w < 2 * limit + 50_000_000, w  # both waits ran to their limit, no longer
    assert dt < 5.0
    # the context is intact: clear the word and run a loss against the oracle
    R.rl_workspace_init(ws)
    case = make_case("tiny", seed=3)
    out = run_loss(R, case, ws=ws)
    compare(case, out, "loss after the timeout")
