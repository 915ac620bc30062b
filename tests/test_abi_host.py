"""Host-only checks of the C ABI: the library builds and loads, exports every
function that include/rl_loss.h declares, and rejects bad arguments before
launching anything (no GPU needed: every call here returns during argument
validation, before the first CUDA runtime call)."""

import ctypes
import os
import re

import pytest

from paper_2608_16798_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")]


@pytest.fixture(scope="module")
def R():
    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    R.lib()
    return R


def declared_functions():
    names = []
    for h in HEADERS:
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        names += re.findall(r"\b(rl_[a-z0-9_]+)\s*\(", src)
    return sorted(set(names))


def test_header_declares_the_four_path_functions():
    names = declared_functions()
    for f in ("rl_group_advantages", "rl_token_logprobs", "rl_policy_loss_fwd_bwd"):
        assert f in names


def test_every_declared_function_is_exported(R):
    handle = ctypes.CDLL(R.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(handle, n)]
    assert not missing, missing
    # and the binding knows each of them
    assert set(declared_functions()) <= set(R.EXPORTS)


def test_version_and_workspace_size(R):
    assert R.rl_version() >= 10000
    assert R.rl_workspace_size(0, 0) == 256
    assert R.rl_workspace_size(16384, 151936) == 256 + 16384 * 8
    assert R.rl_workspace_size(3, 10) == 256 + 256


def test_fused_head_workspace_is_one_chunk_of_logits_gradient(R):
    """The smallest fused-head workspace holds the bf16 logits gradient of one 4,096-token
    chunk, not of all T tokens: at 32,768 x 151,936 x 4,096 it stays near 1.24 GB (plus the
    per-token and per-tile buffers) while the logits of all tokens would take 9.96 GB. Each
    further chunk of a grouped workspace costs exactly one chunk's bf16 gradient."""
    T, V, D = 32768, 151936, 4096
    chunk_dz = 4096 * V * 2  # V is a multiple of 8
    minimum = R.rl_workspace_size(T, V, D)
    assert chunk_dz <= minimum < chunk_dz + 200 * 2**20
    assert minimum < T * V * 2 / 7
    assert R.rl_fused_head_workspace_size(T, V, D, 0) == minimum
    assert R.rl_fused_head_workspace_size(T, V, D, 4096) == minimum
    assert R.rl_fused_head_workspace_size(T, V, D, 4097) == minimum + chunk_dz
    assert R.rl_fused_head_workspace_size(T, V, D, T) == minimum + 7 * chunk_dz
    # a group never exceeds the call's chunks
    assert R.rl_fused_head_workspace_size(T, V, D, 10 * T) == minimum + 7 * chunk_dz
    assert R.rl_fused_head_workspace_size(100, 1000, 64, 10**6) == R.rl_workspace_size(100, 1000, 64)


FAKE = 0x10000  # never dereferenced: every call below fails validation first
PARAMS = None


def _params(R, **kw):
    return ctypes.byref(R.make_params(**kw))


def _loss(R, **over):
    L = R.lib()
    a = dict(logits=FAKE, dt=R.RL_BF16, rows=4, V=8, ld=8, ids=FAKE, mask=FAKE, tt=FAKE, n_traj=2, adv=FAKE,
             coef=FAKE, old=FAKE, ref=None, roll=None, params=_params(R), grad=FAKE, loss=FAKE, stats=None,
             ws=FAKE, ws_bytes=1 << 20, stream=None)
    a.update(over)
    return L.rl_policy_loss_fwd_bwd(a["logits"], a["dt"], a["rows"], a["V"], a["ld"], a["ids"], a["mask"], a["tt"],
                                    a["n_traj"], a["adv"], a["coef"], a["old"], a["ref"], a["roll"], a["params"],
                                    a["grad"], a["loss"], a["stats"], a["ws"], a["ws_bytes"], a["stream"])


def test_policy_loss_argument_checks(R):
    assert _loss(R, dt=7) == 1
    assert _loss(R, rows=-1) == 1
    assert _loss(R, V=0) == 1
    assert _loss(R, ld=7) == 1
    assert _loss(R, ws=None) == 1
    assert _loss(R, ws_bytes=100) == 4
    assert _loss(R, logits=FAKE + 2) == 3
    assert _loss(R, grad=FAKE + 8) == 3
    assert _loss(R, ws=FAKE + 4) == 3
    assert _loss(R, params=None) == 1
    assert _loss(R, params=_params(R, kl_estimator=2)) == 2
    assert _loss(R, params=_params(R, clip_eps_low=-0.1)) == 1
    assert _loss(R, loss=None) == 1
    assert _loss(R, ids=None) == 1
    assert _loss(R, n_traj=-1) == 1
    assert _loss(R, V=10_000_000, ld=10_000_000) == 2  # row larger than 16 CTAs x 100 KB
    assert "rl_policy_loss_fwd_bwd" in R.rl_last_error_message()
    assert _loss(R, rows=0) == 0      # nothing to do: returns before any launch


def test_largest_vocabulary_rows(R):
    """A row is spread over at most 16 CTAs of 100 KB: up to 819,200 bf16 or 409,600 fp32 entries
    pass the shape checks (these calls then stop at the NULL params, before any launch); one
    more entry is unsupported."""
    assert _loss(R, V=819_200, ld=819_200, params=None) == 1
    assert _loss(R, V=819_201, ld=819_201, params=None) == 2
    assert _loss(R, dt=R.RL_F32, V=409_600, ld=409_600, params=None) == 1
    assert _loss(R, dt=R.RL_F32, V=409_601, ld=409_601, params=None) == 2
    assert "16 x 100 KB" in R.rl_last_error_message()


def test_token_logprobs_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(logits=FAKE, dt=R.RL_F32, rows=4, V=8, ld=8, ids=FAKE, logp=FAKE, ent=None, lse=None, ws=FAKE,
                 ws_bytes=1 << 20, stream=None)
        a.update(over)
        return L.rl_token_logprobs(a["logits"], a["dt"], a["rows"], a["V"], a["ld"], a["ids"], a["logp"], a["ent"],
                                   a["lse"], a["ws"], a["ws_bytes"], a["stream"])

    assert call(dt=3) == 1
    assert call(ld=4) == 1
    assert call(logp=None) == 1
    assert call(logits=FAKE + 4) == 3
    assert call(ws_bytes=8) == 4
    assert call(rows=0) == 0


def test_group_advantages_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(n=4, g=1, go=FAKE, rw=FAKE, valid=None, T=16, to=FAKE, mask=FAKE, params=_params(R), adv=FAKE,
                 coef=FAKE, ntok=FAKE, tt=None, ws=FAKE, ws_bytes=1024, stream=None)
        a.update(over)
        return L.rl_group_advantages(a["n"], a["g"], a["go"], a["rw"], a["valid"], a["T"], a["to"], a["mask"],
                                     a["params"], a["adv"], a["coef"], a["ntok"], a["tt"], a["ws"], a["ws_bytes"],
                                     a["stream"])

    assert call(n=-1) == 1
    assert call(params=None) == 1
    assert call(params=_params(R, loss_agg=5)) == 1
    assert call(params=_params(R, adv_eps=-1.0)) == 1
    assert call(ws_bytes=16) == 4
    assert call(rw=None) == 1
    assert call(mask=None) == 1
    assert call(n=0) == 0


def test_selftest_bounded_wait_argument_checks(R):
    L = R.lib()
    assert L.rl_selftest_bounded_wait(None, 1 << 20, 1_000_000, None, None) == 1
    assert L.rl_selftest_bounded_wait(FAKE, 100, 1_000_000, None, None) == 4
    assert L.rl_selftest_bounded_wait(FAKE + 8, 1 << 20, 1_000_000, None, None) == 3
    assert L.rl_selftest_bounded_wait(FAKE, 1 << 20, 999, None, None) == 1
    assert L.rl_selftest_bounded_wait(FAKE, 1 << 20, 2_000_000_001, None, None) == 1
    assert "limit_ns" in R.rl_last_error_message()


def test_status_and_init_argument_checks(R):
    L = R.lib()
    assert L.rl_workspace_init(None, 1024, None) == 1
    assert L.rl_workspace_init(FAKE, 16, None) == 4
    word = ctypes.c_int32(0)
    assert L.rl_query_status(None, None, ctypes.byref(word)) == 1


def test_fused_head_logprobs_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(h=FAKE, w=FAKE, T=4, D=128, V=1000, ids=FAKE, logp=FAKE, ent=None, lse=None, ws=FAKE,
                 ws_bytes=1 << 20, stream=None)
        a.update(over)
        return L.rl_fused_head_token_logprobs(a["h"], a["w"], a["T"], a["D"], a["V"], a["ids"], a["logp"], a["ent"],
                                              a["lse"], a["ws"], a["ws_bytes"], a["stream"])

    assert call(T=-1) == 1
    assert call(D=32) == 1
    assert call(D=96) == 2
    assert call(V=0) == 1
    assert call(ws=None) == 1
    assert call(ws_bytes=300) == 4
    assert call(logp=None) == 1
    assert call(h=FAKE + 2) == 3
    assert call(ws=FAKE + 8) == 3
    assert call(T=0) == 0
    # rl_workspace_size(T, V, D) always suffices; one chunk of partials (two per token and
    # 4,096-entry vocabulary block) is the minimum (logp=None makes a call that passed the
    # workspace check stop at the next one)
    big = dict(T=20000, V=151936, logp=None)
    assert call(ws_bytes=R.rl_workspace_size(20000, 151936, 4096), **big) == 1
    assert call(ws_bytes=256 + 2 * 16 * 38 * 4096, **big) == 1
    assert call(ws_bytes=256 + 2 * 16 * 38 * 4096 - 1, **big) == 4


def test_masked_gae_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(n=4, offs=FAKE, T=100, mask=FAKE, V=FAKE, rt=None, rr=None, g=0.99, l=0.95, skip=1, adv=FAKE,
                 ret=None, ws=FAKE, ws_bytes=1024, stream=None)
        a.update(over)
        return L.rl_masked_gae(a["n"], a["offs"], a["T"], a["mask"], a["V"], a["rt"], a["rr"], a["g"], a["l"],
                               a["skip"], a["adv"], a["ret"], a["ws"], a["ws_bytes"], a["stream"])

    assert call(n=-1) == 1
    assert call(T=-5) == 1
    assert call(g=1.5) == 1
    assert call(l=-0.1) == 1
    assert call(g=float("nan")) == 1
    assert call(skip=2) == 1
    assert call(ws=None) == 1
    assert call(ws_bytes=16) == 4
    assert call(offs=None) == 1
    assert call(adv=None) == 1
    assert call(n=0) == 0


def test_value_loss_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(rows=16, V=FAKE, G=FAKE, mask=FAKE, tt=FAKE, n=2, coef=FAKE, dV=FAKE, loss=FAKE, ws=FAKE,
                 ws_bytes=1 << 16, stream=None)
        a.update(over)
        return L.rl_value_loss_fwd_bwd(a["rows"], a["V"], a["G"], a["mask"], a["tt"], a["n"], a["coef"], a["dV"],
                                       a["loss"], a["ws"], a["ws_bytes"], a["stream"])

    assert call(rows=-1) == 1
    assert call(n=-1) == 1
    assert call(loss=None) == 1
    assert call(ws_bytes=256 + 8 * 16 - 1) == 4
    assert call(dV=None) == 1
    assert call(coef=None) == 1
    assert call(rows=0) == 0


def test_token_level_adv_flag_checks(R):
    assert _loss(R, params=_params(R, token_level_adv=2)) == 1
    assert _loss(R, params=_params(R, token_level_adv=1), adv=None, n_traj=0) == 1


def test_sequence_is_weights_argument_checks(R):
    L = R.lib()

    def call(**over):
        a = dict(n=4, T=100, tt=FAKE, mask=FAKE, old=FAKE, roll=FAKE, cap=2.0, w=FAKE, S=None, ta=None, tk=None,
                 ws=FAKE, ws_bytes=1024, stream=None)
        a.update(over)
        return L.rl_sequence_is_weights(a["n"], a["T"], a["tt"], a["mask"], a["old"], a["roll"], a["cap"], a["w"],
                                        a["S"], a["ta"], a["tk"], a["ws"], a["ws_bytes"], a["stream"])

    assert call(n=-1) == 1
    assert call(T=-1) == 1
    assert call(cap=float("nan")) == 1
    assert call(ws=None) == 1
    assert call(n=200, ws_bytes=256 + 8 * 200 - 1) == 4
    assert call(w=None) == 1
    assert call(roll=None) == 1
    assert call(n=0) == 0


def test_owner_and_tree_argument_checks(R):
    L = R.lib()
    p = _params(R)
    assert L.rl_group_advantages_by_owner(-1, 0, None, FAKE, None, 10, FAKE, FAKE, p, FAKE, FAKE, FAKE, FAKE, 1024,
                                          None) == 1
    assert L.rl_group_advantages_by_owner(4, 1, FAKE, FAKE, None, 10, None, FAKE, p, FAKE, FAKE, FAKE, FAKE, 1024,
                                          None) == 1
    assert L.rl_group_advantages_by_owner(4, 1, FAKE, FAKE, None, 10, FAKE, FAKE, p, FAKE, FAKE, FAKE, FAKE, 16,
                                          None) == 4
    assert L.rl_rollout_value_advantages(-1, FAKE, FAKE, FAKE, FAKE, 2, FAKE, None, FAKE, 1024, None) == 1
    assert L.rl_rollout_value_advantages(10, FAKE, FAKE, FAKE, None, 2, FAKE, None, FAKE, 1024, None) == 1
    n_tok = ctypes.c_int64(0)
    assert L.rl_prefix_tree_build_batch(-1, *([None] * 8), 0, 1, 0, *([None] * 11), ctypes.byref(n_tok)) == 1
    import numpy as np
    bad = np.array([0, 3, 1], np.int64)  # decreasing offsets
    co = np.array([0, 0, 0], np.int32)
    ptr = lambda a: a.ctypes.data_as(ctypes.c_void_p)  # noqa: E731
    assert L.rl_prefix_tree_build_batch(2, ptr(bad), ptr(np.zeros(4, np.int32)), ptr(co), ptr(np.zeros(1, np.int64)),
                                        None, ptr(np.zeros(1, np.int64)), None, None, 0, 1, 0,
                                        *([None] * 11), ctypes.byref(n_tok)) == 1



def test_stats_summary_argument_checks(R):
    L = R.lib()
    assert L.rl_token_stats_summary(-1, FAKE, FAKE, FAKE, 2, FAKE, FAKE, FAKE, 1024, None) == 1
    assert L.rl_token_stats_summary(10, FAKE, FAKE, FAKE, 2, FAKE, None, FAKE, 1024, None) == 1
    assert L.rl_token_stats_summary(10, FAKE, FAKE, FAKE, 2, FAKE, FAKE, FAKE, 16, None) == 4
    assert L.rl_token_stats_summary(10, None, FAKE, FAKE, 2, FAKE, FAKE, FAKE, 1024, None) == 1
    assert L.rl_token_stats_summary(0, None, None, None, 0, None, FAKE, FAKE, 1024, None) == 0



def test_fused_head_loss_shape_limits(R):
    L = R.lib()
    p = _params(R)
    loss = FAKE

    def call(T=16, D=128, V=1000):
        return L.rl_fused_head_loss_fwd_bwd(FAKE, FAKE, T, D, V, FAKE, FAKE, FAKE, 2, FAKE, FAKE, FAKE, None, None, p,
                                            FAKE, R.RL_BF16, FAKE, loss, None, FAKE, 1 << 40, None)

    assert call(D=96) == 2          # not a multiple of 64
    assert call(D=32) == 1
    assert call(V=524_289) == 2     # above the fix-up kernel's shared-memory tile factors
    assert call(D=65_600) == 2
    assert call(T=-1) == 1


def test_binding_fails_loudly_without_the_library(R, monkeypatch):
    """No CPU fallback: with the shared library absent every entry point raises."""
    import pytest as _pytest
    import torch

    monkeypatch.setattr(R, "_lib", None)
    monkeypatch.setattr(R, "LIB_PATH", R.LIB_PATH + ".absent")
    with _pytest.raises(RuntimeError, match="missing"):
        R.lib()
    with _pytest.raises(RuntimeError, match="missing"):
        R.rl_workspace_size(16, 128)
    # host tensors are refused outright: there is no CPU path to fall back to
    with _pytest.raises(ValueError, match="CUDA tensor"):
        R.rl_token_logprobs(torch.zeros((2, 8)), torch.zeros(2, dtype=torch.int32), torch.zeros(1024, dtype=torch.uint8))
