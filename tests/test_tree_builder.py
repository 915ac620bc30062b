"""The native prefix-tree builder (host C++ behind the C ABI) against the oracle, bit for bit.

No GPU is involved: rl_prefix_tree_build_batch is a host function. Random rollouts come from
the pins' generator (retries, compactions, auxiliary calls) and from the workload generator
at realistic sizes; unplaced calls, empty responses and discarded rollouts are included."""

import numpy as np
import pytest

import oracle.prefix_tree as T
from oracle_tree_pins import random_rollout
from paper_2608_16798_gb300 import build as B
from paper_2608_16798_gb300 import workloads as W


@pytest.fixture(scope="module")
def R():
    B.build()
    import paper_2608_16798_gb300.rl_loss as R

    R.lib()
    return R


def oracle_batch(prompts, calls, aux, max_leaves):
    toks, mask, parent, depth, owner, node_call, leaf_call, leaf_end = ([] for _ in range(8))
    offs, loffs, stats = [0], [0], []
    call_base = 0
    for r, (p, cs, a) in enumerate(zip(prompts, calls, aux)):
        out = T.build_prefix_tree(p, cs, a, max_leaves)
        base = offs[-1]
        if out["valid"]:
            toks += out["tokens"]
            mask += out["mask"]
            parent += [q + base if q >= 0 else -1 for q in out["parent"]]
            depth += out["depth"]
            owner += [r] * len(out["tokens"])
            node_call += [c + call_base if c >= 0 else -1 for c in out["node_call"]]
            leaf_call += [c + call_base for c in out["leaf_calls"]]
            leaf_end += [q + base if q >= 0 else -1 for q in out["leaf_end"]]
        offs.append(len(toks))
        loffs.append(len(leaf_call))
        stats.append(dict(valid=int(out["valid"]), n_leaves=out["n_leaves"], n_unplaced=len(out["unplaced"]),
                          n_kept_leaves=len(out["leaf_calls"]) if out["valid"] else 0,
                          n_tokens=len(out["tokens"]) if out["valid"] else 0,
                          n_trainable=int(sum(out["mask"])) if out["valid"] else 0))
        call_base += len(cs)
    return dict(tokens=toks, mask=mask, parent=parent, depth=depth, owner=owner, node_call=node_call,
                leaf_call=leaf_call, leaf_end=leaf_end, rollout_offsets=offs, leaf_offsets=loffs, stats=stats)


def compare(got, ref):
    for k in ("tokens", "mask", "parent", "depth", "owner", "node_call", "leaf_call", "leaf_end", "rollout_offsets",
              "leaf_offsets"):
        assert np.array_equal(np.asarray(got[k], dtype=np.int64), np.asarray(ref[k], dtype=np.int64)), k
    assert got["stats"] == ref["stats"]


@pytest.mark.parametrize("threads", [1, 4])
def test_random_rollouts_bit_exact(R, threads):
    rng = np.random.default_rng(7)
    prompts, calls, aux = [], [], []
    for k in range(80):
        p, c, a = random_rollout(rng, turns=int(rng.integers(0, 12)))
        if k % 9 == 0 and c:
            c = c + [([99] + list(c[0][0]), [1, 2])]  # does not start with the prompt
            a = a + [0]
        prompts.append(p)
        calls.append(c)
        aux.append(a)
    for max_leaves in (0, 3):
        got = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=max_leaves, n_threads=threads)
        compare(got, oracle_batch(prompts, calls, aux, max_leaves))


def test_workload_rollouts_bit_exact(R):
    """Rollouts of the tree workload (long histories, retries, compactions, subagents)."""
    w = W.WORKLOADS["tree"]
    prompts, calls, aux = W.tree_rollouts(w, seed=1, n_rollouts=12)
    got = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves)
    ref = oracle_batch(prompts, calls, aux, w.tree_max_leaves)
    compare(got, ref)
    assert sum(s["n_kept_leaves"] for s in ref["stats"]) > 12  # compactions keep several segments


def test_workload_batch_properties(R):
    """The full tree workload (128 rollouts) through the native builder alone: runaway rollouts
    are discarded, shared histories are stored once (the packed stream is several times shorter
    than the captured calls), and every kept leaf's path is its call's history."""
    w = W.WORKLOADS["tree"]
    prompts, calls, aux = W.tree_rollouts(w, seed=0)
    got = R.rl_prefix_tree_build_batch(prompts, calls, aux, max_leaves=w.tree_max_leaves)
    st = got["stats"]
    assert any(s["valid"] == 0 for s in st) and sum(s["valid"] for s in st) > 100
    captured = sum(len(x) + len(y) for cs in calls for x, y in cs)
    assert captured > 4 * len(got["tokens"])
    flat = [c for cs in calls for c in cs]
    toks, par = got["tokens"], got["parent"]
    for c, last in zip(got["leaf_call"][::7], got["leaf_end"][::7]):
        path = []
        t = int(last)
        while t >= 0:
            path.append(int(toks[t]))
            t = int(par[t])
        x, y = flat[c]
        assert path[::-1] == list(x) + list(y)


def test_empty_and_size_query(R):
    got = R.rl_prefix_tree_build_batch([], [])
    assert len(got["tokens"]) == 0 and list(got["rollout_offsets"]) == [0]
    got = R.rl_prefix_tree_build_batch([[5, 6]], [[]])
    assert list(got["tokens"]) == [5, 6] and list(got["mask"]) == [0, 0] and len(got["leaf_call"]) == 0
