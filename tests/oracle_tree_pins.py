"""Pins for the prefix-tree oracle: a hand-worked tree, and properties that follow from the
definition on random rollouts (every kept trajectory is recovered exactly by following the
parent links, each kept node's tokens appear once, responses and only responses are
trainable, a plain chain flattens to its last call, parents are the longest matching
histories) plus the ownership bookkeeping. Each pin is ``pin_xxx(T)`` of a tree oracle ``T``."""

from __future__ import annotations

import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def random_rollout(rng, prompt_len=6, turns=8, p_retry=0.25, p_compact=0.15, p_aux=0.15, vocab=50):
    """Calls of one synthetic rollout: a main chain with retries, compactions (new segment from
    the prompt plus a summary) and auxiliary calls; tokens drawn from [0, vocab)."""
    tok = lambda n: [int(v) for v in rng.integers(0, vocab, n)]  # noqa: E731
    prompt = tok(prompt_len)
    calls, aux = [], []
    hist = list(prompt)
    for _ in range(turns):
        x = hist + (tok(int(rng.integers(0, 4))) if len(hist) > len(prompt) else [])
        if rng.random() < p_retry:
            calls.append((x, tok(int(rng.integers(0, 4)))))
            aux.append(0)
        y = tok(int(rng.integers(0, 5)))
        calls.append((x, y))
        aux.append(0)
        hist = x + y
        if rng.random() < p_aux:
            calls.append((hist + tok(2), tok(3)))
            aux.append(1)
        if rng.random() < p_compact:
            hist = prompt + tok(int(rng.integers(1, 4)))
    return prompt, calls, aux


def pin_tree_golden(T):
    with open(os.path.join(GOLDEN, "prefix_tree_worked_example.json")) as f:
        ex = json.load(f)
    out = T.build_prefix_tree(ex["prompt"], [(c["x"], c["y"]) for c in ex["calls"]], [c["aux"] for c in ex["calls"]])
    for k, v in ex["expected"].items():
        assert list(out[k]) == v if isinstance(v, list) else out[k] == v, (k, out[k], v)
    dropped = T.build_prefix_tree(ex["prompt"], [(c["x"], c["y"]) for c in ex["calls"]],
                                  [c["aux"] for c in ex["calls"]], max_leaves=2)
    assert dropped["valid"] is False and dropped["tokens"] == []


def pin_tree_paths_recovered(T):
    """Following parent links from each kept leaf's last token gives exactly x + y of its call;
    depth is the index along that path; the trainable tokens are exactly the responses."""
    rng = np.random.default_rng(3)
    for _ in range(60):
        prompt, calls, aux = random_rollout(rng)
        out = T.build_prefix_tree(prompt, calls, aux)
        toks, par, dep = out["tokens"], out["parent"], out["depth"]
        assert len(set(out["leaf_calls"])) == len(out["leaf_calls"])
        for c, last in zip(out["leaf_calls"], out["leaf_end"]):
            assert not aux[c]
            x, y = calls[c]
            path = []
            t = last
            while t >= 0:
                path.append(toks[t])
                t = par[t]
            path.reverse()
            assert path == list(x) + list(y), (path, x, y)
        for t in range(len(toks)):
            assert par[t] < t
            assert dep[t] == (dep[par[t]] + 1 if par[t] >= 0 else 0)
        # responses of kept calls are the trainable tokens; everything else (prompt, harness) is not
        kept_calls = set(out["node_call"]) - {-1}
        n_resp = sum(len(calls[c][1]) for c in kept_calls)
        assert sum(out["mask"]) == n_resp


def pin_tree_chain_and_sharing(T):
    """A plain chain (no retries, compactions or auxiliary calls) flattens to the last call's
    history; two retries that both continue keep only the longer branch; shared tokens once."""
    rng = np.random.default_rng(4)
    prompt, calls, aux = random_rollout(rng, p_retry=0.0, p_compact=0.0, p_aux=0.0)
    out = T.build_prefix_tree(prompt, calls, aux)
    x, y = calls[-1]
    assert out["tokens"] == list(x) + list(y)
    assert out["leaf_calls"] == [len(calls) - 1]
    assert out["mask"] == [0] * len(prompt) + sum(
        ([0] * (len(calls[i][0]) - (len(calls[i - 1][0]) + len(calls[i - 1][1]) if i else len(prompt))) +
         [1] * len(calls[i][1]) for i in range(len(calls))), [])
    p = [1, 2]
    two = [([1, 2], [5, 6]), ([1, 2, 5, 6, 9], [7]), ([1, 2, 5, 6, 9], [8, 8, 8])]
    out = T.build_prefix_tree(p, two)
    assert out["tokens"] == [1, 2, 5, 6, 9, 8, 8, 8] and out["leaf_calls"] == [2] and out["n_leaves"] == 2


def pin_tree_longest_prefix_parent(T):
    """Brute force over every earlier node: the parent is the longest history that prefixes x
    (checked through the recovered paths: the kept leaf's path shares its longest prefix)."""
    p = [1]
    calls = [([1], [2, 3]), ([1, 2], [9]), ([1, 2, 3, 4], [5]), ([1, 2, 9, 4], [6])]
    # histories: n1 [1,2,3], n2 [1,2,9] (parent root: [1,2,3] is not a prefix of [1,2]),
    # n3 [1,2,3,4,5] under n1, n4 [1,2,9,4,6] under n2
    out = T.build_prefix_tree(p, calls)
    # one segment per distinct root-child input: [1] and [1, 2]
    assert sorted(out["leaf_calls"]) == [2, 3]
    assert out["tokens"] == [1, 2, 3, 4, 5, 2, 9, 4, 6]
    assert out["parent"] == [-1, 0, 1, 2, 3, 0, 5, 6, 7]
    # two identical calls give two nodes with equal histories; a continuation attaches to the
    # earlier one, which the kept path then goes through
    same = [([1], [4]), ([1], [4]), ([1, 4, 8], [6])]
    out = T.build_prefix_tree(p, same)
    assert out["tokens"] == [1, 4, 8, 6] and out["node_call"] == [-1, 0, 2, 2] and out["leaf_calls"] == [2]


def pin_owner_counts(T):
    """Counts by owner equal span counts for contiguous owners and are order-independent."""
    from oracle import grpo_objective as G

    rng = np.random.default_rng(6)
    lengths = rng.integers(0, 9, 30)
    offs = np.concatenate([[0], np.cumsum(lengths)])
    mask = (rng.random(offs[-1]) < 0.6).astype(np.uint8)
    L_span, tt = G.trajectory_token_counts(mask, offs)
    L = T.owner_token_counts(tt, mask, 30)
    assert np.array_equal(L, L_span)
    perm = rng.permutation(len(tt))
    assert np.array_equal(T.owner_token_counts(tt[perm], mask[perm], 30), L)
    a, g = T.rollout_value_advantages([0, 1, 1], [1, 0, 1], [0.25, 9.0, 0.5], [1.0, 2.0])
    assert list(a) == [0.75, 0.0, 1.5] and list(g) == [1.0, 0.0, 2.0]


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
