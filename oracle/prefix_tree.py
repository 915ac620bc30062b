"""Plain CPU statement of the rollout-level prefix tree and of the loss bookkeeping over it.

TEST INFRASTRUCTURE. Like the other oracle modules, only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may import this module; it imports
nothing from the product path.

Passages followed (arXiv 2608.16798, "ClawGym II"):

* ``build_prefix_tree`` -- Sec. 3.2.1 "Prefix Tree Construction": a tree rooted at the
  initial task prompt; each captured call (x_i, y_i) is attached to the existing node whose
  accumulated history is the longest prefix of x_i; comparing x_i with that history recovers
  the harness content in between (tool outputs, environment feedback). Sec. 3.2.2
  "Trajectory Extraction and Filtering": dead leaves of retries are dropped (per segment the
  leaf with the longest continuation is kept), over-branching rollouts are discarded and
  auxiliary (subagent, compaction) trajectories are excluded. Shared prefixes are stored
  once (Sec. 3.2.1) and counted once in the loss (Sec. 3.2.3).
* ``owner_token_counts``, ``advantages_and_coefficients_by_owner`` -- the GRPO advantage of
  a rollout assigned to all trainable token nodes of its retained trajectories, each shared
  token once (Sec. 3.2.3), with tokens in any order.
* ``rollout_value_advantages`` -- PPO on the tree: A_t = R_i - V(s_t) (Sec. 2.3.4, gamma =
  lambda = 1, every trajectory backed up on its own; on a shared token all of them agree).

Readings where the paper leaves details open:

* a node holds its call's input past the parent's history (M = 0) followed by the call's
  response (M = 1); its accumulated history is x_i followed by y_i; the root holds the
  prompt (M = 0);
* a call whose input does not start with the task prompt cannot be placed in the tree and is
  reported as unplaced;
* among equally long matching histories the earliest node is the parent;
* over-branching counts the leaves of the whole tree (auxiliary calls included) and discards
  the rollout when there are more than ``max_leaves`` (> 0);
* auxiliary calls are flagged by the caller and removed with their subtrees before leaves are
  taken for training;
* a segment is the set of root children with the same input (retries of the first call of a
  segment share it; a compaction starts from a new input) together with their subtrees; in
  each segment the leaf with the longest accumulated history is kept (ties: the earliest);
* retained nodes (the kept leaves' ancestors) are laid out in depth-first preorder, children
  in creation order; per token the output gives the position of the previous token on its
  path (-1 for the first prompt token) and the token's depth on its path.
"""

from __future__ import annotations

import numpy as np


def build_prefix_tree(prompt, calls, aux=None, max_leaves: int = 0):
    """prompt: token list; calls: list of (x, y) token lists in capture order; aux: per-call
    flags (truthy = auxiliary). Returns a dict with ``valid`` and, when valid, the flattened
    ``tokens``, ``mask``, ``parent``, ``depth``, ``node_call`` (call index of each token's node,
    -1 for the prompt), ``leaf_calls`` (retained leaves in layout order), ``leaf_end`` (position
    of each retained leaf's last token, -1 if its path is empty), ``n_leaves`` (whole tree) and
    ``unplaced`` (calls whose input does not start with the prompt)."""
    prompt = [int(v) for v in prompt]
    aux = [False] * len(calls) if aux is None else [bool(a) for a in aux]
    hist = [prompt]
    own = [prompt]
    own_mask = [[0] * len(prompt)]
    par = [-1]
    call_of = [-1]
    unplaced = []
    for i, (x, y) in enumerate(calls):
        x = [int(v) for v in x]
        y = [int(v) for v in y]
        if x[:len(prompt)] != prompt:
            unplaced.append(i)
            continue
        best = 0
        for n in range(len(hist)):
            h = hist[n]
            if len(h) <= len(x) and x[:len(h)] == h and len(h) > len(hist[best]):
                best = n
        inter = x[len(hist[best]):]
        hist.append(x + y)
        own.append(inter + y)
        own_mask.append([0] * len(inter) + [1] * len(y))
        par.append(best)
        call_of.append(i)
    n_nodes = len(hist)
    children = [[] for _ in range(n_nodes)]
    for n in range(1, n_nodes):
        children[par[n]].append(n)
    n_leaves = sum(1 for n in range(1, n_nodes) if not children[n])
    out = dict(valid=True, n_leaves=n_leaves, unplaced=unplaced)
    if max_leaves > 0 and n_leaves > max_leaves:
        out.update(valid=False, tokens=[], mask=[], parent=[], depth=[], node_call=[], leaf_calls=[], leaf_end=[])
        return out

    # auxiliary calls leave the tree with their subtrees
    main = [True] * n_nodes
    for n in range(1, n_nodes):  # parents precede children in creation order
        main[n] = main[par[n]] and not aux[call_of[n]]
    main_children = [[c for c in children[n] if main[c]] for n in range(n_nodes)]

    def top(n):  # the root child above n
        while par[n] != 0:
            n = par[n]
        return n

    seg_key = {}
    for n in range(1, n_nodes):
        if main[n] and par[n] == 0:
            x = calls[call_of[n]][0]
            seg_key[n] = tuple(int(v) for v in x)
    best_leaf = {}
    for n in range(1, n_nodes):
        if not main[n] or main_children[n]:
            continue
        key = seg_key[top(n)]
        if key not in best_leaf or len(hist[n]) > len(hist[best_leaf[key]]):
            best_leaf[key] = n
    keep = [False] * n_nodes
    keep[0] = True
    for n in best_leaf.values():
        while n >= 0 and not keep[n]:
            keep[n] = True
            n = par[n]
    kept_leaves = set(best_leaf.values())

    tokens, mask, parent, depth, node_call, leaf_calls, leaf_end = [], [], [], [], [], [], []
    path_end = [-1] * n_nodes

    def visit(n):
        prev = path_end[par[n]] if n else -1
        for k, tok in enumerate(own[n]):
            p = prev if k == 0 else len(tokens) - 1
            parent.append(p)
            depth.append(depth[p] + 1 if p >= 0 else 0)
            tokens.append(tok)
            mask.append(own_mask[n][k])
            node_call.append(call_of[n])
        path_end[n] = len(tokens) - 1 if own[n] else prev
        if n in kept_leaves:
            leaf_calls.append(call_of[n])
            leaf_end.append(path_end[n])
        for c in children[n]:
            if keep[c]:
                visit(c)

    visit(0)
    out.update(tokens=tokens, mask=mask, parent=parent, depth=depth, node_call=node_call, leaf_calls=leaf_calls,
               leaf_end=leaf_end)
    return out


def owner_token_counts(token_traj, mask, n_traj: int):
    """L_i = number of tokens t with owner i and M_t = 1 (any token order)."""
    tt = np.asarray(token_traj, dtype=np.int64)
    M = np.asarray(mask) != 0
    L = np.zeros(n_traj, dtype=np.int64)
    for t in range(len(tt)):
        if M[t] and 0 <= tt[t] < n_traj:
            L[tt[t]] += 1
    return L


def advantages_and_coefficients_by_owner(rewards, group_offsets, token_traj, mask, n_traj: int, traj_valid=None,
                                         params=None):
    """Group advantages per rollout and loss coefficients from the deduplicated trainable-token
    counts of each rollout (Sec. 3.2.3), tokens in any order."""
    from oracle import grpo_objective as G

    params = G.LossParams() if params is None else params
    L = owner_token_counts(token_traj, mask, n_traj)
    adv = G.group_advantages(rewards, group_offsets, traj_valid, params.adv_eps)
    coef = G.loss_coefficients(L, traj_valid, params.loss_agg)
    return adv, coef, L


def rollout_value_advantages(token_traj, mask, values, rewards):
    """A_t = R_{i(t)} - V_t and G_t = R_{i(t)} on trainable tokens, 0 elsewhere."""
    tt = np.asarray(token_traj, dtype=np.int64)
    M = np.asarray(mask) != 0
    R = np.asarray(rewards, dtype=np.float64)[tt]
    V = np.asarray(values, dtype=np.float64)
    return np.where(M, R - V, 0.0), np.where(M, R, 0.0)
