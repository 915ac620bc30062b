"""The prefix-tree oracle against its pins, and planted mistakes that the pins must catch."""

import inspect
import sys
import types

import pytest

import oracle.prefix_tree as T
from oracle_tree_pins import ALL_PINS

SRC = inspect.getsource(T)

MUTANTS = {
    "shortest matching parent": ("len(h) > len(hist[best])", "len(h) < len(hist[best]) and n > 0"),
    "latest tie wins": ("len(h) > len(hist[best])", "len(h) >= len(hist[best])"),
    "harness content trainable": ("own_mask.append([0] * len(inter) + [1] * len(y))",
                                  "own_mask.append([1] * len(inter) + [1] * len(y))"),
    "intervening dropped": ("own.append(inter + y)", "own.append(y)"),
    "aux kept": ("main[n] = main[par[n]] and not aux[call_of[n]]", "main[n] = main[par[n]]"),
    "shortest leaf kept": ("len(hist[n]) > len(hist[best_leaf[key]])", "len(hist[n]) < len(hist[best_leaf[key]])"),
    "no over-branching": ("if max_leaves > 0 and n_leaves > max_leaves:", "if False:"),
    "parent link off by one": ("p = prev if k == 0 else len(tokens) - 1", "p = prev if k == 0 else len(tokens) - 2"),
    "branch links to previous token": ("prev = path_end[par[n]] if n else -1", "prev = len(tokens) - 1 if n else -1"),
    "prompt not required": ("if x[:len(prompt)] != prompt:", "if False:"),
    "owner counts ignore mask": ("if M[t] and 0 <= tt[t] < n_traj:", "if 0 <= tt[t] < n_traj:"),
    "value advantage sign": ("return np.where(M, R - V, 0.0)", "return np.where(M, V - R, 0.0)"),
}


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(T)


def _mutant(old, new):
    assert SRC.count(old) >= 1, f"snippet not in oracle: {old}"
    mod = types.ModuleType("tree_oracle_mutant")
    mod.__file__ = T.__file__
    sys.modules["tree_oracle_mutant"] = mod
    try:
        exec(compile(SRC.replace(old, new, 1), "<tree oracle mutant>", "exec"), mod.__dict__)
    finally:
        del sys.modules["tree_oracle_mutant"]
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name):
    mod = _mutant(*MUTANTS[name])
    failed = []
    for pin in ALL_PINS:
        try:
            pin(mod)
        except Exception as e:
            failed.append((pin.__name__, type(e).__name__))
    assert failed, f"no pin catches the planted mistake '{name}'"
