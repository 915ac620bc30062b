"""The PPO oracle against its pins, and planted mistakes that the pins must catch."""

import inspect
import sys
import types

import pytest

import oracle.ppo_objective as P
from oracle_ppo_pins import ALL_PINS

SRC = inspect.getsource(P)

MUTANTS = {
    "bootstrap ignores mask": ("boot = Vv[t + 1] if (t + 1 < e and M[t + 1]) else 0.0",
                               "boot = Vv[t + 1] if (t + 1 < e) else 0.0"),
    "bootstrap across trajectories": ("boot = Vv[t + 1] if (t + 1 < e and M[t + 1]) else 0.0",
                                      "boot = Vv[t + 1] if (t + 1 < len(Vv) and M[t + 1]) else 0.0"),
    "discount without lambda": ("cur = (delta if M[t] else 0.0) + gamma * lam * nxt",
                                "cur = (delta if M[t] else 0.0) + gamma * nxt"),
    "delta not masked": ("cur = (delta if M[t] else 0.0) + gamma * lam * nxt", "cur = delta + gamma * lam * nxt"),
    "bootstrap without gamma": ("delta = r[t] + gamma * boot - Vv[t]", "delta = r[t] + boot - Vv[t]"),
    "skip bootstraps own value": ("delta = r[t] + gamma * nxt_v - Vv[t]", "delta = r[t] + gamma * Vv[t] - Vv[t]"),
    "skip drops lambda": ("adv[t] = delta + gamma * lam * nxt_a", "adv[t] = delta + gamma * nxt_a"),
    "reward at last token": ("r[s + valid[-1]] += float(traj_rewards[i])", "r[e - 1] += float(traj_rewards[i])"),
    "returns without value": ("return adv, np.where(M, adv + Vv, 0.0)\n\n\ndef masked_gae_skip",
                              "return adv, np.where(M, adv, 0.0)\n\n\ndef masked_gae_skip"),
    "value grad without 2": ("return math.fsum(contrib.tolist()), 2.0 * w * d, contrib",
                             "return math.fsum(contrib.tolist()), w * d, contrib"),
    "value grad sign": ("return math.fsum(contrib.tolist()), 2.0 * w * d, contrib",
                        "return math.fsum(contrib.tolist()), -2.0 * w * d, contrib"),
    "value loss unmasked": ("w = np.where(M, c, 0.0)", "w = c"),
}


@pytest.mark.parametrize("pin", ALL_PINS, ids=lambda f: f.__name__)
def test_pin(pin):
    pin(P)


def _mutant(old, new):
    assert SRC.count(old) >= 1, f"snippet not in oracle: {old}"
    mod = types.ModuleType("ppo_oracle_mutant")
    mod.__file__ = P.__file__
    sys.modules["ppo_oracle_mutant"] = mod
    try:
        exec(compile(SRC.replace(old, new, 1), "<ppo oracle mutant>", "exec"), mod.__dict__)
    finally:
        del sys.modules["ppo_oracle_mutant"]
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
