"""The oracle's chain budgets against hand-derived values (no GPU).

App. C.2 gives the two budgets of one hop of a sequential chain: relative
B = T_old + ceil(T_new / r) and fixed B = min(B_max, T_old + T_new).  Sec. 4
states what they do over a chain whose agents each add H positions: the
relative budget grows by H / r per agent (N H / r after N agents), the fixed
one stops growing at B_max.  tests/golden/chain_budget_cases.json holds values
worked out by hand from those statements, each with its reasoning; they are
checked here against oracle.chain_budget alone (the library is compared with
the oracle elsewhere).  Planted mistakes in a copy of the oracle's function
must each fail at least one of them.
"""
import inspect
import json
import os

import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "chain_budget_cases.json")


def _cases():
    with open(GOLDEN) as f:
        return json.load(f)


def _check(fn):
    """Every hand-derived value, single hops and whole chains, through `fn`."""
    data = _cases()
    for c in data["cases"]:
        got = fn(c["T_old"], c["T_new"], c["keep"], mode=c["mode"], B_max=c["B_max"])
        assert got == c["expected"], (c, got)
    for ch in data["chains"]:
        msg, got = 0, []
        for _ in range(ch["hops"]):
            msg = fn(msg, ch["H"], ch["keep"], mode=ch["mode"], B_max=ch["B_max"])   # the message is inherited
            got.append(msg)
        assert got == ch["expected"], (ch, got)


def test_chain_budget_hand_derived():
    _check(oracle.chain_budget)


MUTANTS = [
    ("fixed_ignores_inherited", "B = min(B_max, T)", "B = min(B_max, T_new)"),
    ("fixed_ignores_cap", "B = min(B_max, T)", "B = T"),
    ("relative_drops_inherited", "B = T_old + budget(T_new, keep)", "B = budget(T_new, keep)"),
    ("relative_over_all_positions", "B = T_old + budget(T_new, keep)", "B = budget(T, keep)"),
    ("relative_floor", "B = T_old + budget(T_new, keep)", "B = T_old + int(keep * T_new)"),
    ("relative_rounded", "B = T_old + budget(T_new, keep)", "B = T_old + round(keep * T_new)"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(name, old, new):
    src = inspect.getsource(oracle.chain_budget)
    assert src.count(old) == 1, name
    ns = dict(vars(oracle))
    exec(compile(src.replace(old, new), "<mutant %s>" % name, "exec"), ns)
    with pytest.raises(AssertionError):
        _check(ns["chain_budget"])
