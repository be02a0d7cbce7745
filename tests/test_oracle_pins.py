"""The CPU oracle against its pins (no GPU)."""
import pytest

import oracle
import oracle_pins


@pytest.fixture(scope="module")
def o():
    return oracle.default()


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_pin(o, pin):
    pin(o)


def test_budget_rounding():
    # App. C.2: B_i = ceil(T_i / r); keep = 1/r, computed in double
    assert oracle.budget(8192, 0.25) == 2048
    assert oracle.budget(8192, 0.10) == 820
    assert oracle.budget(65536, 0.10) == 6554
    assert oracle.budget(16384, 0.25) == 4096
    assert oracle.budget(512, 0.25) == 128
    assert oracle.budget(100, 0.0) == 0
    assert oracle.budget(100, 2.0) == 100


def test_thread_count_does_not_change_results(o):
    import numpy as np
    from oracle_pins import _rand_case
    K, _, Q = _rand_case(3, 8, 2, 32, 300, 9, seed=2)
    a = o.score(K, Q, n_threads=1)
    b = o.score(K, Q, n_threads=4)
    for k in a:
        assert np.array_equal(a[k], b[k])
