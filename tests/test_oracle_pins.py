"""CPU: the float64 oracle against the closed forms, special cases and
algorithms that pin it (see ``oracle_pins.py`` for the list)."""
import pytest

import oracle
from oracle_pins import ALL_PINS


@pytest.fixture(scope="module")
def orc():
    return oracle.load()


@pytest.mark.parametrize("pin", ALL_PINS, ids=[p.__name__ for p in ALL_PINS])
def test_pin(orc, pin):
    pin(orc)


def test_openmp_matches_serial(orc):
    import numpy as np
    rng = np.random.default_rng(5)
    B, L, D = 3, 40, 16
    x = rng.standard_normal((B, L, D))
    gl = rng.standard_normal((B, L, 2 * D))
    lam = rng.standard_normal(D)
    dh = rng.standard_normal((B, L, D))
    h1, _ = orc.fwd(x, gl, lam, threads=1)
    h4, _ = orc.fwd(x, gl, lam, threads=4)
    assert np.array_equal(h1, h4)
    g1 = orc.bwd(dh, x, gl, lam, threads=1)
    g4 = orc.bwd(dh, x, gl, lam, threads=4)
    for a, b in zip(g1, g4):
        assert np.array_equal(a, b)
