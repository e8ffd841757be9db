"""Service-interval accounting (App. D.2): the oracle against the identity
and bounds the paper derives, and the library's as2d_interval_accounting
against the oracle.  Host code only."""
import random
from fractions import Fraction

import pytest

from oracle.accounting import accounting


def test_worked_cases():
    # disjoint: serial comparator, no overlap
    assert accounting([(0, 2)], [(2, 5)], 6) == (2, 3, 0, 1)
    # nested: the verifier inside the producer
    assert accounting([(0, 10)], [(2, 3), (5, 6)], 10) == (10, 2, 2, 0)
    # overlapping pieces of one set are merged before summing
    assert accounting([(0, 2), (1, 3)], [(2.5, 5)], 6) == (3, Fraction(5, 2), Fraction(1, 2), 1)
    # clipping to [0, T]
    assert accounting([(-1, 1)], [(4, 9)], 5) == (1, 1, 0, 3)
    assert accounting([], [], 4) == (0, 0, 0, 4)
    with pytest.raises(ValueError):
        accounting([(2, 1)], [], 3)


@pytest.mark.parametrize("seed", range(30))
def test_identity_and_bounds(seed):
    """T = D + V - O + H exactly, 0 <= O <= min(D, V), T >= max(D, V) + H,
    and brute force over unit cells of an integer grid agrees."""
    rng = random.Random(seed)
    T = rng.randint(1, 40)
    P = [tuple(sorted((rng.randint(-3, T + 3), rng.randint(-3, T + 3))))
         for _ in range(rng.randint(0, 6))]
    V = [tuple(sorted((rng.randint(-3, T + 3), rng.randint(-3, T + 3))))
         for _ in range(rng.randint(0, 6))]
    d, v, o, h = accounting(P, V, T)
    assert d + v - o + h == T
    assert 0 <= o <= min(d, v) and T >= max(d, v) + h
    cells = [(t, t + 1) for t in range(T)]
    inp = [any(a <= t and t + 1 <= b for a, b in P) for t, _ in cells]
    inv = [any(a <= t and t + 1 <= b for a, b in V) for t, _ in cells]
    assert d == sum(inp) and v == sum(inv)
    assert o == sum(x and y for x, y in zip(inp, inv))
    assert h == sum(not (x or y) for x, y in zip(inp, inv))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._lib_build_module().build()
    import paper_2609_37617_gb300 as p
    return p


@pytest.mark.parametrize("seed", range(30))
def test_library_matches_oracle(lib, seed):
    rng = random.Random(100 + seed)
    T = rng.uniform(0.5, 20)
    mk = lambda: [tuple(sorted((rng.uniform(-1, T + 1), rng.uniform(-1, T + 1))))
                  for _ in range(rng.randint(0, 12))]
    P, V = mk(), mk()
    st, out = lib.as2d_interval_accounting(P, V, T)
    assert st == lib.AS2D_OK
    want = [float(x) for x in accounting(P, V, T)] + [T]
    assert out == pytest.approx(want, abs=1e-12)
    assert out[0] + out[1] - out[2] + out[3] == pytest.approx(T, abs=1e-12)


def test_library_argument_errors(lib):
    assert lib.as2d_interval_accounting([(2, 1)], [], 3)[0] == lib.AS2D_ERR_INVALID_ARG
    assert lib.as2d_interval_accounting([], [], -1)[0] == lib.AS2D_ERR_INVALID_ARG
    import ctypes
    stats = lib.as2d_session_stats()
    assert lib._lib.as2d_session_run(None, None, ctypes.byref(stats)) == lib.AS2D_ERR_INVALID_ARG
    spec = lib.as2d_session_spec()
    assert lib._lib.as2d_session_run(ctypes.byref(spec), None, ctypes.byref(stats)) \
        == lib.AS2D_ERR_INVALID_ARG
