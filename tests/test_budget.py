"""Offline budget selection: the oracle (oracle/budget.py) against cases the
definitions fix, and the library's as2d_budget_select against the oracle.
Host code only."""
import random

import pytest

from oracle import budget as OB

MAXK = 16


def _noisy(ref, rng, p, vocab):
    return [rng.randrange(vocab) if rng.random() < p else t for t in ref]


def test_cost_reduction_closed_forms():
    assert OB.cost_reduction([2.0, 4.0, 6.0]) == [0.0, 0.0, 0.0]        # linear: no saving
    assert OB.cost_reduction([2.0, 2.0, 2.0, 2.0]) == pytest.approx([0, 50, 200 / 3, 75])
    # the paper's example shape: saving can drop as K grows
    r = OB.cost_reduction([1.0, 1.0, 1.2, 1.6, 2.5])
    assert r[3] > r[4]


def test_linear_cost_selects_no_candidates():
    """With cost proportional to width, a call of k candidates costs k + 1
    single calls and commits at most k + 1 tokens, so b = 0 is never beaten."""
    rng = random.Random(0)
    ref = [rng.randrange(30) for _ in range(200)]
    traces = [(ref, _noisy(ref, rng, 0.2, 30))]
    cost = [10.0 * (k + 1) for k in range(MAXK + 1)]
    best, est = OB.select(traces, cost, 8, 120)
    assert best == 0
    assert all(est[0][0] >= r for r, _ in est)


def test_flat_cost_perfect_producer_selects_the_largest_budget():
    ref = list(range(1000, 1300))
    cost = [50.0] * (MAXK + 1)
    best, est = OB.select([(ref, list(ref))], cost, 12, 200)
    assert best == 12
    # every call commits b + 1 tokens: exact call counts
    for b, (_, n) in enumerate(est):
        assert n == -(-200 // (b + 1))


def test_hand_worked_trace():
    """Reference 0..39, producer wrong at position 3, b = 2, flat cost 1 us:
    calls (k, n) = (2,2) (2,0: 3 rejected, corr 3) (2,0: realign fails,
    corr 4) then from 5: (2,2) ... -- counted by hand below."""
    ref = list(range(40))
    prod = list(range(40))
    prod[3] = 99
    cost = [1.0] * (MAXK + 1)
    rate, n_calls = OB.estimate([(ref, prod)], cost, 2, 12)
    # call 1: cands 0 1, both accepted, bonus 2 -> L = 3 (buffer holds 2 at 2: cursor 3)
    # call 2: cands 99 4, rejected at once, corr 3 -> L = 4; realign at 3
    # call 3: root 3 with cands 99 4: rejected, corr 4 -> search finds 4 at 4 -> cursor 5
    # calls 4..: cands 5 6 + bonus -> L = 5 + 3 j
    # L after call 3 = 5; calls 4, 5, 6 -> L = 8, 11, 14 >= 12
    assert n_calls == 6
    assert rate == pytest.approx(14 / 6e-6)


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._lib_build_module().build()
    import paper_2609_37617_gb300 as p
    return p


@pytest.mark.parametrize("seed", range(12))
def test_library_matches_oracle(lib, seed):
    rng = random.Random(50 + seed)
    vocab = rng.choice([4, 50, 1000])
    traces = []
    for _ in range(rng.randint(1, 4)):
        ref = [rng.randrange(vocab) for _ in range(220)]
        prod = _noisy(ref, rng, rng.choice([0.0, 0.1, 0.3, 0.9]), vocab)
        if rng.random() < 0.5:
            prod = prod[:rng.randint(0, len(prod))]
        traces.append((ref, prod))
    cost = sorted(rng.uniform(100, 400) for _ in range(MAXK + 1))
    b_max = rng.choice([0, 4, 8, 16])
    window = rng.choice([4, 8, 16])
    st, best, tok_s, calls = lib.as2d_budget_select(cost, traces, 150, window, b_max)
    assert st == lib.AS2D_OK
    obest, est = OB.select(traces, cost, b_max, 150, window)
    assert calls == [n for _, n in est]
    assert tok_s == pytest.approx([r for r, _ in est], rel=1e-12)
    assert best == obest


def test_library_argument_errors(lib):
    ref = list(range(40))
    st, *_ = lib.as2d_budget_select([1.0] * 17, [(ref, ref)], 30, 8, 17)
    assert st == lib.AS2D_ERR_INVALID_ARG                     # b_max > AS2D_MAX_K
    st, *_ = lib.as2d_budget_select([1.0] * 17, [(ref, ref)], 35, 8, 8)
    assert st == lib.AS2D_ERR_INVALID_ARG                     # reference too short
    st, *_ = lib.as2d_budget_select([0.0] + [1.0] * 16, [(ref, ref)], 20, 8, 8)
    assert st == lib.AS2D_ERR_INVALID_ARG                     # non-positive cost
    st, *_ = lib.as2d_budget_select([1.0] * 17, [], 20, 8, 8)
    assert st == lib.AS2D_ERR_INVALID_ARG                     # no traces
