"""Pins of the candidate-buffer oracle (oracle/candidates.py) against the
paper's worked example (Fig. 4) and the invariants the method fixes."""
import random

import pytest

from oracle import candidates as C

A, B, Cc, D, E, F, X, Y, Z, Q, R, Wt = range(10, 22)
ALL = lambda i: 10 ** 9  # everything published before every call


def test_fig4_token_flow():
    """Fig. 4: the target checks A B C D, accepts A B, corrects C to X and
    commits A B X; its next token D matches the buffer and becomes the root
    for verifying the ready E F."""
    ref = [A, B, X, D, E, F, Y, Y, Y, Y, Y, Y, Y]
    prod = [A, B, Cc, D, E, F]
    calls, committed = C.run_session(ref, prod, ALL, b=4, target_len=7)
    (k0, n0, c0, cur0, _), (k1, n1, c1, cur1, m1), (k2, n2, c2, cur2, m2) = calls[:3]
    assert (k0, n0, c0, cur0) == (4, 2, X, 0)             # A B accepted, X corrects C
    assert committed[:3] == [A, B, X]
    assert (cur1, m1, n1, c1) == (2, C.REALIGN, 0, D)     # C re-offered; target says D
    assert (cur2, m2, k2, n2) == (4, C.NORMAL, 2, 2)      # cursor past D: E F verified, accepted
    assert committed[:6] == [A, B, X, D, E, F]


def test_insertion_keeps_the_mismatch_position():
    ref = [A, B, X, Cc, D, E, F, Y, Y, Y, Y, Y]
    prod = [A, B, Cc, D, E, F]
    calls, _ = C.run_session(ref, prod, ALL, b=4, target_len=7)
    assert calls[0][:3] == (4, 2, X)
    assert calls[1][1] == 4 and calls[1][3] == 2          # C D E F all accepted after X


def test_correction_anchor_when_next_token_is_absent():
    # the target's next token Y is nowhere in the window; the correction X is
    # at 4, so the producer's R (after X) stands in for Y and Z W follow
    ref = [A, B, X, Y, Z, Wt, Y, Y, Y, Y, Y, Y]
    prod = [A, B, Cc, Q, X, R, Z, Wt]
    calls, committed = C.run_session(ref, prod, ALL, b=4, target_len=7)
    assert calls[1][1:3] == (0, Y)
    assert calls[2][3] == 6 and calls[2][1] == 2          # Z W verified and accepted
    assert committed[:6] == [A, B, X, Y, Z, Wt]


def test_unrelated_producer_decodes_alone():
    ref = list(range(100, 140))
    prod = [7] * 24
    calls, committed = C.run_session(ref, prod, ALL, b=4, target_len=20)
    assert committed == ref[:len(committed)] and len(committed) >= 20
    modes = [m for *_, m in calls]
    assert C.ALONE in modes
    assert all(k == 0 for k, _, _, _, m in calls if m == C.ALONE)


def test_substitution_costs_one_call():
    """R2/R3: after a substitution the insertion reading fails once, the next
    target token is found right after the mismatch and the rest is reused."""
    ref = list(range(100, 160))
    prod = list(ref)
    prod[5] = 7
    calls, committed = C.run_session(ref, prod, ALL, b=8, target_len=40)
    k0, n0, c0, _, _ = calls[0]
    assert (k0, n0, c0) == (8, 5, 105)
    assert calls[1][1:5] == (0, 106, 5, C.REALIGN)
    assert calls[2][3] == 7 and calls[2][1] == 8          # cursor past 106: 107.. accepted


def test_bonus_step_over_waits_for_publication():
    """R1: after full acceptance of everything published, the bonus token's
    buffer position is checked once the producer publishes it."""
    ref = list(range(200, 260))
    sched = lambda i: [4, 4, 16, 64][min(i, 3)]
    calls, committed = C.run_session(ref, list(ref), sched, b=8, target_len=30)
    assert calls[0][:2] == (4, 4)                         # 200..203 accepted, bonus 204
    assert calls[1][0] == 0 and calls[1][4] == C.REALIGN  # 204 not yet published: k = 0
    # 205 was decoded alone; once published, the window from position 5 finds it
    assert calls[2][4] == C.NORMAL and calls[2][3] == 6 and calls[2][1] == 8
    assert committed == ref[:len(committed)]


def test_slow_producer_catches_up():
    """The target decodes alone while the producer is behind; the sliding
    window realigns once the producer's text reaches the target's position."""
    ref = list(range(300, 400))
    calls, committed = C.run_session(ref, list(ref), lambda i: max(0, 4 * (i - 10)), b=8,
                                     target_len=90)
    assert committed == ref[:len(committed)]
    modes = [m for *_, m in calls]
    assert C.ALONE in modes
    last_alone = max(i for i, m in enumerate(modes) if m == C.ALONE)
    after = calls[last_alone + 1:]
    assert after and all(n == k for k, n, *_ in after) and max(k for k, *_ in after) >= 2


def test_alone_search_looks_back_after_a_deletion():
    """R3: the producer's text lost a token inside the stretch the target
    decoded alone, so the target's tokens sit one position behind the window
    start; the look-back finds the anchor and candidates resume."""
    ref = list(range(100, 200))
    prod = list(ref)
    for i in range(1, 12):
        prod[i] = 900 + i      # junk: the realign search fails, the target decodes alone
    del prod[5]                # every later position moves back by one
    calls, comm = C.run_session(ref, prod, lambda i: 10 ** 9, b=4, window=4, target_len=60)
    assert comm == ref[:len(comm)]
    modes = [m for *_, m in calls]
    first_normal_after = next(i for i in range(3, len(calls)) if modes[i] == C.NORMAL)
    # the anchor 112 sits at position 11 while the window starts at 12
    assert calls[first_normal_after][3] == 12
    assert any(n >= 2 for _, n, *_ in calls[first_normal_after:first_normal_after + 3])
    assert len(calls) < 30


def test_batches_are_immutable_and_bounded():
    buf = C.CandidateBuffer()
    with pytest.raises(ValueError):
        buf.publish(list(range(9)), None)
    buf.publish([1, 2, 3], C.SourceRecord(0, 0, 0, 0, 0.0))
    snap = buf.candidates(8)
    buf.publish([4, 5], C.SourceRecord(0, 0, 0, 3, 1.0))
    assert snap == [1, 2, 3] and buf.candidates(8) == [1, 2, 3, 4, 5]
    assert [r[0] for r in buf.records] == [0, 3]
    assert buf.source_of(2).offset == 0 and buf.source_of(3).offset == 3
    with pytest.raises(IndexError):
        buf.source_of(5)


@pytest.mark.parametrize("seed", range(20))
def test_session_invariants(seed):
    """Random producers (the target's text with substitutions, insertions,
    deletions) published 8 at a time: the committed text is always the
    target's own greedy text (Prop. 1), the cursor never moves back, and
    only published tokens are ever verified."""
    rng = random.Random(seed)
    ref = [rng.randrange(50) for _ in range(400)]
    prod = []
    for t in ref:
        r = rng.random()
        if r < 0.08:
            prod.append(rng.randrange(50))           # substitution
        elif r < 0.12:
            prod += [t, rng.randrange(50)]           # insertion
        elif r < 0.15:
            pass                                     # deletion
        else:
            prod.append(t)
    rate = rng.choice([4, 8, 16])
    calls, committed = C.run_session(ref, prod, lambda i: 8 + rate * i, b=8, target_len=300)
    assert committed == ref[:len(committed)] and len(committed) >= 300
    curs = [c for _, _, _, c, m in calls if m != C.ALONE]
    assert all(a <= b for a, b in zip(curs, curs[1:]))
    published = 8
    for i, (k, n, corr, cur, mode) in enumerate(calls):
        published = min(8 + rate * i, len(prod))
        assert 0 <= k <= 8 and cur + k <= max(published, cur)


def test_perfect_producer_accepts_every_block():
    ref = list(range(1000, 1200))
    calls, committed = C.run_session(ref, list(ref), ALL, b=8, target_len=180)
    assert all(n == k == 8 for k, n, *_ in calls)
    assert len(calls) == -(-180 // 9)
