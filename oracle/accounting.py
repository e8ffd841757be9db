"""Service-interval accounting of a producer/verifier run, from the paper
(App. D.2 "Overlap, added work, and performance limits": the interval sets
P and V over [0, T], D = |P|, V = |V|, O = |P n V|, H = |[0, T] \\ (P u V)|,
and T = D + V - O + H by inclusion-exclusion).

TEST INFRASTRUCTURE: only tests import it; it shares no code with the
library's C++ (csrc/session.cu).

Written from the definitions: [0, T] is cut at every interval endpoint into
elementary segments; each segment lies wholly inside or wholly outside each
set, so its length is added to the measures of the sets it belongs to.
"""
from fractions import Fraction


def accounting(P, V, T):
    """P, V: iterables of (start, end); returns (D, V, O, H) as Fractions."""
    T = Fraction(T)
    P = [(Fraction(a), Fraction(b)) for a, b in P]
    V = [(Fraction(a), Fraction(b)) for a, b in V]
    cuts = {Fraction(0), T}
    for a, b in P + V:
        if b < a:
            raise ValueError("interval with end < start")
        for x in (a, b):
            if 0 <= x <= T:
                cuts.add(x)
    cuts = sorted(cuts)
    d = v = o = h = Fraction(0)
    for lo, hi in zip(cuts, cuts[1:]):
        mid = (lo + hi) / 2
        in_p = any(a <= mid <= b for a, b in P)
        in_v = any(a <= mid <= b for a, b in V)
        w = hi - lo
        d += w if in_p else 0
        v += w if in_v else 0
        o += w if in_p and in_v else 0
        h += w if not (in_p or in_v) else 0
    return d, v, o, h
