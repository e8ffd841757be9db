"""The library's candidate buffer (C-ABI as2d_cbuf_*) against the oracle's
(oracle/candidates.py): the same sessions give the same candidates, cursor
and mode at every call.  Host code only: no GPU needed."""
import random
import threading

import pytest

from oracle import candidates as C


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._lib_build_module().build()
    import paper_2609_37617_gb300 as p
    return p


def _noisy(ref, rng, sub, ins, dele, vocab):
    out = []
    for t in ref:
        r = rng.random()
        if r < sub:
            out.append(rng.randrange(vocab))
        elif r < sub + ins:
            out += [t, rng.randrange(vocab)]
        elif r < sub + ins + dele:
            pass
        else:
            out.append(t)
    return out


def _lockstep(lib, ref, prod, sched, b, window, target_len):
    """Drive the oracle's buffer and the library's with the same publications
    and the same simulated target; compare everything each call."""
    ob = C.CandidateBuffer(window)
    lb = lib.CandidateBuffer(window)
    L, published, calls = 0, 0, 0
    while L < target_len:
        want = min(sched(calls), len(prod))
        while published < want:
            nb = min(8, want - published)
            batch = prod[published:published + nb]
            ob.publish(batch, C.SourceRecord(0, 0, 0, published, calls))
            lb.publish(batch, offset=published, time=float(calls))
            published += nb
        oc = ob.candidates(b)
        lc = lb.candidates(b)
        assert lc == oc, f"call {calls}"
        ready, cursor, mode = lb.state()
        assert (ready, cursor, mode) == (len(ob.tokens), ob.cursor, ob.mode), f"call {calls}"
        n, corr = C.verify(ref, L, oc)
        ob.after_call(len(oc), n, corr)
        lb.after_call(len(lc), n, corr)
        L += n + 1
        calls += 1
        assert calls < 10000
    return calls


def test_fig4_session_matches_oracle(lib):
    A, B, Cc, D, E, F, X, Y = range(10, 18)
    _lockstep(lib, [A, B, X, D, E, F] + [Y] * 12, [A, B, Cc, D, E, F], lambda i: 99, 4, 8, 7)


@pytest.mark.parametrize("seed", range(40))
def test_random_sessions_match_oracle(lib, seed):
    rng = random.Random(1000 + seed)
    vocab = rng.choice([3, 20, 1000])       # tiny vocabularies make repeated-token anchors
    ref = [rng.randrange(vocab) for _ in range(600)]
    sub, ins, dele = rng.choice([(0.0, 0.0, 0.0), (0.05, 0.03, 0.03), (0.2, 0.1, 0.1),
                                 (1.0, 0.0, 0.0)])
    prod = _noisy(ref, rng, sub, ins, dele, vocab)
    rate = rng.choice([1, 3, 8, 16, 64])
    start = rng.choice([0, 8, 40])
    b = rng.choice([0, 1, 4, 8, 16])
    window = rng.choice([1, 4, 8, 32])
    _lockstep(lib, ref, prod, lambda i: start + rate * i, b, window, 450)


def test_source_records(lib):
    buf = lib.CandidateBuffer()
    buf.publish([1, 2, 3], request=4, source=1, producer=2, offset=0, time=0.5)
    buf.publish([4, 5], request=4, source=1, producer=2, offset=3, time=0.75, confidence=0.9)
    assert buf.source_of(0)["offset"] == 0 and buf.source_of(2)["time"] == 0.5
    r = buf.source_of(4)
    assert r["offset"] == 3 and r["request"] == 4 and abs(r["confidence"] - 0.9) < 1e-6
    assert buf.source_of(1)["confidence"] is None
    with pytest.raises(lib.AS2DError):
        buf.source_of(5)
    with pytest.raises(lib.AS2DError):
        buf.source_of(-1)


def test_argument_errors(lib):
    import ctypes
    st, h = lib.as2d_cbuf_create(0)
    assert st == lib.AS2D_ERR_INVALID_ARG and h is None
    buf = lib.CandidateBuffer()
    for bad in ([], list(range(9)), [1, -2]):
        with pytest.raises(lib.AS2DError):
            buf.publish(bad)
    assert lib.as2d_cbuf_publish(buf.handle, [1], None) == lib.AS2D_ERR_INVALID_ARG
    assert buf.state() == (0, 0, "normal")                # nothing was published
    with pytest.raises(lib.AS2DError):
        buf.candidates(17)
    buf.publish([5, 6])
    assert buf.candidates(8) == [5, 6]
    for k, n, x in ((1, 0, 3), (2, 3, 3), (2, 1, -1)):      # wrong k, n > k, bad token
        with pytest.raises(lib.AS2DError):
            buf.after_call(k, n, x)
    buf.after_call(2, 2, 7)
    with pytest.raises(lib.AS2DError):                    # no candidates() since
        buf.after_call(0, 0, 7)
    assert lib._lib.as2d_cbuf_state(None, None, None, None) == lib.AS2D_ERR_INVALID_ARG
    vb = (ctypes.c_void_p * 1)(buf.handle)
    assert lib._lib.as2d_verify_from_buffers(None, vb, 4, None, None, None, None) \
        == lib.AS2D_ERR_INVALID_ARG
    lib.as2d_cbuf_free(None)


def test_concurrent_publisher(lib):
    """A producer thread publishes while the verifier reads: every snapshot is
    a run of the producer's sequence, and the session still commits exactly
    the target's text."""
    rng = random.Random(7)
    ref = [rng.randrange(50) for _ in range(3000)]
    prod = _noisy(ref, rng, 0.05, 0.02, 0.02, 50)
    buf = lib.CandidateBuffer()

    def producer():
        for i in range(0, len(prod), 8):
            buf.publish(prod[i:i + 8], offset=i)

    th = threading.Thread(target=producer)
    th.start()
    L, committed = 0, []
    while L < 2000:
        _, cursor, _ = buf.state()
        cands = buf.candidates(8)
        ready, cur2, mode = buf.state()
        if cands:
            assert cands == prod[cur2:cur2 + len(cands)]
        n, corr = C.verify(ref, L, cands)
        committed += cands[:n] + [corr]
        buf.after_call(len(cands), n, corr)
        L += n + 1
    th.join()
    assert committed == ref[:len(committed)]


def test_long_session_holds_a_bounded_buffer(lib):
    """Long sessions: the library's buffer drops what no rule reads again
    (positions stay absolute) and still agrees call by call with the
    oracle's, which keeps everything."""
    rng = random.Random(99)
    ref = [rng.randrange(200) for _ in range(30500)]
    prod = _noisy(ref, rng, 0.05, 0.02, 0.02, 200)
    _lockstep(lib, ref, prod, lambda i: 64 + 16 * i, 16, 8, 20000)
    buf = lib.CandidateBuffer()
    L = 0
    for i in range(0, 24000, 8):
        buf.publish(prod[i:i + 8], offset=i)
    seen_max = 0
    while L < 20000:
        c = buf.candidates(16)
        n, corr = C.verify(ref, L, c)
        buf.after_call(len(c), n, corr)
        L += n + 1
        seen_max = max(seen_max, buf.held()[0])
    held, recs = buf.held()
    ready, cursor, _ = buf.state()
    assert ready == 24000 and cursor > 15000
    assert held < 24000 - 8000 and recs <= held // 8 + 2
    with pytest.raises(lib.AS2DError):
        buf.source_of(0)                      # dropped
    assert buf.source_of(ready - 1)["offset"] == 24000 - 8

