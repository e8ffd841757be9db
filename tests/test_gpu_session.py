"""Verification driven by candidate buffers on the GPU (as2d_verify_from_buffers):
a synthetic producer publishes a noisy copy of the target's greedy text in
8-token batches; the session must commit exactly the target's greedy text
(Prop. 1), the buffer must hand out what the oracle's buffer hands out, and
the committed text must equal plain one-token decoding on the same path."""
import random

import numpy as np
import pytest

import oracle
from oracle import candidates as C
from synth import workloads as W
from tests.helpers import MARGIN_SURE, Pair

pytestmark = pytest.mark.gpu

L0, CAP, N_TOK = 200, 512, 72


@pytest.fixture(scope="module")
def pair():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.TINY, seed=0)


def _producer(cont, seed, vocab):
    """The target's text with seeded substitutions, insertions and deletions."""
    rng = random.Random(seed)
    out = []
    for t in cont:
        r = rng.random()
        if r < 0.08:
            out.append(rng.randrange(vocab))
        elif r < 0.12:
            out += [int(t), rng.randrange(vocab)]
        elif r < 0.15:
            continue
        else:
            out.append(int(t))
    return out


def _session(lib, st, prods, b, n_tok, rate):
    """Run calls until every request committed n_tok tokens; mirror each
    request's buffer with the oracle's buffer fed the GPU's outcomes."""
    B = len(prods)
    bufs = [lib.CandidateBuffer(8) for _ in range(B)]
    mirrors = [C.CandidateBuffer(8) for _ in range(B)]
    published = [0] * B
    committed = [[] for _ in range(B)]
    calls = 0
    while min(len(c) for c in committed) < n_tok:
        for r in range(B):
            want = min(8 + rate * calls, len(prods[r]))
            while published[r] < want:
                nb = min(8, want - published[r])
                batch = prods[r][published[r]:published[r] + nb]
                bufs[r].publish(batch, request=r, offset=published[r], time=float(calls))
                mirrors[r].publish(batch, C.SourceRecord(r, 0, 0, published[r], calls))
                published[r] += nb
        expect = [m.candidates(b) for m in mirrors]
        k_used, rows = st.verify_from_buffers(bufs, b)
        for r in range(B):
            n, corr = len(rows[r]) - 1, rows[r][-1]
            assert k_used[r] == len(expect[r]), f"call {calls} request {r}"
            assert rows[r][:n] == expect[r][:n]
            mirrors[r].after_call(len(expect[r]), n, corr)
            committed[r] += rows[r]
        calls += 1
        assert calls <= 4 * n_tok
    st.check()
    return committed, calls


def _sure_prefix(margins):
    """Number of leading greedy tokens whose oracle margin is decisive."""
    bad = np.nonzero(margins <= MARGIN_SURE)[0]
    return int(bad[0]) if bad.size else len(margins)


def test_session_commits_the_greedy_text(pair):
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    root = int(W.root_tokens(cfg, 1, 0)[0])
    oc = pair.oracle_cache(L0, CAP)
    cont, margins = oracle.greedy_continuation(pair.oracle, oc, L0, root, N_TOK + 16)
    prod = _producer(cont, 5, cfg.vocab)
    st = pair.state([L0], CAP, [root])
    (got,), calls = _session(lib, st, [prod], 8, N_TOK, 16)
    sure = _sure_prefix(margins)
    m = min(sure, len(got))
    assert got[:m] == [int(t) for t in cont[:m]]
    assert calls < len(got)                     # candidates were accepted
    ln, rt = st.read_state()
    assert ln == [L0 + len(got)] and rt == [got[-1]]
    st.close()

    # the same text by plain one-token decoding on the same path
    import torch
    st2 = pair.state([L0], CAP, [root])
    nn = torch.zeros(1, dtype=torch.int32, device="cuda")
    cc = torch.zeros(1, dtype=torch.int32, device="cuda")
    plain = []
    for _ in range(len(got)):
        st2.decode(nn, cc)
        torch.cuda.synchronize()
        plain.append(int(cc.item()))
    assert plain == got
    st2.close()


def test_two_requests_perfect_and_unrelated_producers(pair):
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    roots = [int(t) for t in W.root_tokens(cfg, 2, 0)]
    conts, sures = [], []
    for r in range(2):
        oc = pair.oracle_cache(L0, CAP, req=r)
        cont, margins = oracle.greedy_continuation(pair.oracle, oc, L0, roots[r], 48 + 16)
        conts.append([int(t) for t in cont])
        sures.append(_sure_prefix(margins))
    prods = [list(conts[0]), [(t * 7 + 3) % cfg.vocab for t in range(200)]]
    st = pair.state([L0, L0], CAP, roots)
    got, calls = _session(lib, st, prods, 8, 48, 64)
    for r in range(2):
        m = min(sures[r], len(got[r]))
        assert got[r][:m] == conts[r][:m], f"request {r}"
    st.close()


def test_empty_buffer_is_plain_decoding(pair):
    """No producer at all: every call has k = 0 (the target decodes alone)."""
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    root = int(W.root_tokens(cfg, 1, 0)[0])
    st = pair.state([L0], CAP, [root])
    buf = lib.CandidateBuffer()
    for _ in range(5):
        k_used, rows = st.verify_from_buffers([buf], 8)
        assert k_used == [0] and len(rows[0]) == 1
    assert buf.state()[2] in ("realign", "alone")
    st.close()


def _run_session(lib, pair, drafter, root, script, overlapped, n_commit):
    import torch
    st = pair.state([L0], CAP, [root])
    dst = drafter.state([L0], CAP, [int(W.root_tokens(drafter.cfg, 1, 1)[0])])
    s_t, s_d = torch.cuda.Stream(), torch.cuda.Stream()
    buf = lib.CandidateBuffer(8)
    comm, stats = lib.session_run(st, dst, buf, script, 8, n_commit, overlapped,
                                  target_stream=s_t.cuda_stream, drafter_stream=s_d.cuda_stream)
    ln, rt = st.read_state()
    assert ln == [L0 + len(comm)] and rt == [comm[-1]]
    st.check()
    dst.check()
    st.close()
    dst.close()
    return comm, stats


def test_session_runner_serial_and_overlapped(pair):
    """as2d_session_run with a drafter decoding on its own stream: both
    schedules commit the target's greedy text, and the accounting satisfies
    T = D + V - O + H with no overlap in the serial comparator."""
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    drafter = Pair(W.TINY, seed=1)
    root = int(W.root_tokens(cfg, 1, 0)[0])
    oc = pair.oracle_cache(L0, CAP)
    cont, margins = oracle.greedy_continuation(pair.oracle, oc, L0, root, N_TOK + 24)
    script = _producer(cont, 9, cfg.vocab)[:N_TOK + 16]
    sure = _sure_prefix(margins)
    runs = {}
    for overlapped in (False, True):
        comm, stats = _run_session(lib, pair, drafter, root, script, overlapped, N_TOK)
        assert len(comm) >= N_TOK and len(comm) == stats["committed"]
        m = min(sure, len(comm))
        assert comm[:m] == [int(t) for t in cont[:m]]
        T, D, V, O, H = (stats[x] for x in "TDVOH")
        assert abs(D + V - O + H - T) < 1e-9 * max(T, 1.0)
        assert 0 <= O <= min(D, V) + 1e-12 and T >= max(D, V) + H - 1e-9
        assert stats["accepted"] == stats["committed"] - stats["rounds"]
        assert stats["producer_steps"] == stats["published"] <= len(script)
        runs[overlapped] = (comm, stats)
    assert runs[False][1]["O"] == 0.0
    n = min(len(runs[False][0]), len(runs[True][0]))
    assert runs[False][0][:n] == runs[True][0][:n]
