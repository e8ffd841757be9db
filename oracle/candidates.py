"""Candidate buffer, read cursor and candidate alignment, written from the
paper (Section 3.1 "Ordered publication and buffering"; Section 3.2
"Candidate alignment"; App. C.1 "Source records and incremental
publication"; App. C.3 "Candidate alignment"; Fig. 4).

TEST INFRASTRUCTURE: plain Python, no shared code with the library's C++
implementation (csrc/cand_buffer.cu); only tests import it.

The producer appends immutable batches of at most eight tokens, each with a
source record.  Verification reads only published tokens.  A read cursor,
separate from the producer, says where the next usable candidates start.

Readings taken where the paper leaves the rule open (also listed in the
design notes):
  R1  a call that verified k candidates from the cursor c and accepted n of
      them ends with the target's own token x (the correction when n < k,
      the bonus token when n == k); x stands at buffer position m = c + n.
      If the buffer holds x at m (possible only after full acceptance, and
      checked again once m is published), the cursor steps over it to m + 1;
      so full acceptance advances the cursor by k, plus one when the
      producer also predicted the bonus token;
  R2  otherwise m stays eligible: the next call verifies root x followed by
      the candidates from m (the target may have inserted x), and if it
      accepts n >= 1 of them, R1 applies to it;
  R3  if that call accepts none, its correction t is the next target token,
      the first alignment anchor: the cursor moves just past the first
      position j in (m, m + W] holding t; failing that, to j + 2 for the
      first position j in [m, m + W] holding x (the producer's token after x
      stands in for t, and its continuation after that is verified under
      root t); failing that, the target decodes alone (k = 0).  While it
      does, its latest token u is the anchor, looked for before each call
      first in the published positions [s, s + W) in increasing order, then
      in [max(f, s - W), s) from s - 1 down, f = m + 1 being where the
      target began decoding alone and s starting at f; a match at j moves
      the cursor to j + 1.  Every token decoded alone advances s by one, so
      the window keeps pace with the target when the producer is behind, and
      looking back W positions recovers from deletions in the producer's
      text (positions below f, or more than W behind s, are retired).
  W is the search bound (default 8).
Correctness does not depend on any of this: every candidate is verified
under the current committed prefix, so the committed text is the target's
own greedy text whatever the buffer holds (Prop. 1).
"""

NORMAL, REALIGN, ALONE = "normal", "realign", "alone"


class SourceRecord:
    """App. C.1: request, audio view (source), producer, token offset,
    publication time, confidence (None when unavailable)."""

    def __init__(self, request, source, producer, offset, time, confidence=None):
        self.request = request
        self.source = source
        self.producer = producer
        self.offset = offset
        self.time = time
        self.confidence = confidence


class CandidateBuffer:
    """Published tokens of one request and source, in publication order."""

    BATCH = 8

    def __init__(self, window=8):
        self.tokens = []
        self.records = []      # (start index, record) per published batch
        self.window = window
        self.cursor = 0
        self.mode = NORMAL
        self.m = 0             # REALIGN: position of x; ALONE: search start
        self.x = None          # REALIGN: the call's final token; ALONE: the anchor
        self.f = 0             # ALONE: the first position of the alone search

    def publish(self, tokens, record):
        """Append one immutable batch of at most eight tokens."""
        tokens = list(tokens)
        if not 1 <= len(tokens) <= self.BATCH:
            raise ValueError("a batch holds 1..8 tokens")
        self.records.append((len(self.tokens), record))
        self.tokens.extend(tokens)

    def ready(self):
        return len(self.tokens)

    def source_of(self, i):
        """App. C.1: the source record of the batch that published position i."""
        if not 0 <= i < len(self.tokens):
            raise IndexError(i)
        rec = None
        for start, r in self.records:
            if start > i:
                break
            rec = r
        return rec

    def _settle(self):
        """Before each call: R1's step over position m once the buffer holds x
        there, and R3's search for the anchor while the target decodes alone."""
        tok = self.tokens
        if self.mode == REALIGN and self.m < len(tok) and tok[self.m] == self.x:
            self.cursor, self.mode = self.m + 1, NORMAL
        elif self.mode == ALONE:
            ahead = range(self.m, min(self.m + self.window, len(tok)))
            behind = range(min(self.m, len(tok)) - 1, max(self.f, self.m - self.window) - 1, -1)
            for j in list(ahead) + list(behind):
                if tok[j] == self.x:
                    self.cursor, self.mode = j + 1, NORMAL
                    return

    def candidates(self, b):
        """Candidates for the next call: up to b published tokens from the
        cursor; none while the target decodes alone."""
        self._settle()
        if self.mode == ALONE:
            return []
        return self.tokens[self.cursor:self.cursor + b]

    def after_call(self, k, n, corr):
        """Update the cursor after a call that verified k candidates from the
        cursor, accepted n of them and ended with the target token corr."""
        if self.mode == ALONE:                    # k == 0: corr is the new anchor
            self.m += 1
            self.cursor, self.x = self.m, corr
        elif self.mode == NORMAL or n >= 1:       # R1 / R2
            self.m, self.x = self.cursor + n, corr
            self.cursor, self.mode = self.m, REALIGN
        else:                                     # R3: the insertion reading failed
            self._search(corr)

    def _search(self, t):
        W, tok, m = self.window, self.tokens, self.m
        last = len(tok) - 1
        for j in range(m + 1, min(m + W, last) + 1):
            if tok[j] == t:
                self.cursor, self.mode = j + 1, NORMAL
                return
        for j in range(m, min(m + W, last) + 1):
            if tok[j] == self.x:
                self.cursor, self.mode = j + 2, NORMAL
                return
        self.mode, self.m, self.x = ALONE, m + 1, t
        self.f = self.m
        self.cursor = self.m


def verify(ref, L, cands):
    """The greedy verification rule against the target's reference greedy
    text ref (ref[i] is the target token at committed position i):
    returns (n_accepted, correction)."""
    n = 0
    while n < len(cands) and cands[n] == ref[L + n]:
        n += 1
    return n, ref[L + n]


def run_session(ref, producer, publish_before_call, b=8, window=8, max_calls=10000,
                target_len=None):
    """Drive verification calls with a synthetic producer.

    ref      target's greedy text (the committed text must equal its prefix)
    producer the producer's own token sequence, published in batches of 8
    publish_before_call(i) -> number of producer tokens published before call i
    Returns (calls, committed) with calls = [(k, n, corr, cursor_before, mode_before)].
    """
    buf = CandidateBuffer(window)
    target_len = len(ref) - b - 1 if target_len is None else target_len
    L, calls, published = 0, [], 0
    for i in range(max_calls):
        if L >= target_len:
            break
        want = min(publish_before_call(i), len(producer))
        while published < want:
            nb = min(CandidateBuffer.BATCH, want - published)
            buf.publish(producer[published:published + nb],
                        SourceRecord(0, 0, 0, published, i))
            published += nb
        cands = buf.candidates(b)
        cur, mode = buf.cursor, buf.mode
        n, corr = verify(ref, L, cands)
        calls.append((len(cands), n, corr, cur, mode))
        L += n + 1
        buf.after_call(len(cands), n, corr)
    return calls, ref[:L]
