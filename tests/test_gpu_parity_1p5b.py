"""GPU parity on the 1.5B-class decoder (28 layers, hidden 1536, 12/2 heads,
head_dim 128, FFN 8960, vocab 151936) with 814 prefilled positions (750 audio
+ 64 instruction), k swept over {0, 1, 2, 4, 8}, candidates = the target's
greedy continuation with each place corrupted w.p. 0.3."""
import numpy as np
import pytest

import oracle
from synth import workloads as W
from tests.helpers import ExactTally, Pair, check_parity, oracle_block, run_gpu_block

pytestmark = pytest.mark.gpu
TALLY = ExactTally()

L0 = 814
CAP = L0 + 64


@pytest.fixture(scope="module")
def pair():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.M1P5B, seed=0)


@pytest.fixture(scope="module")
def continuation(pair):
    root = int(W.root_tokens(pair.cfg, 1, 0)[0])
    oc = pair.oracle_cache(L0, CAP)
    cont, margins = oracle.greedy_continuation(pair.oracle, oc, L0, root, 9)
    return root, oc, cont, margins


@pytest.mark.parametrize("k", [0, 1, 2, 4, 8])
def test_1p5b_k_sweep(pair, continuation, k):
    root, oc, cont, margins = continuation
    rng = np.random.default_rng(100 + k)
    cand = W.corrupt_each(cont[:k], 0.3, rng, pair.cfg.vocab)
    ores = oracle_block(pair, oc.copy(pair.oracle), L0, root, cand)
    st = pair.state([L0], CAP, [root])
    gpu = run_gpu_block(st, pair.cfg, [cand])
    check_parity(ores, gpu, 0, k, f"k={k}", TALLY)
    ln, rt = st.read_state()
    assert ln == [L0 + gpu[0][0] + 1] and rt == [gpu[1][0]]
    st.check()
    st.close()


def test_1p5b_two_consecutive_blocks(pair, continuation):
    """State carried across calls: the second block starts from the first
    block's committed length and root, on both sides."""
    root, oc, cont, _ = continuation
    cache = oc.copy(pair.oracle)
    st = pair.state([L0], CAP, [root])
    length, r = L0, root
    cands = [list(cont[:4]), None]
    for blk in range(2):
        if cands[blk] is None:
            nxt, _ = oracle.greedy_continuation(pair.oracle, cache, length, r, 4)
            cands[blk] = list(W.corrupt_each(nxt, 0.3, np.random.default_rng(7), pair.cfg.vocab))
        ores = oracle_block(pair, cache, length, r, cands[blk])
        gpu = run_gpu_block(st, pair.cfg, [cands[blk]])
        d, sure, n, corr = check_parity(ores, gpu, 0, 4, f"block {blk}", TALLY)
        if not sure and (gpu[0][0] != n or gpu[1][0] != corr):
            pytest.skip("a near tie (margin <= 0.1) changed the committed tokens")
        length, r = ores["new_len"], ores["new_root"]
        assert st.read_state() == ([length], [r])
    st.close()


def test_zz_exact_checks_ran():
    """Some of this module's greedy rows and commits were compared bit for
    bit (their oracle margins exceed 0.1), not only the logits."""
    TALLY.assert_ran(rows=1, blocks=1)
