"""GPU parity on the tiny decoder (2 layers, hidden 256, 4/2 heads, head_dim
64, FFN 704, vocab 4096, 200 prefilled positions, k = 4 with place 2
replaced), and the verification invariants on the GPU path, all through the
C-ABI."""
import numpy as np
import pytest

import oracle
from synth import workloads as W
from tests.helpers import (ExactTally, Pair, bf16_bits, compare_block, run_gpu_block,
                           sharp_root)

pytestmark = pytest.mark.gpu

L0, CAP = 200, 256
TALLY = ExactTally()


@pytest.fixture(scope="module")
def pair():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.TINY, seed=0)


@pytest.fixture(scope="module")
def pair_sharp():
    """The tiny shape with the final norm's gain at 8 (logits x 8), so that
    greedy decisions are separated by more than the 0.1 margin."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.TINY, seed=0, gains="sharp")


@pytest.fixture(scope="module")
def sharp_continuation(pair_sharp):
    """Searched on the oracle: the first root whose 9-token greedy
    continuation from 200 positions has every margin above 0.1."""
    p = pair_sharp
    root, cont, margins = sharp_root(p.oracle, lambda: p.oracle_cache(L0, CAP), L0, 9)
    return root, cont, margins


@pytest.fixture(scope="module")
def pair_gains():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.TINY, seed=3, gains="random")


def _workload_block(p, gains_seed=0):
    cfg = p.cfg
    root = int(W.root_tokens(cfg, 1, p.seed)[0])
    oc = p.oracle_cache(L0, CAP)
    cont, _ = oracle.greedy_continuation(p.oracle, oc, L0, root, 4)
    cand = W.replace_at(cont, 2, np.random.default_rng(gains_seed), cfg.vocab)
    return root, oc, cont, cand


def test_device_inputs_match_host_inputs(pair):
    import torch
    from synth import device as D
    cfg = W.TINY
    dw = D.device_weights(cfg, 0)
    hw = W.host_weights(cfg, 0)
    for name in ("embed", "w_q.0", "w_down.1", "lm_head", "attn_norm.0"):
        assert np.array_equal(bf16_bits(dw[name]), hw[name]), name
    kc, vc = D.device_kv(cfg, [L0], CAP, 0)
    ks, vs = W.host_kv_request(cfg, 0, L0, CAP, 0)
    for l in range(cfg.n_layers):
        assert np.array_equal(bf16_bits(kc[l, 0])[:, :L0], ks[l][:, :L0])
        assert np.array_equal(bf16_bits(vc[l, 0])[:, :L0], vs[l][:, :L0])
    torch.cuda.synchronize()


@pytest.mark.parametrize("which", ["unit_gains", "random_gains"])
def test_tiny_block_parity(which, request):
    p = request.getfixturevalue("pair" if which == "unit_gains" else "pair_gains")
    cfg = p.cfg
    root, oc, cont, cand = _workload_block(p)
    ores = p.oracle.verify_block(oc, L0, root, cand)
    st = p.state([L0], CAP, [root])
    n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
    compare_block(ores, logits[:5], greedy[:5], n[0], corr[0], 4, TALLY)
    ln, rt = st.read_state()
    assert ln == [L0 + n[0] + 1] and rt == [corr[0]]
    # the KV entries kept for the committed rows match the oracle's
    keep = L0 + n[0] + 1
    for l in range(cfg.n_layers):
        gk = bf16_bits(st.kc[l, 0])[:, L0:keep].view(np.uint16)
        ok = oc.k[l][:, L0:keep]
        dk = np.abs(((gk.astype(np.uint32) << 16).view(np.float32)) -
                    ((ok.astype(np.uint32) << 16).view(np.float32)))
        assert dk.max() < 3e-2
    st.check()
    st.close()


def test_full_acceptance_and_bonus(pair_sharp, sharp_continuation):
    """Invariant I1 (Prop. 1): candidates equal to the target's own greedy
    continuation are all accepted and the correction is the bonus token.
    Every margin of the continuation exceeds 0.1, so this is asserted
    unconditionally."""
    cfg = pair_sharp.cfg
    root, cont, margins = sharp_continuation
    assert np.all(np.asarray(margins) > 0.1)
    st = pair_sharp.state([L0], CAP, [root])
    n, corr, greedy, _ = run_gpu_block(st, cfg, [cont[:8]], want_logits=False)
    assert n[0] == 8 and corr[0] == cont[8]
    assert np.array_equal(greedy, np.asarray(cont[:9]))
    TALLY.rows += 9
    TALLY.blocks += 1
    ln, rt = st.read_state()
    assert ln == [L0 + 9] and rt == [cont[8]]
    st.close()


def test_sharp_workload_block(pair_sharp, sharp_continuation):
    """The workload's block shape (k = 4, place 2 replaced) on the sharp
    model: the rejection at place 2 and its correction are compared bit for
    bit, since every row they depend on has a margin above 0.1."""
    cfg = pair_sharp.cfg
    root, cont, _ = sharp_continuation
    cand = W.replace_at(cont[:4], 2, np.random.default_rng(0), cfg.vocab)
    oc = pair_sharp.oracle_cache(L0, CAP)
    ores = pair_sharp.oracle.verify_block(oc, L0, root, cand)
    assert ores["n_accepted"] == 2 and ores["correction"] == cont[2]
    st = pair_sharp.state([L0], CAP, [root])
    n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
    blocks = TALLY.blocks
    compare_block(ores, logits[:5], greedy[:5], n[0], corr[0], 4, TALLY)
    assert TALLY.blocks == blocks + 1
    st.close()


def test_block_equals_sequential_decode_bitwise(pair):
    """Pathwise equivalence held bit for bit: row i of a k-block has exactly the
    logits of the i-th of k+1 single-token decode steps (App. C.4, req. 1)."""
    import torch
    cfg = pair.cfg
    root = int(W.root_tokens(cfg, 1, 0)[0])
    cand = [11, 22, 33, 44, 55, 66]
    st = pair.state([L0], CAP, [root])
    n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
    st2 = pair.state([L0], CAP, [root])
    toks = [root] + cand
    for i in range(len(toks)):
        # force the next root to be the block's token i+1 by rolling back
        nn = torch.zeros(1, dtype=torch.int32, device="cuda")
        cc = torch.zeros(1, dtype=torch.int32, device="cuda")
        lg = torch.empty((1, cfg.vocab), dtype=torch.float32, device="cuda")
        st2.rollback([L0 + i], [toks[i]])
        st2.decode(nn, cc, None, lg)
        torch.cuda.synchronize()
        assert np.array_equal(lg.cpu().numpy()[0], logits[i]), f"row {i}"
    st.close()
    st2.close()


def test_k0_is_decode_and_rollback_restores(pair):
    import torch
    cfg = pair.cfg
    root = int(W.root_tokens(cfg, 1, 0)[0])
    st = pair.state([L0], CAP, [root])
    n0, c0, g0, lg0 = run_gpu_block(st, cfg, [[]])
    assert n0[0] == 0 and c0[0] == g0[0] == int(np.argmax(lg0[0]))
    ln, rt = st.read_state()
    assert ln == [L0 + 1] and rt == [c0[0]]
    st.rollback([L0], [root])
    n1, c1, g1, lg1 = run_gpu_block(st, cfg, [[]])
    assert np.array_equal(lg0, lg1) and c1[0] == c0[0]
    st.close()


def test_rejected_rows_never_read(pair):
    """Reject at place 1, then continue: the NaN-poisoned tail beyond the
    prefix and the rejected rows' stale entries never reach a logit."""
    cfg = pair.cfg
    root = int(W.root_tokens(cfg, 1, 0)[0])
    st = pair.state([L0], CAP, [root])
    for _ in range(6):
        n, corr, greedy, logits = run_gpu_block(st, cfg, [[1, 2, 3, 4, 5]])
        assert np.all(np.isfinite(logits))
    st.check()
    st.close()


def test_batch_of_requests_matches_single(pair):
    """Three requests with different lengths and k in one call give, row for
    row, the bitwise logits of each request verified alone."""
    cfg = pair.cfg
    lens = [200, 37, 120]
    roots = [5, 6, 7]
    cands = [[1, 2, 3], [], [9, 8, 7, 6, 5, 4, 3, 2, 1, 0, 11, 12, 13, 14, 15, 16]]
    st = pair.state(lens, CAP, roots)
    n, corr, greedy, logits = run_gpu_block(st, cfg, cands)
    row = 0
    for b in range(3):
        single = pair.state([lens[b]], CAP, [roots[b]], kv_seed=None)
        # request b of the batch drew its cache from stream (layer, b, head);
        # rebuild the same cache for a batch-of-one state
        import torch
        from synth import device as D
        kc, vc = D.device_kv(cfg, lens, CAP, pair.seed)
        single.kc.copy_(kc[:, b:b + 1])
        single.vc.copy_(vc[:, b:b + 1])
        torch.cuda.synchronize()
        n1, c1, g1, lg1 = run_gpu_block(single, cfg, [cands[b]])
        k = len(cands[b])
        assert np.array_equal(lg1, logits[row:row + k + 1])
        assert n1[0] == n[b] and c1[0] == corr[b]
        row += k + 1
        single.close()
    st.close()


LAYOUT_BATCHES = {
    # 2, 4, 1, 3, 4 and 4 chunks: 36 clusters of 8 over the two kv heads
    "narrow": ([1500, 3100, 300, 2600, 4000, 3900], (4, 2, 6, 0, 3, 5)),
    # 36 chunks: 72 clusters of 8, more than the narrow layout keeps resident
    "quad": ([1500, 3100, 300, 2600, 4000, 3900, 3500, 2000, 1000, 3800, 4050, 2500],
             (4, 2, 6, 0, 3, 5, 1, 7, 2, 0, 4, 3)),
}


@pytest.mark.parametrize("layout", sorted(LAYOUT_BATCHES))
def test_attention_layouts_give_the_same_rows(pair, layout):
    """The attention runs a call in one of four layouts with the same
    arithmetic: wide (clusters of 8, two CTAs per SM), wide with clusters of
    16 folding two 1024-key chunks in one cluster (every request of at most
    two chunks), narrow (V loaded over K, three CTAs per SM) and quad (the
    first product in halves of d, P in TMEM, four CTAs per SM).  A batch of
    requests takes the narrow or the quad layout (36 or 72 clusters of 8 over
    the two kv heads); each request alone takes a wide one (the two-chunk
    request: clusters of 16).  Every request's rows agree bit for bit, and
    the two-chunk request matches the oracle."""
    import torch
    from synth import device as D
    cfg = pair.cfg
    lens, ks = LAYOUT_BATCHES[layout]
    cap = 4100
    roots = [int(t) for t in W.root_tokens(cfg, len(lens), 7)]
    rng = np.random.default_rng(13)
    cands = [[int(t) for t in rng.integers(0, cfg.vocab, k)] for k in ks]
    st = pair.state(lens, cap, roots)
    gpu = run_gpu_block(st, cfg, cands)
    st.check()
    starts = np.cumsum([0] + [len(c) + 1 for c in cands])
    kc, vc = D.device_kv(cfg, lens, cap, pair.seed)
    for b in range(len(lens)):
        single = pair.state([lens[b]], cap, [roots[b]])
        single.kc.copy_(kc[:, b:b + 1])
        single.vc.copy_(vc[:, b:b + 1])
        torch.cuda.synchronize()
        g1 = run_gpu_block(single, cfg, [cands[b]])
        single.check()
        assert np.array_equal(g1[3], gpu[3][starts[b]:starts[b + 1]]), f"request {b}"
        assert g1[0][0] == gpu[0][b] and g1[1][0] == gpu[1][b]
        single.close()
    oc = pair.oracle_cache(lens[0], cap, req=0)
    ores = pair.oracle.verify_block(oc, lens[0], roots[0], cands[0])
    compare_block(ores, gpu[3][0:5], gpu[2][0:5], gpu[0][0], gpu[1][0], 4)
    st.close()


def test_argument_and_device_errors(pair):
    import torch
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    st = pair.state([L0], L0 + 8, [3])
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    c = torch.zeros(1, dtype=torch.int32, device="cuda")
    cand = torch.tensor(list(range(17)), dtype=torch.int32, device="cuda")
    with pytest.raises(lib.AS2DError) as e:
        st.verify(cand, [17], n, c)
    assert e.value.status == lib.AS2D_ERR_INVALID_ARG
    with pytest.raises(lib.AS2DError) as e:
        st.verify(cand, [8], n, c)           # 200 + 8 + 1 > 208
    assert e.value.status == lib.AS2D_ERR_CAPACITY
    bad = torch.tensor([cfg.vocab + 5], dtype=torch.int32, device="cuda")
    st.verify(bad, [1], n, c)
    torch.cuda.synchronize()
    assert int(n.item()) == -1
    with pytest.raises(lib.AS2DError) as e:
        st.check()
    assert e.value.status == lib.AS2D_ERR_DEVICE
    ln, rt = st.read_state()
    assert ln == [L0] and rt == [3]           # the bad call changed nothing
    st.check()                                # flag cleared
    st.rollback([L0 + 3], [1])                # beyond the committed length
    with pytest.raises(lib.AS2DError):
        st.check()
    st.close()


def test_reduced_sm_budget_keeps_parity(pair):
    """A model whose grids are sized for 16 SMs (as2d_model_set_sm_budget)
    still matches the oracle and stays batch invariant; a budget that grows
    after a state was sized is refused."""
    import torch
    import paper_2609_37617_gb300 as lib
    from synth import device as D
    cfg = pair.cfg
    dw = D.device_weights(cfg, 0)
    torch.cuda.synchronize()
    model = lib.Model(cfg, D.weight_pointers(cfg, dw))
    del dw
    with pytest.raises(lib.AS2DError):
        model.set_sm_budget(0)
    model.set_sm_budget(16)
    root, oc, cont, cand = _workload_block(pair)
    ores = pair.oracle.verify_block(oc, L0, root, cand)
    kc, vc = D.device_kv(cfg, [L0], CAP, 0)
    st = lib.State(model, [L0], CAP, kc, vc, [root])
    n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
    compare_block(ores, logits[:5], greedy[:5], n[0], corr[0], 4)
    # the same row alone (k = 0 after a rollback) gives bitwise the same logits
    st.rollback([L0], [root])
    n0, c0, g0, lg0 = run_gpu_block(st, cfg, [[]])
    assert np.array_equal(lg0[0], logits[0])
    model.set_sm_budget(torch.cuda.get_device_properties(0).multi_processor_count)
    with pytest.raises(lib.AS2DError):
        run_gpu_block(st, cfg, [[]])
    st.close()
    model.close()



def test_max_batch_max_k_and_capacity_edge(pair):
    """AS2D_MAX_BATCH requests with AS2D_MAX_K candidates each (1088 rows, so
    the projections run in several row chunks), ragged lengths, one request
    ending exactly at the capacity: every request matches the oracle, and a
    request verified alone gives bitwise the same rows."""
    import paper_2609_37617_gb300 as lib
    from synth import device as D
    import torch
    cfg = pair.cfg
    B, K, cap = lib.AS2D_MAX_BATCH, lib.AS2D_MAX_K, CAP
    lens = [cap - K - 1] + [16 + 3 * b for b in range(1, B)]
    roots = [int(t) for t in W.root_tokens(cfg, B, 5)]
    rng = np.random.default_rng(11)
    cands = [[int(t) for t in rng.integers(0, cfg.vocab, K)] for _ in range(B)]
    st = pair.state(lens, cap, roots)
    n, corr, greedy, logits = run_gpu_block(st, cfg, cands)
    ln, _ = st.read_state()
    assert ln[0] <= cap
    for b in (0, 1, 17, B - 1):
        oc = pair.oracle_cache(lens[b], cap, req=b)
        ores = pair.oracle.verify_block(oc, lens[b], roots[b], cands[b])
        r0 = b * (K + 1)
        compare_block(ores, logits[r0:r0 + K + 1], greedy[r0:r0 + K + 1], n[b], corr[b], K)
    # request B-1 alone, on a copy of its cache
    single = pair.state([lens[-1]], cap, [roots[-1]])
    kc, vc = D.device_kv(cfg, lens, cap, pair.seed)
    single.kc.copy_(kc[:, B - 1:B])
    single.vc.copy_(vc[:, B - 1:B])
    torch.cuda.synchronize()
    n1, c1, g1, lg1 = run_gpu_block(single, cfg, [cands[-1]])
    assert np.array_equal(lg1, logits[(B - 1) * (K + 1):])
    st.check()
    single.close()
    st.close()


def test_bounded_wait_expiry_is_reported_and_recovers(pair):
    """The kernels' bounded waits running out (failure detection, exercised
    without a GPU fault): with a wait limit of 0 every wait that is not
    already satisfied gives up at once, the call's blocks abandon their work
    after draining their own copies and products, and as2d_kv_check reports
    the timeout.  With the limit restored and the state rolled back, the next
    call matches the oracle again."""
    import torch
    import paper_2609_37617_gb300 as lib
    cfg = pair.cfg
    root, oc, cont, cand = _workload_block(pair)
    ores = pair.oracle.verify_block(oc, L0, root, cand)
    st = pair.state([L0], CAP, [root])
    st.set_wait_limit(0)
    for _ in range(3):
        run_gpu_block(st, cfg, [cand])
        st.rollback([L0], [root])
    torch.cuda.synchronize()
    with pytest.raises(lib.AS2DError) as e:
        st.check()
    assert e.value.status == lib.AS2D_ERR_DEVICE
    assert "timed out" in str(e.value)
    st.check()                                # the flag was cleared
    st.set_wait_limit(2_000_000_000)
    st.rollback([L0], [root])
    n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
    compare_block(ores, logits[:5], greedy[:5], n[0], corr[0], 4)
    st.check()
    st.close()


def test_zz_exact_checks_ran():
    """The module's bit-exact half ran: greedy rows and at least one full
    (n_accepted, correction) comparison (the sharp-model blocks above)."""
    TALLY.assert_ran(rows=9, blocks=2)
