"""Instruction-suffix prefill on the GPU (as2d_prefill, App. A.1): the tiny
workload's 150 retained "audio" positions plus 50 instruction tokens
prefilled by the library, against the oracle; chunking invariance; the
first verification block after it; argument errors."""
import numpy as np
import pytest

import oracle
from synth import workloads as W
from tests.helpers import MARGIN_SURE, Pair, bf16_bits, compare_block, run_gpu_block

pytestmark = pytest.mark.gpu

L0, N_INSTR, CAP = 150, 50, 256


@pytest.fixture(scope="module")
def pair():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return Pair(W.TINY, seed=0)


def _bf16_f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _prefill_gpu(pair, tokens, chunks=None):
    import torch
    st = pair.state([L0], CAP, [0])
    first = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    tok_d = torch.tensor(tokens, dtype=torch.int32, device="cuda")
    if chunks is None:
        st.prefill(tok_d, first)
    else:
        s0 = 0
        for c in chunks:
            st.prefill(tok_d[s0:s0 + c], first)
            s0 += c
    torch.cuda.synchronize()
    return st, int(first.item())


def test_prefill_matches_oracle(pair):
    cfg = pair.cfg
    instr = [int(t) for t in W.instruction_tokens(cfg, N_INSTR, 0)]
    oc = pair.oracle_cache(L0, CAP)
    ofirst, margin, _ = oracle.prefill(pair.oracle, oc, L0, instr)
    st, first = _prefill_gpu(pair, instr)
    ln, rt = st.read_state()
    assert ln == [L0 + N_INSTR] and rt == [first]
    if margin > MARGIN_SURE:
        assert first == ofirst
    for l in range(cfg.n_layers):
        for gpu, ref in ((st.kc, oc.k), (st.vc, oc.v)):
            g = _bf16_f32(bf16_bits(gpu[l, 0])[:, L0:L0 + N_INSTR])
            o = _bf16_f32(ref[l][:, L0:L0 + N_INSTR])
            assert np.max(np.abs(g - o)) < 3e-2, f"layer {l}"
    st.check()

    # the first verification block after the prefill, against the oracle
    cont, _ = oracle.greedy_continuation(pair.oracle, oc, L0 + N_INSTR, ofirst, 4)
    cand = W.replace_at(cont, 2, np.random.default_rng(0), cfg.vocab)
    if first == ofirst:
        ores = pair.oracle.verify_block(oc, L0 + N_INSTR, ofirst, cand)
        n, corr, greedy, logits = run_gpu_block(st, cfg, [cand])
        compare_block(ores, logits[:5], greedy[:5], n[0], corr[0], 4)
    st.close()


@pytest.mark.parametrize("chunks", [[1] * 100, [17, 83], [64, 36], [5, 90, 5], [99, 1]])
def test_prefill_is_chunking_invariant(pair, chunks):
    """Any split of the suffix into prefill calls gives bitwise the same cache
    and first token as one call of 100 tokens (passes of 64 + 36 rows):
    pathwise equivalence and batch invariance."""
    cfg = pair.cfg
    instr = [int(t) for t in W.instruction_tokens(cfg, 100, 1)]
    ref, first_ref = _prefill_gpu(pair, instr)
    st, first = _prefill_gpu(pair, instr, chunks)
    assert first == first_ref
    for l in range(cfg.n_layers):
        assert np.array_equal(bf16_bits(st.kc[l, 0])[:, :L0 + 100], bf16_bits(ref.kc[l, 0])[:, :L0 + 100])
        assert np.array_equal(bf16_bits(st.vc[l, 0])[:, :L0 + 100], bf16_bits(ref.vc[l, 0])[:, :L0 + 100])
    assert st.read_state() == ref.read_state()
    st.close()
    ref.close()


def test_prefill_argument_errors(pair):
    import torch
    import paper_2609_37617_gb300 as lib
    tok = torch.zeros(4, dtype=torch.int32, device="cuda")
    st = pair.state([L0], L0 + 3, [0])
    with pytest.raises(lib.AS2DError) as e:
        st.prefill(tok)                      # L0 + 4 > capacity
    assert e.value.status == lib.AS2D_ERR_CAPACITY
    assert lib._lib.as2d_prefill(st.handle, tok.data_ptr(), 0, None, None) == lib.AS2D_ERR_INVALID_ARG
    st.close()
    st2 = pair.state([L0, L0], CAP, [0, 0])
    with pytest.raises(lib.AS2DError) as e:
        st2.prefill(tok)
    assert e.value.status == lib.AS2D_ERR_UNSUPPORTED
    st2.close()
    bad = torch.full((3,), cfg_vocab(pair) + 5, dtype=torch.int32, device="cuda")
    st3 = pair.state([L0], CAP, [0])
    st3.prefill(bad)
    with pytest.raises(lib.AS2DError) as e:
        st3.check()
    assert e.value.status == lib.AS2D_ERR_DEVICE
    st3.close()


def cfg_vocab(pair):
    return pair.cfg.vocab
