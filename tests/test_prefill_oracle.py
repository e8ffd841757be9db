"""The oracle's instruction-suffix prefill (App. A.1) against what the greedy
definition fixes.  CPU only."""
import numpy as np

import oracle
from synth import workloads as W

L0, CAP = 150, 256


def _model():
    cfg = W.TINY
    return cfg, oracle.Model(cfg, W.host_weights(cfg, 0))


def test_prefill_of_the_greedy_text_continues_it():
    """Prefilling the model's own greedy text yields the next greedy token,
    and the cache it leaves is the one greedy decoding leaves."""
    cfg, om = _model()
    ks, vs = W.host_kv_request(cfg, 0, L0, CAP, 0)
    root = int(W.root_tokens(cfg, 1, 0)[0])
    cont, margins = oracle.greedy_continuation(om, om.cache(ks, vs), L0, root, 12)
    c1 = om.cache(ks, vs)
    first, m, _ = oracle.prefill(om, c1, L0, [root] + [int(t) for t in cont[:8]])
    assert first == int(cont[8]) and m == margins[8]
    c2 = om.cache(ks, vs)
    oracle.greedy_continuation(om, c2, L0, root, 0)          # copies: c2 untouched
    for i, t in enumerate([root] + [int(t) for t in cont[:8]]):
        om.decode_step(c2, L0 + i, t)
    for l in range(cfg.n_layers):
        assert np.array_equal(c1.k[l][:, :L0 + 9], c2.k[l][:, :L0 + 9])
        assert np.array_equal(c1.v[l][:, :L0 + 9], c2.v[l][:, :L0 + 9])


def test_prefill_then_verify_equals_one_long_greedy_pass():
    """After prefill, a verification block of the greedy continuation is fully
    accepted (Prop. 1 applied to the prefilled state)."""
    cfg, om = _model()
    ks, vs = W.host_kv_request(cfg, 0, L0, CAP, 0)
    instr = [int(t) for t in W.instruction_tokens(cfg, 50, 0)]
    c = om.cache(ks, vs)
    first, _, _ = oracle.prefill(om, c, L0, instr)
    cont, margins = oracle.greedy_continuation(om, c, L0 + 50, first, 4)
    res = om.verify_block(c, L0 + 50, first, cont)
    if np.all(margins > 0.1):
        assert res["n_accepted"] == 4
    assert res["new_len"] == L0 + 50 + res["n_accepted"] + 1


def test_single_token_prefill_is_a_decode_step():
    cfg, om = _model()
    ks, vs = W.host_kv_request(cfg, 0, L0, CAP, 0)
    tok = int(W.instruction_tokens(cfg, 1, 3)[0])
    first, m, lg = oracle.prefill(om, om.cache(ks, vs), L0, [tok])
    lg2 = om.decode_step(om.cache(ks, vs), L0, tok)
    assert np.array_equal(lg, lg2) and first == int(np.argmax(lg2))
