"""The host-core decoder (as2d_cpu_decoder_*) that serves as a producer on the
CPU: its logits follow the oracle's decode steps on the same weights.  Host
code only."""
import numpy as np
import pytest

import oracle
from synth import workloads as W


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._lib_build_module().build()
    import paper_2609_37617_gb300 as p
    return p


def f32(bits):
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def host_f32(cfg, hw):
    out = {k: f32(hw[k]) for k in ("embed", "final_norm", "lm_head")}
    for name in ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm", "w_gate", "w_up", "w_down"):
        out[name] = [f32(hw[f"{name}.{l}"]) for l in range(cfg.n_layers)]
    return out


def test_cpu_decoder_follows_the_oracle(lib):
    cfg = W.TINY
    hw = W.host_weights(cfg, 0)
    om = oracle.Model(cfg, hw)
    cap = 32
    ks, vs = W.host_kv_request(cfg, 0, 0, cap, 0)
    cache = om.cache(ks, vs)
    root = int(W.root_tokens(cfg, 1, 0)[0])
    dec = lib.CpuDecoder(cfg, host_f32(cfg, hw), cap, 4, root)
    tok = root
    for pos in range(12):
        ref = om.decode_step(cache, pos, tok)
        got_tok = dec.step()
        lg = dec.logits()
        assert np.max(np.abs(lg - ref)) < 5e-2, pos
        want, margin = oracle.argmax(ref)
        if margin > 0.1:
            assert got_tok == want
        tok = want
        dec.reset(pos + 1, tok)           # both continue from the oracle's token
    with pytest.raises(lib.AS2DError):
        dec.reset(cap + 1, 0)
    dec.close()


def test_cpu_decoder_capacity_and_arguments(lib):
    cfg = W.TINY
    hw = host_f32(cfg, W.host_weights(cfg, 0))
    dec = lib.CpuDecoder(cfg, hw, 2, 1, 0)
    dec.step()
    dec.step()
    with pytest.raises(lib.AS2DError) as e:
        dec.step()
    assert e.value.status == lib.AS2D_ERR_CAPACITY
    dec.close()
    with pytest.raises(lib.AS2DError):
        lib.CpuDecoder(cfg, hw, 0, 1, 0)
