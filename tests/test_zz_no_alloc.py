"""as2d_decode_step_static, the decode step that allocates nothing, against
as2d_decode_step on the same model and cache, two calls in a row.

Collected last on purpose: if it fails, a run that stops at the first failure
has already run every other test.  It also passes on its own in a fresh
process.
"""
import numpy as np
import pytest

from synth import workloads as W
from tests.helpers import LOGIT_TOL

pytestmark = pytest.mark.gpu

L0, CAP = 200, 256


@pytest.fixture(scope="module")
def setup():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_37617_gb300 as lib
    from synth import device as D
    cfg = W.TINY
    dw = D.device_weights(cfg, seed=0)
    torch.cuda.synchronize()
    model = lib.Model(cfg, D.weight_pointers(cfg, dw))
    del dw
    return lib, D, cfg, model


def test_static_decode_matches_allocating_decode(setup):
    import torch
    lib, D, cfg, model = setup
    root0 = int(W.root_tokens(cfg, 1, 0)[0])

    # the existing entry point, on a state that owns its working memory
    kc_a, vc_a = D.device_kv(cfg, [L0], CAP, seed=0)
    state = lib.State(model, [L0], CAP, kc_a, vc_a, [root0])
    ref_corr, ref_logits = [], []
    for _ in range(2):
        n = torch.zeros(1, dtype=torch.int32, device="cuda")
        c = torch.zeros(1, dtype=torch.int32, device="cuda")
        lg = torch.empty(cfg.vocab, dtype=torch.float32, device="cuda")
        state.decode(n, c, None, lg)
        torch.cuda.synchronize()
        ref_corr.append(int(c.item()))
        ref_logits.append(lg.cpu().numpy())
    ref_len, ref_root = state.read_state()

    # the no-allocation entry point, on an identical cache of its own
    kc_b, vc_b = D.device_kv(cfg, [L0], CAP, seed=0)
    ln = torch.tensor([L0], dtype=torch.int32, device="cuda")
    rt = torch.tensor([root0], dtype=torch.int32, device="cuda")
    for step in range(2):
        c = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        lg = torch.empty(cfg.vocab, dtype=torch.float32, device="cuda")
        st = lib.as2d_decode_step_static(model.handle, kc_b.data_ptr(), vc_b.data_ptr(), CAP,
                                         ln.data_ptr(), rt.data_ptr(), c.data_ptr(),
                                         lg.data_ptr())
        assert st == lib.AS2D_OK, lib.as2d_last_error()
        torch.cuda.synchronize()
        assert int(c.item()) == ref_corr[step]
        assert np.max(np.abs(lg.cpu().numpy() - ref_logits[step])) <= LOGIT_TOL
    assert int(ln.item()) == ref_len[0] == L0 + 2
    assert int(rt.item()) == ref_root[0] == ref_corr[1]
    # the cache entries both paths appended agree too
    assert torch.equal(kc_a[:, :, :, L0:L0 + 2], kc_b[:, :, :, L0:L0 + 2])
    assert torch.equal(vc_a[:, :, :, L0:L0 + 2], vc_b[:, :, :, L0:L0 + 2])
    state.close()


def test_static_decode_rejects_oversize(setup):
    import torch
    lib, D, cfg, model = setup
    big = 5000
    kc = torch.zeros(1, dtype=torch.bfloat16, device="cuda")
    ln = torch.zeros(1, dtype=torch.int32, device="cuda")
    st = lib.as2d_decode_step_static(model.handle, kc.data_ptr(), kc.data_ptr(), big,
                                     ln.data_ptr(), ln.data_ptr(), ln.data_ptr())
    assert st == lib.AS2D_ERR_CAPACITY
    assert "4096" in lib.as2d_last_error()
