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


def test_static_decode_length_guard(setup):
    """The length lives on the device, so the kernels check it: a step at
    len = capacity - 1 runs, the next (len = capacity) is refused on the
    device -- correction -1, len and root unchanged, the capacity bit in the
    error output, and nothing written past the request's cache slots (the
    slots beyond the last head of the last layer hold a sentinel)."""
    import torch
    lib, D, cfg, model = setup
    cap = 64
    root0 = int(W.root_tokens(cfg, 1, 0)[0])
    kc, vc = D.device_kv(cfg, [cap - 1], cap, seed=3)
    # the caches plus one guard position of sentinels past the end of each
    shape = (cfg.n_layers, 1, cfg.n_kv, cap, cfg.head_dim)
    pad = cfg.head_dim * cfg.n_kv
    kbuf = torch.full((kc.numel() + pad,), 7.0, dtype=torch.bfloat16, device="cuda")
    vbuf = torch.full((vc.numel() + pad,), 7.0, dtype=torch.bfloat16, device="cuda")
    kbuf[:kc.numel()].copy_(kc.reshape(-1))
    vbuf[:vc.numel()].copy_(vc.reshape(-1))
    k_before, v_before = kbuf.clone(), vbuf.clone()
    ln = torch.tensor([cap - 1], dtype=torch.int32, device="cuda")
    rt = torch.tensor([root0], dtype=torch.int32, device="cuda")
    errb = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    c = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    st = lib.as2d_decode_step_static(model.handle, kbuf.data_ptr(), vbuf.data_ptr(), cap,
                                     ln.data_ptr(), rt.data_ptr(), c.data_ptr(), 0,
                                     errb.data_ptr())
    assert st == lib.AS2D_OK, lib.as2d_last_error()
    torch.cuda.synchronize()
    assert int(errb.item()) == 0 and int(c.item()) >= 0 and int(ln.item()) == cap
    root1 = int(rt.item())
    assert root1 == int(c.item())
    # the step appended at position cap - 1 of every (layer, head): the last
    # position of each slot, not past it
    k_mid = kbuf.clone()
    assert torch.equal(k_mid[kc.numel():], k_before[kc.numel():])
    # now len == capacity: refused on the device
    c.fill_(-7)
    st = lib.as2d_decode_step_static(model.handle, kbuf.data_ptr(), vbuf.data_ptr(), cap,
                                     ln.data_ptr(), rt.data_ptr(), c.data_ptr(), 0,
                                     errb.data_ptr())
    assert st == lib.AS2D_OK, lib.as2d_last_error()
    torch.cuda.synchronize()
    assert int(c.item()) == -1
    assert int(ln.item()) == cap and int(rt.item()) == root1
    assert int(errb.item()) & lib.AS2D_DEVERR_CAPACITY
    assert torch.equal(kbuf, k_mid)            # nothing written anywhere
    assert torch.equal(vbuf[vc.numel():], v_before[vc.numel():])
    # a negative length is refused the same way
    ln.fill_(-3)
    c.fill_(-7)
    st = lib.as2d_decode_step_static(model.handle, kbuf.data_ptr(), vbuf.data_ptr(), cap,
                                     ln.data_ptr(), rt.data_ptr(), c.data_ptr(), 0,
                                     errb.data_ptr())
    assert st == lib.AS2D_OK
    torch.cuda.synchronize()
    assert int(c.item()) == -1 and int(ln.item()) == -3
    assert int(errb.item()) & lib.AS2D_DEVERR_CAPACITY
    assert torch.equal(kbuf, k_mid)
    # the array is reused: a valid step afterwards still matches a fresh state
    ln.fill_(cap - 1)
    rt.fill_(root0)
    kc2, vc2 = D.device_kv(cfg, [cap - 1], cap, seed=3)
    state = lib.State(model, [cap - 1], cap, kc2, vc2, [root0])
    n_ref = torch.zeros(1, dtype=torch.int32, device="cuda")
    c_ref = torch.zeros(1, dtype=torch.int32, device="cuda")
    state.decode(n_ref, c_ref)
    st = lib.as2d_decode_step_static(model.handle, kbuf.data_ptr(), vbuf.data_ptr(), cap,
                                     ln.data_ptr(), rt.data_ptr(), c.data_ptr(), 0,
                                     errb.data_ptr())
    assert st == lib.AS2D_OK
    torch.cuda.synchronize()
    assert int(errb.item()) == 0 and int(c.item()) == int(c_ref.item())
    state.close()
