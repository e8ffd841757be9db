"""Shared test scaffolding: the same seeded inputs on the oracle (host) and
on the CUDA path (device), and comparison helpers."""
import numpy as np

from synth import workloads as W

LOGIT_TOL = 5e-2      # max |logit difference| allowed against the oracle
MARGIN_SURE = 0.1     # top-1 minus top-2 above which the greedy token must agree


def bf16_bits(t):
    """uint16 numpy view of a bf16 torch tensor."""
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


class Pair:
    """A model with identical weights on the oracle and on the GPU library."""

    def __init__(self, cfg, seed=0, gains="unit", host_weights=None, precision="f64"):
        import torch
        import oracle
        import paper_2609_37617_gb300 as lib
        from synth import device as D
        self.cfg = cfg
        self.seed = seed
        self.gains = gains
        self.dev_w = D.device_weights(cfg, seed, gains)
        torch.cuda.synchronize()
        self.model = lib.Model(cfg, D.weight_pointers(cfg, self.dev_w))
        self.dev_w = None  # the library keeps its own copy
        torch.cuda.empty_cache()
        hw = host_weights if host_weights is not None else W.host_weights(cfg, seed, gains)
        self.oracle = oracle.Model(cfg, hw, precision)

    def state(self, kv_lens, capacity, roots, poison=True, kv_seed=None):
        import paper_2609_37617_gb300 as lib
        from synth import device as D
        kc, vc = D.device_kv(self.cfg, kv_lens, capacity, self.seed if kv_seed is None else kv_seed,
                             poison=poison)
        st = lib.State(self.model, list(kv_lens), capacity, kc, vc, list(roots))
        st.kc, st.vc = kc, vc
        return st

    def oracle_cache(self, kv_len, capacity, req=0, kv_seed=None):
        ks, vs = W.host_kv_request(self.cfg, req, kv_len, capacity,
                                   self.seed if kv_seed is None else kv_seed)
        return self.oracle.cache(ks, vs)


def run_gpu_block(st, cfg, cand_lists, want_logits=True):
    """Run one as2d_verify_block over requests with candidate lists; returns
    numpy (n_accepted, correction, greedy, logits)."""
    import torch
    ks = [len(c) for c in cand_lists]
    flat = [int(t) for c in cand_lists for t in c]
    rows = sum(k + 1 for k in ks)
    cand = torch.tensor(flat if flat else [0], dtype=torch.int32, device="cuda")
    n = torch.full((len(ks),), -7, dtype=torch.int32, device="cuda")
    corr = torch.full((len(ks),), -7, dtype=torch.int32, device="cuda")
    greedy = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    logits = torch.empty((rows, cfg.vocab), dtype=torch.float32, device="cuda") if want_logits else None
    st.verify(cand if flat else None, ks, n, corr, greedy, logits)
    torch.cuda.synchronize()
    return (n.cpu().numpy(), corr.cpu().numpy(), greedy.cpu().numpy(),
            logits.cpu().numpy() if want_logits else None)


def compare_block(oracle_res, gpu_logits, gpu_greedy, gpu_n, gpu_corr, k):
    """Parity rule: logits within LOGIT_TOL everywhere; greedy tokens equal
    where the oracle's margin exceeds MARGIN_SURE; n_accepted and the
    correction equal whenever every margin they depend on exceeds it."""
    d = np.max(np.abs(oracle_res["logits"] - gpu_logits))
    assert d <= LOGIT_TOL, f"max |dlogit| = {d}"
    sure = oracle_res["margin"] > MARGIN_SURE
    assert np.array_equal(oracle_res["greedy"][sure], gpu_greedy[sure])
    n = oracle_res["n_accepted"]
    if np.all(sure[: n + 1]):
        assert gpu_n == n and gpu_corr == oracle_res["correction"]
    return d


def oracle_block(pair, cache, length, root, cand):
    """Oracle verification of one block on `cache` (modified in place)."""
    return pair.oracle.verify_block(cache, length, root, list(cand))


def check_parity(ores, gpu, row0, k, where=""):
    """Compare one request's oracle result with its rows of a GPU call
    (gpu = (n, corr, greedy, logits) arrays; request at row offset row0)."""
    n, corr, greedy, logits = gpu
    d = np.max(np.abs(ores["logits"] - logits[row0:row0 + k + 1]))
    assert d <= LOGIT_TOL, f"{where}: max |dlogit| = {d}"
    sure = ores["margin"] > MARGIN_SURE
    g = greedy[row0:row0 + k + 1]
    assert np.array_equal(ores["greedy"][sure], g[sure]), where
    m = ores["n_accepted"]
    return d, bool(np.all(sure[: m + 1])), m, ores["correction"]
