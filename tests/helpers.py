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


class ExactTally:
    """How many bit-exact comparisons actually ran: greedy tokens compared on
    rows whose oracle margin exceeds MARGIN_SURE, and (n_accepted,
    correction) pairs compared on blocks whose deciding rows all do.  A test
    module asserts at the end that its exact half was not skipped."""

    def __init__(self):
        self.rows = 0
        self.blocks = 0

    def assert_ran(self, rows=1, blocks=1):
        assert self.rows >= rows and self.blocks >= blocks, (
            f"bit-exact checks ran on {self.rows} rows and {self.blocks} blocks only")


def compare_block(oracle_res, gpu_logits, gpu_greedy, gpu_n, gpu_corr, k, tally=None):
    """Parity rule: logits within LOGIT_TOL everywhere; greedy tokens equal
    where the oracle's margin exceeds MARGIN_SURE; n_accepted and the
    correction equal whenever every margin they depend on exceeds it."""
    d = np.max(np.abs(oracle_res["logits"] - gpu_logits))
    assert d <= LOGIT_TOL, f"max |dlogit| = {d}"
    sure = oracle_res["margin"] > MARGIN_SURE
    assert np.array_equal(oracle_res["greedy"][sure], gpu_greedy[sure])
    n = oracle_res["n_accepted"]
    exact = bool(np.all(sure[: n + 1]))
    if exact:
        assert gpu_n == n and gpu_corr == oracle_res["correction"]
    if tally is not None:
        tally.rows += int(sure.sum())
        tally.blocks += int(exact)
    return d


def sharp_root(oracle_model, cache_fn, length, n, start=0, limit=400):
    """The first root token, searching upward from `start`, whose n-token
    oracle greedy continuation from `length` has every top-1 minus top-2
    margin above MARGIN_SURE (cache_fn() gives a fresh oracle cache).  Returns
    (root, continuation, margins).  A search on the oracle only."""
    import oracle
    for root in range(start, start + limit):
        cont, m = oracle.greedy_continuation(oracle_model, cache_fn(), length, root, n)
        if np.all(np.asarray(m) > MARGIN_SURE):
            return root, cont, m
    raise AssertionError("no root with well-separated greedy decisions found")


def oracle_block(pair, cache, length, root, cand):
    """Oracle verification of one block on `cache` (modified in place)."""
    return pair.oracle.verify_block(cache, length, root, list(cand))


def check_parity(ores, gpu, row0, k, where="", tally=None, b=0):
    """Compare request b's oracle result with its rows of a GPU call (gpu =
    (n, corr, greedy, logits) arrays; the request's rows start at row0):
    logits within LOGIT_TOL, greedy tokens where the margin is sure, and
    n_accepted / correction when every row they depend on is sure.  Returns
    (max |dlogit|, whether the commit was compared, oracle n, oracle corr)."""
    n, corr, greedy, logits = gpu
    d = np.max(np.abs(ores["logits"] - logits[row0:row0 + k + 1]))
    assert d <= LOGIT_TOL, f"{where}: max |dlogit| = {d}"
    sure = ores["margin"] > MARGIN_SURE
    g = greedy[row0:row0 + k + 1]
    assert np.array_equal(ores["greedy"][sure], g[sure]), where
    m = ores["n_accepted"]
    exact = bool(np.all(sure[: m + 1]))
    if exact:
        assert n[b] == m and corr[b] == ores["correction"], where
    if tally is not None:
        tally.rows += int(sure.sum())
        tally.blocks += int(exact)
    return d, exact, m, ores["correction"]
