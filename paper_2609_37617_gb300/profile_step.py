"""Run a few verification blocks of one synthetic workload, for profiler
captures (ncu) of the library's kernels.

    python -m paper_2609_37617_gb300.profile_step --model 7b-2l --kv-len 1564 --k 8 \
        --warmup 2 --blocks 2

Weights and the prefilled cache are the seeded synthetic inputs of the
benchmark (random-init bf16 weights, N(0, 1) cache entries); candidates are
uniform tokens, since a block's work does not depend on what is accepted.
Each block starts from the same prefix (a rollback), so every captured launch
sees the same length.  The blocks after the warm-up run inside the NVTX range
"blocks" (ncu --nvtx --nvtx-include blocks/); each is a rollback launch and
one verification pass of 3 + 9 x n_layers launches.
"""
import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main(argv=None):
    import numpy as np
    import torch

    import paper_2609_37617_gb300 as lib
    from synth import device as D
    from synth import workloads as W

    ap = argparse.ArgumentParser()
    ap.add_argument("--model", default="7b-2l")
    ap.add_argument("--kv-len", type=int, nargs="+", default=[1564],
                    help="prefix length of each request (one value per request)")
    ap.add_argument("--k", type=int, nargs="+", default=[8],
                    help="candidates per request (one value, or one per request)")
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--blocks", type=int, default=2)
    ap.add_argument("--seed", type=int, default=0)
    a = ap.parse_args(argv)
    cfg = W.MODELS[a.model]
    lens = list(a.kv_len)
    ks = list(a.k) * (len(lens) if len(a.k) == 1 else 1)
    assert len(ks) == len(lens), "--k takes one value or one per request"
    B = len(lens)
    torch.cuda.set_device(0)
    w = D.device_weights(cfg, a.seed)
    torch.cuda.synchronize()
    model = lib.Model(cfg, D.weight_pointers(cfg, w))
    del w
    torch.cuda.empty_cache()
    cap = max(lens) + max(ks) + 64
    kc, vc = D.device_kv(cfg, lens, cap, a.seed, poison=False)
    roots = [int(t) for t in W.root_tokens(cfg, B, a.seed)]
    st = lib.State(model, lens, cap, kc, vc, roots)
    rng = np.random.default_rng(a.seed + 1)
    cand = torch.from_numpy(rng.integers(0, cfg.vocab, max(sum(ks), 1)).astype(np.int32)).cuda()
    n = torch.zeros(B, dtype=torch.int32, device="cuda")
    c = torch.zeros(B, dtype=torch.int32, device="cuda")
    for i in range(a.warmup + a.blocks):
        if i == a.warmup:
            torch.cuda.synchronize()
            torch.cuda.nvtx.range_push("blocks")
        st.rollback(lens, roots)
        st.verify(cand, ks, n, c)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    st.check()
    st.close()
    model.close()
    print(f"profile_step ok: {a.model}, lens={lens}, k={ks}, {a.warmup}+{a.blocks} blocks")


if __name__ == "__main__":
    main()
