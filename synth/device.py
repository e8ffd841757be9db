"""Device copies of the seeded synthetic inputs (torch tensors on a CUDA
device), filled by the device generator with the same bits as the host
generator.  Input construction only: no part of the method's arithmetic."""
import torch

import synth
from synth import workloads as W


def device_weights(cfg, seed=0, gains="unit", device="cuda"):
    """dict name -> bf16 tensor in logical layout (as workloads.host_weights)."""
    out = {}
    for s in W.weight_specs(cfg, gains):
        t = torch.empty(s.shape, dtype=torch.bfloat16, device=device)
        if s.sigma == 0.0:
            t.fill_(s.base)
        else:
            synth.cuda_normal_bf16(t.data_ptr(), t.numel(), seed, s.stream, s.sigma,
                                   s.base, torch.cuda.current_stream().cuda_stream)
        out[s.name] = t
    return out


def weight_pointers(cfg, tensors):
    ptrs = {n: tensors[n].data_ptr() for n in ("embed", "final_norm", "lm_head")}
    for kind in W.LAYER_KINDS:
        ptrs[kind] = [tensors[f"{kind}.{l}"].data_ptr() for l in range(cfg.n_layers)]
    return ptrs


def device_kv(cfg, kv_lens, capacity, seed=0, poison=True, device="cuda"):
    """Caller-side caches [n_layers][batch][n_kv][capacity][head_dim] bf16 with
    request b's positions [0, kv_lens[b]) drawn N(0, 1) (workloads.kv_stream);
    the rest holds NaN when poison is set."""
    B = len(kv_lens)
    shape = (cfg.n_layers, B, cfg.n_kv, capacity, cfg.head_dim)
    kc = torch.full(shape, float("nan") if poison else 0.0, dtype=torch.bfloat16, device=device)
    vc = torch.full(shape, float("nan") if poison else 0.0, dtype=torch.bfloat16, device=device)
    st = torch.cuda.current_stream().cuda_stream
    for l in range(cfg.n_layers):
        for b, L in enumerate(kv_lens):
            for g in range(cfg.n_kv):
                for which, t in ((0, kc), (1, vc)):
                    view = t[l, b, g]
                    if L > 0:
                        synth.cuda_normal_bf16(view.data_ptr(), L * cfg.head_dim, seed,
                                               W.kv_stream(l, b, g, which), 1.0, 0.0, st)
    return kc, vc


def host_kv_from_device(cfg, kc, vc, b):
    """One request's cache as the oracle's per-layer uint16 arrays."""
    ks = [kc[l, b].contiguous().view(torch.int16).cpu().numpy().view("uint16") for l in range(cfg.n_layers)]
    vs = [vc[l, b].contiguous().view(torch.int16).cpu().numpy().view("uint16") for l in range(cfg.n_layers)]
    return ks, vs
