"""Benchmark of the target-side block verification step on GB300.

Default workload (one JSON line): the 7B-class decoder (28 layers, hidden
3584, 28/4 heads, head_dim 128, FFN 18944, vocab 152064, bf16 random-init
weights), one request whose cache holds 1564 prefilled positions (60 s of
audio at 25 tokens/s plus 64 instruction tokens), candidate blocks of k = 8
whose accepted length is geometric with mean 3 (capped at k), 256
consecutive verification blocks.  A step is one verification block: the
whole hot path (embedding, 28 layers, LM head + argmax, accept scan and
rollback) through the C-ABI.

value  = committed tokens / s over the timed blocks (inputs resident in HBM).
e2e    = the same metric through the C-ABI with host buffers: each block's
         candidates copied host->device and its (n_accepted, correction)
         copied device->host inside the timed region.
--impl reference times the CPU oracle on the same workload instead.
--session prints a different line instead: one request decoded by a drafter
(producer) and the 7B target (verifier) through a candidate buffer, serially
and overlapped on two streams, with the service-interval accounting
T = D + V - O + H of each run.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "7B verify-step µs & committed tok/s vs block k; fraction of HBM roofline"
UNIT = "committed tok/s"
WORKLOAD = "7b"

# dram__bytes_read.sum + dram__bytes_write.sum per launch from one ncu capture
# of the kernel as it stands (profiles/); None once the kernel has changed.
TRAFFIC = {"gate_up": 272168960}  # 271,877,632 read + 291,328 written

# Diagnostic legs that reuse the headline state (each rolls it back to L0 first).
BUDGET_WIN, BUDGET_COMMIT, BUDGET_TRACES = 220, 180, 4
MAX_K = 16


def plan_capacity(L0, k, steps, warmup, sweep_ks, sweep_blocks, committed_plan):
    """Cache positions the headline state needs, and the length of the greedy
    trajectory, for every leg that runs on it.  Each leg starts from L0 (a
    rollback).  Between read-backs the library's host bound of the length
    grows by k + 1 per call whatever is accepted, and a call is refused once
    bound + k + 1 exceeds the capacity, so a leg of n calls of width k needs
    n (k + 1) positions past L0.  Returns (trajectory length, capacity, the
    positions past L0 of each leg)."""
    sweep_ks = list(sweep_ks)
    sweep_need = max(((kk + 1) * sweep_blocks for kk in sweep_ks), default=0)
    # the trajectory feeds the timed blocks' candidates (up to the planned
    # committed length + k), the k-sweep's (up to its own advance + k) and
    # the budget leg's development windows
    traj_len = max(committed_plan + k + 2, BUDGET_TRACES * BUDGET_WIN + 1,
                   max(((kk + 1) * sweep_blocks + kk + 1 for kk in sweep_ks), default=0))
    needs = {
        "trajectory": traj_len,                    # k = 0 decode steps
        "warmup": warmup * (k + 1),
        "timed": steps * (k + 1),                  # also the e2e leg
        "breakdown": min(8, steps) * (k + 1),
        "k_sweep": sweep_need,
        # sessions read every call's outcome back, so the bound stays exact:
        # the committed tokens plus one call of the widest block
        "budget": BUDGET_COMMIT + 2 * (MAX_K + 1),
        "prefill": 0,                              # rewrites positions below L0
    }
    return traj_len, L0 + max(needs.values()) + 64, needs


def guarded(errors, name, fn, *a, **kw):
    """Run one diagnostic leg; a failure is recorded under `name` in `errors`
    (and reported as None) instead of ending the run."""
    import traceback
    try:
        return fn(*a, **kw)
    except Exception as exc:  # noqa: BLE001 -- every leg failure is reported, not raised
        errors[name] = f"{type(exc).__name__}: {exc}"
        traceback.print_exc(file=sys.stderr)
        return None


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--k", type=int, default=8)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--profile-class", default="gate_up",
                    help="kernel class timed live for the roofline (the dominant one, "
                         "gate_up, by default)")
    ap.add_argument("--model", default="7b", help="model shape (7b; smaller ones for quick checks)")
    ap.add_argument("--kv-len", type=int, default=1564)
    ap.add_argument("--sweep", default=",".join(str(i) for i in range(17)),
                    help="block sizes k for the verify-time sweep ('' to skip); the budget "
                         "selection needs all of 0..16")
    ap.add_argument("--sweep-blocks", type=int, default=24)
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the 1.5B k-sweep and the ragged 16-request rounds")
    ap.add_argument("--long-kv-len", type=int, default=15128,
                    help="prefix length of the long-context sweep (0 to skip)")
    ap.add_argument("--session", action="store_true",
                    help="producer/verifier session line instead of the verify-step line")
    ap.add_argument("--drafter", default="1.5b", help="drafter model shape for --session")
    ap.add_argument("--drafter-kv-len", type=int, default=814)
    ap.add_argument("--session-tokens", type=int, default=256)
    ap.add_argument("--session-b", type=int, default=8)
    ap.add_argument("--cpu-drafter", action="store_true",
                    help="--session: the producer runs the cpu-draft decoder on the host cores "
                         "instead of a GPU drafter")
    ap.add_argument("--cpu-threads", type=int, default=0,
                    help="host threads of the CPU drafter (0: half the cores, at most 8)")
    ap.add_argument("--drafter-sms", type=int, default=0,
                    help="--session: confine the drafter's grids to this many SMs and the "
                         "target's to the rest (0: both use every SM)")
    ap.add_argument("--session-noise", type=float, default=0.25,
                    help="per-token substitution probability of the producer's text")
    return ap.parse_args()


def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def model_shape(name):
    from synth import workloads as W
    return W.MODELS[name]


def draw_plans(args, steps, vocab, k=None, seed_offset=17):
    from synth import workloads as W
    k = args.k if k is None else k
    rng = np.random.default_rng(args.seed + seed_offset)
    return np.stack([W.geometric_plan(rng, k, vocab) for _ in range(steps)])


def reduce_ranks(elapsed_ms, committed, device):
    """Replicas: the job's time is the slowest rank's, its work the sum of
    every rank's committed tokens (no exchange between replicas otherwise)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([elapsed_ms, float(committed)], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    sm = t.clone()
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(sm[1])


def bytes_per_block(cfg, L, k):
    """Algorithmic HBM bytes of one block: every weight once plus the KV read
    by attention (all layers), as the roofline of the workload defines it."""
    return cfg.weight_bytes() + (L + k + 1) * cfg.kv_bytes_per_pos()


def run_ours(args, ws, rank, local):
    import torch
    import torch.distributed as dist

    import paper_2609_37617_gb300 as lib
    import synth
    from synth import device as D
    from synth import workloads as W

    torch.cuda.set_device(local)
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    cfg = model_shape(args.model)
    k, L0, steps, warm = args.k, args.kv_len, args.steps, args.warmup
    seed = args.seed + rank
    stream = torch.cuda.Stream()
    sh = stream.cuda_stream

    with torch.cuda.stream(stream):
        dev_w = D.device_weights(cfg, seed)
        torch.cuda.synchronize()
        model = lib.Model(cfg, D.weight_pointers(cfg, dev_w))
        del dev_w
        torch.cuda.empty_cache()
        plans = draw_plans(args, steps, cfg.vocab)
        committed_plan = int((plans[:, 0] + 1).sum())
        sweep_ks = [int(x) for x in args.sweep.split(",") if x != ""] if args.sweep else []
        traj_len, cap, _ = plan_capacity(L0, k, steps, warm, sweep_ks, args.sweep_blocks,
                                         committed_plan)
        kc, vc = D.device_kv(cfg, [L0], cap, seed, poison=False)
        root0 = int(W.root_tokens(cfg, 1, seed)[0])
        state = lib.State(model, [L0], cap, kc, vc, [root0])
        len_dev, _ = state.device_state()

        # greedy trajectory from the initial state (untimed), on the device
        traj = torch.zeros(traj_len + 1, dtype=torch.int32, device="cuda")
        traj[0] = root0
        nbuf = torch.zeros(1, dtype=torch.int32, device="cuda")
        for j in range(traj_len):
            out = lib.make_verify_out(nbuf.data_ptr(), traj.data_ptr() + 4 * (j + 1))
            lib._check(lib.as2d_decode_step(state.handle, out, sh), "as2d_decode_step")
        state.check(sh)
        state.rollback([L0], [root0], sh)
        state.read_state(sh)

        # every block's candidates, resident in HBM before the timed region:
        # block i continues the greedy trajectory from the length the plans
        # of blocks < i leave (checked afterwards: plan_match)
        traj_h = traj.cpu().numpy()
        cand_h = np.zeros((steps, k), dtype=np.int32)
        m_off = 0
        for i in range(steps):
            cand_h[i] = W.apply_plan(traj_h[m_off + 1:m_off + 1 + k], plans[i], cfg.vocab)
            m_off += int(plans[i, 0]) + 1
        cand_all = torch.from_numpy(cand_h).cuda()
        n_all = torch.zeros(steps, dtype=torch.int32, device="cuda")
        c_all = torch.zeros(steps, dtype=torch.int32, device="cuda")

        def block(i, plan_row):
            out = lib.make_verify_out(n_all.data_ptr() + 4 * i, c_all.data_ptr() + 4 * i)
            lib._check(lib.as2d_verify_block(state.handle, cand_all[plan_row].data_ptr(), [k],
                                             out, sh), "as2d_verify_block")

        for w in range(warm):
            block(w % steps, w % steps)
        state.check(sh)
        state.rollback([L0], [root0], sh)
        state.read_state(sh)
        n_all.zero_()

        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)

        def timed_pass(profile_class, per_block=False):
            """`steps` consecutive blocks from the initial state, timed with
            CUDA events on the launching stream; optionally with an event pair
            around every block, or with the library's event pairs around one
            kernel class."""
            state.rollback([L0], [root0], sh)
            state.read_state(sh)
            n_all.zero_()
            state.profile(None if profile_class in (None, "none") else profile_class)
            state.profile_read()
            if ws > 1:
                dist.barrier()
            torch.cuda.synchronize()
            torch.cuda.nvtx.range_push("timed")
            t0.record(stream)
            for i in range(steps):
                if per_block:
                    ev[i][0].record(stream)
                block(i, i)
                if per_block:
                    ev[i][1].record(stream)
            t1.record(stream)
            torch.cuda.nvtx.range_pop()
            torch.cuda.synchronize()
            if ws > 1:
                dist.barrier()
            res = state.profile_read()
            state.profile(None)
            return res

        # pass 1 (the headline): no event inside the timed region, so
        # programmatic dependent launch overlaps every kernel boundary, also
        # between blocks
        clocks = ClockSampler(local)
        clocks.start()
        time.sleep(0.3)
        _, _, all_launches = timed_pass(None)
        clk = clocks.stop()
        state.check(sh)
        elapsed_ms = t0.elapsed_time(t1)
        n_np = n_all.cpu().numpy()
        committed = int((n_np + 1).sum())
        plan_match = float(np.mean(n_np == plans[:, 0]))
        # everything below is diagnostic: a leg that fails is reported in the
        # line's "errors" instead of ending the run
        errors = {}
        # pass 2: the same blocks again with event pairs around every launch of
        # the dominant kernel class, for its live average duration
        prof_cls = args.profile_class

        def pass2():
            # run twice and keep the faster: a transient stall of the shared
            # host would otherwise set the kernel's figure
            prof = []
            for _ in range(2):
                pn, pms, _ = timed_pass(prof_cls)
                prof.append((pms / pn if pn else float("inf"), pn, pms, t0.elapsed_time(t1)))
            state.check(sh)
            return min(prof)[1:]

        prof_n, prof_ms, pass2_ms = guarded(errors, "kernel_timing", pass2) or (0, 0.0, 0.0)

        def pass3():
            # an event pair around every block for the distribution of block times
            timed_pass(None, per_block=True)
            state.check(sh)
            return np.array([a.elapsed_time(b) * 1e3 for a, b in ev])

        per_block_us = guarded(errors, "per_block", pass3)

        def class_breakdown():
            # per-class device time per block (after the timed region)
            breakdown = {}
            for cls_name in ("qkv", "attention", "o", "gate_up", "down", "lm_head", "other"):
                state.rollback([L0], [root0], sh)
                state.read_state(sh)
                state.profile(cls_name)
                state.profile_read()
                nb_blocks = min(8, steps)
                for i in range(nb_blocks):
                    block(i, i)
                n_cls, ms_cls, _ = state.profile_read()
                if n_cls:
                    breakdown[cls_name] = round(ms_cls / nb_blocks * 1e3, 1)
            state.profile(None)
            state.check(sh)
            return breakdown

        breakdown = guarded(errors, "class_us_per_block", class_breakdown)

        def k_sweep():
            # verify time and committed tokens/s versus k (same acceptance law,
            # capped at k), and the per-position cost reduction R(K) of Eq. 2
            sweep = []
            nbk = args.sweep_blocks
            for kk in sweep_ks:
                pl = draw_plans(args, nbk, cfg.vocab, k=kk, seed_offset=1000 + kk) if kk > 0 else None
                pl_d = torch.from_numpy(pl.astype(np.int32)).cuda() if kk > 0 else None
                cand_k = torch.zeros(max(kk, 1), dtype=torch.int32, device="cuda")
                nk = torch.zeros(nbk, dtype=torch.int32, device="cuda")
                ck = torch.zeros(nbk, dtype=torch.int32, device="cuda")
                evk = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(nbk)]
                state.rollback([L0], [root0], sh)
                state.read_state(sh)
                torch.cuda.synchronize()
                for i in range(nbk):
                    evk[i][0].record(stream)
                    if kk > 0:
                        rc = synth._load_cuda().synth_cuda_build_candidates(
                            cand_k.data_ptr(), traj.data_ptr(), traj_len + 1, len_dev, L0,
                            pl_d[i].data_ptr(), kk, cfg.vocab, sh)
                        if rc != 0:
                            raise RuntimeError(f"synth_cuda_build_candidates returned {rc}")
                    out = lib.make_verify_out(nk.data_ptr() + 4 * i, ck.data_ptr() + 4 * i)
                    lib._check(lib.as2d_verify_block(state.handle, cand_k.data_ptr() if kk else 0,
                                                     [kk], out, sh), "as2d_verify_block")
                    evk[i][1].record(stream)
                torch.cuda.synchronize()
                us = np.array([a.elapsed_time(b) * 1e3 for a, b in evk])
                ncommit = int((nk.cpu().numpy() + 1).sum())
                sweep.append({"k": kk, "K": kk + 1, "verify_us_median": round(float(np.median(us)), 1),
                              "verify_us_mean": round(float(us.mean()), 1),
                              "committed_tok_s": round(ncommit / (us.sum() / 1e6), 1),
                              "mean_committed": round(ncommit / nbk, 3)})
                state.check(sh)
            v1 = next((e["verify_us_mean"] for e in sweep if e["k"] == 0), None)
            if v1:
                for e in sweep:
                    e["R_pct"] = round(100.0 * (1.0 - e["verify_us_mean"] / (e["K"] * v1)), 1)
            return sweep

        sweep = (guarded(errors, "k_sweep", k_sweep) or []) if sweep_ks else []

        budget = None
        if len(sweep) == MAX_K + 1 and [e["k"] for e in sweep] == list(range(MAX_K + 1)):
            budget = guarded(errors, "budget", select_budget, args, lib, state, traj, sweep, cfg,
                             L0, root0, sh)

        e2e = None
        if not args.no_e2e:
            e2e = guarded(errors, "e2e", run_e2e, args, lib, W, state, traj, plans, cfg, L0,
                          root0, sh, stream)
        prefill = guarded(errors, "prefill", measure_prefill, args, lib, W, state, cfg, L0,
                          root0, sh, stream)
        long_ctx = None
        if args.long_kv_len > 0 and args.model == "7b":
            long_ctx = guarded(errors, "long_context", measure_long_context, args, lib, D, W,
                               model, cfg, sh, stream, seed)
        other_cfgs = None
        if not args.no_configs and args.model == "7b":
            other_cfgs = {"7b_ragged16": guarded(errors, "7b_ragged16", measure_ragged, args, lib,
                                                 D, model, cfg, sh, stream, seed)}
            guarded(errors, "close_7b", lambda: (state.close(), model.close()))
            torch.cuda.empty_cache()
            other_cfgs["1.5b_k_sweep"] = guarded(errors, "1.5b_k_sweep", measure_1p5b, args, lib,
                                                 D, sh, stream, seed)

    if ws > 1:
        elapsed_ms, committed_all = reduce_ranks(elapsed_ms, committed, "cuda")
    else:
        committed_all = committed
    value = committed_all / (elapsed_ms / 1e3)
    peak, peak_kind = load_peaks()

    # roofline of the dominant kernel class (per layer: one pair of events)
    H, F = cfg.hidden, cfg.ffn
    rows = k + 1
    cls = prof_cls
    mean_len = L0 + committed / 2.0
    per_unit = {
        "gate_up": 2 * F * H * 2 + rows * (H * 4 + 2 * H * 2 + F * 2),
        "down": H * F * 2 + rows * (F * 2 + 2 * H * 4),
        "qkv": (cfg.n_q + 2 * cfg.n_kv) * cfg.head_dim * H * 2 + rows * (H * 4 + 2 * H * 2),
        "o": H * cfg.n_q * cfg.head_dim * 2 + rows * (cfg.n_q * cfg.head_dim * 2 + 2 * H * 4),
        "lm_head": cfg.vocab * H * 2 + rows * (H * 4 + 2 * H * 2),
    }.get(cls)
    roofline = None
    if prof_n and per_unit:
        avg_ms = prof_ms / prof_n
        achieved = per_unit / (avg_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                    "unit": "GB/s", "frac": round(achieved / peak, 4),
                    "traffic": TRAFFIC.get(cls), "kernel": cls, "peak_kind": peak_kind,
                    "launches": prof_n, "avg_us": round(avg_ms * 1e3, 2),
                    "bytes_per_launch": int(per_unit),
                    "measured": f"CUDA event pair around each {cls} launch on the "
                                f"launching stream during a second timed pass over the same "
                                f"{steps} blocks ({pass2_ms / steps:.3f} ms/block with the "
                                "event pairs; the faster of two such passes); value comes "
                                "from the first pass, without them"}
    step_bytes = bytes_per_block(cfg, L0 + committed / 2.0, k)  # mean length over the blocks
    mean_us = elapsed_ms * 1e3 / steps
    med_us = float(np.median(per_block_us)) if per_block_us is not None else None
    step_roof = {"bytes_per_block": int(step_bytes),
                 "kv_bytes_written_per_block": int((k + 1) * cfg.kv_bytes_per_pos()),
                 "roofline_us": round(step_bytes / (peak * 1e9) * 1e6, 1),
                 "frac_of_mean_block": round(step_bytes / (peak * 1e9) / (mean_us / 1e6), 4),
                 "frac_of_median_block": (round(step_bytes / (peak * 1e9) / (med_us / 1e6), 4)
                                          if med_us else None),
                 "note": "mean over the headline pass (no event between blocks); median from "
                         "a diagnostic pass with an event pair around every block"}
    verify_us = None
    if per_block_us is not None:
        verify_us = {"mean": round(mean_us, 1), "median": round(med_us, 1),
                     "p10": round(float(np.percentile(per_block_us, 10)), 1),
                     "p90": round(float(np.percentile(per_block_us, 90)), 1)}

    line = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": ws,
        "steps": steps, "warmup": warm, "ms_per_step": round(elapsed_ms / steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded random-init weights and KV; greedy-derived candidates)",
        "config": {"workload": f"{args.model} verify, k={k}, L0={L0}, {steps} consecutive blocks, "
                               "geometric acceptance (mean 3, capped at k)",
                   "k": k, "kv_len": L0, "blocks": steps, "batch": 1, "capacity": cap,
                   "l2": f"inputs larger than L2 ({cfg.weight_bytes() / 1e9:.2f} GB of weights "
                         "streamed per step)",
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU"},
        "verify_us": verify_us,
        "mean_committed_per_block": round(committed / steps, 3),
        "plan_match": plan_match,
        "step_roofline": step_roof,
        "roofline": roofline,
        "gpu_launches": int(all_launches),
        "gpu_launches_detail": f"{int(all_launches)} libas2d kernels in the timed pass "
                               "(candidates of every block built before it)",
        "class_us_per_block": breakdown,
        "k_sweep": sweep,
        "budget": budget,
        "prefill": prefill,
        "long_context": long_ctx,
        "other_configs": other_cfgs,
        "clocks": clk,
        "e2e": e2e,
        "errors": errors or None,
        "profiles": {"launch_list": "profiles/launches_7b_k8_verify.md",
                     "kernel_classes": "profiles/kernels_7b2l_k8_L1564.md",
                     "attention": "profiles/attention_7b2l_k8.md",
                     "gate_up": "profiles/gemm_gateup_7b_k8.md",
                     "ragged": "profiles/kernels_7b2l_ragged16.md",
                     "1.5b": "profiles/kernels_1p5b_k8_L814.md"},
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = guarded(errors, "cpu_baseline", cpu_baseline, args, cfg, L0, plans)
        line["errors"] = errors or None
    if rank == 0:
        print(json.dumps(line), flush=True)
    if other_cfgs is None:
        guarded(errors, "close", lambda: (state.close(), model.close()))
    if ws > 1:
        dist.destroy_process_group()


def measure_long_context(args, lib, D, W, model, cfg, sh, stream, seed, ks=(1, 4, 8, 16),
                         blocks=16):
    """Verify time at a long retained prefix (10 min of audio at 25 tokens/s
    plus 128 instruction positions): `blocks` blocks per k from the same
    prefix, uniform candidates (the time does not depend on acceptance), CUDA
    events on the launching stream; the roofline counts the prefix's KV."""
    import torch
    L = args.long_kv_len
    cap = L + (max(ks) + 1) * blocks + 64
    kc, vc = D.device_kv(cfg, [L], cap, seed, poison=False)
    st = lib.State(model, [L], cap, kc, vc, [1])
    peak, _ = load_peaks()
    rng = np.random.default_rng(seed + 77)
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    c = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = []
    for k in ks:
        cand = torch.from_numpy(rng.integers(0, cfg.vocab, (blocks, k)).astype(np.int32)).cuda()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(blocks)]
        st.rollback([L], [1], sh)
        st.read_state(sh)
        st.verify(cand[0], [k], n, c, stream=sh)          # warm-up
        st.rollback([L], [1], sh)
        st.read_state(sh)
        torch.cuda.synchronize()
        for i in range(blocks):
            ev[i][0].record(stream)
            st.verify(cand[i], [k], n, c, stream=sh)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        us = float(np.mean([a.elapsed_time(b) * 1e3 for a, b in ev]))
        ln, _ = st.read_state(sh)
        mean_len = (L + ln[0]) / 2.0
        bts = bytes_per_block(cfg, mean_len, k)
        out.append({"k": k, "verify_us_mean": round(us, 1),
                    "kv_bytes": int((mean_len + k + 1) * cfg.kv_bytes_per_pos()),
                    "frac": round(bts / (peak * 1e9) / (us / 1e6), 4)})
    st.check(sh)
    st.close()
    del kc, vc
    torch.cuda.empty_cache()
    return {"kv_len": L, "blocks_per_k": blocks, "sweep": out}


def _timed_blocks(st, cands, ks, sh, stream):
    """Run one verification call per entry of `cands` (lists of per-request
    candidate lists) with CUDA events around each; returns (µs per call,
    committed tokens per call)."""
    import torch
    B = len(ks[0])
    n = torch.zeros(B, dtype=torch.int32, device="cuda")
    c = torch.zeros(B, dtype=torch.int32, device="cuda")
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in cands]
    n_all = []
    torch.cuda.synchronize()
    for i, (cd, kk) in enumerate(zip(cands, ks)):
        ev[i][0].record(stream)
        st.verify(cd, kk, n, c, stream=sh)
        ev[i][1].record(stream)
        n_all.append(n.clone())
    torch.cuda.synchronize()
    us = [a.elapsed_time(b) * 1e3 for a, b in ev]
    committed = [int((x + 1).sum().item()) for x in n_all]
    return us, committed


def measure_ragged(args, lib, D, model, cfg, sh, stream, seed, B=16, rounds=128):
    """The ragged workload: 16 requests with prefixes uniform in [250, 7500] and
    k uniform in {0..16} per request and round, verified together; uniform
    candidates (the work of a round does not depend on acceptance)."""
    import torch
    rng = np.random.default_rng(seed + 505)
    lens = [int(x) for x in rng.integers(250, 7501, B)]
    cap = max(lens) + 17 * rounds + 64
    kc, vc = D.device_kv(cfg, lens, cap, seed, poison=False)
    st = lib.State(model, lens, cap, kc, vc, [1] * B)
    ks = [[int(x) for x in rng.integers(0, 17, B)] for _ in range(rounds)]
    cands = [torch.from_numpy(rng.integers(0, cfg.vocab, max(sum(kk), 1)).astype(np.int32)).cuda()
             for kk in ks]
    _timed_blocks(st, cands[:3], ks[:3], sh, stream)       # warm-up
    st.rollback(lens, [1] * B, sh)
    st.read_state(sh)
    us, committed = _timed_blocks(st, cands, ks, sh, stream)
    ln, _ = st.read_state(sh)
    st.check(sh)
    peak, _ = load_peaks()
    kv_read = sum((lens[b] + ln[b]) / 2.0 for b in range(B)) * cfg.kv_bytes_per_pos()
    bts = cfg.weight_bytes() + kv_read
    mean_us = float(np.mean(us))
    st.close()
    del kc, vc
    torch.cuda.empty_cache()
    return {"requests": B, "rounds": rounds, "round_us_mean": round(mean_us, 1),
            "round_us_median": round(float(np.median(us)), 1),
            "mean_rows_per_round": round(float(np.mean([sum(kk) + B for kk in ks])), 1),
            "committed_tok_s": round(sum(committed) / (sum(us) / 1e6), 1),
            "frac": round(bts / (peak * 1e9) / (mean_us / 1e6), 4),
            "note": "uniform candidates: acceptance (and so committed tok/s) is low; the "
                    "work of a round does not depend on it"}


def measure_1p5b(args, lib, D, sh, stream, seed, L0=814, blocks=24):
    """The 1.5B-class decoder (814 prefilled positions), verify time versus
    k in {0, 1, 2, 4, 8}, uniform candidates."""
    import torch
    cfg = model_shape("1.5b")
    w = D.device_weights(cfg, seed)
    torch.cuda.synchronize()
    model = lib.Model(cfg, D.weight_pointers(cfg, w))
    del w
    torch.cuda.empty_cache()
    cap = L0 + 9 * (blocks + 2) + 64
    kc, vc = D.device_kv(cfg, [L0], cap, seed, poison=False)
    st = lib.State(model, [L0], cap, kc, vc, [1])
    peak, _ = load_peaks()
    rng = np.random.default_rng(seed + 606)
    out = []
    for k in (0, 1, 2, 4, 8):
        cands = [torch.from_numpy(rng.integers(0, cfg.vocab, max(k, 1)).astype(np.int32)).cuda()
                 for _ in range(blocks + 1)]
        st.rollback([L0], [1], sh)
        st.read_state(sh)
        _timed_blocks(st, cands[:1], [[k]], sh, stream)
        st.rollback([L0], [1], sh)
        st.read_state(sh)
        us, _ = _timed_blocks(st, cands[1:], [[k]] * blocks, sh, stream)
        ln, _ = st.read_state(sh)
        mean_us = float(np.mean(us))
        bts = bytes_per_block(cfg, (L0 + ln[0]) / 2.0, k)
        out.append({"k": k, "verify_us_mean": round(mean_us, 1),
                    "verify_us_median": round(float(np.median(us)), 1),
                    "frac": round(bts / (peak * 1e9) / (mean_us / 1e6), 4)})
    st.check(sh)
    st.close()
    model.close()
    return {"kv_len": L0, "blocks_per_k": blocks, "sweep": out}


def measure_prefill(args, lib, W, state, cfg, L0, root0, sh, stream, n_instr=64, reps=5):
    """Instruction-suffix prefill (App. A.1): the last n_instr positions of the
    workload's prefix forwarded by as2d_prefill over the retained audio
    positions before them (CUDA events on the launching stream; after every
    other measurement, since it rewrites those cache entries)."""
    import torch
    audio = L0 - n_instr
    tok = torch.from_numpy(W.instruction_tokens(cfg, n_instr, args.seed)).cuda()
    first = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    times = []
    for r in range(reps + 1):
        state.rollback([audio], [root0], sh)
        state.read_state(sh)
        t0.record(stream)
        state.prefill(tok, first, sh)
        t1.record(stream)
        torch.cuda.synchronize()
        if r > 0:
            times.append(t0.elapsed_time(t1))
    state.check(sh)
    ms = float(np.mean(times))
    return {"tokens": n_instr, "audio_positions": audio, "ms": round(ms, 3),
            "tok_s": round(n_instr / (ms / 1e3), 1),
            "passes": -(-n_instr // 64), "reps": reps}


def select_budget(args, lib, state, traj, sweep, cfg, L0, root0, sh):
    """Offline budget choice (Section 3.3; App. D.2): the measured mean call
    time of every k and development traces -- windows of the target's greedy
    text, the producer's copy with each token substituted w.p. 0.25 (the
    acceptance of this workload) -- rank b = 0..16 by estimated committed
    tok/s (as2d_budget_select).  The chosen b and b = 8 are then run as real
    sessions through the candidate buffer (producer text published ahead, no
    drafter cost) and measured."""
    rng = np.random.default_rng(args.seed + 4242)
    traj_h = [int(x) for x in traj.cpu().numpy()[1:]]
    win, n_commit = 220, 180
    traces = []
    for w in range(min(4, len(traj_h) // win)):
        ref = traj_h[w * win:(w + 1) * win]
        prod = [int(rng.integers(cfg.vocab)) if rng.random() < 0.25 else t for t in ref]
        traces.append((ref, prod))
    if not traces:
        return None
    cost = [e["verify_us_mean"] for e in sweep]
    st, best, tok_s, calls = lib.as2d_budget_select(cost, traces, n_commit, 8, 16)
    lib._check(st, "as2d_budget_select")
    measured = {}
    ref, prod = traces[0]
    for b in sorted({best, 8}):
        state.rollback([L0], [root0], sh)
        state.read_state(sh)
        buf = lib.CandidateBuffer(8)
        comm, stats = lib.session_run(state, None, buf, prod, b, n_commit, False,
                                      target_stream=sh)
        assert comm[:len(ref)] == ref[:len(comm)], "session text differs from greedy decoding"
        measured[str(b)] = {"tok_s": round(stats["committed"] / stats["V"], 1),
                            "calls": stats["rounds"], "committed": stats["committed"]}
    state.check(sh)
    v1 = cost[0]
    return {"selected_b": best,
            "est_tok_s": [round(x, 1) for x in tok_s],
            "est_calls": calls,
            "R_pct": [round(100.0 * (1.0 - c / ((k + 1) * v1)), 1) for k, c in enumerate(cost)],
            "measured_first_trace": measured,
            "dev": f"{len(traces)} windows of {win} greedy tokens, producer substitution "
                   f"p=0.25, {n_commit} committed per window, window W=8",
            "measured_note": "verifier service time only (producer text published ahead)"}


def run_e2e(args, lib, W, state, traj, plans, cfg, L0, root0, sh, stream):
    """Host-buffer loop through the C-ABI: per block, host candidates ->
    device, verify, (n_accepted, correction) -> host, host bookkeeping."""
    import torch
    k = args.k
    state.rollback([L0], [root0], sh)
    state.read_state(sh)
    traj_h = traj.cpu().numpy()
    cand_h = torch.zeros(k, dtype=torch.int32).pin_memory()
    out_h = torch.zeros(2, dtype=torch.int32).pin_memory()
    cand_d = torch.zeros(k, dtype=torch.int32, device="cuda")
    out_d = torch.zeros(2, dtype=torch.int32, device="cuda")
    steps = min(args.steps, len(plans))
    out = lib.make_verify_out(out_d.data_ptr(), out_d.data_ptr() + 4)
    m = 0
    committed = 0
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(steps):
        cand_h.numpy()[:] = W.apply_plan(traj_h[m + 1:m + 1 + k], plans[i], cfg.vocab)
        cand_d.copy_(cand_h, non_blocking=True)
        lib._check(lib.as2d_verify_block(state.handle, cand_d.data_ptr(), [k], out, sh),
                   "as2d_verify_block")
        out_h.copy_(out_d, non_blocking=True)
        stream.synchronize()
        n = int(out_h[0])
        m += n + 1
        committed += n + 1
    t1 = time.perf_counter()
    state.check(sh)
    return {"value": round(committed / (t1 - t0), 2), "unit": UNIT,
            "h2d_bytes_per_step": 4 * k, "d2h_bytes_per_step": 8, "steps": steps}


def cpu_baseline(args, cfg, L0, plans):
    """The CPU oracle (as it stands) on the same workload, on the host cores:
    one k-block forward at L0 with every core (OpenMP over output rows), and
    one decode row (one of the block's k + 1 rows) on a single thread."""
    import oracle
    from synth import workloads as W
    k = args.k
    hw = W.host_weights(cfg, args.seed)
    om = oracle.Model(cfg, hw)
    ks, vs = W.host_kv_request(cfg, 0, L0, L0 + k + 8, args.seed, poison=False)
    cache = om.cache(ks, vs)
    root = int(W.root_tokens(cfg, 1, args.seed)[0])
    cand = plans[0, 2:2 + k]
    mean_committed = float((plans[:, 0] + 1).mean())
    default_threads = oracle.set_threads(0)
    try:
        cores = oracle.set_threads(default_threads)
        t0 = time.perf_counter()
        om.verify_block(cache, L0, root, cand, want_logits=False)
        dt = time.perf_counter() - t0
        # one row single-threaded, at the block's last position (the rows of a
        # block cost the same up to the few extra keys)
        oracle.set_threads(1)
        t0 = time.perf_counter()
        om.decode_step(cache, L0, root)
        dt1 = time.perf_counter() - t0
    finally:
        oracle.set_threads(default_threads)
    v1 = mean_committed / (dt1 * (k + 1))
    return {"value": round(mean_committed / dt, 4), "unit": UNIT, "cores": cores,
            "kind": "oracle",
            "sample": f"one k={k} verification block of the {cfg.name} decoder at L={L0} "
                      f"({dt:.2f} s, fp64, OpenMP over output rows on {cores} threads); value = "
                      "mean committed tokens per block of the timed plan / that block time",
            "single_thread": {"value": round(v1, 4), "unit": UNIT, "cores": 1,
                              "sample": f"one decode row at L={L0} on one thread ({dt1:.2f} s); "
                                        f"value = mean committed tokens per block / ({k + 1} x "
                                        "that row time)"},
            "host_cores": os.cpu_count()}


def run_reference(args, ws, rank):
    """The CPU oracle timed as the reference arm: each step is one of the
    k+1 rows of a verification block (one decode step of the oracle)."""
    if rank != 0:
        return
    import oracle
    from synth import workloads as W
    cfg = model_shape(args.model)
    k, L0 = args.k, args.kv_len
    steps, warm = args.steps, args.warmup
    hw = W.host_weights(cfg, args.seed)
    om = oracle.Model(cfg, hw)
    cap = L0 + steps + warm + 8
    ks, vs = W.host_kv_request(cfg, 0, L0, cap, args.seed, poison=False)
    cache = om.cache(ks, vs)
    plans = draw_plans(args, max(steps, 1), cfg.vocab)
    tok = int(W.root_tokens(cfg, 1, args.seed)[0])
    pos = L0
    for _ in range(warm):
        om.decode_step(cache, pos, tok)
        pos += 1
    t0 = time.perf_counter()
    for i in range(steps):
        om.decode_step(cache, pos, tok)
        pos += 1
    dt = time.perf_counter() - t0
    rows_per_s = steps / dt
    mean_committed = float((plans[:, 0] + 1).mean())
    value = rows_per_s * mean_committed / (k + 1)
    cores = oracle.set_threads(0)
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
            "n_gpus": ws, "steps": steps, "warmup": warm,
            "ms_per_step": round(dt / steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{args.model} verify, k={k}, L0={L0}", "k": k, "kv_len": L0},
            "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": cores,
                             "kind": "oracle",
                             "sample": f"each step = one of the {k + 1} rows of a k={k} block "
                                       "(one oracle decode step); value = rows/s x mean "
                                       "committed tokens per block / (k+1)"},
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def producer_script(greedy, noise, vocab, seed):
    """The producer's text: the target's greedy text with each token replaced
    w.p. `noise`, plus one insertion and one deletion per 50 tokens (seeded)."""
    rng = np.random.default_rng(seed)
    out = []
    for t in greedy:
        r = rng.random()
        if r < noise:
            out.append(int(rng.integers(vocab)))
        elif r < noise + 0.02:
            out += [int(t), int(rng.integers(vocab))]
        elif r < noise + 0.04:
            continue
        else:
            out.append(int(t))
    return out


def run_session(args, ws, rank, local):
    """Target-decoupled decoding of one request (Section 3.1-3.2; App. D.2):
    the drafter decodes on its own stream and publishes its text in 8-token
    batches; the target verifies up to b ready candidates per call and decodes
    alone when none is ready.  Serial comparator, overlapped run and
    target-only decoding commit the same N tokens."""
    import torch

    import paper_2609_37617_gb300 as lib
    from synth import device as D
    from synth import workloads as W

    torch.cuda.set_device(local)
    cfg, dcfg = model_shape(args.model), model_shape(args.drafter)
    L0, DL0, N, b = args.kv_len, args.drafter_kv_len, args.session_tokens, args.session_b
    seed = args.seed + rank
    s_t = torch.cuda.Stream(priority=-1)   # the verifier is the critical path
    s_d = torch.cuda.Stream(priority=0)
    models, states = [], []
    n_script = 2 * N + 64
    cpu = None
    if args.cpu_drafter:
        ccfg = model_shape("cpu-draft")
        hw = W.host_weights(ccfg, seed + 202)
        f32 = lambda b: (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)
        host = {k: f32(hw[k]) for k in ("embed", "final_norm", "lm_head")}
        for name in ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm", "w_gate", "w_up", "w_down"):
            host[name] = [f32(hw[f"{name}.{l}"]) for l in range(ccfg.n_layers)]
        # half the host cores: more threads slow the verifier's own host thread
        cpu_threads = args.cpu_threads or max(1, min(8, (os.cpu_count() or 8) // 2))
        cpu = lib.CpuDecoder(ccfg, host, n_script + 16, cpu_threads, 1)
        del host, hw
        dcfg = None
    for c, L, sd in ((cfg, L0, seed), (dcfg, DL0, seed + 101)):
        if c is None:
            continue
        w = D.device_weights(c, sd)
        torch.cuda.synchronize()
        models.append(lib.Model(c, D.weight_pointers(c, w)))
        del w
        torch.cuda.empty_cache()
    if args.drafter_sms > 0 and cpu is None:
        n_sm = torch.cuda.get_device_properties(local).multi_processor_count
        models[0].set_sm_budget(n_sm - args.drafter_sms)
        models[1].set_sm_budget(args.drafter_sms)
    cap_t = L0 + 2 * N + 64
    cap_d = DL0 + n_script + 16
    kc, vc = D.device_kv(cfg, [L0], cap_t, seed, poison=False)
    root_t = int(W.root_tokens(cfg, 1, seed)[0])
    target = lib.State(models[0], [L0], cap_t, kc, vc, [root_t])
    drafter = None
    if cpu is None:
        dkc, dvc = D.device_kv(dcfg, [DL0], cap_d, seed + 101, poison=False)
        root_d = int(W.root_tokens(dcfg, 1, seed + 101)[0])
        drafter = lib.State(models[1], [DL0], cap_d, dkc, dvc, [root_d])

    # the target's greedy text (untimed), then the producer's noisy copy
    nbuf = torch.zeros(1, dtype=torch.int32, device="cuda")
    greedy = torch.zeros(N + 32, dtype=torch.int32, device="cuda")
    for j in range(N + 32):
        out = lib.make_verify_out(nbuf.data_ptr(), greedy.data_ptr() + 4 * j)
        lib._check(lib.as2d_decode_step(target.handle, out, s_t.cuda_stream), "as2d_decode_step")
    target.check(s_t.cuda_stream)
    greedy_h = [int(x) for x in greedy.cpu()]
    script = producer_script(greedy_h, args.session_noise, cfg.vocab, seed + 7)[:n_script]

    def one(kind):
        target.rollback([L0], [root_t], s_t.cuda_stream)
        target.read_state(s_t.cuda_stream)
        if drafter is not None:
            drafter.rollback([DL0], [root_d], s_d.cuda_stream)
            drafter.read_state(s_d.cuda_stream)
        else:
            cpu.reset(0, 1)
        torch.cuda.synchronize()
        buf = lib.CandidateBuffer(8)
        sc = [] if kind == "target_only" else script
        comm, st = lib.session_run(target, drafter if sc else None, buf, sc, b, N,
                                   kind == "overlapped", target_stream=s_t.cuda_stream,
                                   drafter_stream=s_d.cuda_stream,
                                   cpu_drafter=cpu if sc else None)
        target.check(s_t.cuda_stream)
        if drafter is not None:
            drafter.check(s_d.cuda_stream)
        m = min(len(comm), len(greedy_h))
        assert comm[:m] == greedy_h[:m], f"{kind}: committed text differs from greedy decoding"
        st["tok_s"] = st["committed"] / st["T"]
        return {k: (round(v, 6) if isinstance(v, float) else v) for k, v in st.items()}

    for _ in range(max(args.warmup, 1)):
        one("overlapped")
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    runs = {kind: one(kind) for kind in ("target_only", "serial", "overlapped")}
    clk = clocks.stop()
    s, a = runs["serial"], runs["overlapped"]
    dD, dV, dH = a["D"] - s["D"], a["V"] - s["V"], a["H"] - s["H"]
    line = {
        "metric": "target-decoupled session: committed tok/s and overlap accounting "
                  "T = D + V - O + H",
        "value": round(a["tok_s"], 2), "unit": UNIT, "n_gpus": 1, "steps": 1,
        "warmup": max(args.warmup, 1), "ms_per_step": round(a["T"] * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded random-init weights and KV; the producer publishes the "
                "target's greedy text with seeded corruption while running the drafter's "
                "own decode steps for their cost)",
        "config": {"workload": f"{args.model} target (L0={L0}) + "
                               + (f"cpu-draft drafter on {cpu_threads} host threads"
                                  if cpu is not None else f"{args.drafter} drafter (L0={DL0})")
                               + f", N={N} committed tokens, b={b}, 8-token batches, "
                               f"substitution p={args.session_noise}, 2% insertions, 2% deletions"
                               + (f", drafter on {args.drafter_sms} SMs and target on the rest"
                                  if args.drafter_sms > 0 else ", both on every SM"),
                   "l2": "inputs larger than L2 (weights streamed per call)"},
        "runs": runs,
        "speedup_overlapped_vs_serial": round(s["T"] / a["T"], 4),
        "speedup_overlapped_vs_target_only": round(runs["target_only"]["T"] / a["T"], 4),
        "break_even": {"O_a": round(a["O"], 6), "dD_plus_dV_plus_dH": round(dD + dV + dH, 6),
                       "Ts_minus_Ta": round(s["T"] - a["T"], 6)},
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    target.close()
    if drafter is not None:
        drafter.close()
    if cpu is not None:
        cpu.close()
    for m in models:
        m.close()


def main():
    args = parse()
    ws, rank, local = dist_setup(args)
    if args.session:
        run_session(args, ws, rank, local)
        return
    if args.impl == "reference":
        run_reference(args, ws, rank)
        return
    run_ours(args, ws, rank, local)


if __name__ == "__main__":
    main()
