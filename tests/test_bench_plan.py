"""bench.py's capacity plan: every leg that reuses the headline state fits its
cache at any --steps / --warmup, under the library's own rule (a call is
refused once the host bound of the length + k + 1 exceeds the capacity; the
bound grows by k + 1 per call until it is read back).  CPU only."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402

L0, K = 1564, 8
SWEEP = list(range(17))


def leg_fits(cap, L0, calls, k):
    """Simulate one leg's calls from a rollback to L0 under the capacity rule."""
    bound = L0
    for _ in range(calls):
        if bound + k + 1 > cap:
            return False
        bound += k + 1
    return True


@pytest.mark.parametrize("steps", [1, 5, 20, 256])
@pytest.mark.parametrize("warmup", [1, 3, 5, 40])
@pytest.mark.parametrize("sweep_blocks", [1, 24, 64])
def test_every_leg_fits(steps, warmup, sweep_blocks):
    rng = np.random.default_rng(steps * 31 + warmup)
    # planned commits per block: between 1 and k + 1
    committed_plan = int(rng.integers(1, K + 2, steps).sum())
    traj_len, cap, needs = bench.plan_capacity(L0, K, steps, warmup, SWEEP, sweep_blocks,
                                               committed_plan)
    # the greedy trajectory: traj_len k = 0 steps from L0
    assert leg_fits(cap, L0, traj_len, 0)
    assert leg_fits(cap, L0, warmup, K)
    assert leg_fits(cap, L0, steps, K)             # timed passes and the e2e leg
    assert leg_fits(cap, L0, min(8, steps), K)     # per-class breakdown
    for kk in SWEEP:
        assert leg_fits(cap, L0, sweep_blocks, kk), kk
    # budget sessions read every outcome back: commits + one widest call
    assert L0 + bench.BUDGET_COMMIT + 2 * (bench.MAX_K + 1) <= cap
    # the trajectory covers every timed block's candidates, the sweep's
    # candidate reads, and the budget leg's development windows
    assert traj_len >= committed_plan + K + 1
    assert traj_len >= max((kk + 1) * sweep_blocks + kk + 1 for kk in SWEEP)
    assert traj_len // bench.BUDGET_WIN >= bench.BUDGET_TRACES
    assert set(needs) >= {"trajectory", "warmup", "timed", "k_sweep", "budget"}


def test_driver_command_was_short():
    """The command the harness runs (--steps 20 --warmup 5) used to
    overrun the capacity in the k-sweep (24 blocks of k = 16 need 408
    positions past L0; the old plan gave 9 x 20 + trajectory)."""
    traj_len, cap, needs = bench.plan_capacity(L0, K, 20, 5, SWEEP, 24, 20 * 4)
    assert needs["k_sweep"] == 17 * 24
    assert cap >= L0 + 17 * 24


def test_guarded_records_failures():
    errors = {}
    assert bench.guarded(errors, "ok", lambda: 3) == 3
    assert bench.guarded(errors, "bad", lambda: 1 / 0) is None
    assert list(errors) == ["bad"] and "ZeroDivisionError" in errors["bad"]
