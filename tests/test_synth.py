"""The seeded input generator: Philox4x32-10 against its published
known-answer vectors, and the distribution of the drawn values."""
import json
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_philox_known_answers(built):
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.json")) as f:
        kat = json.load(f)
    for v in kat["vectors"]:
        ctr = [int(x, 16) for x in v["ctr"]]
        key = [int(x, 16) for x in v["key"]]
        want = tuple(int(x, 16) for x in v["out"])
        assert synth.philox4x32_10(ctr, key) == want


def test_normal_moments(built):
    x = synth.normal_bf16(1 << 20, seed=7, stream=99, sigma=0.02)
    f = (x.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert abs(f.mean()) < 1e-4
    assert abs(f.std() - 0.02) < 2e-4
    # Irwin-Hall(8) is bounded at sqrt(3*8) = 4.9 sigma.
    assert np.abs(f).max() <= 0.02 * np.sqrt(24) * 1.01


def test_streams_and_seeds_differ(built):
    a = synth.normal_bf16(1000, 0, 1)
    b = synth.normal_bf16(1000, 0, 2)
    c = synth.normal_bf16(1000, 1, 1)
    assert (a != b).mean() > 0.9 and (a != c).mean() > 0.9
    assert np.array_equal(a, synth.normal_bf16(1000, 0, 1))


def test_uniform_int_range(built):
    t = synth.uniform_int(100000, 3, 5, 37)
    assert t.min() == 0 and t.max() == 36
    counts = np.bincount(t, minlength=37)
    assert counts.min() > 100000 / 37 * 0.9


def test_offset_gains(built):
    g = synth.normal_bf16(4096, 0, 3, sigma=0.1, base=1.0)
    f = (g.astype(np.uint32) << 16).view(np.float32)
    assert abs(f.mean() - 1.0) < 0.01


def test_sharp_gains_scale_only_the_final_norm():
    """gains="sharp": layer gains stay 1.0, the final norm's gain is 8.0
    (exact in bf16), every other tensor is the unit-gain model's."""
    from synth import workloads as W
    unit = W.host_weights(W.TINY, 0)
    sharp = W.host_weights(W.TINY, 0, gains="sharp")
    assert np.all(sharp["final_norm"] == 0x4100)          # 8.0 in bf16
    for name in unit:
        if name != "final_norm":
            assert np.array_equal(unit[name], sharp[name]), name


def test_sharp_root_search_finds_separated_decisions():
    """The exactness tests' root search, on the oracle only: on the sharp tiny
    model it finds a root whose 9-token greedy continuation from 200
    positions has every margin above 0.1 (the unit-gain model's margins are
    mostly below it)."""
    import oracle
    from synth import workloads as W
    from tests.helpers import MARGIN_SURE, sharp_root
    cfg = W.TINY
    om = oracle.Model(cfg, W.host_weights(cfg, 0, gains="sharp"))
    ks, vs = W.host_kv_request(cfg, 0, 200, 256, 0)
    root, cont, m = sharp_root(om, lambda: om.cache(ks, vs), 200, 9)
    assert len(cont) == 9 and np.all(np.asarray(m) > MARGIN_SURE)
