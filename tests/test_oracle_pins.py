"""Pins of the CPU oracle to facts outside itself: closed forms, invariants,
special cases that reduce to a library routine (numpy/torch), brute force on
tiny inputs, and the paper's worked example (Section 3.2, Fig. 4).

Each sub-step test is chosen so that a plausible mistake (a dropped term, a
wrong sign, a wrong pairing index, a transposed operand, a wrong scale) fails.
"""
import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from synth import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16_decode(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def bf16_bits_of(x):
    """Exact bf16 bits for values that are bf16-representable."""
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


# ---- bf16 rounding ------------------------------------------------------------

def _exact_rne_bf16(x):
    """Brute force: nearest bf16 value by exact rational comparison."""
    f = Fraction(x)
    if f == 0:
        return 0.0
    sign = -1 if f < 0 else 1
    a = abs(f)
    e = math.floor(math.log2(a))
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    ulp = Fraction(2) ** (max(e, -126) - 7)
    q = a / ulp
    lo = math.floor(q)
    rem = q - lo
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and lo % 2 == 1):
        lo += 1
    return sign * float(lo * ulp)


def test_bf16_known_values(built):
    assert oracle.double_to_bf16(1.0) == 0x3F80
    assert oracle.double_to_bf16(-2.0) == 0xC000
    assert oracle.double_to_bf16(1.0 + 2 ** -8) == 0x3F80          # tie -> even
    assert oracle.double_to_bf16(1.0 + 3 * 2 ** -8) == 0x3F82      # tie -> even (up)
    assert oracle.double_to_bf16(1.0 + 2 ** -8 + 2 ** -30) == 0x3F81  # above tie
    assert oracle.double_to_bf16(float("nan")) & 0x7F80 == 0x7F80
    assert oracle.double_to_bf16(1e39) == 0x7F80


def test_bf16_matches_torch_and_exact(built):
    rng = np.random.default_rng(0)
    x = rng.standard_normal(3000) * np.exp(rng.uniform(-20, 20, 3000))
    # float32 inputs: torch's float32 -> bfloat16 conversion (round to nearest even)
    xf = x.astype(np.float32)
    want = torch.from_numpy(xf).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.double_to_bf16(float(v)) for v in xf], np.uint16)
    assert np.array_equal(got, want)
    # double inputs (no double rounding through float): exact rational rounding
    for v in x[:400]:
        assert bf16_decode(oracle.double_to_bf16(float(v))) == _exact_rne_bf16(float(v))


# ---- RMSNorm ------------------------------------------------------------------

def test_rmsnorm_unit_rms_and_scale_invariance(built):
    rng = np.random.default_rng(1)
    x = rng.standard_normal(256) * 3.0 + 0.5
    ones = np.full(256, W.ONE_BF16, np.uint16)
    y = oracle.rmsnorm(x, ones, 0.0)
    assert abs(np.sqrt(np.mean(y ** 2)) - 1.0) < 1e-12
    assert np.allclose(oracle.rmsnorm(7.5 * x, ones, 0.0), y, rtol=1e-12, atol=0)
    # direction is kept (no mean subtraction: RMSNorm, not LayerNorm)
    assert np.allclose(y / np.linalg.norm(y), x / np.linalg.norm(x), atol=1e-12)
    # gains multiply elementwise
    g = bf16_bits_of(rng.uniform(0.5, 1.5, 256).astype(np.float32))
    yg = oracle.rmsnorm(x, g, 0.0)
    assert np.allclose(yg, y * bf16_decode(g), rtol=1e-12)
    # eps enters under the root: mean(x^2) = 1 and eps = 3 gives a factor 1/2
    z = np.ones(64)
    assert np.allclose(oracle.rmsnorm(z, np.full(64, W.ONE_BF16, np.uint16), 3.0), 0.5)


# ---- linear -------------------------------------------------------------------

def test_linear_matches_numpy_matmul(built):
    rng = np.random.default_rng(2)
    w = bf16_bits_of(rng.standard_normal((37, 53)).astype(np.float32))
    x = rng.standard_normal(53)
    want = bf16_decode(w) @ x          # library matmul; non-square, so a transpose fails
    assert np.allclose(oracle.linear(w, x), want, rtol=1e-12, atol=1e-12)


# ---- RoPE ---------------------------------------------------------------------

def test_rope_closed_forms(built):
    d, theta = 8, 10000.0
    rng = np.random.default_rng(3)
    v = rng.standard_normal(d)
    assert np.allclose(oracle.rope(v, 0, theta), v)                       # identity at 0
    for pos in (1, 17, 15127):
        assert abs(np.linalg.norm(oracle.rope(v, pos, theta)) - np.linalg.norm(v)) < 1e-9
    # unit vector e_i turns towards e_{i+d/2} by pos * theta^(-2i/d)
    for i in range(d // 2):
        e = np.zeros(d)
        e[i] = 1.0
        pos = 3
        w = pos * theta ** (-2.0 * i / d)
        want = np.zeros(d)
        want[i] = math.cos(w)
        want[i + d // 2] = math.sin(w)
        assert np.allclose(oracle.rope(e, pos, theta), want, atol=1e-14)
    # e_0 at position 1: frequency 1 -> angle 1 rad
    e0 = np.eye(d)[0]
    assert np.allclose(oracle.rope(e0, 1, theta)[[0, d // 2]], [math.cos(1), math.sin(1)])


def test_rope_group_and_relative_position(built):
    d, theta = 16, 1e6
    rng = np.random.default_rng(4)
    v = rng.standard_normal(d)
    q = rng.standard_normal(d)
    # rotations compose: angles are linear in the position
    assert np.allclose(oracle.rope(oracle.rope(v, 5, theta), 9, theta), oracle.rope(v, 14, theta))
    # scores depend on the offset only
    s1 = oracle.rope(q, 100, theta) @ oracle.rope(v, 40, theta)
    s2 = oracle.rope(q, 1060, theta) @ oracle.rope(v, 1000, theta)
    assert abs(s1 - s2) < 1e-9


# ---- attention ----------------------------------------------------------------

def test_attention_single_key_returns_value(built):
    rng = np.random.default_rng(5)
    d = 64
    k = bf16_bits_of(rng.standard_normal((1, d)).astype(np.float32))
    v = bf16_bits_of(rng.standard_normal((1, d)).astype(np.float32))
    out = oracle.attend(rng.standard_normal(d), k, v)
    assert np.allclose(out, bf16_decode(v[0]), atol=1e-15)


def test_attention_equal_keys_give_mean(built):
    rng = np.random.default_rng(6)
    d, n = 32, 9
    k = np.tile(bf16_bits_of(rng.standard_normal(d).astype(np.float32)), (n, 1))
    v = bf16_bits_of(rng.standard_normal((n, d)).astype(np.float32))
    out = oracle.attend(rng.standard_normal(d), k, v)
    assert np.allclose(out, bf16_decode(v).mean(axis=0), atol=1e-14)


def test_attention_two_keys_logistic_scale(built):
    """Two keys with scores a/sqrt(d) and 0: the first value gets weight
    1 / (1 + exp(-a / sqrt(d))).  Fails for a missing or wrong 1/sqrt(d)."""
    d, a = 64, 3.0
    q = np.zeros(d)
    q[0] = a
    k = np.zeros((2, d), np.uint16)
    k[0, 0] = W.ONE_BF16
    v = np.zeros((2, d), np.uint16)
    v[0, 1] = W.ONE_BF16          # V1 = e_1
    v[1, 2] = W.ONE_BF16          # V2 = e_2
    out = oracle.attend(q, k, v)
    p = 1.0 / (1.0 + math.exp(-a / math.sqrt(d)))
    assert abs(out[1] - p) < 1e-14 and abs(out[2] - (1 - p)) < 1e-14


def test_attention_permutation_invariant(built):
    rng = np.random.default_rng(7)
    d, n = 32, 11
    k = bf16_bits_of(rng.standard_normal((n, d)).astype(np.float32))
    v = bf16_bits_of(rng.standard_normal((n, d)).astype(np.float32))
    q = rng.standard_normal(d)
    perm = rng.permutation(n)
    assert np.allclose(oracle.attend(q, k, v), oracle.attend(q, k[perm], v[perm]), atol=1e-13)


# ---- SiLU, argmax, accept rule -----------------------------------------------

def test_silu_closed_forms(built):
    assert oracle.silu(0.0) == 0.0
    assert abs(oracle.silu(1.0) - 1.0 / (1.0 + math.exp(-1.0))) < 1e-15
    for x in (-3.0, -0.5, 0.7, 4.0):
        assert abs((oracle.silu(x) - oracle.silu(-x)) - x) < 1e-14   # silu(x) - silu(-x) = x
    assert abs(oracle.silu(40.0) - 40.0) < 1e-12


def test_argmax_lowest_index_tie_break(built):
    assert oracle.argmax([1.0, 3.0, 3.0, 2.0]) == (1, 0.0)
    i, m = oracle.argmax([0.5, -1.0, 2.0, 1.25])
    assert i == 2 and abs(m - 0.75) < 1e-15
    assert oracle.argmax([-5.0])[0] == 0


def test_accept_worked_example_fig4(built):
    with open(os.path.join(GOLDEN, "fig_token_flow.json")) as f:
        g = json.load(f)
    T = g["tokens"]
    cand = [T[c] for c in g["candidates"]]
    greedy = [T[c] for c in g["greedy"]]
    n, corr = oracle.accept(cand, greedy)
    assert n == g["expected"]["n_accepted"]
    assert corr == T[g["expected"]["correction"]]
    committed = cand[:n] + [corr]
    assert committed == [T[c] for c in g["expected"]["committed"]]


def test_accept_brute_force_tiny_vocab(built):
    """Over every candidate block of length <= 4 on a 3-token vocabulary and
    every greedy sequence, n is the largest j such that the first j
    candidates equal the first j greedy tokens, and the correction is the
    greedy token at place n (the bonus token when n = k)."""
    V = 3
    for k in range(0, 5):
        for cand in itertools.product(range(V), repeat=k):
            for greedy in itertools.product(range(V), repeat=k + 1):
                n, corr = oracle.accept(list(cand), list(greedy))
                best = max(j for j in range(k + 1) if list(cand[:j]) == list(greedy[:j]))
                assert n == best and corr == greedy[best]


# ---- whole-model special cases ------------------------------------------------

def _zero_like(w, keep=()):
    out = {}
    for name, a in w.items():
        kind = name.split(".")[0]
        if kind in ("embed", "lm_head", "final_norm", "attn_norm", "mlp_norm") or kind in keep:
            out[name] = a
        else:
            out[name] = np.zeros_like(a)
    return out


TINYCFG = W.ModelConfig("pin", 2, 64, 4, 2, 16, 96, 50, rope_theta=1e4, rms_eps=1e-6)


def _cache(cfg, L, cap, seed=0, poison=True):
    return W.host_kv_request(cfg, 0, L, cap, seed=seed, poison=poison)


def test_zero_layers_reduce_to_lm_head_gemv(built):
    """All layer matrices zero: the residual stream is the embedding row, so the
    logits are W_lm . rmsnorm(E[t]) -- a plain matrix-vector product."""
    cfg = TINYCFG
    w = _zero_like(W.host_weights(cfg, seed=1, gains="random"))
    m = oracle.Model(cfg, w)
    ks, vs = _cache(cfg, 5, 8)
    c = m.cache(ks, vs)
    t = 17
    logits = m.decode_step(c, 5, t)
    e = bf16_decode(w["embed"][t])
    n = e / np.sqrt(np.mean(e ** 2) + cfg.rms_eps) * bf16_decode(w["final_norm"])
    want = bf16_decode(w["lm_head"]) @ n
    assert np.allclose(logits, want, rtol=1e-10, atol=1e-12)


def test_uniform_attention_layer_closed_form(built):
    """One layer, W_q = W_k = 0 (all scores 0, so attention is the mean of the
    values at positions 0..pos, the new token's value included), MLP zero.
    h' = E[t] + W_o [mean V_{g(j)}]_j with g(j) = j // group."""
    cfg = W.ModelConfig("pin1", 1, 64, 4, 2, 16, 96, 50, rope_theta=1e4, rms_eps=1e-6)
    w = W.host_weights(cfg, seed=2, gains="random")
    for kind in ("w_q", "w_k", "w_gate", "w_up", "w_down"):
        w[f"{kind}.0"] = np.zeros_like(w[f"{kind}.0"])
    m = oracle.Model(cfg, w)
    L, cap, t = 6, 10, 33
    ks, vs = _cache(cfg, L, cap, seed=3)
    c = m.cache(ks, vs)
    logits = m.decode_step(c, L, t)
    # expected residual stream
    h = bf16_decode(w["embed"][t])
    a = h / np.sqrt(np.mean(h ** 2) + cfg.rms_eps) * bf16_decode(w["attn_norm.0"])
    vnew = bf16_decode(w["w_v.0"]) @ a                      # [n_kv * d]
    d = cfg.head_dim
    o = []
    for j in range(cfg.n_q):
        g = j // cfg.group
        vals = bf16_decode(vs[0][g, :L, :])
        newv = bf16_decode([oracle.double_to_bf16(x) for x in vnew[g * d:(g + 1) * d]])
        o.append(np.vstack([vals, newv]).mean(axis=0))
    h2 = h + bf16_decode(w["w_o.0"]) @ np.concatenate(o)
    f = h2 / np.sqrt(np.mean(h2 ** 2) + cfg.rms_eps) * bf16_decode(w["final_norm"])
    want = bf16_decode(w["lm_head"]) @ f
    assert np.allclose(logits, want, rtol=1e-9, atol=1e-11)
    # the appended value row is stored rounded to bf16
    assert np.array_equal(c.v[0][1, L], np.array([oracle.double_to_bf16(x) for x in vnew[d:2 * d]], np.uint16))


def test_mlp_one_hot_closed_form(built):
    """Attention output zero (W_o = 0), embedding row c*e_j: rmsnorm gives
    sqrt(H) sign(c) e_j, so gate/up are columns j of W_gate/W_up scaled by
    sqrt(H) and h' = c e_j + W_down (silu(gate) * up)."""
    cfg = W.ModelConfig("pin2", 1, 64, 4, 2, 16, 96, 50, rope_theta=1e4, rms_eps=0.0)
    w = W.host_weights(cfg, seed=4)
    w["w_o.0"] = np.zeros_like(w["w_o.0"])
    emb = np.zeros_like(w["embed"])
    j, t, cval = 5, 9, -0.375
    emb[t, j] = bf16_bits_of(np.float32(cval))
    w["embed"] = emb
    m = oracle.Model(cfg, w)
    ks, vs = _cache(cfg, 3, 6)
    logits = m.decode_step(m.cache(ks, vs), 3, t)
    H = cfg.hidden
    s = math.sqrt(H) * np.sign(cval)
    gate = s * bf16_decode(w["w_gate.0"])[:, j]
    up = s * bf16_decode(w["w_up.0"])[:, j]
    h2 = np.zeros(H)
    h2[j] = cval
    h2 = h2 + bf16_decode(w["w_down.0"]) @ (gate / (1 + np.exp(-gate)) * up)
    f = h2 / np.sqrt(np.mean(h2 ** 2)) * bf16_decode(w["final_norm"])
    assert np.allclose(logits, bf16_decode(w["lm_head"]) @ f, rtol=1e-9, atol=1e-11)


# ---- verification invariants (I1-I6) ----------------------------------------

@pytest.fixture(scope="module")
def tiny_model(built):
    cfg = TINYCFG
    w = W.host_weights(cfg, seed=11, gains="random")
    return cfg, oracle.Model(cfg, w)


def test_I1_greedy_candidates_fully_accepted(tiny_model):
    cfg, m = tiny_model
    L, cap, k = 12, 40, 6
    ks, vs = _cache(cfg, L, cap, seed=5)
    c = m.cache(ks, vs)
    root = 7
    cont, _ = oracle.greedy_continuation(m, c, L, root, k + 1)
    r = m.verify_block(c.copy(m), L, root, cont[:k])
    assert r["n_accepted"] == k
    assert r["correction"] == cont[k]                  # the bonus token
    assert r["new_len"] == L + k + 1 and r["new_root"] == cont[k]


def test_I2_I3_block_equals_sequential_decode_brute_force(built):
    """Vocabulary of 8, every candidate block of length <= 3: the accepted
    length is the first mismatch against the greedy tokens of sequential
    decode steps, and every row's logits equal that decode step's logits."""
    cfg = W.ModelConfig("pin3", 1, 32, 2, 1, 16, 48, 8, rope_theta=1e4, rms_eps=1e-6)
    m = oracle.Model(cfg, W.host_weights(cfg, seed=12, gains="random"))
    L, cap, root = 4, 12, 3
    ks, vs = _cache(cfg, L, cap, seed=6)
    base = m.cache(ks, vs)
    for k in range(0, 4):
        for cand in itertools.product(range(cfg.vocab), repeat=k):
            r = m.verify_block(base.copy(m), L, root, list(cand))
            seq = base.copy(m)
            toks = [root] + list(cand)
            greedy = []
            for i, t in enumerate(toks):
                lg = m.decode_step(seq, L + i, t)
                assert np.array_equal(lg, r["logits"][i])
                greedy.append(oracle.argmax(lg)[0])
            n = 0
            while n < k and cand[n] == greedy[n]:
                n += 1
            assert r["n_accepted"] == n and r["correction"] == greedy[n]


def test_I4_k0_is_plain_decode(tiny_model):
    cfg, m = tiny_model
    L, cap = 9, 20
    ks, vs = _cache(cfg, L, cap, seed=7)
    c = m.cache(ks, vs)
    lg = m.decode_step(c.copy(m), L, 21)
    r = m.verify_block(c.copy(m), L, 21, [])
    assert r["n_accepted"] == 0
    assert np.array_equal(r["logits"][0], lg)
    assert r["correction"] == oracle.argmax(lg)[0]
    assert r["new_len"] == L + 1


def test_I5_state_restoration_after_rejection(tiny_model):
    """After a rejection the retained cache equals the cache built by decoding
    the committed tokens one by one, and the rejected slots are never read by
    later steps (they hold NaN; every later logit stays finite)."""
    cfg, m = tiny_model
    L, cap, k = 10, 40, 5
    ks, vs = _cache(cfg, L, cap, seed=8)
    c0 = m.cache(ks, vs)
    root = 4
    cont, _ = oracle.greedy_continuation(m, c0, L, root, k)
    cand = cont.copy()
    cand[2] = (cand[2] + 1) % cfg.vocab                   # reject at place 2
    c = c0.copy(m)
    r = m.verify_block(c, L, root, cand)
    assert r["n_accepted"] == 2
    keep = r["new_len"]
    assert keep == L + 3
    ref = c0.copy(m)
    for i, t in enumerate([root] + list(cand[:2])):
        m.decode_step(ref, L + i, t)
    for l in range(cfg.n_layers):
        assert np.array_equal(c.k[l][:, :keep], ref.k[l][:, :keep])
        assert np.array_equal(c.v[l][:, :keep], ref.v[l][:, :keep])
        assert np.all(c.k[l][:, keep:L + k + 1] == W.NAN_BF16)
    r2 = m.verify_block(c, keep, r["new_root"], cont[:3])
    assert np.all(np.isfinite(r2["logits"]))


def test_I6_commit_then_next_root(tiny_model):
    """The committed tokens of a block are the accepted candidates followed by
    the correction, which is carried as the next root and not forwarded."""
    cfg, m = tiny_model
    L, cap = 10, 40
    ks, vs = _cache(cfg, L, cap, seed=9)
    c = m.cache(ks, vs)
    cont, _ = oracle.greedy_continuation(m, c, L, 2, 4)
    cand = cont.copy()
    cand[1] = (cand[1] + 3) % cfg.vocab
    r = m.verify_block(c, L, 2, cand)
    assert r["n_accepted"] == 1 and r["correction"] == cont[1]
    assert r["new_root"] == cont[1] and r["new_len"] == L + 2


def test_fp32_build_agrees_with_fp64(built):
    cfg = W.TINY
    w = W.host_weights(cfg, seed=0)
    L, cap = 200, 216
    ks, vs = W.host_kv_request(cfg, 0, L, cap, seed=0)
    m64 = oracle.Model(cfg, w, "f64")
    m32 = oracle.Model(cfg, w, "f32")
    assert oracle.load("f32").oracle_real_bytes() == 4
    cand = [5, 6, 7, 8]
    r64 = m64.verify_block(m64.cache(ks, vs), L, 100, cand)
    r32 = m32.verify_block(m32.cache(ks, vs), L, 100, cand)
    assert np.max(np.abs(r64["logits"] - r32["logits"])) < 1e-3
    sure = r64["margin"] > 1e-2
    assert np.array_equal(r64["greedy"][sure], r32["greedy"][sure])
