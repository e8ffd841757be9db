"""Model shapes, stream ids and seeded input recipes of the five workloads.

The paper measures on phone ASR/translation/QA corpora with trained Qwen
weights; none are available, so seeded synthetic inputs with the workloads'
shapes stand in for them: weights N(0, 0.02) stored bf16, prefilled KV caches
N(0, 1) bf16 (25 audio tokens per second plus instruction tokens), and
candidate blocks derived from the target's own greedy continuation with a
stated corruption rule.

Every tensor is keyed by a stream id and filled in its logical row-major
order, so host (oracle) and device copies agree element by element whatever
layout either side uses afterwards.
"""
from dataclasses import dataclass, field

import numpy as np

import synth

NAN_BF16 = 0x7FC0
ONE_BF16 = 0x3F80


@dataclass(frozen=True)
class ModelConfig:
    name: str
    n_layers: int
    hidden: int
    n_q: int
    n_kv: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6

    @property
    def group(self):
        return self.n_q // self.n_kv

    def weight_bytes(self):
        """bf16 bytes streamed per block: all layer matrices and the LM head
        (the embedding contributes only the gathered rows)."""
        h, d = self.hidden, self.head_dim
        per_layer = (self.n_q * d + 2 * self.n_kv * d) * h + h * self.n_q * d \
            + 2 * self.ffn * h + h * self.ffn + 2 * h
        return 2 * (self.n_layers * per_layer + self.vocab * h + h)

    def kv_bytes_per_pos(self):
        return 2 * 2 * self.n_layers * self.n_kv * self.head_dim


TINY = ModelConfig("tiny", 2, 256, 4, 2, 64, 704, 4096)
M1P5B = ModelConfig("1.5b", 28, 1536, 12, 2, 128, 8960, 151936)
M7B = ModelConfig("7b", 28, 3584, 28, 4, 128, 18944, 152064)
# 7B-shaped decoder with two layers: small enough for profiler captures
M7B_2L = ModelConfig("7b-2l", 2, 3584, 28, 4, 128, 18944, 152064)
# a small drafter for the host cores (its own vocabulary: the producer's text
# is re-tokenised for the target)
CPU_DRAFT = ModelConfig("cpu-draft", 4, 512, 8, 2, 64, 1408, 8192)
MODELS = {m.name: m for m in (TINY, M1P5B, M7B, M7B_2L, CPU_DRAFT)}

# ---- stream ids ------------------------------------------------------------
S_EMBED, S_LM_HEAD, S_FINAL_NORM = 1, 2, 3
LAYER_KINDS = ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm",
               "w_gate", "w_up", "w_down")
GAINS = ("attn_norm", "mlp_norm")
S_ROOT = 0x20000000
S_INSTR = 0x20000001


def layer_stream(layer, kind):
    return 0x100 + 16 * layer + LAYER_KINDS.index(kind)


def kv_stream(layer, req, head, which):
    """which: 0 = keys, 1 = values."""
    return 0x40000000 | ((((layer * 1024 + req) * 64 + head) * 2 + which) & 0x3FFFFFFF)


def layer_shape(cfg, kind):
    h, d = cfg.hidden, cfg.head_dim
    return {
        "attn_norm": (h,), "mlp_norm": (h,),
        "w_q": (cfg.n_q * d, h), "w_k": (cfg.n_kv * d, h), "w_v": (cfg.n_kv * d, h),
        "w_o": (h, cfg.n_q * d),
        "w_gate": (cfg.ffn, h), "w_up": (cfg.ffn, h), "w_down": (h, cfg.ffn),
    }[kind]


@dataclass
class WeightSpec:
    name: str            # "embed", "lm_head", "final_norm" or "<kind>.<layer>"
    shape: tuple
    stream: int
    sigma: float
    base: float


def weight_specs(cfg, gains="unit", sigma=0.02, gain_sigma=0.1):
    """All tensors of a model.  gains="unit" gives RMSNorm gains of exactly 1.0
    (the workloads' reading); gains="random" draws 1 + N(0, gain_sigma);
    gains="sharp" keeps the layer gains at 1.0 and sets the final norm's gain
    to 8.0, which scales every logit by 8: the same arithmetic with greedy
    decisions separated by wider margins (the exactness tests use it)."""
    gs, gb = (0.0, 1.0) if gains in ("unit", "sharp") else (gain_sigma, 1.0)
    fb = 8.0 if gains == "sharp" else gb
    specs = [WeightSpec("embed", (cfg.vocab, cfg.hidden), S_EMBED, sigma, 0.0),
             WeightSpec("final_norm", (cfg.hidden,), S_FINAL_NORM, gs, fb),
             WeightSpec("lm_head", (cfg.vocab, cfg.hidden), S_LM_HEAD, sigma, 0.0)]
    for l in range(cfg.n_layers):
        for kind in LAYER_KINDS:
            if kind in GAINS:
                specs.append(WeightSpec(f"{kind}.{l}", layer_shape(cfg, kind),
                                        layer_stream(l, kind), gs, gb))
            else:
                specs.append(WeightSpec(f"{kind}.{l}", layer_shape(cfg, kind),
                                        layer_stream(l, kind), sigma, 0.0))
    return specs


def host_tensor(spec, seed):
    n = int(np.prod(spec.shape))
    if spec.sigma == 0.0:
        v = np.full(n, _bf16_bits(spec.base), dtype=np.uint16)
    else:
        v = synth.normal_bf16(n, seed, spec.stream, spec.sigma, spec.base)
    return v.reshape(spec.shape)


def _bf16_bits(x):
    u = np.array([x], dtype=np.float32).view(np.uint32)[0]
    u = (int(u) + 0x7FFF + ((int(u) >> 16) & 1)) >> 16
    return np.uint16(u & 0xFFFF)


def host_weights(cfg, seed=0, gains="unit"):
    """dict name -> uint16 array (bf16 bits) in logical layout."""
    return {s.name: host_tensor(s, seed) for s in weight_specs(cfg, gains)}


def host_kv_request(cfg, req, kv_len, capacity, seed=0, poison=True):
    """One request's prefilled cache: lists over layers of uint16 arrays
    [n_kv][capacity][head_dim].  Positions >= kv_len hold bf16 NaN when
    poison is set, so any read past the committed length shows up."""
    d = cfg.head_dim
    ks, vs = [], []
    for l in range(cfg.n_layers):
        pair = []
        for which in (0, 1):
            a = np.full((cfg.n_kv, capacity, d), NAN_BF16 if poison else 0,
                        dtype=np.uint16)
            for g in range(cfg.n_kv):
                a[g, :kv_len, :] = synth.normal_bf16(
                    kv_len * d, seed, kv_stream(l, req, g, which), 1.0).reshape(kv_len, d)
            pair.append(a)
        ks.append(pair[0])
        vs.append(pair[1])
    return ks, vs


def instruction_tokens(cfg, n, seed=0):
    """n instruction-suffix token ids, uniform over the vocabulary (the text
    that follows the retained audio positions in the prompt)."""
    return synth.uniform_int(n, seed, S_INSTR, cfg.vocab)


def root_tokens(cfg, batch, seed=0):
    return synth.uniform_int(batch, seed, S_ROOT, cfg.vocab)


# ---- candidate recipes -----------------------------------------------------

def replace_at(greedy_cont, pos, rng, vocab):
    """The greedy continuation with place `pos` replaced by a uniform token
    different from the greedy one (tiny workload: k = 4, place 2)."""
    c = np.array(greedy_cont, dtype=np.int32).copy()
    t = int(rng.integers(vocab))
    if t == c[pos]:
        t = (t + 1) % vocab
    c[pos] = t
    return c


def corrupt_each(greedy_cont, p, rng, vocab):
    """Each place independently replaced w.p. p by a uniform token != greedy."""
    c = np.array(greedy_cont, dtype=np.int32).copy()
    for i in range(len(c)):
        if rng.random() < p:
            t = int(rng.integers(vocab))
            if t == c[i]:
                t = (t + 1) % vocab
            c[i] = t
    return c


def geometric_plan(rng, k, vocab, q=0.75):
    """Accepted length ell with P(ell) = q^ell (1 - q), capped at k: places
    < ell follow the greedy continuation, place ell is corrupted, later places
    are uniform.  Returned as {ell, corrupt_token, tail[0..k-1]} int32."""
    ell = 0
    while ell < k and rng.random() < q:
        ell += 1
    plan = np.empty(k + 2, dtype=np.int32)
    plan[0] = ell
    plan[1] = rng.integers(vocab)
    plan[2:] = rng.integers(vocab, size=k)
    return plan


def apply_plan(greedy_cont, plan, vocab):
    """Host equivalent of the device candidate builder for one block."""
    k = len(plan) - 2
    ell = int(plan[0])
    c = np.empty(k, dtype=np.int32)
    for i in range(k):
        want = int(greedy_cont[i]) if i < len(greedy_cont) else -1
        if i < ell and want >= 0:
            c[i] = want
        elif i == ell:
            t = int(plan[1])
            c[i] = (t + 1) % vocab if t == want else t
        else:
            c[i] = int(plan[2 + i])
    return c


@dataclass
class Workload:
    name: str
    model: ModelConfig
    batch: int
    kv_len: list
    k: list
    recipe: str
    blocks: int = 1
    seed: int = 0
    notes: str = ""
    extra: dict = field(default_factory=dict)


def ragged_lengths(seed=0, batch=16):
    rng = np.random.default_rng(seed + 5)
    kv_len = rng.integers(250, 7501, size=batch).tolist()
    k = rng.integers(0, 17, size=batch).tolist()
    return kv_len, k


WORKLOADS = {
    "tiny": Workload("tiny", TINY, 1, [200], [4], "replace_at_2",
                     notes="150 audio + 50 instruction positions"),
    "1.5b": Workload("1.5b", M1P5B, 1, [814], [0, 1, 2, 4, 8], "corrupt_0.3",
                     notes="750 audio (30 s at 25 tok/s) + 64 instruction; k swept"),
    "7b": Workload("7b", M7B, 1, [1564], [8], "geometric_mean3", blocks=256,
                   notes="1500 audio (60 s) + 64 instruction; 256 consecutive blocks"),
    "7b-long": Workload("7b-long", M7B, 1, [15128], [1, 4, 8, 16], "geometric_mean3",
                        notes="15000 audio (10 min) + 128 instruction; k swept"),
    "7b-ragged": Workload("7b-ragged", M7B, 16, *ragged_lengths(), "corrupt_0.25",
                          blocks=128,
                          notes="16 requests, L ~ U[250, 7500], k ~ U{0..16}"),
}
