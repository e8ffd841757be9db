"""ctypes binding of the CPU oracle (oracle.c).

TEST INFRASTRUCTURE: only the tests, __graft_entry__.smoke() and bench.py's
CPU-baseline / reference legs may import this package.  The product path
(paper_2609_37617_gb300) never imports it.
"""
import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
_LIBS = {}

_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_D = ctypes.c_double


class _Config(ctypes.Structure):
    _fields_ = [("n_layers", _I32), ("hidden", _I32), ("n_q", _I32),
                ("n_kv", _I32), ("head_dim", _I32), ("ffn", _I32),
                ("vocab", _I32), ("rope_theta", _D), ("rms_eps", _D)]


class _Weights(ctypes.Structure):
    _fields_ = [(n, _P) for n in ("embed", "final_norm", "lm_head", "attn_norm",
                                  "w_q", "w_k", "w_v", "w_o", "mlp_norm",
                                  "w_gate", "w_up", "w_down")]


class _KV(ctypes.Structure):
    _fields_ = [("k", _P), ("v", _P), ("capacity", _I64)]


def load(precision="f64"):
    """The oracle library: 'f64' (default) or 'f32' (self-check build)."""
    if precision not in _LIBS:
        name = {"f64": "liboracle.so", "f32": "liboracle_f32.so"}[precision]
        path = os.path.join(HERE, name)
        if not os.path.exists(path):
            from . import build as _b
            _b.build()
        lib = ctypes.CDLL(path)
        lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.oracle_bf16_to_double.restype = _D
        lib.oracle_double_to_bf16.argtypes = [_D]
        lib.oracle_double_to_bf16.restype = ctypes.c_uint16
        lib.oracle_rmsnorm.argtypes = [_I32, _P, _P, _D, _P]
        lib.oracle_linear.argtypes = [_I32, _I32, _P, _P, _P]
        lib.oracle_rope.argtypes = [_I32, _P, _I64, _D]
        lib.oracle_attend.argtypes = [_I32, _I64, _P, _P, _P, _P]
        lib.oracle_silu.argtypes = [_D]
        lib.oracle_silu.restype = _D
        lib.oracle_argmax.argtypes = [_I32, _P, _P]
        lib.oracle_argmax.restype = _I32
        lib.oracle_accept.argtypes = [_I32, _P, _P, _P, _P]
        lib.oracle_decode_step.argtypes = [_P, _P, _P, _I64, _I32, _P]
        lib.oracle_decode_step.restype = _I32
        lib.oracle_verify_block.argtypes = [_P, _P, _P, _I64, _I32, _I32, _P,
                                            _P, _P, _P, _P, _P, _P, _P]
        lib.oracle_verify_block.restype = _I32
        lib.oracle_real_bytes.restype = _I32
        lib.oracle_set_threads.argtypes = [_I32]
        lib.oracle_set_threads.restype = _I32
        _LIBS[precision] = lib
    return _LIBS[precision]


def set_threads(n, precision="f64"):
    """Threads of the oracle's OpenMP loops (n <= 0: the default); returns
    the count in effect.  The thread count changes no result."""
    return int(load(precision).oracle_set_threads(int(n)))


def _ptr(a):
    return ctypes.c_void_p(a.ctypes.data)


def _f64(x):
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


# ---- sub-steps -------------------------------------------------------------

def bf16_to_double(bits, precision="f64"):
    return load(precision).oracle_bf16_to_double(int(bits))


def double_to_bf16(x, precision="f64"):
    return int(load(precision).oracle_double_to_bf16(float(x)))


def rmsnorm(x, gain_bits, eps, precision="f64"):
    x = _f64(x)
    g = np.ascontiguousarray(gain_bits, dtype=np.uint16)
    y = np.empty_like(x)
    load(precision).oracle_rmsnorm(len(x), _ptr(x), _ptr(g), float(eps), _ptr(y))
    return y


def linear(w_bits, x, precision="f64"):
    w = np.ascontiguousarray(w_bits, dtype=np.uint16)
    x = _f64(x)
    y = np.empty(w.shape[0], dtype=np.float64)
    load(precision).oracle_linear(w.shape[0], w.shape[1], _ptr(w), _ptr(x), _ptr(y))
    return y


def rope(v, pos, theta, precision="f64"):
    v = _f64(v).copy()
    load(precision).oracle_rope(len(v), _ptr(v), int(pos), float(theta))
    return v


def attend(q, k_bits, v_bits, precision="f64"):
    q = _f64(q)
    k = np.ascontiguousarray(k_bits, dtype=np.uint16)
    v = np.ascontiguousarray(v_bits, dtype=np.uint16)
    out = np.empty(len(q), dtype=np.float64)
    load(precision).oracle_attend(len(q), k.shape[0], _ptr(q), _ptr(k), _ptr(v), _ptr(out))
    return out


def silu(x, precision="f64"):
    return load(precision).oracle_silu(float(x))


def argmax(x, precision="f64"):
    x = _f64(x)
    m = np.zeros(1, dtype=np.float64)
    i = load(precision).oracle_argmax(len(x), _ptr(x), _ptr(m))
    return int(i), float(m[0])


def accept(cand, greedy, precision="f64"):
    cand = np.ascontiguousarray(cand, dtype=np.int32)
    greedy = np.ascontiguousarray(greedy, dtype=np.int32)
    assert len(greedy) == len(cand) + 1
    n = np.zeros(1, dtype=np.int32)
    c = np.zeros(1, dtype=np.int32)
    load(precision).oracle_accept(len(cand), _ptr(cand), _ptr(greedy), _ptr(n), _ptr(c))
    return int(n[0]), int(c[0])


# ---- model -----------------------------------------------------------------

class Model:
    """The oracle's view of a model: host bf16 weights in logical layout
    (dict name -> uint16 array, names as synth.workloads.weight_specs)."""

    def __init__(self, cfg, weights, precision="f64"):
        self.cfg = cfg
        self.lib = load(precision)
        self._keep = []
        c = _Config(cfg.n_layers, cfg.hidden, cfg.n_q, cfg.n_kv, cfg.head_dim,
                    cfg.ffn, cfg.vocab, float(cfg.rope_theta), float(cfg.rms_eps))
        self._cfg = c
        w = _Weights()
        for name in ("embed", "final_norm", "lm_head"):
            a = np.ascontiguousarray(weights[name], dtype=np.uint16)
            self._keep.append(a)
            setattr(w, name, a.ctypes.data)
        for kind in ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm",
                     "w_gate", "w_up", "w_down"):
            arrs = [np.ascontiguousarray(weights[f"{kind}.{l}"], dtype=np.uint16)
                    for l in range(cfg.n_layers)]
            self._keep.extend(arrs)
            ptrs = (ctypes.c_void_p * cfg.n_layers)(*[a.ctypes.data for a in arrs])
            self._keep.append(ptrs)
            setattr(w, kind, ctypes.cast(ptrs, ctypes.c_void_p).value)
        self._w = w

    def cache(self, k_layers, v_layers):
        """Wrap one request's cache (lists over layers of uint16 arrays
        [n_kv][capacity][d], modified in place by the oracle)."""
        return Cache(self, k_layers, v_layers)

    def decode_step(self, cache, pos, token):
        logits = np.empty(self.cfg.vocab, dtype=np.float64)
        rc = self.lib.oracle_decode_step(ctypes.byref(self._cfg), ctypes.byref(self._w),
                                         ctypes.byref(cache._kv), int(pos), int(token),
                                         _ptr(logits))
        if rc != 0:
            raise ValueError("oracle_decode_step rejected its arguments")
        return logits

    def verify_block(self, cache, length, root, cand, want_logits=True):
        cand = np.ascontiguousarray(cand, dtype=np.int32)
        k = len(cand)
        V = self.cfg.vocab
        n = np.zeros(1, np.int32)
        corr = np.zeros(1, np.int32)
        greedy = np.zeros(k + 1, np.int32)
        logits = np.empty((k + 1, V), np.float64) if want_logits else None
        margin = np.zeros(k + 1, np.float64)
        new_len = np.zeros(1, np.int64)
        new_root = np.zeros(1, np.int32)
        rc = self.lib.oracle_verify_block(
            ctypes.byref(self._cfg), ctypes.byref(self._w), ctypes.byref(cache._kv),
            int(length), int(root), k, _ptr(cand) if k else None, _ptr(n), _ptr(corr),
            _ptr(greedy), _ptr(logits) if want_logits else None, _ptr(margin),
            _ptr(new_len), _ptr(new_root))
        if rc != 0:
            raise ValueError("oracle_verify_block rejected its arguments")
        return dict(n_accepted=int(n[0]), correction=int(corr[0]), greedy=greedy,
                    logits=logits, margin=margin, new_len=int(new_len[0]),
                    new_root=int(new_root[0]))


class Cache:
    def __init__(self, model, k_layers, v_layers):
        self.k = [np.ascontiguousarray(a, dtype=np.uint16) for a in k_layers]
        self.v = [np.ascontiguousarray(a, dtype=np.uint16) for a in v_layers]
        L = model.cfg.n_layers
        self._kp = (ctypes.c_void_p * L)(*[a.ctypes.data for a in self.k])
        self._vp = (ctypes.c_void_p * L)(*[a.ctypes.data for a in self.v])
        self._kv = _KV(ctypes.cast(self._kp, ctypes.c_void_p).value,
                       ctypes.cast(self._vp, ctypes.c_void_p).value,
                       int(self.k[0].shape[1]))

    def copy(self, model):
        return Cache(model, [a.copy() for a in self.k], [a.copy() for a in self.v])


def greedy_continuation(model, cache, length, root, n):
    """The target's own greedy tokens after `root` (n of them), by n+1 decode
    steps on a copy of the cache (Eq. 3); returns (tokens[n], margins[n+1])."""
    c = cache.copy(model)
    toks, margins = [], []
    tok = int(root)
    for i in range(n + 1):
        logits = model.decode_step(c, length + i, tok)
        tok, m = argmax(logits)
        margins.append(m)
        toks.append(tok)
    return np.array(toks[:n], dtype=np.int32), np.array(margins)


def prefill(model, cache, length, tokens):
    """Instruction-suffix prefill (App. A.1): the tokens forwarded one greedy
    decode step at a time after the `length` retained positions (Eq. 3), their
    keys and values appended to `cache` in place.  Returns (the first token of
    the response -- the greedy token after the last one --, its margin, the
    last row's logits)."""
    logits = None
    for i, t in enumerate(tokens):
        logits = model.decode_step(cache, length + i, int(t))
    tok, m = argmax(logits)
    return tok, m, logits

