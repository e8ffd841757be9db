"""Python binding of libas2d.so, the GB300 (sm_103a) target-side block
verification library (C-ABI: include/as2d.h).

The functions below carry the C names and only marshal arguments: every step
of the verification pass runs in the library's CUDA kernels.  PyTorch is used
by callers for device memory and streams only.  Importing this package fails
loudly if libas2d.so has not been built: there is no fallback path.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libas2d.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
        "(or python paper_2609_37617_gb300/build.py). There is no CPU fallback.")

_lib = ctypes.CDLL(LIB_PATH)

AS2D_OK = 0
AS2D_ERR_INVALID_ARG = -1
AS2D_ERR_CAPACITY = -2
AS2D_ERR_CUDA = -3
AS2D_ERR_UNSUPPORTED = -4
AS2D_ERR_DEVICE = -5
AS2D_ERR_NO_MEMORY = -6
AS2D_DEVERR_BAD_TOKEN = 1
AS2D_DEVERR_ROLLBACK = 2
AS2D_DEVERR_TIMEOUT = 4
AS2D_DEVERR_CAPACITY = 8
AS2D_CBUF_BATCH = 8
CBUF_MODES = {0: "normal", 1: "realign", 2: "alone"}
AS2D_MAX_K = 16
AS2D_MAX_BATCH = 64

EXPORTED = ("as2d_model_load", "as2d_kv_init_prefilled", "as2d_verify_block",
            "as2d_decode_step", "as2d_kv_rollback", "as2d_kv_read_state",
            "as2d_kv_device_state", "as2d_kv_check", "as2d_kv_free",
            "as2d_model_free", "as2d_last_error", "as2d_kv_profile",
            "as2d_kv_profile_read", "as2d_decode_step_static", "as2d_kv_set_wait_limit",
            "as2d_cbuf_create", "as2d_cbuf_publish", "as2d_cbuf_candidates", "as2d_cbuf_after_call",
            "as2d_cbuf_state", "as2d_cbuf_source_of", "as2d_cbuf_free", "as2d_cbuf_held",
            "as2d_verify_from_buffers", "as2d_interval_accounting", "as2d_session_run",
            "as2d_budget_select", "as2d_prefill", "as2d_model_set_sm_budget",
            "as2d_cpu_decoder_create", "as2d_cpu_decoder_step", "as2d_cpu_decoder_logits",
            "as2d_cpu_decoder_reset", "as2d_cpu_decoder_free")
KERNEL_CLASSES = {"qkv": 0, "attention": 1, "o": 2, "gate_up": 3, "down": 4,
                  "lm_head": 5, "other": 6}


class as2d_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rope_theta", ctypes.c_float),
                ("rms_eps", ctypes.c_float)]


class as2d_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "embed", "final_norm", "lm_head", "attn_norm", "w_q", "w_k", "w_v",
        "w_o", "mlp_norm", "w_gate", "w_up", "w_down")]


class as2d_verify_out(ctypes.Structure):
    _fields_ = [("n_accepted", ctypes.c_void_p), ("correction_token", ctypes.c_void_p),
                ("greedy", ctypes.c_void_p), ("logits", ctypes.c_void_p)]


class as2d_source_record(ctypes.Structure):
    _fields_ = [("request", ctypes.c_int32), ("source", ctypes.c_int32),
                ("producer", ctypes.c_int32), ("offset", ctypes.c_int32),
                ("time", ctypes.c_double), ("confidence", ctypes.c_float),
                ("has_confidence", ctypes.c_int32)]


class as2d_session_spec(ctypes.Structure):
    _fields_ = [("target", ctypes.c_void_p), ("drafter", ctypes.c_void_p),
                ("buf", ctypes.c_void_p), ("script", ctypes.c_void_p),
                ("n_script", ctypes.c_int32), ("b", ctypes.c_int32),
                ("publish_every", ctypes.c_int32), ("n_commit", ctypes.c_int32),
                ("overlapped", ctypes.c_int32), ("target_stream", ctypes.c_void_p),
                ("drafter_stream", ctypes.c_void_p), ("cpu_drafter", ctypes.c_void_p)]


class as2d_session_stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_double) for n in ("T", "D", "V", "O", "H")] + \
               [(n, ctypes.c_int32) for n in ("rounds", "alone_rounds", "committed", "accepted",
                                              "producer_steps", "published")]


_P = ctypes.c_void_p
_S = ctypes.c_int32
_lib.as2d_model_load.argtypes = [ctypes.POINTER(as2d_config), ctypes.POINTER(as2d_weights),
                                 ctypes.POINTER(ctypes.c_void_p)]
_lib.as2d_model_load.restype = _S
_lib.as2d_kv_init_prefilled.argtypes = [_P, ctypes.c_int32, _P, ctypes.c_int32, _P, _P, _P,
                                        ctypes.POINTER(ctypes.c_void_p)]
_lib.as2d_kv_init_prefilled.restype = _S
_lib.as2d_verify_block.argtypes = [_P, _P, _P, ctypes.POINTER(as2d_verify_out), _P]
_lib.as2d_verify_block.restype = _S
_lib.as2d_decode_step.argtypes = [_P, ctypes.POINTER(as2d_verify_out), _P]
_lib.as2d_decode_step.restype = _S
_lib.as2d_kv_rollback.argtypes = [_P, _P, _P, _P]
_lib.as2d_kv_rollback.restype = _S
_lib.as2d_kv_read_state.argtypes = [_P, _P, _P, _P]
_lib.as2d_kv_read_state.restype = _S
_lib.as2d_kv_device_state.argtypes = [_P, ctypes.POINTER(ctypes.c_void_p),
                                      ctypes.POINTER(ctypes.c_void_p)]
_lib.as2d_kv_device_state.restype = _S
_lib.as2d_kv_check.argtypes = [_P, _P]
_lib.as2d_kv_check.restype = _S
_lib.as2d_kv_free.argtypes = [_P]
_lib.as2d_kv_free.restype = None
_lib.as2d_model_free.argtypes = [_P]
_lib.as2d_model_free.restype = None
_lib.as2d_kv_profile.argtypes = [_P, ctypes.c_int32]
_lib.as2d_kv_profile.restype = _S
_lib.as2d_kv_profile_read.argtypes = [_P, ctypes.POINTER(ctypes.c_int32),
                                      ctypes.POINTER(ctypes.c_double),
                                      ctypes.POINTER(ctypes.c_int64)]
_lib.as2d_kv_profile_read.restype = _S
_lib.as2d_decode_step_static.argtypes = [_P, _P, _P, ctypes.c_int32, _P, _P, _P, _P, _P, _P]
_lib.as2d_kv_set_wait_limit.argtypes = [_P, ctypes.c_uint64]
_lib.as2d_kv_set_wait_limit.restype = _S
_lib.as2d_decode_step_static.restype = _S
_lib.as2d_cbuf_create.argtypes = [_S, ctypes.POINTER(ctypes.c_void_p)]
_lib.as2d_cbuf_publish.argtypes = [_P, _P, _S, ctypes.POINTER(as2d_source_record)]
_lib.as2d_cbuf_candidates.argtypes = [_P, _S, _P, ctypes.POINTER(ctypes.c_int32)]
_lib.as2d_cbuf_after_call.argtypes = [_P, _S, _S, _S]
_lib.as2d_cbuf_state.argtypes = [_P, _P, _P, _P]
_lib.as2d_cbuf_source_of.argtypes = [_P, _S, ctypes.POINTER(as2d_source_record)]
_lib.as2d_cbuf_held.argtypes = [_P, _P, _P]
_lib.as2d_cbuf_held.restype = _S
_lib.as2d_cbuf_free.argtypes = [_P]
_lib.as2d_cbuf_free.restype = None
_lib.as2d_verify_from_buffers.argtypes = [_P, _P, _S, _P, _P, _P, _P]
for _n in ("as2d_cbuf_create", "as2d_cbuf_publish", "as2d_cbuf_candidates",
           "as2d_cbuf_after_call", "as2d_cbuf_state", "as2d_cbuf_source_of",
           "as2d_verify_from_buffers"):
    getattr(_lib, _n).restype = _S
_lib.as2d_interval_accounting.argtypes = [_P, _S, _P, _S, ctypes.c_double, _P]
_lib.as2d_interval_accounting.restype = _S
_lib.as2d_session_run.argtypes = [ctypes.POINTER(as2d_session_spec), _P,
                                  ctypes.POINTER(as2d_session_stats)]
_lib.as2d_session_run.restype = _S
_lib.as2d_budget_select.argtypes = [_P, _P, _P, _P, _P, _S, _S, _S, _S, _P, _P, _P]
_lib.as2d_budget_select.restype = _S
_lib.as2d_model_set_sm_budget.argtypes = [_P, _S]
_lib.as2d_model_set_sm_budget.restype = _S
_lib.as2d_prefill.argtypes = [_P, _P, _S, _P, _P]
_lib.as2d_prefill.restype = _S
_lib.as2d_cpu_decoder_create.argtypes = [ctypes.POINTER(as2d_config), ctypes.POINTER(as2d_weights),
                                         _S, _S, _S, ctypes.POINTER(ctypes.c_void_p)]
_lib.as2d_cpu_decoder_step.argtypes = [_P, ctypes.POINTER(ctypes.c_int32)]
_lib.as2d_cpu_decoder_logits.argtypes = [_P, _P]
_lib.as2d_cpu_decoder_reset.argtypes = [_P, _S, _S]
_lib.as2d_cpu_decoder_free.argtypes = [_P]
_lib.as2d_cpu_decoder_free.restype = None
for _n in ("as2d_cpu_decoder_create", "as2d_cpu_decoder_step", "as2d_cpu_decoder_logits",
           "as2d_cpu_decoder_reset"):
    getattr(_lib, _n).restype = _S
_lib.as2d_last_error.argtypes = []
_lib.as2d_last_error.restype = ctypes.c_char_p


class AS2DError(RuntimeError):
    def __init__(self, status, where):
        msg = _lib.as2d_last_error().decode(errors="replace")
        super().__init__(f"{where} returned {status}: {msg}")
        self.status = status


def _check(status, where):
    if status != AS2D_OK:
        raise AS2DError(status, where)
    return status


def _i32_array(values):
    arr = (ctypes.c_int32 * len(values))(*[int(v) for v in values])
    return arr


# ---- the C entry points, one wrapper each -------------------------------------

def as2d_last_error():
    return _lib.as2d_last_error().decode(errors="replace")


def as2d_model_load(cfg, weights_ptrs, n_layers):
    """cfg: as2d_config; weights_ptrs: dict name -> device pointer (int) for
    embed/final_norm/lm_head and name -> list of n_layers pointers for the
    per-layer tensors.  Returns (status, model handle)."""
    keep = []
    w = as2d_weights()
    for name in ("embed", "final_norm", "lm_head"):
        setattr(w, name, int(weights_ptrs[name]))
    for name in ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm", "w_gate",
                 "w_up", "w_down"):
        arr = (ctypes.c_void_p * n_layers)(*[int(p) for p in weights_ptrs[name]])
        keep.append(arr)
        setattr(w, name, ctypes.cast(arr, ctypes.c_void_p).value)
    out = ctypes.c_void_p()
    st = _lib.as2d_model_load(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(out))
    return st, out.value


def as2d_kv_init_prefilled(model, batch, kv_len, capacity, k_cache_ptr, v_cache_ptr,
                           root_tokens):
    out = ctypes.c_void_p()
    st = _lib.as2d_kv_init_prefilled(_P(model), int(batch), _i32_array(kv_len),
                                     int(capacity), _P(int(k_cache_ptr)),
                                     _P(int(v_cache_ptr)), _i32_array(root_tokens),
                                     ctypes.byref(out))
    return st, out.value


def make_verify_out(n_accepted_ptr, correction_ptr, greedy_ptr=0, logits_ptr=0):
    return as2d_verify_out(int(n_accepted_ptr) or None, int(correction_ptr) or None,
                           int(greedy_ptr) or None, int(logits_ptr) or None)


def as2d_verify_block(kv, candidates_ptr, k, out, stream=0):
    return _lib.as2d_verify_block(_P(kv), _P(int(candidates_ptr) or None), _i32_array(k),
                                  ctypes.byref(out), _P(int(stream) or None))


def as2d_decode_step(kv, out, stream=0):
    return _lib.as2d_decode_step(_P(kv), ctypes.byref(out), _P(int(stream) or None))


def as2d_kv_rollback(kv, new_len, new_root, stream=0):
    return _lib.as2d_kv_rollback(_P(kv), _i32_array(new_len), _i32_array(new_root),
                                 _P(int(stream) or None))


def as2d_kv_read_state(kv, batch, stream=0):
    ln = (ctypes.c_int32 * batch)()
    rt = (ctypes.c_int32 * batch)()
    st = _lib.as2d_kv_read_state(_P(kv), ln, rt, _P(int(stream) or None))
    return st, list(ln), list(rt)


def as2d_kv_device_state(kv):
    ln = ctypes.c_void_p()
    rt = ctypes.c_void_p()
    st = _lib.as2d_kv_device_state(_P(kv), ctypes.byref(ln), ctypes.byref(rt))
    return st, ln.value, rt.value


def as2d_kv_check(kv, stream=0):
    return _lib.as2d_kv_check(_P(kv), _P(int(stream) or None))


def as2d_kv_free(kv):
    _lib.as2d_kv_free(_P(kv))


def as2d_model_free(model):
    _lib.as2d_model_free(_P(model))


def as2d_kv_profile(kv, kernel_class):
    return _lib.as2d_kv_profile(_P(kv), int(kernel_class))


def as2d_kv_profile_read(kv):
    n = ctypes.c_int32()
    ms = ctypes.c_double()
    alln = ctypes.c_int64()
    st = _lib.as2d_kv_profile_read(_P(kv), ctypes.byref(n), ctypes.byref(ms), ctypes.byref(alln))
    return st, n.value, ms.value, alln.value


def as2d_decode_step_static(model, k_cache_ptr, v_cache_ptr, capacity, len_ptr, root_ptr,
                            correction_ptr, logits_ptr=0, error_bits_ptr=0, stream=0):
    """Single-request decode step whose working memory is the library's fixed
    array (no allocation); see include/as2d.h."""
    return _lib.as2d_decode_step_static(_P(model), _P(int(k_cache_ptr)), _P(int(v_cache_ptr)),
                                        int(capacity), _P(int(len_ptr)), _P(int(root_ptr)),
                                        _P(int(correction_ptr)), _P(int(logits_ptr) or None),
                                        _P(int(error_bits_ptr) or None),
                                        _P(int(stream) or None))


def as2d_cbuf_create(window):
    h = ctypes.c_void_p()
    st = _lib.as2d_cbuf_create(window, ctypes.byref(h))
    return st, h.value


def as2d_cbuf_publish(buf, tokens, record):
    arr = _i32_array(tokens) if len(tokens) else None
    return _lib.as2d_cbuf_publish(buf, arr, len(tokens),
                                  ctypes.byref(record) if record is not None else None)


def as2d_cbuf_candidates(buf, b):
    arr = (ctypes.c_int32 * max(b, 1))()
    k = ctypes.c_int32(-1)
    st = _lib.as2d_cbuf_candidates(buf, b, arr, ctypes.byref(k))
    return st, list(arr[:max(k.value, 0)])


def as2d_cbuf_after_call(buf, k, n_accepted, correction):
    return _lib.as2d_cbuf_after_call(buf, k, n_accepted, correction)


def as2d_cbuf_state(buf):
    r, c, m = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    st = _lib.as2d_cbuf_state(buf, ctypes.byref(r), ctypes.byref(c), ctypes.byref(m))
    return st, r.value, c.value, m.value


def as2d_cbuf_source_of(buf, position):
    rec = as2d_source_record()
    st = _lib.as2d_cbuf_source_of(buf, position, ctypes.byref(rec))
    return st, rec


def as2d_cbuf_free(buf):
    _lib.as2d_cbuf_free(buf)


def as2d_verify_from_buffers(kv, bufs, b, batch, stream=0):
    """Returns (status, k_used, committed lists)."""
    hb = (ctypes.c_void_p * batch)(*bufs)
    k_used = (ctypes.c_int32 * batch)()
    comm = (ctypes.c_int32 * (batch * (b + 1)))()
    ncomm = (ctypes.c_int32 * batch)()
    st = _lib.as2d_verify_from_buffers(kv, hb, b, k_used, comm, ncomm, stream)
    rows = [list(comm[r * (b + 1): r * (b + 1) + ncomm[r]]) for r in range(batch)]
    return st, list(k_used), rows


def as2d_interval_accounting(p, v, T):
    """p, v: lists of (start, end).  Returns (status, [D, V, O, H, T])."""
    pa = (ctypes.c_double * max(2 * len(p), 1))(*[x for iv in p for x in iv])
    va = (ctypes.c_double * max(2 * len(v), 1))(*[x for iv in v for x in iv])
    out = (ctypes.c_double * 5)()
    st = _lib.as2d_interval_accounting(pa, len(p), va, len(v), T, out)
    return st, list(out)


def as2d_session_run(spec, n_commit, b):
    """Returns (status, committed list, stats dict)."""
    comm = (ctypes.c_int32 * (n_commit + AS2D_MAX_K + 1))()
    stats = as2d_session_stats()
    st = _lib.as2d_session_run(ctypes.byref(spec), comm, ctypes.byref(stats))
    d = {n: getattr(stats, n) for n, _ in as2d_session_stats._fields_}
    return st, list(comm[:max(stats.committed, 0)]), d


class CpuDecoder:
    """Owns an as2d_cpu_decoder built from host fp32 weights: `host` maps the
    names of as2d_weights to float32 numpy arrays (per-layer names to lists)."""

    def __init__(self, shape, host, capacity, threads, root):
        import numpy as np
        self._keep = {k: ([np.ascontiguousarray(a, dtype=np.float32) for a in v]
                          if isinstance(v, list) else np.ascontiguousarray(v, dtype=np.float32))
                      for k, v in host.items()}
        w = as2d_weights()
        for name in ("embed", "final_norm", "lm_head"):
            setattr(w, name, self._keep[name].ctypes.data)
        self._arrs = []
        for name in ("attn_norm", "w_q", "w_k", "w_v", "w_o", "mlp_norm", "w_gate", "w_up",
                     "w_down"):
            arr = (ctypes.c_void_p * shape.n_layers)(*[a.ctypes.data for a in self._keep[name]])
            self._arrs.append(arr)
            setattr(w, name, ctypes.cast(arr, ctypes.c_void_p))
        cfg = as2d_config(shape.n_layers, shape.hidden, shape.n_q, shape.n_kv, shape.head_dim,
                          shape.ffn, shape.vocab, float(shape.rope_theta), float(shape.rms_eps))
        h = ctypes.c_void_p()
        _check(_lib.as2d_cpu_decoder_create(ctypes.byref(cfg), ctypes.byref(w), capacity, threads,
                                            root, ctypes.byref(h)), "as2d_cpu_decoder_create")
        self.handle = h.value
        self.vocab = shape.vocab
        self._keep = None  # copied by the library

    def step(self):
        t = ctypes.c_int32()
        _check(_lib.as2d_cpu_decoder_step(self.handle, ctypes.byref(t)), "as2d_cpu_decoder_step")
        return t.value

    def logits(self):
        import numpy as np
        out = np.empty(self.vocab, dtype=np.float32)
        _check(_lib.as2d_cpu_decoder_logits(self.handle, out.ctypes.data),
               "as2d_cpu_decoder_logits")
        return out

    def reset(self, length, root):
        _check(_lib.as2d_cpu_decoder_reset(self.handle, length, root), "as2d_cpu_decoder_reset")

    def close(self):
        if self.handle:
            _lib.as2d_cpu_decoder_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def session_run(target, drafter, buf, script, b, n_commit, overlapped, publish_every=8,
                target_stream=0, drafter_stream=0, cpu_drafter=None):
    """Run a producer/verifier session (as2d_session_run) on State objects and
    a CandidateBuffer; returns (committed tokens, stats dict)."""
    arr = _i32_array(script) if len(script) else None
    spec = as2d_session_spec(target.handle, drafter.handle if drafter is not None else None,
                             buf.handle, ctypes.cast(arr, ctypes.c_void_p) if arr else None,
                             len(script), b, publish_every, n_commit, int(bool(overlapped)),
                             target_stream, drafter_stream,
                             cpu_drafter.handle if cpu_drafter is not None else None)
    st, comm, stats = as2d_session_run(spec, n_commit, b)
    _check(st, "as2d_session_run")
    return comm, stats


def as2d_budget_select(cost_us, traces, n_commit, window, b_max):
    """cost_us: AS2D_MAX_K + 1 mean call times by k; traces: list of
    (reference text, producer text).  Returns (status, best b, tok/s per b,
    calls per b)."""
    cost = (ctypes.c_double * (AS2D_MAX_K + 1))(*[float(c) for c in cost_us])
    refs = [int(t) for r, _ in traces for t in r]
    prods = [int(t) for _, p in traces for t in p]
    ra = _i32_array(refs or [0])
    pa = _i32_array(prods or [0])
    rl = _i32_array([len(r) for r, _ in traces] or [0])
    pl = _i32_array([len(p) for _, p in traces] or [0])
    tok_s = (ctypes.c_double * (max(b_max, 0) + 1))()
    calls = (ctypes.c_int32 * (max(b_max, 0) + 1))()
    best = ctypes.c_int32(-1)
    st = _lib.as2d_budget_select(cost, ra, rl, pa, pl, len(traces), n_commit, window, b_max,
                                 tok_s, calls, ctypes.byref(best))
    return st, best.value, list(tok_s), list(calls)


def exported_symbols():
    """Names of include/as2d.h's entry points that the loaded library exports."""
    return [n for n in EXPORTED if hasattr(_lib, n)]


# ---- thin owners of the handles (marshalling only) ---------------------------

class Model:
    """Owns an as2d_model.  `shape` has the fields of as2d_config
    (n_layers, hidden, n_q, n_kv, head_dim, ffn, vocab, rope_theta, rms_eps);
    `pointers` maps weight names to device pointers (see as2d_model_load)."""

    def __init__(self, shape, pointers):
        self.shape = shape
        self.cfg = as2d_config(shape.n_layers, shape.hidden, shape.n_q, shape.n_kv,
                               shape.head_dim, shape.ffn, shape.vocab,
                               float(shape.rope_theta), float(shape.rms_eps))
        st, h = as2d_model_load(self.cfg, pointers, shape.n_layers)
        _check(st, "as2d_model_load")
        self.handle = h

    def set_sm_budget(self, n_sms):
        _check(_lib.as2d_model_set_sm_budget(self.handle, int(n_sms)), "as2d_model_set_sm_budget")

    def close(self):
        if self.handle:
            as2d_model_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class CandidateBuffer:
    """Owns an as2d_cbuf: one request's published candidates, read cursor and
    alignment state (host side)."""

    def __init__(self, window=8):
        st, h = as2d_cbuf_create(window)
        _check(st, "as2d_cbuf_create")
        self.handle = h

    def publish(self, tokens, request=0, source=0, producer=0, offset=0, time=0.0,
                confidence=None):
        rec = as2d_source_record(request, source, producer, offset, time,
                                 0.0 if confidence is None else confidence,
                                 0 if confidence is None else 1)
        _check(as2d_cbuf_publish(self.handle, list(tokens), rec), "as2d_cbuf_publish")

    def candidates(self, b):
        st, toks = as2d_cbuf_candidates(self.handle, b)
        _check(st, "as2d_cbuf_candidates")
        return toks

    def after_call(self, k, n_accepted, correction):
        _check(as2d_cbuf_after_call(self.handle, k, n_accepted, correction),
               "as2d_cbuf_after_call")

    def state(self):
        st, ready, cursor, mode = as2d_cbuf_state(self.handle)
        _check(st, "as2d_cbuf_state")
        return ready, cursor, CBUF_MODES[mode]

    def held(self):
        """(tokens, batch records) the buffer still holds."""
        t, r = ctypes.c_int32(), ctypes.c_int32()
        _check(_lib.as2d_cbuf_held(self.handle, ctypes.byref(t), ctypes.byref(r)), "as2d_cbuf_held")
        return t.value, r.value

    def source_of(self, position):
        st, rec = as2d_cbuf_source_of(self.handle, position)
        _check(st, "as2d_cbuf_source_of")
        return {"request": rec.request, "source": rec.source, "producer": rec.producer,
                "offset": rec.offset, "time": rec.time,
                "confidence": rec.confidence if rec.has_confidence else None}

    def close(self):
        if self.handle:
            as2d_cbuf_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class State:
    """Owns an as2d_kv bound to caller caches (torch tensors kept alive here)."""

    def __init__(self, model, kv_len, capacity, k_cache, v_cache, roots):
        self.model = model
        self.batch = len(kv_len)
        self._caches = (k_cache, v_cache)
        st, h = as2d_kv_init_prefilled(model.handle, self.batch, kv_len, capacity,
                                       k_cache.data_ptr(), v_cache.data_ptr(), roots)
        _check(st, "as2d_kv_init_prefilled")
        self.handle = h

    def verify(self, candidates, k, n_accepted, correction, greedy=None, logits=None,
               stream=0):
        out = make_verify_out(n_accepted.data_ptr(), correction.data_ptr(),
                              greedy.data_ptr() if greedy is not None else 0,
                              logits.data_ptr() if logits is not None else 0)
        cptr = candidates.data_ptr() if candidates is not None and candidates.numel() else 0
        _check(as2d_verify_block(self.handle, cptr, k, out, stream), "as2d_verify_block")

    def decode(self, n_accepted, correction, greedy=None, logits=None, stream=0):
        out = make_verify_out(n_accepted.data_ptr(), correction.data_ptr(),
                              greedy.data_ptr() if greedy is not None else 0,
                              logits.data_ptr() if logits is not None else 0)
        _check(as2d_decode_step(self.handle, out, stream), "as2d_decode_step")

    def verify_from_buffers(self, bufs, b, stream=0):
        """One verification call with candidates from CandidateBuffer objects
        (one per request); returns (k_used, committed token lists)."""
        st, k_used, rows = as2d_verify_from_buffers(
            self.handle, [x.handle for x in bufs], b, self.batch, stream)
        _check(st, "as2d_verify_from_buffers")
        return k_used, rows

    def prefill(self, tokens, first_token=None, stream=0):
        """as2d_prefill: tokens and first_token are device int32 tensors."""
        _check(_lib.as2d_prefill(self.handle, tokens.data_ptr(), tokens.numel(),
                                 first_token.data_ptr() if first_token is not None else None,
                                 stream), "as2d_prefill")

    def rollback(self, new_len, new_root, stream=0):
        _check(as2d_kv_rollback(self.handle, new_len, new_root, stream), "as2d_kv_rollback")

    def read_state(self, stream=0):
        st, ln, rt = as2d_kv_read_state(self.handle, self.batch, stream)
        _check(st, "as2d_kv_read_state")
        return ln, rt

    def device_state(self):
        st, ln, rt = as2d_kv_device_state(self.handle)
        _check(st, "as2d_kv_device_state")
        return ln, rt

    def profile(self, kernel_class):
        cls = KERNEL_CLASSES[kernel_class] if isinstance(kernel_class, str) else kernel_class
        _check(as2d_kv_profile(self.handle, -1 if cls is None else cls), "as2d_kv_profile")

    def profile_read(self):
        st, n, ms, alln = as2d_kv_profile_read(self.handle)
        _check(st, "as2d_kv_profile_read")
        return n, ms, alln

    def set_wait_limit(self, ns):
        _check(_lib.as2d_kv_set_wait_limit(self.handle, int(ns)), "as2d_kv_set_wait_limit")

    def check(self, stream=0):
        _check(as2d_kv_check(self.handle, stream), "as2d_kv_check")

    def close(self):
        if self.handle:
            as2d_kv_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
