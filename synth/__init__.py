"""Seeded synthetic inputs shared by the oracle and the CUDA path.

Every value is a pure function of (seed, stream, index) through Philox4x32-10
(Salmon et al., SC 2011).  The host filler (libsynth_host.so, C + OpenMP) and
the device filler (libsynth_cuda.so, sm_103a) are bit-identical, so large
models can be generated on the GPU while the oracle gets the same bits on the
host.  Nothing here computes any part of the verification method.
"""
import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
_HOST = None
_CUDA = None


def _load_host():
    global _HOST
    if _HOST is None:
        path = os.path.join(HERE, "libsynth_host.so")
        if not os.path.exists(path):
            from . import build as _b
            _b.build_host()
        lib = ctypes.CDLL(path)
        lib.synth_philox4x32_10.argtypes = [ctypes.POINTER(ctypes.c_uint32),
                                            ctypes.POINTER(ctypes.c_uint32),
                                            ctypes.POINTER(ctypes.c_uint32)]
        lib.synth_normal_scale.argtypes = [ctypes.c_double]
        lib.synth_normal_scale.restype = ctypes.c_float
        lib.synth_fill_normal_bf16_offset.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
            ctypes.c_float, ctypes.c_float]
        lib.synth_fill_uniform_int.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
            ctypes.c_uint32]
        _HOST = lib
    return _HOST


def _load_cuda():
    global _CUDA
    if _CUDA is None:
        path = os.path.join(HERE, "libsynth_cuda.so")
        if not os.path.exists(path):
            raise RuntimeError("libsynth_cuda.so is not built; run __graft_entry__.build()")
        lib = ctypes.CDLL(path)
        lib.synth_cuda_fill_normal_bf16.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
            ctypes.c_float, ctypes.c_float, ctypes.c_void_p]
        lib.synth_cuda_fill_normal_bf16.restype = ctypes.c_int
        lib.synth_cuda_fill_uniform_int.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
            ctypes.c_uint32, ctypes.c_void_p]
        lib.synth_cuda_fill_uniform_int.restype = ctypes.c_int
        lib.synth_cuda_build_candidates.argtypes = [
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p,
            ctypes.c_int32, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_void_p]
        lib.synth_cuda_build_candidates.restype = ctypes.c_int
        _CUDA = lib
    return _CUDA


def philox4x32_10(ctr, key):
    """One Philox4x32-10 block (4 x uint32) for counter ctr[4] and key key[2]."""
    lib = _load_host()
    c = (ctypes.c_uint32 * 4)(*[int(v) & 0xFFFFFFFF for v in ctr])
    k = (ctypes.c_uint32 * 2)(*[int(v) & 0xFFFFFFFF for v in key])
    out = (ctypes.c_uint32 * 4)()
    lib.synth_philox4x32_10(c, k, out)
    return tuple(int(v) for v in out)


def normal_scale(sigma):
    return float(_load_host().synth_normal_scale(float(sigma)))


def normal_bf16(n, seed, stream, sigma=0.02, base=0.0):
    """bf16 bit patterns (uint16) of n draws of base + N(0, sigma)."""
    out = np.empty(int(n), dtype=np.uint16)
    _load_host().synth_fill_normal_bf16_offset(
        out.ctypes.data, int(n), int(seed), int(stream) & 0xFFFFFFFF,
        normal_scale(sigma), float(base))
    return out


def uniform_int(n, seed, stream, upper):
    """n integers uniform in [0, upper) as int32."""
    out = np.empty(int(n), dtype=np.int32)
    _load_host().synth_fill_uniform_int(out.ctypes.data, int(n), int(seed),
                                        int(stream) & 0xFFFFFFFF, int(upper))
    return out


def cuda_normal_bf16(ptr, n, seed, stream, sigma=0.02, base=0.0, cuda_stream=0):
    """Fill n bf16 values at device pointer ptr; same bits as normal_bf16."""
    rc = _load_cuda().synth_cuda_fill_normal_bf16(
        ctypes.c_void_p(int(ptr)), int(n), int(seed), int(stream) & 0xFFFFFFFF,
        normal_scale(sigma), float(base), ctypes.c_void_p(int(cuda_stream)))
    if rc != 0:
        raise RuntimeError(f"synth_cuda_fill_normal_bf16 failed: cudaError {rc}")


def cuda_uniform_int(ptr, n, seed, stream, upper, cuda_stream=0):
    rc = _load_cuda().synth_cuda_fill_uniform_int(
        ctypes.c_void_p(int(ptr)), int(n), int(seed), int(stream) & 0xFFFFFFFF,
        int(upper), ctypes.c_void_p(int(cuda_stream)))
    if rc != 0:
        raise RuntimeError(f"synth_cuda_fill_uniform_int failed: cudaError {rc}")
