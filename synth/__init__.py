"""Seeded synthetic inputs for the sentinel-compressed KV decode path.

This module is shared by the CUDA path's tests/bench and by the CPU oracle's
tests.  It holds none of the method's arithmetic: it generates K, V and q
values (Philox4x32-10 counter-based generator, see ``synth_gen.h``) and the
token-kind structure of each workload (``synth.workloads``).

Two builds of the same generator exist: ``libsynth_host.so`` (host, used to
regenerate slices for the oracle) and ``libsynth_cuda.so`` (device, used to
fill tens of GB of workload inputs in HBM).  They give identical bits.
"""
from __future__ import annotations

import ctypes
import math
import os

import numpy as np

from . import build as _build

K_TENSOR, V_TENSOR, Q_TENSOR = 0, 1, 2
DTYPE_F16, DTYPE_BF16 = 0, 1
_DTYPE_CODES = {"f16": DTYPE_F16, "bf16": DTYPE_BF16}

_host = None
_cuda = None


def dtype_code(dtype: str) -> int:
    return _DTYPE_CODES[dtype]


def tag(tensor: int, layer: int) -> int:
    """Counter word 3: which tensor (K, V, q) and which layer."""
    return int(tensor) | (int(layer) << 8)


def scale_for(sigma: float) -> np.float32:
    """binary32 multiplier giving standard deviation ``sigma`` (Irwin-Hall(4) of 16-bit uniforms)."""
    return np.float32(sigma * math.sqrt(3.0) / 65536.0)


def host_lib():
    global _host
    if _host is None:
        path = _build.build_host()
        lib = ctypes.CDLL(path)
        u64, i32, i64, f32, u32, p = (ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_float,
                                      ctypes.c_uint32, ctypes.c_void_p)
        lib.syn_fill_tokens.argtypes = [u64, i32, f32, u32, i64, p, p, i32, i32, p]
        lib.syn_fill_tokens.restype = None
        lib.syn_centred_sums.argtypes = [u64, u32, i64, p, p, p, p]
        lib.syn_centred_sums.restype = None
        lib.syn_philox_blocks.argtypes = [i64, p, p, p]
        lib.syn_philox_blocks.restype = None
        lib.syn_f32_to_f16_array.argtypes = [i64, p, p]
        lib.syn_f32_to_bf16_array.argtypes = [i64, p, p]
        _host = lib
    return _host


def cuda_lib():
    global _cuda
    if _cuda is None:
        path = _build.build_cuda()
        lib = ctypes.CDLL(path)
        u64, i32, i64, f32, u32, p = (ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_float,
                                      ctypes.c_uint32, ctypes.c_void_p)
        lib.syn_cuda_fill_tokens.argtypes = [u64, i32, f32, u32, i64, p, p, i32, i32, p, p]
        lib.syn_cuda_fill_tokens.restype = ctypes.c_int
        _cuda = lib
    return _cuda


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def fill_tokens_host(seed: int, dtype: str, scale, tag_: int, tok_t, tok_s, H: int, d: int) -> np.ndarray:
    """uint16 bit patterns, shape [n_tok, H, d]; token ``i`` uses counters (tok_t[i], tok_s[i], h*1024+e)."""
    tok_t = np.ascontiguousarray(tok_t, dtype=np.int32)
    tok_s = np.ascontiguousarray(tok_s, dtype=np.int32)
    assert tok_t.shape == tok_s.shape and tok_t.ndim == 1
    out = np.empty((tok_t.size, H, d), dtype=np.uint16)
    host_lib().syn_fill_tokens(seed, dtype_code(dtype), float(np.float32(scale)), tag_, tok_t.size, _ptr(tok_t),
                               _ptr(tok_s), H, d, _ptr(out))
    return out


def fill_tokens_cuda(seed: int, dtype: str, scale, tag_: int, tok_t, tok_s, H: int, d: int, out, stream=None):
    """Device fill of ``out`` (a CUDA tensor of n_tok*H*d 16-bit elements) from device int32 ``tok_t``/``tok_s``."""
    import torch

    assert tok_t.is_cuda and tok_s.is_cuda and out.is_cuda
    assert tok_t.dtype == torch.int32 and tok_s.dtype == torch.int32
    assert out.element_size() == 2 and out.is_contiguous() and out.numel() == tok_t.numel() * H * d
    if stream is None:
        stream = torch.cuda.current_stream()
    rc = cuda_lib().syn_cuda_fill_tokens(seed, dtype_code(dtype), float(np.float32(scale)), tag_, tok_t.numel(),
                                         tok_t.data_ptr(), tok_s.data_ptr(), H, d, out.data_ptr(),
                                         stream.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"syn_cuda_fill_tokens failed with CUDA error {rc}")
    return out


def centred_sums(seed: int, tag_: int, i0, i1, i2) -> np.ndarray:
    i0 = np.ascontiguousarray(i0, dtype=np.uint32)
    i1 = np.ascontiguousarray(i1, dtype=np.uint32)
    i2 = np.ascontiguousarray(i2, dtype=np.uint32)
    out = np.empty(i0.size, dtype=np.int32)
    host_lib().syn_centred_sums(seed, tag_, i0.size, _ptr(i0), _ptr(i1), _ptr(i2), _ptr(out))
    return out


def philox_blocks(ctr4: np.ndarray, key2: np.ndarray) -> np.ndarray:
    ctr4 = np.ascontiguousarray(ctr4, dtype=np.uint32).reshape(-1, 4)
    key2 = np.ascontiguousarray(key2, dtype=np.uint32).reshape(-1, 2)
    out = np.empty_like(ctr4)
    host_lib().syn_philox_blocks(ctr4.shape[0], _ptr(ctr4), _ptr(key2), _ptr(out))
    return out


def f32_to_f16_bits(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    host_lib().syn_f32_to_f16_array(x.size, _ptr(x), _ptr(out))
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    host_lib().syn_f32_to_bf16_array(x.size, _ptr(x), _ptr(out))
    return out
