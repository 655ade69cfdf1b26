"""Sentinel-compressed KV cache decode path for GB300 (sm_103a).

Thin Python binding of the C ABI in ``include/kvc.h`` (libkvc.so, loaded with
ctypes).  Every step of the path runs in the library's CUDA kernels; this
module only marshals arguments.  PyTorch provides device memory and streams.

Functions named like the C ABI (``kvc_append``, ``kvc_compress_spans``,
``kvc_decode_attention``, ``kvc_masked_reference_layout``, ...) take a cache
handle; ``KVCache`` wraps them and owns the device buffers.
"""
from __future__ import annotations

import ctypes
from typing import Optional

import numpy as np

from . import _lib

NORMAL, CL, CR = 0, 1, 2
POLICY_PAPER, POLICY_KEEP_CL, POLICY_LOCAL = 0, 1, 2
F16, BF16 = 0, 1
_DTYPES = {"f16": F16, "bf16": BF16}
STATUS_NAMES = {0: "KVC_OK", 1: "KVC_ERR_INVALID_ARG", 2: "KVC_ERR_UNSUPPORTED", 3: "KVC_ERR_CAPACITY",
                4: "KVC_ERR_SPAN", 5: "KVC_ERR_STATE", 6: "KVC_ERR_CUDA", 7: "KVC_ERR_DEVICE_CHECK",
                8: "KVC_ERR_TIMEOUT", 9: "KVC_ERR_NO_MEMORY"}


class KvcError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status
        self.message = message


def lib():
    return _lib.load()


def _check(rc: int):
    if rc != 0:
        L = lib()
        raise KvcError(rc, (L.kvc_last_error() or b"").decode())


def _np(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _ptr(a) -> Optional[int]:
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        return a.ctypes.data
    return a.data_ptr()


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        import torch

        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def stream_handle(stream=None) -> int:
    """The cudaStream_t (as an int) that a call given `stream` runs on: None means torch's current
    stream.  Resolve it once and pass the int to a run of calls to skip the per-call lookup."""
    return _stream_handle(stream)


def _dev(t, name, dtype=None, numel=None):
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} must have {numel} elements, got {t.numel()}")
    return t


# ------------------------------------------------------------------------------------------
# span book (host only)
# ------------------------------------------------------------------------------------------

def kvc_book_create(b: int, capacity, policy: int = POLICY_PAPER, local_ratio: float = 0.0) -> int:
    cap = _np(capacity, np.int64)
    h = ctypes.c_void_p()
    if policy == POLICY_LOCAL:
        _check(lib().kvc_book_create_local(b, float(local_ratio), cap.ctypes.data, ctypes.byref(h)))
    else:
        _check(lib().kvc_book_create(b, policy, cap.ctypes.data, ctypes.byref(h)))
    return h.value


def kvc_book_destroy(book: int):
    lib().kvc_book_destroy(book)


def kvc_book_next_positions(book: int, n_new, kinds) -> np.ndarray:
    n_new = _np(n_new, np.int32)
    kinds = _np(kinds, np.uint8)
    pos = np.empty(max(int(n_new.sum()), 1), dtype=np.int32)
    _check(lib().kvc_book_next_positions(book, n_new.ctypes.data, kinds.ctypes.data, pos.ctypes.data))
    return pos[:int(n_new.sum())]


def kvc_book_append(book: int, n_new, kinds, pos):
    n_new, kinds, pos = _np(n_new, np.int32), _np(kinds, np.uint8), _np(pos, np.int32)
    _check(lib().kvc_book_append(book, n_new.ctypes.data, kinds.ctypes.data, pos.ctypes.data))


def kvc_book_append_free_closed(book: int, n_new, kinds, pos):
    n_new, kinds, pos = _np(n_new, np.int32), _np(kinds, np.uint8), _np(pos, np.int32)
    _check(lib().kvc_book_append_free_closed(book, n_new.ctypes.data, kinds.ctypes.data, pos.ctypes.data))


def kvc_book_compress(book: int, seq, cl, cr):
    seq, cl, cr = _np(seq, np.int32), _np(cl, np.int64), _np(cr, np.int64)
    _check(lib().kvc_book_compress(book, seq.ctypes.data, cl.ctypes.data, cr.ctypes.data, seq.size))


def kvc_book_pending_spans(book: int, seq: int):
    n = ctypes.c_int64()
    _check(lib().kvc_book_pending_spans(book, seq, None, None, 0, ctypes.byref(n)))
    cl = np.empty(max(n.value, 1), np.int64)
    cr = np.empty(max(n.value, 1), np.int64)
    _check(lib().kvc_book_pending_spans(book, seq, cl.ctypes.data, cr.ctypes.data, n.value, ctypes.byref(n)))
    return [(int(cl[i]), int(cr[i])) for i in range(n.value)]


def kvc_book_lengths(book: int, b: int):
    ln = np.empty(b, np.int64)
    at = np.empty(b, np.int64)
    _check(lib().kvc_book_lengths(book, ln.ctypes.data, at.ctypes.data))
    return ln, at


def kvc_book_prefill_keys(book: int, seq: int, n_q: int) -> np.ndarray:
    """Per stored row of `seq`: (hid << 1) | is_cl, the masked-prefill bounds for its last n_q tokens."""
    n = ctypes.c_int64()
    rc = lib().kvc_book_prefill_keys(book, seq, n_q, None, 0, ctypes.byref(n))
    if rc != 0 and n.value == 0:
        _check(rc)
    meta = np.empty(max(n.value, 1), np.int32)
    _check(lib().kvc_book_prefill_keys(book, seq, n_q, meta.ctypes.data, n.value, ctypes.byref(n)))
    return meta[:n.value].copy()


def _layout_sizes(fn, *args):
    nf, ns = ctypes.c_int64(), ctypes.c_int64()
    rc = fn(*args, 0, None, None, None, ctypes.byref(nf), None, None, ctypes.byref(ns))
    if rc not in (0, 3):
        _check(rc)
    return max(nf.value, ns.value)


def kvc_book_layout(book: int, seq: int, cap: Optional[int] = None):
    if cap is None:
        cap = _layout_sizes(lib().kvc_book_layout, book, seq)
    cap = max(int(cap), 1)
    kind = np.empty(cap, np.uint8)
    pos = np.empty(cap, np.int32)
    vis = np.empty(cap, np.uint8)
    so = np.empty(cap, np.int32)
    sp = np.empty(cap, np.int32)
    nf, ns = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().kvc_book_layout(book, seq, cap, kind.ctypes.data, pos.ctypes.data, vis.ctypes.data,
                                 ctypes.byref(nf), so.ctypes.data, sp.ctypes.data, ctypes.byref(ns)))
    return {"kinds": kind[:nf.value], "pos": pos[:nf.value], "visible": vis[:nf.value].astype(bool),
            "stored_orig": so[:ns.value], "stored_pos": sp[:ns.value]}


class Book:
    """Host-only span bookkeeping of b token histories (positions, spans, stored rows).

    A cache's own book (``KVCache.book``) is a read-only view: appends and compactions go through
    the cache so that its device state follows."""

    def __init__(self, b: int, capacity, policy: int = POLICY_PAPER, _handle: Optional[int] = None,
                 local_ratio: float = 0.0):
        self.b = b
        self._owned = _handle is None
        self.readonly = _handle is not None
        self.handle = kvc_book_create(b, capacity, policy, local_ratio) if _handle is None else _handle

    def next_positions(self, n_new, kinds):
        return kvc_book_next_positions(self.handle, n_new, kinds)

    def append(self, n_new, kinds, pos=None, free_closed: bool = False):
        if self.readonly:
            raise KvcError(5, "a cache's book is read-only; append through the cache")
        if pos is None:
            pos = self.next_positions(n_new, kinds)
        (kvc_book_append_free_closed if free_closed else kvc_book_append)(self.handle, n_new, kinds, pos)
        return pos

    def compress(self, seq, cl, cr):
        if self.readonly:
            raise KvcError(5, "a cache's book is read-only; compress through the cache")
        kvc_book_compress(self.handle, seq, cl, cr)

    def pending_spans(self, seq: int):
        return kvc_book_pending_spans(self.handle, seq)

    def prefill_keys(self, seq: int, n_q: int) -> np.ndarray:
        return kvc_book_prefill_keys(self.handle, seq, n_q)

    def lengths(self):
        return kvc_book_lengths(self.handle, self.b)

    def layout(self, seq: int):
        return kvc_book_layout(self.handle, seq, None)

    def __del__(self):
        if getattr(self, "_owned", False) and getattr(self, "handle", None):
            try:
                kvc_book_destroy(self.handle)
            except Exception:
                pass
            self.handle = None


# ------------------------------------------------------------------------------------------
# cache
# ------------------------------------------------------------------------------------------

def make_config(M, H, d_head, capacity, dtype="f16", rotary_dim=0, rope_base=10000.0, policy=POLICY_PAPER,
                local_ratio=0.0):
    cap = _np(capacity, np.int64)
    cfg = _lib.KvcConfig()
    cfg.M, cfg.H, cfg.d_head, cfg.b = M, H, d_head, cap.size
    cfg.dtype = _DTYPES[dtype]
    cfg.rotary_dim = rotary_dim
    cfg.rope_base = rope_base
    cfg.policy = policy
    cfg.local_ratio = local_ratio
    cfg.seq_capacity = cap.ctypes.data
    return cfg, cap


def kvc_required_bytes(cfg) -> dict:
    k, v, m, w = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    _check(lib().kvc_required_bytes(ctypes.byref(cfg), ctypes.byref(k), ctypes.byref(v), ctypes.byref(m),
                                    ctypes.byref(w)))
    return {"k": k.value, "v": v.value, "meta": m.value, "workspace": w.value}


def kvc_create(cfg) -> int:
    h = ctypes.c_void_p()
    _check(lib().kvc_create(ctypes.byref(cfg), ctypes.byref(h)))
    return h.value


def kvc_destroy(cache: int):
    lib().kvc_destroy(cache)


def kvc_append(cache: int, layer: int, k, v, n_new, pos, kinds, stream=None):
    n_new = _np(n_new, np.int32) if n_new is not None else None
    pos = _np(pos, np.int32) if pos is not None else None
    kinds = _np(kinds, np.uint8) if kinds is not None else None
    _check(lib().kvc_append(cache, layer, _ptr(k), _ptr(v), _ptr(n_new), _ptr(pos), _ptr(kinds),
                            _stream_handle(stream)))


def kvc_append_free_closed(cache: int, layer: int, k, v, n_new, pos, kinds, stream=None):
    """kvc_append that frees spans opened and closed among the new tokens as they are written."""
    n_new = _np(n_new, np.int32) if n_new is not None else None
    pos = _np(pos, np.int32) if pos is not None else None
    kinds = _np(kinds, np.uint8) if kinds is not None else None
    _check(lib().kvc_append_free_closed(cache, layer, _ptr(k), _ptr(v), _ptr(n_new), _ptr(pos), _ptr(kinds),
                                        _stream_handle(stream)))


def kvc_compress_spans(cache: int, seq, cl, cr, stream=None):
    seq, cl, cr = _np(seq, np.int32), _np(cl, np.int64), _np(cr, np.int64)
    _check(lib().kvc_compress_spans(cache, seq.ctypes.data, cl.ctypes.data, cr.ctypes.data, seq.size,
                                    _stream_handle(stream)))


def kvc_decode_attention(cache: int, layer: int, q, scale: float, out, stream=None):
    _check(lib().kvc_decode_attention(cache, layer, _ptr(q), float(scale), _ptr(out), _stream_handle(stream)))


def kvc_decode_attention_layers(cache: int, first: int, n_layers: int, q, q_layer_stride: int, scale: float, out,
                                out_layer_stride: int, stream=None):
    """kvc_decode_attention of layers [first, first + n_layers) in one call (strides in elements)."""
    _check(lib().kvc_decode_attention_layers(cache, first, n_layers, _ptr(q), int(q_layer_stride), float(scale),
                                             _ptr(out), int(out_layer_stride), _stream_handle(stream)))


def kvc_decode_attention_static_scratch(cache: int, layer: int, q, scale: float, out, stream=None):
    """Decode whose split-K scratch is the library's static device array (no allocation anywhere)."""
    _check(lib().kvc_decode_attention_static_scratch(cache, layer, _ptr(q), float(scale), _ptr(out),
                                                     _stream_handle(stream)))


def kvc_prefill_attention(cache: int, layer: int, q, n_q, scale: float, out, stream=None):
    n_q = _np(n_q, np.int32)
    _check(lib().kvc_prefill_attention(cache, layer, _ptr(q), n_q.ctypes.data, float(scale), _ptr(out),
                                       _stream_handle(stream)))


def kvc_masked_reference_layout(cache: int, seq: int, cap: int, stream=None):
    kind = np.empty(cap, np.uint8)
    pos = np.empty(cap, np.int32)
    vis = np.empty(cap, np.uint8)
    so = np.empty(cap, np.int32)
    sp = np.empty(cap, np.int32)
    nf, ns = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().kvc_masked_reference_layout(cache, seq, cap, kind.ctypes.data, pos.ctypes.data, vis.ctypes.data,
                                             ctypes.byref(nf), so.ctypes.data, sp.ctypes.data, ctypes.byref(ns),
                                             _stream_handle(stream)))
    return {"kinds": kind[:nf.value], "pos": pos[:nf.value], "visible": vis[:nf.value].astype(bool),
            "stored_orig": so[:ns.value], "stored_pos": sp[:ns.value]}


def kvc_device_status(cache: int, stream=None) -> int:
    w = ctypes.c_int32()
    _check(lib().kvc_device_status(cache, _stream_handle(stream), ctypes.byref(w)))
    return w.value


def kvc_check_bounded_wait(cache: int, limit_ns: int, stream=None):
    _check(lib().kvc_check_bounded_wait(cache, int(limit_ns), _stream_handle(stream)))


def kvc_launch_count(cache: int) -> int:
    return lib().kvc_launch_count(cache)


def kvc_set_compaction_timing(cache: int, enable: bool):
    _check(lib().kvc_set_compaction_timing(cache, 1 if enable else 0))


def kvc_last_compaction_ms(cache: int):
    """(scan ms, row-move ms) of the last timed compaction."""
    a = ctypes.c_float()
    b = ctypes.c_float()
    _check(lib().kvc_last_compaction_ms(cache, ctypes.byref(a), ctypes.byref(b)))
    return float(a.value), float(b.value)


def kvc_last_decode_plan(cache: int) -> dict:
    a = np.zeros(4, np.int32)
    _check(lib().kvc_last_decode_plan(cache, a.ctypes.data))
    return {"mode": int(a[0]), "workers": int(a[1]), "tile_rows": int(a[2]), "stages": int(a[3])}


class KVCache:
    """A sentinel-compressed KV cache: owns its device buffers (torch) and the library handle."""

    def __init__(self, M: int, H: int, d_head: int, capacity, dtype: str = "f16", rotary_dim: int = 0,
                 rope_base: float = 10000.0, policy: int = POLICY_PAPER, device=None, local_ratio: float = 0.0):
        import torch

        self.M, self.H, self.d, self.dtype = M, H, d_head, dtype
        self.rotary_dim, self.rope_base, self.policy = rotary_dim, rope_base, policy
        self.local_ratio = local_ratio
        cfg, cap = make_config(M, H, d_head, capacity, dtype, rotary_dim, rope_base, policy, local_ratio)
        self.capacity = cap
        self.b = cap.size
        self.C = int(cap.sum())
        self.offsets = np.concatenate([[0], np.cumsum(cap)[:-1]]).astype(np.int64)
        sizes = kvc_required_bytes(cfg)
        device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
        tdt = torch.float16 if dtype == "f16" else torch.bfloat16
        self.torch_dtype = tdt
        self.k = torch.empty(sizes["k"] // 2, dtype=tdt, device=device)
        self.v = torch.empty(sizes["v"] // 2, dtype=tdt, device=device)
        self.pos = torch.empty(sizes["meta"] // 4, dtype=torch.int32, device=device)
        self.orig = torch.empty(sizes["meta"] // 4, dtype=torch.int32, device=device)
        self.workspace = torch.empty(sizes["workspace"], dtype=torch.uint8, device=device)
        self.sizes = sizes
        cfg.k_base, cfg.v_base = self.k.data_ptr(), self.v.data_ptr()
        cfg.pos_base, cfg.orig_base = self.pos.data_ptr(), self.orig.data_ptr()
        cfg.workspace, cfg.workspace_bytes = self.workspace.data_ptr(), sizes["workspace"]
        self._cfg = cfg
        self.handle = kvc_create(cfg)
        self.book = Book(self.b, cap, policy, _handle=lib().kvc_get_book(self.handle))

    # views of the device layout (rows of d_head elements)
    def k_plane(self, layer: int):
        return self.k.view(self.M, self.H * self.C, self.d)[layer]

    def v_plane(self, layer: int):
        return self.v.view(self.M, self.H * self.C, self.d)[layer]

    def stream_rows(self, plane, s: int, h: int, n: int):
        """Rows [0, n) of sequence s, head h in a (layer, K/V) plane."""
        base = self.H * int(self.offsets[s]) + h * int(self.capacity[s])
        return plane[base:base + n]

    def append(self, k, v, n_new, kinds, pos=None, layer: int = -1, stream=None, free_closed: bool = False):
        """k, v: device [M or 1][N][H][d] in the cache dtype.  Positions default to the tied positions.
        free_closed: free spans opened and closed among these tokens as they are written."""
        n_new = _np(n_new, np.int32)
        kinds = _np(kinds, np.uint8)
        if layer <= 0 and pos is None:
            pos = self.book.next_positions(n_new, kinds)
        N = int(n_new.sum())
        nl = self.M if layer < 0 else 1
        _dev(k, "k", self.torch_dtype, nl * N * self.H * self.d)
        _dev(v, "v", self.torch_dtype, nl * N * self.H * self.d)
        (kvc_append_free_closed if free_closed else kvc_append)(self.handle, layer, k, v, n_new, pos, kinds, stream)
        return pos

    def compress_spans(self, seq, cl, cr, stream=None):
        kvc_compress_spans(self.handle, seq, cl, cr, stream)

    def decode_attention(self, layer: int, q, scale: float, out=None, stream=None):
        import torch

        _dev(q, "q", self.torch_dtype, self.b * self.H * self.d)
        if out is None:
            out = torch.empty(self.b, self.H, self.d, dtype=torch.float32, device=q.device)
        _dev(out, "out", torch.float32, self.b * self.H * self.d)
        kvc_decode_attention(self.handle, layer, q, scale, out, stream)
        return out

    def prefill_attention(self, layer: int, q, n_q, scale: float, out=None, stream=None):
        """Masked prefill of the last n_q[s] tokens of every sequence s (q: [sum n_q, H, d_head])."""
        import torch

        n_tok = int(np.sum(n_q))
        _dev(q, "q", self.torch_dtype, n_tok * self.H * self.d)
        if out is None:
            out = torch.empty(n_tok, self.H, self.d, dtype=torch.float32, device=q.device)
        _dev(out, "out", torch.float32, n_tok * self.H * self.d)
        kvc_prefill_attention(self.handle, layer, q, n_q, scale, out, stream)
        return out

    def prefill_keys(self, seq: int, n_q: int) -> np.ndarray:
        return kvc_book_prefill_keys(lib().kvc_get_book(self.handle), seq, n_q)

    def decode_attention_layers(self, q, scale: float, out=None, stream=None):
        """Decode attention of every layer in one call: q [M][b][H][d_head], out fp32 [M][b][H][d_head]."""
        import torch

        _dev(q, "q", self.torch_dtype, self.M * self.b * self.H * self.d)
        if out is None:
            out = torch.empty(self.M, self.b, self.H, self.d, dtype=torch.float32, device=q.device)
        _dev(out, "out", torch.float32, self.M * self.b * self.H * self.d)
        n = self.b * self.H * self.d
        kvc_decode_attention_layers(self.handle, 0, self.M, q, n, scale, out, n, stream)
        return out

    def masked_reference_layout(self, seq: int, stream=None):
        cap = _layout_sizes(lib().kvc_book_layout, lib().kvc_get_book(self.handle), seq)
        return kvc_masked_reference_layout(self.handle, seq, max(cap, 1), stream)

    def device_status(self, stream=None) -> int:
        return kvc_device_status(self.handle, stream)

    def pending_spans(self, seq: int):
        return self.book.pending_spans(seq)

    def lengths(self):
        return self.book.lengths()

    @property
    def launch_count(self) -> int:
        return kvc_launch_count(self.handle)

    @property
    def last_decode_plan(self) -> dict:
        return kvc_last_decode_plan(self.handle)

    def close(self):
        if getattr(self, "handle", None):
            kvc_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
