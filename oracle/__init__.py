"""fp64 CPU oracle for the decode step over a sentinel-compressed KV cache.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, by ``__graft_entry__.smoke``
and by the CPU-baseline leg of ``bench.py``, never by the library.  It shares
no code with the CUDA path; see ``kvc_oracle.c`` for the definitions, the
paper passages they follow and the readings taken where the paper is silent.

The wrappers here only marshal numpy arrays into the C functions.
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import build as _build

NORMAL, CL, CR = 0, 1, 2
POLICY_PAPER, POLICY_KEEP_CL = 0, 1
F16, BF16 = 0, 1
_DT = {"f16": F16, "bf16": BF16}

_lib = None


class OracleError(RuntimeError):
    pass


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(_build.build())
        p, i64, i32, f64, u16 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double, ctypes.c_uint16
        L.orc_f16_to_f64.argtypes = [u16]
        L.orc_f16_to_f64.restype = f64
        L.orc_bf16_to_f64.argtypes = [u16]
        L.orc_bf16_to_f64.restype = f64
        L.orc_f64_to_f16.argtypes = [f64]
        L.orc_f64_to_f16.restype = u16
        L.orc_f64_to_bf16.argtypes = [f64]
        L.orc_f64_to_bf16.restype = u16
        L.orc_decode16_array.argtypes = [i64, p, i32, p]
        L.orc_decode16_array.restype = None
        L.orc_encode16_array.argtypes = [i64, p, i32, p]
        L.orc_encode16_array.restype = None
        L.orc_tied_positions.argtypes = [p, i64, p]
        L.orc_pair_spans.argtypes = [p, i64, p, p, p, p]
        L.orc_visible.argtypes = [p, i64, i32, p]
        L.orc_stored_rows.argtypes = [i64, p, p, i64, i32, p, p]
        L.orc_rope.argtypes = [p, i32, i32, f64, f64, p]
        L.orc_rope.restype = None
        L.orc_attend.argtypes = [i32, i32, p, p, p, p, p, i64, f64, i32, f64, i32, p]
        L.orc_masked_decode.argtypes = [i64, i64, i32, i32, p, p, p, p, p, p, p, p, f64, i32, f64, i32, p, i32]
        L.orc_max_threads.argtypes = []
        L.orc_visible_local.argtypes = [i64, f64, p]
        L.orc_local_decode.argtypes = [i64, i64, i32, i32, p, p, p, p, p, p, p, f64, i32, f64, f64, p, i32]
        L.orc_masked_prefill.argtypes = [i64, i64, i32, i32, p, p, p, p, p, p, p, p, p, p, f64, i32, f64, i32, p,
                                         i32]
        _lib = L
    return _lib


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _check(rc: int, what: str):
    if rc != 0:
        raise OracleError(f"{what} failed with code {rc}")


def max_threads() -> int:
    return lib().orc_max_threads()


def decode16(bits, dtype: str) -> np.ndarray:
    bits = _c(bits, np.uint16)
    out = np.empty(bits.shape, dtype=np.float64)
    lib().orc_decode16_array(bits.size, bits.ctypes.data, _DT[dtype], out.ctypes.data)
    return out


def encode16(x, dtype: str) -> np.ndarray:
    x = _c(x, np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().orc_encode16_array(x.size, x.ctypes.data, _DT[dtype], out.ctypes.data)
    return out


def tied_positions(kinds) -> np.ndarray:
    kinds = _c(kinds, np.uint8)
    pos = np.empty(kinds.size, dtype=np.int32)
    _check(lib().orc_tied_positions(kinds.ctypes.data, kinds.size, pos.ctypes.data), "tied_positions")
    return pos


def pair_spans(kinds):
    """(closed spans as a list of (cl, cr), open <CL> index or -1)."""
    kinds = _c(kinds, np.uint8)
    n = kinds.size
    cl = np.empty(n // 2 + 1, dtype=np.int64)
    cr = np.empty(n // 2 + 1, dtype=np.int64)
    nc = ctypes.c_int64()
    op = ctypes.c_int64()
    _check(lib().orc_pair_spans(kinds.ctypes.data, n, cl.ctypes.data, cr.ctypes.data, ctypes.byref(nc),
                                ctypes.byref(op)), "pair_spans")
    return [(int(cl[i]), int(cr[i])) for i in range(nc.value)], int(op.value)


def visible(kinds, t_q: int, policy: int = POLICY_PAPER) -> np.ndarray:
    """bool[t_q+1]: which history tokens the query at ``t_q`` attends to."""
    kinds = _c(kinds, np.uint8)
    vis = np.empty(t_q + 1, dtype=np.uint8)
    _check(lib().orc_visible(kinds.ctypes.data, t_q, policy, vis.ctypes.data), "visible")
    return vis.astype(bool)


def stored_rows(n_hist: int, spans, policy: int = POLICY_PAPER) -> np.ndarray:
    """Increasing history indices kept after freeing ``spans`` [(cl, cr), ...]."""
    cl = _c([s[0] for s in spans], np.int64)
    cr = _c([s[1] for s in spans], np.int64)
    rows = np.empty(max(n_hist, 1), dtype=np.int64)
    n = ctypes.c_int64()
    _check(lib().orc_stored_rows(n_hist, cl.ctypes.data, cr.ctypes.data, len(spans), policy, rows.ctypes.data,
                                 ctypes.byref(n)), "stored_rows")
    return rows[:n.value].copy()


def rope(x, rot: int, base: float, pos: float) -> np.ndarray:
    x = _c(x, np.float64)
    y = np.empty_like(x)
    lib().orc_rope(x.ctypes.data, x.size, rot, base, float(pos), y.ctypes.data)
    return y


def attend(q_bits, K_bits, V_bits, pos, rows, dtype: str, scale: float, rot: int = 0, base: float = 10000.0,
           qpos: int = 0) -> np.ndarray:
    """Softmax attention of one query over the listed rows of one (sequence, head)."""
    q_bits = _c(q_bits, np.uint16)
    K_bits = _c(K_bits, np.uint16)
    V_bits = _c(V_bits, np.uint16)
    d = q_bits.size
    pos = _c(pos if pos is not None else np.zeros(K_bits.shape[0]), np.int32)
    rows = _c(rows, np.int64)
    out = np.empty(d, dtype=np.float64)
    _check(lib().orc_attend(d, _DT[dtype], q_bits.ctypes.data, K_bits.ctypes.data, V_bits.ctypes.data,
                            pos.ctypes.data, rows.ctypes.data, rows.size, scale, rot, base, int(qpos),
                            out.ctypes.data), "attend")
    return out


def masked_decode(kinds_list, pos_list, K_list, V_list, q, dtype: str, scale: float, rot: int = 0,
                  base: float = 10000.0, policy: int = POLICY_PAPER, n_threads: int = 0) -> np.ndarray:
    """Decode step over full histories under the sentinel mask.

    kinds_list[s], pos_list[s]: history of sequence s (its query is the last token);
    K_list[s], V_list[s]: uint16 [H, T_s, d]; q: uint16 [n_seq, H, d].  Returns fp64 [n_seq, H, d].
    """
    n_seq = len(kinds_list)
    H, d = q.shape[1], q.shape[2]
    n_hist = _c([k.size for k in kinds_list], np.int64)
    hist_off = np.zeros(n_seq, dtype=np.int64)
    hist_off[1:] = np.cumsum(n_hist)[:-1]
    kinds = _c(np.concatenate(kinds_list), np.uint8)
    pos = _c(np.concatenate(pos_list), np.int32)
    kv_sizes = np.array([K.size for K in K_list], dtype=np.int64)
    for s in range(n_seq):
        assert K_list[s].shape == (H, n_hist[s], d) and V_list[s].shape == (H, n_hist[s], d)
    kv_off = np.zeros(n_seq, dtype=np.int64)
    kv_off[1:] = np.cumsum(kv_sizes)[:-1]
    K = _c(np.concatenate([k.reshape(-1) for k in K_list]), np.uint16)
    V = _c(np.concatenate([v.reshape(-1) for v in V_list]), np.uint16)
    q = _c(q, np.uint16)
    out = np.empty((n_seq, H, d), dtype=np.float64)
    _check(lib().orc_masked_decode(n_seq, H, d, _DT[dtype], n_hist.ctypes.data, hist_off.ctypes.data,
                                   kinds.ctypes.data, pos.ctypes.data, kv_off.ctypes.data, K.ctypes.data,
                                   V.ctypes.data, q.ctypes.data, scale, rot, base, policy, out.ctypes.data,
                                   n_threads), "masked_decode")
    return out


def visible_local(t_q: int, ratio: float) -> np.ndarray:
    """Local Attention mask (Sec. 4.1): bool[t_q+1], the history indices the query at t_q sees."""
    vis = np.empty(t_q + 1, dtype=np.uint8)
    _check(lib().orc_visible_local(t_q, float(ratio), vis.ctypes.data), "visible_local")
    return vis.astype(bool)


def local_decode(pos_list, K_list, V_list, q, dtype: str, scale: float, ratio: float, rot: int = 0,
                 base: float = 10000.0, n_threads: int = 0) -> np.ndarray:
    """Decode under the Local Attention mask: the query of sequence s is its last history token."""
    n_seq = len(pos_list)
    H, d = q.shape[1], q.shape[2]
    n_hist = _c([p.size for p in pos_list], np.int64)
    hist_off = np.zeros(n_seq, dtype=np.int64)
    hist_off[1:] = np.cumsum(n_hist)[:-1]
    pos = _c(np.concatenate(pos_list), np.int32)
    kv_sizes = np.array([k.size for k in K_list], dtype=np.int64)
    kv_off = np.zeros(n_seq, dtype=np.int64)
    kv_off[1:] = np.cumsum(kv_sizes)[:-1]
    K = _c(np.concatenate([k.reshape(-1) for k in K_list]), np.uint16)
    V = _c(np.concatenate([v.reshape(-1) for v in V_list]), np.uint16)
    q = _c(q, np.uint16)
    out = np.empty((n_seq, H, d), dtype=np.float64)
    _check(lib().orc_local_decode(n_seq, H, d, _DT[dtype], n_hist.ctypes.data, hist_off.ctypes.data,
                                  pos.ctypes.data, kv_off.ctypes.data, K.ctypes.data, V.ctypes.data, q.ctypes.data,
                                  scale, rot, base, float(ratio), out.ctypes.data, n_threads), "local_decode")
    return out


def masked_prefill(kinds_list, pos_list, K_list, V_list, n_q, Q, dtype: str, scale: float, rot: int = 0,
                   base: float = 10000.0, policy: int = POLICY_PAPER, n_threads: int = 0) -> np.ndarray:
    """Prefill under the sentinel mask: sequence s's queries are its last n_q[s] history tokens.

    kinds_list/pos_list/K_list/V_list as ``masked_decode``; Q: uint16 [sum n_q, H, d] (sequence s's
    queries consecutive, oldest first).  Returns fp64 [sum n_q, H, d].
    """
    n_seq = len(kinds_list)
    H, d = Q.shape[1], Q.shape[2]
    n_hist = _c([k.size for k in kinds_list], np.int64)
    hist_off = np.zeros(n_seq, dtype=np.int64)
    hist_off[1:] = np.cumsum(n_hist)[:-1]
    n_q = _c(n_q, np.int64)
    assert n_q.size == n_seq and Q.shape[0] == int(n_q.sum())
    q_off = np.zeros(n_seq, dtype=np.int64)
    q_off[1:] = np.cumsum(n_q)[:-1]
    kinds = _c(np.concatenate(kinds_list), np.uint8)
    pos = _c(np.concatenate(pos_list), np.int32)
    for s in range(n_seq):
        assert K_list[s].shape == (H, n_hist[s], d) and V_list[s].shape == (H, n_hist[s], d)
    kv_sizes = np.array([k.size for k in K_list], dtype=np.int64)
    kv_off = np.zeros(n_seq, dtype=np.int64)
    kv_off[1:] = np.cumsum(kv_sizes)[:-1]
    K = _c(np.concatenate([k.reshape(-1) for k in K_list]), np.uint16)
    V = _c(np.concatenate([v.reshape(-1) for v in V_list]), np.uint16)
    Q = _c(Q, np.uint16)
    out = np.empty(Q.shape, dtype=np.float64)
    _check(lib().orc_masked_prefill(n_seq, H, d, _DT[dtype], n_hist.ctypes.data, hist_off.ctypes.data,
                                    kinds.ctypes.data, pos.ctypes.data, kv_off.ctypes.data, K.ctypes.data,
                                    V.ctypes.data, n_q.ctypes.data, q_off.ctypes.data, Q.ctypes.data, scale, rot,
                                    base, policy, out.ctypes.data, n_threads), "masked_prefill")
    return out
