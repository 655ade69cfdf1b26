"""Oracle-side regeneration of a workload's inputs and its expected decode outputs.

TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU baseline).  Regenerates K, V
and q with the host build of the seeded generator, using the same counter
conventions as the CUDA-path harness (K/V of history token t of sequence s:
(i0=t, i1=s) with tag (K|V, layer); the query of layer m at history token t:
tag (q, m), (i0=t, i1=s)), and runs the fp64 oracle over the FULL history under
the mask -- never over a compacted cache.
"""
from __future__ import annotations

import numpy as np

import synth
from synth import workloads as wl

from . import local_decode, masked_decode, masked_prefill, tied_positions, POLICY_PAPER


def history(w: wl.Workload, s: int, steps_done: int):
    """Kinds and positions of sequence s after the prompt and `steps_done` generated tokens."""
    kinds = w.kinds_history(s, steps_done)
    return kinds, tied_positions(kinds)


def kv_bits(w: wl.Workload, layer: int, s: int, T: int, heads=None):
    """uint16 K, V of sequence s for history tokens [0, T): shapes [len(heads), T, d]."""
    tok_t = np.arange(T, dtype=np.int32)
    tok_s = np.full(T, s, dtype=np.int32)
    sc = synth.scale_for(w.kv_sigma)
    K = synth.fill_tokens_host(w.seed, w.dtype, sc, synth.tag(synth.K_TENSOR, layer), tok_t, tok_s, w.H, w.d)
    V = synth.fill_tokens_host(w.seed, w.dtype, sc, synth.tag(synth.V_TENSOR, layer), tok_t, tok_s, w.H, w.d)
    K = K.transpose(1, 0, 2)
    V = V.transpose(1, 0, 2)
    if heads is not None:
        K, V = K[heads], V[heads]
    return np.ascontiguousarray(K), np.ascontiguousarray(V)


def q_bits(w: wl.Workload, layer: int, s: int, t: int, heads=None):
    sc = synth.scale_for(w.q_sigma)
    q = synth.fill_tokens_host(w.seed, w.dtype, sc, synth.tag(synth.Q_TENSOR, layer), np.array([t], np.int32),
                               np.array([s], np.int32), w.H, w.d)[0]
    return q if heads is None else q[heads]


def expected_decode(w: wl.Workload, steps_done: int, layer: int, seqs, heads=None, policy: int = POLICY_PAPER,
                    n_threads: int = 0) -> np.ndarray:
    """fp64 [len(seqs), n_heads, d]: decode of `layer` for the query at the last token of each sequence's
    history (prompt + `steps_done` generated tokens), under the mask over the full history."""
    kinds_l, pos_l, K_l, V_l, q_l = [], [], [], [], []
    for s in seqs:
        kinds, pos = history(w, s, steps_done)
        T = kinds.size
        K, V = kv_bits(w, layer, s, T, heads)
        kinds_l.append(kinds)
        pos_l.append(pos)
        K_l.append(K)
        V_l.append(V)
        q_l.append(q_bits(w, layer, s, T - 1, heads))
    q = np.stack(q_l)
    return masked_decode(kinds_l, pos_l, K_l, V_l, q, w.dtype, w.scale, rot=w.rotary_dim, base=w.rope_base,
                         policy=policy, n_threads=n_threads)


def expected_local_decode(w: wl.Workload, steps_done: int, layer: int, seqs, ratio: float, heads=None,
                          n_threads: int = 0) -> np.ndarray:
    """fp64 decode under the Local Attention mask (the paper's Sec. 4.1 baseline) for the query at the
    last token of each sequence's history; `ratio` as the cache holds it (a binary32 value)."""
    pos_l, K_l, V_l, q_l = [], [], [], []
    for s in seqs:
        kinds, pos = history(w, s, steps_done)
        T = kinds.size
        K, V = kv_bits(w, layer, s, T, heads)
        pos_l.append(pos)
        K_l.append(K)
        V_l.append(V)
        q_l.append(q_bits(w, layer, s, T - 1, heads))
    return local_decode(pos_l, K_l, V_l, np.stack(q_l), w.dtype, w.scale, ratio, rot=w.rotary_dim, base=w.rope_base,
                        n_threads=n_threads)


def expected_prefill(w: wl.Workload, layer: int, seqs, end, n_q, heads=None, policy: int = POLICY_PAPER,
                     n_threads: int = 0) -> np.ndarray:
    """fp64 [sum n_q over seqs, n_heads, d]: masked prefill of `layer` for prompt tokens
    [end[s] - n_q[s], end[s]) of each listed sequence, over its prompt history [0, end[s])."""
    kinds_l, pos_l, K_l, V_l, Q_l, nq_l = [], [], [], [], [], []
    for s in seqs:
        T, n = int(end[s]), int(n_q[s])
        kinds = np.asarray(w.prompt_kinds[s][:T], dtype=np.uint8)
        K, V = kv_bits(w, layer, s, T, heads)
        t = np.arange(T - n, T, dtype=np.int32)
        Q = synth.fill_tokens_host(w.seed, w.dtype, synth.scale_for(w.q_sigma), synth.tag(synth.Q_TENSOR, layer), t,
                                   np.full(n, s, np.int32), w.H, w.d)
        kinds_l.append(kinds)
        pos_l.append(tied_positions(kinds))
        K_l.append(K)
        V_l.append(V)
        Q_l.append(Q if heads is None else Q[:, heads])
        nq_l.append(n)
    return masked_prefill(kinds_l, pos_l, K_l, V_l, nq_l, np.concatenate(Q_l), w.dtype, w.scale, rot=w.rotary_dim,
                          base=w.rope_base, policy=policy, n_threads=n_threads)
