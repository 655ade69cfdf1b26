"""Runs a synthetic workload (synth.workloads) through the CUDA path.

Shared by the GPU tests, ``__graft_entry__.smoke`` and ``bench.py``.  Inputs come
from the device build of the seeded generator, so tens of GB of K/V never cross
the host link.  Counter conventions (also used by the oracle side): K and V of
history token t of sequence s use counters (i0=t, i1=s) with tag (K|V, layer);
the query of layer m at history token t uses tag (q, m) and (i0=t, i1=s).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import numpy as np
import torch

import paper_2310_08152_gb300 as kvc
import synth
from synth import workloads as wl


@dataclass
class StepInputs:
    kinds: np.ndarray            # [b] uint8
    kv_k: torch.Tensor           # [M][b][H][d]
    kv_v: torch.Tensor           # [M][b][H][d]
    q: torch.Tensor              # [M][b][H][d]


class Runner:
    def __init__(self, w: wl.Workload, steps: int, policy: int = kvc.POLICY_PAPER, device=None,
                 capacity_slack: int = 0, capacity=None, local_ratio: float = 0.0):
        if w.extra.get("policy") == "local":  # the workload names its own cache policy
            policy, local_ratio = kvc.POLICY_LOCAL, w.extra["local_ratio"]
        self.w = w
        self.steps = steps
        self.policy = policy
        self.device = torch.device("cuda", 0) if device is None else torch.device(device)
        self.tdt = torch.float16 if w.dtype == "f16" else torch.bfloat16
        cap = (w.capacity(steps) if capacity is None else np.asarray(capacity, np.int64)) + capacity_slack
        if policy == kvc.POLICY_LOCAL and capacity is None:
            # a ring holding the largest window the run reaches: x_t sees (floor(t r), t]
            T = w.prompt_len + steps
            cap = T - np.floor(T * np.float64(np.float32(local_ratio))).astype(np.int64) + capacity_slack
        self.cache = kvc.KVCache(w.M, w.H, w.d, cap, w.dtype, w.rotary_dim, w.rope_base, policy, device=self.device,
                                 local_ratio=local_ratio)
        self.L = w.prompt_len.copy()
        self.open_cl = [-1] * w.b      # history index of an open <CL>
        self.g = 0                      # generated tokens so far
        self.kv_scale = synth.scale_for(w.kv_sigma)
        self.q_scale = synth.scale_for(w.q_sigma)

    # ---------------------------------------------------------------------------------------
    def _fill(self, tensor_kind: int, layer: int, tok_t: torch.Tensor, tok_s: torch.Tensor, out: torch.Tensor,
              scale) -> torch.Tensor:
        synth.fill_tokens_cuda(self.w.seed, self.w.dtype, scale, synth.tag(tensor_kind, layer), tok_t, tok_s,
                               self.w.H, self.w.d, out)
        return out

    def load_prompt(self, compress: bool = True, stream=None, mode: str = "compact", block: int = 0, timer=None):
        """Append every prompt layer by layer and free the prompt spans (Sec. 3.1).

        mode "compact": append all tokens, then free every span with one compaction ("in one go").
        mode "free": append with write-time freeing -- spans inside the prompt are never stored.
        mode "progressive": append `block` tokens per sequence at a time with write-time freeing, and
        after each block compact the spans that straddled blocks (the paper's for-loop over blocks).
        """
        w = self.w
        if mode == "compact":
            self._append_tokens(np.zeros(w.b, np.int64), self.L.astype(np.int64), False, stream, timer)
            if compress:
                self.compress_prompt(stream)
            return
        if mode == "free":
            self._append_tokens(np.zeros(w.b, np.int64), self.L.astype(np.int64), True, stream, timer)
            return
        assert mode == "progressive" and block > 0
        start = np.zeros(w.b, np.int64)
        while (start < self.L).any():
            n = np.minimum(self.L - start, block)
            self._append_tokens(start, n, True, stream, timer)
            start = start + n
            seq, cl, cr = [], [], []
            for s in range(w.b):
                for a, c in self.cache.pending_spans(s):
                    seq.append(s)
                    cl.append(a)
                    cr.append(c)
            if seq:
                self.cache.compress_spans(seq, cl, cr, stream)

    def _append_tokens(self, start, n, free_closed: bool, stream=None, timer=None):
        """Prompt tokens [start[s], start[s] + n[s]) of every sequence, layer by layer.  timer: a list
        that receives a (start, end) CUDA event pair around every append call."""
        w = self.w
        n_new = n.astype(np.int32)
        kinds = np.concatenate([w.prompt_kinds[s][start[s]:start[s] + n[s]] for s in range(w.b)]).astype(np.uint8)
        N = int(n_new.sum())
        if N == 0:
            return
        tok_t = torch.from_numpy(np.concatenate([np.arange(start[s], start[s] + n[s], dtype=np.int32)
                                                 for s in range(w.b)])).to(self.device)
        tok_s = torch.from_numpy(np.repeat(np.arange(w.b, dtype=np.int32), n)).to(self.device)
        kbuf = torch.empty(N * w.H * w.d, dtype=self.tdt, device=self.device)
        vbuf = torch.empty_like(kbuf)
        append = kvc.kvc_append_free_closed if free_closed else kvc.kvc_append
        for m in range(w.M):
            self._fill(synth.K_TENSOR, m, tok_t, tok_s, kbuf, self.kv_scale)
            self._fill(synth.V_TENSOR, m, tok_t, tok_s, vbuf, self.kv_scale)
            if timer is not None:
                ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                ev[0].record(stream)
            if m == 0:
                pos = self.cache.book.next_positions(n_new, kinds)
                append(self.cache.handle, 0, kbuf, vbuf, n_new, pos, kinds, stream)
            else:
                append(self.cache.handle, m, kbuf, vbuf, None, None, None, stream)
            if timer is not None:
                ev[1].record(stream)
                timer.append(ev)
        del kbuf, vbuf

    def prefill_prompt(self, block: int = 0, stream=None, out_cb=None, layers=None, events=None):
        """Prompt ingestion with masked prefill attention (Sec. 3.1): per block of `block` tokens of
        every sequence (0: the whole prompt in one go), append the block's K/V layer by layer, run the
        prefill of that layer's queries (the block's tokens) over the stored rows, and once every layer
        is written free the spans closed so far -- the paper's for-loop over blocks.

        out_cb(start, n, layer, out): receives each prefilled layer's output, fp32 [sum n, H, d]
        (sequence-major).  events: a list that receives a (start, end) CUDA event pair around each
        prefill call."""
        w = self.w
        start = np.zeros(w.b, np.int64)
        while (start < self.L).any():
            n = self.L - start if block <= 0 else np.minimum(self.L - start, block)
            self._prefill_block(start, n, stream, out_cb, layers, events)
            start = start + n
            seq, cl, cr = [], [], []
            for s in range(w.b):
                for a, c in self.cache.pending_spans(s):
                    seq.append(s)
                    cl.append(a)
                    cr.append(c)
            if seq:
                self.cache.compress_spans(seq, cl, cr, stream)

    def _prefill_block(self, start, n, stream, out_cb, layers, events):
        w = self.w
        n_new = n.astype(np.int32)
        kinds = np.concatenate([w.prompt_kinds[s][start[s]:start[s] + n[s]] for s in range(w.b)]).astype(np.uint8)
        N = int(n_new.sum())
        tok_t = torch.from_numpy(np.concatenate([np.arange(start[s], start[s] + n[s], dtype=np.int32)
                                                 for s in range(w.b)])).to(self.device)
        tok_s = torch.from_numpy(np.repeat(np.arange(w.b, dtype=np.int32), n)).to(self.device)
        kbuf = torch.empty(N * w.H * w.d, dtype=self.tdt, device=self.device)
        vbuf = torch.empty_like(kbuf)
        qbuf = torch.empty_like(kbuf)
        out = torch.empty(N, w.H, w.d, dtype=torch.float32, device=self.device)
        for m in range(w.M):
            self._fill(synth.K_TENSOR, m, tok_t, tok_s, kbuf, self.kv_scale)
            self._fill(synth.V_TENSOR, m, tok_t, tok_s, vbuf, self.kv_scale)
            if m == 0:
                pos = self.cache.book.next_positions(n_new, kinds)
                kvc.kvc_append(self.cache.handle, 0, kbuf, vbuf, n_new, pos, kinds, stream)
            else:
                kvc.kvc_append(self.cache.handle, m, kbuf, vbuf, None, None, None, stream)
            if layers is not None and m not in layers:
                continue
            self._fill(synth.Q_TENSOR, m, tok_t, tok_s, qbuf, self.q_scale)
            if events is not None:
                ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                ev[0].record(stream)
            kvc.kvc_prefill_attention(self.cache.handle, m, qbuf, n_new, w.scale, out, stream)
            if events is not None:
                ev[1].record(stream)
                events.append(ev)
            if out_cb is not None:
                out_cb(start, n, m, out)

    def compress_prompt(self, stream=None):
        seq, cl, cr = [], [], []
        for s in range(self.w.b):
            for a, c in self.w.prompt_spans[s]:
                seq.append(s)
                cl.append(a)
                cr.append(c)
        if seq:
            self.cache.compress_spans(seq, cl, cr, stream)

    # ---------------------------------------------------------------------------------------
    def make_step_inputs(self, g: int) -> StepInputs:
        """Inputs of generated token g: its K/V rows (all layers) and the queries of all layers."""
        w = self.w
        kinds = np.array([w.gen_kind(s, g) for s in range(w.b)], dtype=np.uint8)
        tok_t = torch.from_numpy((self.L + g).astype(np.int32)).to(self.device)
        tok_s = torch.arange(w.b, dtype=torch.int32, device=self.device)
        shape = (w.M, w.b, w.H, w.d)
        k = torch.empty(shape, dtype=self.tdt, device=self.device)
        v = torch.empty(shape, dtype=self.tdt, device=self.device)
        q = torch.empty(shape, dtype=self.tdt, device=self.device)
        for m in range(w.M):
            self._fill(synth.K_TENSOR, m, tok_t, tok_s, k[m], self.kv_scale)
            self._fill(synth.V_TENSOR, m, tok_t, tok_s, v[m], self.kv_scale)
            self._fill(synth.Q_TENSOR, m, tok_t, tok_s, q[m], self.q_scale)
        return StepInputs(kinds, k, v, q)

    def step_spans(self, kinds: np.ndarray):
        """Spans closed by this step's tokens (to free right after the step's decode)."""
        seq, cl, cr = [], [], []
        for s in range(self.w.b):
            t = int(self.L[s]) + self.g
            if kinds[s] == wl.CL:
                self.open_cl[s] = t
            elif kinds[s] == wl.CR:
                seq.append(s)
                cl.append(self.open_cl[s])
                cr.append(t)
                self.open_cl[s] = -1
        return seq, cl, cr

    def append_only(self, inp: StepInputs, stream=None):
        """The first part of a step: append the token's K/V rows of every layer (decode follows)."""
        self.cache.append(inp.kv_k, inp.kv_v, np.ones(self.w.b, dtype=np.int32), inp.kinds, layer=-1,
                          stream=kvc.stream_handle(stream))

    def finish_step(self, inp: StepInputs, stream=None):
        """The last part of a step after its decode: free the span the token closed, if any."""
        seq, cl, cr = self.step_spans(inp.kinds)
        self.g += 1
        if seq:
            self.cache.compress_spans(seq, cl, cr, kvc.stream_handle(stream))
        return seq

    def step(self, inp: StepInputs, out: torch.Tensor, stream=None, events=None, compress: bool = True):
        """One decode step: append the token, decode all M layers into out[M][b][H][d], free closed spans.

        events: optional list of (start, end) CUDA event pairs, one per layer, recorded around each decode."""
        w = self.w
        n_new = np.ones(w.b, dtype=np.int32)
        sh = kvc.stream_handle(stream)  # resolved once: every call of the step goes on this stream
        self.cache.append(inp.kv_k, inp.kv_v, n_new, inp.kinds, layer=-1, stream=sh)
        if events is None:  # all layers in one call
            n = w.b * w.H * w.d
            kvc.kvc_decode_attention_layers(self.cache.handle, 0, w.M, inp.q, n, w.scale, out, n, sh)
        else:
            for m in range(w.M):
                events[m][0].record(stream)
                kvc.kvc_decode_attention(self.cache.handle, m, inp.q[m], w.scale, out[m], sh)
                events[m][1].record(stream)
        seq, cl, cr = self.step_spans(inp.kinds)
        self.g += 1
        if compress and seq:
            self.cache.compress_spans(seq, cl, cr, sh)
        return seq

    # ---------------------------------------------------------------------------------------
    def attended_rows(self) -> np.ndarray:
        """Rows the next decode reads per sequence."""
        return self.cache.lengths()[1]

    def decode_bytes(self) -> int:
        """Algorithmic bytes of one decode launch: kept K+V rows read, q read, out written."""
        w = self.w
        rows = int(self.attended_rows().sum())
        return 2 * rows * w.H * w.d * 2 + w.b * w.H * w.d * 2 + w.b * w.H * w.d * 4
