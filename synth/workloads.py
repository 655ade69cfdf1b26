"""Workload recipes: shapes and sentinel structure of the synthetic caches.

No dataset or trained weight is available, so seeded synthetic inputs stand in
for the paper's WikiText-2 / C4 / WritingPrompts runs on OPT-1.3B, OPT-2.7B and
RedPajama-3B (paper Sec. 4).  A recipe fixes the cache shape (M layers, H heads,
d_head, batch b), the token kinds of every prompt and of every generated token
(NORMAL, <CL>, <CR>), and the K/V/q value distributions.  It contains no
position, mask, attention or compaction arithmetic.

Token-kind geometry of the periodic recipes: in every 64-token block k of a
prompt, <CL> sits at 64k+7, the I enclosed tokens at [64k+8, 64k+8+I) and
<CR> at 64k+8+I, so a prompt of L tokens encloses I/64 of its tokens (the
paper's compression ratio r, Sec. 3.1 "Input Transformation").

The ragged recipe follows the paper's span sampler (Sec. 3.1: spans drawn
repeatedly, lengths uniform, no overlap, until ratio r is reached) with
interior lengths U[8, 64] and r = 0.5.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Callable, List, Tuple

import numpy as np

NORMAL, CL, CR = 0, 1, 2
SEED_BASE = 0xC0FFEE


def block_kinds(L: int, interior: int, cl_off: int = 7, period: int = 64):
    """Kinds and spans of a prompt with one <CL>..<CR> pair per ``period`` tokens."""
    kinds = np.zeros(L, dtype=np.uint8)
    spans = []
    for k in range(L // period + 1):
        cl = period * k + cl_off
        cr = cl + 1 + interior
        if cr >= L:
            break
        kinds[cl] = CL
        kinds[cr] = CR
        spans.append((cl, cr))
    return kinds, spans


def sampled_kinds(L: int, ratio: float, lo: int, hi: int, rng: np.random.Generator, max_tries: int = 200000):
    """Non-overlapping spans with interior length ~ U[lo, hi] at random offsets until ``ratio`` of L is enclosed."""
    kinds = np.zeros(L, dtype=np.uint8)
    taken = np.zeros(L, dtype=bool)
    spans = []
    enclosed = 0
    target = ratio * L
    tries = 0
    while enclosed < target and tries < max_tries:
        tries += 1
        interior = int(rng.integers(lo, hi + 1))
        if interior + 2 > L:
            continue
        cl = int(rng.integers(0, L - interior - 1))
        cr = cl + 1 + interior
        if taken[cl:cr + 1].any():
            continue
        taken[cl:cr + 1] = True
        kinds[cl] = CL
        kinds[cr] = CR
        spans.append((cl, cr))
        enclosed += interior
    spans.sort()
    return kinds, spans


@dataclass
class Workload:
    name: str
    index: int
    M: int
    H: int
    d: int
    dtype: str
    b: int
    prompt_kinds: List[np.ndarray]
    prompt_spans: List[List[Tuple[int, int]]]
    n_steps: int
    gen_kind: Callable[[int, int], int]
    scale: float
    q_sigma: float = 1.0
    kv_sigma: float = 1.0
    rotary_dim: int = 0
    rope_base: float = 10000.0
    seed: int = SEED_BASE
    note: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def prompt_len(self) -> np.ndarray:
        return np.array([k.size for k in self.prompt_kinds], dtype=np.int64)

    def capacity(self, steps: int) -> np.ndarray:
        return self.prompt_len + int(steps)

    def gen_kinds(self, steps: int) -> np.ndarray:
        """[steps, b] kinds of the generated tokens."""
        return np.array([[self.gen_kind(s, g) for s in range(self.b)] for g in range(steps)], dtype=np.uint8)

    def kinds_history(self, s: int, steps: int) -> np.ndarray:
        gk = np.array([self.gen_kind(s, g) for g in range(steps)], dtype=np.uint8)
        return np.concatenate([self.prompt_kinds[s], gk])

    def gen_spans(self, s: int, steps: int):
        """(cl, cr) orig indices of spans opened and closed within the first ``steps`` generated tokens."""
        L = self.prompt_kinds[s].size
        out = []
        open_cl = None
        for g in range(steps):
            k = self.gen_kind(s, g)
            if k == CL:
                open_cl = L + g
            elif k == CR:
                out.append((open_cl, L + g))
                open_cl = None
        return out

    def kv_bytes_per_token(self) -> int:
        return self.M * 2 * self.H * self.d * 2


def _periodic_gen(cl_at: int, cr_at: int, period: int):
    def f(s: int, g: int) -> int:
        r = g % period
        if r == cl_at:
            return CL
        if r == cr_at:
            return CR
        return NORMAL

    return f


def _normal_gen(s: int, g: int) -> int:
    return NORMAL


def tiny() -> Workload:
    kinds, spans = block_kinds(512, 32)
    return Workload("tiny", 0, M=1, H=4, d=64, dtype="f16", b=2, prompt_kinds=[kinds.copy(), kinds.copy()],
                    prompt_spans=[list(spans), list(spans)], n_steps=1, gen_kind=_normal_gen,
                    scale=1.0 / math.sqrt(64), seed=SEED_BASE + 0,
                    note="1 layer, b=2, H=4, d=64, L=512, spans [64k+8, 64k+40)")


def opt13b(b: int = 16, L: int = 2048, M: int = 24) -> Workload:
    kinds, spans = block_kinds(L, 32)
    return Workload("opt1.3b", 1, M=M, H=32, d=64, dtype="f16", b=b, prompt_kinds=[kinds.copy() for _ in range(b)],
                    prompt_spans=[list(spans) for _ in range(b)], n_steps=128, gen_kind=_periodic_gen(0, 32, 33),
                    scale=1.0 / math.sqrt(64), seed=SEED_BASE + 1,
                    note=f"OPT-1.3B-shaped: M={M}, H=32, d=64, fp16, b={b}, L={L}, 32 enclosed per 64; "
                         "generated: <CL> at g%33==0, <CR> at g%33==32")


def opt13b_uncompressed(b: int = 16, L: int = 2048, M: int = 24) -> Workload:
    """The OPT-1.3B-shaped cache with no sentinel spans (r = 0): every token is kept.  Used as the
    reference point for DRAM traffic scaling with the compressed length."""
    kinds = np.zeros(L, dtype=np.uint8)
    return Workload("opt1.3b_r0", 1, M=M, H=32, d=64, dtype="f16", b=b, prompt_kinds=[kinds.copy() for _ in range(b)],
                    prompt_spans=[[] for _ in range(b)], n_steps=128, gen_kind=_normal_gen,
                    scale=1.0 / math.sqrt(64), seed=SEED_BASE + 1,
                    note=f"OPT-1.3B-shaped, no spans (r=0): M={M}, H=32, d=64, fp16, b={b}, L={L}")


def opt13b_local(ratio: float = 0.5, b: int = 16, L: int = 2048, M: int = 24) -> Workload:
    """The paper's Local Attention baseline (Sec. 4.1; FIFO queue at inference, Sec. 4.2) on the
    OPT-1.3B-shaped cache: no sentinels, each token attends within a window of ~(1 - r) of its
    history.  At r = 0.5 it keeps as many rows as the compressed cache with 32 of 64 tokens enclosed."""
    kinds = np.zeros(L, dtype=np.uint8)
    w = Workload(f"opt1.3b_local{ratio:g}", 1, M=M, H=32, d=64, dtype="f16", b=b,
                 prompt_kinds=[kinds.copy() for _ in range(b)], prompt_spans=[[] for _ in range(b)], n_steps=128,
                 gen_kind=_normal_gen, scale=1.0 / math.sqrt(64), seed=SEED_BASE + 1,
                 note=f"OPT-1.3B-shaped Local Attention FIFO cache (r={ratio:g}): M={M}, H=32, d=64, fp16, b={b}, "
                      f"L={L}")
    w.extra = {"policy": "local", "local_ratio": ratio}
    return w


def opt27b(b: int = 32, L: int = 4096, M: int = 32) -> Workload:
    kinds, spans = block_kinds(L, 44)
    return Workload("opt2.7b", 2, M=M, H=32, d=80, dtype="bf16", b=b, prompt_kinds=[kinds.copy() for _ in range(b)],
                    prompt_spans=[list(spans) for _ in range(b)], n_steps=64, gen_kind=_periodic_gen(7, 52, 64),
                    scale=1.0, q_sigma=1.0 / math.sqrt(80), seed=SEED_BASE + 2,
                    note=f"OPT-2.7B-shaped: M={M}, H=32, d=80, bf16, b={b}, L={L}, 44 enclosed per 64; "
                         "q std d^-1/2 with softmax scale 1; generated: one span per 64 steps")


def rope3b(interior: int = 32, b: int = 64, L: int = 2048, M: int = 32) -> Workload:
    assert interior in (19, 32, 45) or True
    kinds, spans = block_kinds(L, interior)
    r = interior / 64.0
    return Workload(f"rope3b_I{interior}", 3, M=M, H=32, d=80, dtype="f16", b=b,
                    prompt_kinds=[kinds.copy() for _ in range(b)], prompt_spans=[list(spans) for _ in range(b)],
                    n_steps=128, gen_kind=_normal_gen, scale=1.0 / math.sqrt(80), rotary_dim=80, rope_base=10000.0,
                    seed=SEED_BASE + 3,
                    note=f"3B rotary-shaped: M={M}, H=32, d=80, fp16, RoPE base 1e4 on K at write and q at its "
                         f"position, b={b}, L={L}, {interior} enclosed per 64 (r={r:.2f})")


def ragged(b: int = 128, lmin: int = 256, lmax: int = 8192, M: int = 24, steps: int = 32) -> Workload:
    seed = SEED_BASE + 4
    rng = np.random.default_rng(seed)
    lens = rng.integers(lmin, lmax + 1, size=b)
    kinds, spans = [], []
    for s in range(b):
        k, sp = sampled_kinds(int(lens[s]), 0.5, 8, 64, rng)
        kinds.append(k)
        spans.append(sp)
    opens = rng.integers(0, 16, size=b)
    gaps = rng.integers(8, 16, size=b)

    def gen(s: int, g: int) -> int:
        if g == opens[s]:
            return CL
        if g == opens[s] + gaps[s]:
            return CR
        return NORMAL

    return Workload("ragged", 4, M=M, H=32, d=64, dtype="f16", b=b, prompt_kinds=kinds, prompt_spans=spans,
                    n_steps=steps, gen_kind=gen, scale=1.0 / math.sqrt(64), seed=seed,
                    note=f"ragged stress: M={M}, H=32, d=64, fp16, b={b}, L_s ~ U[{lmin},{lmax}], sampled spans "
                         "U[8,64] to r=0.5; each sequence opens <CL> at a step in [0,16) and closes 8-15 steps later",
                    extra={"opens": opens, "gaps": gaps})


def throughput_3b(ratio: float, b: int, prefix: int = 800, M: int = 32, steps: int = 64) -> Workload:
    """The paper's throughput setting (Sec. 4.3): RedPajama-3B shapes (M=32, H=32, d=80, fp16, RoPE),
    a dummy prefix of 800 tokens transformed to compression ratio r, then normal generated tokens.
    Spans: one <CL>..<CR> pair per 64-token block, <CL> first, round(64 r) enclosed tokens."""
    interior = int(round(64 * ratio))
    if interior == 0:
        kinds, spans = np.zeros(prefix, dtype=np.uint8), []
    else:
        assert interior + 2 <= 64, "r too high for one span per 64-token block"
        kinds, spans = block_kinds(prefix, interior, cl_off=0)
    return Workload(f"throughput3b_r{ratio:.2f}", 3, M=M, H=32, d=80, dtype="f16", b=b,
                    prompt_kinds=[kinds.copy() for _ in range(b)], prompt_spans=[list(spans) for _ in range(b)],
                    n_steps=steps, gen_kind=_normal_gen, scale=1.0 / math.sqrt(80), rotary_dim=80,
                    rope_base=10000.0, seed=SEED_BASE + 5,
                    note=f"3B rotary shapes, prefix {prefix} at r={ratio:.2f} ({interior} enclosed per 64), b={b}")


def by_name(name: str, **kw) -> Workload:
    table = {"tiny": tiny, "opt1.3b": opt13b, "opt1.3b_r0": opt13b_uncompressed, "opt2.7b": opt27b,
             "ragged": ragged, "opt1.3b_local0.5": opt13b_local}
    if name.startswith("rope3b"):
        interior = int(name.split("_I")[1]) if "_I" in name else 32
        return rope3b(interior=interior, **kw)
    return table[name](**kw)
