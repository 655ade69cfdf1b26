"""Helpers shared by the GPU parity tests (not collected by pytest)."""
from __future__ import annotations

import numpy as np
import torch

import harness
import oracle as orc
import oracle.workload as ow
import paper_2310_08152_gb300 as kvc
import synth

# Tolerance for fp16/bf16 K/V with fp32 accumulation against the fp64 oracle.
MAX_ABS = 2e-3
MAX_REL = 1e-2
REL_FLOOR = 0.2  # |ref| below this is governed by the absolute bound (MAX_ABS / MAX_REL)


def compare(got: np.ndarray, ref: np.ndarray, what: str = ""):
    got = np.asarray(got, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - ref)
    max_abs = float(err.max())
    max_rel = float((err / np.maximum(np.abs(ref), REL_FLOOR)).max())
    assert max_abs <= MAX_ABS and max_rel <= MAX_REL, f"{what}: max_abs={max_abs:.3g} max_rel={max_rel:.3g}"
    return max_abs, max_rel


def check_metadata(run: harness.Runner, steps_done: int, seqs=None, policy=orc.POLICY_PAPER):
    """Stored rows of each sequence (history index, position, count) read back from the device equal the
    oracle's rows left after freeing the spans freed so far -- bit-exact."""
    w = run.w
    seqs = range(w.b) if seqs is None else seqs
    ln = run.cache.lengths()[0]
    for s in seqs:
        kinds, pos = ow.history(w, s, steps_done)
        freed = _freed_spans(run, s, kinds)
        rows = orc.stored_rows(kinds.size, freed, policy)
        lay = run.cache.masked_reference_layout(s)
        assert np.array_equal(lay["kinds"], kinds)
        assert np.array_equal(lay["pos"], pos)
        assert ln[s] == rows.size, (s, ln[s], rows.size)
        assert np.array_equal(lay["stored_orig"], rows.astype(np.int32)), f"seq {s}: stored history indices"
        assert np.array_equal(lay["stored_pos"], pos[rows]), f"seq {s}: stored positions"


def _freed_spans(run, s, kinds):
    # the harness frees every span right after its <CR> step, and every prompt span after the prompt
    closed, _ = orc.pair_spans(kinds)
    return closed


def check_rows(run: harness.Runner, steps_done: int, layer: int, s: int, heads, check_k: bool = True):
    """Cache rows of (layer, s, h) equal the generator's values of the stored history tokens, bit-exact."""
    w = run.w
    lay = run.cache.masked_reference_layout(s)
    orig = lay["stored_orig"]
    T = int(orig.max()) + 1 if orig.size else 0
    K, V = ow.kv_bits(w, layer, s, T)
    n = orig.size
    kp = run.cache.k_plane(layer)
    vp = run.cache.v_plane(layer)
    for h in heads:
        v_dev = run.cache.stream_rows(vp, s, h, n).cpu().view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(v_dev, V[h][orig]), f"V rows (layer {layer}, seq {s}, head {h})"
        if check_k:
            k_dev = run.cache.stream_rows(kp, s, h, n).cpu().view(torch.int16).numpy().view(np.uint16)
            assert np.array_equal(k_dev, K[h][orig]), f"K rows (layer {layer}, seq {s}, head {h})"


def run_workload(w, steps: int, policy=orc.POLICY_PAPER, layers=None, seqs=None, heads=None, check_steps=None,
                 meta_every_compaction: bool = True):
    """Prompt + `steps` decode steps; compare decode outputs with the oracle at the chosen steps."""
    run = harness.Runner(w, steps, policy)
    run.load_prompt()
    check_metadata(run, 0, policy=policy)
    out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device=run.device)
    layers = range(w.M) if layers is None else layers
    seqs = list(range(w.b)) if seqs is None else list(seqs)
    worst = (0.0, 0.0)
    for g in range(steps):
        inp = run.make_step_inputs(g)
        out.fill_(float("nan"))
        closed = run.step(inp, out)
        if check_steps is None or g in check_steps or len(closed) or (inp.kinds != 0).any():
            torch.cuda.synchronize()
            o = out.cpu().numpy()
            for m in layers:
                ref = ow.expected_decode(w, g + 1, m, seqs, heads, policy)
                got = o[m][seqs] if heads is None else o[m][seqs][:, heads]
                a, r = compare(got, ref, f"{w.name} step {g} layer {m}")
                worst = (max(worst[0], a), max(worst[1], r))
        if closed and meta_every_compaction:
            check_metadata(run, g + 1, policy=policy)
    assert run.cache.device_status() == 0
    return run, worst
