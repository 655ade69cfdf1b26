"""Parity at the workloads' full sizes, in the launch configuration the benchmark times: compaction
metadata of every sequence bit-exact, sampled cache rows bit-exact, and sampled decode outputs
(layers first/middle/last, sequences first/middle/last, every head) within tolerance of the fp64
oracle at the first step, right after compactions and at the last step checked."""
import numpy as np
import pytest
import torch

import harness
import oracle.workload as ow
from synth import workloads as wl

from _parity import check_metadata, check_rows, compare

pytestmark = pytest.mark.gpu


def _full(w, steps, check_at, rope=False):
    run = harness.Runner(w, steps)
    run.load_prompt()
    check_metadata(run, 0)
    seqs = sorted({0, w.b // 2, w.b - 1})
    layers = sorted({0, w.M // 2, w.M - 1})
    for s in seqs:
        check_rows(run, 0, layers[-1], s, [0, w.H - 1], check_k=not rope)
    out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device=run.device)
    for g in range(steps):
        inp = run.make_step_inputs(g)
        closed = run.step(inp, out)
        if g in check_at:
            torch.cuda.synchronize()
            o = out.cpu().numpy()
            for m in layers:
                ref = ow.expected_decode(w, g + 1, m, seqs)
                compare(o[m][seqs], ref, f"{w.name} step {g} layer {m}")
        if closed:
            check_metadata(run, g + 1)
    assert run.cache.device_status() == 0
    return run


def test_full_opt13b_shaped():
    # 128 steps as in the workload: compactions after g = 32, 65, 98
    _full(wl.opt13b(), 128, check_at={0, 1, 32, 33, 34, 66, 127})


def test_full_opt27b_shaped():
    _full(wl.opt27b(), 64, check_at={0, 7, 8, 52, 53, 63})


@pytest.mark.parametrize("interior", [19, 32, 45])
def test_full_rope3b_shaped(interior):
    # all 128 steps of the workload: the query positions run up to 2048 + 127 over the full cache
    _full(wl.rope3b(interior), 128, check_at={0, 64, 127}, rope=True)


# --------------------------------------------------------------------------
# The capacity / throughput sweep's shapes (Sec. 4.3, App. C): RedPajama-3B-shaped caches (H = 32,
# d_head = 80, fp16, RoPE), an 800-token prefix at r = 0.9 with the <CL> at offset 0 of every
# 64-token block, ingested with write-time freeing, and the sweep's largest batch, b = 4096: 131,072
# (sequence, head) segments per layer.  Two layers stand for the model's 32 (layers are independent
# and processed identically); the bench's step calls decode all of them in one launch.
# --------------------------------------------------------------------------

def _sweep_run(w, steps, seqs, rng):
    kept = [int(w.prompt_len[s]) - sum(c - a for a, c in w.prompt_spans[s]) for s in range(w.b)]
    run = harness.Runner(w, steps, capacity=np.asarray(kept, np.int64) + steps)
    run.load_prompt(mode="free")
    assert int(run.cache.lengths()[0].sum()) == sum(kept)
    out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device=run.device)
    plans = []
    for g in range(steps):
        inp = run.make_step_inputs(g)
        out.fill_(float("nan"))
        run.step(inp, out)
        plans.append(run.cache.last_decode_plan)
        torch.cuda.synchronize()
        o = out.cpu().numpy()
        assert np.all(np.isfinite(o))
        if g in (0, steps - 1):
            for m in range(w.M):
                compare(o[m][seqs], ow.expected_decode(w, g + 1, m, seqs), f"{w.name} step {g} layer {m}")
    assert run.cache.device_status() == 0
    return run, plans


def test_capacity_sweep_shapes_b4096():
    w = wl.throughput_3b(0.9, b=4096, M=2, steps=4)
    rng = np.random.default_rng(9)
    seqs = sorted({0, 1, 2047, 4095, *rng.integers(0, 4096, size=6).tolist()})
    run, plans = _sweep_run(w, 4, seqs, rng)
    # balanced segments: several whole segments per warp, both layers in one launch
    assert all(p["mode"] == 3 for p in plans), plans


def test_capacity_sweep_shapes_b4096_unbalanced_stream_k():
    """The same cache with one sequence's prefix ten times longer: the segments are unbalanced, so each
    layer's rows are split evenly over a full wave of warps (stream-K).  Every warp then covers dozens
    of whole segments plus split pieces at both ends, and the long sequence's segments are split over
    several warps and merged by the log-sum-exp combine."""
    import dataclasses

    w = wl.throughput_3b(0.9, b=4096, M=1, steps=3)
    k_long, s_long = wl.block_kinds(8000, 58, cl_off=0)
    kinds = list(w.prompt_kinds)
    spans = list(w.prompt_spans)
    kinds[1], spans[1] = k_long, s_long
    w = dataclasses.replace(w, prompt_kinds=kinds, prompt_spans=spans, name="throughput3b_r0.90_long1")
    rng = np.random.default_rng(10)
    seqs = sorted({0, 1, 2, 4095, *rng.integers(0, 4096, size=6).tolist()})
    run, plans = _sweep_run(w, 3, seqs, rng)
    assert all(p["mode"] == 0 for p in plans), plans
    rows = int(run.attended_rows().sum()) * w.H
    assert rows // plans[-1]["workers"] > 20 * 110  # dozens of ~100-row segments per warp


def test_full_ragged():
    w = wl.ragged()
    run = _full(w, 32, check_at={0, 15, 31})
    # the benchmark's launch configuration: every layer in one launch, whole segments cut by rows
    assert run.cache.last_decode_plan["mode"] == 4, run.cache.last_decode_plan
    ln = run.cache.lengths()[0]
    assert ln.max() > 3000 and ln.min() < 400  # ragged: lengths span more than an order of magnitude


# --------------------------------------------------------------------------
# Masked prefill at the workloads' full sizes: whole prompts (OPT-1.3B, 3B rotary, OPT-2.7B shapes
# and the ragged prompts), in one go and in blocks of 512 tokens, every layer prefilled as the bench
# times it; sampled queries (block edges, <CL>/<CR> tokens, random) of three layers, three
# sequences and two heads against the oracle's single-query attention over the mask.
# --------------------------------------------------------------------------

@pytest.mark.parametrize("name,block", [("opt1.3b", 0), ("opt1.3b", 512), ("rope3b_I32", 0), ("rope3b_I32", 512),
                                        ("opt2.7b", 0), ("opt2.7b", 512), ("ragged", 512)])
def test_full_prefill(name, block):
    """d_head 64 (OPT-1.3B shape), d_head 80 with RoPE (3B rotary shape, r = 0.5), d_head 80 in bf16
    (OPT-2.7B shape: the rotated query and P go to the tensor cores as high and low bf16 parts) and
    the ragged prompts (b = 128, 256-8192 tokens), in one go and in blocks of 512 tokens; only the
    sampled sequences' outputs are read back."""
    import oracle as orc

    w = wl.by_name(name)
    layers, seqs, heads = {0, w.M // 2, w.M - 1}, [0, w.b // 2, w.b - 1], [0, w.H - 1]
    run = harness.Runner(w, 0)
    got = []

    def keep(start, n, m, out):
        if m in layers:
            row0 = np.concatenate([[0], np.cumsum(n)[:-1]])
            sel = {s: out[int(row0[s]):int(row0[s] + n[s])][:, heads].cpu().numpy() for s in seqs}
            got.append((start.copy(), n.copy(), m, sel))

    run.prefill_prompt(block=block, out_cb=keep)
    assert run.cache.device_status() == 0
    rng = np.random.default_rng(block + 1)
    n_checked = 0
    for start, n, m, sel in got:
        for s in seqs:
            if n[s] == 0:  # a ragged prompt that ended in an earlier block
                continue
            T = int(start[s] + n[s])
            kinds = np.asarray(w.prompt_kinds[s][:T], np.uint8)
            pos = orc.tied_positions(kinds)
            K, V = ow.kv_bits(w, m, s, T, heads)
            lo = int(start[s])
            special = [t for t in range(lo, T) if kinds[t] != 0][:6]
            ts = sorted({lo, T - 1, *special, *rng.integers(lo, T, size=8).tolist()})
            for t in ts:
                rows = np.nonzero(orc.visible(kinds[:t + 1], t))[0]
                q = ow.q_bits(w, m, s, t, heads)
                ref = np.stack([orc.attend(q[i], K[i], V[i], pos, rows, w.dtype, w.scale, w.rotary_dim, w.rope_base,
                                           int(pos[t])) for i in range(len(heads))])
                compare(sel[s][t - lo], ref, f"{name} prefill block={block} layer {m} seq {s} token {t}")
                n_checked += 1
    assert n_checked > 100
