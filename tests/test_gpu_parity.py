"""Parity of the CUDA path (through the C ABI) with the fp64 oracle, at sizes the oracle finishes in
seconds: several tiles per segment, split segments, ragged tails, every step kind (normal, <CL>
query, open-span queries, <CR> query, compaction right after it), both policies, every built d_head."""
import dataclasses
import math

import numpy as np
import pytest
import torch

import harness
import oracle as orc
import oracle.workload as ow
import paper_2310_08152_gb300 as kvc
import synth
from synth import workloads as wl

from _parity import MAX_ABS, check_metadata, check_rows, compare, run_workload

pytestmark = pytest.mark.gpu


def test_device_generator_matches_host():
    rng = np.random.default_rng(1)
    for dtype, sigma in (("f16", 1.0), ("bf16", 80 ** -0.5)):
        t = rng.integers(0, 9000, size=300).astype(np.int32)
        s = rng.integers(0, 128, size=300).astype(np.int32)
        sc = synth.scale_for(sigma)
        tag = synth.tag(synth.V_TENSOR, 17)
        host = synth.fill_tokens_host(77, dtype, sc, tag, t, s, 5, 80)
        out = torch.empty(300 * 5 * 80, dtype=torch.int16, device="cuda")
        synth.fill_tokens_cuda(77, dtype, sc, tag, torch.from_numpy(t).cuda(), torch.from_numpy(s).cuda(), 5, 80, out)
        assert np.array_equal(out.cpu().numpy().view(np.uint16).reshape(300, 5, 80), host)


def test_tiny_config_every_output():
    run, worst = run_workload(wl.tiny(), steps=1)
    for s in range(2):
        check_rows(run, 1, 0, s, range(4))
    assert worst[0] <= MAX_ABS


def test_opt13b_shaped_small():
    # H=32, d=64, fp16: <CL> query at g=0 and 33, open-span queries, <CR> at g=32 then compaction
    w = wl.opt13b(b=3, L=640, M=2)
    run, _ = run_workload(w, steps=36)
    for s in range(3):
        check_rows(run, 36, 1, s, [0, 31])


def test_opt27b_shaped_small():
    # d=80, bf16, q std d^-1/2 with scale 1; span opened at g=7, closed at g=52
    w = wl.opt27b(b=3, L=704, M=2)
    run, _ = run_workload(w, steps=54, check_steps={0, 7, 8, 30, 51, 52, 53})
    check_rows(run, 54, 0, 2, [5])


@pytest.mark.parametrize("interior", [19, 32, 45])
def test_rope3b_shaped_small(interior):
    w = wl.rope3b(interior, b=3, L=640, M=2)
    run, _ = run_workload(w, steps=6)
    check_rows(run, 6, 1, 0, [3], check_k=False)  # K is stored rotated


def test_ragged_small():
    w = wl.ragged(b=6, lmin=64, lmax=900, M=2, steps=32)
    run_workload(w, steps=32, check_steps={0, 10, 20, 31})


def test_keep_cl_policy():
    w = wl.opt13b(b=2, L=384, M=1)
    run_workload(w, steps=35, policy=orc.POLICY_KEEP_CL)


@pytest.mark.parametrize("d,dtype", [(96, "f16"), (128, "bf16"), (64, "bf16"), (80, "f16")])
def test_every_built_head_dim(d, dtype):
    w = dataclasses.replace(wl.opt13b(b=2, L=448, M=2), d=d, dtype=dtype, name=f"d{d}-{dtype}")
    run_workload(w, steps=34, check_steps={0, 1, 31, 32, 33})


@pytest.mark.parametrize("d,rot", [(96, 96), (128, 64)])
def test_rope_other_head_dims(d, rot):
    # rotation of 6 / 4 vector pairs per head (d_head 96 whole, 128 half), four lanes per row
    w = dataclasses.replace(wl.rope3b(32, b=2, L=384, M=1), d=d, rotary_dim=rot, scale=1.0 / math.sqrt(d),
                            name=f"rope-d{d}-r{rot}")
    run, _ = run_workload(w, steps=3)
    check_rows(run, 3, 0, 0, [1], check_k=False)  # K is stored rotated


def test_rope_partial_rotary_dim():
    w = dataclasses.replace(wl.rope3b(32, b=2, L=384, M=1), rotary_dim=32, name="rope-partial")
    run_workload(w, steps=3)


def test_long_segments_split_over_many_ctas():
    # one long sequence and a short one: stream-K splits the long segments across many CTAs
    w = dataclasses.replace(wl.opt13b(b=2, L=64, M=1), name="long")
    kinds_long, spans_long = wl.block_kinds(9000, 32)
    kinds_short, spans_short = wl.block_kinds(70, 8)
    w.prompt_kinds = [kinds_long, kinds_short]
    w.prompt_spans = [spans_long, spans_short]
    run_workload(w, steps=2)


def test_sequences_without_tokens_are_skipped():
    w = wl.opt13b(b=3, L=320, M=1)
    run = harness.Runner(w, steps=1)
    n_new = np.array([320, 0, 320], np.int32)
    kinds = np.concatenate([w.prompt_kinds[0], w.prompt_kinds[2]])
    N = 640
    k = torch.empty(N * w.H * w.d, dtype=torch.float16, device="cuda")
    v = torch.empty_like(k)
    tok_t = torch.from_numpy(np.concatenate([np.arange(320), np.arange(320)]).astype(np.int32)).cuda()
    tok_s = torch.from_numpy(np.repeat(np.int32([0, 2]), 320)).cuda()
    run._fill(synth.K_TENSOR, 0, tok_t, tok_s, k, run.kv_scale)
    run._fill(synth.V_TENSOR, 0, tok_t, tok_s, v, run.kv_scale)
    run.cache.append(k, v, n_new, kinds)
    q = torch.empty(1, 3, w.H, w.d, dtype=torch.float16, device="cuda")
    run._fill(synth.Q_TENSOR, 0, torch.full((3,), 319, dtype=torch.int32, device="cuda"),
              torch.arange(3, dtype=torch.int32, device="cuda"), q[0], run.q_scale)
    out = torch.full((3, w.H, w.d), float("nan"), device="cuda")
    # two pending spans hide more than one run: the decode must refuse until they are freed
    with pytest.raises(kvc.KvcError) as e:
        run.cache.decode_attention(0, q[0], w.scale, out)
    assert e.value.status == 5
    run.cache.compress_spans([s for s in (0, 2) for _ in w.prompt_spans[s]],
                             [a for s in (0, 2) for a, _ in w.prompt_spans[s]],
                             [c for s in (0, 2) for _, c in w.prompt_spans[s]])
    run.cache.decode_attention(0, q[0], w.scale, out)
    torch.cuda.synchronize()
    o = out.cpu().numpy()
    assert np.isnan(o[1]).all()  # untouched
    kinds0, pos0 = w.prompt_kinds[0], orc.tied_positions(w.prompt_kinds[0])
    K, V = ow.kv_bits(w, 0, 0, 320)
    ref = orc.masked_decode([kinds0], [pos0], [K], [V], ow.q_bits(w, 0, 0, 319)[None], "f16", w.scale)
    compare(o[0:1], ref)
    assert run.cache.device_status() == 0


def test_capacity_edge_and_errors_through_the_cache():
    w = dataclasses.replace(wl.opt13b(b=1, L=128, M=1), name="no-spans")
    w.prompt_kinds = [np.zeros(128, np.uint8)]
    w.prompt_spans = [[]]
    run = harness.Runner(w, steps=2)
    run.load_prompt()
    out = torch.empty(1, 1, w.H, w.d, device="cuda")
    for g in range(2):
        run.step(run.make_step_inputs(g), out)
    # the cache is full now (capacity = L + 2): one more row must be refused on the host
    inp = run.make_step_inputs(2)
    with pytest.raises(kvc.KvcError) as e:
        run.cache.append(inp.kv_k, inp.kv_v, np.ones(1, np.int32), np.zeros(1, np.uint8))
    assert e.value.status == 3
    # compaction of something that is not a closed span
    with pytest.raises(kvc.KvcError) as e:
        run.cache.compress_spans([0], [7], [40])
    assert e.value.status == 4
    assert run.cache.device_status() == 0


def test_span_at_history_start_and_empty_interior():
    # <CL> at index 0 (first dropped row is row 0) and, under KEEP_CL, a <CL><CR> pair with nothing inside
    w = dataclasses.replace(wl.opt13b(b=2, L=64, M=1), name="edges")
    k0 = np.zeros(200, np.uint8)
    k0[0], k0[9] = wl.CL, wl.CR
    k0[50], k0[51] = wl.CL, wl.CR
    k1 = np.zeros(150, np.uint8)
    k1[149 - 5], k1[149] = wl.CL, wl.CR
    w.prompt_kinds = [k0, k1]
    w.prompt_spans = [[(0, 9), (50, 51)], [(144, 149)]]
    for policy in (orc.POLICY_PAPER, orc.POLICY_KEEP_CL):
        run_workload(w, steps=2, policy=policy)


def test_per_layer_append_equals_all_layer_append():
    w = wl.opt13b(b=2, L=192, M=3)
    a = harness.Runner(w, steps=1)
    a.load_prompt()  # per-layer appends
    b = harness.Runner(w, steps=1)
    # all layers in one call
    n_new = b.L.astype(np.int32)
    N = int(n_new.sum())
    tok_t = torch.from_numpy(np.concatenate([np.arange(L, dtype=np.int32) for L in b.L])).cuda()
    tok_s = torch.from_numpy(np.repeat(np.arange(w.b, dtype=np.int32), b.L)).cuda()
    k = torch.empty(w.M, N * w.H * w.d, dtype=torch.float16, device="cuda")
    v = torch.empty_like(k)
    for m in range(w.M):
        b._fill(synth.K_TENSOR, m, tok_t, tok_s, k[m], b.kv_scale)
        b._fill(synth.V_TENSOR, m, tok_t, tok_s, v[m], b.kv_scale)
    b.cache.append(k, v, n_new, np.concatenate(w.prompt_kinds))
    b.compress_prompt()
    torch.cuda.synchronize()
    for s in range(w.b):
        la, lb = a.cache.masked_reference_layout(s), b.cache.masked_reference_layout(s)
        n = la["stored_orig"].size
        assert np.array_equal(la["stored_orig"], lb["stored_orig"])
        for m in range(w.M):
            for h in (0, 17, 31):
                for pa, pb in ((a.cache.k_plane(m), b.cache.k_plane(m)), (a.cache.v_plane(m), b.cache.v_plane(m))):
                    assert torch.equal(a.cache.stream_rows(pa, s, h, n), b.cache.stream_rows(pb, s, h, n))


def test_launch_counter_counts_kernels():
    w = wl.tiny()
    run = harness.Runner(w, steps=1)
    run.load_prompt()  # one append (M=1) + scan + move
    assert run.cache.launch_count == 3
    out = torch.empty(1, 2, 4, 64, device="cuda")
    run.step(run.make_step_inputs(0), out)  # append + decode
    assert run.cache.launch_count == 5


def _mode_workloads():
    sms = torch.cuda.get_device_properties(0).multi_processor_count if torch.cuda.is_available() else 152
    b_narrow = (5 * sms + 31) // 32  # more segments than one wave of the wide pipeline holds (3 warps/SM at d=64)
    # more segments than one wave of the narrow pipeline holds (8 warps/SM at d=64), and a count that
    # k does not divide, so the last worker takes fewer segments
    b_multi = (10 * sms + 31) // 32 + 1
    b_multi80 = (9 * sms) // 32 + 1  # d=80 rotary: beyond a wave of the narrow pipeline (7 warps/SM)
    long_short = dataclasses.replace(wl.opt13b(b=2, L=64, M=1), name="long-short")
    k_long, s_long = wl.block_kinds(5000, 32)
    k_short, s_short = wl.block_kinds(70, 8)
    long_short.prompt_kinds = [k_long, k_short]
    long_short.prompt_spans = [s_long, s_short]
    return [("wide", wl.opt13b(b=3, L=640, M=1), 1),
            ("narrow", wl.opt13b(b=b_narrow, L=192, M=1), 2),
            ("several segments per warp", wl.opt13b(b=b_multi, L=192, M=1), 3),
            ("several segments per warp, d=80 rotary", wl.rope3b(32, b=b_multi80, L=192, M=1), 3),
            ("stream-k", long_short, 0),
            ("ragged stream-k", wl.ragged(b=40, lmin=64, lmax=1500, M=1, steps=4), 0)]


@pytest.mark.parametrize("name,w,mode", _mode_workloads(), ids=lambda x: x if isinstance(x, str) else "")
def test_every_scheduling_mode(name, w, mode):
    # each way of dividing the decode work (one warp per segment, wide or narrow pipeline; several
    # whole segments per warp; stream-K with split segments) must agree with the oracle
    run, _ = run_workload(w, steps=2, check_steps={0, 1}, seqs=None)
    plan = run.cache.last_decode_plan
    assert plan["mode"] == mode, plan


def test_bounded_wait_reports_timeout_and_context_survives():
    # a wait that nothing completes must give up, report KVC_ERR_TIMEOUT and leave the GPU usable
    w = wl.tiny()
    run = harness.Runner(w, steps=1)
    run.load_prompt()
    assert run.cache.device_status() == 0
    kvc.kvc_check_bounded_wait(run.cache.handle, 2_000_000)  # 2 ms
    with pytest.raises(kvc.KvcError) as e:
        run.cache.device_status()
    assert e.value.status == 8
    assert run.cache.device_status() == 0  # read and cleared
    out = torch.empty(1, 2, 4, 64, device="cuda")
    inp = run.make_step_inputs(0)
    run.step(inp, out)
    torch.cuda.synchronize()
    ref = ow.expected_decode(w, 1, 0, [0, 1])
    compare(out[0].cpu().numpy(), ref)
    assert run.cache.device_status() == 0


@pytest.mark.parametrize("mode,block", [("free", 0), ("progressive", 100), ("progressive", 64)])
def test_write_time_freeing_prompt_modes(mode, block):
    # freeing at write time (in one go, or block by block with compaction of the spans that straddle
    # blocks) leaves exactly the rows the paper keeps; decode over them matches the oracle
    for w in (wl.opt13b(b=3, L=640, M=2), wl.ragged(b=5, lmin=64, lmax=700, M=2, steps=4)):
        run = harness.Runner(w, steps=3)
        run.load_prompt(mode=mode, block=block)
        check_metadata(run, 0)
        for s in range(w.b):
            check_rows(run, 0, 1, s, [0, 17])
        out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device="cuda")
        for g in range(3):
            inp = run.make_step_inputs(g)
            run.step(inp, out)
            torch.cuda.synchronize()
            for m in range(w.M):
                compare(out[m].cpu().numpy(), ow.expected_decode(w, g + 1, m, list(range(w.b))), f"{mode} {g} {m}")
        assert run.cache.device_status() == 0


@pytest.mark.parametrize("ratio", [0.5, 0.8, 0.0])
def test_local_attention_fifo_cache(ratio):
    # the paper's Local Attention baseline (Sec. 4.1; FIFO queue at inference, Sec. 4.2): a ring per
    # (layer, K/V, head), decode over the window, compared with the oracle's local mask
    for w in (wl.opt13b_uncompressed(b=3, L=700, M=2), dataclasses.replace(wl.rope3b(32, b=2, L=300, M=1),
                                                                           prompt_kinds=[np.zeros(300, np.uint8)] * 2,
                                                                           prompt_spans=[[], []], name="rope-local")):
        run = harness.Runner(w, steps=6, policy=kvc.POLICY_LOCAL, local_ratio=ratio)
        run.load_prompt()
        out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device="cuda")
        r32 = float(np.float32(ratio))
        for g in range(6):
            run.step(run.make_step_inputs(g), out)
            torch.cuda.synchronize()
            for m in range(w.M):
                ref = ow.expected_local_decode(w, g + 1, m, list(range(w.b)), r32)
                compare(out[m].cpu().numpy(), ref, f"local r={ratio} step {g} layer {m}")
            for s in range(w.b):
                lay = run.cache.masked_reference_layout(s)
                T = lay["kinds"].size
                first = int(np.floor(T * np.float64(r32)))
                assert np.array_equal(lay["stored_orig"], np.arange(first, T))
        assert run.cache.device_status() == 0


def test_multi_layer_decode_call_equals_per_layer_calls():
    """kvc_decode_attention_layers over balanced segments is one launch in which every segment is
    processed whole with the per-layer launches' tile shape: identical outputs."""
    w = wl.opt13b(b=3, L=400, M=3)
    run = harness.Runner(w, 2)
    run.load_prompt()
    inp = run.make_step_inputs(0)
    run.cache.append(inp.kv_k, inp.kv_v, np.ones(w.b, np.int32), inp.kinds)
    one = torch.full((w.M, w.b, w.H, w.d), float("nan"), dtype=torch.float32, device="cuda")
    for m in range(w.M):
        kvc.kvc_decode_attention(run.cache.handle, m, inp.q[m], w.scale, one[m])
    l0 = run.cache.launch_count
    many = run.cache.decode_attention_layers(inp.q, w.scale)
    torch.cuda.synchronize()
    assert run.cache.launch_count == l0 + 1
    assert torch.equal(one, many)
    # a run of layers in the middle, with padded strides
    n = w.b * w.H * w.d
    qpad = torch.zeros(w.M, n + 64, dtype=inp.q.dtype, device="cuda")
    qpad[:, :n] = inp.q.reshape(w.M, n)
    opad = torch.full((w.M, n + 32), float("nan"), dtype=torch.float32, device="cuda")
    kvc.kvc_decode_attention_layers(run.cache.handle, 1, 2, qpad[1], n + 64, w.scale, opad[1], n + 32)
    torch.cuda.synchronize()
    assert torch.equal(opad[1:, :n], one[1:].reshape(2, n))
    assert torch.isnan(opad[0]).all()
    assert run.cache.device_status() == 0


def _layers_without_some_tokens(b, M, L=192, dead=lambda s: s % 3 == 1):
    """An OPT-1.3B-shaped cache of M layers whose `dead` sequences hold no token; the prompt spans of
    the others are freed.  Returns the runner, the live sequences and every layer's queries at the
    last prompt token."""
    w = wl.opt13b(b=b, L=L, M=M)
    run = harness.Runner(w, steps=1)
    live = [s for s in range(b) if not dead(s)]
    n_new = np.array([0 if dead(s) else L for s in range(b)], np.int32)
    kinds = np.concatenate([w.prompt_kinds[s] for s in live])
    N = L * len(live)
    k = torch.empty(M, N * w.H * w.d, dtype=torch.float16, device="cuda")
    v = torch.empty_like(k)
    tok_t = torch.from_numpy(np.tile(np.arange(L, dtype=np.int32), len(live))).cuda()
    tok_s = torch.from_numpy(np.repeat(np.int32(live), L)).cuda()
    for m in range(M):
        run._fill(synth.K_TENSOR, m, tok_t, tok_s, k[m], run.kv_scale)
        run._fill(synth.V_TENSOR, m, tok_t, tok_s, v[m], run.kv_scale)
    run.cache.append(k, v, n_new, kinds)
    run.cache.compress_spans([s for s in live for _ in w.prompt_spans[s]],
                             [a for s in live for a, _ in w.prompt_spans[s]],
                             [c for s in live for _, c in w.prompt_spans[s]])
    q = torch.empty(M, b, w.H, w.d, dtype=torch.float16, device="cuda")
    for m in range(M):
        run._fill(synth.Q_TENSOR, m, torch.full((b,), L - 1, dtype=torch.int32, device="cuda"),
                  torch.arange(b, dtype=torch.int32, device="cuda"), q[m], run.q_scale)
    return w, run, live, q


@pytest.mark.parametrize("b", [53, 61])
def test_fused_layers_several_segments_per_warp_with_empty_sequences(b):
    """One launch over five layers with more segments than a wave of warps holds: each warp takes k
    consecutive whole segments and skips the sequences that hold no token.  With a prime b the 32 b
    segments of a layer are a multiple of k only when k is a power of two, so workers' runs of
    segments cross from one layer to the next.  Every live output against the oracle; the empty
    sequences' outputs untouched."""
    M = 5
    w, run, live, q = _layers_without_some_tokens(b, M)
    fused = torch.full((M, b, w.H, w.d), float("nan"), dtype=torch.float32, device="cuda")
    l0 = run.cache.launch_count
    run.cache.decode_attention_layers(q, w.scale, fused)
    torch.cuda.synchronize()
    assert run.cache.launch_count == l0 + 1
    plan = run.cache.last_decode_plan
    assert plan["mode"] == 3, plan
    one = torch.full_like(fused, float("nan"))
    for m in range(M):
        kvc.kvc_decode_attention(run.cache.handle, m, q[m], w.scale, one[m])
    torch.cuda.synchronize()
    o, o1 = fused.cpu().numpy(), one.cpu().numpy()
    dead = [s for s in range(b) if s not in live]
    assert np.isnan(o[:, dead]).all() and np.isnan(o1[:, dead]).all()
    for m in range(M):
        ref = ow.expected_decode(w, 0, m, live)  # queries at the last prompt token, spans freed
        compare(o[m][live], ref, f"fused layer {m}")
        compare(o1[m][live], ref, f"per-layer layer {m}")
    assert run.cache.device_status() == 0


def test_fused_layers_fall_back_to_per_layer_launches_when_unbalanced():
    """Unbalanced segments are split over a wave of warps (stream-K) one layer per launch: the
    multi-layer call makes M launches and matches the per-layer calls bit for bit."""
    w = dataclasses.replace(wl.opt13b(b=2, L=64, M=3), name="long-short")
    k_long, s_long = wl.block_kinds(3000, 32)
    k_short, s_short = wl.block_kinds(70, 8)
    w.prompt_kinds = [k_long, k_short]
    w.prompt_spans = [s_long, s_short]
    run = harness.Runner(w, 3)
    run.load_prompt()
    out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device="cuda")
    run.step(run.make_step_inputs(0), out)  # a <CL>: its query sees one row, balanced by itself
    inp = run.make_step_inputs(1)           # a normal token inside the open span
    run.append_only(inp)
    one = torch.full((w.M, w.b, w.H, w.d), float("nan"), dtype=torch.float32, device="cuda")
    for m in range(w.M):
        kvc.kvc_decode_attention(run.cache.handle, m, inp.q[m], w.scale, one[m])
    l0 = run.cache.launch_count
    many = run.cache.decode_attention_layers(inp.q, w.scale)
    torch.cuda.synchronize()
    assert run.cache.launch_count == l0 + w.M
    assert run.cache.last_decode_plan["mode"] == 0
    assert torch.equal(one, many)
    o = many.cpu().numpy()
    for m in range(w.M):
        compare(o[m], ow.expected_decode(w, 2, m, [0, 1]), f"layer {m}")
    assert run.cache.device_status() == 0


def test_fused_layers_whole_segments_cut_by_rows():
    """Unbalanced (ragged) segments over many layers, each short beside a warp's even share of all the
    layers' rows: one launch in which every warp takes a run of whole segments cut by rows (no split,
    no combine).  Against the per-layer stream-K launches, which split segments and combine them, and
    against the oracle on the first, a middle and the last layer."""
    w = wl.ragged(b=64, lmin=64, lmax=700, M=24, steps=2)
    run = harness.Runner(w, 2)
    run.load_prompt()
    inp = run.make_step_inputs(0)
    run.append_only(inp)
    rows = run.attended_rows()
    assert rows.max() * w.b > 1.3 * rows.sum()  # unbalanced: the longest segment is above 1.3x the mean
    one = torch.full((w.M, w.b, w.H, w.d), float("nan"), dtype=torch.float32, device="cuda")
    for m in range(w.M):
        kvc.kvc_decode_attention(run.cache.handle, m, inp.q[m], w.scale, one[m])
    assert run.cache.last_decode_plan["mode"] == 0
    l0 = run.cache.launch_count
    many = run.cache.decode_attention_layers(inp.q, w.scale)
    torch.cuda.synchronize()
    plan = run.cache.last_decode_plan
    assert run.cache.launch_count == l0 + 1
    assert plan["mode"] == 4, plan
    # the precondition of the plan: the longest segment within 1/16 of a warp's share of the rows
    assert 16 * rows.max() <= w.M * w.H * rows.sum() // plan["workers"]
    assert plan["tile_rows"] == 32  # segments of ~200 rows: the narrow shape
    o, o1 = many.cpu().numpy(), one.cpu().numpy()
    seqs = list(range(w.b))
    for m in (0, w.M // 2, w.M - 1):
        ref = ow.expected_decode(w, 1, m, seqs)
        compare(o[m], ref, f"fused layer {m}")
        compare(o1[m], ref, f"per-layer layer {m}")
    compare(o.reshape(-1), o1.reshape(-1).astype(np.float64), "fused against per-layer, every layer")
    assert run.cache.device_status() == 0


def test_local_attention_ragged_rings_fused_layers():
    """Local Attention rings of different sizes over 24 layers (prompts of 64-700 tokens, window about
    half the history, so every ring has wrapped): one decode launch in which warps take runs of whole
    windows cut by rows, each window read in two parts around its ring's end.  Against the oracle's
    Local Attention decode on the first, a middle and the last layer, two steps."""
    base = wl.ragged(b=64, lmin=64, lmax=700, M=24, steps=3)
    kinds = [np.zeros(int(n), np.uint8) for n in base.prompt_len]
    w = dataclasses.replace(base, prompt_kinds=kinds, prompt_spans=[[] for _ in kinds], gen_kind=wl._normal_gen,
                            name="ragged-local")
    ratio = 0.5
    r32 = float(np.float32(ratio))
    run = harness.Runner(w, steps=3, policy=kvc.POLICY_LOCAL, local_ratio=ratio)
    run.load_prompt()
    out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device="cuda")
    seqs = list(range(w.b))
    for g in range(2):
        l0 = run.cache.launch_count
        run.step(run.make_step_inputs(g), out)
        torch.cuda.synchronize()
        assert run.cache.last_decode_plan["mode"] == 4, run.cache.last_decode_plan
        assert run.cache.launch_count == l0 + 2  # the append and one decode launch
        o = out.cpu().numpy()
        for m in (0, w.M // 2, w.M - 1):
            compare(o[m], ow.expected_local_decode(w, g + 1, m, seqs, r32), f"ragged local step {g} layer {m}")
    assert run.cache.device_status() == 0
