"""Parity of the tensor-core masked prefill (kvc_prefill_attention, through the C ABI) with the fp64
oracle: every query of a prompt block under the sentinel mask (Sec. 3.1), in one go and block by
block with the spans each block closed freed in between, ragged lengths and query tiles that start
mid-tile, RoPE (full and partial rotary dimension, f16 and bf16), both policies, every built d_head
and both 16-bit types."""
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

from _parity import MAX_ABS, MAX_REL, REL_FLOOR, check_metadata

pytestmark = pytest.mark.gpu

# One tolerance for both 16-bit types, the decode's (fp16/bf16 K/V with fp32 accumulation).  The
# kernel feeds the rotated query and the softmax weights P to the tensor cores in the cache type; with
# bf16 it passes each as a high and a low bf16 part, so both products keep 16 significant bits.
TOL = {"f16": (MAX_ABS, MAX_REL), "bf16": (MAX_ABS, MAX_REL)}


def _compare(got, ref, dtype, what):
    got = np.asarray(got, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - ref)
    a, r = float(err.max()), float((err / np.maximum(np.abs(ref), REL_FLOOR)).max())
    ta, tr = TOL[dtype]
    assert a <= ta and r <= tr, f"{what}: max_abs={a:.3g} max_rel={r:.3g}"
    return a, r


def run_prefill(w, block, layers, heads=None, policy=orc.POLICY_PAPER):
    run = harness.Runner(w, 0, policy)
    outs = []

    def keep(start, n, m, out):
        outs.append((start.copy(), n.copy(), m, out.cpu().numpy()))

    run.prefill_prompt(block=block, out_cb=keep, layers=layers)
    worst = (0.0, 0.0)
    for start, n, m, o in outs:
        ref = ow.expected_prefill(w, m, range(w.b), start + n, n, heads, policy)
        got = o if heads is None else o[:, heads]
        a, r = _compare(got, ref, w.dtype, f"{w.name} block at {start.tolist()} layer {m}")
        worst = (max(worst[0], a), max(worst[1], r))
    check_metadata(run, 0, policy=policy)
    assert run.cache.device_status() == 0
    print(f"{w.name} block={block}: max_abs={worst[0]:.3g} max_rel={worst[1]:.3g}")
    return run, worst


def test_prefill_one_go_opt13b_shaped():
    # the whole prompt appended, every query over every stored row; spans closed earlier in the
    # prompt are masked, not freed; <CL> queries at 64k+7, <CR> queries at 64k+40
    w = wl.opt13b(b=2, L=520, M=2)
    run_prefill(w, 0, layers=[1], heads=[0, 17, 31])


def test_prefill_progressive_blocks_straddling_spans():
    # blocks of 200 tokens: spans open at a block's end close in the next one, so rows of the
    # earlier block become hidden from the later queries of the next block
    w = wl.opt13b(b=3, L=700, M=1)
    run_prefill(w, 200, layers=[0], heads=[0, 9])


@pytest.mark.parametrize("block", [0, 256])
def test_prefill_ragged_lengths(block):
    w = wl.ragged(b=5, lmin=60, lmax=620, M=1, steps=1)
    run_prefill(w, block, layers=[0], heads=[3, 30])


def test_prefill_rope():
    w = wl.rope3b(32, b=2, L=400, M=2)
    run_prefill(w, 0, layers=[1], heads=[0, 31])


def test_prefill_bf16_d80_prescaled_queries():
    w = wl.opt27b(b=2, L=384, M=1)
    run_prefill(w, 160, layers=[0], heads=[1, 2])


@pytest.mark.parametrize("d,dtype", [(96, "f16"), (128, "bf16"), (64, "bf16"), (80, "f16")])
def test_prefill_every_built_head_dim(d, dtype):
    w = dataclasses.replace(wl.opt13b(b=2, L=300, M=1), d=d, dtype=dtype, name=f"d{d}-{dtype}")
    run_prefill(w, 0, layers=[0], heads=[0, 7])


def test_prefill_keep_cl_policy():
    w = wl.opt13b(b=2, L=330, M=1)
    run_prefill(w, 128, layers=[0], heads=[4], policy=orc.POLICY_KEEP_CL)


def test_prefill_query_subsets_and_errors():
    """n_q = 0 for a sequence (skipped), a single query (= the decode at that token), and the host
    errors: a query token that is not stored, the local policy, a non-positive scale."""
    w = wl.opt13b(b=3, L=300, M=1)
    run = harness.Runner(w, 0)
    run.load_prompt(compress=False)
    H, d = w.H, w.d
    n_q = np.array([0, 1, 37], np.int32)
    q = torch.empty(int(n_q.sum()) * H * d, dtype=torch.float16, device="cuda")
    tok_t = torch.tensor([299] + list(range(263, 300)), dtype=torch.int32, device="cuda")
    tok_s = torch.tensor([1] + [2] * 37, dtype=torch.int32, device="cuda")
    synth.fill_tokens_cuda(w.seed, w.dtype, synth.scale_for(w.q_sigma), synth.tag(synth.Q_TENSOR, 0), tok_t, tok_s,
                           H, d, q)
    out = torch.full((int(n_q.sum()), H, d), float("nan"), dtype=torch.float32, device="cuda")
    kvc.kvc_prefill_attention(run.cache.handle, 0, q, n_q, w.scale, out)
    got = out.cpu().numpy()
    ref = ow.expected_prefill(w, 0, [1, 2], np.array([0, 300, 300]), n_q, None)
    _compare(got, ref, "f16", "subsets")
    # the single query equals the decode oracle at that token
    dec = ow.expected_decode(w, 0, 0, [1])
    assert np.max(np.abs(got[0] - dec[0])) <= MAX_ABS
    with pytest.raises(kvc.KvcError) as e:
        kvc.kvc_prefill_attention(run.cache.handle, 0, q, n_q, 0.0, out)
    assert e.value.status == 1
    # tokens freed at write time cannot be queried
    run2 = harness.Runner(w, 0)
    run2.load_prompt(mode="free")
    with pytest.raises(kvc.KvcError) as e:
        kvc.kvc_prefill_attention(run2.cache.handle, 0, q, n_q, w.scale, out)
    assert e.value.status == 5
    # no prefill for the local-attention cache
    loc = kvc.KVCache(1, H, d, [64] * 3, "f16", policy=kvc.POLICY_LOCAL, local_ratio=0.5)
    loc.append(torch.zeros(3 * H * d, dtype=torch.float16, device="cuda"),
               torch.zeros(3 * H * d, dtype=torch.float16, device="cuda"), [1, 1, 1], [0, 0, 0])
    with pytest.raises(kvc.KvcError) as e:
        kvc.kvc_prefill_attention(loc.handle, 0, q[:3 * H * d], [1, 1, 1], 0.125, out)
    assert e.value.status == 2
    assert run.cache.device_status() == 0


@pytest.mark.parametrize("policy", [orc.POLICY_PAPER, orc.POLICY_KEEP_CL])
def test_prefill_query_tile_offsets(policy):
    """The first query row at several offsets within a 128-row key tile (1, 127, 129, 200): key tiles
    that end exactly at the first query, query tiles straddling two key tiles, and <CL> queries (tokens
    64k + 7) in each of them, which must see their own key alone."""
    w = wl.opt13b(b=4, L=330, M=1)
    run = harness.Runner(w, 0, policy)
    run.load_prompt(compress=False)
    H, d, L = w.H, w.d, 330
    q0 = np.array([1, 127, 129, 200])
    n_q = (L - q0).astype(np.int32)
    tok_t = torch.tensor(np.concatenate([np.arange(a, L) for a in q0]), dtype=torch.int32, device="cuda")
    tok_s = torch.tensor(np.repeat(np.arange(4), n_q), dtype=torch.int32, device="cuda")
    q = torch.empty(int(n_q.sum()) * H * d, dtype=torch.float16, device="cuda")
    synth.fill_tokens_cuda(w.seed, w.dtype, synth.scale_for(w.q_sigma), synth.tag(synth.Q_TENSOR, 0), tok_t, tok_s,
                           H, d, q)
    out = torch.full((int(n_q.sum()), H, d), float("nan"), dtype=torch.float32, device="cuda")
    kvc.kvc_prefill_attention(run.cache.handle, 0, q, n_q, w.scale, out)
    heads = [0, 13, 31]
    got = out.cpu().numpy()[:, heads]
    ref = ow.expected_prefill(w, 0, range(4), np.full(4, L), n_q, heads, policy)
    _compare(got, ref, "f16", f"query tiles at {q0.tolist()}")
    assert run.cache.device_status() == 0


def test_prefill_blocks_of_512_cl_key_in_last_column():
    """Blocks of 512 tokens: once the first block's spans are freed, the second block's queries start
    at stored row 248, so the <CL> at token 519 is stored row 255, the last column of key tile 1.
    Its query tile runs its key tiles in reverse, so the tile before holds no visible key for that
    query and its own tile holds one, in the last column: the row maximum must take that column."""
    w = wl.opt13b(b=2, L=1100, M=1)
    run_prefill(w, 512, layers=[0], heads=[0, 31])


@pytest.mark.parametrize("d,rot,block", [(80, 80, 0), (80, 32, 200), (64, 64, 0), (96, 96, 0), (128, 64, 256)])
def test_prefill_rope_bf16(d, rot, block):
    # bf16 with RoPE: the rotated query goes to the tensor cores as a high and a low bf16 part (its low
    # part in TMEM with two CTAs per SM, d_head 64 / 80, and in shared memory with one, d_head 96 /
    # 128; zero past the rotary dimensions), P likewise; held to the f16 bound
    w = dataclasses.replace(wl.rope3b(32, b=2, L=400, M=1), dtype="bf16", d=d, rotary_dim=rot,
                            scale=1.0 / math.sqrt(d), name=f"rope-bf16-d{d}-r{rot}")
    run_prefill(w, block, layers=[0], heads=[0, 31])


@pytest.mark.parametrize("d,rot", [(96, 96), (128, 64)])
def test_prefill_rope_other_head_dims(d, rot):
    # one CTA per SM (d_head 96 / 128) with the query rotated over 48 / 32 pairs
    w = dataclasses.replace(wl.rope3b(32, b=2, L=384, M=1), d=d, rotary_dim=rot, scale=1.0 / math.sqrt(d),
                            name=f"rope-d{d}-r{rot}")
    run_prefill(w, 0, layers=[0], heads=[3, 30])


def test_prefill_rope_partial_rotary_dim():
    # only the first 32 of 80 dimensions rotated (pairs (e, e + 16)); blocks of 200 tokens
    w = dataclasses.replace(wl.rope3b(32, b=2, L=384, M=1), rotary_dim=32, name="rope-partial")
    run_prefill(w, 200, layers=[0], heads=[5, 30])
