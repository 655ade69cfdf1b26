"""kvc_decode_attention_static_scratch: the decode for callers that cannot allocate device memory.

Some callers run where new device allocations are not allowed -- inside a fixed, pre-sized memory
pool, or under an allocator that forbids cudaMalloc once serving has started -- so they cannot
give the decode a scratch buffer of its own.  This entry point keeps its split-K scratch in a
file-scope device array of the library instead.  Its results must equal those of the regular entry
point bit for bit, on two calls in a row (the array keeps the previous call's contents, so each call
must start from a clean state), and the calls must allocate no device memory.  Collected last on purpose: a failure here leaves every other test already run.
"""
import dataclasses

import numpy as np
import pytest
import torch

import harness
import paper_2310_08152_gb300 as kvc
from synth import workloads as wl

from _parity import compare

pytestmark = pytest.mark.gpu


def _workloads():
    # one (sequence, head) per warp, and a stream-K split with partials combined through the scratch
    long_short = dataclasses.replace(wl.opt13b(b=2, L=64, M=2), name="long-short")
    k_long, s_long = wl.block_kinds(9000, 32)
    k_short, s_short = wl.block_kinds(70, 8)
    long_short.prompt_kinds = [k_long, k_short]
    long_short.prompt_spans = [s_long, s_short]
    return [wl.opt13b(b=3, L=640, M=2), wl.ragged(b=6, lmin=64, lmax=900, M=2, steps=4), long_short]


@pytest.mark.parametrize("w", _workloads(), ids=lambda w: w.name)
def test_static_scratch_decode_matches_workspace_decode(w):
    """Same kernel, same plan, same inputs as kvc_decode_attention: the outputs are equal bit for bit,
    on two calls in a row, and the calls allocate no device memory."""
    run = harness.Runner(w, steps=2)
    run.load_prompt()
    for g in range(2):
        inp = run.make_step_inputs(g)
        out = torch.empty(w.M, w.b, w.H, w.d, dtype=torch.float32, device="cuda")
        run.append_only(inp)
        # the regular entry point (split-K scratch in the cache workspace), layer by layer
        for m in range(w.M):
            kvc.kvc_decode_attention(run.cache.handle, m, inp.q[m], w.scale, out[m])
        alt = torch.full((2, w.M, w.b, w.H, w.d), float("nan"), device="cuda")
        torch.cuda.synchronize()
        # the same query through the static scratch, twice; the second time no lookup is left to do
        for rep in range(2):
            free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
            for m in range(w.M):
                kvc.kvc_decode_attention_static_scratch(run.cache.handle, m, inp.q[m], w.scale, alt[rep, m])
            torch.cuda.synchronize()
            if rep == 1:
                assert torch.cuda.mem_get_info()[0] == free0, "device memory was allocated"
                assert torch.cuda.memory_allocated() == alloc0
            assert torch.equal(alt[rep], out), f"{w.name} step {g} call {rep}: not bit-identical"
        compare(alt[1, 0].cpu().numpy(), out[0].cpu().numpy().astype(np.float64), f"{w.name} step {g}")
        run.finish_step(inp)  # frees the span a <CR> closed
    assert run.cache.device_status() == 0


def test_static_scratch_rejects_caches_beyond_its_size():
    # 2048 sequences x 32 heads at d_head=128 need more split-K scratch than the 8 MiB array holds
    cap = np.full(2048, 4, np.int64)
    cache = kvc.KVCache(1, 32, 128, cap, "f16")
    n_new = np.ones(2048, np.int32)
    k = torch.zeros(2048 * 32 * 128, dtype=torch.float16, device="cuda")
    cache.append(k, k, n_new, np.zeros(2048, np.uint8))
    q = torch.zeros(2048, 32, 128, dtype=torch.float16, device="cuda")
    out = torch.empty(2048, 32, 128, device="cuda")
    with pytest.raises(kvc.KvcError) as e:
        kvc.kvc_decode_attention_static_scratch(cache.handle, 0, q, 1.0, out)
    assert e.value.status == 2 and "static array" in e.value.message
    cache.decode_attention(0, q, 1.0, out)  # the regular entry point still serves it
    torch.cuda.synchronize()
    assert cache.device_status() == 0
