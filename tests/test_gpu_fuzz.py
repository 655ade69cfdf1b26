"""Randomised parity: caches of random shapes and histories through the whole path (prompt append,
compaction, per-step append, decode of every layer in one call, span freeing), against the oracle at
every step.  Prompts of 1 to 600 tokens (single-row segments, sequences far apart in length), spans
at random places with interiors of 0 to 40 tokens (one may start at the history's first token),
spans opened and closed while generating (some left open at the end, some opened at step 0), both
mask policies, f16 and bf16, with and without RoPE.  The stored rows' metadata is checked bit-exact
after every compaction."""
import dataclasses

import numpy as np
import pytest

import oracle as orc
from synth import workloads as wl

from _parity import run_workload

pytestmark = pytest.mark.gpu

NORMAL, CL, CR = 0, 1, 2


def _random_history(rng, L):
    kinds = np.zeros(L, np.uint8)
    spans = []
    t = 0 if rng.random() < 0.2 else int(rng.integers(0, 12))
    while t + 1 < L:
        interior = int(rng.integers(0, 41))
        cl, cr = t, t + 1 + interior
        if cr >= L:
            break
        kinds[cl], kinds[cr] = CL, CR
        spans.append((cl, cr))
        t = cr + 1 + int(rng.integers(0, 30))
    return kinds, spans


def _fuzz_workload(seed, d, dtype, M, rot, steps, b=None):
    rng = np.random.default_rng(seed)
    b = int(rng.integers(6, 33)) if b is None else b
    lens = rng.integers(1, 601, size=b)
    lens[rng.integers(0, b)] = 1
    hist = [_random_history(rng, int(n)) for n in lens]
    opens = rng.integers(0, steps, size=b)
    gaps = rng.integers(1, steps + 2, size=b)  # some spans stay open past the last step

    def gen(s, g):
        if g == opens[s]:
            return CL
        if g == opens[s] + gaps[s]:
            return CR
        return NORMAL

    base = wl.opt13b(b=b, L=64, M=M)
    return dataclasses.replace(base, name=f"fuzz{seed}", d=d, dtype=dtype, b=b,
                               prompt_kinds=[k for k, _ in hist], prompt_spans=[sp for _, sp in hist],
                               n_steps=steps, gen_kind=gen, scale=1.0 / np.sqrt(d), rotary_dim=rot,
                               seed=wl.SEED_BASE + 100 + seed)


@pytest.mark.parametrize("seed,d,dtype,M,rot,policy", [
    (1, 64, "f16", 3, 0, orc.POLICY_PAPER),
    (2, 80, "bf16", 2, 80, orc.POLICY_KEEP_CL),
    (3, 64, "f16", 6, 32, orc.POLICY_PAPER),
    (4, 128, "f16", 2, 0, orc.POLICY_PAPER),
    (5, 96, "bf16", 2, 96, orc.POLICY_PAPER),
    (6, 80, "f16", 4, 0, orc.POLICY_KEEP_CL),
])
def test_random_histories(seed, d, dtype, M, rot, policy):
    steps = 10
    w = _fuzz_workload(seed, d, dtype, M, rot, steps)
    run_workload(w, steps=steps, policy=policy)


def test_random_histories_one_launch_over_all_layers():
    """128 random histories over 24 layers: short segments far apart in length, decoded in one launch
    whose warps take runs of whole segments cut by rows (narrow shape), every step against the oracle."""
    steps = 6
    w = _fuzz_workload(7, 64, "f16", 24, 0, steps, b=128)
    run, _ = run_workload(w, steps=steps, layers=[0, 11, 23])
    plan = run.cache.last_decode_plan
    assert plan["mode"] == 4 and plan["tile_rows"] == 32, plan
