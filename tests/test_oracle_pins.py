"""Pins of the fp64 CPU oracle to facts outside itself (CPU only).

Each test checks the oracle against something the paper or the mathematics
fixes: library float16/bfloat16 conversions, a library softmax-attention
routine in the span-free case, closed-form row counts of the periodic span
geometry, the rotation-matrix / complex-number forms of RoPE, the stated
special cases of the mask (a <CL> query sees only itself), the
compaction-equivalence invariant (attention under the mask over the full
history equals plain attention over the rows left after freeing the closed
spans), and brute force over every well-formed kind sequence of length <= 8.
"""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle as orc
from synth import workloads as wl

NORMAL, CL, CR = orc.NORMAL, orc.CL, orc.CR


# --------------------------------------------------------------------------
# 16-bit formats
# --------------------------------------------------------------------------

def test_f16_decode_exhaustive_vs_numpy():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = orc.decode16(bits, "f16")
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])


def test_bf16_decode_exhaustive_vs_torch():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = orc.decode16(bits, "bf16")
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])


def _f32_probe_values(rng):
    # every half/bfloat16 tie and neighbour region, subnormals, overflow edges, plus random values
    f = []
    for e in range(-30, 17):
        base = 2.0 ** e
        m = rng.integers(0, 2 ** 23, size=200)
        f.append(np.float32(base) * (1 + m.astype(np.float64) / 2 ** 23))
    v = np.concatenate(f).astype(np.float32)
    # exact midpoints between adjacent float16 values and between adjacent bfloat16 values
    h = np.arange(0, 0x7C00, 7, dtype=np.uint16)
    hv = h.view(np.float16).astype(np.float64)
    hn = (h + 1).view(np.float16).astype(np.float64)
    mids16 = ((hv + hn) / 2).astype(np.float32)
    b = np.arange(0, 0x7F80, 5, dtype=np.uint32)
    bv = (b << 16).astype(np.uint32).view(np.float32).astype(np.float64)
    bn = ((b + 1) << 16).astype(np.uint32).view(np.float32).astype(np.float64)
    mids_b = ((bv + bn) / 2).astype(np.float32)
    allv = np.concatenate([v, mids16, mids_b, np.float32([65504, 65519.99, 65520, 65536, 1e-8, 3e-8, 5.96e-8])])
    return np.concatenate([allv, -allv])


def test_f16_encode_vs_numpy():
    rng = np.random.default_rng(1)
    x = _f32_probe_values(rng).astype(np.float64)
    ours = orc.encode16(x, "f16")
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)


def test_bf16_encode_vs_torch():
    rng = np.random.default_rng(2)
    x = _f32_probe_values(rng)  # binary32 values: torch's float -> bfloat16 rounding is the reference
    ours = orc.encode16(x.astype(np.float64), "bf16")
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


# --------------------------------------------------------------------------
# Positions (Sec. 3.1, Input Transformation)
# --------------------------------------------------------------------------

def _random_wellformed(rng, n, p_open=0.15, p_close=0.2):
    kinds = np.zeros(n, dtype=np.uint8)
    open_ = False
    for t in range(n):
        r = rng.random()
        if not open_ and r < p_open:
            kinds[t] = CL
            open_ = True
        elif open_ and r < p_close:
            kinds[t] = CR
            open_ = False
    return kinds


def test_positions_closed_form():
    rng = np.random.default_rng(3)
    for _ in range(200):
        n = int(rng.integers(1, 300))
        kinds = _random_wellformed(rng, n)
        if rng.random() < 0.3:
            kinds[0] = CL if kinds[0] == NORMAL and not (kinds == CR).any() else kinds[0]
        pos = orc.tied_positions(kinds)
        normal_count = np.cumsum(kinds == NORMAL)
        assert np.array_equal(pos, np.maximum(0, normal_count - 1))


def test_positions_sentinels_occupy_no_position():
    # removing the sentinels must leave the normal tokens at 0, 1, 2, ... (the untransformed input)
    rng = np.random.default_rng(4)
    for _ in range(100):
        kinds = _random_wellformed(rng, int(rng.integers(2, 200)))
        pos = orc.tied_positions(kinds)
        normals = pos[kinds == NORMAL]
        assert np.array_equal(normals, np.arange(normals.size))
        # each sentinel shares the position of the token before it
        for t in np.nonzero(kinds != NORMAL)[0]:
            assert pos[t] == (pos[t - 1] if t > 0 else 0)


# --------------------------------------------------------------------------
# Span pairing
# --------------------------------------------------------------------------

def test_pairing_rejects_overlap_and_nesting():
    with pytest.raises(orc.OracleError):
        orc.pair_spans(np.array([CL, NORMAL, CL, NORMAL, CR, CR], dtype=np.uint8))
    with pytest.raises(orc.OracleError):
        orc.pair_spans(np.array([NORMAL, CR], dtype=np.uint8))
    spans, op = orc.pair_spans(np.array([CL, NORMAL, CR, NORMAL, CL, NORMAL], dtype=np.uint8))
    assert spans == [(0, 2)] and op == 4


@pytest.mark.parametrize("make", [wl.tiny, lambda: wl.opt13b(b=2), lambda: wl.opt27b(b=2),
                                  lambda: wl.rope3b(19, b=1), lambda: wl.rope3b(45, b=1),
                                  lambda: wl.ragged(b=4, lmax=1024)])
def test_recipes_are_wellformed(make):
    w = make()
    for s in range(w.b):
        spans, op = orc.pair_spans(w.prompt_kinds[s])
        assert spans == [tuple(x) for x in w.prompt_spans[s]] and op == -1
        hist = w.kinds_history(s, w.n_steps)
        spans_all, _ = orc.pair_spans(hist)
        assert spans_all[len(spans):] == w.gen_spans(s, w.n_steps)


# --------------------------------------------------------------------------
# Mask + freeing: closed-form counts of the periodic geometry
# --------------------------------------------------------------------------

@pytest.mark.parametrize("L,interior,expect", [(512, 32, 248), (2048, 32, 992), (4096, 44, 1216),
                                               (2048, 19, 1408), (2048, 45, 576)])
def test_closed_form_counts(L, interior, expect):
    kinds, spans = wl.block_kinds(L, interior)
    blocks = L // 64
    assert len(spans) == blocks
    # each block frees its <CL> and its I enclosed tokens: 64 - I - 1 rows survive
    assert expect == blocks * (64 - interior - 1)
    rows = orc.stored_rows(L, spans, orc.POLICY_PAPER)
    assert rows.size == expect
    rows_keep = orc.stored_rows(L, spans, orc.POLICY_KEEP_CL)
    assert rows_keep.size == blocks * (64 - interior)
    # a following normal query sees exactly the survivors plus itself
    hist = np.concatenate([kinds, np.uint8([NORMAL])])
    assert orc.visible(hist, L, orc.POLICY_PAPER).sum() == expect + 1
    assert orc.visible(hist, L, orc.POLICY_KEEP_CL).sum() == blocks * (64 - interior) + 1
    # compression ratio (Sec. 3.1): fraction of the L tokens enclosed
    assert math.isclose(sum(cr - cl - 1 for cl, cr in spans) / L, interior / 64)


# --------------------------------------------------------------------------
# Brute force over every well-formed kind sequence of length <= 8
# --------------------------------------------------------------------------

def _all_wellformed(n):
    for seq in itertools.product((NORMAL, CL, CR), repeat=n):
        open_ = False
        ok = True
        for k in seq:
            if k == CL:
                if open_:
                    ok = False
                    break
                open_ = True
            elif k == CR:
                if not open_:
                    ok = False
                    break
                open_ = False
        if ok:
            yield np.array(seq, dtype=np.uint8)


def _rand_bits(rng, shape, dtype="f16"):
    x = rng.standard_normal(shape)
    return orc.encode16(x, dtype)


@pytest.mark.parametrize("policy", [orc.POLICY_PAPER, orc.POLICY_KEEP_CL])
def test_bruteforce_compaction_equivalence(policy):
    """Masked attention over the full history == plain attention over the rows that remain once
    every span closed before the query is freed (minus an open span's <CL> under the paper policy)."""
    rng = np.random.default_rng(5)
    d = 8
    n_checked = 0
    for n in range(1, 9):
        for kinds in _all_wellformed(n):
            K = _rand_bits(rng, (n, d))
            V = _rand_bits(rng, (n, d))
            q = _rand_bits(rng, (d,))
            for t_q in range(n):
                sub = kinds[:t_q + 1]
                vis = orc.visible(sub, t_q, policy)
                assert vis[t_q]  # every query attends to itself
                full = orc.attend(q, K, V, None, np.nonzero(vis)[0], "f16", 0.5)
                if kinds[t_q] == CL:
                    # Sec. 3.1: <CL> attends only to itself -> its own value row, exactly
                    assert vis.sum() == 1
                    assert np.array_equal(full, orc.decode16(V[t_q], "f16"))
                    continue
                closed, open_cl = orc.pair_spans(sub)
                before = [(a, b) for a, b in closed if b < t_q]
                rows = orc.stored_rows(t_q + 1, before, policy)
                if policy == orc.POLICY_PAPER:
                    # <CL> rows of spans still open or just closed are stored but never attended to
                    rows = np.array([r for r in rows if sub[r] != CL], dtype=np.int64)
                compact = orc.attend(q, K, V, None, rows, "f16", 0.5)
                assert np.max(np.abs(full - compact)) <= 1e-12
                n_checked += 1
    assert n_checked > 2000


@pytest.mark.parametrize("policy", [orc.POLICY_PAPER, orc.POLICY_KEEP_CL])
def test_bruteforce_stored_rows_vs_next_query(policy):
    """After freeing every closed span, the kept rows are exactly what a next normal query sees,
    plus (paper policy) the <CL> row of a span that is still open."""
    for n in range(1, 9):
        for kinds in _all_wellformed(n):
            closed, open_cl = orc.pair_spans(kinds)
            rows = set(orc.stored_rows(n, closed, policy).tolist())
            hist = np.concatenate([kinds, np.uint8([NORMAL])])
            vis = set(np.nonzero(orc.visible(hist, n, policy))[0].tolist()) - {n}
            extra = {open_cl} if (open_cl >= 0 and policy == orc.POLICY_PAPER) else set()
            assert rows == vis | extra


def test_bruteforce_dependence_on_values():
    """Perturbing a row's K/V changes a query's output exactly when the mask shows that row:
    tokens after a <CR> are unaffected by the span's interior (Sec. 1), <CL> rows never
    affect later queries under the paper policy (Sec. 3.1)."""
    rng = np.random.default_rng(6)
    d = 4
    for n in range(2, 8):
        for kinds in _all_wellformed(n):
            pos = orc.tied_positions(kinds)
            K = _rand_bits(rng, (1, n, d))
            V = _rand_bits(rng, (1, n, d))
            q = _rand_bits(rng, (1, 1, d))
            t_q = n - 1
            base = orc.masked_decode([kinds], [pos], [K], [V], q, "f16", 0.7)[0, 0]
            vis = orc.visible(kinds, t_q)
            for j in range(n):
                K2, V2 = K.copy(), V.copy()
                V2[0, j] = orc.encode16(orc.decode16(V2[0, j], "f16") + 1.0, "f16")
                K2[0, j] = orc.encode16(orc.decode16(K2[0, j], "f16") + 0.5, "f16")
                out = orc.masked_decode([kinds], [pos], [K2], [V2], q, "f16", 0.7)[0, 0]
                changed = np.max(np.abs(out - base)) > 0
                assert changed == bool(vis[j]), (kinds, j)
                # the intro's rule: tokens after a <CR> never depend on that span's interior
                closed, _ = orc.pair_spans(kinds)
                for a, b in closed:
                    if b < t_q and a < j < b:
                        assert not changed
                if kinds[j] == CL and j != t_q:
                    assert not changed


# --------------------------------------------------------------------------
# Attention arithmetic: library routine in the span-free case
# --------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_spanfree_equals_sdpa(dtype):
    rng = np.random.default_rng(7)
    H, T, d = 3, 57, 16
    kinds = np.zeros(T, dtype=np.uint8)
    pos = orc.tied_positions(kinds)
    K = _rand_bits(rng, (H, T, d), dtype)
    V = _rand_bits(rng, (H, T, d), dtype)
    q = _rand_bits(rng, (1, H, d), dtype)
    scale = 0.3
    ours = orc.masked_decode([kinds], [pos], [K], [V], q, dtype, scale)[0]
    Kt = torch.from_numpy(orc.decode16(K, dtype))
    Vt = torch.from_numpy(orc.decode16(V, dtype))
    qt = torch.from_numpy(orc.decode16(q[0], dtype)).unsqueeze(1)  # [H, 1, d]
    ref = torch.nn.functional.scaled_dot_product_attention(qt, Kt, Vt, scale=scale)[:, 0].numpy()
    assert np.max(np.abs(ours - ref)) < 1e-12
    # intermediate queries: causal attention over the prefix
    for t in (0, 1, 20):
        o = orc.attend(q[0, 1], K[1], V[1], pos, np.arange(t + 1), dtype, scale)
        r = torch.nn.functional.scaled_dot_product_attention(qt[1:2], Kt[1:2, :t + 1], Vt[1:2, :t + 1],
                                                             scale=scale)[0, 0].numpy()
        assert np.max(np.abs(o - r)) < 1e-12


def test_zero_query_is_mean_of_visible_values():
    rng = np.random.default_rng(8)
    kinds, spans = wl.block_kinds(300, 20)
    hist = np.concatenate([kinds, np.uint8([NORMAL, CL, NORMAL, NORMAL])])  # an open span at the end
    T = hist.size
    pos = orc.tied_positions(hist)
    K = _rand_bits(rng, (1, T, 8))
    V = _rand_bits(rng, (1, T, 8))
    q = np.zeros((1, 1, 8), dtype=np.uint16)
    out = orc.masked_decode([hist], [pos], [K], [V], q, "f16", 1.0)[0, 0]
    vis = orc.visible(hist, T - 1)
    expect = orc.decode16(V[0][vis], "f16").mean(axis=0)
    assert np.max(np.abs(out - expect)) < 1e-12
    # closed form: 4 blocks of 64 keep 64-20-1 each; the tail 256..299 holds one more span
    # (<CL> 263, 20 enclosed, <CR> 284) leaving 44-21 = 23; then NORMAL, (<CL> hidden), NORMAL, NORMAL
    assert vis.sum() == 4 * 43 + 23 + 3


def test_one_hot_values_give_probabilities():
    rng = np.random.default_rng(9)
    hist = np.array([NORMAL, NORMAL, CL, NORMAL, NORMAL, CR, NORMAL, NORMAL], dtype=np.uint8)
    T = hist.size
    d = 8
    pos = orc.tied_positions(hist)
    K = _rand_bits(rng, (1, T, d))
    V = np.zeros((1, T, d), dtype=np.uint16)
    for j in range(T):
        V[0, j, j] = 0x3C00  # 1.0 in binary16
    q = _rand_bits(rng, (1, 1, d))
    p = orc.masked_decode([hist], [pos], [K], [V], q, "f16", 0.5)[0, 0]
    assert abs(p.sum() - 1) < 1e-14
    # query 7 (after the <CR> at 5): <CL> 2 and enclosed 3, 4 get exactly zero
    assert p[2] == 0 and p[3] == 0 and p[4] == 0
    kf = orc.decode16(K[0], "f16")
    qf = orc.decode16(q[0, 0], "f16")
    z = 0.5 * kf[[0, 1, 5, 6, 7]] @ qf
    w = np.exp(z - z.max())
    assert np.max(np.abs(p[[0, 1, 5, 6, 7]] - w / w.sum())) < 1e-14


# --------------------------------------------------------------------------
# RoPE
# --------------------------------------------------------------------------

def test_rope_matches_complex_rotation():
    rng = np.random.default_rng(10)
    for d, rot in [(80, 80), (64, 64), (80, 32), (2, 2)]:
        x = rng.standard_normal(d)
        for p in (0.0, 1.0, 17.0, 8191.0):
            y = orc.rope(x, rot, 10000.0, p)
            h = rot // 2
            theta = p * 10000.0 ** (-2.0 * np.arange(h) / rot)
            z = (x[:h] + 1j * x[h:rot]) * np.exp(1j * theta)
            tol = 1e-14 * (1.0 + p)  # 1-ulp differences in theta grow with the position
            assert np.allclose(y[:h], z.real, atol=tol, rtol=0)
            assert np.allclose(y[h:rot], z.imag, atol=tol, rtol=0)
            assert np.array_equal(y[rot:], x[rot:])
            assert math.isclose(np.linalg.norm(y), np.linalg.norm(x), rel_tol=1e-12)


def test_rope_relative_position_identity():
    rng = np.random.default_rng(11)
    q = rng.standard_normal(80)
    k = rng.standard_normal(80)
    a = orc.rope(q, 80, 1e4, 100) @ orc.rope(k, 80, 1e4, 37)
    b = orc.rope(q, 80, 1e4, 100 + 555) @ orc.rope(k, 80, 1e4, 37 + 555)
    assert abs(a - b) < 1e-9
    x = np.array([0.3, -1.2])
    y = orc.rope(x, 2, 1e4, 1.0)
    R = np.array([[math.cos(1.0), -math.sin(1.0)], [math.sin(1.0), math.cos(1.0)]])
    assert np.allclose(y, R @ x, atol=1e-15)


def test_rope_attention_depends_on_relative_positions_only():
    # with RoPE and unrounded inputs, shifting every position by s leaves the output unchanged up to the
    # storage rounding of rotated K; with K stored rounded the difference stays at rounding level
    rng = np.random.default_rng(12)
    T, d = 40, 16
    kinds = np.zeros(T, dtype=np.uint8)
    pos = orc.tied_positions(kinds)
    K = _rand_bits(rng, (1, T, d))
    V = _rand_bits(rng, (1, T, d))
    q = _rand_bits(rng, (1, 1, d))
    a = orc.masked_decode([kinds], [pos], [K], [V], q, "f16", 0.25, rot=d)[0, 0]
    b = orc.masked_decode([kinds], [pos + 1000], [K], [V], q, "f16", 0.25, rot=d)[0, 0]
    assert np.max(np.abs(a - b)) < 5e-3
    c = orc.masked_decode([kinds], [pos], [K], [V], q, "f16", 0.25, rot=0)[0, 0]
    assert np.max(np.abs(a - c)) > 1e-3  # the rotation is really applied


# --------------------------------------------------------------------------
# Local Attention baseline (Sec. 4.1)
# --------------------------------------------------------------------------

def test_local_window_closed_form_and_fifo_growth():
    for r in (0.0, 0.3, 0.5, 0.75, 0.9):
        prev_first = 0
        for t in range(0, 400):
            vis = orc.visible_local(t, r)
            first = int(np.argmax(vis))
            # 1-based x_{t+1} attends within (floor((t+1) r), t+1]: a contiguous window ending at the query
            assert vis[t] and vis[first:].all() and not vis[:first].any()
            assert first == math.floor((t + 1) * r)
            # FIFO: the window's left end never moves back, and it admits exactly one new token per step
            assert first >= prev_first
            prev_first = first
        # r = 0 is plain causal attention
        assert orc.visible_local(57, 0.0).all()


def test_local_decode_equals_sdpa_over_the_window():
    rng = np.random.default_rng(13)
    H, T, d = 2, 90, 16
    K = _rand_bits(rng, (H, T, d))
    V = _rand_bits(rng, (H, T, d))
    q = _rand_bits(rng, (1, H, d))
    pos = np.arange(T, dtype=np.int32)
    for r in (0.0, 0.5, 0.8):
        ours = orc.local_decode([pos], [K], [V], q, "f16", 0.4, r)[0]
        first = math.floor(T * r)
        Kt = torch.from_numpy(orc.decode16(K[:, first:], "f16"))
        Vt = torch.from_numpy(orc.decode16(V[:, first:], "f16"))
        qt = torch.from_numpy(orc.decode16(q[0], "f16")).unsqueeze(1)
        ref = torch.nn.functional.scaled_dot_product_attention(qt, Kt, Vt, scale=0.4)[:, 0].numpy()
        assert np.max(np.abs(ours - ref)) < 1e-12


# --------------------------------------------------------------------------
# Masked prefill (Sec. 3.1: the mask over every token of a prompt block)
# --------------------------------------------------------------------------

def _sdpa(q, k, v, scale, mask=None, causal=False):
    """fp64 library attention: q [H, Tq, d], k/v [H, Tk, d]."""
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q), torch.from_numpy(k), torch.from_numpy(v), scale=scale,
        attn_mask=None if mask is None else torch.from_numpy(mask), is_causal=causal).numpy()


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_prefill_spanfree_equals_causal_sdpa(dtype):
    """No spans: every query of the block is plain causal attention (library routine)."""
    rng = np.random.default_rng(21)
    H, d, scale = 3, 16, 0.35
    Ts, nqs = [70, 41], [70, 13]
    kinds_l = [np.zeros(T, np.uint8) for T in Ts]
    pos_l = [orc.tied_positions(k) for k in kinds_l]
    K_l = [_rand_bits(rng, (H, T, d), dtype) for T in Ts]
    V_l = [_rand_bits(rng, (H, T, d), dtype) for T in Ts]
    Q_full = [_rand_bits(rng, (T, H, d), dtype) for T in Ts]
    Q = np.concatenate([q[T - n:] for q, T, n in zip(Q_full, Ts, nqs)])
    ours = orc.masked_prefill(kinds_l, pos_l, K_l, V_l, nqs, Q, dtype, scale)
    row = 0
    for s, (T, n) in enumerate(zip(Ts, nqs)):
        qf = orc.decode16(Q_full[s], dtype).transpose(1, 0, 2)  # [H, T, d]
        ref = _sdpa(qf, orc.decode16(K_l[s], dtype), orc.decode16(V_l[s], dtype), scale, causal=True)
        got = ours[row:row + n].transpose(1, 0, 2)
        assert np.max(np.abs(got - ref[:, T - n:])) < 1e-12
        row += n


@pytest.mark.parametrize("policy", [orc.POLICY_PAPER, orc.POLICY_KEEP_CL])
@pytest.mark.parametrize("rot", [0, 16])
def test_prefill_equals_sdpa_with_the_mask_matrix(policy, rot):
    """With spans (closed, open, at the block's edges) and RoPE: the block's outputs equal library
    attention with a boolean mask whose row t is the query-t mask, on keys rotated at their tied
    positions and rounded to the cache type, and queries rotated at theirs."""
    rng = np.random.default_rng(22 + rot + policy)
    H, d, scale, base = 2, 16, 0.3, 10000.0
    kinds_l = [np.concatenate([wl.block_kinds(128, 20)[0], _random_wellformed(rng, 61)]),
               _random_wellformed(rng, 97, p_open=0.3, p_close=0.3)]
    nqs = [100, 97]
    pos_l = [orc.tied_positions(k) for k in kinds_l]
    K_l = [_rand_bits(rng, (H, k.size, d)) for k in kinds_l]
    V_l = [_rand_bits(rng, (H, k.size, d)) for k in kinds_l]
    Q_full = [_rand_bits(rng, (k.size, H, d)) for k in kinds_l]
    Q = np.concatenate([q[q.shape[0] - n:] for q, n in zip(Q_full, nqs)])
    ours = orc.masked_prefill(kinds_l, pos_l, K_l, V_l, nqs, Q, "f16", scale, rot=rot, base=base, policy=policy)
    row = 0
    for s, kinds in enumerate(kinds_l):
        T, n = kinds.size, nqs[s]
        mask = np.zeros((n, T), dtype=bool)
        for i in range(n):
            t = T - n + i
            mask[i, :t + 1] = orc.visible(kinds[:t + 1], t, policy)
        pos = pos_l[s]
        kf = orc.decode16(K_l[s], "f16")
        qf = orc.decode16(Q_full[s][T - n:], "f16").transpose(1, 0, 2)
        if rot:
            kf = np.stack([[orc.decode16(orc.encode16(orc.rope(kf[h, j], rot, base, pos[j]), "f16"), "f16")
                            for j in range(T)] for h in range(H)])
            qf = np.stack([[orc.rope(qf[h, i], rot, base, pos[T - n + i]) for i in range(n)] for h in range(H)])
        ref = _sdpa(qf, kf, orc.decode16(V_l[s], "f16"), scale, mask=mask)
        got = ours[row:row + n].transpose(1, 0, 2)
        assert np.max(np.abs(got - ref)) < 1e-12
        # Sec. 3.1: a <CL> query attends only to itself -> exactly its value row
        for i in range(n):
            if kinds[T - n + i] == CL:
                assert np.array_equal(got[:, i], orc.decode16(V_l[s][:, T - n + i], "f16"))
        row += n
    assert any((k == CL).any() for k in kinds_l)


def test_prefill_row_equals_decode_at_its_prefix():
    """Query t of a prefill block is the decode step whose history ends at t."""
    rng = np.random.default_rng(23)
    H, d = 2, 8
    kinds = np.concatenate([wl.block_kinds(64, 30)[0], np.uint8([NORMAL, CL, NORMAL, NORMAL, CR, NORMAL])])
    T = kinds.size
    pos = orc.tied_positions(kinds)
    K = _rand_bits(rng, (H, T, d))
    V = _rand_bits(rng, (H, T, d))
    Q = _rand_bits(rng, (T, H, d))
    pre = orc.masked_prefill([kinds], [pos], [K], [V], [T], Q, "f16", 0.6, rot=8)
    for t in (0, 6, 7, 8, 38, 39, 40, 63, 64, 65, 66, 68, 69):
        dec = orc.masked_decode([kinds[:t + 1]], [pos[:t + 1]], [K[:, :t + 1]], [V[:, :t + 1]], Q[t:t + 1], "f16",
                                0.6, rot=8)[0]
        assert np.array_equal(pre[t], dec)
