"""The C ABI on the host (CPU only): exported symbols, argument/state errors, and the span book
(a2: span bookkeeping, positions, stored rows, mask) against the fp64 oracle, bit-exact."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as orc
import paper_2310_08152_gb300 as kvc
from paper_2310_08152_gb300 import _lib
from synth import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
NORMAL, CL, CR = kvc.NORMAL, kvc.CL, kvc.CR


def declared_functions():
    text = open(os.path.join(ROOT, "include", "kvc.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvc_[a-z_]+)\s*\(", text)))


def test_library_exports_every_declared_function():
    names = declared_functions()
    assert len(names) >= 20
    L = kvc.lib()
    for n in names:
        assert hasattr(L, n), n
    assert sorted(n for n, _, _ in _lib.SIGNATURES) == names


def test_status_strings():
    L = kvc.lib()
    for s in range(10):
        assert L.kvc_status_string(s)
    assert L.kvc_status_string(0) == b"ok"


# --------------------------------------------------------------------------------------------
# book vs oracle
# --------------------------------------------------------------------------------------------

def _random_kinds(rng, n, open_=False):
    kinds = np.zeros(n, np.uint8)
    for t in range(n):
        r = rng.random()
        if not open_ and r < 0.12:
            kinds[t] = CL
            open_ = True
        elif open_ and r < 0.15:
            kinds[t] = CR
            open_ = False
    return kinds, open_


@pytest.mark.parametrize("policy", [kvc.POLICY_PAPER, kvc.POLICY_KEEP_CL])
def test_book_matches_oracle_random_histories(policy):
    rng = np.random.default_rng(20)
    b = 4
    cap = np.full(b, 4000, np.int64)
    book = kvc.Book(b, cap, policy)
    hist = [np.zeros(0, np.uint8) for _ in range(b)]
    freed = [[] for _ in range(b)]
    open_ = [False] * b
    for rnd in range(40):
        n_new = rng.integers(0, 12, size=b).astype(np.int32)
        parts = []
        for s in range(b):
            k, open_[s] = _random_kinds(rng, int(n_new[s]), open_[s])
            parts.append(k)
        kinds = np.concatenate(parts)
        pos = book.append(n_new, kinds)
        # positions continue each history with the tie rule
        off = 0
        for s in range(b):
            hist[s] = np.concatenate([hist[s], parts[s]])
            expect = orc.tied_positions(hist[s])[hist[s].size - n_new[s]:]
            assert np.array_equal(pos[off:off + n_new[s]], expect)
            off += n_new[s]
        # free a random subset of the pending spans
        seq, cl, cr = [], [], []
        for s in range(b):
            for a, c in book.pending_spans(s):
                if rng.random() < 0.6:
                    seq.append(s)
                    cl.append(a)
                    cr.append(c)
                    freed[s].append((a, c))
        if seq:
            book.compress(seq, cl, cr)
        ln, at = book.lengths()
        for s in range(b):
            lay = book.layout(s)
            T = hist[s].size
            assert np.array_equal(lay["kinds"], hist[s])
            rows = orc.stored_rows(T, freed[s], policy)
            assert np.array_equal(lay["stored_orig"], rows)
            assert ln[s] == rows.size
            assert np.array_equal(lay["stored_pos"], orc.tied_positions(hist[s])[rows])
            closed, _ = orc.pair_spans(hist[s])
            assert book.pending_spans(s) == [sp for sp in closed if sp not in freed[s]]
            if T:
                vis = orc.visible(hist[s], T - 1, policy)
                assert np.array_equal(lay["visible"], vis)
                # rows the next decode reads: the visible ones, when every hidden row sits in one run
                hidden = set(rows.tolist()) - set(np.nonzero(vis)[0].tolist())
                idx = sorted(np.searchsorted(rows, list(hidden)))
                one_run = not idx or idx[-1] - idx[0] + 1 == len(idx)
                if one_run or hist[s][T - 1] == CL:
                    # the decode reads exactly the stored rows the mask shows (a <CR> query whose span
                    # was already freed sees the rows that are left)
                    assert at[s] == vis[rows].sum()
                else:
                    assert at[s] == 0


def test_book_workload_counts():
    for w in (wl.tiny(), wl.opt13b(b=2), wl.rope3b(45, b=1)):
        book = kvc.Book(w.b, w.capacity(0), kvc.POLICY_PAPER)
        book.append(w.prompt_len.astype(np.int32), np.concatenate(w.prompt_kinds))
        seq = [s for s in range(w.b) for _ in w.prompt_spans[s]]
        cl = [a for s in range(w.b) for a, _ in w.prompt_spans[s]]
        cr = [c for s in range(w.b) for _, c in w.prompt_spans[s]]
        book.compress(seq, cl, cr)
        ln, at = book.lengths()
        L = int(w.prompt_len[0])
        I = w.prompt_spans[0][0][1] - w.prompt_spans[0][0][0] - 1
        assert np.all(ln == (L // 64) * (64 - I - 1))


# --------------------------------------------------------------------------------------------
# host-side errors
# --------------------------------------------------------------------------------------------

def _err(fn, *a):
    with pytest.raises(kvc.KvcError) as e:
        fn(*a)
    return e.value.status


def test_book_span_errors_leave_state_unchanged():
    book = kvc.Book(2, [100, 100])
    book.append([3, 1], [NORMAL, CL, NORMAL, NORMAL])
    before = (book.layout(0), book.layout(1), book.lengths())
    assert _err(book.append, [1, 0], [CL]) == 4          # <CL> inside the open span of sequence 0
    assert _err(book.append, [0, 1], [CR]) == 4          # <CR> without an open span in sequence 1
    assert _err(book.append, [0, 200], [NORMAL] * 200) == 3  # capacity
    assert _err(book.append, [1, 0], [7]) == 1           # not a kind
    assert _err(book.append, [-1, 0], []) == 1
    after = (book.layout(0), book.layout(1), book.lengths())
    for x, y in zip(before[:2], after[:2]):
        for key in x:
            assert np.array_equal(x[key], y[key])
    book.append([2, 0], [NORMAL, CR])
    assert book.pending_spans(0) == [(1, 4)]
    assert _err(book.compress, [0], [0], [4]) == 4       # not a span
    assert _err(book.compress, [0], [1], [3]) == 4       # wrong <CR>
    assert _err(book.compress, [0, 0], [1, 1], [4, 4]) == 4  # listed twice
    assert _err(book.compress, [5], [1], [4]) == 4       # sequence out of range
    book.compress([0], [1], [4])
    assert _err(book.compress, [0], [1], [4]) == 4       # already freed
    assert book.lengths()[0][0] == 2


def test_book_open_span_cannot_be_freed():
    book = kvc.Book(1, [50])
    book.append([3], [NORMAL, CL, NORMAL])
    assert _err(book.compress, [0], [1], [3]) == 4


def test_decode_view_needs_spans_freed():
    # two closed spans that are not freed leave two hidden runs: the next decode must refuse
    book = kvc.Book(1, [50])
    book.append([9], [NORMAL, CL, NORMAL, CR, NORMAL, CL, NORMAL, CR, NORMAL])
    ln, at = book.lengths()
    assert at[0] == 0
    book.compress([0], [1], [3])
    ln, at = book.lengths()
    assert at[0] == orc.visible(np.array([0, 1, 0, 2, 0, 1, 0, 2, 0], np.uint8), 8).sum()


def test_cache_config_errors_on_host():
    cfg, cap = kvc.make_config(2, 4, 72, [16, 16])
    assert _err(kvc.kvc_required_bytes, cfg) == 2        # d_head not built
    cfg, cap = kvc.make_config(2, 4, 64, [16, 16], rotary_dim=24)
    assert _err(kvc.kvc_required_bytes, cfg) == 2        # rotary_dim not a multiple of 16
    cfg, cap = kvc.make_config(2, 4, 64, [16, 0])
    assert _err(kvc.kvc_required_bytes, cfg) == 1
    cfg, cap = kvc.make_config(2, 4, 64, [16, 16])
    sizes = kvc.kvc_required_bytes(cfg)
    assert sizes["k"] == 2 * 4 * 32 * 64 * 2 and sizes["meta"] == 32 * 4
    assert _err(kvc.kvc_create, cfg) == 1                # NULL device buffers
    cfg.k_base = cfg.v_base = cfg.pos_base = cfg.orig_base = cfg.workspace = 0x1000 + 8
    cfg.workspace_bytes = sizes["workspace"]
    assert _err(kvc.kvc_create, cfg) == 1                # unaligned


def test_cache_validates_before_any_device_work():
    # Fake (never dereferenced) addresses: every call below must fail on the host before touching CUDA.
    cfg, cap = kvc.make_config(2, 4, 64, [16, 16])
    sizes = kvc.kvc_required_bytes(cfg)
    cfg.k_base = cfg.v_base = cfg.pos_base = cfg.orig_base = cfg.workspace = 1 << 40
    cfg.workspace_bytes = sizes["workspace"]
    h = kvc.kvc_create(cfg)
    try:
        fake = 1 << 40
        L = kvc.lib()
        n_new = np.array([1, 1], np.int32)
        pos = np.zeros(2, np.int32)
        assert L.kvc_append(h, 5, fake, fake, n_new.ctypes.data, pos.ctypes.data, np.uint8([0, 0]).ctypes.data,
                            None) == 1
        assert L.kvc_append(h, -1, fake, fake, n_new.ctypes.data, pos.ctypes.data, np.uint8([2, 0]).ctypes.data,
                            None) == 4
        big = np.array([17, 0], np.int32)
        assert L.kvc_append(h, -1, fake, fake, big.ctypes.data, np.zeros(17, np.int32).ctypes.data,
                            np.zeros(17, np.uint8).ctypes.data, None) == 3
        assert L.kvc_append(h, 1, fake, fake, None, None, None, None) == 5   # layer 1 before layer 0
        # inputs the bulk copies cannot start from: not 16-byte aligned
        assert L.kvc_append(h, -1, fake + 8, fake, n_new.ctypes.data, pos.ctypes.data, np.uint8([0, 0]).ctypes.data,
                            None) == 1
        assert L.kvc_append(h, 0, fake, fake + 2, n_new.ctypes.data, pos.ctypes.data, np.uint8([0, 0]).ctypes.data,
                            None) == 1
        assert L.kvc_decode_attention(h, 0, fake, ctypes.c_float(0.125), fake, None) == 5  # nothing appended
        assert L.kvc_decode_attention(h, 9, fake, ctypes.c_float(0.125), fake, None) == 1
        n = 2 * 4 * 64
        assert L.kvc_decode_attention_layers(h, 1, 2, fake, n, ctypes.c_float(0.125), fake, n, None) == 1  # > M
        assert L.kvc_decode_attention_layers(h, 0, 2, fake, n - 1, ctypes.c_float(0.125), fake, n, None) == 1
        assert L.kvc_decode_attention_layers(h, 0, 2, fake, n, ctypes.c_float(0.125), fake, n, None) == 5
        assert L.kvc_decode_attention_layers(h, 0, 0, None, 0, ctypes.c_float(0.125), None, 0, None) == 0
        assert L.kvc_compress_spans(h, np.int32([0]).ctypes.data, np.int64([0]).ctypes.data,
                                    np.int64([1]).ctypes.data, 1, None) == 4
        assert b"span" in L.kvc_last_error() or b"closed" in L.kvc_last_error()
    finally:
        kvc.kvc_destroy(h)


def test_cache_fails_loudly_without_a_gpu():
    import torch

    if torch.cuda.is_available():
        pytest.skip("only meaningful where no GPU exists (it would dereference fake addresses)")
    cfg, cap = kvc.make_config(1, 2, 64, [8])
    sizes = kvc.kvc_required_bytes(cfg)
    cfg.k_base = cfg.v_base = cfg.pos_base = cfg.orig_base = cfg.workspace = 1 << 40
    cfg.workspace_bytes = sizes["workspace"]
    h = kvc.kvc_create(cfg)
    try:
        L = kvc.lib()
        rc = L.kvc_append(h, -1, 1 << 40, 1 << 40, np.int32([1]).ctypes.data, np.int32([0]).ctypes.data,
                          np.uint8([0]).ctypes.data, None)
        assert rc == 6  # KVC_ERR_CUDA: no silent CPU path
    finally:
        kvc.kvc_destroy(h)


@pytest.mark.parametrize("policy", [kvc.POLICY_PAPER, kvc.POLICY_KEEP_CL])
def test_book_write_time_freeing_matches_oracle(policy):
    """Spans opened and closed within one append are freed as they are written (Sec. 3.1, freeing in
    one go / block by block); the stored rows equal the oracle's rows left after freeing them, and a
    later compaction of the spans that straddled calls gives the same rows as freeing everything."""
    rng = np.random.default_rng(21)
    b = 3
    book = kvc.Book(b, np.full(b, 5000, np.int64), policy)
    hist = [np.zeros(0, np.uint8) for _ in range(b)]
    freed = [[] for _ in range(b)]
    open_ = [False] * b
    for rnd in range(30):
        n_new = rng.integers(0, 40, size=b).astype(np.int32)
        parts = []
        for s in range(b):
            k, open_[s] = _random_kinds(rng, int(n_new[s]), open_[s])
            parts.append(k)
        book.append(n_new, np.concatenate(parts), free_closed=True)
        for s in range(b):
            T0 = hist[s].size
            hist[s] = np.concatenate([hist[s], parts[s]])
            closed, _ = orc.pair_spans(hist[s])
            freed[s] += [(a, c) for a, c in closed if a >= T0]  # opened and closed in this call
        ln, _ = book.lengths()
        for s in range(b):
            rows = orc.stored_rows(hist[s].size, freed[s], policy)
            assert np.array_equal(book.layout(s)["stored_orig"], rows)
            assert ln[s] == rows.size
            closed, _ = orc.pair_spans(hist[s])
            assert book.pending_spans(s) == [sp for sp in closed if sp not in freed[s]]
    # free what straddled calls: the same rows as freeing every closed span
    seq, cl, cr = [], [], []
    for s in range(b):
        for a, c in book.pending_spans(s):
            seq.append(s)
            cl.append(a)
            cr.append(c)
    if seq:
        book.compress(seq, cl, cr)
    for s in range(b):
        closed, _ = orc.pair_spans(hist[s])
        assert np.array_equal(book.layout(s)["stored_orig"], orc.stored_rows(hist[s].size, closed, policy))


def test_write_time_freeing_capacity_counts_stored_rows():
    book = kvc.Book(1, [5])
    # 9 tokens, of which <CL> and 4 enclosed are freed at write time: 4 stored rows fit capacity 5
    book.append([9], [NORMAL, CL, NORMAL, NORMAL, NORMAL, NORMAL, CR, NORMAL, NORMAL], free_closed=True)
    assert book.lengths()[0][0] == 4
    assert _err(book.append, [2], [NORMAL, NORMAL]) == 3


@pytest.mark.parametrize("ratio", [0.0, 0.3, 0.5, 0.8])
def test_local_book_window_matches_oracle(ratio):
    """The Local Attention FIFO cache (Sec. 4.1/4.2) keeps exactly the window the mask shows."""
    rng = np.random.default_rng(22)
    r32 = float(np.float32(ratio))
    cap = np.array([700, 700], np.int64)
    book = kvc.Book(2, cap, kvc.POLICY_LOCAL, local_ratio=ratio)
    T = [0, 0]
    for _ in range(25):
        n_new = rng.integers(0, 30, size=2).astype(np.int32)
        book.append(n_new, np.zeros(int(n_new.sum()), np.uint8))
        ln, at = book.lengths()
        for s in range(2):
            T[s] += int(n_new[s])
            if not T[s]:
                continue
            vis = orc.visible_local(T[s] - 1, r32)
            lay = book.layout(s)
            assert np.array_equal(lay["visible"], vis)
            assert np.array_equal(lay["stored_orig"], np.nonzero(vis)[0])
            assert ln[s] == at[s] == vis.sum()
    assert _err(book.append, [1, 0], [CL]) == 4  # no sentinels in a local-attention cache


def test_local_book_capacity_is_the_window():
    book = kvc.Book(1, [10], kvc.POLICY_LOCAL, local_ratio=0.5)
    book.append([19], np.zeros(19, np.uint8))  # x_19 sees (9, 19]: 10 rows
    assert book.lengths()[0][0] == 10
    book.append([1], [NORMAL])  # x_20 sees (10, 20]: still 10
    assert _err(book.append, [2], [NORMAL, NORMAL]) == 3  # x_22 would see (11, 22]: 11 rows


def _wellformed(n):
    import itertools
    for seq in itertools.product((NORMAL, CL, CR), repeat=n):
        open_ = False
        ok = True
        for k in seq:
            if (k == CL and open_) or (k == CR and not open_):
                ok = False
                break
            if k != NORMAL:
                open_ = k == CL
        if ok:
            yield np.array(seq, np.uint8)


def _prefill_visible(meta, iq):
    """The documented prefill rule: row i is visible to the query at stored row iq iff
    i <= iq <= hid(i), and a <CL> query (its own is_cl bit) sees only itself."""
    hid = meta >> 1
    i = np.arange(meta.size)
    vis = (i <= iq) & (iq <= hid)
    if meta[iq] & 1:
        vis = i == iq
    return vis


@pytest.mark.parametrize("policy", [kvc.POLICY_PAPER, kvc.POLICY_KEEP_CL])
def test_book_prefill_mask_bounds_match_oracle_bruteforce(policy):
    """Every well-formed history of up to 7 tokens, split into a first part (appended, its closed
    spans freed) and a prefill block: the per-row bounds give, for every query of the block, exactly
    the oracle's visible set mapped onto the stored rows (Sec. 3.1 mask)."""
    n_checked = 0
    for n in range(1, 8):
        for kinds in _wellformed(n):
            for k in range(n):  # block = tokens [k, n)
                book = kvc.Book(1, [n], policy)
                if k:
                    book.append([k], kinds[:k])
                    spans = book.pending_spans(0)
                    if spans:
                        book.compress([0] * len(spans), [a for a, _ in spans], [c for _, c in spans])
                book.append([n - k], kinds[k:])
                meta = book.prefill_keys(0, n - k)
                rows = book.layout(0)["stored_orig"]
                assert meta.size == rows.size
                for t in range(k, n):
                    iq = int(np.nonzero(rows == t)[0][0])
                    assert iq == rows.size - (n - t)  # the queries are the last stored rows
                    vis_hist = orc.visible(kinds[:t + 1], t, policy)
                    expect = np.zeros(rows.size, bool)
                    for r, j in enumerate(rows):
                        expect[r] = j <= t and vis_hist[j]
                    assert np.array_equal(_prefill_visible(meta, iq), expect), (kinds, k, t)
                    # nothing the query may see was freed
                    assert set(np.nonzero(vis_hist)[0]) <= set(rows.tolist())
                    n_checked += 1
    assert n_checked > 5000


def test_book_prefill_keys_errors():
    book = kvc.Book(1, [16])
    book.append([6], [NORMAL, CL, NORMAL, CR, NORMAL, NORMAL], free_closed=True)  # rows 1..2 freed
    assert _err(book.prefill_keys, 0, 5) == 5   # token 1 is not stored
    assert _err(book.prefill_keys, 0, 7) == 5   # more queries than tokens
    assert book.prefill_keys(0, 3).size == 4    # tokens 3..5 are the last stored rows
    assert book.prefill_keys(0, 0).size == 0
    local = kvc.Book(1, [16], kvc.POLICY_LOCAL, local_ratio=0.5)
    local.append([3], [NORMAL] * 3)
    assert _err(local.prefill_keys, 0, 1) == 2
