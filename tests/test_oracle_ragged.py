"""Pins for the oracle's page fills and ragged eviction (cache_model).

Ragged eviction packs only the pages a span touches and drops the rest by
remapping; every other operation must then read its rows through the page
fills.  What pins it, independently of the model's own code:
  * hand-worked layouts (page ids, fills, moved and zeroed rows);
  * the logical contents do not depend on the eviction mode: a twin cache
    that runs every eviction densely holds the same token ids, in order;
  * physical mode: reading each page's filled slots in page order gives the
    logical contents, and no unused slot of a page that ends early (not the
    last) is memory no row was ever written to (zeros or a row once appended);
  * reference counts equal the number of holders, the free set is the
    complement;
  * the work is O(spans x P): at most 2 P rows move per span, and pages
    outside the touched windows keep their ids and slots;
  * a fork alive during the eviction keeps its view (copy-on-write of the
    shared pages whose rows change), an empty span set changes nothing;
  * attention over the rows read back through the fills equals attention
    over the original rows with the evicted tokens masked out (Algorithm 2's
    BuildMask reading of Algorithm 1's clear_kv).
"""
import math
import random

import numpy as np
import pytest

from oracle import attention as oatt
from oracle import cache_model as ocm
from synthetic import bf16_bits, bf16_normal


def test_hand_worked_window_packing():
    c = ocm.OracleCache(8, 4, physical=True)
    s = c.seq_new()
    c.append(s, 14)                       # pages 0..3, fills 4 4 4 2
    assert c.page_table(s) == [0, 1, 2, 3] and c.page_fills(s) == [4, 4, 4, 2]
    r = c.evict(s, [(9, 10), (2, 5)], mode="ragged")
    # removed 2 3 4 9: pages 0, 1, 2 are touched and form one window; its
    # kept rows 0 1 5 6 7 8 10 11 fill pages 0 and 1; page 2 leaves
    assert c.tokens(s) == [0, 1, 5, 6, 7, 8, 10, 11, 12, 13]
    assert c.page_table(s) == [0, 1, 3] and c.page_fills(s) == [4, 4, 2]
    assert r["moved_rows"] == 6 and r["windows"] == 1 and r["zeroed_rows"] == 0
    assert r["released_pages"] == 1 and c.ref[2] == 0
    assert c.physical_tokens(s) == c.tokens(s)


def test_hand_worked_separate_windows_and_zeros():
    c = ocm.OracleCache(8, 4, physical=True)
    s = c.seq_new()
    c.append(s, 16)
    r = c.evict(s, [(13, 14), (1, 2)], mode="ragged")
    # pages 0 and 3 are touched, not adjacent: two windows, each packed in
    # place with one zeroed slot; pages 1 and 2 untouched
    assert c.page_table(s) == [0, 1, 2, 3] and c.page_fills(s) == [3, 4, 4, 3]
    assert r["windows"] == 2 and r["moved_rows"] == 4 and r["zeroed_rows"] == 2
    assert c.phys[0] == [0, 2, 3, ocm.ZERO] and c.phys[3] == [12, 14, 15, ocm.ZERO]
    assert c.phys[1] == [4, 5, 6, 7] and c.phys[2] == [8, 9, 10, 11]
    # an append after it fills the last page's free slot, then a new page
    ids = c.append(s, 2)
    assert ids == [16, 17]
    assert c.page_fills(s) == [3, 4, 4, 4, 1] and c.page_table(s) == [0, 1, 2, 3, 4]
    assert c.phys[3] == [12, 14, 15, 16] and c.phys[4][0] == 17
    assert c.physical_tokens(s) == c.tokens(s)
    # a dense eviction packs through the fills: every page full but the last
    c.evict(s, [(0, 1)])
    assert c.page_fills(s) == [4, 4, 4, 3] and c.page_table(s) == [0, 1, 2, 3]
    assert c.ref[4] == 0
    assert c.tokens(s) == [2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 14, 15, 16, 17]
    assert c.physical_tokens(s) == c.tokens(s)


def test_whole_pages_are_dropped_without_a_copy():
    c = ocm.OracleCache(40, 8, physical=True)
    s = c.seq_new()
    c.append(s, 200)                      # 25 full pages
    r = c.evict(s, [(16, 40), (80, 120)], mode="ragged")   # page-aligned spans
    # every removed row sits in a page the span covers whole: nothing moves,
    # nothing is zeroed, the five pages leave by remapping alone
    assert r["moved_rows"] == 0 and r["zeroed_rows"] == 0 and r["released_pages"] == 8
    assert c.page_table(s) == [0, 1] + list(range(5, 10)) + list(range(15, 25))
    assert c.page_fills(s) == [8] * 17
    assert c.physical_tokens(s) == c.tokens(s)


def test_shared_pages_are_copied_on_write():
    c = ocm.OracleCache(64, 8, physical=True)
    m = c.seq_new()
    c.append(m, 100)                      # pages 0..12 (fills 8 x 12, 4)
    a = c.fork(m)
    aux_view = c.physical_tokens(a)
    r = c.evict(m, [(20, 30), (70, 71)], mode="ragged")
    # windows: pages 2..3 (rows 16..31) and page 8 (rows 64..71); the pages
    # whose rows change are shared with the fork, so they are copied
    assert r["cow_pages"] == 2
    assert c.physical_tokens(a) == aux_view == c.tokens(a)
    assert c.physical_tokens(m) == c.tokens(m)
    pt_m, pt_a = c.page_table(m), c.page_table(a)
    assert pt_m[:2] == pt_a[:2] and all(c.ref[p] == 2 for p in pt_m[:2])
    # page 3 left main, so the second fresh page sits at index 7
    assert pt_m[2] == 13 and pt_m[7] == 14   # fresh pages, lowest ids, increasing order
    assert c.page_fills(m)[2] == 6 and c.page_fills(m)[7] == 7
    assert c.ref[pt_a[3]] == 1               # main dropped page 3, the fork still holds it


def test_empty_span_set_is_the_identity():
    c = ocm.OracleCache(30, 16, physical=True)
    s = c.seq_new()
    c.append(s, 300)
    c.evict(s, [(17, 40)], mode="ragged")
    before = (c.page_table(s), c.page_fills(s), list(c.ref), {p: list(v) for p, v in c.phys.items()})
    for mode in ("ragged", "dense"):
        r = c.evict(s, [], mode=mode)
        assert r["moved_rows"] == 0
        assert (c.page_table(s), c.page_fills(s), list(c.ref),
                {p: list(v) for p, v in c.phys.items()}) == before


def _invariants(c, P):
    holders = [0] * c.num_pages
    for sid, s in c.seqs.items():
        assert len(s.pages) == len(s.fills)
        assert all(1 <= f <= P for f in s.fills)
        assert sum(s.fills) == len(s.tokens)
        for p in s.pages:
            holders[p] += 1
        assert c.physical_tokens(sid) == c.tokens(sid)
        for p, f in zip(s.pages[:-1], s.fills[:-1]):
            if f < P:                     # a page that ends early: zeros or rows once appended
                assert all(x == ocm.ZERO or x >= 0 for x in c.phys[p][f:])
    assert holders == c.ref
    assert c.free_count() == sum(1 for r in c.ref if r == 0)


@pytest.mark.parametrize("seed", range(12))
def test_random_ops_against_a_dense_twin(seed):
    rng = random.Random(seed)
    P = rng.choice([4, 8, 16])
    rag = ocm.OracleCache(4000, P, physical=True)
    den = ocm.OracleCache(4000, P)
    ids = {}                              # ragged sid -> dense sid
    for step in range(60):
        live = list(ids)
        op = rng.random()
        if not live or op < 0.1:
            a = rag.seq_new()
            ids[a] = den.seq_new()
            n = rng.randint(1, 6 * P)
            assert rag.append(a, n) == den.append(ids[a], n)
        elif op < 0.25:
            src = rng.choice(live)
            a = rag.fork(src)
            ids[a] = den.fork(ids[src])
        elif op < 0.5:
            a = rng.choice(live)
            n = rng.choice([1, 1, 2, P - 1, P, P + 1, rng.randint(1, 5 * P)])
            assert rag.append(a, n) == den.append(ids[a], n)
        elif op < 0.85:
            a = rng.choice(live)
            n = rag.n_tokens(a)
            if n < 2:
                continue
            spans, pos = [], 0
            for _ in range(rng.randint(1, 6)):
                lo = rng.randint(pos, n - 1)
                hi = rng.randint(lo + 1, min(n, lo + 3 * P))
                spans.append((lo, hi))
                pos = hi
                if pos >= n - 1:
                    break
            rng.shuffle(spans)
            mode = rng.choice(["ragged", "ragged", "dense"])
            r = rag.evict(a, spans, mode=mode)
            den.evict(ids[a], spans)
            if mode == "ragged":
                assert r["moved_rows"] <= 2 * P * len(spans)
                assert r["zeroed_rows"] < P * max(1, r["windows"])
            else:
                f = rag.page_fills(a)
                assert all(x == P for x in f[:-1])
        else:
            a = rng.choice(live)
            rag.release(a)
            den.release(ids.pop(a))
        for a, d in ids.items():
            assert rag.tokens(a) == den.tokens(d)
        _invariants(rag, P)


def test_untouched_pages_keep_their_ids_and_slots():
    rng = random.Random(5)
    c = ocm.OracleCache(200, 16, physical=True)
    s = c.seq_new()
    c.append(s, 1500)
    for trial in range(8):
        n = c.n_tokens(s)
        a = rng.randint(0, n - 40)
        b = a + rng.randint(1, 40)
        untouched = []
        j = 0
        for p, f in zip(c.page_table(s), c.page_fills(s)):
            if j + f <= a or j >= b:
                untouched.append((p, f, list(c.phys[p][:f])))
            j += f
        r = c.evict(s, [(a, b)], mode="ragged")
        assert r["moved_rows"] <= 2 * 16
        after = {p: f for p, f in zip(c.page_table(s), c.page_fills(s))}
        order = [p for p in c.page_table(s) if p in {u[0] for u in untouched}]
        assert order == [u[0] for u in untouched]        # same pages, same order
        for p, f, rows in untouched:
            assert after[p] == f and c.phys[p][:f] == rows
        assert c.physical_tokens(s) == c.tokens(s)


def test_evict_then_attend_equals_masked_attention():
    P, L, Hq, Hkv, d = 8, 1, 8, 2, 64
    c = ocm.OracleCache(300, P, physical=True)
    s = c.seq_new()
    n = 700
    c.append(s, n)
    k = bf16_bits(bf16_normal((n, Hkv, d), 1))
    v = bf16_bits(bf16_normal((n, Hkv, d), 2))
    q = bf16_bits(bf16_normal((Hq, d), 3))
    spans = [(5, 9), (40, 200), (333, 334), (690, 700)]
    c.evict(s, spans, mode="ragged")
    # rows read back through the page table and the fills
    toks = []
    for p, f in zip(c.page_table(s), c.page_fills(s)):
        toks.extend(c.phys[p][:f])
    toks = np.array(toks)
    got = oatt.decode(q, k[toks], v[toks], 0.125)
    exp = oatt.decode(q, k, v, 0.125, mask=oatt.removed_mask(n, spans))
    np.testing.assert_allclose(got, exp, rtol=1e-12, atol=1e-13)
