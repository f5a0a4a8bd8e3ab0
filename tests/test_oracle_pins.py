"""Pins for the CPU oracle: each test checks the oracle against something other
than itself — a closed form, an invariant, brute force on tiny inputs, a
library routine, or a worked example from the paper — chosen so that a
plausible slip (a dropped term, a wrong sign or head index, a transposed
operand, an off-by-one page rule) fails at least one of them.
"""
import json
import math
import os
import random

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import cache_model as ocm
from synthetic import bf16_bits, bf16_normal

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def widen(bits: np.ndarray) -> np.ndarray:
    """bf16 bits -> float64, via torch (independent of the oracle's C code)."""
    t = torch.from_numpy(bits.astype(np.int16).copy()).view(torch.bfloat16)
    return t.to(torch.float64).numpy()


def rand_qkv(seed, n, Hq, Hkv, d, kscale=1.0):
    q = bf16_bits(bf16_normal((Hq, d), seed))
    k = bf16_bits(bf16_normal((n, Hkv, d), seed + 1, scale=kscale))
    v = bf16_bits(bf16_normal((n, Hkv, d), seed + 2))
    return q, k, v


def sdpa_f64(q, k, v, scale, mask=None):
    """torch scaled_dot_product_attention in float64 with K/V heads repeated
    for the query group (library routine)."""
    Hq, d = q.shape
    n, Hkv, _ = k.shape
    G = Hq // Hkv
    qt = torch.from_numpy(widen(q)).view(1, Hq, 1, d)
    kt = torch.from_numpy(widen(k)).permute(1, 0, 2).repeat_interleave(G, dim=0).unsqueeze(0)
    vt = torch.from_numpy(widen(v)).permute(1, 0, 2).repeat_interleave(G, dim=0).unsqueeze(0)
    am = None
    if mask is not None:
        am = torch.zeros(1, 1, 1, n, dtype=torch.float64)
        am[..., torch.from_numpy(mask.astype(bool))] = -math.inf
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=am, scale=scale)
    return o.view(Hq, d).numpy()


# ---------------------------------------------------------------------------
# decode attention
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("n,Hq,Hkv,d", [(1, 4, 4, 8), (37, 16, 4, 64), (300, 8, 1, 32), (129, 32, 8, 128)])
def test_softmax_weights_sum_to_one(n, Hq, Hkv, d):
    q, k, v = rand_qkv(11, n, Hq, Hkv, d)
    out, w, lse = oatt.decode(q, k, v, 1.0 / math.sqrt(d), want_weights=True, want_lse=True)
    assert np.all(w >= 0)
    np.testing.assert_allclose(w.sum(axis=1), 1.0, rtol=0, atol=1e-12)
    # out is exactly the weight-average of V (checked with numpy, float64)
    G = Hq // Hkv
    vf = widen(v)
    for h in range(Hq):
        np.testing.assert_allclose(out[h], w[h] @ vf[:, h // G, :], rtol=1e-12, atol=1e-12)


def test_single_token_returns_its_value():
    for d in (8, 64, 128):
        q, k, v = rand_qkv(5 + d, 1, 8, 2, d)
        out = oatt.decode(q, k, v, 0.37)
        vf = widen(v)
        for h in range(8):
            assert np.array_equal(out[h], vf[0, h // 4])  # exact: p = 1, l = 1


def test_constant_value_rows_give_that_constant():
    n, Hq, Hkv, d = 200, 8, 2, 16
    q, k, _ = rand_qkv(3, n, Hq, Hkv, d)
    c = bf16_bits(bf16_normal((1, Hkv, d), 99))
    v = np.ascontiguousarray(np.broadcast_to(c, (n, Hkv, d)))
    out = oatt.decode(q, k, v, 0.2)
    cf = widen(c)[0]
    for h in range(Hq):
        np.testing.assert_allclose(out[h], cf[h // 4], rtol=1e-13, atol=1e-14)


def test_zero_keys_give_mean_of_values():
    n, Hq, Hkv, d = 97, 4, 4, 32
    q, _, v = rand_qkv(7, n, Hq, Hkv, d)
    k = np.zeros((n, Hkv, d), dtype=np.uint16)  # +0.0 bits
    out = oatt.decode(q, k, v, 1.0)
    vf = widen(v)
    for h in range(Hq):
        np.testing.assert_allclose(out[h], vf[:, h].mean(axis=0), rtol=1e-12, atol=1e-14)


def test_two_tokens_logistic_closed_form():
    # With two tokens the softmax weight of token 1 is sigmoid(s1 - s0):
    # o = V0 + sigmoid(s1 - s0) * (V1 - V0).  Keys are chosen so that the
    # logits are known exactly: K0 = 0, K1 = e_0 (unit vector), q[0] = x.
    d = 16
    for x in (-3.0, -0.5, 0.0, 0.75, 2.0, 9.0):
        q = np.zeros((1, d), dtype=np.float32)
        q[0, 0] = x
        qb = bf16_bits(torch.from_numpy(q).to(torch.bfloat16))
        k = np.zeros((2, 1, d), dtype=np.float32)
        k[1, 0, 0] = 1.0
        kb = bf16_bits(torch.from_numpy(k).to(torch.bfloat16))
        vb = bf16_bits(bf16_normal((2, 1, d), 21))
        scale = 0.5
        out = oatt.decode(qb, kb, vb, scale)
        s = float(widen(qb)[0, 0]) * scale
        sig = 1.0 / (1.0 + math.exp(-s))
        vf = widen(vb)
        np.testing.assert_allclose(out[0], vf[0, 0] + sig * (vf[1, 0] - vf[0, 0]), rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("n,Hq,Hkv,d,scale", [
    (1, 1, 1, 16, 0.25), (50, 4, 4, 64, 0.125),      # G = 1: textbook MHA decode
    (333, 16, 4, 64, 0.125), (70, 32, 8, 128, 1.0),  # GQA groups of 4
    (45, 64, 8, 128, 0.0884),                        # groups of 8
])
def test_matches_torch_sdpa_float64(n, Hq, Hkv, d, scale):
    q, k, v = rand_qkv(n + Hq, n, Hq, Hkv, d)
    out = oatt.decode(q, k, v, scale)
    ref = sdpa_f64(q, k, v, scale)
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)


def test_head_group_mapping_is_contiguous():
    # Changing KV head g must change exactly query heads g*G .. g*G+G-1.
    n, Hq, Hkv, d = 40, 16, 4, 32
    q, k, v = rand_qkv(1, n, Hq, Hkv, d)
    base = oatt.decode(q, k, v, 0.3)
    k2 = k.copy()
    v2 = v.copy()
    k2[:, 2] = bf16_bits(bf16_normal((n, d), 77))
    v2[:, 2] = bf16_bits(bf16_normal((n, d), 78))
    out = oatt.decode(q, k2, v2, 0.3)
    changed = [h for h in range(Hq) if not np.array_equal(out[h], base[h])]
    assert changed == [8, 9, 10, 11]


def test_token_permutation_invariance():
    n, Hq, Hkv, d = 123, 8, 2, 64
    q, k, v = rand_qkv(4, n, Hq, Hkv, d)
    perm = np.random.default_rng(0).permutation(n)
    a = oatt.decode(q, k, v, 0.125)
    b = oatt.decode(q, k[perm], v[perm], 0.125)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-13)


def test_mask_equals_removal_and_sdpa_mask():
    # Algorithm 2, BuildMask: masking a closed cursor's tokens out of attention
    # stands for their eviction.  Masked attention over all rows must equal
    # attention over the kept rows, and torch SDPA with a -inf mask.
    n, Hq, Hkv, d = 260, 16, 4, 64
    q, k, v = rand_qkv(8, n, Hq, Hkv, d)
    mask = np.zeros(n, dtype=np.uint8)
    for a, b in [(3, 40), (100, 101), (180, 250)]:
        mask[a:b] = 1
    kept = np.nonzero(mask == 0)[0]
    masked = oatt.decode(q, k, v, 0.125, mask=mask)
    removed = oatt.decode(q, k[kept], v[kept], 0.125)
    assert np.array_equal(masked, removed)  # zero weights add exact zeros
    np.testing.assert_allclose(masked, sdpa_f64(q, k, v, 0.125, mask=mask), rtol=1e-10, atol=1e-12)


def test_batch_matches_single():
    Hq, Hkv, d = 8, 2, 32
    ns = [1, 17, 64, 65]
    qs, ks, vs, ref = [], [], [], []
    for i, n in enumerate(ns):
        q, k, v = rand_qkv(30 + i, n, Hq, Hkv, d)
        qs.append(q); ks.append(k); vs.append(v)
        ref.append(oatt.decode(q, k, v, 0.2))
    out = oatt.decode_batch(np.stack(qs), ks, vs, 0.2)
    for i in range(len(ns)):
        assert np.array_equal(out[i], ref[i])


def test_empty_sequence_rejected():
    q = np.zeros((4, 8), dtype=np.uint16)
    k = np.zeros((0, 4, 8), dtype=np.uint16)
    with pytest.raises(ValueError):
        oatt.decode(q, k, k, 1.0)


# ---------------------------------------------------------------------------
# cache model
# ---------------------------------------------------------------------------
def check_invariants(c: ocm.OracleCache):
    counts = [0] * c.num_pages
    for sid, s in c.seqs.items():
        assert len(s.pages) == ocm.ceil_div(len(s.tokens), c.P)
        assert len(set(s.pages)) == len(s.pages)
        for p in s.pages:
            counts[p] += 1
    assert counts == c.ref, "reference counts must equal the number of holders"
    assert sorted(c._free) == [p for p in range(c.num_pages) if c.ref[p] == 0]
    # a page shared by several sequences sits at the same logical index in all
    where = {}
    for sid, s in c.seqs.items():
        for q, p in enumerate(s.pages):
            assert where.setdefault(p, q) == q
    if c.phys is not None:
        for sid in c.seqs:
            assert c.physical_tokens(sid) == c.tokens(sid)


def brute_kept(tokens, spans):
    return [t for j, t in enumerate(tokens) if not any(a <= j < b for a, b in spans)]


def random_spans(rng, n, k):
    if n == 0:
        return []
    cuts = sorted(rng.sample(range(n + 1), min(2 * k, n + 1)))
    spans = [(cuts[i], cuts[i + 1]) for i in range(0, len(cuts) - 1, 2) if cuts[i] < cuts[i + 1]]
    rng.shuffle(spans)
    return spans


@pytest.mark.parametrize("seed", range(12))
def test_random_operation_sequences(seed):
    rng = random.Random(seed)
    P = rng.choice([1, 2, 4, 16])
    c = ocm.OracleCache(num_pages=rng.choice([40, 96, 200]), page_size=P,
                        max_pages_per_seq=rng.choice([None, 30]), physical=True)
    live = [c.seq_new()]
    for step in range(120):
        op = rng.random()
        sid = rng.choice(live) if live else None
        free_before = sorted(c._free)
        before_pages = {s: c.page_table(s) for s in c.seqs}
        try:
            if sid is None or op < 0.08:
                live.append(c.seq_new())
            elif op < 0.25:
                child = c.fork(sid)
                assert c.page_table(child) == c.page_table(sid)
                assert c.tokens(child) == c.tokens(sid)
                assert sorted(c._free) == free_before  # zero K/V copies (Sec. 3.4)
                live.append(child)
            elif op < 0.65:
                others = {s: c.tokens(s) for s in c.seqs if s != sid}
                c.append(sid, rng.choice([0, 1, 1, 2, P - 1, P, P + 1, 3 * P + 2]))
                for s, toks in others.items():
                    assert c.tokens(s) == toks
            elif op < 0.9:
                old = c.tokens(sid)
                others = {s: c.tokens(s) for s in c.seqs if s != sid}
                spans = random_spans(rng, len(old), rng.choice([0, 1, 2, 5]))
                c.evict(sid, spans)
                assert c.tokens(sid) == brute_kept(old, spans)
                for s, toks in others.items():
                    assert c.tokens(s) == toks  # a fork keeps its own view
            else:
                c.release(sid)
                live.remove(sid)
        except (ocm.NoPages, ocm.Capacity):
            # transactional: nothing changed
            assert sorted(c._free) == free_before
            assert {s: c.page_table(s) for s in c.seqs} == before_pages
        # lowest-free-id: every page newly taken by this op is among the
        # smallest free ids before it, and taken ids form a prefix of them
        taken = sorted(set(free_before) - set(c._free))
        assert taken == free_before[:len(taken)]
        check_invariants(c)


def test_append_cow_of_shared_partial_page():
    c = ocm.OracleCache(num_pages=10, page_size=4, physical=True)
    m = c.seq_new()
    c.append(m, 6)                   # pages [0, 1], page 1 half full
    a = c.fork(m)
    assert c.ref[:2] == [2, 2]
    c.append(m, 1)                   # last page shared and partial -> CoW
    assert c.page_table(m) == [0, 2] and c.page_table(a) == [0, 1]
    assert c.ref[:3] == [2, 1, 1]
    c.append(a, 3)                   # aux's page 1 is now private: no CoW
    assert c.page_table(a) == [0, 1, 3]
    check_invariants(c)


def test_evict_cow_rules_worked_by_hand():
    # P = 4, n = 12 (pages A B C), fork, evict [2, 5) from main.
    # kept = 0 1 5 6 7 8 9 10 11 -> n' = 9, pages q = 0, 1, 2 (q = 2 has 1 row)
    # q = 0 changed (rows 2, 3 now hold old 5, 6); q = 1, 2 changed too; all
    # shared -> three fresh pages 3, 4, 5 in increasing q; nothing trails.
    c = ocm.OracleCache(num_pages=8, page_size=4, physical=True)
    m = c.seq_new()
    c.append(m, 12)
    aux = c.fork(m)
    r = c.evict(m, [(2, 5)])
    assert c.page_table(m) == [3, 4, 5]
    assert c.page_table(aux) == [0, 1, 2]
    assert r == {"n_before": 12, "n_after": 9, "moved_rows": 9, "cow_pages": 3, "released_pages": 0}
    assert c.ref[:6] == [1, 1, 1, 1, 1, 1]
    c.release(aux)
    # without a fork: in place.  evict [0, 4) from [0..9): pages [3, 4, 5]
    # n' = 5 -> pages q = 0, 1 kept in place, page 5 released
    r = c.evict(m, [(0, 4)])
    assert c.page_table(m) == [3, 4]
    assert r["cow_pages"] == 0 and r["released_pages"] == 1 and r["moved_rows"] == 5
    check_invariants(c)


def test_empty_span_set_is_identity():
    c = ocm.OracleCache(num_pages=16, page_size=4, physical=True)
    m = c.seq_new()
    c.append(m, 13)
    aux = c.fork(m)
    c.append(aux, 2)
    snap = (c.page_table(m), c.tokens(m), list(c.ref), sorted(c._free),
            {p: list(v) for p, v in c.phys.items()})
    r = c.evict(m, [])
    assert r["moved_rows"] == 0 and r["cow_pages"] == 0 and r["released_pages"] == 0
    assert snap == (c.page_table(m), c.tokens(m), list(c.ref), sorted(c._free),
                    {p: list(v) for p, v in c.phys.items()})


@pytest.mark.parametrize("spans", [
    [(3, 2)], [(4, 4)], [(-1, 2)], [(0, 11)], [(0, 5), (4, 6)], [(2, 6), (0, 3)],
])
def test_bad_spans_rejected_without_change(spans):
    c = ocm.OracleCache(num_pages=8, page_size=4)
    m = c.seq_new()
    c.append(m, 10)
    before = (c.page_table(m), c.tokens(m), list(c.ref))
    with pytest.raises(ocm.InvalidArg):
        c.evict(m, spans)
    assert before == (c.page_table(m), c.tokens(m), list(c.ref))


def test_adjacent_and_unsorted_spans_accepted():
    c = ocm.OracleCache(num_pages=8, page_size=4)
    m = c.seq_new()
    c.append(m, 10)
    toks = c.tokens(m)
    c.evict(m, [(6, 8), (2, 4), (4, 6)])
    assert c.tokens(m) == toks[:2] + toks[8:]


def test_no_pages_is_transactional():
    c = ocm.OracleCache(num_pages=3, page_size=4)
    m = c.seq_new()
    c.append(m, 10)                  # 3 pages, last one half full
    aux = c.fork(m)
    with pytest.raises(ocm.NoPages):
        c.append(m, 1)               # needs a CoW page: none free
    with pytest.raises(ocm.NoPages):
        c.evict(m, [(0, 1)])         # every page changes and is shared
    assert c.page_table(m) == [0, 1, 2] and c.ref == [2, 2, 2]
    c.release(aux)
    c.evict(m, [(0, 1)])             # now private: in place
    assert c.page_table(m) == [0, 1, 2]


def test_capacity_limit():
    c = ocm.OracleCache(num_pages=10, page_size=4, max_pages_per_seq=2)
    m = c.seq_new()
    c.append(m, 8)
    with pytest.raises(ocm.Capacity):
        c.append(m, 1)
    assert c.n_tokens(m) == 8


def test_release_frees_only_private_pages():
    # Sec. 3.4 / Algorithm 1: the aux thread's own tokens are discarded.
    c = ocm.OracleCache(num_pages=20, page_size=4)
    m = c.seq_new()
    c.append(m, 16)
    aux = c.fork(m)
    c.append(aux, 9)                 # 3 private pages
    live = c.live_pages()
    c.release(aux)
    assert c.live_pages() == live - 3
    assert all(c.ref[p] == 1 for p in c.page_table(m))


def test_fig1_walkthrough_golden():
    g = json.load(open(os.path.join(GOLDEN, "fig1_walkthrough.json")))
    c = ocm.OracleCache(num_pages=200, page_size=g["page_size"], physical=True)
    m = c.seq_new()
    ranges = {}
    for msg in g["messages"]:
        ids = c.append(m, msg["len"])
        ranges[msg["name"]] = ids
    # the caller maps each cursor to its call + response tokens
    n0 = 0
    spans = []
    pos = 0
    for msg in g["messages"]:
        if msg.get("cursor") in g["del_cursors"]:
            spans.append((pos, pos + msg["len"]))
        pos += msg["len"]
    # merge the adjacent call/response pieces of one cursor into one span
    merged = []
    for a, b in sorted(spans):
        if merged and merged[-1][1] == a:
            merged[-1] = (merged[-1][0], b)
        else:
            merged.append((a, b))
    assert merged == [tuple(g["expected_span"])]
    aux = c.fork(m)   # the aux thread that issued the command is still alive
    c.evict(m, merged)
    assert c.n_tokens(m) == g["expected_n_after"]
    toks = c.tokens(m)
    for name, (a, b) in g["expected_after"].items():
        assert toks[a:b] == ranges[name], name
    # the aux thread's view is untouched
    assert c.n_tokens(aux) == sum(msg["len"] for msg in g["messages"])
    check_invariants(c)


def test_forked_aux_attends_exactly_like_parent():
    # Sec. 3.4: the aux thread works on the shared context.  Its decode over
    # the same query equals the parent's bit for bit, also after the parent
    # evicts (the aux keeps its view).
    Hq, Hkv, d, P = 8, 2, 32, 4
    c = ocm.OracleCache(num_pages=64, page_size=P)
    m = c.seq_new()
    ids = c.append(m, 50)
    rows_k = bf16_bits(bf16_normal((200, Hkv, d), 1))
    rows_v = bf16_bits(bf16_normal((200, Hkv, d), 2))
    q = bf16_bits(bf16_normal((Hq, d), 3))
    aux = c.fork(m)
    km = rows_k[c.tokens(m)]
    ka = rows_k[c.tokens(aux)]
    assert np.array_equal(km, ka)
    o_m = oatt.decode(q, km, rows_v[c.tokens(m)], 0.17)
    o_a = oatt.decode(q, ka, rows_v[c.tokens(aux)], 0.17)
    assert np.array_equal(o_m, o_a)
    c.evict(m, [(5, 20)])
    o_a2 = oatt.decode(q, rows_k[c.tokens(aux)], rows_v[c.tokens(aux)], 0.17)
    assert np.array_equal(o_a, o_a2)
    # evict-then-attend equals masked attention over the pre-eviction rows
    mask = np.zeros(50, dtype=np.uint8)
    mask[5:20] = 1
    o_m2 = oatt.decode(q, rows_k[c.tokens(m)], rows_v[c.tokens(m)], 0.17)
    assert np.array_equal(o_m2, oatt.decode(q, km, rows_v[ids], 0.17, mask=mask))


# ---------------------------------------------------------------------------
# masked prefill attention (Algorithm 2, BuildMask)
# ---------------------------------------------------------------------------
def prefill_reference_f64(q, k, v, scale, spans):
    """Causal attention with the spans' tokens removed, written with torch
    float64 ops: an explicit [n_q, n] mask and torch's SDPA (library routine),
    and the log-sum-exp from torch.logsumexp over the masked logits."""
    n_q, Hq, d = q.shape
    n, Hkv, _ = k.shape
    G = Hq // Hkv
    pos = torch.arange(n - n_q, n).view(n_q, 1)
    key = torch.arange(n).view(1, n)
    allowed = key <= pos
    for a, b in spans:
        allowed[:, a:b] = False
    qt = torch.from_numpy(widen(q)).permute(1, 0, 2)                               # [Hq, n_q, d]
    kt = torch.from_numpy(widen(k)).permute(1, 0, 2).repeat_interleave(G, dim=0)  # [Hq, n, d]
    vt = torch.from_numpy(widen(v)).permute(1, 0, 2).repeat_interleave(G, dim=0)
    logits = scale * qt @ kt.transpose(1, 2)                                       # [Hq, n_q, n]
    logits = logits.masked_fill(~allowed, -math.inf)
    lse = torch.logsumexp(logits, dim=-1)                                          # [Hq, n_q]
    rows = allowed.any(dim=1)
    am = torch.zeros(n_q, n, dtype=torch.float64).masked_fill(~allowed, -math.inf)
    am[~rows] = 0.0  # keep SDPA finite on rows with nothing to see; zeroed below
    o = torch.nn.functional.scaled_dot_product_attention(
        qt.unsqueeze(0), kt.unsqueeze(0), vt.unsqueeze(0), attn_mask=am, scale=scale)[0]
    o[:, ~rows] = 0.0
    return o.permute(1, 0, 2).numpy(), lse.permute(1, 0).numpy()


def rand_prefill(seed, n, n_q, Hq, Hkv, d):
    q = bf16_bits(bf16_normal((n_q, Hq, d), seed))
    k = bf16_bits(bf16_normal((n, Hkv, d), seed + 1))
    v = bf16_bits(bf16_normal((n, Hkv, d), seed + 2))
    return q, k, v


@pytest.mark.parametrize("n,n_q,Hq,Hkv,d,spans", [
    (1, 1, 4, 4, 16, []),                              # one token, G = 1
    (40, 40, 4, 4, 32, []),                            # textbook causal MHA
    (40, 40, 8, 2, 32, [(5, 9), (20, 33)]),            # GQA, full prefill
    (97, 13, 16, 4, 64, [(60, 90), (2, 3), (95, 97)]),  # queries at the tail
    (64, 64, 6, 2, 16, [(0, 10)]),                     # a masked prefix: empty rows
    (150, 7, 12, 4, 64, [(143, 146)]),                 # spans among the queries
])
def test_prefill_matches_masked_causal_sdpa(n, n_q, Hq, Hkv, d, spans):
    q, k, v = rand_prefill(n * 7 + n_q, n, n_q, Hq, Hkv, d)
    out, lse = oatt.prefill(q, k, v, 0.21, spans, want_lse=True)
    ref, ref_lse = prefill_reference_f64(q, k, v, 0.21, spans)
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)
    fin = np.isfinite(ref_lse)
    assert np.array_equal(np.isfinite(lse), fin)
    np.testing.assert_allclose(lse[fin], ref_lse[fin], rtol=1e-12, atol=1e-12)


def test_prefill_causal_reach_is_exact():
    # Changing token t's K/V changes exactly the queries at positions >= t,
    # and none when t lies in a masked span.
    n, n_q, Hq, Hkv, d = 30, 30, 4, 2, 16
    q, k, v = rand_prefill(5, n, n_q, Hq, Hkv, d)
    spans = [(11, 14)]
    base = oatt.prefill(q, k, v, 0.3, spans)
    for t in (0, 7, 12, 29):
        k2, v2 = k.copy(), v.copy()
        k2[t] = bf16_bits(bf16_normal((Hkv, d), 90 + t))
        v2[t] = bf16_bits(bf16_normal((Hkv, d), 190 + t))
        out = oatt.prefill(q, k2, v2, 0.3, spans)
        changed = [i for i in range(n_q) if not np.array_equal(out[i], base[i])]
        expect = [] if 11 <= t < 14 else list(range(t, n))
        assert changed == expect, t


def test_prefill_single_visible_key_and_empty_rows():
    # spans [1, n): every query sees token 0 only -> output = V[0] of its
    # group exactly, lse = its logit; spans [0, n): nothing -> zeros, -inf.
    n, Hq, Hkv, d = 20, 8, 2, 16
    q, k, v = rand_prefill(11, n, n, Hq, Hkv, d)
    out, lse = oatt.prefill(q, k, v, 0.5, [(1, n)], want_lse=True)
    vw, kw, qw = widen(v), widen(k), widen(q)
    for h in range(Hq):
        g = h // (Hq // Hkv)
        assert np.array_equal(out[:, h], np.broadcast_to(vw[0, g], (n, d)))
        np.testing.assert_allclose(lse[:, h], 0.5 * qw[:, h] @ kw[0, g], rtol=1e-13)
    out, lse = oatt.prefill(q, k, v, 0.5, [(0, n)], want_lse=True)
    assert not out.any() and np.all(lse == -np.inf)


def test_prefill_last_row_equals_decode_after_eviction():
    # Algorithm 2 masks the closed cursors' tokens while training; Algorithm 1
    # evicts them at inference.  The last query of a masked prefill must equal
    # decode over the evicted cache, up to the order of the sums.
    Hq, Hkv, d, P = 8, 2, 32, 4
    c = ocm.OracleCache(num_pages=64, page_size=P)
    m = c.seq_new()
    ids = c.append(m, 90)
    k = bf16_bits(bf16_normal((90, Hkv, d), 21))
    v = bf16_bits(bf16_normal((90, Hkv, d), 22))
    q = bf16_bits(bf16_normal((1, Hq, d), 23))
    spans = [(30, 41), (4, 9), (60, 88)]
    pre = oatt.prefill(q, k[ids], v[ids], 0.2, spans)
    c.evict(m, spans)
    kept = c.tokens(m)
    dec = oatt.decode(q[0], k[kept], v[kept], 0.2)
    np.testing.assert_allclose(pre[0], dec, rtol=1e-12, atol=1e-13)


def test_prefill_constant_values():
    n, Hq, Hkv, d = 50, 4, 1, 8
    q, k, _ = rand_prefill(3, n, 25, Hq, Hkv, d)
    v = np.full((n, Hkv, d), bf16_bits(torch.tensor([0.375], dtype=torch.bfloat16))[0], dtype=np.uint16)
    out = oatt.prefill(q, k, v, 0.4, [(26, 31)])
    np.testing.assert_allclose(out, 0.375, rtol=1e-14)


def test_prefill_rejects_bad_shapes():
    q, k, v = rand_prefill(1, 10, 11, 4, 2, 8)
    with pytest.raises(ValueError):
        oatt.prefill(q, k, v, 1.0)
