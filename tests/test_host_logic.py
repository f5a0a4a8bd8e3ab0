"""CPU tests of the library's host logic (page allocator, copy-on-write and
eviction planning, decode planning), driven through libsq_host.so — the same
C++ the CUDA library runs on the host — and compared with the oracle."""
import random

import pytest

from oracle import cache_model as ocm
from tests.hostlib import HostCache, lib

CODES = {ocm.InvalidArg: -1, ocm.BadHandle: -2, ocm.NoPages: -3, ocm.Capacity: -4}
STAGE = 64  # tokens per decode stage


def oracle_call(fn, *args):
    try:
        return 0, fn(*args)
    except ocm.OracleError as e:
        return CODES[type(e)], None


def random_spans(rng, n, k):
    if n == 0:
        return []
    cuts = sorted(rng.sample(range(n + 1), min(2 * k, n + 1)))
    spans = [(cuts[i], cuts[i + 1]) for i in range(0, len(cuts) - 1, 2) if cuts[i] < cuts[i + 1]]
    rng.shuffle(spans)
    return spans


def compare_state(hc, oc, pairs):
    for h, o in pairs.items():
        assert hc.page_table(h) == oc.page_table(o)
        assert hc.page_fill(h) == oc.page_fills(o)
        assert hc.info(h)[1] == oc.n_tokens(o)
    assert hc.free_count() == oc.free_count()
    for p in range(oc.num_pages):
        assert hc.refcount(p) == oc.ref[p]


@pytest.mark.parametrize("seed", range(16))
def test_page_tables_match_oracle_bit_exact(seed):
    rng = random.Random(1000 + seed)
    P = rng.choice([8, 16, 32, 64])
    num_pages = rng.choice([24, 64, 150])
    mpps = rng.choice([None, 12])
    hc = HostCache(1, 8, 2, 64, P, num_pages, max_seqs=32, max_pages_per_seq=mpps)
    oc = ocm.OracleCache(num_pages, P, max_pages_per_seq=mpps)
    pairs = {}
    rc, h = hc.seq_new()
    pairs[h] = oc.seq_new()
    for step in range(150):
        live = list(pairs)
        op = rng.random()
        if not live or op < 0.05:
            rc, h = hc.seq_new()
            if rc == 0:
                pairs[h] = oc.seq_new()
            continue
        h = rng.choice(live)
        o = pairs[h]
        if op < 0.2:
            rc, child = hc.fork(h)
            orc, ochild = oracle_call(oc.fork, o)
            assert rc == orc
            if rc == 0:
                pairs[child] = ochild
        elif op < 0.6:
            n = rng.choice([1, 1, 3, P - 1, P, P + 1, 2 * P + 5, 7 * P])
            rc = hc.append(h, n)
            orc, _ = oracle_call(oc.append, o, n)
            assert rc == orc
        elif op < 0.9:
            spans = random_spans(rng, oc.n_tokens(o), rng.choice([1, 2, 4, 9]))
            if rng.random() < 0.1 and spans:
                spans.append((spans[0][0], spans[0][0] + 1))  # overlap -> rejected
            ragged = rng.random() < 0.5
            rc, st = hc.evict(h, spans, ragged)
            orc, ost = oracle_call(oc.evict, o, spans, "ragged" if ragged else "dense")
            assert rc == orc, (spans, rc, orc)
            if rc == 0 and spans:
                assert st["moved_rows"] == ost["moved_rows"]
                assert st["cow_pages"] == ost["cow_pages"]
                if ragged:
                    assert st["zeroed_rows"] == ost["zeroed_rows"]
                    assert st["windows"] == ost["windows"]
        else:
            assert hc.release(h) == 0
            oc.release(o)
            del pairs[h]
        compare_state(hc, oc, pairs)
    assert hc.peak_live_pages() == oc.peak_live_pages


def test_bad_handles_rejected():
    hc = HostCache(1, 4, 4, 64, 16, 32)
    rc, h = hc.seq_new()
    assert hc.append(h, 5) == 0
    assert hc.release(h) == 0
    assert hc.append(h, 1) == -2       # released handle
    assert hc.fork(h)[0] == -2
    assert hc.evict(h, [(0, 1)])[0] == -2
    assert hc.append(12345, 1) == -2
    assert hc.append(-1, 1) == -2
    rc, h2 = hc.seq_new()               # the slot is reused with a new generation
    assert h2 != h
    assert hc.append(h2, -1) == -1


def _check_plan(hc, handles, plan, n_ctas, G):
    P, Hkv = hc.P, hc.Hkv
    segs, items = plan["segs"], plan["items"]
    cb = plan["cta_begin"]
    assert cb[0] == 0 and cb[-1] == len(items)
    assert all(cb[i] <= cb[i + 1] for i in range(len(cb) - 1))
    assert len(cb) - 1 <= n_ctas
    # work per CTA (stages + a fixed cost per item) is balanced: within one
    # unit start-up cost plus one stage
    C = 2
    per_cta = [sum(items[i][3] - items[i][2] + C for i in range(cb[c], cb[c + 1]))
               for c in range(len(cb) - 1)]
    busy = [x for x in per_cta if x > 0]
    assert max(busy) - min(busy) <= 2 * C + 1
    for s in segs:
        assert 1 <= s["n_grp"] <= 16 // G
        assert max(s["grp_lim"]) == s["n_tok"] and min(s["grp_lim"]) > 0
        assert s["n_tok"] <= s["n_pages"] * P
    # every (sequence, head) covers its slots exactly once, through its own
    # pages (slot space: page index x P + slot; rows = filled slots)
    tables = [hc.page_table(h) for h in handles]
    fills = [hc.page_fill(h) for h in handles]
    ends = [(len(f) - 1) * P + f[-1] for f in fills]
    ragged = any(x < P for f in fills for x in f[:-1])
    assert (plan["page_fill"] is not None) == ragged
    if ragged:
        for s in segs:
            pids = plan["page_ids"][s["page_off"]:s["page_off"] + s["n_pages"]]
            pf = plan["page_fill"][s["page_off"]:s["page_off"] + s["n_pages"]]
            for j in range(s["n_grp"]):
                i = s["grp_seq"][j]
                q0 = tables[i].index(pids[0])
                assert fills[i][q0:q0 + s["n_pages"]] == pf
    for i in range(len(handles)):
        for head in range(Hkv):
            key = i * Hkv + head
            ents = plan["comb_ent"][plan["comb_off"][key]:plan["comb_off"][key + 1]]
            covered = []
            seg_start = {}
            for it_idx, j in ents:
                seg_i, hd, s0, s1 = items[it_idx]
                s = segs[seg_i]
                assert hd == head and s["grp_seq"][j] == i
                # first logical page of the segment: find where its pages sit
                pids = plan["page_ids"][s["page_off"]:s["page_off"] + s["n_pages"]]
                q0 = tables[i].index(pids[0])
                assert tables[i][q0:q0 + s["n_pages"]] == pids
                lim = s["grp_lim"][j]
                # the limit is the sequence's end from the run's first slot,
                # within the run's pages (an append inside the last page
                # rewrites it this way in a kept plan)
                assert s["q0"] == q0
                assert min(ends[i] - q0 * P, s["n_pages"] * P) == lim
                # the tail bit: the run holds the member's last page; the
                # others' limit is the whole run
                is_tail = q0 + s["n_pages"] == len(tables[i])
                assert bool((s["tail"] >> j) & 1) == is_tail
                if not is_tail:
                    assert lim == s["n_pages"] * P
                lo, hi = s0 * STAGE, min(s1 * STAGE, lim)
                if hi > lo:
                    covered.append((q0 * P + lo, q0 * P + hi))
            covered.sort()
            pos = 0
            for a, b in covered:
                assert a == pos
                pos = b
            assert pos == ends[i]


@pytest.mark.parametrize("seed", range(10))
def test_decode_plan_covers_every_token_once(seed):
    rng = random.Random(seed)
    P = rng.choice([8, 16, 64, 128])
    G = rng.choice([1, 4, 8, 16])
    Hkv = rng.choice([1, 2, 8])
    hc = HostCache(2, G * Hkv, Hkv, 128, P, 4000, max_seqs=64)
    mains = []
    for _ in range(rng.randint(1, 4)):
        rc, h = hc.seq_new()
        assert hc.append(h, rng.randint(1, 40 * P)) == 0
        mains.append(h)
    seqs = list(mains)
    for h in mains:
        for _ in range(rng.randint(0, 3)):
            rc, a = hc.fork(h)
            assert rc == 0
            assert hc.append(a, rng.randint(0, 3 * P)) == 0
            seqs.append(a)
        assert hc.append(h, rng.randint(0, 2 * P)) == 0
        if rng.random() < 0.5:
            n = hc.info(h)[1]
            hc.evict(h, random_spans(rng, n, 3), ragged=rng.random() < 0.5)
    rng.shuffle(seqs)
    for n_ctas in (1, 3, 152, 304, 5000):
        rc, plan = hc.plan_decode(seqs, n_ctas)
        assert rc == 0
        _check_plan(hc, seqs, plan, n_ctas, G)
        assert plan["logical_tokens"] == sum(hc.info(h)[1] for h in seqs)
        assert plan["unique_tokens"] <= plan["logical_tokens"]


def test_decode_plan_reads_shared_prefix_once():
    # main + fork with a 4096-token shared prefix: the shared pages form one
    # segment read for both query groups (Sec. 3.4, shared-context kernels)
    hc = HostCache(1, 32, 8, 128, 64, 1000)
    rc, m = hc.seq_new()
    hc.append(m, 4096)
    rc, a = hc.fork(m)
    hc.append(a, 8)
    hc.append(m, 1)
    rc, plan = hc.plan_decode([m, a], 304)
    assert rc == 0
    shared = [s for s in plan["segs"] if s["n_grp"] == 2]
    assert len(shared) == 1 and shared[0]["n_tok"] == 4096
    assert plan["unique_tokens"] == 4096 + 1 + 8
    assert plan["logical_tokens"] == 4097 + 4104


def test_decode_plan_spreads_fork_tails():
    # 8 requests of 32,768 tokens, each with a fork holding an 8-token tail
    # of its own (the aux trigger): 64 one-stage tail units among 64 prefix
    # units of 512 stages.  Units go family by family, head by head, so each
    # tail follows the prefix unit of its own head: no CTA holds more than a
    # few tails, and each tail's CTA also holds the end of that prefix.
    Hkv = 8
    hc = HostCache(1, 32, Hkv, 128, 64, 8 * 520)
    seqs = []
    for _ in range(8):
        rc, m = hc.seq_new()
        assert hc.append(m, 32768) == 0
        rc, a = hc.fork(m)
        assert hc.append(a, 8) == 0
        seqs += [m, a]
    rc, plan = hc.plan_decode(seqs, 304)
    assert rc == 0
    _check_plan(hc, seqs, plan, 304, 4)
    segs, items, cb = plan["segs"], plan["items"], plan["cta_begin"]
    tails_per_cta = []
    for c in range(len(cb) - 1):
        its = items[cb[c]:cb[c + 1]]
        tails = [it for it in its if segs[it[0]]["n_tok"] == 8]
        tails_per_cta.append(len(tails))
        for t in tails:
            # the same CTA ends the shared prefix of the tail's head (or the
            # tail starts the CTA right after it)
            fork_seq = segs[t[0]]["grp_seq"][0]
            prefix = [it for it in items[max(0, cb[c] - 1):cb[c + 1]]
                      if segs[it[0]]["n_grp"] == 2 and fork_seq in segs[it[0]]["grp_seq"]
                      and it[1] == t[1]]
            assert prefix, (c, t)
    assert sum(tails_per_cta) == 8 * Hkv
    assert max(tails_per_cta) <= 2
    # a fork's (sequence, head) run: its prefix entries and its tail; the
    # tails are never alone, so no tail member is marked sole
    assert all(len(plan["comb_ent"][plan["comb_off"][k]:plan["comb_off"][k + 1]]) > 1
               for k in range(len(plan["comb_off"]) - 1))


def test_decode_plan_marks_single_item_runs():
    # many short sequences, one CTA: every (sequence, head) run is one item,
    # so every member is marked sole (the parse of the plan checks the mark
    # against the run lengths)
    hc = HostCache(1, 16, 4, 64, 16, 400)
    seqs = []
    for n in (1, 5, 16, 17, 40):
        rc, h = hc.seq_new()
        assert hc.append(h, n) == 0
        seqs.append(h)
    rc, plan = hc.plan_decode(seqs, 1)
    assert rc == 0
    offs = plan["comb_off"]
    assert all(offs[k + 1] - offs[k] == 1 for k in range(len(offs) - 1))


def test_decode_plan_rejects_bad_input():
    hc = HostCache(1, 8, 2, 64, 16, 100)
    rc, m = hc.seq_new()
    assert hc.plan_decode([m], 10)[0] == -1          # empty sequence
    hc.append(m, 5)
    assert hc.plan_decode([m, m], 10)[0] == -1       # duplicate
    assert hc.plan_decode([m, 999], 10)[0] == -2     # bad handle


def test_decode_plan_limits_entries_per_run():
    # The kernel counts a run's arrivals in 16 bits: one KV head of one
    # sequence may have at most 65,535 partial results.  66,000 stages of 64
    # tokens dealt to 66,000 CTAs give ~65,998 (the unit's start-up share
    # leaves the first CTAs without stages): SQ_ERR_CAPACITY.  65,000 CTAs
    # are accepted.
    n = 66000 * 64
    hc = HostCache(1, 1, 1, 64, 64, n // 64 + 4, max_pages_per_seq=n // 64 + 4)
    rc, m = hc.seq_new()
    assert hc.append(m, n) == 0
    assert hc.plan_decode([m], 66000)[0] == -4      # SQ_ERR_CAPACITY
    rc, plan = hc.plan_decode([m], 65000)
    assert rc == 0


@pytest.mark.parametrize("seed", range(20))
def test_evict_tiles_compact_in_place(seed):
    """Replaying the compaction tiles in order — each tile's reads before its
    writes, on a physical model of the pool — gives the oracle's result; no
    tile reads a slot an earlier tile wrote (so loads may run ahead of
    earlier stores); forks sharing pages are untouched."""
    rng = random.Random(500 + seed)
    P = rng.choice([8, 16, 64, 128])
    tile_rows = rng.choice([t for t in (8, 16, 32, 64) if t <= P])
    hc = HostCache(1, 4, 1, 64, P, 600)
    oc = ocm.OracleCache(600, P, physical=True)
    rc, m = hc.seq_new()
    om = oc.seq_new()
    n0 = rng.randint(1, 40 * P)
    hc.append(m, n0)
    oc.append(om, n0)
    forks = []
    if rng.random() < 0.5:
        rc, a = hc.fork(m)
        forks.append((a, oc.fork(om)))
        k = rng.randint(0, 2 * P)
        hc.append(a, k)
        oc.append(forks[-1][1], k)
        k = rng.randint(0, P)
        hc.append(m, k)
        oc.append(om, k)
    # a first ragged eviction leaves partial pages for the one under test
    if rng.random() < 0.5:
        pre = random_spans(rng, oc.n_tokens(om), 4)
        assert hc.evict(m, pre, ragged=True)[0] == 0
        oc.evict(om, pre, mode="ragged")
    ragged = rng.random() < 0.5
    n = oc.n_tokens(om)
    spans = random_spans(rng, n, rng.choice([1, 3, 8, 20]))
    # physical state before, as {page: [token ids]}
    phys = {p: list(v) for p, v in oc.phys.items()}
    max_chunks = rng.choice([1, 2, 5, 64])
    rc, tiles, pieces, chunks = hc.evict_tiles(m, spans, tile_rows, ragged, max_chunks=max_chunks,
                                               want_chunks=True)
    oc.evict(om, spans, mode="ragged" if ragged else "dense")
    assert rc == 0
    # chunks cover the tiles in order; a dense eviction is one chunk
    assert chunks[0] == 0 and chunks[-1] == len(tiles) and chunks == sorted(set(chunks))
    assert len(chunks) - 1 <= max(1, max_chunks)
    if not ragged:
        assert len(chunks) == 2 or len(tiles) == 0
    # chunks run in any order (here: last first), each in order, against
    # one pool; chunk c's tiles read no slot another chunk writes
    order = []
    for c in reversed(range(len(chunks) - 1)):
        order.extend(range(chunks[c], chunks[c + 1]))
    chunk_of = {}
    for c in range(len(chunks) - 1):
        for t in range(chunks[c], chunks[c + 1]):
            chunk_of[t] = c
    writes = {}
    for t in range(len(tiles)):
        dpage, dslot, nrows, _ = (int(x) for x in tiles[t])
        for i in range(nrows):
            writes[(dpage, dslot + i)] = chunk_of[t]
    for t in range(len(tiles)):
        pb = int(tiles[t][3])
        pe = int(tiles[t + 1][3]) if t + 1 < len(tiles) else len(pieces)
        for k in range(pb, pe):
            spage, sslot, pn, _ = (int(x) for x in pieces[k])
            for i in range(pn):
                assert writes.get((spage, sslot + i), chunk_of[t]) == chunk_of[t]
    written = set()
    for t in order:
        dpage, dslot, nrows, pb = (int(x) for x in tiles[t])
        pe = int(tiles[t + 1][3]) if t + 1 < len(tiles) else len(pieces)
        assert 0 < nrows <= tile_rows and dslot + nrows <= P
        if pe == pb:                      # a tile of zeros
            assert ragged
            buf = [ocm.ZERO] * nrows
        else:
            buf = [None] * nrows
        for k in range(pb, pe):
            spage, sslot, pn, drow = (int(x) for x in pieces[k])
            assert 0 < pn and sslot + pn <= P and drow + pn <= nrows
            for i in range(pn):
                assert (spage, sslot + i) not in written
                buf[drow + i] = phys[spage][sslot + i]
        assert all(x is not None for x in buf)
        for i in range(nrows):
            phys.setdefault(dpage, [-1] * P)[dslot + i] = buf[i]
            written.add((dpage, dslot + i))

    def read(h):
        rows = []
        for pg, f in zip(hc.page_table(h), hc.page_fill(h)):
            rows.extend(phys[pg][:f])
        return rows

    assert hc.page_table(m) == oc.page_table(om)
    assert hc.page_fill(m) == oc.page_fills(om)
    assert read(m) == oc.tokens(om)
    # every slot the oracle holds, unused ones included, as the tiles left it
    for pg in hc.page_table(m):
        assert phys[pg] == oc.phys[pg], pg
    for a, oa in forks:
        assert read(a) == oc.tokens(oa)


# ---------------------------------------------------------------------------
# masked prefill planning (Algorithm 2, BuildMask)
# ---------------------------------------------------------------------------
NO_KEYS = 0x7fffffc0


def _brute_prefill_plan(n, n_q, spans, P=64):
    """Key tiles by their definition: with pages of >= 64 tokens, the 64-key
    boxes holding a visible key, two by two; otherwise aligned 128-key tiles
    holding one.  Each as (key0, full, vis words, key0b)."""
    removed = [False] * n
    for a, b in spans:
        for j in range(a, b):
            removed[j] = True

    def bits_of(base):
        return [base + c < n and not removed[base + c] for c in range(64)]

    tiles = []
    if P >= 64:
        boxes = [b for b in range(0, n, 64) if any(bits_of(b))]
        for i in range(0, len(boxes), 2):
            lo = boxes[i]
            hi = boxes[i + 1] if i + 1 < len(boxes) else NO_KEYS
            bits = bits_of(lo) + (bits_of(hi) if hi != NO_KEYS else [False] * 64)
            words = [sum(1 << c for c in range(32) if bits[32 * w + c]) for w in range(4)]
            tiles.append((lo, int(all(bits)), words, hi))
    else:
        for key0 in range(0, n, 128):
            bits = bits_of(key0) + bits_of(key0 + 64)
            if any(bits):
                words = [sum(1 << c for c in range(32) if bits[32 * w + c]) for w in range(4)]
                tiles.append((key0, int(all(bits)), words, key0 + 64))
    pairs = sum(sum(1 for j in range(p + 1) if not removed[j]) for p in range(n - n_q, n))
    return tiles, pairs


@pytest.mark.parametrize("seed", range(10))
def test_prefill_plan_visibility_matches_brute_force(seed):
    from tests.hostlib import plan_prefill
    rng = random.Random(seed)
    n = rng.choice([1, 5, 127, 128, 129, 700, 1500])
    n_q = rng.choice([1, n, max(1, n // 3)])
    Hkv = rng.choice([1, 2, 8])
    G = rng.choice([1, 3, 4, 16])
    k = rng.randint(0, 6)
    cuts = sorted(rng.sample(range(n + 1), min(2 * k, n + 1)))
    spans = [(cuts[i], cuts[i + 1]) for i in range(0, len(cuts) - 1, 2) if cuts[i] < cuts[i + 1]]
    rng.shuffle(spans)
    P = rng.choice([16, 64, 256])
    rc, info, tiles = plan_prefill(G * Hkv, Hkv, n, n_q, spans, P=P)
    assert rc == 0
    exp_tiles, exp_pairs = _brute_prefill_plan(n, n_q, spans, P)
    assert info["tile_bytes"] == 32
    assert info["n_tiles"] == len(exp_tiles)
    for got, (key0, full, words, key0b) in zip(tiles, exp_tiles):
        assert got[0] == key0 and got[1] == full and list(got[2:6]) == words and got[6] == key0b
    assert info["visible_pairs"] == exp_pairs
    assert info["BP"] == 128 // G
    span = 2 * (128 // G)          # two query tiles per CTA
    assert info["n_qt"] == -(-n_q // span)
    # each CTA tile reaches the listed tiles up to its last query position
    for qt, cnt in enumerate(info["qt_tiles"]):
        p_last = n - n_q + min((qt + 1) * span, n_q) - 1
        assert cnt == sum(1 for t in exp_tiles if t[0] <= p_last), qt
    units = info["n_qt"] * Hkv
    assert info["n_split"] >= 1
    if units >= 152:
        assert info["n_split"] == 1
    else:
        assert info["n_split"] <= max(1, min(64, len(exp_tiles)))


def test_prefill_plan_rejects_bad_input():
    from tests.hostlib import plan_prefill
    assert plan_prefill(8, 2, 100, 101, [])[0] == -1      # more queries than tokens
    assert plan_prefill(8, 2, 100, 0, [])[0] == -1
    assert plan_prefill(8, 2, 100, 10, [(5, 5)])[0] == -1      # empty span
    assert plan_prefill(8, 2, 100, 10, [(5, 9), (8, 12)])[0] == -1  # overlap
    assert plan_prefill(8, 2, 100, 10, [(90, 101)])[0] == -1   # past the end
    assert plan_prefill(8, 2, 100, 10, [(-1, 3)])[0] == -1
    rc, info, _ = plan_prefill(8, 2, 100, 10, [(0, 100)])      # everything masked
    assert rc == 0 and info["n_tiles"] == 0 and info["visible_pairs"] == 0


def test_prefill_plan_splits_short_query_blocks():
    # 8 trigger tokens over a long context: one query tile per KV head, so the
    # key range is split to fill the GPU; a full prefill is not split.
    from tests.hostlib import plan_prefill
    rc, info, _ = plan_prefill(32, 8, 131072, 8, [])
    assert rc == 0 and info["n_qt"] == 1 and info["n_split"] == 19
    # 512 queries: 64 CTA tiles; the split fills its waves of 152 CTAs (not
    # 3 splits = 192 CTAs, whose second wave is 26% full)
    rc, info, _ = plan_prefill(32, 8, 131072, 512, [])
    ctas = 64 * info["n_split"]
    assert rc == 0 and info["n_qt"] == 8 and info["n_split"] > 1
    assert ctas / (-(-ctas // 152) * 152) >= 0.9
    rc, info, _ = plan_prefill(32, 8, 32768, 32768, [(100, 5000)])
    assert rc == 0 and info["n_split"] == 1 and info["n_qt"] == 512


def test_next_position_counts_appends_not_evictions():
    # the position of a sequence's next token: every appended token advances
    # it, a fork starts from its parent's, eviction leaves it (kept keys keep
    # the rotary phase of their original positions), a refused append does not
    hc = HostCache(1, 8, 2, 64, 16, 40)
    rc, m = hc.seq_new()
    assert rc == 0 and hc.next_pos(m) == 0
    assert hc.append(m, 100) == 0
    assert hc.next_pos(m) == 100
    rc, a = hc.fork(m)
    assert rc == 0 and hc.next_pos(a) == 100
    assert hc.append(a, 7) == 0
    assert (hc.next_pos(a), hc.next_pos(m)) == (107, 100)
    rc, _ = hc.evict(m, [(10, 50), (60, 61)])
    assert rc == 0
    assert hc.info(m)[1] == 59 and hc.next_pos(m) == 100
    assert hc.append(m, 1) == 0
    assert (hc.info(m)[1], hc.next_pos(m)) == (60, 101)
    assert hc.append(m, 16 * 40) != 0           # more pages than the pool holds
    assert (hc.info(m)[1], hc.next_pos(m)) == (60, 101)
    assert hc.release(a) == 0
    rc, b = hc.seq_new()                         # a fresh handle starts at 0
    assert rc == 0 and hc.next_pos(b) == 0


@pytest.mark.parametrize("seed", range(10))
def test_prefill_slot_spans_on_partial_pages(seed):
    """A masked prefill over a sequence with partial pages runs in slot space:
    the masked slots are exactly the slots of the spans' rows plus the unused
    slots of every page but the last, the end is (pages - 1) x P + last fill,
    and queries that a partial page would split are refused."""
    rng = random.Random(900 + seed)
    P = rng.choice([8, 16, 64])
    hc = HostCache(1, 8, 2, 64, P, 3000)
    oc = ocm.OracleCache(3000, P)
    rc, m = hc.seq_new()
    om = oc.seq_new()
    n0 = rng.randint(4 * P, 30 * P)
    hc.append(m, n0)
    oc.append(om, n0)
    pre = random_spans(rng, n0, rng.choice([1, 3, 6]))
    assert hc.evict(m, pre, ragged=True)[0] == 0
    oc.evict(om, pre, mode="ragged")
    tail = rng.randint(1, 3 * P)
    hc.append(m, tail)
    oc.append(om, tail)
    n = oc.n_tokens(om)
    fills = oc.page_fills(om)
    slot_of = [q * P + t for q, f in enumerate(fills) for t in range(f)]
    end = (len(fills) - 1) * P + fills[-1]
    spans = random_spans(rng, n - tail, rng.choice([0, 1, 4]))
    for n_q in (1, tail, min(n, tail + rng.randint(1, 4 * P)), n):
        rc, sl, n_slots = hc.prefill_slot_spans(m, n_q, spans)
        contiguous = slot_of[n - n_q] == end - n_q
        if not contiguous:
            assert rc == -8            # unsupported
            continue
        assert rc == 0 and n_slots == end
        masked = set()
        for a, b in spans:
            masked.update(slot_of[j] for j in range(a, b))
        for q, f in enumerate(fills[:-1]):
            masked.update(range(q * P + f, (q + 1) * P))
        got = set()
        prev = -1
        for a, b in sl:
            assert prev < a < b        # sorted, disjoint, not touching (merged)
            prev = b
            got.update(range(a, b))
        assert got == masked
    assert hc.prefill_slot_spans(m, tail, [(0, n + 1)])[0] == -1   # bad span


def test_prefill_tiles_skip_boxes_a_span_covers():
    """With 64-token pages a key tile pairs the visible 64-key boxes: a box
    that a span covers entirely costs no tile half, even when its aligned
    128-key neighbour is visible."""
    from tests.hostlib import plan_prefill
    rc, info, tiles = plan_prefill(8, 2, 512, 512, [(64, 128), (256, 384)], P=64)
    assert rc == 0
    # visible boxes 0, 128, 192, 384, 448 -> tiles (0, 128), (192, 384), (448, -)
    assert [(int(t[0]), int(t[6])) for t in tiles] == [(0, 128), (192, 384), (448, NO_KEYS)]
    assert all(int(t[1]) == 1 for t in tiles[:2]) and int(tiles[2][1]) == 0
    # the same spans with 16-token pages keep aligned 128-key tiles
    rc, info, tiles = plan_prefill(8, 2, 512, 512, [(64, 128), (256, 384)], P=16)
    assert [int(t[0]) for t in tiles] == [0, 128, 384]


def test_evict_shape_rule():
    # 8 KiB tiles, at most a page; ring slots by the planes per SM
    L_ = lib()
    assert L_.sqh_evict_tile_rows(64, 128) == 32
    assert L_.sqh_evict_tile_rows(64, 64) == 64
    assert L_.sqh_evict_tile_rows(16, 128) == 16
    assert L_.sqh_evict_tile_rows(8, 64) == 8
    assert L_.sqh_evict_tile_rows(256, 64) == 64
    for planes, stages in ((1, 6), (128, 6), (152, 6), (153, 3), (512, 3), (608, 3), (609, 4),
                           (1280, 4), (100000, 4)):
        assert L_.sqh_evict_stages(planes, 152) == stages, planes
