"""GPU parity of the CUDA path against the CPU oracle (through the C ABI).

Page tables, token counts, reference counts and post-compaction K/V contents
must match bit for bit; decode attention within max-abs 1e-2 and mean-abs
1e-3 of the double-precision oracle."""
import math
import random

import numpy as np
import pytest
import torch

import paper_2602_22603_gb300 as sq
from synthetic import TINY, bf16_normal, random_spans, shuffled
from tests.gpu_harness import MAX_ABS, MEAN_ABS, Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _q(seed, S, Hq, D):
    q = bf16_normal((S, Hq, D), seed)
    return q, q.cuda()


def _decode_check(p: Pair, seqs, layer, scale, seed):
    q_cpu, q = _q(seed, len(seqs), p.Hq, p.D)
    exp, budget = p.oracle_decode_budget(seqs, layer, scale, q_cpu)
    out32 = p.decode(seqs, layer, scale, q, sq.SQ_OUT_F32)
    out16 = p.decode(seqs, layer, scale, q, sq.SQ_OUT_BF16)
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    e32 = assert_budget(out32, exp, budget)
    e16 = assert_close(out16, exp)
    # the bf16 output is the fp32 output rounded to nearest even
    assert torch.equal(out16, out32.to(torch.bfloat16))
    return e32, e16


def test_tiny_workload_full_parity():
    """1 layer, 16 q / 4 kv heads, d 64, P 16, seed 0: 2,048-token prefix,
    fork, main +32 / aux +64, one decode step each, evict 5 spans (30% of the
    prefix) from main while the aux is alive, one more decode step each."""
    s = TINY
    p = Pair(s.num_layers, s.num_q_heads, s.num_kv_heads, s.head_dim, s.page_size,
             num_pages=400, seed=0)
    scale = 1.0 / math.sqrt(s.head_dim)
    keep = []
    main = p.seq_new()
    keep.append(p.append(main, 2048))
    aux = p.fork(main)
    p.check_tables()
    assert p.cache.stats()["live_pages"] == 2048 // 16   # the fork copied nothing
    keep.append(p.append(main, 32))
    keep.append(p.append(aux, 64))
    for step in range(2):
        keep.append(p.append(main, 1))
        keep.append(p.append(aux, 1))
        _decode_check(p, [main, aux], 0, scale, 10 + step)
        if step == 0:
            spans = random_spans(seed=1, n_spans=5, total=int(0.3 * 2048), lo=s.page_size,
                                 hi=2048, median=100)
            r = p.evict(main, shuffled(spans, 2))
            assert r["cow_pages"] > 0          # shared changed pages were copied
        p.check_tables()
        p.check_contents(main)
        p.check_contents(aux)
    st = p.cache.stats()
    assert st["evict_calls"] == 1 and st["evicted_tokens"] == int(0.3 * 2048)
    p.close()


@pytest.mark.parametrize("P,G,D", [(16, 1, 64), (16, 4, 128), (64, 4, 128), (64, 8, 128),
                                   (64, 8, 64), (32, 16, 64), (128, 2, 128), (8, 4, 64),
                                   (256, 4, 128), (64, 3, 64), (16, 6, 128), (32, 5, 128)])
def test_ragged_lengths(P, G, D):
    Hkv = 2
    p = Pair(2, G * Hkv, Hkv, D, P, num_pages=4000 // max(1, P // 16), seed=P * 31 + G * 7 + D)
    keep = []
    lengths = [1, P - 1, P, P + 1, 3 * P + 7, 700]
    seqs = []
    for n in lengths:
        h = p.seq_new()
        keep.append(p.append(h, n))
        seqs.append(h)
    p.check_tables()
    for h in seqs:
        p.check_contents(h)
    for layer in range(2):
        _decode_check(p, seqs, layer, 1.0 / math.sqrt(D), 5 + layer)
    p.close()


def test_split_invariance_over_cta_counts():
    """The same decode with 1 .. many persistent CTAs (so 1 .. many partials
    per sequence and head) agrees with the oracle and with itself."""
    outs = []
    budget = None
    for ctas in (1, 2, 7, 64, 304, 1000):
        p = Pair(1, 32, 8, 128, 64, num_pages=600, decode_ctas=ctas, seed=3)
        keep = []
        m = p.seq_new()
        keep.append(p.append(m, 9000))
        a = p.fork(m)
        keep.append(p.append(a, 40))
        keep.append(p.append(m, 3))
        q_cpu, q = _q(77, 2, 32, 128)
        out = p.decode([m, a], 0, 0.0884, q, sq.SQ_OUT_F32)
        torch.cuda.synchronize()
        exp, budget = p.oracle_decode_budget([m, a], 0, 0.0884, q_cpu)
        assert_budget(out, exp, budget)
        outs.append(out.cpu())
        p.close()
    # every split is within the budget of the exact result, so two splits
    # are within twice the budget of each other
    for o in outs[1:]:
        assert np.all((o - outs[0]).abs().double().numpy() <= 2 * budget)


@pytest.mark.parametrize("Hq,Hkv,D,P,ctas,n", [
    (32, 2, 64, 32, 400, 9000),    # G = 16: runs of ~140 entries merge in chunks of 22
    (6, 2, 128, 256, 200, 3000),   # G = 3: several runs per merge round (96 outputs each)
    (8, 8, 64, 16, 300, 2000),     # G = 1, d = 64: 16 outputs per run, many runs per CTA
    (16, 4, 64, 16, 1, 700),       # one CTA: every run is one item (direct outputs)
    (16, 1, 128, 64, 304, 5000),   # one KV head, G = 16: a run fills a round's 512 outputs
])
def test_merge_paths_across_shapes(Hq, Hkv, D, P, ctas, n):
    """The in-kernel merge across group sizes, head dims and CTA counts: main
    and fork share a prefix, each adds its own tail; every (sequence, KV head)
    run is merged by the CTA that completes it (or written directly when it is
    one item) and must equal the oracle."""
    p = Pair(1, Hq, Hkv, D, P, num_pages=3 * (n // P) + 40, decode_ctas=ctas, seed=n + ctas)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, n))
    a = p.fork(m)
    keep.append(p.append(a, 37))
    keep.append(p.append(m, 5))
    b = p.fork(a)
    keep.append(p.append(b, 1))
    _decode_check(p, [m, a, b], 0, 1.0 / math.sqrt(D), n + 1)
    p.close()


def test_one_cta_merges_hundreds_of_runs():
    """decode_ctas = 1: the one CTA holds every item (40 sequences, 8 KV heads:
    320 arrivals, three rounds of 128) and completes, so merges, every
    (sequence, KV head) run itself; forks make two-member groups too."""
    p = Pair(1, 32, 8, 128, 16, num_pages=700, decode_ctas=1, seed=52)
    rng = np.random.default_rng(52)
    keep = []
    seqs = []
    for i in range(30):
        h = p.seq_new()
        keep.append(p.append(h, int(rng.integers(1, 300))))
        seqs.append(h)
    for h in seqs[:10]:
        f = p.fork(h)
        keep.append(p.append(f, int(rng.integers(1, 20))))
        seqs.append(f)
    _decode_check(p, seqs, 0, 0.0884, 53)
    p.close()


def test_cached_plan_reused_across_streams():
    """The same sequences decoded on stream A, then B, then A again: each later
    call reuses the cached plan (its arrival counts and partial buffers too)
    after waiting for the other stream's use of it, and every result equals
    the oracle."""
    p = Pair(2, 32, 8, 128, 64, num_pages=200, decode_ctas=300, seed=56)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 2500))
    a = p.fork(m)
    keep.append(p.append(a, 24))
    seqs = [m, a]
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    sa.wait_stream(torch.cuda.current_stream())
    sb.wait_stream(torch.cuda.current_stream())
    checks = []
    for i, st in enumerate((sa, sb, sa, sb, sb, sa)):
        q_cpu, q = _q(700 + i, 2, 32, 128)
        keep.append(q)
        st.wait_stream(torch.cuda.current_stream())   # q was copied on the default stream
        with torch.cuda.stream(st):
            out = p.decode(seqs, i % 2, 0.09, q, sq.SQ_OUT_F32, st)
        checks.append((out, i % 2, q_cpu))
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    for out, layer, q_cpu in checks:
        assert_budget(out, *p.oracle_decode_budget(seqs, layer, 0.09, q_cpu))
    p.close()


def test_decode_replayed_from_a_cuda_graph():
    """Replays of a captured decode repeat its kernel arguments, the merge's
    arrival tag among them: every replay must still merge each run once
    (the last arrival clears the word), with fresh queries each time."""
    p = Pair(2, 32, 8, 128, 64, num_pages=200, decode_ctas=300, seed=54)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 3000))
    a = p.fork(m)
    keep.append(p.append(a, 40))
    seqs = [m, a]
    q = torch.zeros(2, 32, 128, dtype=torch.bfloat16, device="cuda")
    outs = [torch.zeros(2, 32, 128, device="cuda") for _ in range(2)]
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for layer in range(2):      # plans made and cached on the capture stream
            p.cache.decode_attention(seqs, layer, q, outs[layer], sq.SQ_OUT_F32, 0.09)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for layer in range(2):
            p.cache.decode_attention(seqs, layer, q, outs[layer], sq.SQ_OUT_F32, 0.09)
    for rep in range(3):
        q_cpu = bf16_normal((2, 32, 128), 60 + rep)
        q.copy_(q_cpu.cuda())
        for o in outs:
            o.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert p.cache.sync_status() == sq.SQ_OK
        for layer in range(2):
            assert_budget(outs[layer], *p.oracle_decode_budget(seqs, layer, 0.09, q_cpu))
    del g
    p.close()


@pytest.mark.parametrize("seed", range(5))
def test_random_forks_appends_evictions(seed):
    rng = random.Random(seed)
    P = (8, 16, 32, 64, 256)[seed % 5]
    D = rng.choice([64, 128])
    G = rng.choice([1, 4, 8])
    Hkv = rng.choice([1, 2, 4])
    L = 2
    p = Pair(L, G * Hkv, Hkv, D, P, num_pages=3000, seed=seed)
    keep = []
    mains = []
    for _ in range(2):
        h = p.seq_new()
        keep.append(p.append(h, rng.randint(P, 60 * P)))
        mains.append(h)
    live = list(mains)
    for it in range(6):
        h = rng.choice(live)
        op = rng.random()
        if op < 0.3 and len(live) < 8:
            live.append(p.fork(h))
        elif op < 0.7:
            keep.append(p.append(h, rng.choice([1, 2, P - 1, P + 3, 5 * P])))
        else:
            n = p.cache.seq_info(h)[0]
            k = rng.randint(1, 6)
            if n > 4 * k:
                spans = random_spans(seed=seed * 100 + it, n_spans=k,
                                     total=rng.randint(k, n // 2), lo=0, hi=n,
                                     median=max(1, n // (4 * k)))
                p.evict(h, shuffled(spans, it))
        p.check_tables()
        for x in live:
            p.check_contents(x)
        _decode_check(p, live, rng.randrange(L), 1.0 / math.sqrt(D), 1000 + it)
    # releasing forks frees exactly their private pages
    for x in live[2:]:
        p.release(x)
    p.check_tables()
    p.close()


def test_evict_edge_cases():
    p = Pair(1, 8, 2, 64, 16, num_pages=200, seed=11)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 100))
    snap = p.cache.page_table(m)
    p.evict(m, [])                                   # no spans: identity
    assert p.cache.page_table(m) == snap
    p.check_contents(m)
    p.evict(m, [(0, 1)])                             # first token
    p.evict(m, [(98, 99)])                           # last token
    p.evict(m, [(10, 20), (20, 30)])                 # adjacent spans
    p.evict(m, [(0, 16)])                            # exactly one page
    p.check_tables()
    p.check_contents(m)
    n = p.cache.seq_info(m)[0]
    p.evict(m, [(5, n)])                             # everything after a prefix
    p.check_tables()
    p.check_contents(m)
    for bad in ([(3, 2)], [(-1, 2)], [(0, 999)], [(0, 3), (2, 4)]):
        before = p.cache.page_table(m)
        with pytest.raises(sq.SqError) as e:
            p.cache.evict_spans(m, bad)
        assert e.value.code == sq.SQ_ERR_INVALID_ARG
        assert p.cache.page_table(m) == before
    p.evict(m, [(0, 5)])                             # everything: empty sequence
    assert p.cache.seq_info(m) == (0, 0)
    out = torch.empty(1, 8, 64, device="cuda")
    with pytest.raises(sq.SqError) as e:
        p.cache.decode_attention([m], 0, torch.zeros(1, 8, 64, dtype=torch.bfloat16,
                                                     device="cuda"), out, sq.SQ_OUT_F32)
    assert e.value.code == sq.SQ_ERR_INVALID_ARG     # empty-sequence decode
    keep.append(p.append(m, 20))                     # it can grow again
    p.check_tables()
    p.check_contents(m)
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


def test_no_pages_is_transactional():
    p = Pair(1, 4, 1, 64, 16, num_pages=6, seed=5)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 90))                     # 6 pages, the last one partial
    a = p.fork(m)
    before = (p.cache.page_table(m), p.cache.free_pages())
    with pytest.raises(sq.SqError) as e:
        p.cache.append_kv(m, 1, keep[0][0], keep[0][1])
    assert e.value.code == sq.SQ_ERR_NO_PAGES
    with pytest.raises(sq.SqError) as e:
        p.cache.evict_spans(m, [(0, 1)])
    assert e.value.code == sq.SQ_ERR_NO_PAGES
    assert (p.cache.page_table(m), p.cache.free_pages()) == before
    p.release(a)
    p.evict(m, [(0, 1)])                             # private now: in place
    p.check_tables()
    p.check_contents(m)
    p.close()


def test_argument_errors():
    c = sq.Cache(2, 8, 2, 64, 16, 50)
    m = c.seq_new()
    k = torch.zeros(2, 4, 2, 64, dtype=torch.bfloat16, device="cuda")
    c.append_kv(m, 4, k, k)
    q = torch.zeros(1, 8, 64, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(1, 8, 64, device="cuda")
    for kwargs, code in [
        (dict(seqs=[m], layer=2), sq.SQ_ERR_INVALID_ARG),
        (dict(seqs=[m], layer=-1), sq.SQ_ERR_INVALID_ARG),
        (dict(seqs=[m, m], layer=0), sq.SQ_ERR_INVALID_ARG),
        (dict(seqs=[m + 1], layer=0), sq.SQ_ERR_BAD_HANDLE),
    ]:
        with pytest.raises(sq.SqError) as e:
            c.decode_attention(kwargs["seqs"], kwargs["layer"], q, out, sq.SQ_OUT_F32)
        assert e.value.code == code
    with pytest.raises(sq.SqError) as e:
        c.decode_attention([m], 0, q, out, 7)
    assert e.value.code == sq.SQ_ERR_INVALID_ARG
    with pytest.raises(sq.SqError) as e:                # misaligned input
        c.append_kv(m, 1, k.view(-1)[1:].data_ptr(), k)
    assert e.value.code == sq.SQ_ERR_INVALID_ARG
    with pytest.raises(sq.SqError) as e:
        c.append_kv(m, -3, k, k)
    assert e.value.code == sq.SQ_ERR_INVALID_ARG
    c.release(m)
    with pytest.raises(sq.SqError) as e:
        c.append_kv(m, 1, k, k)
    assert e.value.code == sq.SQ_ERR_BAD_HANDLE
    assert c.sync_status() == sq.SQ_OK
    c.close()


def test_two_streams_main_and_aux():
    """Main and aux decode on two streams, interleaved from one host thread
    (single-agent workload shape, at a reduced size); then the aux is
    released on its stream and main evicts on its own."""
    p = Pair(2, 32, 8, 128, 64, num_pages=800, seed=21, k_scale=1 / math.sqrt(128))
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 4096))
    torch.cuda.synchronize()
    a = p.fork(m)
    checks = []
    for step in range(6):
        with torch.cuda.stream(sa):
            keep.append(p.append(m, 1, sa))
            q_cpu, q = _q(500 + step, 1, 32, 128)
            keep.append(q)
            out = p.decode([m], step % 2, 1.0, q, sq.SQ_OUT_F32, sa)
            checks.append((out, p.oracle_decode_budget([m], step % 2, 1.0, q_cpu)))
        if step % 2 == 0:
            with torch.cuda.stream(sb):
                keep.append(p.append(a, 1, sb))
                q_cpu, q = _q(900 + step, 1, 32, 128)
                keep.append(q)
                out = p.decode([a], step % 2, 1.0, q, sq.SQ_OUT_F32, sb)
                checks.append((out, p.oracle_decode_budget([a], step % 2, 1.0, q_cpu)))
    torch.cuda.synchronize()
    for out, (exp, budget) in checks:
        assert_budget(out, exp, budget)
    p.release(a, sb)
    with torch.cuda.stream(sa):
        spans = random_spans(seed=4, n_spans=12, total=int(0.4 * 4096), lo=64, hi=4096, median=150)
        p.evict(m, spans, sa)
        keep.append(p.append(m, 70, sa))     # may reuse pages the aux released on sb
    torch.cuda.synchronize()
    p.check_tables()
    p.check_contents(m)
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


@pytest.mark.parametrize("sm_scale", [1.0, 1.0 / math.sqrt(128)])
def test_agent_shape_key_scaling_readings(sm_scale):
    """Single-agent shape with keys N(0,1)/sqrt(128): the reading taken
    (sm_scale 1, the 1/sqrt(d) folded into the keys) and the alternate one
    (1/sqrt(d) applied again at decode) both match the oracle."""
    p = Pair(2, 32, 8, 128, 64, num_pages=400, seed=31, k_scale=1 / math.sqrt(128))
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 5000))
    a = p.fork(m)
    keep.append(p.append(a, 8))
    for layer in range(2):
        _decode_check(p, [m, a], layer, sm_scale, 40 + layer)
    p.close()


def test_short_agent_loop_trace():
    """Algorithm 1 at a reduced size: 2 agents x 9 turns; every turn 6 main
    decode steps then a tool response; every 4 turns an aux fork (trigger +
    3 steps, decoded with the mains in one call); at the next turn release
    it and evict whole tool responses older than 2 turns until >= 60% of
    their tokens are covered.  Page tables, contents and attention outputs
    are checked against the oracle along the way."""
    rng = random.Random(77)
    P = 16
    p = Pair(2, 16, 4, 64, P, num_pages=3000, seed=77)
    keep = []
    mains = [p.seq_new() for _ in range(2)]
    for m in mains:
        keep.append(p.append(m, 40))            # the user query
    responses = {m: [] for m in mains}          # (turn, start, end)
    auxs = []
    for t in range(9):
        if auxs:
            for x in auxs:
                p.release(x)
            auxs = []
            for m in mains:
                old = [r for r in responses[m] if r[0] < t - 2]
                if not old:
                    continue
                rng.shuffle(old)
                total = sum(e - s for _, s, e in old)
                chosen, cov = [], 0
                for r in old:
                    if cov >= 0.6 * total:
                        break
                    chosen.append(r)
                    cov += r[2] - r[1]
                p.evict(m, [(s, e) for _, s, e in chosen])
                gone = sorted((s, e) for _, s, e in chosen)
                kept = []
                for r in responses[m]:
                    if r in chosen:
                        continue
                    sh = sum(e - s for s, e in gone if e <= r[1])
                    kept.append((r[0], r[1] - sh, r[2] - sh))
                responses[m] = kept
            p.check_tables()
            for m in mains:
                p.check_contents(m)
        if t % 4 == 0:
            for m in mains:
                a = p.fork(m)
                keep.append(p.append(a, 8))
                auxs.append(a)
        for s_ in range(6):
            seqs = mains + (auxs if s_ < 3 else [])
            for h in seqs:
                keep.append(p.append(h, 1))
            if s_ in (0, 5):
                _decode_check(p, seqs, s_ % 2, 0.125, 1000 * t + s_)
        for m in mains:
            n = p.cache.seq_info(m)[0]
            ln = rng.choice([17, 60, 150, 333])
            keep.append(p.append(m, ln))
            responses[m].append((t, n, n + ln))
    p.check_tables()
    for h in mains + auxs:
        p.check_contents(h)
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


def test_batched_single_token_append():
    """sq_append_kv_batch = one sq_append_kv of one token per sequence, in the
    order given: same page tables (including the copy-on-write of a shared
    partial last page right after a fork), same contents."""
    P = 16
    p = Pair(2, 8, 2, 64, P, num_pages=400, seed=61)
    keep = []
    seqs = []
    for n in (1, P - 1, P, 37):
        h = p.seq_new()
        keep.append(p.append(h, n))
        seqs.append(h)
    seqs.append(p.fork(seqs[3]))            # shares a partial last page
    for step in range(2 * P + 3):
        keep.append(p.append_batch(seqs))
    p.check_tables()
    for h in seqs:
        p.check_contents(h)
    _decode_check(p, seqs, 1, 0.125, 7)
    # all or nothing: a bad handle in the batch changes nothing
    before = [p.cache.page_table(h) for h in seqs]
    with pytest.raises(sq.SqError) as e:
        p.cache.append_kv_batch(seqs + [123456789], keep[-1][0], keep[-1][1])
    assert e.value.code == sq.SQ_ERR_BAD_HANDLE
    with pytest.raises(sq.SqError) as e:
        p.cache.append_kv_batch([seqs[0], seqs[0]], keep[-1][0], keep[-1][1])
    assert e.value.code == sq.SQ_ERR_INVALID_ARG
    assert before == [p.cache.page_table(h) for h in seqs]
    p.close()


def test_many_sequences_in_one_call():
    """64 sequences of mixed lengths (some sharing prefixes) in one decode
    call: many segments, items and combine lists."""
    rng = random.Random(5)
    p = Pair(1, 32, 8, 128, 64, num_pages=4000, max_seqs=128, seed=55)
    keep = []
    seqs = []
    for i in range(40):
        h = p.seq_new()
        keep.append(p.append(h, rng.choice([1, 63, 64, 65, 500, 3000])))
        seqs.append(h)
    for i in range(24):
        a = p.fork(seqs[i])
        keep.append(p.append(a, rng.choice([1, 7, 70])))
        seqs.append(a)
    rng.shuffle(seqs)
    _decode_check(p, seqs, 0, 0.0884, 3)
    p.close()


def test_next_position_through_the_api():
    # the same counter through the C ABI: appends advance it, a fork inherits
    # it, eviction leaves it, a bad handle is refused
    p = Pair(1, 16, 4, 64, 16, num_pages=40, seed=3)
    try:
        m = p.seq_new()
        p.append(m, 100)
        assert p.cache.next_pos(m) == 100
        a = p.fork(m)
        p.append(a, 5)
        assert (p.cache.next_pos(a), p.cache.next_pos(m)) == (105, 100)
        p.evict(m, [(0, 30)])
        assert p.cache.seq_info(m)[0] == 70 and p.cache.next_pos(m) == 100
        with pytest.raises(sq.SqError) as ei:
            sq.sq_seq_next_pos(p.cache.handle, 123456789)
        assert ei.value.code == sq.SQ_ERR_BAD_HANDLE
    finally:
        p.close()


def test_decode_steps_reuse_plans_with_early_loads():
    """Decode steps as a model runs them: one batched append, then every
    layer's call on one stream.  Every call after a step's first reuses the
    step's plan and loads its first stages before its dependency wait (the
    pages the step's append wrote are excluded until that append is known
    complete); each output must equal the oracle."""
    L = 6
    p = Pair(L, 32, 8, 128, 64, num_pages=900, seed=88)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 20000))
    a = p.fork(m)
    keep.append(p.append(a, 30))
    seqs = [m, a]
    checks = []
    st0 = p.cache.stats()
    rebuilds = 0
    for step in range(3):
        # a plan is built for the first step, and again only when an append
        # opens a page (P = 64: also a 64-token stage) of some sequence
        if step == 0 or any(p.oracle.n_tokens(p.o[h]) % 64 == 0 for h in seqs):
            rebuilds += 1
        keep.append(p.append_batch(seqs))
        for layer in range(L):
            q_cpu, q = _q(900 + 10 * step + layer, 2, 32, 128)
            keep.append(q)
            out = p.decode(seqs, layer, 0.09, q, sq.SQ_OUT_F32)
            checks.append((out, layer, q_cpu, [p.oracle.n_tokens(p.o[h]) for h in seqs]))
        torch.cuda.synchronize()
        for out, layer, q_cpu, ns in checks:
            assert_budget(out, *p.oracle_decode_budget(seqs, layer, 0.09, q_cpu))
        checks.clear()
    st1 = p.cache.stats()
    # the calls after each step's first reused the plan and loaded early (in
    # steps 1 and 2 at least: every earlier write had completed by then)
    assert st1["decode_early_calls"] - st0["decode_early_calls"] >= 2 * (L - 1)
    # the batched appends inside both sequences' last pages kept the plan
    # (the fork's third append opens a page: 20,032 rows before it)
    assert st1["decode_plans_built"] - st0["decode_plans_built"] == rebuilds == 2
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


@pytest.mark.parametrize("P", [64, 128])
def test_decode_plan_survives_in_page_appends(P):
    """One-token appends (sq_append_kv) between decode steps: an append
    inside the sequence's last page and 64-token stage keeps the cached plan
    (the append kernel rewrites the sequence's length in it), one that opens
    a page or a stage has it rebuilt; every output equals the oracle."""
    L = 3
    p = Pair(L, 16, 4, 64, P, num_pages=400, seed=91)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 4 * 64 + 58))   # the 6th step's append starts at 320
    st0 = p.cache.stats()
    rebuilds = 1                             # the first step plans
    for step in range(10):
        n_before = p.oracle.n_tokens(p.o[m])
        if step > 0 and n_before % 64 == 0:  # a new 64-token stage (for P = 64 a new page)
            rebuilds += 1
        keep.append(p.append(m, 1))
        for layer in range(L):
            q_cpu, q = _q(1300 + 10 * step + layer, 1, 16, 64)
            keep.append(q)
            out = p.decode([m], layer, 0.125, q, sq.SQ_OUT_F32)
            torch.cuda.synchronize()
            assert_budget(out, *p.oracle_decode_budget([m], layer, 0.125, q_cpu))
    st1 = p.cache.stats()
    assert st1["decode_plans_built"] - st0["decode_plans_built"] == rebuilds == 2
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()
