"""GPU parity of ragged-page eviction (sq_evict_spans_ragged) and of the
kernels that read partial pages, against the CPU oracle.

Page tables, page fills, reference counts and the K/V rows of every sequence
(read through the page table and the fills) must match the oracle bit for
bit; so must the zeros the eviction writes past a window's last rows.
Decode outputs are checked against the oracle within the contract's
tolerance and element by element within the kernel's error budget; masked
prefill over a sequence with partial pages within the contract's tolerance."""
import math
import random

import numpy as np
import pytest
import torch

import paper_2602_22603_gb300 as sq
from oracle import attention as oatt
from synthetic import TINY, bf16_bits, bf16_normal, random_spans, shuffled
from tests.gpu_harness import Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _decode_check(p, seqs, layer, scale, seed):
    q_cpu = bf16_normal((len(seqs), p.Hq, p.D), seed)
    q = q_cpu.cuda()
    exp, budget = p.oracle_decode_budget(seqs, layer, scale, q_cpu)
    out32 = p.decode(seqs, layer, scale, q, sq.SQ_OUT_F32)
    out16 = p.decode(seqs, layer, scale, q, sq.SQ_OUT_BF16)
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    assert_budget(out32, exp, budget)
    assert_close(out16, exp)
    assert torch.equal(out16, out32.to(torch.bfloat16))


def test_tiny_workload_ragged():
    """The tiny workload (1 layer, 16q/4kv, d64, P16, seed 0) with the
    eviction done by ragged packing while the fork is alive: the shared pages
    whose rows change are copied, untouched pages stay shared."""
    s = TINY
    p = Pair(s.num_layers, s.num_q_heads, s.num_kv_heads, s.head_dim, s.page_size,
             num_pages=400, seed=0, physical=True)
    scale = 1.0 / math.sqrt(s.head_dim)
    keep = []
    main = p.seq_new()
    keep.append(p.append(main, 2048))
    aux = p.fork(main)
    keep.append(p.append(main, 32))
    keep.append(p.append(aux, 64))
    for step in range(2):
        keep.append(p.append(main, 1))
        keep.append(p.append(aux, 1))
        _decode_check(p, [main, aux], 0, scale, 10 + step)
        if step == 0:
            spans = random_spans(seed=1, n_spans=5, total=int(0.3 * 2048), lo=s.page_size,
                                 hi=2048, median=100)
            r = p.evict(main, shuffled(spans, 2), ragged=True)
            assert r["cow_pages"] > 0 and r["moved_rows"] <= 2 * s.page_size * len(spans)
            st = p.cache.stats()
            assert st["evict_moved_rows"] == r["moved_rows"]
        p.check_tables()
        p.check_contents(main)
        p.check_contents(aux)
        p.check_zero_slots()
    p.close()


@pytest.mark.parametrize("seed", range(12))
def test_random_ops_with_ragged_evictions(seed):
    rng = random.Random(seed)
    P = (8, 16, 32, 64, 128, 256)[seed % 6]   # every page size twice
    D = rng.choice([64, 128])
    G = rng.choice([1, 4, 8])
    Hkv = 2
    p = Pair(2, G * Hkv, Hkv, D, P, num_pages=8000 // max(1, P // 8), seed=40 + seed,
             decode_ctas=rng.choice([0, 7, 300]), physical=True)
    scale = 1.0 / math.sqrt(D)
    keep = []
    live = []
    for step in range(14):
        op = rng.random()
        if not live or op < 0.12:
            h = p.seq_new()
            keep.append(p.append(h, rng.randint(1, 30 * P)))
            live.append(h)
        elif op < 0.3:
            f = p.fork(rng.choice(live))
            keep.append(p.append(f, rng.randint(0, 2 * P)))
            live.append(f)
        elif op < 0.5:
            h = rng.choice(live)
            keep.append(p.append(h, rng.choice([1, P - 1, P + 1, rng.randint(1, 4 * P)])))
        elif op < 0.9:
            h = rng.choice(live)
            n = p.cache.seq_info(h)[0]
            if n < 4:
                continue
            k = rng.randint(1, 8)
            total = rng.randint(1, max(1, n // 2))
            spans = random_spans(seed=1000 * seed + step, n_spans=min(k, total), total=total,
                                 lo=0, hi=n, median=max(1.0, total / k))
            p.evict(h, shuffled(spans, step), ragged=rng.random() < 0.75)
        elif len(live) > 1:
            h = live.pop(rng.randrange(len(live)))
            p.release(h)
        p.check_tables()
        for h in live:
            p.check_contents(h)
        p.check_zero_slots()
        _decode_check(p, live, step % 2, scale, 100 * seed + step)
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


@pytest.mark.parametrize("P,ctas", [(8, 1), (8, 300), (64, 7), (64, 304), (256, 50)])
def test_ragged_decode_over_many_windows(P, ctas):
    """A long main thread and its fork after a ragged eviction of 40 spans:
    dozens of partial pages (fill masks in every stage kind: several pages
    per stage, one page per stage, several stages per page), read by 1 to
    hundreds of CTAs."""
    p = Pair(1, 32, 8, 128, P, num_pages=40000 // P + 64, decode_ctas=ctas, seed=P + ctas)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 20000))
    spans = random_spans(seed=P, n_spans=40, total=9000, lo=0, hi=20000, median=200)
    r = p.evict(m, shuffled(spans, 3), ragged=True)
    assert r["windows"] > 10
    assert any(f < P for f in p.cache.page_fills(m)[:-1])
    a = p.fork(m)
    keep.append(p.append(a, 70))
    keep.append(p.append(m, 1))
    p.check_tables()
    p.check_contents(m)
    _decode_check(p, [m, a], 0, 0.0884, 9)
    p.close()


def test_ragged_then_dense_packs_again():
    p = Pair(2, 16, 4, 64, 16, num_pages=800, seed=77, physical=True)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 3000))
    p.evict(m, [(17, 40), (500, 777), (1024, 1025), (2999, 3000)], ragged=True)
    keep.append(p.append(m, 20))
    p.evict(m, [(0, 3), (1500, 1600)])           # dense: packs every page
    fills = p.cache.page_fills(m)
    assert all(f == 16 for f in fills[:-1])
    p.check_tables()
    p.check_contents(m)
    _decode_check(p, [m], 1, 0.125, 5)
    p.close()


def _prefill_check(p, h, layer, n_q, spans, seed, scale):
    q_cpu = bf16_normal((n_q, p.Hq, p.D), seed)
    out = torch.empty(n_q, p.Hq, p.D, dtype=torch.float32, device="cuda")
    lse = torch.empty(n_q, p.Hq, dtype=torch.float32, device="cuda")
    p.cache.prefill_attention(h, layer, n_q, q_cpu.cuda(), out, sq.SQ_OUT_F32, lse, scale, spans)
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    k, v = p.store.rows(p.oracle.tokens(p.o[h]), layer)
    exp, exp_lse = oatt.prefill(bf16_bits(q_cpu), k, v, scale, spans, want_lse=True)
    assert_close(out, exp)
    fin = np.isfinite(exp_lse)
    got = lse.cpu().numpy().astype(np.float64)
    assert np.abs(got[fin] - exp_lse[fin]).max() <= 1e-2


def test_ragged_prefill():
    """Algorithm 1 after a ragged eviction: a new aux thread appends its
    trigger tokens and prefills them over the packed context (the unused
    slots of partial pages are masked); a masked prefill of the main thread's
    tail with closed-cursor spans; queries that a partial page splits are
    refused."""
    P = 64
    p = Pair(2, 32, 8, 128, P, num_pages=600, seed=91)
    scale = 1.0 / math.sqrt(128)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 12000))
    spans = random_spans(seed=5, n_spans=12, total=4000, lo=P, hi=12000, median=300)
    p.evict(m, shuffled(spans, 1), ragged=True)
    a = p.fork(m)
    keep.append(p.append(a, 8))
    for layer in range(2):
        _prefill_check(p, a, layer, 8, [], 300 + layer, scale)
    keep.append(p.append(m, 300))
    n = p.cache.seq_info(m)[0]
    _prefill_check(p, m, 1, 300, [(100, 900), (n - 250, n - 240)], 400, scale)
    # queries from the first row of the last partial page on: its unused
    # slots would split them, so the call is refused
    fills = p.cache.page_fills(m)
    qs = max(q for q, f in enumerate(fills[:-1]) if f < P)
    n_q = n - sum(fills[:qs])
    q = torch.zeros(n_q, 32, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(n_q, 32, 128, dtype=torch.float32, device="cuda")
    with pytest.raises(sq.SqError) as e:
        p.cache.prefill_attention(m, 0, n_q, q, out, sq.SQ_OUT_F32, None, scale, [])
    assert e.value.code == sq.SQ_ERR_UNSUPPORTED
    # one row fewer starts on the next page: accepted
    _prefill_check(p, m, 0, n_q - fills[qs], [], 401, scale)
    p.close()


def test_decode_plan_survives_in_page_appends_after_ragged_eviction():
    """After a ragged eviction (partial pages before the last), one-token
    appends inside the last page keep the cached plan: the append kernel
    rewrites the last run's limit and the last page's fill in it.  An append
    that opens a page has the plan rebuilt; every output equals the oracle."""
    L, P = 2, 64
    p = Pair(L, 16, 4, 64, P, num_pages=300, seed=95, physical=True)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 14 * P + 20))
    p.evict(m, [(100, 150), (400, 420), (880, 900)], ragged=True)
    fills = p.cache.page_fills(m)
    assert min(fills[:-1]) < P                      # partial pages before the last
    st0 = p.cache.stats()
    rebuilds = 0
    for step in range(P + 4):                       # long enough to open a page
        f = p.cache.page_fills(m)
        if step == 0 or f[-1] == P:                 # first plan, or the append opens a page
            rebuilds += 1
        keep.append(p.append(m, 1))
        for layer in range(L):
            q_cpu, q = bf16_normal((1, 16, 64), 1500 + 7 * step + layer), None
            q = q_cpu.cuda()
            keep.append(q)
            out = p.decode([m], layer, 0.125, q, sq.SQ_OUT_F32)
            torch.cuda.synchronize()
            assert_budget(out, *p.oracle_decode_budget([m], layer, 0.125, q_cpu))
    st1 = p.cache.stats()
    assert st1["decode_plans_built"] - st0["decode_plans_built"] == rebuilds
    assert rebuilds >= 2
    p.check_tables()
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()
