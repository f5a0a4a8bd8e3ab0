"""Parity at the benchmark's full sizes, in the launch configuration bench.py
times (all decoding sequences of a step in one call, default persistent CTA
count): attention outputs on sampled sequences and layers against the oracle,
complete page tables, and sampled (layer, K/V, head) planes of the pool bit
for bit after eviction."""
import math

import numpy as np
import pytest
import torch

import paper_2602_22603_gb300 as sq
from oracle import attention as oatt
from synthetic import bf16_bits, bf16_normal, random_spans, request_spans, shuffled
from tests.bankfill import BankPair
from tests.budget import decode_budget
from tests.gpu_harness import assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _decode_and_check(bp, seqs, layer, scale, seed, sample):
    S = len(seqs)
    q_cpu = bf16_normal((S, bp.Hq, bp.D), seed)
    out = torch.empty(S, bp.Hq, bp.D, dtype=torch.float32, device="cuda")
    bp.cache.decode_attention(seqs, layer, q_cpu.cuda(), out, sq.SQ_OUT_F32, scale)
    torch.cuda.synchronize()
    assert bp.cache.sync_status() == sq.SQ_OK
    qb = bf16_bits(q_cpu)
    for i in (range(S) if sample is None else sample):
        K, V = bp.rows(seqs[i], layer)
        exp, dev, absv = oatt.decode_dev(qb[i], K, V, scale)
        assert_budget(out[i], exp, decode_budget(dev, absv, K.shape[0]))


def _check_request_planes(bp, h, r):
    """32 (layer, K/V, head) planes of a request: every plane of one layer,
    and four planes of each of four more layers."""
    rng = np.random.default_rng(1000 + r)
    full = (5 * r + 3) % bp.L
    bp.check_planes(h, full)
    others = [x for x in range(bp.L) if x != full]
    for layer in rng.choice(others, size=4, replace=False):
        picks = rng.choice(2 * bp.Hkv, size=4, replace=False)
        bp.check_planes(h, int(layer), [(int(x) // bp.Hkv, int(x) % bp.Hkv) for x in picks])


def test_serving_128k_full_size():
    """8 requests x 131,072 tokens + 8 forks (16 decoding sequences), 32
    layers, 32q/8kv, d128, P64; evict 20-65% per request in 10-40 spans."""
    L, Hq, Hkv, D, P = 32, 32, 8, 128, 64
    R, ctx = 8, 131072
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=R * (ctx // P + 4) + R * 4 + 64, seed=0)
    try:
        scale = 1.0 / math.sqrt(D)
        mains = []
        for r in range(R):
            m = bp.seq_new()
            bp.fill(m, ctx, 4096)
            mains.append(m)
        auxs = []
        for m in mains:
            a = bp.fork(m)
            bp.append(a, 8)
            auxs.append(a)
        seqs = [x for pair in zip(mains, auxs) for x in pair]
        for h in seqs:
            bp.append(h, 1)
        bp.check_tables(seqs)
        st = bp.cache.stats()
        assert st["live_pages"] == bp.oracle.live_pages()
        # every sequence at two layers
        for layer in (0, 31):
            _decode_and_check(bp, seqs, layer, scale, 100 + layer, None)
        # the shared prefix is read once per call
        st2 = bp.cache.stats()
        calls = st2["decode_calls"] - st["decode_calls"]
        uniq = (st2["decode_unique_bytes"] - st["decode_unique_bytes"]) / calls
        logi = (st2["decode_logical_bytes"] - st["decode_logical_bytes"]) / calls
        assert uniq < 0.51 * logi
        # Algorithm 1: release the aux threads, then evict
        for a in auxs:
            bp.release(a)
        for r, m in enumerate(mains):
            n = bp.cache.seq_info(m)[0]
            bp.evict(m, request_spans(0, r, n, P))
        bp.check_tables(mains)
        for r, m in enumerate(mains):
            _check_request_planes(bp, m, r)
        auxs = []
        for m in mains:
            a = bp.fork(m)
            bp.append(a, 8)
            auxs.append(a)
        seqs = [x for pair in zip(mains, auxs) for x in pair]
        for h in seqs:
            bp.append(h, 1)
        for layer in (5, 30):
            _decode_and_check(bp, seqs, layer, scale, 999 + layer, None)
        bp.check_tables(seqs)
    finally:
        bp.close()


def test_large_ragged_full_size():
    """64q/8kv (G = 8), d128, 80 layers, P64: requests of 32k, 96k, 192k and
    262,144 tokens, each with a fork; evict 50% of each in 25 spans — the
    32k one while its fork is alive (copy-on-write of every changed page)."""
    L, Hq, Hkv, D, P = 80, 64, 8, 128, 64
    ctxs = [32768, 98304, 196608, 262144]
    pages = sum(c // P for c in ctxs) + 4 * 8 + 64 + ctxs[0] // P  # + CoW room
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=pages, seed=3)
    try:
        scale = 1.0 / math.sqrt(D)
        mains = []
        for n in ctxs:
            m = bp.seq_new()
            bp.fill(m, n, 2048)
            mains.append(m)
        auxs = []
        for m in mains:
            a = bp.fork(m)
            bp.append(a, 8)
            auxs.append(a)
        seqs = [x for pair in zip(mains, auxs) for x in pair]
        for h in seqs:
            bp.append(h, 1)
        bp.check_tables(seqs)
        _decode_and_check(bp, seqs, 0, scale, 7, None)
        _decode_and_check(bp, seqs, 79, scale, 8, None)
        for r in range(1, 4):
            bp.release(auxs[r])
        for r, m in enumerate(mains):
            n = bp.cache.seq_info(m)[0]
            spans = shuffled(random_spans(500 + r, 25, n // 2, P, n, median=n / 50), r)
            bp.evict(m, spans)
        kept = [mains[0], auxs[0], mains[1], mains[2], mains[3]]
        bp.check_tables(kept)
        for r, h in enumerate(mains):
            _check_request_planes(bp, h, r)
        bp.check_planes(auxs[0], 40)
        for h in kept:
            bp.append(h, 1)
        _decode_and_check(bp, kept, 33, scale, 9, None)
    finally:
        bp.close()


def test_prefill_32k_full_size():
    """Masked prefill at the bench's size and launch configuration: one
    32,768-token context, 32 layers, 32q/8kv, d128, P64, 12 spans holding 40%
    of it masked, every token a query.  Sampled query rows (masked and
    unmasked positions, tile edges, the first and last) of two layers, with
    their log-sum-exp, against the oracle."""
    L, Hq, Hkv, D, P = 32, 32, 8, 128, 64
    n = 32768
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=n // P + 64, seed=4)
    try:
        m = bp.seq_new()
        bp.fill(m, n, 2048)
        spans = shuffled(random_spans(21, 12, int(0.4 * n), P, n, median=1500), 1)
        scale = 1.0 / math.sqrt(D)
        inside = spans[0][0] + 3
        for layer in (0, 31):
            q = bf16_normal((n, Hq, D), 400 + layer, device="cuda")
            out = torch.empty(n, Hq, D, dtype=torch.float32, device="cuda")
            lse = torch.empty(n, Hq, dtype=torch.float32, device="cuda")
            bp.cache.prefill_attention(m, layer, n, q, out, sq.SQ_OUT_F32, lse, scale, spans)
            torch.cuda.synchronize()
            assert bp.cache.sync_status() == sq.SQ_OK
            qb = bf16_bits(q.cpu())
            K, V = bp.rows(m, layer)
            for p in (0, 31, 32, 127, 128, 4095, inside, 20000, n - 129, n - 1):
                vis = [(a, min(b, p + 1)) for a, b in spans if a < p + 1]
                exp, exp_lse = oatt.prefill(qb[p:p + 1], K[:p + 1], V[:p + 1], scale, vis,
                                            want_lse=True)
                assert_close(out[p:p + 1], exp)
                got = lse[p].cpu().numpy().astype(np.float64)
                assert np.abs(got - exp_lse[0]).max() <= 1e-2, p
    finally:
        bp.close()


def test_aux_trigger_prefill_128k_full_size():
    """The aux thread's trigger prefill at the bench's size and launch
    configuration: a fork of a 131,072-token context (32q/8kv, d128, P64)
    appends 8 tokens and prefills them over all 131,080 keys (each KV head's
    key range split across the SMs, dual-key mode, split merge).  Every output
    row and log-sum-exp at two layers against the oracle, bf16 outputs too."""
    L, Hq, Hkv, D, P = 2, 32, 8, 128, 64
    n0, n_q = 131072, 8
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=n0 // P + 64, seed=5)
    try:
        m = bp.seq_new()
        bp.fill(m, n0, 4096)
        a = bp.fork(m)
        bp.append(a, n_q)
        scale = 1.0 / math.sqrt(D)
        for layer in (0, 1):
            q = bf16_normal((n_q, Hq, D), 500 + layer, device="cuda")
            out = torch.empty(n_q, Hq, D, dtype=torch.float32, device="cuda")
            out16 = torch.empty(n_q, Hq, D, dtype=torch.bfloat16, device="cuda")
            lse = torch.empty(n_q, Hq, dtype=torch.float32, device="cuda")
            bp.cache.prefill_attention(a, layer, n_q, q, out, sq.SQ_OUT_F32, lse, scale, [])
            bp.cache.prefill_attention(a, layer, n_q, q, out16, sq.SQ_OUT_BF16, None, scale, [])
            torch.cuda.synchronize()
            assert bp.cache.sync_status() == sq.SQ_OK
            K, V = bp.rows(a, layer)
            assert K.shape[0] == n0 + n_q
            exp, exp_lse = oatt.prefill(bf16_bits(q.cpu()), K, V, scale, [], want_lse=True)
            assert_close(out, exp)
            assert_close(out16, exp)
            assert np.abs(lse.cpu().numpy().astype(np.float64) - exp_lse).max() <= 1e-2
    finally:
        bp.close()


def test_serving_128k_ragged_eviction_full_size():
    """The serving workload's requests at full length (8 x 131,072 tokens,
    32q/8kv, d128, P64; two layers) evicted by ragged packing with the
    bench's spans (20-65% of each request in 10-40 spans): page tables and
    fills bit-exact, every plane of both layers of every request bit-exact,
    a few P rows copied per span, and decode of all 16 sequences (each request
    re-forked, Algorithm 1's next trigger) at both layers against the oracle."""
    L, Hq, Hkv, D, P = 2, 32, 8, 128, 64
    R, ctx = 8, 131072
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=R * (ctx // P + 4) + R * 4 + 64, seed=6)
    try:
        scale = 1.0 / math.sqrt(D)
        mains = []
        for r in range(R):
            m = bp.seq_new()
            bp.fill(m, ctx, 8192)
            mains.append(m)
        moved, spans_total = 0, 0
        for r, m in enumerate(mains):
            n = bp.cache.seq_info(m)[0]
            spans = request_spans(0, r, n, P)
            res = bp.evict(m, spans, ragged=True)
            assert res["moved_rows"] <= 2 * P * len(spans)
            moved += res["moved_rows"]
            spans_total += len(spans)
        st = bp.cache.stats()
        assert st["evict_moved_rows"] == moved
        bp.check_tables(mains)
        for m in mains:
            assert any(f < P for f in bp.cache.page_fills(m)[:-1])
            for layer in range(L):
                bp.check_planes(m, layer)
        auxs = []
        for m in mains:
            a = bp.fork(m)
            bp.append(a, 8)
            auxs.append(a)
        seqs = [x for pair in zip(mains, auxs) for x in pair]
        for h in seqs:
            bp.append(h, 1)
        bp.check_tables(seqs)
        for layer in range(L):
            _decode_and_check(bp, seqs, layer, scale, 700 + layer, None)
    finally:
        bp.close()


@pytest.mark.parametrize("L,D,ctx", [(32, 128, 16384), (80, 128, 8192), (32, 64, 16384)])
def test_eviction_ring_depths_many_planes(L, D, ctx):
    """Dense and ragged evictions with 32 and 80 layers of 8 KV heads (512 and
    1,280 (layer, K/V, head) planes: a cache on 152 SMs drives them with a
    ring of 3 and of 4 tiles; the small caches of the other tests use 6), at
    d = 128 (32-row tiles) and d = 64 (64-row tiles).  Two requests, each with
    a fork alive while its request is evicted (the changed shared pages are
    copied on write); page tables and fills bit-exact, every plane of three
    layers of every sequence bit-exact, then decode of all four sequences
    against the oracle."""
    Hq, Hkv, P = 32, 8, 64
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=4 * (ctx // P + 4) + 64, seed=L)
    try:
        mains, auxs = [], []
        for r in range(2):
            m = bp.seq_new()
            bp.fill(m, ctx, 1024)   # chunks that fit the bank at 80 layers
            mains.append(m)
            auxs.append(bp.fork(m))
        for r, m in enumerate(mains):
            spans = request_spans(L, r, ctx, P)
            bp.evict(m, spans, ragged=(r == 1))
        seqs = mains + auxs
        bp.check_tables(seqs)
        for h in seqs:
            for layer in (0, L // 2, L - 1):
                bp.check_planes(h, layer)
        for h in seqs:
            bp.append(h, 1)
        _decode_and_check(bp, seqs, L - 1, 1.0 / math.sqrt(D), 900 + L, None)
    finally:
        bp.close()


def test_d64_long_contexts_decode_evict_prefill():
    """The d = 64 kernels (a six-stage decode ring, the 64-column prefill
    tiles) at long contexts: 2 requests x 49,152 tokens + forks, G = 8, P = 64,
    every sequence decoded at two layers; request 0 loses 30% in 10 spans while
    its fork is alive (copy-on-write), tables and planes checked, decode again;
    then a masked prefill of its last 4,096 tokens at one layer, sampled rows
    with their log-sum-exp against the oracle."""
    L, Hq, Hkv, D, P = 4, 32, 4, 64, 64
    R, ctx = 2, 49152
    # the eviction with the fork alive copies most of a request's pages on write
    bp = BankPair(L, Hq, Hkv, D, P, num_pages=2 * R * (ctx // P + 4) + 256, seed=6)
    try:
        scale = 1.0 / math.sqrt(D)
        mains, auxs = [], []
        for r in range(R):
            m = bp.seq_new()
            bp.fill(m, ctx, 4096)
            mains.append(m)
            a = bp.fork(m)
            bp.append(a, 8)
            auxs.append(a)
        seqs = [x for pair in zip(mains, auxs) for x in pair]
        for layer in (0, L - 1):
            _decode_and_check(bp, seqs, layer, scale, 700 + layer, None)
        n = bp.cache.seq_info(mains[0])[0]
        spans = shuffled(random_spans(33, 10, int(0.3 * n), P, n, median=1200), 2)
        bp.evict(mains[0], spans)                   # the fork still holds the old pages
        bp.check_tables(seqs)
        bp.check_planes(mains[0], 1)
        bp.check_planes(auxs[0], 2)
        for h in seqs:
            bp.append(h, 1)
        for layer in (1, 2):
            _decode_and_check(bp, seqs, layer, scale, 800 + layer, None)
        # masked prefill of request 1's last 4,096 tokens
        m = mains[1]
        n = bp.cache.seq_info(m)[0]
        n_q = 4096
        pspans = shuffled(random_spans(34, 6, 6000, P, n - n_q, median=900), 3)
        q = bf16_normal((n_q, Hq, D), 900, device="cuda")
        out = torch.empty(n_q, Hq, D, dtype=torch.float32, device="cuda")
        lse = torch.empty(n_q, Hq, dtype=torch.float32, device="cuda")
        bp.cache.prefill_attention(m, 3, n_q, q, out, sq.SQ_OUT_F32, lse, scale, pspans)
        torch.cuda.synchronize()
        assert bp.cache.sync_status() == sq.SQ_OK
        qb = bf16_bits(q.cpu())
        K, V = bp.rows(m, 3)
        for i in (0, 1, 7, 8, 63, 64, 2047, n_q - 9, n_q - 1):
            p = n - n_q + i
            vis = [(a, min(b, p + 1)) for a, b in pspans if a < p + 1]
            exp, exp_lse = oatt.prefill(qb[i:i + 1], K[:p + 1], V[:p + 1], scale, vis,
                                        want_lse=True)
            assert_close(out[i:i + 1], exp)
            got = lse[i].cpu().numpy().astype(np.float64)
            assert np.abs(got - exp_lse[0]).max() <= 1e-2, i
    finally:
        bp.close()
