"""Masked prefill attention (Algorithm 2, BuildMask) on the GPU against the
oracle: every output row and log-sum-exp at small sizes that still span
several query and key tiles with ragged tails, across GQA groups, head dims,
page sizes, span layouts (including a masked prefix and masked queries), the
split-key path for short query blocks, forked sequences and evicted ones."""
import math

import numpy as np
import pytest
import torch

import paper_2602_22603_gb300 as sq
from oracle import attention as oatt
from synthetic import bf16_bits, bf16_normal, random_spans
from tests.budget import decode_budget
from tests.gpu_harness import Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu

LSE_ABS = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def run_prefill(p: Pair, h, layer, n_q, spans, seed, scale, out_dtype=sq.SQ_OUT_F32):
    q_cpu = bf16_normal((n_q, p.Hq, p.D), seed)
    dt = torch.float32 if out_dtype == sq.SQ_OUT_F32 else torch.bfloat16
    out = torch.full((n_q, p.Hq, p.D), float("nan"), dtype=dt, device="cuda")
    lse = torch.full((n_q, p.Hq), float("nan"), dtype=torch.float32, device="cuda")
    p.cache.prefill_attention(h, layer, n_q, q_cpu.cuda(), out, out_dtype, lse, scale, spans)
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    return q_cpu, out, lse


def oracle_prefill(p: Pair, h, layer, q_cpu, spans, scale):
    k, v = p.store.rows(p.oracle.tokens(p.o[h]), layer)
    return oatt.prefill(bf16_bits(q_cpu), k, v, scale, spans, want_lse=True)


def check_budget_rows(p: Pair, h, layer, q_cpu, out, spans, scale, rows):
    """Element by element within the error budget of the bf16 softmax weights
    (tests/budget.py): the normaliser sums the same rounded weights the PV
    product takes, so each output row is a convex combination of V rows, as in
    decode.  Query row r at position n - n_q + r is decode over the keys it
    sees; rows that see no key are left to the exact check."""
    k, v = p.store.rows(p.oracle.tokens(p.o[h]), layer)
    n, n_q = k.shape[0], q_cpu.shape[0]
    qb = bf16_bits(q_cpu)
    got = out.detach().float().cpu()
    for r in rows:
        pos = n - n_q + r
        mask = oatt.removed_mask(pos + 1, spans)
        if mask.all():
            continue
        exp, dev, absv = oatt.decode_dev(qb[r], k[:pos + 1], v[:pos + 1], scale, mask)
        assert_budget(got[r], exp, decode_budget(dev, absv, pos + 1))


def check(p, h, layer, n_q, spans, seed, scale=None, out_dtype=sq.SQ_OUT_F32):
    scale = scale if scale is not None else 1.0 / math.sqrt(p.D)
    q_cpu, out, lse = run_prefill(p, h, layer, n_q, spans, seed, scale, out_dtype)
    exp, exp_lse = oracle_prefill(p, h, layer, q_cpu, spans, scale)
    assert_close(out, exp)
    if out_dtype == sq.SQ_OUT_F32:
        rows = sorted(set(np.linspace(0, n_q - 1, min(n_q, 40)).round().astype(int).tolist()))
        check_budget_rows(p, h, layer, q_cpu, out, spans, scale, rows)
    got_lse = lse.cpu().numpy().astype(np.float64)
    fin = np.isfinite(exp_lse)
    assert np.array_equal(np.isfinite(got_lse), fin)
    if fin.any():
        assert np.abs(got_lse[fin] - exp_lse[fin]).max() <= LSE_ABS
    return out, lse


def spans_for(n, k, seed):
    if n < 4 or k == 0:
        return []
    total = max(k, n // 3)
    return random_spans(seed, k, total, 0, n, median=max(1.0, total / k))


@pytest.mark.parametrize("Hq,Hkv,D,P", [
    (16, 4, 64, 16),    # G = 4, the tiny shape
    (32, 8, 128, 64),   # G = 4, d = 128, the 8B-class shape
    (8, 8, 64, 8),      # G = 1: textbook MHA, 8-token pages
    (6, 2, 128, 256),   # G = 3: padded query tiles, 256-token pages
    (32, 2, 64, 32),    # G = 16: 8 positions per query tile
])
@pytest.mark.parametrize("n,n_q,k", [(1, 1, 0), (129, 129, 2), (300, 37, 3), (517, 517, 5)])
def test_prefill_matches_oracle(Hq, Hkv, D, P, n, n_q, k):
    p = Pair(2, Hq, Hkv, D, P, num_pages=(n + P - 1) // P + 8, seed=n + Hq)
    try:
        h = p.seq_new()
        p.append(h, n)
        spans = spans_for(n, k, n * 3 + k)
        check(p, h, 1, n_q, spans, seed=n + 7)
    finally:
        p.close()


def test_prefill_bf16_output_and_long_ragged_sequence():
    p = Pair(1, 32, 8, 128, 64, num_pages=40, seed=5)
    try:
        h = p.seq_new()
        for chunk in (700, 1, 1000, 333):   # several appends, a ragged last page
            p.append(h, chunk)
        n = 2034
        spans = random_spans(9, 6, 800, 64, n, median=130)
        check(p, h, 0, n, spans, seed=11)
        # bf16 outputs of the queries that average hundreds of rows (|o| << 1);
        # an early query's output is a mean of a few N(0,1) rows, |o| up to
        # ~3, where one bf16 rounding alone is worth up to 2^-7
        check(p, h, 0, 1024, spans, seed=12, out_dtype=sq.SQ_OUT_BF16)
    finally:
        p.close()


def test_prefill_split_key_ranges():
    # 8 query positions over 3000 keys: one query tile per KV head, so the key
    # range is split across CTAs and merged by the combine kernel.
    p = Pair(1, 32, 8, 128, 64, num_pages=60, seed=6)
    try:
        h = p.seq_new()
        p.append(h, 3000)
        spans = random_spans(4, 10, 1200, 0, 3000, median=120)
        check(p, h, 0, 8, spans, seed=3)
        check(p, h, 0, 8, [], seed=4, out_dtype=sq.SQ_OUT_BF16)
    finally:
        p.close()


@pytest.mark.parametrize("Hq,Hkv,D,P,n,n_q,scale", [
    (32, 8, 128, 64, 1100, 1100, 0.35),   # maxima grow a few powers of two: kept, weights > 1
    (32, 8, 128, 64, 1100, 1100, 1.0),    # grow by ~10: some tiles redone with a raised maximum
    (32, 8, 128, 64, 1100, 1100, 4.0),    # grow far past 2^16: raised on most tiles
    (16, 4, 64, 16, 700, 700, 1.5),       # d = 64
    (32, 8, 128, 64, 3000, 8, 4.0),       # short block: dual-key halves and split key ranges
])
def test_prefill_running_maximum_under_growing_logits(Hq, Hkv, D, P, n, n_q, scale):
    # Large softmax scales make each row's maximum grow from key tile to key
    # tile.  A tile's weights are kept with the old maximum while every row's
    # sum of them stays at most 2^16; past that the tile is redone with the
    # raised maximum and O rescaled.  Both, and the mix of rows in one warp
    # taking either, must give the softmax over all visible keys.
    p = Pair(1, Hq, Hkv, D, P, num_pages=(n + P - 1) // P + 8, seed=n + 5)
    try:
        h = p.seq_new()
        p.append(h, n)
        check(p, h, 0, n_q, spans_for(n, 3, n + 1), seed=n + 2, scale=scale)
    finally:
        p.close()


def test_prefill_masked_prefix_gives_empty_rows():
    # spans covering [0, 200): the first 200 queries see nothing (zeros,
    # -inf), later ones see only the unmasked suffix
    p = Pair(1, 16, 4, 64, 16, num_pages=40, seed=8)
    try:
        h = p.seq_new()
        p.append(h, 400)
        out, lse = check(p, h, 0, 400, [(0, 150), (150, 200)], seed=1)
        assert not out[:200].any()
        assert torch.isinf(lse[:200]).all() and (lse[:200] < 0).all()
        # only the last token visible: the last query sees itself, the rest nothing
        out, _ = check(p, h, 0, 400, [(0, 399)], seed=2)
    finally:
        p.close()


def test_prefill_on_fork_and_after_eviction():
    # the aux thread's prefill reads the shared pages; after the main thread
    # evicts, the aux keeps its view and the main thread's masked prefill over
    # the evicted context equals decode over it
    p = Pair(2, 32, 8, 128, 64, num_pages=80, seed=9)
    try:
        m = p.seq_new()
        p.append(m, 1500)
        a = p.fork(m)
        p.append(a, 24)                       # trigger + aux tokens
        check(p, a, 1, 24, [], seed=5)        # aux prefill over the shared context
        spans = [(100, 400), (700, 710), (900, 1300)]
        p.evict(m, spans)
        p.append(m, 1)
        check(p, a, 1, 24, [(64, 128)], seed=6)
        n = p.cache.seq_info(m)[0]
        q_cpu, out, _ = run_prefill(p, m, 0, 1, [], 7, 0.088)
        dec = p.decode([m], 0, 0.088, q_cpu.cuda())
        torch.cuda.synchronize()
        assert (out[0] - dec[0]).abs().max().item() < 2e-3
        exp = p.oracle_decode([m], 0, 0.088, q_cpu)
        assert_close(out, exp)
        assert n == 1500 - 710 + 1
    finally:
        p.close()


def test_prefill_masked_equals_evicted():
    # Algorithm 2 (mask) vs Algorithm 1 (evict): the masked prefill's last
    # query over the full context equals prefill's last query after the spans
    # are evicted, both on the GPU.
    p = Pair(1, 16, 4, 64, 16, num_pages=80, seed=10)
    try:
        m = p.seq_new()
        p.append(m, 900)
        spans = [(17, 90), (300, 301), (500, 870)]
        q_cpu = bf16_normal((1, 16, 64), 77)
        out_mask = torch.empty(1, 16, 64, dtype=torch.float32, device="cuda")
        p.cache.prefill_attention(m, 0, 1, q_cpu.cuda(), out_mask, sq.SQ_OUT_F32, None, 0.125, spans)
        p.evict(m, spans)
        out_evict = torch.empty_like(out_mask)
        p.cache.prefill_attention(m, 0, 1, q_cpu.cuda(), out_evict, sq.SQ_OUT_F32, None, 0.125, [])
        torch.cuda.synchronize()
        assert (out_mask - out_evict).abs().max().item() < 2e-3
    finally:
        p.close()


def test_prefill_rejects_bad_arguments():
    p = Pair(1, 16, 4, 64, 16, num_pages=20, seed=11)
    try:
        h = p.seq_new()
        p.append(h, 100)
        q = torch.zeros(10, 16, 64, dtype=torch.bfloat16, device="cuda")
        out = torch.zeros(10, 16, 64, dtype=torch.float32, device="cuda")
        c = p.cache
        bad = [
            dict(n_q=101), dict(n_q=0), dict(layer=1), dict(spans=[(5, 5)]),
            dict(spans=[(5, 9), (8, 12)]), dict(spans=[(90, 101)]), dict(sm_scale=-1.0),
            dict(sm_scale=float("nan")), dict(out_dtype=7),
            dict(out=q.view(torch.float32)[:5]),             # out overlaps q
            dict(lse=out.view(-1)[:160]),                     # lse overlaps out
        ]
        for kw in bad:
            args = dict(seq=h, layer=0, n_q=10, q=q, out=out, out_dtype=sq.SQ_OUT_F32,
                        lse=None, sm_scale=0.1, spans=[])
            args.update(kw)
            with pytest.raises(sq.SqError) as ei:
                c.prefill_attention(**args)
            assert ei.value.code == sq.SQ_ERR_INVALID_ARG, kw
        with pytest.raises(sq.SqError) as ei:
            c.prefill_attention(123456789, 0, 10, q, out, sq.SQ_OUT_F32, None, 0.1, [])
        assert ei.value.code == sq.SQ_ERR_BAD_HANDLE
        torch.cuda.synchronize()
        assert c.sync_status() == sq.SQ_OK
    finally:
        p.close()


@pytest.mark.parametrize("n,n_q,spans", [
    (5 * 128 + 3, 5, [(10, 200)]),             # 6 key tiles: the two halves take 3 + 3
    (7 * 128 + 1, 3, [(0, 600)]),              # 8 key tiles; rows see keys only past 600
    (4 * 128, 8, [(0, 130), (260, 384)]),      # keys only in tiles 1 and 3 (one half)
    (3 * 128 + 64, 1, []),                     # 4 key tiles, one query
])
def test_prefill_short_block_dual_key_split(n, n_q, spans):
    # All queries of a CTA tile fit in its first query tile, so the second takes
    # every other key tile and the two partial results are merged per row.
    p = Pair(1, 32, 8, 128, 64, num_pages=n // 64 + 4, seed=n_q + 40)
    try:
        h = p.seq_new()
        p.append(h, n)
        check(p, h, 0, n_q, spans, seed=n + 1)
        check(p, h, 0, n_q, spans, seed=n + 2, out_dtype=sq.SQ_OUT_BF16)
    finally:
        p.close()


def test_prefill_plan_reuse_follows_sequence_changes():
    # a plan is reused across layers while the sequence, the query count and
    # the spans are unchanged; every change (append, n_q, spans, eviction, a
    # fork's copy-on-write) gives a new one, and more distinct plans than the
    # cache holds cycle through it
    p = Pair(2, 16, 4, 64, 16, num_pages=120, seed=12)
    try:
        h = p.seq_new()
        p.append(h, 700)
        s1, s2 = [(40, 90), (300, 420)], [(0, 10), (500, 650)]
        check(p, h, 0, 100, s1, seed=1)
        check(p, h, 1, 100, s1, seed=2)
        p.append(h, 50)
        check(p, h, 0, 100, s1, seed=3)
        check(p, h, 0, 120, s1, seed=4)
        check(p, h, 1, 120, s2, seed=5)
        p.evict(h, [(200, 260)])
        check(p, h, 0, 80, [], seed=6)
        a = p.fork(h)
        p.append(a, 10)
        for layer in (0, 1):
            check(p, a, layer, 30, [(5, 25)], seed=7 + layer)
            check(p, h, layer, 30, [(5, 25)], seed=9 + layer)
        for rep in range(2):
            for n_q in (1, 7, 33, 64, 65, 129):
                check(p, h, rep, n_q, s2, seed=20 + n_q)
    finally:
        p.close()
