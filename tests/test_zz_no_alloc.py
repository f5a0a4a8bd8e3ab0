"""sq_decode_attention_noalloc: decode attention for callers that may not
allocate GPU memory while decoding (runtimes that reserve the device for their
KV pool up front, or hosts whose allocator C code cannot reach).  Its result
must equal the regular entry point's, call after call, although every call
reuses the same fixed library scratch.

Collected last on purpose (file name), so a run that stops at the first
failure has already run every other test; it also passes on its own."""
import ctypes
import math

import pytest
import torch

import paper_2602_22603_gb300 as sq
from synthetic import bf16_normal
from tests.gpu_harness import MAX_ABS, MEAN_ABS, Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _noalloc_c(cache, seqs, layer, q, out, out_dtype, scale):
    """Direct C-ABI call; returns the status code."""
    arr = (ctypes.c_int32 * len(seqs))(*seqs)
    return sq.lib().sq_decode_attention_noalloc(
        cache.handle, arr, len(seqs), layer, q.data_ptr(), out.data_ptr(), out_dtype,
        ctypes.c_float(scale), torch.cuda.current_stream().cuda_stream)


def test_noalloc_matches_regular_entry_point_two_calls_in_a_row():
    p = Pair(2, 32, 8, 128, 64, num_pages=1200, seed=41)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 20000))
    a = p.fork(m)
    keep.append(p.append(a, 8))
    keep.append(p.append(m, 37))
    lone = p.seq_new()
    keep.append(p.append(lone, 333))
    seqs = [m, a, lone]
    scale = 1.0 / math.sqrt(128)
    torch.cuda.synchronize()
    for call in range(2):
        layer = call % 2
        q_cpu = bf16_normal((3, 32, 128), 7 + call)
        q = q_cpu.cuda()
        outs = {}
        for dt, tdt in ((sq.SQ_OUT_F32, torch.float32), (sq.SQ_OUT_BF16, torch.bfloat16)):
            ref = torch.empty(3, 32, 128, dtype=tdt, device="cuda")
            got = torch.full((3, 32, 128), float("nan"), dtype=tdt, device="cuda")
            p.cache.decode_attention(seqs, layer, q, ref, dt, scale)
            torch.cuda.synchronize()
            # the free device memory the driver reports does not move across
            # the allocation-free call (the scratch was made resident when
            # the cache was created)
            free0 = torch.cuda.mem_get_info()[0]
            assert _noalloc_c(p.cache, seqs, layer, q, got, dt, scale) == sq.SQ_OK
            torch.cuda.synchronize()
            assert torch.cuda.mem_get_info()[0] == free0
            assert p.cache.sync_status() == sq.SQ_OK
            assert_close(got, ref.double().cpu().numpy(), MAX_ABS, MEAN_ABS)
            assert torch.equal(got, ref)   # same plan, same kernels
            outs[dt] = got
        exp, budget = p.oracle_decode_budget(seqs, layer, scale, q_cpu)
        assert_budget(outs[sq.SQ_OUT_F32], exp, budget)
        assert_close(outs[sq.SQ_OUT_BF16], exp)
        keep.append(p.append(m, 1))        # the next call sees a changed sequence
    p.close()


def test_decode_rejects_output_over_queries():
    # the merged rows of a call are written while other CTAs still read their
    # queries, so both entry points refuse an output that overlaps q
    p = Pair(1, 16, 4, 64, 16, num_pages=40, seed=45)
    keep = [None]
    m = p.seq_new()
    keep.append(p.append(m, 300))
    buf = torch.zeros(4096, dtype=torch.float32, device="cuda")     # 16 KiB
    q = buf.view(torch.bfloat16)[:1024].view(1, 16, 64)               # bytes [0, 2048)
    arr = (ctypes.c_int32 * 1)(m)
    bad = [
        (buf[256:256 + 1024].view(1, 16, 64), sq.SQ_OUT_F32),        # fp32 out from byte 1024
        (q, sq.SQ_OUT_BF16),                                           # in place
    ]
    for out, dt in bad:
        rc = sq.lib().sq_decode_attention(p.cache.handle, arr, 1, 0, q.data_ptr(), out.data_ptr(),
                                          dt, ctypes.c_float(0.1),
                                          torch.cuda.current_stream().cuda_stream)
        assert rc == sq.SQ_ERR_INVALID_ARG
        assert _noalloc_c(p.cache, [m], 0, q, out, dt, 0.1) == sq.SQ_ERR_INVALID_ARG
    # adjacent (the output starts at q's end): accepted
    out = buf[512:512 + 1024].view(1, 16, 64)
    assert _noalloc_c(p.cache, [m], 0, q, out, sq.SQ_OUT_F32, 0.1) == sq.SQ_OK
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


def test_noalloc_rejects_plans_beyond_the_scratch():
    # 8 KV heads x 2048 stages over 16384 persistent CTAs -> about 16,390
    # partial entries of G = 8 rows (8 x (128 + 4) floats each): ~69 MB of
    # partials plus ~1.4 MB of plan, twice what the fixed scratch holds
    n = 131072
    c = sq.Cache(1, 64, 8, 128, 64, n // 64 + 4, max_seqs=4, decode_ctas=16384)
    try:
        m = c.seq_new()
        kv = torch.zeros(1, 4096, 8, 128, dtype=torch.bfloat16, device="cuda")
        for _ in range(n // 4096):
            c.append_kv(m, 4096, kv, kv)
        q = bf16_normal((1, 64, 128), 1).cuda()
        out = torch.zeros(1, 64, 128, device="cuda")
        assert _noalloc_c(c, [m], 0, q, out, sq.SQ_OUT_F32, 0.1) == sq.SQ_ERR_CAPACITY
        torch.cuda.synchronize()
        assert torch.count_nonzero(out).item() == 0     # nothing was enqueued
        assert c.sync_status() == sq.SQ_OK
    finally:
        c.close()
