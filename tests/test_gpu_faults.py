"""Failure detection on the GPU without a fault: a bounded wait runs out.

The test hook makes one persistent CTA of the next decode call leave its
first pipeline stage unsignalled, so its consumer warps wait on a barrier
that nothing completes.  The wait gives up after ~2 s; the kernel winds down
(no trap, no fault); the host reads SQ_ERR_DEVICE_TIMEOUT; the cache and the
CUDA context keep working."""
import math
import time

import pytest
import torch

import paper_2602_22603_gb300 as sq
from synthetic import bf16_normal
from tests.gpu_harness import Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_unsignalled_stage_times_out_and_context_survives():
    p = Pair(1, 8, 2, 64, 16, num_pages=600, seed=9)
    keep = []
    m = p.seq_new()
    keep.append(p.append(m, 3000))
    a = p.fork(m)
    keep.append(p.append(a, 20))
    q_cpu = bf16_normal((2, 8, 64), 1)
    q = q_cpu.cuda()
    out = torch.empty(2, 8, 64, device="cuda")
    assert p.cache.sync_status() == sq.SQ_OK
    sq.sq_debug_set(p.cache.handle, sq.SQ_DEBUG_DROP_DECODE_STAGE)
    t0 = time.monotonic()
    p.cache.decode_attention([m, a], 0, q, out, sq.SQ_OUT_F32, 0.125)
    rc = p.cache.sync_status()
    dt = time.monotonic() - t0
    assert rc == sq.SQ_ERR_DEVICE_TIMEOUT
    assert 1.0 < dt < 60.0
    # the status was cleared, the hook too; the same call now succeeds
    out2 = p.decode([m, a], 0, 0.125, q, sq.SQ_OUT_F32)
    torch.cuda.synchronize()
    assert p.cache.sync_status() == sq.SQ_OK
    assert_budget(out2, *p.oracle_decode_budget([m, a], 0, 0.125, q_cpu))
    # and so do appends and evictions
    keep.append(p.append(m, 5))
    p.evict(m, [(100, 400)])
    p.check_tables()
    p.check_contents(m)
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()


def test_debug_flags_are_validated():
    c = sq.Cache(1, 4, 1, 64, 16, 10)
    with pytest.raises(sq.SqError) as e:
        sq.sq_debug_set(c.handle, 1 << 5)
    assert e.value.code == sq.SQ_ERR_INVALID_ARG
    sq.sq_debug_set(c.handle, 0)
    c.close()
