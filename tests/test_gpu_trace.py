"""End-to-end GPU parity of the Algorithm 1 loop at a small scale: every
library call of the hot path interleaved as an agent runs them, with the
oracle in lockstep.

Two agents, eight turns (32q/8kv, d128, P64, 2 layers).  A turn: (1) when
the aux thread has finished, release it and evict the tool responses older
than two turns (alternately by dense and by ragged packing); (2) every other
turn fork an aux thread, append its 8-token trigger and prefill the trigger
over the whole context (Algorithm 1 phase 2, Sec. 3.2); (3) three decode
steps: one batched append of a new row for every decoding sequence, then
attention at each layer; (4) append a tool response.  Page tables, fills,
counts and contents match the oracle bit for bit after every turn; decode
within the error budget, prefill within the contract's tolerance."""
import math

import numpy as np
import pytest
import torch

import paper_2602_22603_gb300 as sq
from oracle import attention as oatt
from synthetic import bf16_bits, bf16_normal
from tests.gpu_harness import Pair, assert_budget, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2602_22603_gb300 import build
    build.build_libsq()
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_agent_loop_two_agents_eight_turns():
    L, Hq, Hkv, D, P = 2, 32, 8, 128, 64
    p = Pair(L, Hq, Hkv, D, P, num_pages=3000, seed=123, physical=True)
    scale = 1.0 / math.sqrt(D)
    rng = np.random.default_rng(7)
    keep = []
    mains = []
    for _ in range(2):
        m = p.seq_new()
        keep.append(p.append(m, 300))             # the user query Q
        mains.append(m)
    responses = [[] for _ in mains]               # (turn, start, end), current positions
    auxs = []
    qseed = 1000
    evictions = 0
    for turn in range(8):
        # (1) aux finished: release, then evict the responses older than two turns
        if auxs:
            for a in auxs:
                p.release(a)
            auxs = []
            for i, m in enumerate(mains):
                old = [r for r in responses[i] if r[0] < turn - 2]
                if not old:
                    continue
                spans = [(s, e) for _, s, e in old]
                p.evict(m, spans, ragged=evictions % 2 == 1)
                evictions += 1
                gone = sorted(spans)
                kept = []
                for r in responses[i]:
                    if r in old:
                        continue
                    shift = sum(e - s for s, e in gone if e <= r[1])
                    kept.append((r[0], r[1] - shift, r[2] - shift))
                responses[i] = kept
        # (2) every other turn: fork an aux thread, append and prefill its trigger
        if turn % 2 == 0:
            for m in mains:
                a = p.fork(m)
                keep.append(p.append(a, 8))
                auxs.append(a)
                layer = turn % L
                q_cpu = bf16_normal((8, Hq, D), qseed)
                qseed += 1
                out = torch.empty(8, Hq, D, dtype=torch.float32, device="cuda")
                p.cache.prefill_attention(a, layer, 8, q_cpu.cuda(), out, sq.SQ_OUT_F32, None, scale, [])
                torch.cuda.synchronize()
                k, v = p.store.rows(p.oracle.tokens(p.o[a]), layer)
                assert_close(out, oatt.prefill(bf16_bits(q_cpu), k, v, scale, []))
        # (3) decode steps over every decoding sequence
        seqs = mains + auxs
        for step in range(3):
            keep.append(p.append_batch(seqs))
            for layer in range(L):
                q_cpu = bf16_normal((len(seqs), Hq, D), qseed)
                qseed += 1
                out = p.decode(seqs, layer, scale, q_cpu.cuda(), sq.SQ_OUT_F32)
                torch.cuda.synchronize()
                assert_budget(out, *p.oracle_decode_budget(seqs, layer, scale, q_cpu))
        # (4) the tool response
        for i, m in enumerate(mains):
            n = p.cache.seq_info(m)[0]
            k = int(rng.integers(40, 700))
            keep.append(p.append(m, k))
            responses[i].append((turn, n, n + k))
        p.check_tables()
        for h in mains + auxs:
            p.check_contents(h)
        p.check_zero_slots()
    assert evictions >= 4
    assert p.cache.sync_status() == sq.SQ_OK
    p.close()
