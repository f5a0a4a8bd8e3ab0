"""Drives the CUDA library and the CPU oracle side by side on the same seeded
inputs, and compares them: page tables and KV contents bit for bit, decode
attention within the stated tolerance."""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

import paper_2602_22603_gb300 as sq
from oracle import attention as oatt
from oracle import cache_model as ocm
from synthetic import bf16_bits, bf16_normal
from tests.budget import decode_budget

# Attention tolerance against the double-precision oracle (max / mean abs).
MAX_ABS = 1e-2
MEAN_ABS = 1e-3


class RowStore:
    """Contents of every appended token row: token id -> [L, 2, Hkv, D]
    bf16 bits, for small workloads."""

    def __init__(self, L, Hkv, D):
        self.L, self.Hkv, self.D = L, Hkv, D
        self.k: List[np.ndarray] = []   # chunks [n, L, Hkv, D]
        self.v: List[np.ndarray] = []
        self.first: List[int] = []

    def add(self, first_id: int, k_bits: np.ndarray, v_bits: np.ndarray):
        # k_bits: [L, n, Hkv, D] -> stored token-major
        self.first.append(first_id)
        self.k.append(np.ascontiguousarray(k_bits.transpose(1, 0, 2, 3)))
        self.v.append(np.ascontiguousarray(v_bits.transpose(1, 0, 2, 3)))

    def _cat(self):
        if not hasattr(self, "_kk") or self._kk.shape[0] != sum(x.shape[0] for x in self.k):
            self._kk = np.concatenate(self.k, axis=0)
            self._vv = np.concatenate(self.v, axis=0)
        return self._kk, self._vv

    def rows(self, token_ids: Sequence[int], layer: int):
        """K, V bits [n, Hkv, D] of the given tokens at one layer."""
        kk, vv = self._cat()
        ids = np.asarray(token_ids, dtype=np.int64)
        return kk[ids, layer], vv[ids, layer]


class Pair:
    """One library cache and one oracle cache, kept in lockstep."""

    def __init__(self, L, Hq, Hkv, D, P, num_pages, max_seqs=64, decode_ctas=0, seed=0,
                 k_scale=1.0, physical=False):
        self.L, self.Hq, self.Hkv, self.D, self.P = L, Hq, Hkv, D, P
        self.cache = sq.Cache(L, Hq, Hkv, D, P, num_pages, max_seqs=max_seqs,
                              decode_ctas=decode_ctas)
        self.oracle = ocm.OracleCache(num_pages, P, physical=physical)
        self.store = RowStore(L, Hkv, D)
        self.o: Dict[int, int] = {}     # library handle -> oracle sequence id
        self.seed = seed
        self.k_scale = k_scale
        self._draws = 0

    def close(self):
        self.cache.close()

    def _next_seed(self):
        self._draws += 1
        return self.seed * 100003 + self._draws

    def seq_new(self) -> int:
        h = self.cache.seq_new()
        self.o[h] = self.oracle.seq_new()
        return h

    def fork(self, parent: int) -> int:
        h = self.cache.fork_aux(parent)
        self.o[h] = self.oracle.fork(self.o[parent])
        return h

    def append(self, h: int, n: int, stream=None):
        if n == 0:
            return None
        s = self._next_seed()
        k = bf16_normal((self.L, n, self.Hkv, self.D), s, scale=self.k_scale)
        v = bf16_normal((self.L, n, self.Hkv, self.D), s + 50000)
        ids = self.oracle.append(self.o[h], n)
        self.store.add(ids[0], bf16_bits(k), bf16_bits(v))
        kd, vd = k.cuda(), v.cuda()
        self.cache.append_kv(h, n, kd, vd, stream)
        return kd, vd  # keep alive until the stream has run

    def append_batch(self, hs, stream=None):
        """One new token for each sequence of hs, in one library call."""
        S = len(hs)
        s = self._next_seed()
        k = bf16_normal((self.L, S, self.Hkv, self.D), s, scale=self.k_scale)
        v = bf16_normal((self.L, S, self.Hkv, self.D), s + 50000)
        ids = [self.oracle.append(self.o[h], 1)[0] for h in hs]
        assert ids == list(range(ids[0], ids[0] + S))
        self.store.add(ids[0], bf16_bits(k), bf16_bits(v))
        kd, vd = k.cuda(), v.cuda()
        self.cache.append_kv_batch(list(hs), kd, vd, stream)
        return kd, vd

    def evict(self, h: int, spans, stream=None, ragged=False):
        r = self.oracle.evict(self.o[h], spans, mode="ragged" if ragged else "dense")
        if ragged:
            self.cache.evict_spans_ragged(h, spans, stream)
        else:
            self.cache.evict_spans(h, spans, stream)
        return r

    def release(self, h: int, stream=None):
        self.cache.release(h, stream)
        self.oracle.release(self.o.pop(h))

    # ---- checks --------------------------------------------------------------
    def check_tables(self):
        for h, o in self.o.items():
            assert self.cache.page_table(h) == self.oracle.page_table(o)
            assert self.cache.page_fills(h) == self.oracle.page_fills(o)
            assert self.cache.seq_info(h)[0] == self.oracle.n_tokens(o)
        assert self.cache.free_pages() == self.oracle.free_count()
        for p in range(self.oracle.num_pages):
            assert self.cache.page_refcount(p) == self.oracle.ref[p], p

    def check_contents(self, h: int, layers: Optional[Sequence[int]] = None):
        """Every valid row of the sequence, read from the device pool through
        the library's page table, equals the row the oracle says is there."""
        torch.cuda.synchronize()
        pool = self.cache.pool_view()
        page, slot = row_slots(self.cache, h)
        toks = self.oracle.tokens(self.o[h])
        for layer in (layers if layers is not None else range(self.L)):
            for kv in (0, 1):
                got = pool[layer, page, kv, :, slot, :]           # [n, Hkv, D]
                got = bf16_bits(got.cpu())
                ek, ev = self.store.rows(toks, layer)
                exp = ek if kv == 0 else ev
                assert np.array_equal(got, exp), f"layer {layer} kv {kv}"

    def check_zero_slots(self):
        """Every slot the (physical) oracle says was set to zero holds zero
        bits in the device pool, in every layer, K and V, and head."""
        torch.cuda.synchronize()
        pool = self.cache.pool_view()
        for p, slots in self.oracle.phys.items():
            z = [t for t, x in enumerate(slots) if x == ocm.ZERO]
            if z:
                got = pool[:, p, :, :, z, :]
                assert not torch.any(got.view(torch.int16) != 0).item(), (p, z)

    def decode(self, seqs: Sequence[int], layer: int, sm_scale: float, q: torch.Tensor,
               out_dtype=sq.SQ_OUT_F32, stream=None) -> torch.Tensor:
        S = len(seqs)
        dt = torch.float32 if out_dtype == sq.SQ_OUT_F32 else torch.bfloat16
        out = torch.empty(S, self.Hq, self.D, dtype=dt, device="cuda")
        self.cache.decode_attention(list(seqs), layer, q, out, out_dtype, sm_scale, stream)
        return out

    def oracle_decode_budget(self, seqs: Sequence[int], layer: int, sm_scale: float,
                             q_cpu) -> Tuple[np.ndarray, np.ndarray]:
        """The oracle's outputs [S, Hq, D] and the kernel's per-element error
        budget for them (tests/budget.py)."""
        qb = bf16_bits(q_cpu)
        res, bud = [], []
        for i, h in enumerate(seqs):
            k, v = self.store.rows(self.oracle.tokens(self.o[h]), layer)
            o, dev, absv = oatt.decode_dev(qb[i], k, v, sm_scale)
            res.append(o)
            bud.append(decode_budget(dev, absv, k.shape[0]))
        return np.stack(res), np.stack(bud)

    def oracle_decode(self, seqs: Sequence[int], layer: int, sm_scale: float, q_cpu) -> np.ndarray:
        qb = bf16_bits(q_cpu)
        res = []
        for i, h in enumerate(seqs):
            k, v = self.store.rows(self.oracle.tokens(self.o[h]), layer)
            res.append(oatt.decode(qb[i], k, v, sm_scale))
        return np.stack(res)


def row_slots(cache, h):
    """(page, slot) of every row of sequence h in logical order, as CUDA
    long tensors, through the library's page table and page fills."""
    pt = cache.page_table(h)
    fills = cache.page_fills(h)
    page = np.repeat(np.asarray(pt, dtype=np.int64), fills)
    slot = np.concatenate([np.arange(f, dtype=np.int64) for f in fills]) if fills else \
        np.zeros(0, dtype=np.int64)
    return torch.from_numpy(page).cuda(), torch.from_numpy(slot).cuda()


def assert_close(got: torch.Tensor, exp: np.ndarray, max_abs=MAX_ABS, mean_abs=MEAN_ABS):
    g = got.detach().float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(g)), "non-finite attention output"
    err = np.abs(g - exp)
    assert err.max() <= max_abs, f"max abs error {err.max():.3g}"
    assert err.mean() <= mean_abs, f"mean abs error {err.mean():.3g}"
    return float(err.max()), float(err.mean())


def assert_budget(got: torch.Tensor, exp: np.ndarray, budget: np.ndarray):
    """The contract's tolerance (max-abs 1e-2, mean-abs 1e-3) and, element by
    element, the error budget the kernel's arithmetic allows (tests/budget.py)."""
    e = assert_close(got, exp)
    g = got.detach().float().cpu().numpy().astype(np.float64)
    over = np.abs(g - exp) - budget
    assert over.max() <= 0.0, f"error above its budget by {over.max():.3g}"
    return e
