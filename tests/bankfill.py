"""Large workloads for parity tests: K/V chunks sliced from a seeded bank
(synthetic.Bank) and appended through the library, with the oracle cache
model tracking token ids, and any token row reconstructed on the host from
its bank offset for the oracle."""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

import numpy as np
import torch

import paper_2602_22603_gb300 as sq
from oracle import cache_model as ocm
from synthetic import Bank, bf16_bits, sub_seed
from tests.gpu_harness import row_slots


class BankPair:
    def __init__(self, L, Hq, Hkv, D, P, num_pages, seed, bank_elems=1 << 28, max_seqs=64,
                 decode_ctas=0):
        self.L, self.Hq, self.Hkv, self.D, self.P = L, Hq, Hkv, D, P
        self.cache = sq.Cache(L, Hq, Hkv, D, P, num_pages, max_seqs=max_seqs,
                              decode_ctas=decode_ctas)
        self.oracle = ocm.OracleCache(num_pages, P)
        self.bank = Bank(bank_elems, sub_seed(seed, 1), device="cuda")
        self.host_bank = None
        self.seed = seed
        self.o: Dict[int, int] = {}
        # appended chunks: (first token id, n, k offset, v offset)
        self.chunks: List[Tuple[int, int, int, int]] = []
        self._firsts = np.zeros(0, dtype=np.int64)
        self._rng = np.random.default_rng(sub_seed(seed, 2))

    def close(self):
        self.cache.close()

    def _offset(self, n):
        elems = self.L * n * self.Hkv * self.D
        hi = (self.bank.n_elems - elems) // 8
        return int(self._rng.integers(0, hi)) * 8

    def seq_new(self):
        h = self.cache.seq_new()
        self.o[h] = self.oracle.seq_new()
        return h

    def fork(self, parent):
        h = self.cache.fork_aux(parent)
        self.o[h] = self.oracle.fork(self.o[parent])
        return h

    def append(self, h, n, stream=None):
        ok, ov = self._offset(n), self._offset(n)
        shape = (self.L, n, self.Hkv, self.D)
        self.cache.append_kv(h, n, self.bank.view(ok, shape), self.bank.view(ov, shape), stream)
        ids = self.oracle.append(self.o[h], n)
        self.chunks.append((ids[0], n, ok, ov))
        self._firsts = np.array([c[0] for c in self.chunks], dtype=np.int64)

    def fill(self, h, n, chunk):
        while n > 0:
            k = min(chunk, n)
            self.append(h, k)
            n -= k

    def evict(self, h, spans, stream=None, ragged=False):
        r = self.oracle.evict(self.o[h], spans, mode="ragged" if ragged else "dense")
        if ragged:
            self.cache.evict_spans_ragged(h, spans, stream)
        else:
            self.cache.evict_spans(h, spans, stream)
        return r

    def release(self, h, stream=None):
        self.cache.release(h, stream)
        self.oracle.release(self.o.pop(h))

    # ---- host reconstruction of rows -----------------------------------------
    def _host(self):
        if self.host_bank is None:
            self.host_bank = bf16_bits(self.bank.data.cpu())
        return self.host_bank

    def rows(self, h, layer, heads=None) -> Tuple[np.ndarray, np.ndarray]:
        """K, V bf16 bits [n, Hkv, D] of sequence h at one layer, in logical
        order, rebuilt from the bank (what the oracle says is there)."""
        hb = self._host()
        toks = np.asarray(self.oracle.tokens(self.o[h]), dtype=np.int64)
        n = len(toks)
        K = np.empty((n, self.Hkv, self.D), dtype=np.uint16)
        V = np.empty_like(K)
        if n == 0:
            return K, V
        # runs of consecutive token ids inside one chunk
        brk = np.nonzero(np.diff(toks) != 1)[0] + 1
        starts = np.concatenate([[0], brk])
        ends = np.concatenate([brk, [n]])
        row = self.Hkv * self.D
        for a, b in zip(starts, ends):
            t0 = int(toks[a])
            pos = a
            while pos < b:
                t = int(toks[pos])
                c = int(np.searchsorted(self._firsts, t, side="right") - 1)
                first, cn, ok, ov = self.chunks[c]
                i0 = t - first
                cnt = min(b - pos, cn - i0)
                base = (layer * cn + i0) * row
                K[pos:pos + cnt] = hb[ok + base: ok + base + cnt * row].reshape(cnt, self.Hkv, self.D)
                V[pos:pos + cnt] = hb[ov + base: ov + base + cnt * row].reshape(cnt, self.Hkv, self.D)
                pos += cnt
        return K, V

    def check_tables(self, handles: Sequence[int]):
        for h in handles:
            assert self.cache.page_table(h) == self.oracle.page_table(self.o[h])
            assert self.cache.page_fills(h) == self.oracle.page_fills(self.o[h])
            assert self.cache.seq_info(h)[0] == self.oracle.n_tokens(self.o[h])
        assert self.cache.free_pages() == self.oracle.free_count()

    def check_planes(self, h, layer, planes=None):
        """The listed (K/V, head) planes of one layer of a sequence (all
        2 x Hkv of them by default), read through the page table from the
        device pool, equal the oracle's rows bit for bit."""
        if planes is None:
            planes = [(kv, head) for kv in (0, 1) for head in range(self.Hkv)]
        torch.cuda.synchronize()
        pool = self.cache.pool_view()
        page, slot = row_slots(self.cache, h)
        K, V = self.rows(h, layer)
        for kv, head in planes:
            got = bf16_bits(pool[layer, page, kv, head, slot, :].cpu())
            exp = (K if kv == 0 else V)[:, head, :]
            assert np.array_equal(got, exp), (layer, kv, head)
