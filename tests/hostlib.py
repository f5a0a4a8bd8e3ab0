"""ctypes face of libsq_host.so: the library's host-side cache state and
planners, built without CUDA, for CPU tests."""
import ctypes
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2602_22603_gb300 import build as _build  # noqa: E402

_lib = None

SEG_INTS = 4 + 2 * 16 + 2  # DecodeSeg: page_off, n_pages, n_tok, n_grp, grp_seq[16], grp_lim[16], q0, tail
ITEM_INTS = 5 + 16     # DecodeItem: seg, head, s0, s1, sole, ent[16]


def lib():
    global _lib
    if _lib is None:
        path = _build.build_host_lib()
        L = ctypes.CDLL(path)
        P, I32, I32P, I64P = ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32), \
            ctypes.POINTER(ctypes.c_int64)
        L.sqh_create.restype = P
        L.sqh_create.argtypes = [I32] * 8
        L.sqh_destroy.argtypes = [P]
        L.sqh_seq_new.argtypes = [P, I32P]
        L.sqh_fork.argtypes = [P, I32, I32P]
        L.sqh_append.argtypes = [P, I32, I32]
        L.sqh_evict.argtypes = [P, I32, I32P, I32, I32, I64P]
        L.sqh_release.argtypes = [P, I32]
        L.sqh_evict_tiles.argtypes = [P, I32, I32P, I32, I32, I32, I32P, I32, I32P, I32, I32P,
                                      I32P, I32, I32P, I32, I32P]
        L.sqh_page_fill.argtypes = [P, I32, I32P, I32, I32P]
        L.sqh_prefill_slot_spans.argtypes = [P, I32, I32, I32P, I32, I32P, I32, I32P, I32P]
        L.sqh_seq_info.argtypes = [P, I32, I32P, I32P]
        L.sqh_next_pos.argtypes = [P, I32]
        L.sqh_next_pos.restype = ctypes.c_int64
        L.sqh_page_table.argtypes = [P, I32, I32P, I32, I32P]
        L.sqh_refcount.argtypes = [P, I32]
        L.sqh_free_count.argtypes = [P]
        L.sqh_peak_live_pages.argtypes = [P]
        L.sqh_peak_live_pages.restype = ctypes.c_int64
        L.sqh_plan_decode.argtypes = [P, I32P, I32, I32, I64P, ctypes.POINTER(ctypes.c_uint8),
                                      ctypes.c_int64]
        L.sqh_evict_tile_rows.argtypes = [I32, I32]
        L.sqh_evict_tile_rows.restype = ctypes.c_int32
        L.sqh_evict_stages.argtypes = [ctypes.c_int64, I32]
        L.sqh_evict_stages.restype = ctypes.c_int32
        L.sqh_plan_prefill.argtypes = [I32, I32, I32, I32, I32, I32P, I32, I32, I64P, I32P, I32,
                                       I32P, I32]
        _lib = L
    return _lib


def plan_prefill(Hq, Hkv, n, n_q, spans, target_ctas=152, cap=1 << 16, P=64):
    """(rc, info dict, tiles [k, 7] int64 array of key0, flags, vis[4], key0b)."""
    arr = (ctypes.c_int32 * max(2, 2 * len(spans)))(*[int(x) for ab in spans for x in ab])
    info = (ctypes.c_int64 * 6)()
    tiles = (ctypes.c_int32 * (7 * cap))()
    qt = (ctypes.c_int32 * cap)()
    rc = lib().sqh_plan_prefill(Hq, Hkv, P, n, n_q, arr, len(spans), target_ctas, info, tiles,
                                cap, qt, cap)
    d = dict(zip(("n_tiles", "BP", "n_qt", "n_split", "visible_pairs", "tile_bytes"), list(info)))
    d["qt_tiles"] = list(qt[: d["n_qt"]]) if rc == 0 else []
    t = np.frombuffer(tiles, dtype=np.int32).reshape(-1, 7)[: d["n_tiles"] if rc == 0 else 0]
    t = t.astype(np.int64)
    t[:, 1:6] &= 0xffffffff
    return rc, d, t


class HostCache:
    def __init__(self, L, Hq, Hkv, D, P, num_pages, max_seqs=64, max_pages_per_seq=None):
        self.h = lib().sqh_create(L, Hq, Hkv, D, P, num_pages, max_seqs,
                                  max_pages_per_seq or num_pages)
        assert self.h, "invalid geometry"
        self.P, self.Hkv, self.G = P, Hkv, Hq // Hkv

    def __del__(self):
        if getattr(self, "h", None):
            lib().sqh_destroy(self.h)
            self.h = None

    def seq_new(self):
        x = ctypes.c_int32()
        rc = lib().sqh_seq_new(self.h, ctypes.byref(x))
        return rc, x.value

    def fork(self, parent):
        x = ctypes.c_int32()
        rc = lib().sqh_fork(self.h, parent, ctypes.byref(x))
        return rc, x.value

    def append(self, h, n):
        return lib().sqh_append(self.h, h, n)

    def evict(self, h, spans, ragged=False):
        arr = (ctypes.c_int32 * max(2, 2 * len(spans)))(*[int(x) for ab in spans for x in ab])
        st = (ctypes.c_int64 * 6)()
        rc = lib().sqh_evict(self.h, h, arr, len(spans), int(ragged), st)
        return rc, {"moved_rows": st[0], "cow_pages": st[1], "freed": st[2],
                    "zeroed_rows": st[3], "windows": st[4], "n_moves": st[5]}

    def evict_tiles(self, h, spans, tile_rows, ragged=False, cap=100000, max_chunks=1,
                    want_chunks=False):
        arr = (ctypes.c_int32 * max(2, 2 * len(spans)))(*[int(x) for ab in spans for x in ab])
        tiles = np.zeros(4 * cap, dtype=np.int32)
        pieces = np.zeros(4 * cap, dtype=np.int32)
        chunks = np.zeros(cap, dtype=np.int32)
        nt, npc, nch = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        i32p = ctypes.POINTER(ctypes.c_int32)
        rc = lib().sqh_evict_tiles(self.h, h, arr, len(spans), int(ragged), tile_rows,
                                   tiles.ctypes.data_as(i32p), cap, pieces.ctypes.data_as(i32p),
                                   cap, ctypes.byref(nt), ctypes.byref(npc), max_chunks,
                                   chunks.ctypes.data_as(i32p), cap, ctypes.byref(nch))
        if rc != 0:
            return (rc, None, None, None) if want_chunks else (rc, None, None)
        t = tiles[:4 * nt.value].reshape(-1, 4)
        pc = pieces[:4 * npc.value].reshape(-1, 4)
        if want_chunks:
            return 0, t, pc, chunks[:nch.value + 1].tolist()
        return 0, t, pc

    def release(self, h):
        return lib().sqh_release(self.h, h)

    def info(self, h):
        n, p = ctypes.c_int32(), ctypes.c_int32()
        rc = lib().sqh_seq_info(self.h, h, ctypes.byref(n), ctypes.byref(p))
        return rc, n.value, p.value

    def next_pos(self, h):
        return lib().sqh_next_pos(self.h, h)

    def page_table(self, h):
        rc, n, npg = self.info(h)
        assert rc == 0
        buf = (ctypes.c_int32 * max(1, npg))()
        m = ctypes.c_int32()
        assert lib().sqh_page_table(self.h, h, buf, npg, ctypes.byref(m)) == 0
        return list(buf[:m.value])

    def page_fill(self, h):
        rc, n, npg = self.info(h)
        assert rc == 0
        buf = (ctypes.c_int32 * max(1, npg))()
        m = ctypes.c_int32()
        assert lib().sqh_page_fill(self.h, h, buf, npg, ctypes.byref(m)) == 0
        return list(buf[:m.value])

    def prefill_slot_spans(self, h, n_q, spans, cap=1 << 16):
        """(rc, slot-space spans, slot-space end) of a masked prefill."""
        arr = (ctypes.c_int32 * max(2, 2 * len(spans)))(*[int(x) for ab in spans for x in ab])
        out = (ctypes.c_int32 * (2 * cap))()
        m, ns = ctypes.c_int32(), ctypes.c_int32()
        rc = lib().sqh_prefill_slot_spans(self.h, h, n_q, arr, len(spans), out, cap,
                                          ctypes.byref(m), ctypes.byref(ns))
        if rc != 0:
            return rc, None, None
        return 0, [(out[2 * i], out[2 * i + 1]) for i in range(m.value)], ns.value

    def refcount(self, p):
        return lib().sqh_refcount(self.h, p)

    def free_count(self):
        return lib().sqh_free_count(self.h)

    def peak_live_pages(self):
        return lib().sqh_peak_live_pages(self.h)

    def plan_decode(self, handles, n_ctas):
        arr = (ctypes.c_int32 * len(handles))(*handles)
        lay = (ctypes.c_int64 * 17)()
        rc = lib().sqh_plan_decode(self.h, arr, len(handles), n_ctas, lay, None, 0)
        if rc != 0:
            return rc, None
        total = lay[6]
        buf = np.zeros(total, dtype=np.uint8)
        rc = lib().sqh_plan_decode(self.h, arr, len(handles), n_ctas, lay,
                                   buf.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)), total)
        assert rc == 0
        L = list(lay)
        assert L[15] == SEG_INTS * 4
        i32 = buf.view(np.int32)

        def arr_at(off, count, width=1):
            a = i32[off // 4: off // 4 + count * width]
            return a.reshape(count, width) if width > 1 else a

        n_segs, n_items, n_ctas_, n_pid, n_keys, n_ent = L[7:13]
        segs = arr_at(L[0], n_segs, SEG_INTS)
        seg_list = [{"page_off": int(s[0]), "n_pages": int(s[1]), "n_tok": int(s[2]),
                     "n_grp": int(s[3]), "grp_seq": [int(x) for x in s[4:4 + s[3]]],
                     "grp_lim": [int(x) for x in s[20:20 + s[3]]], "q0": int(s[36]),
                     "tail": int(s[37])} for s in segs]
        raw_items = arr_at(L[1], n_items, ITEM_INTS) if n_items else np.zeros((0, ITEM_INTS), np.int32)
        comb_off = arr_at(L[4], n_keys + 1).tolist()
        # each item's group members name their partial entry; every entry is
        # named once, inside the range of its (sequence, KV head)
        comb_ent = [None] * n_ent
        for it, row in enumerate(raw_items):
            seg = seg_list[row[0]]
            for j in range(seg["n_grp"]):
                e = int(row[5 + j])
                key = seg["grp_seq"][j] * self.Hkv + int(row[1])
                assert comb_off[key] <= e < comb_off[key + 1], (it, j, e)
                assert comb_ent[e] is None, e
                comb_ent[e] = [it, j]
                # the sole bit marks exactly the one-entry runs
                assert bool((int(row[4]) >> j) & 1) == (comb_off[key + 1] - comb_off[key] == 1)
        assert all(x is not None for x in comb_ent)
        arrive = buf[L[5]:L[5] + 4 * n_keys]
        assert L[5] % 4 == 0 and not arrive.any()
        plan = {
            "segs": seg_list,
            "items": raw_items[:, :4].tolist(),
            "cta_begin": arr_at(L[2], n_ctas_ + 1).tolist(),
            "page_ids": arr_at(L[3], n_pid).tolist(),
            "comb_off": comb_off,
            "comb_ent": comb_ent,
            "unique_tokens": L[13], "logical_tokens": L[14],
            "page_fill": arr_at(L[16], n_pid).tolist() if L[16] >= 0 else None,
        }
        return 0, plan
