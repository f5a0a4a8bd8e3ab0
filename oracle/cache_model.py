"""CPU oracle: the paged KV cache as a plain integer state machine.

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline / reference legs may import this module.  It shares no code with
the CUDA library and does not import it.

What the paper fixes, and what this model follows:
  * Sec. 3.1 (Overview, steps 1 and 3) and Algorithm 1, phase 2: an auxiliary
    thread is forked on the main thread's context, C_aux <- C + p.
  * Sec. 3.4 (Storage Costs): the auxiliary thread works on the shared
    context and does not duplicate its KV cache; its own tokens are dropped
    once it finishes (Algorithm 1: S_thread <- None).
  * Algorithm 1, phase 1, C.clear_kv(Delta_ids), and Sec. 3 (Goal): the KV
    entries of stale tool calls and responses are removed from the cache; the
    remaining tokens keep their order.
  * Algorithm 1, phase 3: C <- C + R and C <- C + O append to the context.

The paper is silent on paging.  The readings this model fixes (each also in
the design notes) are:
  * pages of P token slots; logical token j of a sequence lives in slot j % P
    of the sequence's page pages[j // P]; len(pages) == ceil(n / P);
  * each page carries a reference count; a page is free iff its count is 0;
    allocation always takes the LOWEST free page id;
  * fork: the child copies the parent's page list and n; every page's count
    grows by one; no K/V row is copied;
  * append(n_new): first, if n % P != 0 and the last page is shared (count
    > 1), a fresh page replaces it (its n % P valid rows copied, the old
    page's count drops by one); then ceil((n+n_new)/P) - ceil(n/P) fresh
    pages are taken in increasing logical order; then the rows are written;
  * evict(spans): spans are half-open [a, b) in current logical positions,
    in any order; overlapping, empty or out-of-range spans are an error and
    leave everything unchanged.  kept = positions in no span, increasing;
    n' = len(kept); new row j <- old row kept[j].  Destination page q
    (q < ceil(n'/P)) is CHANGED when some j in [qP, min(qP+P, n')) has
    kept[j] != j.  A changed page whose count is > 1 is replaced by a fresh
    page (increasing q; the old page's count drops by one); other pages are
    rewritten in place.  Then pages at q >= ceil(n'/P) lose one count each
    and the list is truncated.  Rows past n' in the last page are don't-care;
  * release: every page of the sequence loses one count;
  * PAGE FILLS.  Every page of a sequence carries a fill f (1 <= f <= P):
    its slots 0 .. f-1 hold the sequence's rows, in order, and the logical
    rows are the concatenation of the pages' filled slots.  After the
    operations above every page is full except the last (the dense layout:
    logical j in slot j % P of pages[j // P]).  Appends fill the last page's
    free slots first (after the copy-on-write above, which copies its f rows),
    then take fresh pages.  The dense eviction above reads its sources
    through the fills, so it also packs a sequence that had partial pages;
  * RAGGED eviction (the "next" row of the hot path: drop pages by remapping,
    compact only what the spans touch; not in the paper, whose clear_kv says
    only that the entries go): a page is TOUCHED when a span removes one of
    its rows; a WINDOW is a maximal run of consecutive touched pages.  A
    window's kept rows, in order, are packed from slot 0 of its first page:
    its first ceil(r / P) pages receive them (all full but the last), its
    other pages leave the sequence (one count less each), pages outside every
    window keep their rows, slots and fills untouched.  A window page whose
    rows change (some destination slot receives a row from another page or
    slot) and whose count is > 1 is replaced by a fresh page, in increasing
    logical order (the old page loses one count), others are rewritten in
    place.  When a window's last page is written (its rows change, or it is
    a fresh page), its slots past the fill are set to zero; an unchanged one
    keeps them (they hold rows appended earlier, which a fork may still
    read).  So the unused slots of a page that ends early hold zeros or rows
    once appended, never memory no row was written to.  An empty span set
    changes nothing;
  * an operation that would need more free pages than exist, or more than
    max_pages_per_seq pages for one sequence, fails and changes nothing.

Contents are modelled by TOKEN IDS: every appended row gets a fresh integer,
and "the row at logical position j" is the id now there.  The optional
physical mode additionally keeps, per page, which id sits in each slot and
performs the moves the rules above describe (in-place moves in increasing j),
so a test can check that reading the pages through the page table gives back
the logical contents.
"""
from __future__ import annotations

import heapq
from typing import Dict, List, Optional, Sequence, Tuple


class OracleError(Exception):
    code = "error"


class InvalidArg(OracleError):
    code = "invalid_arg"


class NoPages(OracleError):
    code = "no_pages"


class Capacity(OracleError):
    code = "capacity"


class BadHandle(OracleError):
    code = "bad_handle"


def ceil_div(a: int, b: int) -> int:
    return -(-a // b)


# the physical-mode stand-in for a slot that was set to zero
ZERO = -2


class _Seq:
    __slots__ = ("pages", "fills", "tokens")

    def __init__(self, pages: List[int], fills: List[int], tokens: List[int]):
        self.pages = pages
        self.fills = fills
        self.tokens = tokens

    def locations(self) -> List[Tuple[int, int]]:
        """(page index, slot) of every logical row, in order, through the fills."""
        return [(q, t) for q, f in enumerate(self.fills) for t in range(f)]


class OracleCache:
    def __init__(self, num_pages: int, page_size: int,
                 max_pages_per_seq: Optional[int] = None,
                 physical: bool = False):
        if num_pages <= 0 or page_size <= 0:
            raise InvalidArg("bad geometry")
        self.P = int(page_size)
        self.num_pages = int(num_pages)
        self.max_pages_per_seq = int(max_pages_per_seq or num_pages)
        self.ref = [0] * self.num_pages
        self._free = list(range(self.num_pages))  # min-heap of free ids
        heapq.heapify(self._free)
        self.seqs: Dict[int, _Seq] = {}
        self._next_seq = 0
        self._next_token = 0
        self.phys: Optional[Dict[int, List[int]]] = {} if physical else None
        self.peak_live_pages = 0

    # -- pages ---------------------------------------------------------------
    def free_count(self) -> int:
        return len(self._free)

    def live_pages(self) -> int:
        return self.num_pages - len(self._free)

    def _alloc(self) -> int:
        p = heapq.heappop(self._free)
        assert self.ref[p] == 0
        self.ref[p] = 1
        if self.phys is not None:
            self.phys[p] = [-1] * self.P
        self.peak_live_pages = max(self.peak_live_pages, self.live_pages())
        return p

    def _unref(self, p: int) -> None:
        assert self.ref[p] > 0
        self.ref[p] -= 1
        if self.ref[p] == 0:
            heapq.heappush(self._free, p)
            if self.phys is not None:
                del self.phys[p]

    def _seq(self, sid: int) -> _Seq:
        if sid not in self.seqs:
            raise BadHandle(f"unknown sequence {sid}")
        return self.seqs[sid]

    # -- operations ------------------------------------------------------------
    def seq_new(self) -> int:
        sid = self._next_seq
        self._next_seq += 1
        self.seqs[sid] = _Seq([], [], [])
        return sid

    def fork(self, parent: int) -> int:
        ps = self._seq(parent)
        sid = self._next_seq
        self._next_seq += 1
        for p in ps.pages:
            self.ref[p] += 1
        self.seqs[sid] = _Seq(list(ps.pages), list(ps.fills), list(ps.tokens))
        return sid

    def append(self, sid: int, n_new: int) -> List[int]:
        """Append n_new rows; returns the token ids given to them."""
        s = self._seq(sid)
        if n_new < 0:
            raise InvalidArg("negative token count")
        if n_new == 0:
            return []
        P = self.P
        n = len(s.tokens)
        last_fill = s.fills[-1] if s.pages else P
        room = P - last_fill                       # free slots of the last page
        cow = room > 0 and self.ref[s.pages[-1]] > 1
        grow = ceil_div(max(0, n_new - room), P)
        if len(s.pages) + grow > self.max_pages_per_seq:
            raise Capacity("sequence would exceed max_pages_per_seq")
        if int(cow) + grow > self.free_count():
            raise NoPages("not enough free pages")
        if cow:
            old = s.pages[-1]
            new = self._alloc()
            if self.phys is not None:
                for slot in range(last_fill):
                    self.phys[new][slot] = self.phys[old][slot]
            self._unref(old)
            s.pages[-1] = new
        ids = list(range(self._next_token, self._next_token + n_new))
        self._next_token += n_new
        for tok in ids:
            if not s.pages or s.fills[-1] == P:
                s.pages.append(self._alloc())
                s.fills.append(0)
            if self.phys is not None:
                self.phys[s.pages[-1]][s.fills[-1]] = tok
            s.fills[-1] += 1
        s.tokens.extend(ids)
        return ids

    @staticmethod
    def check_spans(spans: Sequence[Tuple[int, int]], n: int) -> List[Tuple[int, int]]:
        srt = sorted((int(a), int(b)) for a, b in spans)
        prev_end = 0
        for a, b in srt:
            if a < 0 or b > n or a >= b:
                raise InvalidArg(f"span [{a},{b}) empty or outside [0,{n})")
            if a < prev_end:
                raise InvalidArg("overlapping spans")
            prev_end = b
        return srt

    def evict(self, sid: int, spans: Sequence[Tuple[int, int]],
              mode: str = "dense") -> Dict[str, int]:
        """Remove the rows in `spans`; returns counters of the work done.
        mode "dense" packs the kept rows into full pages, "ragged" drops and
        packs pages window by window (see the module notes)."""
        if mode == "ragged":
            return self._evict_ragged(sid, spans)
        if mode != "dense":
            raise InvalidArg(f"unknown eviction mode {mode}")
        s = self._seq(sid)
        P = self.P
        n = len(s.tokens)
        srt = self.check_spans(spans, n)
        if not srt:
            return {"n_before": n, "n_after": n, "moved_rows": 0, "cow_pages": 0,
                    "released_pages": 0}
        removed = set()
        for a, b in srt:
            removed.update(range(a, b))
        kept = [j for j in range(n) if j not in removed]
        n2 = len(kept)
        new_np = ceil_div(n2, P)
        loc = s.locations()
        src = [loc[k] for k in kept]          # (page index, slot) of each kept row
        changed = [any(src[j] != (q, j % P) for j in range(q * P, min(q * P + P, n2)))
                   for q in range(new_np)]
        cow_q = [q for q in range(new_np) if changed[q] and self.ref[s.pages[q]] > 1]
        if len(cow_q) > self.free_count():
            raise NoPages("not enough free pages for copy-on-write")

        old_pages = list(s.pages)
        new_pages = old_pages[:new_np]
        for q in cow_q:                       # fresh pages in increasing q
            new_pages[q] = self._alloc()
        moved = 0
        for j in range(n2):                   # destination rows, increasing j
            q = j // P
            if src[j] == (q, j % P) and new_pages[q] == old_pages[q]:
                continue                      # row stays where it is
            moved += 1
            if self.phys is not None:
                sq_, ss = src[j]
                self.phys[new_pages[q]][j % P] = self.phys[old_pages[sq_]][ss]
        for q in cow_q:                       # the shared originals lose a holder
            self._unref(old_pages[q])
        for p in old_pages[new_np:]:          # trailing pages
            self._unref(p)
        s.pages = new_pages
        s.fills = [min(P, n2 - q * P) for q in range(new_np)]
        s.tokens = [s.tokens[j] for j in kept]
        return {"n_before": n, "n_after": n2, "moved_rows": moved,
                "cow_pages": len(cow_q), "released_pages": len(old_pages) - new_np}

    def _evict_ragged(self, sid: int, spans: Sequence[Tuple[int, int]]) -> Dict[str, int]:
        s = self._seq(sid)
        P = self.P
        n = len(s.tokens)
        srt = self.check_spans(spans, n)
        zero = {"n_before": n, "n_after": n, "moved_rows": 0, "cow_pages": 0,
                "released_pages": 0, "windows": 0, "zeroed_rows": 0}
        if not srt:
            return zero
        removed = set()
        for a, b in srt:
            removed.update(range(a, b))
        # the rows of every page, as logical positions
        rows_of = []
        j = 0
        for f in s.fills:
            rows_of.append(list(range(j, j + f)))
            j += f
        touched = [any(r in removed for r in rows) for rows in rows_of]
        windows = []                          # [first, last] page indices
        q = 0
        while q < len(s.pages):
            if touched[q]:
                e = q
                while e + 1 < len(s.pages) and touched[e + 1]:
                    e += 1
                windows.append((q, e))
                q = e + 1
            else:
                q += 1
        # the new layout, window by window: page index -> (page, rows) with
        # rows the (old page index, slot) of each destination slot
        dest = {}                             # old page index -> [(src q, src slot)]
        dropped = []                          # old page indices that leave
        for qa, qb in windows:
            src = [(q, t) for q in range(qa, qb + 1) for t, r in enumerate(rows_of[q])
                   if r not in removed]
            used = ceil_div(len(src), P)
            for i in range(qb - qa + 1):
                if i < used:
                    dest[qa + i] = src[i * P:(i + 1) * P]
                else:
                    dropped.append(qa + i)
        changed = {q: any(sv != (q, t) for t, sv in enumerate(rows)) for q, rows in dest.items()}
        cow_q = sorted(q for q in dest if changed[q] and self.ref[s.pages[q]] > 1)
        if len(cow_q) > self.free_count():
            raise NoPages("not enough free pages for copy-on-write")

        old_pages = list(s.pages)
        new_page = {q: old_pages[q] for q in dest}
        for q in cow_q:                       # fresh pages in increasing logical order
            new_page[q] = self._alloc()
        moved = 0
        zeroed = 0
        for q in sorted(dest):                # destination pages, increasing; slots increasing
            rows = dest[q]
            fresh = new_page[q] != old_pages[q]
            for t, (sq_, ss) in enumerate(rows):
                if not fresh and (sq_, ss) == (q, t):
                    continue                  # row stays where it is
                moved += 1
                if self.phys is not None:
                    self.phys[new_page[q]][t] = self.phys[old_pages[sq_]][ss]
        for qa, qb in windows:                # zeros past the fill of each window's last page
            last = max((q for q in dest if qa <= q <= qb), default=None)
            if last is None or not (changed[last] or new_page[last] != old_pages[last]):
                continue
            for t in range(len(dest[last]), P):
                zeroed += 1
                if self.phys is not None:
                    self.phys[new_page[last]][t] = ZERO
        for q in cow_q:
            self._unref(old_pages[q])
        for q in dropped:
            self._unref(old_pages[q])
        pages, fills = [], []
        for q in range(len(old_pages)):
            if q in dest:
                pages.append(new_page[q])
                fills.append(len(dest[q]))
            elif q not in dropped:
                pages.append(old_pages[q])
                fills.append(s.fills[q])
        s.pages = pages
        s.fills = fills
        s.tokens = [t for j, t in enumerate(s.tokens) if j not in removed]
        return {"n_before": n, "n_after": len(s.tokens), "moved_rows": moved,
                "cow_pages": len(cow_q), "released_pages": len(dropped),
                "windows": len(windows), "zeroed_rows": zeroed}

    def release(self, sid: int) -> None:
        s = self._seq(sid)
        for p in s.pages:
            self._unref(p)
        del self.seqs[sid]

    # -- views -----------------------------------------------------------------
    def n_tokens(self, sid: int) -> int:
        return len(self._seq(sid).tokens)

    def page_table(self, sid: int) -> List[int]:
        return list(self._seq(sid).pages)

    def page_fills(self, sid: int) -> List[int]:
        return list(self._seq(sid).fills)

    def tokens(self, sid: int) -> List[int]:
        return list(self._seq(sid).tokens)

    def physical_tokens(self, sid: int) -> List[int]:
        """Token ids read back through the page table from the physical
        pages (physical mode only)."""
        assert self.phys is not None
        s = self._seq(sid)
        out = []
        for p, f in zip(s.pages, s.fills):
            out.extend(self.phys[p][:f])
        return out
