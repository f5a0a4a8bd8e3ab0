// Host-side cache state and planners.  See core.hpp for the rules.
#include "core.hpp"

#include <algorithm>
#include <atomic>
#include <cstring>
#include <unordered_map>

namespace sq {

static inline int32_t ceil_div(int64_t a, int64_t b) { return (int32_t)((a + b - 1) / b); }

int check_geometry(const Geometry& g) {
    if (g.L < 1 || g.Hq < 1 || g.Hkv < 1 || g.D < 1 || g.P < 1 ||
        g.num_pages < 1 || g.max_seqs < 1 || g.max_pages_per_seq < 1)
        return kInvalidArg;
    if (g.Hq % g.Hkv != 0) return kInvalidArg;
    if (g.G() > kRowsPerTile) return kUnsupported;
    if (g.D != 64 && g.D != 128) return kUnsupported;
    if (g.P < 8 || g.P > 256 || (g.P & (g.P - 1)) != 0) return kUnsupported;
    if (g.max_seqs >= (1 << 20)) return kUnsupported;
    // logical positions are int32
    if ((int64_t)g.max_pages_per_seq * g.P >= (1LL << 31)) return kUnsupported;
    return kOk;
}

int sorted_spans(int32_t n, const int32_t* starts, const int32_t* ends, int32_t n_spans,
                 std::vector<std::pair<int32_t, int32_t>>* out) {
    out->clear();
    if (n_spans < 0) return kInvalidArg;
    if (n_spans == 0) return kOk;
    if (!starts || !ends) return kInvalidArg;
    auto& sp = *out;
    sp.resize(n_spans);
    for (int32_t i = 0; i < n_spans; ++i) sp[i] = {starts[i], ends[i]};
    std::sort(sp.begin(), sp.end());
    int32_t prev_end = 0;
    for (auto& ab : sp) {
        if (ab.first < 0 || ab.second > n || ab.first >= ab.second || ab.first < prev_end) {
            out->clear();
            return kInvalidArg;
        }
        prev_end = ab.second;
    }
    return kOk;
}

// ---------------------------------------------------------------------------
PageAllocator::PageAllocator(int32_t n)
    : ref_(n, 0), free_bits_((n + 63) / 64, 0), free_count_(n) {
    for (int32_t i = 0; i < n; ++i) free_bits_[i >> 6] |= 1ULL << (i & 63);
}

int32_t PageAllocator::lowest_free() const {
    const int32_t words = (int32_t)free_bits_.size();
    for (int32_t w = hint_; w < words; ++w) {
        if (free_bits_[w]) {
            hint_ = w;
            return w * 64 + __builtin_ctzll(free_bits_[w]);
        }
    }
    hint_ = words;
    return -1;
}

void PageAllocator::take(int32_t p) {
    ref_[p] = 1;
    free_bits_[p >> 6] &= ~(1ULL << (p & 63));
    --free_count_;
}

bool PageAllocator::drop_ref(int32_t p) {
    if (--ref_[p] == 0) {
        free_bits_[p >> 6] |= 1ULL << (p & 63);
        ++free_count_;
        if ((p >> 6) < hint_) hint_ = p >> 6;
        return true;
    }
    return false;
}

// ---------------------------------------------------------------------------
// shared by every cache (of any thread): a version is never handed out twice
static std::atomic<uint64_t> g_version_counter{1};

HostCache::HostCache(const Geometry& g) : g_(g), alloc_(g.num_pages), seqs_(g.max_seqs) {
    free_slots_.reserve(g.max_seqs);
    for (int32_t s = g.max_seqs - 1; s >= 0; --s) free_slots_.push_back(s);
}

int32_t HostCache::take_lowest() {
    int32_t p = alloc_.lowest_free();
    alloc_.take(p);
    int64_t live = live_pages();
    if (live > peak_live_) peak_live_ = live;
    return p;
}

const Seq* HostCache::seq(int32_t h) const {
    if (h <= 0) return nullptr;
    int32_t slot = h & 0xFFFFF;
    uint32_t gen = (uint32_t)h >> 20;
    if (slot >= g_.max_seqs) return nullptr;
    const Seq& s = seqs_[slot];
    if (!s.live || s.gen != gen) return nullptr;
    return &s;
}

Seq* HostCache::seq_mut(int32_t h) { return const_cast<Seq*>(seq(h)); }

int HostCache::seq_new(int32_t* handle) {
    if (free_slots_.empty()) return kCapacity;
    int32_t slot = free_slots_.back();
    free_slots_.pop_back();
    Seq& s = seqs_[slot];
    s.live = true;
    s.gen = (s.gen % 2047) + 1;  // 1 .. 2047: handles stay positive
    s.n = 0;
    s.pages.clear();
    s.fill.clear();
    s.next_pos = 0;
    s.version = g_version_counter++;
    s.last_stream = nullptr;
    *handle = (int32_t)((s.gen << 20) | (uint32_t)slot);
    return kOk;
}

int HostCache::fork(int32_t parent, int32_t* child) {
    const Seq* ps = seq(parent);
    if (!ps) return kBadHandle;
    std::vector<int32_t> pages = ps->pages;
    std::vector<int32_t> fill = ps->fill;
    int32_t n = ps->n;
    const int64_t next_pos = ps->next_pos;
    void* st = ps->last_stream;
    int rc = seq_new(child);
    if (rc != kOk) return rc;
    Seq* cs = seq_mut(*child);
    cs->pages = std::move(pages);
    cs->fill = std::move(fill);
    cs->n = n;
    cs->next_pos = next_pos;
    cs->last_stream = st;
    for (int32_t p : cs->pages) alloc_.add_ref(p);
    return kOk;
}

int HostCache::append(int32_t h, int32_t n_new, AppendPlan* plan) {
    *plan = AppendPlan();
    if (n_new < 0) return kInvalidArg;
    Seq* s = seq_mut(h);
    if (!s) return kBadHandle;
    const int32_t P = g_.P;
    const int32_t n = s->n;
    plan->n0 = n;
    plan->n_new = n_new;
    plan->pos0 = slot_end(*s, P);
    plan->last_fill0 = s->pages.empty() ? 0 : s->fill.back();
    if (n_new == 0) return kOk;
    if ((int64_t)n + n_new >= (1LL << 31)) return kCapacity;
    // the last page's free slots take the first rows, then fresh pages
    const int32_t room = s->pages.empty() ? 0 : P - s->fill.back();
    const int64_t grow = n_new > room ? ((int64_t)n_new - room + P - 1) / P : 0;
    const int64_t new_np = (int64_t)s->pages.size() + grow;
    if (new_np > g_.max_pages_per_seq) return kCapacity;
    const bool cow = room > 0 && alloc_.refcount(s->pages.back()) > 1;
    const int64_t need = (cow ? 1 : 0) + grow;
    if (need > alloc_.free_count()) return kNoPages;

    if (cow) {
        int32_t old = s->pages.back();
        int32_t fresh = take_lowest();
        alloc_.drop_ref(old);  // was > 1: stays held by the other sequences
        s->pages.back() = fresh;
        plan->cow = true;
        plan->cow_old = old;
        plan->cow_new = fresh;
        plan->cow_rows = s->fill.back();
        plan->taken.push_back(fresh);
    }
    plan->first_page_index = plan->pos0 / P;
    int32_t left = n_new;
    if (room > 0) {
        const int32_t k = std::min(room, left);
        s->fill.back() += k;
        left -= k;
    }
    while (left > 0) {
        int32_t p = take_lowest();
        s->pages.push_back(p);
        s->fill.push_back(std::min(P, left));
        left -= s->fill.back();
        plan->taken.push_back(p);
    }
    plan->pages.assign(s->pages.begin() + plan->first_page_index, s->pages.end());
    s->n = n + n_new;
    s->next_pos += n_new;
    s->version = g_version_counter++;
    return kOk;
}

void HostCache::undo_append(int32_t h, const AppendPlan& plan) {
    Seq* s = seq_mut(h);
    if (!s || plan.n_new == 0) return;
    // pages before the append: pos0 = (pages - 1) * P + last fill
    const int32_t keep = plan.last_fill0 > 0 ? (plan.pos0 - plan.last_fill0) / g_.P + 1 : 0;
    while ((int32_t)s->pages.size() > keep) {
        alloc_.drop_ref(s->pages.back());
        s->pages.pop_back();
        s->fill.pop_back();
    }
    if (keep > 0) s->fill.back() = plan.last_fill0;
    if (plan.cow) {
        alloc_.drop_ref(plan.cow_new);
        alloc_.add_ref(plan.cow_old);
        s->pages.back() = plan.cow_old;
    }
    s->n = plan.n0;
    s->next_pos -= plan.n_new;
    s->version = g_version_counter++;
}

bool has_partial_pages(const Seq& s, int32_t P) {
    for (size_t q = 0; q + 1 < s.fill.size(); ++q)
        if (s.fill[q] != P) return true;
    return false;
}

namespace {

// A run of rows moving as one: destination page index / slot, source page
// index / slot (indices into the sequence's page table before the eviction).
struct Run {
    int32_t dq, ds, sq, ss, n;
};

// Packs the kept logical rows `kept` (increasing, disjoint half-open ranges)
// into consecutive slots from slot 0 of page index dq0, splitting at source
// and destination page boundaries.  start[q] = first logical row of page q.
void pack_rows(const std::vector<std::pair<int32_t, int32_t>>& kept,
               const std::vector<int32_t>& start, int32_t P, int32_t dq0, std::vector<Run>* out) {
    int64_t m = 0;  // destination index from slot 0 of page dq0
    size_t q = 0;   // source page index, monotone
    for (const auto& r : kept) {
        int32_t j = r.first;
        while (j < r.second) {
            while (start[q + 1] <= j) ++q;
            const int32_t ds = (int32_t)(m % P);
            const int32_t n = std::min({r.second - j, start[q + 1] - j, P - ds});
            out->push_back({dq0 + (int32_t)(m / P), ds, (int32_t)q, j - start[q], n});
            j += n;
            m += n;
        }
    }
}

}  // namespace

int HostCache::evict(int32_t h, const int32_t* starts, const int32_t* ends,
                     int32_t n_spans, EvictPlan* plan, bool ragged) {
    *plan = EvictPlan();
    Seq* s = seq_mut(h);
    if (!s) return kBadHandle;
    if (n_spans < 0) return kInvalidArg;
    const int32_t n = s->n;
    const int32_t P = g_.P;
    plan->ragged = ragged;
    plan->n_old = n;
    plan->n_new = n;
    plan->old_pages = s->pages;
    plan->old_fill = s->fill;
    plan->new_pages = s->pages;
    plan->new_fill = s->fill;
    if (n_spans == 0) return kOk;
    if (!starts || !ends) return kInvalidArg;

    std::vector<std::pair<int32_t, int32_t>> sp;
    int rc = sorted_spans(n, starts, ends, n_spans, &sp);
    if (rc != kOk) return rc;
    const int32_t np = (int32_t)s->pages.size();
    std::vector<int32_t> start(np + 1, 0);
    for (int32_t q = 0; q < np; ++q) start[q + 1] = start[q] + s->fill[q];
    int64_t removed = 0;
    for (auto& ab : sp) removed += ab.second - ab.first;

    // Windows: the whole table (dense), or the maximal runs of pages a span
    // touches (ragged).  Each window's kept rows are packed from slot 0 of
    // its first page.
    struct Window {
        int32_t qa, qb;                                 // page indices, inclusive
        std::vector<std::pair<int32_t, int32_t>> kept;  // logical row ranges
        int32_t used = 0;                               // pages that receive rows
    };
    std::vector<Window> win;
    if (!ragged) {
        win.push_back({0, np - 1, {}, 0});
    } else {
        std::vector<uint8_t> touched(np, 0);
        int32_t q = 0;
        for (auto& ab : sp) {
            while (start[q + 1] <= ab.first) ++q;
            int32_t e = q;
            while (start[e + 1] < ab.second) ++e;
            for (int32_t x = q; x <= e; ++x) touched[x] = 1;
        }
        for (q = 0; q < np;) {
            if (!touched[q]) {
                ++q;
                continue;
            }
            int32_t e = q;
            while (e + 1 < np && touched[e + 1]) ++e;
            win.push_back({q, e, {}, 0});
            q = e + 1;
        }
    }
    size_t si = 0;
    for (Window& w : win) {
        int32_t cur = start[w.qa];
        const int32_t end = start[w.qb + 1];
        while (si < sp.size() && sp[si].second <= cur) ++si;
        size_t k = si;
        while (cur < end) {
            if (k < sp.size() && sp[k].first < end) {
                if (sp[k].first > cur) w.kept.push_back({cur, sp[k].first});
                cur = std::max(cur, sp[k].second);
                ++k;
            } else {
                w.kept.push_back({cur, end});
                cur = end;
            }
        }
    }

    // runs, and which destination pages change
    std::vector<std::vector<Run>> runs(win.size());
    std::vector<uint8_t> changed(np, 0);
    std::vector<int32_t> dest_fill(np, 0);
    for (size_t wi = 0; wi < win.size(); ++wi) {
        Window& w = win[wi];
        pack_rows(w.kept, start, P, w.qa, &runs[wi]);
        int64_t r = 0;
        for (auto& kr : w.kept) r += kr.second - kr.first;
        w.used = (int32_t)((r + P - 1) / P);
        for (int32_t i = 0; i < w.used; ++i)
            dest_fill[w.qa + i] = (int32_t)std::min<int64_t>(P, r - (int64_t)i * P);
        for (const Run& x : runs[wi])
            if (x.dq != x.sq || x.ds != x.ss) changed[x.dq] = 1;
    }
    // the last page of a ragged window is also written when its unused
    // slots are zeroed, which happens only if its rows change anyway
    int32_t need = 0;
    for (const Window& w : win)
        for (int32_t i = 0; i < w.used; ++i)
            if (changed[w.qa + i] && alloc_.refcount(s->pages[w.qa + i]) > 1) ++need;
    if (need > alloc_.free_count()) return kNoPages;

    // commit
    std::vector<int32_t> page_at(s->pages);   // destination page of each page index
    for (const Window& w : win)
        for (int32_t i = 0; i < w.used; ++i) {
            const int32_t q = w.qa + i;
            if (changed[q] && alloc_.refcount(s->pages[q]) > 1) {
                page_at[q] = take_lowest();
                plan->cow_pages.push_back(page_at[q]);
            }
        }
    for (size_t wi = 0; wi < win.size(); ++wi) {
        const Window& w = win[wi];
        for (const Run& x : runs[wi]) {
            const bool fresh = page_at[x.dq] != s->pages[x.dq];
            if (!fresh && x.dq == x.sq && x.ds == x.ss) continue;  // rows stay where they are
            plan->moves.push_back({page_at[x.dq], x.ds, s->pages[x.sq], x.ss, x.n, (int32_t)wi});
            plan->moved_rows += x.n;
        }
        if (ragged && w.used > 0) {
            const int32_t q = w.qa + w.used - 1;
            const bool fresh = page_at[q] != s->pages[q];
            if ((changed[q] || fresh) && dest_fill[q] < P) {
                plan->moves.push_back({page_at[q], dest_fill[q], -1, 0, P - dest_fill[q], (int32_t)wi});
                plan->zeroed_rows += P - dest_fill[q];
            }
        }
    }
    // references: replaced originals and the pages that leave
    std::vector<int32_t> pages, fill;
    pages.reserve(np);
    fill.reserve(np);
    size_t wi = 0;
    for (int32_t q = 0; q < np;) {
        if (wi < win.size() && win[wi].qa == q) {
            const Window& w = win[wi];
            for (int32_t i = 0; i <= w.qb - w.qa; ++i) {
                const int32_t x = w.qa + i;
                if (i < w.used) {
                    if (page_at[x] != s->pages[x]) alloc_.drop_ref(s->pages[x]);
                    pages.push_back(page_at[x]);
                    fill.push_back(dest_fill[x]);
                } else if (alloc_.drop_ref(s->pages[x])) {
                    plan->freed.push_back(s->pages[x]);
                }
            }
            q = w.qb + 1;
            ++wi;
        } else {
            pages.push_back(s->pages[q]);
            fill.push_back(s->fill[q]);
            ++q;
        }
    }
    plan->new_pages = pages;
    plan->new_fill = fill;
    plan->n_new = (int32_t)(n - removed);
    plan->evicted = (int32_t)removed;
    plan->windows = ragged ? (int32_t)win.size() : 1;
    s->pages = std::move(pages);
    s->fill = std::move(fill);
    s->n = plan->n_new;
    s->version = g_version_counter++;
    return kOk;
}

void HostCache::undo_evict(int32_t h, const EvictPlan& plan) {
    Seq* s = seq_mut(h);
    if (!s || plan.n_new == plan.n_old) return;
    // every page of the old table gains its holder back before the new
    // table's pages lose theirs, so no page shared by both passes zero
    for (int32_t p : plan.old_pages) {
        if (alloc_.refcount(p) == 0) alloc_.take(p);
        else alloc_.add_ref(p);
    }
    for (int32_t p : plan.new_pages) alloc_.drop_ref(p);
    s->pages = plan.old_pages;
    s->fill = plan.old_fill;
    s->n = plan.n_old;
    s->version = g_version_counter++;
}

int HostCache::release(int32_t h, std::vector<int32_t>* freed) {
    Seq* s = seq_mut(h);
    if (!s) return kBadHandle;
    for (int32_t p : s->pages)
        if (alloc_.drop_ref(p) && freed) freed->push_back(p);
    s->pages.clear();
    s->n = 0;
    s->live = false;
    int32_t slot = h & 0xFFFFF;
    free_slots_.push_back(slot);
    return kOk;
}

void evict_tiles(const EvictPlan& p, int32_t tile_rows, std::vector<EvictTile>* tiles,
                 std::vector<EvictPiece>* pieces, std::vector<int32_t>* window_tile) {
    tiles->clear();
    pieces->clear();
    if (window_tile) window_tile->clear();
    EvictTile* open = nullptr;   // the tile being filled
    bool open_zero = false;
    int32_t window = -1;
    for (const EvictMove& m : p.moves) {
        const bool zero = m.src_page < 0;
        if (m.window != window) {
            // a new window starts a new tile
            window = m.window;
            open = nullptr;
            if (window_tile) window_tile->push_back((int32_t)tiles->size());
        }
        int32_t done = 0;
        while (done < m.n) {
            const int32_t dst_slot = m.dst_slot + done;
            // continue the open tile when this move extends it in place
            const bool cont = open && open_zero == zero && open->dst_page == m.dst_page &&
                              open->dst_slot + open->n_rows == dst_slot &&
                              open->n_rows < tile_rows;
            if (!cont) {
                tiles->push_back({m.dst_page, dst_slot, 0, (int32_t)pieces->size()});
                open = &tiles->back();
                open_zero = zero;
            }
            const int32_t k = std::min(m.n - done, tile_rows - open->n_rows);
            if (!zero) pieces->push_back({m.src_page, m.src_slot + done, k, open->n_rows});
            open->n_rows += k;
            done += k;
        }
    }
}

int32_t evict_tile_rows_for(int32_t P, int32_t D) {
    return std::min(P, std::max(8, 8192 / (2 * D)));
}

int32_t evict_stages_for(int64_t planes, int32_t num_sms) {
    return planes <= num_sms ? 6 : (planes <= 4LL * num_sms ? 3 : 4);
}

void evict_chunks(const std::vector<int32_t>& window_tile, int32_t n_tiles, int32_t max_chunks,
                  int32_t min_tiles, std::vector<int32_t>* chunk) {
    chunk->assign(1, 0);
    const int32_t nw = (int32_t)window_tile.size();
    int32_t want = std::min<int32_t>(max_chunks, nw);
    if (min_tiles > 0) want = std::min<int32_t>(want, std::max<int32_t>(1, n_tiles / min_tiles));
    // cut at the window start nearest each even share of the tiles
    int32_t w = 1;
    for (int32_t c = 1; c < want && w < nw; ++c) {
        const int64_t target = (int64_t)n_tiles * c / want;
        while (w < nw && window_tile[w] < target) ++w;
        if (w < nw && window_tile[w] > chunk->back()) chunk->push_back(window_tile[w++]);
    }
    chunk->push_back(n_tiles);
}

// ---------------------------------------------------------------------------
// decode planning

int plan_decode(const HostCache& c, const int32_t* handles, int32_t n_seqs,
                int32_t n_ctas, DecodePlanHost* out) {
    *out = DecodePlanHost();
    const Geometry& g = c.geom();
    if (n_seqs < 1 || !handles || n_ctas < 1) return kInvalidArg;
    std::vector<const Seq*> ss(n_seqs);
    bool ragged = false;
    for (int32_t i = 0; i < n_seqs; ++i) {
        ss[i] = c.seq(handles[i]);
        if (!ss[i]) return kBadHandle;
        if (ss[i]->n < 1) return kInvalidArg;
        for (int32_t j = 0; j < i; ++j)
            if (ss[j] == ss[i]) return kInvalidArg;
        out->logical_tokens += ss[i]->n;
        ragged = ragged || has_partial_pages(*ss[i], g.P);
    }
    const int32_t P = g.P;
    const int32_t max_grp = kRowsPerTile / g.G();

    // Group sequences holding the same physical page, with the same fill, at
    // the same page index into shared runs (depth-first over the prefix tree
    // of pages).  (Two holders of one page can see different fills after a
    // ragged eviction of one of them; they read that page separately.)
    // Every segment also records its family: the subtree of one first page
    // (a request, its forks and whatever they added).
    struct Work {
        std::vector<int32_t> members;
        int32_t q;
        int32_t fam;  // -1 at the root
    };
    std::vector<Work> stack;
    std::vector<int32_t> seg_fam;
    int32_t n_fam = 0;
    {
        Work root;
        for (int32_t i = 0; i < n_seqs; ++i) root.members.push_back(i);
        root.q = 0;
        root.fam = -1;
        stack.push_back(std::move(root));
    }
    while (!stack.empty()) {
        Work w = std::move(stack.back());
        stack.pop_back();
        // partition by the page held at w.q (first-seen order)
        std::vector<std::vector<int32_t>> parts;
        std::vector<std::pair<int32_t, int32_t>> part_page;  // (page, fill)
        for (int32_t i : w.members) {
            if ((int32_t)ss[i]->pages.size() <= w.q) continue;
            const std::pair<int32_t, int32_t> key{ss[i]->pages[w.q], ss[i]->fill[w.q]};
            size_t k = 0;
            while (k < part_page.size() && part_page[k] != key) ++k;
            if (k == part_page.size()) {
                part_page.push_back(key);
                parts.emplace_back();
            }
            parts[k].push_back(i);
        }
        // process parts in order: push in reverse so the first is handled first
        std::vector<Work> next;
        for (auto& part : parts) {
            const int32_t fam = w.fam >= 0 ? w.fam : n_fam++;
            const int32_t q0 = w.q;
            int32_t q_end = q0 + 1;
            const Seq* lead = ss[part[0]];
            for (;;) {
                if (q_end >= (int32_t)lead->pages.size()) break;
                bool same = true;
                for (int32_t i : part) {
                    if ((int32_t)ss[i]->pages.size() <= q_end ||
                        ss[i]->pages[q_end] != lead->pages[q_end] ||
                        ss[i]->fill[q_end] != lead->fill[q_end]) {
                        same = false;
                        break;
                    }
                }
                if (!same) break;
                ++q_end;
            }
            for (size_t b = 0; b < part.size(); b += max_grp) {
                DecodeSeg seg;
                std::memset(&seg, 0, sizeof seg);
                seg.page_off = (int32_t)out->page_ids.size();
                seg.n_pages = q_end - q0;
                seg.n_grp = (int32_t)std::min<size_t>(max_grp, part.size() - b);
                seg.n_tok = 0;
                seg.q0 = q0;
                for (int32_t j = 0; j < seg.n_grp; ++j) {
                    int32_t i = part[b + j];
                    // slot-space limit of this member inside the run
                    int64_t lim = std::min<int64_t>((int64_t)slot_end(*ss[i], P) - (int64_t)q0 * P,
                                                    (int64_t)seg.n_pages * P);
                    seg.grp_seq[j] = i;
                    seg.grp_lim[j] = (int32_t)lim;
                    seg.n_tok = std::max(seg.n_tok, (int32_t)lim);
                    if ((int32_t)ss[i]->pages.size() == q_end) seg.tail |= 1 << j;
                }
                const Seq* sl = ss[part[b]];
                for (int32_t q = q0; q < q_end; ++q) {
                    out->page_ids.push_back(sl->pages[q]);
                    if (ragged) out->page_fill.push_back(sl->fill[q]);
                    // rows read: the filled slots below the run's limit
                    const int64_t below = (int64_t)seg.n_tok - (int64_t)(q - q0) * P;
                    out->unique_tokens += std::max<int64_t>(0, std::min<int64_t>(sl->fill[q], below));
                }
                out->segs.push_back(seg);
                seg_fam.push_back(fam);
            }
            Work nw;
            for (int32_t i : part)
                if ((int32_t)ss[i]->pages.size() > q_end) nw.members.push_back(i);
            nw.q = q_end;
            nw.fam = fam;
            if (!nw.members.empty()) next.push_back(std::move(nw));
        }
        for (auto it = next.rbegin(); it != next.rend(); ++it) stack.push_back(std::move(*it));
    }

    // (segment, head) units and an even split of their cost over the
    // persistent CTAs.  On the cost line a unit occupies kUnitCostStages
    // (its start-up) followed by its stages; an item is the overlap of a
    // CTA's share with a unit's stages.  Units go family by family, head by
    // head, each family's segments in tree order: a fork's own short tail
    // follows the shared prefix of the same head, so it lands in the CTA that
    // finishes that prefix instead of in a pile of tails at the end of the
    // line (whose one CTA would then merge every fork's rows alone).
    const int32_t n_segs = (int32_t)out->segs.size();
    std::vector<int32_t> by_fam(n_segs);
    for (int32_t s = 0; s < n_segs; ++s) by_fam[s] = s;
    std::stable_sort(by_fam.begin(), by_fam.end(),
                     [&](int32_t x, int32_t y) { return seg_fam[x] < seg_fam[y]; });
    std::vector<int32_t> unit_seg, unit_head;
    for (int32_t b = 0; b < n_segs;) {
        int32_t e = b;
        while (e < n_segs && seg_fam[by_fam[e]] == seg_fam[by_fam[b]]) ++e;
        for (int32_t h = 0; h < g.Hkv; ++h)
            for (int32_t x = b; x < e; ++x) {
                unit_seg.push_back(by_fam[x]);
                unit_head.push_back(h);
            }
        b = e;
    }
    std::vector<int64_t> unit_start;  // where the unit's stages begin on the cost line
    std::vector<int64_t> unit_end;
    int64_t total = 0;
    for (size_t v = 0; v < unit_seg.size(); ++v) {
        total += kUnitCostStages;
        unit_start.push_back(total);
        total += ceil_div(out->segs[unit_seg[v]].n_tok, kStageTokens);
        unit_end.push_back(total);
    }
    const int64_t n_units = (int64_t)unit_start.size();
    const int32_t ctas = (int32_t)std::min<int64_t>(n_ctas, total - n_units * kUnitCostStages);
    out->n_ctas = ctas;
    out->cta_begin.resize(ctas + 1);
    int64_t u = 0;
    for (int32_t cta = 0; cta < ctas; ++cta) {
        const int64_t b = total * cta / ctas, e = total * (cta + 1) / ctas;
        out->cta_begin[cta] = (int32_t)out->items.size();
        while (u < n_units && unit_end[u] <= b) ++u;
        for (int64_t v = u; v < n_units && unit_start[v] - kUnitCostStages < e; ++v) {
            const int64_t lo = std::max(b, unit_start[v]), hi = std::min(e, unit_end[v]);
            if (hi <= lo) continue;
            DecodeItem it;
            std::memset(&it, 0, sizeof it);
            it.seg = unit_seg[v];
            it.head = unit_head[v];
            it.s0 = (int32_t)(lo - unit_start[v]);
            it.s1 = (int32_t)(hi - unit_start[v]);
            out->items.push_back(it);
        }
    }
    out->cta_begin[ctas] = (int32_t)out->items.size();

    // partial entries per (sequence, KV head), contiguous, in item order
    const int32_t keys = n_seqs * g.Hkv;
    out->comb_off.assign(keys + 1, 0);
    for (const DecodeItem& it : out->items) {
        const DecodeSeg& s = out->segs[it.seg];
        for (int32_t j = 0; j < s.n_grp; ++j) ++out->comb_off[s.grp_seq[j] * g.Hkv + it.head + 1];
    }
    for (int32_t k = 0; k < keys; ++k) {
        // the kernel counts a run's entries in 16 bits
        if (out->comb_off[k + 1] > kMaxRunEntries) return kCapacity;
        out->comb_off[k + 1] += out->comb_off[k];
    }
    std::vector<int32_t> fill(out->comb_off.begin(), out->comb_off.end() - 1);
    for (DecodeItem& it : out->items) {
        const DecodeSeg& s = out->segs[it.seg];
        it.sole = 0;
        for (int32_t j = 0; j < s.n_grp; ++j) {
            const int32_t key = s.grp_seq[j] * g.Hkv + it.head;
            it.ent[j] = fill[key]++;
            if (out->comb_off[key + 1] - out->comb_off[key] == 1) it.sole |= 1 << j;
        }
    }
    return kOk;
}

static int64_t align16(int64_t x) { return (x + 15) & ~int64_t(15); }

DecodePlanLayout plan_layout(const DecodePlanHost& p, int32_t n_seqs, int32_t Hkv) {
    DecodePlanLayout L;
    L.n_segs = (int32_t)p.segs.size();
    L.n_items = (int32_t)p.items.size();
    L.n_ctas = p.n_ctas;
    L.n_page_ids = (int32_t)p.page_ids.size();
    L.n_comb_keys = n_seqs * Hkv;
    L.n_comb_ent = p.comb_off.empty() ? 0 : p.comb_off.back();
    int64_t o = 0;
    L.segs = o;      o = align16(o + sizeof(DecodeSeg) * L.n_segs);
    L.items = o;     o = align16(o + sizeof(DecodeItem) * L.n_items);
    L.cta_begin = o; o = align16(o + sizeof(int32_t) * (L.n_ctas + 1));
    L.page_ids = o;  o = align16(o + sizeof(int32_t) * L.n_page_ids);
    L.comb_off = o;  o = align16(o + sizeof(int32_t) * (L.n_comb_keys + 1));
    L.arrive = o;    o = align16(o + sizeof(uint32_t) * L.n_comb_keys);
    if (!p.page_fill.empty()) {
        L.page_fill = o; o = align16(o + sizeof(int32_t) * L.n_page_ids);
    } else {
        L.page_fill = -1;
    }
    L.total = o;
    return L;
}

void plan_serialize(const DecodePlanHost& p, const DecodePlanLayout& L, uint8_t* dst) {
    std::memset(dst, 0, L.total);
    std::memcpy(dst + L.segs, p.segs.data(), sizeof(DecodeSeg) * L.n_segs);
    std::memcpy(dst + L.items, p.items.data(), sizeof(DecodeItem) * L.n_items);
    std::memcpy(dst + L.cta_begin, p.cta_begin.data(), sizeof(int32_t) * (L.n_ctas + 1));
    std::memcpy(dst + L.page_ids, p.page_ids.data(), sizeof(int32_t) * L.n_page_ids);
    std::memcpy(dst + L.comb_off, p.comb_off.data(), sizeof(int32_t) * (L.n_comb_keys + 1));
    if (L.page_fill >= 0)
        std::memcpy(dst + L.page_fill, p.page_fill.data(), sizeof(int32_t) * L.n_page_ids);
}

// ---------------------------------------------------------------------------
// Masked prefill planning.  Visibility of key j to the query at position p:
// j <= p (causal) and j in no span (Algorithm 2: a closed cursor's tokens are
// masked for every later token).  The kernel applies the causal part; the
// plan carries the span part as one bit per key, per key tile.
int plan_prefill(const Geometry& g, int32_t n, int32_t n_q, const int32_t* starts,
                 const int32_t* ends, int32_t n_spans, int32_t target_ctas,
                 PrefillPlanHost* out, const int32_t* pages) {
    *out = PrefillPlanHost();
    if (n < 1 || n_q < 1 || n_q > n) return kInvalidArg;
    std::vector<std::pair<int32_t, int32_t>> sp;
    int rc = sorted_spans(n, starts, ends, n_spans, &sp);
    if (rc != kOk) return rc;
    const int32_t n_kt = ceil_div(n, kPrefillKeys);
    std::vector<uint32_t> vis((size_t)n_kt * 4, 0);
    for (int32_t j = 0; j < n; j += 32) {
        const int32_t m = std::min(32, n - j);
        vis[j >> 5] = m == 32 ? 0xffffffffu : ((1u << m) - 1u);
    }
    for (auto& ab : sp)
        for (int32_t j = ab.first; j < ab.second; ++j) vis[j >> 5] &= ~(1u << (j & 31));
    auto box_full = [&](int32_t b) {   // 64 keys from b, all in the sequence and visible
        return vis[(b >> 5)] == 0xffffffffu && vis[(b >> 5) + 1] == 0xffffffffu;
    };
    if (g.P >= 64) {
        // the 64-key boxes with a visible key, two by two
        std::vector<int32_t> boxes;
        for (int32_t b = 0; b < n; b += 64)
            if (vis[b >> 5] | vis[(b >> 5) + 1]) boxes.push_back(b);
        for (size_t i = 0; i < boxes.size(); i += 2) {
            PrefillTile tile{};
            tile.key0 = boxes[i];
            tile.key0b = i + 1 < boxes.size() ? boxes[i + 1] : kPrefillNoKeys;
            tile.vis[0] = vis[tile.key0 >> 5];
            tile.vis[1] = vis[(tile.key0 >> 5) + 1];
            if (i + 1 < boxes.size()) {
                tile.vis[2] = vis[tile.key0b >> 5];
                tile.vis[3] = vis[(tile.key0b >> 5) + 1];
            }
            const bool full = i + 1 < boxes.size() && box_full(tile.key0) && box_full(tile.key0b);
            tile.flags = full ? kPrefillTileFull : 0;
            out->tiles.push_back(tile);
        }
    } else {
        for (int32_t t = 0; t < n_kt; ++t) {
            PrefillTile tile{};
            tile.key0 = t * kPrefillKeys;
            tile.key0b = tile.key0 + 64;
            bool any = false, full = true;
            for (int w = 0; w < 4; ++w) {
                tile.vis[w] = vis[(size_t)t * 4 + w];
                any |= tile.vis[w] != 0;
                full &= tile.vis[w] == 0xffffffffu;
            }
            if (!any) continue;
            tile.flags = full ? kPrefillTileFull : 0;
            out->tiles.push_back(tile);
        }
    }
    // the page of each TMA box (min(P, 64) rows) of each listed tile: the
    // first half's boxes from key0, the second half's from key0b
    const int32_t br = std::min(g.P, 64);
    out->n_pieces = kPrefillKeys / br;
    if (pages) {
        const int32_t half = out->n_pieces / 2;
        out->tile_pages.resize(out->tiles.size() * out->n_pieces);
        for (size_t t = 0; t < out->tiles.size(); ++t)
            for (int32_t i = 0; i < out->n_pieces; ++i) {
                const int64_t key = i < half ? (int64_t)out->tiles[t].key0 + i * br
                                             : (int64_t)out->tiles[t].key0b + (i - half) * br;
                out->tile_pages[t * out->n_pieces + i] = key < n ? pages[key / g.P] : -1;
            }
    }
    // visible keys of each query: the visible keys among 0 .. p
    int64_t seen = 0, pairs = 0;
    const int32_t q0 = n - n_q;
    for (int32_t j = 0; j < n; ++j) {
        seen += (vis[j >> 5] >> (j & 31)) & 1u;
        if (j >= q0) pairs += seen;
    }
    out->visible_pairs = pairs;
    out->n = n;
    out->n_q = n_q;
    out->BP = kPrefillRows / g.G();
    const int32_t span = out->BP * kPrefillQTiles;  // query positions per CTA
    out->n_qt = ceil_div(n_q, span);
    // each CTA tile reaches the key tiles up to its last query position
    out->qt_tiles.resize(out->n_qt);
    for (int32_t qt = 0, t = 0; qt < out->n_qt; ++qt) {
        const int32_t p_last = q0 + std::min((qt + 1) * span, n_q) - 1;
        while (t < (int32_t)out->tiles.size() && out->tiles[t].key0 <= p_last) ++t;
        out->qt_tiles[qt] = t;
    }
    const int64_t units = (int64_t)out->n_qt * g.Hkv;
    const int32_t n_tiles = (int32_t)out->tiles.size();
    // Split each CTA tile's key range when there are too few CTA tiles to
    // fill the GPU: pick the split that minimises the estimated makespan,
    // waves x (key tiles per CTA + a fixed per-CTA cost), CTAs running
    // `target_ctas` at a time.
    int32_t split = 1;
    if (units < target_ctas && n_tiles > 0 && target_ctas > 0) {
        constexpr int32_t kMaxSplit = 64;
        constexpr double kCtaCost = 4.0;  // prologue + epilogue, in key tiles
        double avg = 0;
        for (int32_t c : out->qt_tiles) avg += c;
        avg /= std::max<int32_t>(1, out->n_qt);
        double best = 1e300;
        for (int32_t sp = 1; sp <= kMaxSplit && sp <= n_tiles; ++sp) {
            const int64_t ctas = units * sp;
            const int64_t waves = (ctas + target_ctas - 1) / target_ctas;
            const double cost = (double)waves * (avg / sp + kCtaCost);
            if (cost < best - 1e-9) {
                best = cost;
                split = sp;
            }
        }
    }
    out->n_split = split;
    return kOk;
}

int prefill_slot_spans(const Seq& s, int32_t P, int32_t n_q, const int32_t* starts,
                       const int32_t* ends, int32_t n_spans, std::vector<int32_t>* a_out,
                       std::vector<int32_t>* b_out, int32_t* n_slots) {
    a_out->clear();
    b_out->clear();
    std::vector<std::pair<int32_t, int32_t>> sp;
    int rc = sorted_spans(s.n, starts, ends, n_spans, &sp);
    if (rc != kOk) return rc;
    const int32_t np = (int32_t)s.pages.size();
    *n_slots = slot_end(s, P);
    if (n_q < 1 || n_q > s.n) return kInvalidArg;
    std::vector<int32_t> start(np + 1, 0);
    for (int32_t q = 0; q < np; ++q) start[q + 1] = start[q] + s.fill[q];
    // the queries must sit in consecutive slots: the slot of row n - n_q is
    // n_slots - n_q exactly when no unused slot lies between
    {
        const int32_t j = s.n - n_q;
        int32_t q = (int32_t)(std::upper_bound(start.begin(), start.end(), j) - start.begin()) - 1;
        if (q * P + (j - start[q]) != *n_slots - n_q) return kUnsupported;
    }
    // spans and unused slots, in slot order, adjacent ranges merged
    std::vector<std::pair<int32_t, int32_t>> r;
    auto add = [&](int32_t a, int32_t b) {
        if (a >= b) return;
        if (!r.empty() && r.back().second == a) r.back().second = b;
        else r.push_back({a, b});
    };
    size_t k = 0;
    for (int32_t q = 0; q < np; ++q) {
        // the span parts inside page q
        while (k < sp.size() && sp[k].second <= start[q]) ++k;
        for (size_t x = k; x < sp.size() && sp[x].first < start[q + 1]; ++x) {
            const int32_t a = std::max(sp[x].first, start[q]), b = std::min(sp[x].second, start[q + 1]);
            add(q * P + (a - start[q]), q * P + (b - start[q]));
        }
        if (q + 1 < np) add(q * P + s.fill[q], (q + 1) * P);
    }
    for (auto& ab : r) {
        a_out->push_back(ab.first);
        b_out->push_back(ab.second);
    }
    return kOk;
}

}  // namespace sq
