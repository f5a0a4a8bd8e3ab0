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
    int32_t n = ps->n;
    const int64_t next_pos = ps->next_pos;
    void* st = ps->last_stream;
    int rc = seq_new(child);
    if (rc != kOk) return rc;
    Seq* cs = seq_mut(*child);
    cs->pages = std::move(pages);
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
    if (n_new == 0) return kOk;
    if ((int64_t)n + n_new >= (1LL << 31)) return kCapacity;
    const int32_t new_np = ceil_div((int64_t)n + n_new, P);
    if (new_np > g_.max_pages_per_seq) return kCapacity;
    const bool cow = (n % P != 0) && alloc_.refcount(s->pages.back()) > 1;
    const int32_t need = (cow ? 1 : 0) + new_np - (int32_t)s->pages.size();
    if (need > alloc_.free_count()) return kNoPages;

    if (cow) {
        int32_t old = s->pages.back();
        int32_t fresh = take_lowest();
        alloc_.drop_ref(old);  // was > 1: stays held by the other sequences
        s->pages.back() = fresh;
        plan->cow = true;
        plan->cow_old = old;
        plan->cow_new = fresh;
        plan->cow_rows = n % P;
        plan->taken.push_back(fresh);
    }
    while ((int32_t)s->pages.size() < new_np) {
        int32_t p = take_lowest();
        s->pages.push_back(p);
        plan->taken.push_back(p);
    }
    plan->first_page_index = n / P;
    plan->pages.assign(s->pages.begin() + n / P, s->pages.end());
    s->n = n + n_new;
    s->next_pos += n_new;
    s->version = g_version_counter++;
    return kOk;
}

void HostCache::undo_append(int32_t h, const AppendPlan& plan) {
    Seq* s = seq_mut(h);
    if (!s || plan.n_new == 0) return;
    const int32_t old_np = ceil_div(plan.n0, g_.P);
    while ((int32_t)s->pages.size() > old_np) {
        alloc_.drop_ref(s->pages.back());
        s->pages.pop_back();
    }
    if (plan.cow) {
        alloc_.drop_ref(plan.cow_new);
        alloc_.add_ref(plan.cow_old);
        s->pages.back() = plan.cow_old;
    }
    s->n = plan.n0;
    s->next_pos -= plan.n_new;
    s->version = g_version_counter++;
}

int HostCache::evict(int32_t h, const int32_t* starts, const int32_t* ends,
                     int32_t n_spans, EvictPlan* plan) {
    *plan = EvictPlan();
    Seq* s = seq_mut(h);
    if (!s) return kBadHandle;
    if (n_spans < 0) return kInvalidArg;
    const int32_t n = s->n;
    const int32_t P = g_.P;
    plan->n_old = n;
    plan->n_new = n;
    plan->first_row = n;
    plan->old_pages = s->pages;
    plan->new_pages = s->pages;
    if (n_spans == 0) return kOk;
    if (!starts || !ends) return kInvalidArg;

    std::vector<std::pair<int32_t, int32_t>> sp;
    int rc = sorted_spans(n, starts, ends, n_spans, &sp);
    if (rc != kOk) return rc;
    int64_t removed = 0;
    for (auto& ab : sp) removed += ab.second - ab.first;
    // kept runs
    int32_t cur = 0, dst = 0;
    for (auto& ab : sp) {
        if (ab.first > cur) {
            plan->run_dst.push_back(dst);
            plan->run_src.push_back(cur);
            plan->run_len.push_back(ab.first - cur);
            dst += ab.first - cur;
        }
        cur = ab.second;
    }
    if (n > cur) {
        plan->run_dst.push_back(dst);
        plan->run_src.push_back(cur);
        plan->run_len.push_back(n - cur);
        dst += n - cur;
    }
    const int32_t n2 = (int32_t)(n - removed);
    const int32_t new_np = ceil_div(n2, P);
    const int32_t a0 = sp[0].first;
    const int32_t qc = a0 / P;
    const bool any_change = n2 > a0;  // some kept row moves
    // copy-on-write needs
    int32_t need = 0;
    if (any_change)
        for (int32_t q = qc; q < new_np; ++q)
            if (alloc_.refcount(s->pages[q]) > 1) ++need;
    if (need > alloc_.free_count()) return kNoPages;

    // commit
    std::vector<int32_t> new_pages(s->pages.begin(), s->pages.begin() + new_np);
    int64_t moved = 0;
    if (any_change) {
        for (int32_t q = qc; q < new_np; ++q) {
            const int32_t row_end = std::min<int64_t>((int64_t)q * P + P, n2);
            if (alloc_.refcount(s->pages[q]) > 1) {
                new_pages[q] = take_lowest();
                plan->cow_pages.push_back(new_pages[q]);
                moved += row_end - (int64_t)q * P;
            } else {
                moved += row_end - std::max<int64_t>((int64_t)q * P, a0);
            }
        }
        for (int32_t q = qc; q < new_np; ++q)
            if (new_pages[q] != s->pages[q]) alloc_.drop_ref(s->pages[q]);
    }
    for (size_t q = new_np; q < s->pages.size(); ++q)
        if (alloc_.drop_ref(s->pages[q])) plan->freed.push_back(s->pages[q]);
    plan->new_pages = new_pages;
    plan->n_new = n2;
    plan->first_row = any_change ? qc * P : n2;
    plan->moved_rows = moved;
    plan->evicted = (int32_t)removed;
    s->pages = std::move(new_pages);
    s->n = n2;
    s->version = g_version_counter++;
    return kOk;
}

void HostCache::undo_evict(int32_t h, const EvictPlan& plan) {
    Seq* s = seq_mut(h);
    if (!s || plan.n_new == plan.n_old) return;
    // trailing pages back
    for (size_t q = plan.new_pages.size(); q < plan.old_pages.size(); ++q) {
        int32_t p = plan.old_pages[q];
        if (alloc_.refcount(p) == 0) alloc_.take(p);
        else alloc_.add_ref(p);
    }
    for (size_t q = 0; q < plan.new_pages.size(); ++q) {
        if (plan.new_pages[q] != plan.old_pages[q]) {
            alloc_.drop_ref(plan.new_pages[q]);
            alloc_.add_ref(plan.old_pages[q]);
        }
    }
    s->pages = plan.old_pages;
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

void evict_tiles(const EvictPlan& p, int32_t P, int32_t tile_rows,
                 std::vector<EvictTile>* tiles, std::vector<EvictPiece>* pieces) {
    tiles->clear();
    pieces->clear();
    if (p.first_row >= p.n_new) return;
    size_t r = 0;  // current kept run (monotone in the destination row)
    const int32_t first_q = p.first_row / P;
    const int32_t new_np = (int32_t)p.new_pages.size();
    for (int32_t q = first_q; q < new_np; ++q) {
        const int32_t page_begin = q * P;
        const int32_t row_end = std::min<int64_t>((int64_t)page_begin + P, p.n_new);
        const bool fresh = p.new_pages[q] != p.old_pages[q];
        int32_t row = page_begin;
        if (!fresh) {
            // skip destination rows that keep their row (kept[j] == j)
            while (row < row_end) {
                while (r + 1 < p.run_dst.size() && p.run_dst[r + 1] <= row) ++r;
                const int32_t src = p.run_src[r] + (row - p.run_dst[r]);
                if (src != row) break;
                // the whole rest of this run keeps its rows
                row = std::min<int32_t>(row_end, p.run_dst[r] + p.run_len[r]);
            }
        }
        while (row < row_end) {
            const int32_t t_end = std::min(row_end, row + tile_rows);
            EvictTile t;
            t.dst_page = p.new_pages[q];
            t.dst_slot = row - page_begin;
            t.n_rows = t_end - row;
            t.piece_begin = (int32_t)pieces->size();
            int32_t j = row;
            while (j < t_end) {
                while (r + 1 < p.run_dst.size() && p.run_dst[r + 1] <= j) ++r;
                const int32_t src = p.run_src[r] + (j - p.run_dst[r]);
                const int32_t run_left = p.run_dst[r] + p.run_len[r] - j;
                const int32_t page_left = P - src % P;
                const int32_t n = std::min({t_end - j, run_left, page_left});
                EvictPiece pc;
                pc.src_page = p.old_pages[src / P];
                pc.src_slot = src % P;
                pc.n_rows = n;
                pc.dst_row = j - row;
                pieces->push_back(pc);
                j += n;
            }
            tiles->push_back(t);
            row = t_end;
        }
    }
}

// ---------------------------------------------------------------------------
// decode planning

int plan_decode(const HostCache& c, const int32_t* handles, int32_t n_seqs,
                int32_t n_ctas, DecodePlanHost* out) {
    *out = DecodePlanHost();
    const Geometry& g = c.geom();
    if (n_seqs < 1 || !handles || n_ctas < 1) return kInvalidArg;
    std::vector<const Seq*> ss(n_seqs);
    for (int32_t i = 0; i < n_seqs; ++i) {
        ss[i] = c.seq(handles[i]);
        if (!ss[i]) return kBadHandle;
        if (ss[i]->n < 1) return kInvalidArg;
        for (int32_t j = 0; j < i; ++j)
            if (ss[j] == ss[i]) return kInvalidArg;
        out->logical_tokens += ss[i]->n;
    }
    const int32_t P = g.P;
    const int32_t max_grp = kRowsPerTile / g.G();

    // Group sequences holding the same physical page at the same logical
    // index into shared runs (depth-first over the prefix tree of pages).
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
        std::vector<int32_t> part_page;
        for (int32_t i : w.members) {
            if ((int32_t)ss[i]->pages.size() <= w.q) continue;
            int32_t p = ss[i]->pages[w.q];
            size_t k = 0;
            while (k < part_page.size() && part_page[k] != p) ++k;
            if (k == part_page.size()) {
                part_page.push_back(p);
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
                        ss[i]->pages[q_end] != lead->pages[q_end]) {
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
                for (int32_t j = 0; j < seg.n_grp; ++j) {
                    int32_t i = part[b + j];
                    int64_t lim = std::min<int64_t>((int64_t)ss[i]->n - (int64_t)q0 * P,
                                                    (int64_t)seg.n_pages * P);
                    seg.grp_seq[j] = i;
                    seg.grp_lim[j] = (int32_t)lim;
                    seg.n_tok = std::max(seg.n_tok, (int32_t)lim);
                }
                const Seq* sl = ss[part[b]];
                for (int32_t q = q0; q < q_end; ++q) out->page_ids.push_back(sl->pages[q]);
                out->unique_tokens += seg.n_tok;
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
    for (int32_t k = 0; k < keys; ++k) out->comb_off[k + 1] += out->comb_off[k];
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
    for (int32_t t = 0; t < n_kt; ++t) {
        PrefillTile tile{};
        tile.key0 = t * kPrefillKeys;
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
    // the page of each TMA box (min(P, 64) rows) of each listed tile
    const int32_t br = std::min(g.P, 64);
    out->n_pieces = kPrefillKeys / br;
    if (pages) {
        out->tile_pages.resize(out->tiles.size() * out->n_pieces);
        for (size_t t = 0; t < out->tiles.size(); ++t)
            for (int32_t i = 0; i < out->n_pieces; ++i) {
                const int32_t key = out->tiles[t].key0 + i * br;
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

}  // namespace sq
