// Host-side state of the paged KV cache: page allocator, reference counts,
// sequence table and page tables, and the planners for append, eviction and
// decode.  Plain C++17, no CUDA: the device side consumes the plans.
//
// The rules (Sec. 3.1 and Algorithm 1 for fork / append / clear_kv /
// release; Sec. 3.4 for prefix sharing without duplication) are fixed as:
//   * lowest free page id first;
//   * fork copies the page list, +1 reference per page, no K/V copy;
//   * append: copy-on-write of a shared partial last page, then new pages in
//     increasing logical order;
//   * evict: a destination page whose rows change and that is shared is
//     replaced by a fresh page (increasing logical order), others are
//     compacted in place; pages past the new end lose a reference;
//   * release: every page loses a reference.
//
// Page fills: each page of a sequence holds `fill` rows (1 .. P) in its
// first slots; the logical rows are the pages' filled slots in order.  All
// pages are full but the last (the dense layout, logical j in slot j % P of
// pages[j / P]) unless a ragged eviction left partial pages: it packs only
// the runs of pages the spans touch (windows), each from slot 0 of its first
// page, drops the window pages it no longer needs by remapping, and leaves
// every other page as it was.  Kernels address rows in SLOT SPACE, position
// q * P + slot for slot `slot` of page index q, which keeps the logical
// order; a sequence's slot-space end is (pages - 1) * P + last fill.
#pragma once

#include <stdint.h>

#include <utility>
#include <vector>

#include "plan.hpp"

namespace sq {

enum Status : int {
    kOk = 0,
    kInvalidArg = -1,
    kBadHandle = -2,
    kNoPages = -3,
    kCapacity = -4,
    kCuda = -5,
    kDevice = -6,
    kDeviceTimeout = -7,
    kUnsupported = -8,
    kNoMemory = -9,
};

struct Geometry {
    int32_t L = 0, Hq = 0, Hkv = 0, D = 0, P = 0;
    int32_t num_pages = 0, max_seqs = 0, max_pages_per_seq = 0;
    int32_t G() const { return Hq / Hkv; }
    // K+V bytes of one token of one layer
    int64_t token_layer_bytes() const { return 2LL * Hkv * D * 2; }
};

// Validates a geometry against what the kernels handle.
int check_geometry(const Geometry& g);

// Checks half-open spans against a sequence of n tokens (each non-empty,
// inside [0, n), no two overlapping; any order) and returns them sorted.
int sorted_spans(int32_t n, const int32_t* starts, const int32_t* ends, int32_t n_spans,
                 std::vector<std::pair<int32_t, int32_t>>* out);

class PageAllocator {
  public:
    explicit PageAllocator(int32_t n = 0);
    int32_t size() const { return (int32_t)ref_.size(); }
    int32_t free_count() const { return free_count_; }
    int32_t refcount(int32_t p) const { return ref_[p]; }
    // The lowest free page id, -1 if none.
    int32_t lowest_free() const;
    // Take a free page (reference count 0 -> 1).
    void take(int32_t p);
    void add_ref(int32_t p) { ++ref_[p]; }
    // Drop one reference; true if the page became free.
    bool drop_ref(int32_t p);

  private:
    std::vector<int32_t> ref_;
    std::vector<uint64_t> free_bits_;  // bit set = free
    int32_t free_count_ = 0;
    mutable int32_t hint_ = 0;         // no free page below word hint_
};

struct Seq {
    bool live = false;
    uint32_t gen = 0;
    int32_t n = 0;
    std::vector<int32_t> pages;
    std::vector<int32_t> fill;  // rows held by each page, 1 .. P (sum = n)
    uint64_t version = 0;  // bumped by every change of n or pages
    // position of the next token: tokens ever appended (a fork starts from its
    // parent's); eviction does not lower it, since kept keys keep the rotary
    // phase of their original positions
    int64_t next_pos = 0;
    void* last_stream = nullptr;
};

// Slot-space end of a sequence: (pages - 1) * P + last fill (0 when empty).
inline int32_t slot_end(const Seq& s, int32_t P) {
    return s.pages.empty() ? 0 : ((int32_t)s.pages.size() - 1) * P + s.fill.back();
}
// True when some page other than the last holds fewer than P rows.
bool has_partial_pages(const Seq& s, int32_t P);

struct AppendPlan {
    int32_t n0 = 0, n_new = 0;
    int32_t pos0 = 0;        // slot-space position of the first new row
    int32_t last_fill0 = 0;  // fill of the last page before (0: no page)
    bool cow = false;
    int32_t cow_old = -1, cow_new = -1, cow_rows = 0;
    int32_t first_page_index = 0;  // logical index of the page holding n0
    std::vector<int32_t> pages;    // page ids for logical pages first_page_index ..
    std::vector<int32_t> taken;    // pages newly taken (cow page first)
};

// One contiguous piece of an eviction's row movement: n rows from slots
// src_slot .. of page src_page to slots dst_slot .. of page dst_page, or n
// zero rows when src_page is -1.
struct EvictMove {
    int32_t dst_page, dst_slot, src_page, src_slot, n;
    int32_t window;   // the window (run of packed pages) the move belongs to
};

struct EvictPlan {
    int32_t n_old = 0, n_new = 0;
    bool ragged = false;
    std::vector<int32_t> old_pages, old_fill;   // page table before
    std::vector<int32_t> new_pages, new_fill;   // page table after
    // Row movement in increasing destination (slot-space) order.  Every
    // source of a move lies at a slot-space position >= its destination's,
    // inside the same window, so performing the moves in order (each one's
    // reads before its writes) compacts in place.
    std::vector<EvictMove> moves;
    std::vector<int32_t> cow_pages;    // fresh pages taken (increasing logical page)
    std::vector<int32_t> freed;        // pages whose count reached zero
    int64_t moved_rows = 0;            // rows copied
    int64_t zeroed_rows = 0;           // unused slots set to zero (ragged windows)
    int32_t evicted = 0;
    int32_t windows = 0;               // runs of pages packed
};

class HostCache {
  public:
    explicit HostCache(const Geometry& g);
    const Geometry& geom() const { return g_; }
    const PageAllocator& alloc() const { return alloc_; }

    int seq_new(int32_t* handle);
    int fork(int32_t parent, int32_t* child);
    // Plans and commits an append (host state updated).  `undo_append`
    // restores the state if the device work cannot be enqueued.
    int append(int32_t h, int32_t n_new, AppendPlan* plan);
    void undo_append(int32_t h, const AppendPlan& plan);
    // Validates spans, plans and commits an eviction: dense (the kept rows
    // packed into full pages) or ragged (only the touched windows packed).
    int evict(int32_t h, const int32_t* starts, const int32_t* ends,
              int32_t n_spans, EvictPlan* plan, bool ragged = false);
    void undo_evict(int32_t h, const EvictPlan& plan);
    int release(int32_t h, std::vector<int32_t>* freed);

    // Resolves a handle; nullptr if invalid.
    const Seq* seq(int32_t h) const;
    Seq* seq_mut(int32_t h);
    int32_t live_pages() const { return g_.num_pages - alloc_.free_count(); }
    int64_t peak_live_pages() const { return peak_live_; }

  private:
    int32_t take_lowest();
    Geometry g_;
    PageAllocator alloc_;
    std::vector<Seq> seqs_;
    std::vector<int32_t> free_slots_;  // stack, lowest slot on top
    int64_t peak_live_ = 0;
};

// Splits an eviction's moves into tiles of at most `tile_rows` contiguous
// destination rows of one page, in order, and each copy tile into its
// contiguous source pieces; a tile of zero rows has no pieces.  Every
// source of a tile lies at a slot-space position >= the tile's first
// destination row, so processing tiles in order, each tile's reads before
// its writes, compacts in place.
// `window_tile` (may be null) receives the index of each window's first
// tile: windows share no page, so their tiles may run in any order.
void evict_tiles(const EvictPlan& p, int32_t tile_rows, std::vector<EvictTile>* tiles,
                 std::vector<EvictPiece>* pieces, std::vector<int32_t>* window_tile = nullptr);

// Eviction CTA shape: rows of an 8 KiB tile (at most a page, at least 8;
// 8 KiB copies measured faster than 16 KiB ones and far faster than 4 KiB
// ones), and ring slots by the (layer, K/V, head) planes each SM gets: 6 when
// there is at most one per SM, 3 up to four per SM, 4 beyond (measured on
// dense evictions of 128, 512 and 1,280 planes on 152 SMs).
int32_t evict_tile_rows_for(int32_t P, int32_t D);
int32_t evict_stages_for(int64_t planes, int32_t num_sms);

// Groups consecutive windows into at most `max_chunks` chunks of about equal
// tile counts, at least `min_tiles` tiles each (but the last): chunk c is
// tiles [chunk[c], chunk[c + 1]).  One chunk when there is one window.
void evict_chunks(const std::vector<int32_t>& window_tile, int32_t n_tiles, int32_t max_chunks,
                  int32_t min_tiles, std::vector<int32_t>* chunk);

// ---- decode planning -------------------------------------------------------

struct DecodePlanHost {
    std::vector<DecodeSeg> segs;
    std::vector<DecodeItem> items;
    std::vector<int32_t> cta_begin;   // n_ctas + 1
    std::vector<int32_t> page_ids;
    // rows held by each page of page_ids; filled only when some sequence of
    // the call has a partial page before its last (else every page is full
    // up to the members' limits)
    std::vector<int32_t> page_fill;
    // partial entries of (sequence i, KV head h): [comb_off[k], comb_off[k + 1]),
    // k = i * Hkv + h, in item order
    std::vector<int32_t> comb_off;    // n_seqs * Hkv + 1
    int64_t unique_tokens = 0;        // distinct rows read (one head, one layer)
    int64_t logical_tokens = 0;       // sum over sequences of n
    int32_t n_ctas = 0;
};

// Most partial results one (sequence, KV head) may have in a decode call:
// the kernel counts a run's arrivals in 16 bits.
constexpr int32_t kMaxRunEntries = 65535;

// Plans one decode call over the given sequences (each with n >= 1):
// groups sequences that hold the same physical page at the same logical
// index into shared runs, splits every (run, KV head) into stages of
// kStageTokens tokens and deals the stages out evenly to `n_ctas`
// persistent CTAs.  kCapacity if a (sequence, KV head) would get more than
// kMaxRunEntries partial results (more CTAs than that on one sequence).
int plan_decode(const HostCache& c, const int32_t* handles, int32_t n_seqs,
                int32_t n_ctas, DecodePlanHost* out);

// Serialises a plan into one buffer (8-byte aligned arrays).
DecodePlanLayout plan_layout(const DecodePlanHost& p, int32_t n_seqs,
                             int32_t Hkv);
void plan_serialize(const DecodePlanHost& p, const DecodePlanLayout& lay,
                    uint8_t* dst);

// ---- masked prefill planning ----------------------------------------------

struct PrefillPlanHost {
    std::vector<PrefillTile> tiles;   // key tiles with a visible key, increasing key0
    std::vector<int32_t> qt_tiles;    // per CTA tile: key tiles with key0 <= its last position
    int32_t n_pieces = 0;             // TMA boxes (min(P, 64) rows) per key tile
    std::vector<int32_t> tile_pages;  // [tiles][n_pieces] page of each piece, -1 past the end
    int32_t n = 0, n_q = 0;
    int32_t BP = 0;                   // query positions per query tile
    int32_t n_qt = 0;                 // CTA tiles (kPrefillQTiles query tiles each) per KV head
    int32_t n_split = 1;              // key-range splits per query tile
    int64_t visible_pairs = 0;        // sum over queries of the keys each sees
};

// Plans masked prefill attention over a sequence of n tokens whose last n_q
// tokens are the queries: validates the spans, builds the per-tile visibility
// bitmaps, and splits each query tile's key range in n_split parts when the
// query tiles alone would fill fewer than `target_ctas` CTAs.
// `pages` (may be null) is the sequence's page table; with it the plan also
// lists the page of every piece of every key tile.  Positions are slot-space
// positions: for a sequence with partial pages, n is its slot-space end and
// the spans include its unused slots (see prefill_slot_spans).
int plan_prefill(const Geometry& g, int32_t n, int32_t n_q, const int32_t* starts,
                 const int32_t* ends, int32_t n_spans, int32_t target_ctas,
                 PrefillPlanHost* out, const int32_t* pages = nullptr);

// Slot-space form of a masked prefill over sequence `s`: validates the
// logical spans against s.n, maps them to slot-space ranges, adds the unused
// slots of every partial page before the last, and returns the slot-space
// end.  The last n_q rows must occupy consecutive slots (no partial page
// among the pages holding them, but the last); otherwise kUnsupported.
int prefill_slot_spans(const Seq& s, int32_t P, int32_t n_q, const int32_t* starts,
                       const int32_t* ends, int32_t n_spans, std::vector<int32_t>* a_out,
                       std::vector<int32_t>* b_out, int32_t* n_slots);

}  // namespace sq
