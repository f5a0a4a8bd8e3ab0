// A small C interface over the host-side cache state and planners, built into
// a separate CPU-only library (libsq_host.so) so that the page allocator,
// the copy-on-write / eviction rules and the decode planner can be exercised
// without a GPU.  It drives exactly the code libsq.so runs on the host.
#include <cstring>
#include <new>
#include <vector>

#include "../host/core.hpp"

using namespace sq;

extern "C" {

void* sqh_create(int32_t L, int32_t Hq, int32_t Hkv, int32_t D, int32_t P,
                 int32_t num_pages, int32_t max_seqs, int32_t max_pages_per_seq) {
    Geometry g;
    g.L = L; g.Hq = Hq; g.Hkv = Hkv; g.D = D; g.P = P;
    g.num_pages = num_pages; g.max_seqs = max_seqs; g.max_pages_per_seq = max_pages_per_seq;
    if (check_geometry(g) != kOk) return nullptr;
    return new (std::nothrow) HostCache(g);
}

void sqh_destroy(void* c) { delete static_cast<HostCache*>(c); }

int sqh_seq_new(void* c, int32_t* h) { return static_cast<HostCache*>(c)->seq_new(h); }

int sqh_fork(void* c, int32_t parent, int32_t* child) {
    return static_cast<HostCache*>(c)->fork(parent, child);
}

int sqh_append(void* c, int32_t h, int32_t n) {
    AppendPlan p;
    return static_cast<HostCache*>(c)->append(h, n, &p);
}

// ragged: 0 dense, 1 ragged.  stats_out (may be NULL): moved_rows, cow_pages,
// freed_pages, zeroed_rows, windows, number of moves.
int sqh_evict(void* c, int32_t h, const int32_t* spans, int32_t n_spans, int32_t ragged,
              int64_t* stats_out) {
    std::vector<int32_t> a(n_spans > 0 ? n_spans : 0), b(a.size());
    for (int32_t i = 0; i < n_spans; ++i) { a[i] = spans[2 * i]; b[i] = spans[2 * i + 1]; }
    EvictPlan p;
    int rc = static_cast<HostCache*>(c)->evict(h, a.data(), b.data(), n_spans, &p, ragged != 0);
    if (rc == kOk && stats_out) {
        stats_out[0] = p.moved_rows;
        stats_out[1] = (int64_t)p.cow_pages.size();
        stats_out[2] = (int64_t)p.freed.size();
        stats_out[3] = p.zeroed_rows;
        stats_out[4] = p.windows;
        stats_out[5] = (int64_t)p.moves.size();
    }
    return rc;
}

// Evicts and returns the compaction tiles (4 ints each: dst_page, dst_slot,
// n_rows, piece_begin) and pieces (src_page, src_slot, n_rows, dst_row), and
// the chunks of windows (chunk_out[0 .. n_chunks], tile indices) that the
// library would run in parallel CTAs with `max_chunks`.
int sqh_evict_tiles(void* c, int32_t h, const int32_t* spans, int32_t n_spans, int32_t ragged,
                    int32_t tile_rows, int32_t* tiles_out, int32_t tiles_cap, int32_t* pieces_out,
                    int32_t pieces_cap, int32_t* n_tiles, int32_t* n_pieces, int32_t max_chunks,
                    int32_t* chunk_out, int32_t chunk_cap, int32_t* n_chunks) {
    HostCache* hc = static_cast<HostCache*>(c);
    std::vector<int32_t> a(n_spans > 0 ? n_spans : 0), b(a.size());
    for (int32_t i = 0; i < n_spans; ++i) { a[i] = spans[2 * i]; b[i] = spans[2 * i + 1]; }
    EvictPlan p;
    int rc = hc->evict(h, a.data(), b.data(), n_spans, &p, ragged != 0);
    if (rc != kOk) return rc;
    std::vector<EvictTile> tiles;
    std::vector<EvictPiece> pieces;
    std::vector<int32_t> window_tile, chunk;
    evict_tiles(p, tile_rows, &tiles, &pieces, &window_tile);
    evict_chunks(window_tile, (int32_t)tiles.size(), max_chunks, 4, &chunk);
    *n_tiles = (int32_t)tiles.size();
    *n_pieces = (int32_t)pieces.size();
    *n_chunks = (int32_t)chunk.size() - 1;
    if ((int32_t)tiles.size() > tiles_cap || (int32_t)pieces.size() > pieces_cap ||
        (int32_t)chunk.size() > chunk_cap)
        return kInvalidArg;
    std::memcpy(tiles_out, tiles.data(), tiles.size() * sizeof(EvictTile));
    std::memcpy(pieces_out, pieces.data(), pieces.size() * sizeof(EvictPiece));
    std::memcpy(chunk_out, chunk.data(), chunk.size() * sizeof(int32_t));
    return kOk;
}

int sqh_release(void* c, int32_t h) { return static_cast<HostCache*>(c)->release(h, nullptr); }

int sqh_seq_info(void* c, int32_t h, int32_t* n_tokens, int32_t* n_pages) {
    const Seq* s = static_cast<HostCache*>(c)->seq(h);
    if (!s) return kBadHandle;
    *n_tokens = s->n;
    *n_pages = (int32_t)s->pages.size();
    return kOk;
}

int64_t sqh_next_pos(void* c, int32_t h) {
    const Seq* s = static_cast<HostCache*>(c)->seq(h);
    return s ? s->next_pos : -1;
}

int sqh_page_table(void* c, int32_t h, int32_t* out, int32_t cap, int32_t* n_out) {
    const Seq* s = static_cast<HostCache*>(c)->seq(h);
    if (!s) return kBadHandle;
    *n_out = (int32_t)s->pages.size();
    if (cap < *n_out) return kInvalidArg;
    std::memcpy(out, s->pages.data(), sizeof(int32_t) * s->pages.size());
    return kOk;
}

int sqh_page_fill(void* c, int32_t h, int32_t* out, int32_t cap, int32_t* n_out) {
    const Seq* s = static_cast<HostCache*>(c)->seq(h);
    if (!s) return kBadHandle;
    *n_out = (int32_t)s->fill.size();
    if (cap < *n_out) return kInvalidArg;
    std::memcpy(out, s->fill.data(), sizeof(int32_t) * s->fill.size());
    return kOk;
}

// The slot-space spans and end a masked prefill of the last n_q rows of
// sequence h uses (prefill_slot_spans); out receives start, end pairs.
int sqh_prefill_slot_spans(void* c, int32_t h, int32_t n_q, const int32_t* spans,
                           int32_t n_spans, int32_t* out, int32_t cap, int32_t* n_out,
                           int32_t* n_slots) {
    HostCache* hc = static_cast<HostCache*>(c);
    const Seq* s = hc->seq(h);
    if (!s) return kBadHandle;
    std::vector<int32_t> a(n_spans > 0 ? n_spans : 0), b(a.size()), xa, xb;
    for (int32_t i = 0; i < n_spans; ++i) { a[i] = spans[2 * i]; b[i] = spans[2 * i + 1]; }
    int rc = prefill_slot_spans(*s, hc->geom().P, n_q, a.data(), b.data(), n_spans, &xa, &xb,
                                n_slots);
    if (rc != kOk) return rc;
    *n_out = (int32_t)xa.size();
    if (cap < *n_out) return kInvalidArg;
    for (size_t i = 0; i < xa.size(); ++i) {
        out[2 * i] = xa[i];
        out[2 * i + 1] = xb[i];
    }
    return kOk;
}

int sqh_refcount(void* c, int32_t p) {
    HostCache* hc = static_cast<HostCache*>(c);
    if (p < 0 || p >= hc->geom().num_pages) return -1;
    return hc->alloc().refcount(p);
}

int sqh_free_count(void* c) { return static_cast<HostCache*>(c)->alloc().free_count(); }

int64_t sqh_peak_live_pages(void* c) { return static_cast<HostCache*>(c)->peak_live_pages(); }

// Plans a decode call.  layout_out receives 17 int64 values:
//   offsets segs, items, cta_begin, page_ids, comb_off, arrive, total,
//   counts n_segs, n_items, n_ctas, n_page_ids, n_comb_keys, n_comb_ent,
//   unique_tokens, logical_tokens, sizeof(DecodeSeg), offset page_fill (-1: none).
// If buf is non-NULL and buf_bytes >= total, the serialised plan is written.
// The eviction CTA shape the library picks: tile rows for (P, D) and ring
// slots for (planes, SMs).
int32_t sqh_evict_tile_rows(int32_t P, int32_t D) { return evict_tile_rows_for(P, D); }
int32_t sqh_evict_stages(int64_t planes, int32_t num_sms) { return evict_stages_for(planes, num_sms); }

int sqh_plan_decode(void* c, const int32_t* handles, int32_t n, int32_t n_ctas,
                    int64_t* layout_out, uint8_t* buf, int64_t buf_bytes) {
    HostCache* hc = static_cast<HostCache*>(c);
    DecodePlanHost p;
    int rc = plan_decode(*hc, handles, n, n_ctas, &p);
    if (rc != kOk) return rc;
    DecodePlanLayout L = plan_layout(p, n, hc->geom().Hkv);
    int64_t v[17] = {L.segs, L.items, L.cta_begin, L.page_ids, L.comb_off, L.arrive, L.total,
                     L.n_segs, L.n_items, L.n_ctas, L.n_page_ids, L.n_comb_keys, L.n_comb_ent,
                     p.unique_tokens, p.logical_tokens, (int64_t)sizeof(DecodeSeg), L.page_fill};
    std::memcpy(layout_out, v, sizeof v);
    if (buf) {
        if (buf_bytes < L.total) return kInvalidArg;
        plan_serialize(p, L, buf);
    }
    return kOk;
}

// Plans a masked prefill over a sequence of n tokens (G = Hq / Hkv; spans as
// start, end pairs; page size P).  info_out receives 6 int64 values: n_tiles,
// BP, n_qt, n_split, visible_pairs, sizeof(PrefillTile).  If tiles_out is
// non-NULL, up to `cap` tiles are written as 7 int32 each: key0, flags,
// vis[4], key0b; if qt_out is non-NULL, up to qt_cap per-query-tile counts.
int sqh_plan_prefill(int32_t Hq, int32_t Hkv, int32_t P, int32_t n, int32_t n_q,
                     const int32_t* spans, int32_t n_spans, int32_t target_ctas,
                     int64_t* info_out, int32_t* tiles_out, int32_t cap, int32_t* qt_out,
                     int32_t qt_cap) {
    Geometry g;
    g.L = 1; g.Hq = Hq; g.Hkv = Hkv; g.D = 128; g.P = P;
    g.num_pages = 1; g.max_seqs = 1; g.max_pages_per_seq = 1;
    if (Hkv < 1 || Hq % Hkv != 0) return kInvalidArg;
    std::vector<int32_t> a(n_spans > 0 ? n_spans : 0), b(a.size());
    for (int32_t i = 0; i < n_spans; ++i) {
        a[i] = spans[2 * i];
        b[i] = spans[2 * i + 1];
    }
    PrefillPlanHost p;
    int rc = plan_prefill(g, n, n_q, a.data(), b.data(), n_spans, target_ctas, &p);
    if (rc != kOk) return rc;
    int64_t v[6] = {(int64_t)p.tiles.size(), p.BP, p.n_qt, p.n_split, p.visible_pairs,
                    (int64_t)sizeof(PrefillTile)};
    std::memcpy(info_out, v, sizeof v);
    if (tiles_out) {
        const int32_t m = std::min<int32_t>(cap, (int32_t)p.tiles.size());
        for (int32_t i = 0; i < m; ++i) {
            const PrefillTile& t = p.tiles[i];
            int32_t* o = tiles_out + 7 * i;
            o[0] = t.key0;
            o[1] = t.flags;
            for (int w = 0; w < 4; ++w) o[2 + w] = (int32_t)t.vis[w];
            o[6] = t.key0b;
        }
    }
    if (qt_out) {
        const int32_t m = std::min<int32_t>(qt_cap, (int32_t)p.qt_tiles.size());
        for (int32_t i = 0; i < m; ++i) qt_out[i] = p.qt_tiles[i];
    }
    return kOk;
}

}  // extern "C"
