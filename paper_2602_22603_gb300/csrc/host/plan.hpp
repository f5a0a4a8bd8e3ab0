// Plain-old-data work descriptions the host planners write and the kernels
// read.  Shared by host code (C++) and device code (CUDA); no CUDA types.
#pragma once
#include <stdint.h>

namespace sq {

// Rows of one tensor-core tile: the query rows a decode work item serves
// (Sec. 2.1: a KV head is shared by G query heads; with several sequences
// sharing the same pages, their query groups stack up to this many rows).
constexpr int kRowsPerTile = 16;
// Tokens of K/V one pipeline stage of the decode kernel holds.
constexpr int kStageTokens = 64;
// Consumer warps of the decode kernel; each owns kStageTokens / 4 tokens.
constexpr int kDecodeConsumerWarps = 4;
// Fixed cost of starting a work unit, in stages: its query reload and its
// item-end merge.  The planner balances stages plus this cost per unit, so a
// CTA that gets many short units (e.g. the few-token tails of several forks)
// is not the one every other CTA waits for.
constexpr int kUnitCostStages = 2;

// A run of logical pages read once for a group of sequences that hold the
// same physical pages there (a main thread and its forks, Sec. 3.4).
struct DecodeSeg {
    int32_t page_off;                 // into DecodePlan page_ids
    int32_t n_pages;                  // pages in the run
    int32_t n_tok;                    // tokens to read (max over the group)
    int32_t n_grp;                    // sequences in the group
    int32_t grp_seq[kRowsPerTile];    // call-local sequence indices
    int32_t grp_lim[kRowsPerTile];    // valid tokens of each, from the run start
    int32_t q0;                       // page index of the run's first page in its members
    int32_t tail;                     // bit j: the run holds member j's last page (the
                                      // others' limit is the whole run)
};

// A contiguous range of stages of one (segment, KV head) — one partial result
// per group member.  Member j's G rows go to partial entry ent[j]; the entries
// of one (sequence, KV head) are contiguous, so that its merge reads them
// without an index.  A member whose (sequence, KV head) has this one entry
// only (bit j of `sole`) gets its normalised output written directly.
struct DecodeItem {
    int32_t seg;
    int32_t head;
    int32_t s0, s1;                   // stages [s0, s1)
    int32_t sole;                     // bit j: member j's run is this item alone
    int32_t ent[kRowsPerTile];        // partial entry of each group member (n_grp used)
};

// Eviction compaction, planned once per eviction and shared by every
// (layer, K/V, head) plane: destination tiles (contiguous rows of one page, in
// increasing logical order) and, per tile, the contiguous source pieces that
// fill it.  A tile without pieces writes zeros (the unused slots of a page
// that a ragged eviction leaves partial).
struct EvictTile {
    int32_t dst_page;
    int32_t dst_slot;     // first destination slot in the page
    int32_t n_rows;       // rows written (<= tile capacity)
    int32_t piece_begin;  // pieces [piece_begin, next tile's piece_begin); none: zero rows
};

struct EvictPiece {
    int32_t src_page;
    int32_t src_slot;
    int32_t n_rows;
    int32_t dst_row;      // row offset inside the tile
};

// Masked prefill attention (Algorithm 2, BuildMask).  A query tile holds
// kPrefillRows rows: floor(kPrefillRows / G) consecutive query positions times
// the G query heads of one KV head (Sec. 2.1), so one K/V tile serves them all.
// Keys are taken kPrefillKeys at a time, aligned to kPrefillKeys.
constexpr int kPrefillRows = 128;
constexpr int kPrefillKeys = 128;
// Query tiles one CTA owns; they share every K/V tile it loads.
constexpr int kPrefillQTiles = 2;
constexpr int32_t kPrefillTileFull = 1;  // every key of the tile exists and is visible

// One key tile that holds at least one visible key of the sequence: two
// halves of 64 keys, each 64 consecutive positions starting at a multiple of
// 64 (key0, key0b).  With pages of >= 64 tokens the halves are the visible
// 64-key boxes of the sequence taken two by two, so a box that a span covers
// entirely is skipped even when its neighbour is not; with smaller pages the
// tile is 128 aligned keys (key0b = key0 + 64).  A missing second half has
// key0b = kPrefillNoKeys (past any sequence).
constexpr int32_t kPrefillNoKeys = 0x7fffffc0;
struct PrefillTile {
    int32_t key0;      // first key of the lower half
    int32_t flags;     // kPrefillTileFull or 0
    uint32_t vis[4];   // bit c of word w: key (w < 2 ? key0 : key0b) + 32 (w % 2) + c
                       // exists and lies in no span
    int32_t key0b;     // first key of the upper half
    int32_t pad;
};

// Byte offsets of the arrays of a decode plan inside one upload buffer.
// Byte offsets of the serialised decode plan.  `arrive` holds one 32-bit
// arrival count per (sequence, KV head), zero in the serialised plan; the
// kernel counts on it and leaves it at zero again.
// `page_fill` is -1 when the plan carries no page fills.
struct DecodePlanLayout {
    int64_t segs, items, cta_begin, page_ids, comb_off, arrive, page_fill, total;
    int32_t n_segs, n_items, n_ctas, n_page_ids, n_comb_keys, n_comb_ent;
};

}  // namespace sq
