// Kernel argument blocks and host-side launchers of the sm_103a kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../host/plan.hpp"

namespace sq {

// ---- decode attention -------------------------------------------------------
// Pages whose K/V may still be being written when a decode call starts, at
// most this many per call (see DecodeArgs::kv_early).
constexpr int kDecodeMaxUnsafe = 32;

struct DecodeArgs {
    const DecodeSeg* segs;
    const DecodeItem* items;
    const int32_t* cta_begin;
    const int32_t* page_ids;
    // rows held by each page of page_ids, or null when every page of the
    // call is full up to the members' limits (no sequence with partial pages)
    const int32_t* page_fill;
    const int32_t* comb_off;    // [n_seqs * Hkv + 1] partial entries of each (sequence, KV head)
    unsigned int* arrive;       // [n_seqs * Hkv] arrival counts, zero between calls
    const __nv_bfloat16* q;     // [n_seqs][Hq][D]
    void* out;                  // [n_seqs][Hq][D] bf16 or fp32
    float* part_o;              // [n_ent][G][D]  unnormalised partial outputs
    float* part_ml;             // [n_ent][G][4]  max (log2 units), sum, unused, unused
    int32_t out_f32;
    // 1: the plan was on the device before whatever precedes this launch on
    // the stream, so it may be read before the grid-dependency wait
    int32_t plan_ready;
    int32_t layer, Hq, Hkv, G, P, num_pages;
    float scale_log2;           // sm_scale * log2(e)
    int32_t debug_drop_cta;     // test hook: this CTA leaves its first stage unsignalled (-1: none)
    // 1: every library write to the plan's pages except those in unsafe[] is
    // known complete (the host polled its events), so a CTA may load its
    // first stages before the grid-dependency wait, overlapping the previous
    // kernel's tail, up to its first stage in one of those pages
    int32_t kv_early;
    int32_t n_unsafe;
    int32_t unsafe[kDecodeMaxUnsafe];
    int* err;
};

// Bytes of partial results one decode plan needs (n_ent partial entries).
int64_t decode_partial_bytes(int32_t n_ent, int32_t G, int32_t D);
// Persistent CTAs per SM the decode kernel runs with (occupancy of the kernel).
int decode_ctas_per_sm(int D);
cudaError_t decode_prepare(int D);  // raises the dynamic shared-memory limit once
cudaError_t launch_decode(const CUtensorMap& tmap, const DecodeArgs& a, int n_ctas, int D,
                          cudaStream_t st);

// ---- masked prefill attention -------------------------------------------------
struct PrefillArgs {
    const PrefillTile* tiles;   // key tiles with a visible key, increasing key0
    const int32_t* qt_tiles;    // [n_qt] key tiles each CTA tile reaches (a prefix of tiles)
    const int32_t* tile_pages;  // [n_tiles][n_pieces] page of each min(P, 64)-row piece, -1 past the end
    int32_t n_tiles, n_pieces;
    int32_t n, n_q;             // sequence tokens; queries = its last n_q tokens
    int32_t layer, Hq, Hkv, G, P, num_pages;
    int32_t BP;                 // query positions per query tile (kPrefillRows / G)
    int32_t n_qt, n_split;
    float scale_log2;           // sm_scale * log2(e), >= 0
    void* out;                  // [n_q][Hq][D] bf16 or fp32 (n_split == 1)
    int32_t out_f32;
    float* lse;                 // [n_q][Hq] or null (n_split == 1)
    float* part_o;              // [grid][kPrefillQTiles][kPrefillRows][D] normalised partials
                                // (n_split > 1)
    float* part_ml;             // [grid][kPrefillQTiles][kPrefillRows] their log2-sum-exp
    int* err;
};

struct PrefillCombineArgs {
    const float* part_o;
    const float* part_ml;
    void* out;
    int32_t out_f32;
    float* lse;
    int32_t n_q, Hq, Hkv, G, BP, n_qt, n_split;
};

// Dynamic shared memory of the prefill kernel.
int prefill_smem_bytes(int D);
cudaError_t prefill_prepare(int D);
// qmap: 3-D map of the queries {D, Hq, n_q}, box {64, G, BP}, 128-byte swizzle.
cudaError_t launch_prefill(const CUtensorMap& pool_map, const CUtensorMap& qmap,
                           const PrefillArgs& a, int D, cudaStream_t st);
cudaError_t launch_prefill_combine(const PrefillCombineArgs& a, int D, cudaStream_t st);

// ---- append / copy-on-write / eviction --------------------------------------
constexpr int kAppendMaxPages = 64;

// Words of cached decode plans that an append rewrites (in stream order, by
// block 0): the row limit of the run holding the appended sequence's last
// page, in plans that the append leaves valid (see the API layer).
constexpr int kAppendLenMax = 32;
struct AppendLens {
    int32_t n;
    int32_t* ptr[kAppendLenMax];
    int32_t val[kAppendLenMax];
};

struct AppendArgs {
    __nv_bfloat16* pool;
    const __nv_bfloat16* k;     // [L][n_total][Hkv][D]
    const __nv_bfloat16* v;
    int64_t num_pages;
    int32_t L, Hkv, P, D;
    int32_t n_total;            // tokens in the caller's buffers
    int32_t tok_begin;          // first caller token this launch writes
    int32_t n_tok;              // tokens this launch writes
    int32_t pos0;               // logical position of token tok_begin
    int32_t page_index0;        // logical page index of pages[0]
    int32_t n_pages;
    int32_t pages[kAppendMaxPages];
    AppendLens lens;
    int* err;
};

// One new token for each of up to kAppendBatchMax sequences.
constexpr int kAppendBatchMax = 128;

struct AppendBatchArgs {
    __nv_bfloat16* pool;
    const __nv_bfloat16* k;     // [L][n_total][Hkv][D]
    const __nv_bfloat16* v;
    int64_t num_pages;
    int32_t L, Hkv, P, D;
    int32_t n_total;            // rows in the caller's buffers (sequences of the call)
    int32_t row0;               // first row this launch writes
    int32_t n;                  // rows this launch writes
    int32_t page[kAppendBatchMax];
    int32_t slot[kAppendBatchMax];
    AppendLens lens;
    int* err;
};

struct CowArgs {
    __nv_bfloat16* pool;
    int64_t num_pages;
    int32_t L, Hkv, P, D;
    int32_t src_page, dst_page, rows;
    int* err;
};

struct EvictArgs {
    __nv_bfloat16* pool;
    int64_t num_pages;
    int32_t L, Hkv, P, D;
    const EvictTile* tiles;     // destination tiles, increasing logical order
    const EvictPiece* pieces;   // their contiguous source pieces
    int32_t n_tiles, n_pieces;
    int32_t tile_rows;          // rows a tile holds at most
    int32_t stages;             // shared-memory ring slots: 3, 4 or 6
    int32_t zero_tiles;         // 1: some tiles (those without pieces) write zeros
    // null, or [n_chunks + 1] tile indices: chunk c (tiles [chunk[c],
    // chunk[c + 1]), whole windows) of every plane runs in its own CTA
    const int32_t* chunk;
    int32_t n_chunks;
    int* err;
};

cudaError_t launch_append(const AppendArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_append_batch(const AppendBatchArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_cow_copy(const CowArgs& a, int num_sms, cudaStream_t st);
// Shared memory of one eviction CTA for a tile size and ring depth (plus one
// zero tile when the plan zeroes rows).
int evict_smem_bytes(int tile_rows, int D, int stages, bool zero_tiles = false);
// Resident eviction CTAs per SM for a tile size and ring depth.
int evict_ctas_per_sm(int tile_rows, int D, int stages);
cudaError_t evict_prepare();  // raises the dynamic shared-memory limit once
cudaError_t launch_evict(const EvictArgs& a, cudaStream_t st);

// Read-only streaming probe over `bytes` (multiple of 16) at `buf`.
cudaError_t launch_read_probe(const void* buf, size_t bytes, unsigned int* sink, int num_sms,
                              cudaStream_t st);

}  // namespace sq
