// Masked prefill attention on the 5th-generation tensor cores.
//
// What it computes (Algorithm 2, BuildMask; Sec. 3.3): the last n_q tokens of
// a sequence attend causally to its tokens, with the tokens of the given spans
// (closed cursors) removed from every query's view:
//   query at position p, query head h, KV head g = floor(h / G):
//     s_j = sm_scale * q_h . k_{g,j}   for visible keys j (j <= p, j in no span)
//     o_h = sum_j softmax_j(s) v_{g,j}
//
// A query tile is 128 rows: floor(128 / G) consecutive query positions times
// the G query heads of one KV head (Sec. 2.1).  One CTA owns two consecutive
// query tiles (a, b) of the same KV head, and every K/V tile it loads serves
// both, which halves the loads per tensor-core FLOP.  Keys go 128 at a time,
// aligned to 128; tiles whose keys are all masked are never loaded (the host
// lists the others with a visibility bitmap).  Per key tile j and query tile t:
//   S_t = Q_t K_j^T           tcgen05.mma, Q and K from shared memory, S in TMEM
//   P_t = exp2(S_t - m)       softmax warpgroup t: tcgen05.ld of S, mask, bf16 P
//                             stored back over the first half of S_t
//   O_t += P_t V_j            tcgen05.mma with A = P from TMEM and V read
//                             token-major from shared memory (MN-major B)
// The MMA issuer interleaves the two tiles (PV_a(j), S_a(j+1), PV_b(j),
// S_b(j+1)), so while one warpgroup turns S into P the tensor core works for
// the other.  P_t(j) shares TMEM with S_t: S_t(j+1) is issued after PV_t(j),
// and tcgen05.mma operations of one thread execute in issue order.  The same
// order means that when S_t(j) is ready, PV_t(j-1) is complete, so a
// warpgroup may rescale O_t then without another wait.  The running maximum
// is raised lazily: a key tile's weights are taken with the current maximum
// and accepted while every row's sum of them stays at most 2^16 (so does each
// weight); only then is a maximum raised and O rescaled.  K and V stream through one ring of
// shared-memory slots (K_0, V_0, K_1, ...); a K slot is released once both S
// products are done, a V slot once both PV products are.
//
// Short query blocks: when a CTA tile's queries all fit in tile a, tile b's
// warpgroup takes the same rows over every other key tile (dual-key mode, the
// two results merged per row at the end, loads in the order the MMAs consume
// them), and when there are fewer CTA tiles than SMs each tile's key range is
// split over several CTAs whose normalised partial results a second kernel
// merges.
//
// Warp roles (320 threads): warp 0 loads (lanes 0 and 1 issue the TMA copies,
// two loads at a time), lane 0 of warp 1 issues the MMAs and warp 1 owns the
// TMEM allocation, warps 2-5
// are the softmax warpgroup of tile a and warps 6-9 that of tile b (warp w
// reads TMEM lanes 32 (w mod 4) .. +31, one row per thread).  Every wait is
// bounded; a wait that runs out sets the error word and the CTA winds down
// after its copies and MMAs in flight have completed.
#include "launch.hpp"
#include "ptx.cuh"
#include "tc.cuh"

namespace sq {
namespace dev {
namespace {

template <int D>
struct PreCfg {
    static constexpr int kThreads = 320;
    static constexpr int kColBlocks = D / 64;                  // 64-column (128-byte) blocks
    static constexpr int kBlockBytes = kPrefillRows * 128;      // one block of a 128-row tile
    static constexpr int kQBytes = kColBlocks * kBlockBytes;    // one query tile
    static constexpr int kSlotBytes = kColBlocks * kBlockBytes;  // 128 keys of K or of V
    static constexpr int kSlots = D == 128 ? 5 : 12;
    static constexpr int kOffQ = 0;
    static constexpr int kOffRing = kOffQ + kPrefillQTiles * kQBytes;
    static constexpr int kOffBar = kOffRing + kSlots * kSlotBytes;
    static constexpr int kBarQ = 0;
    static constexpr int kBarFull = 1;                  // [kSlots] tile landed (V: and ready)
    static constexpr int kBarEmpty = kBarFull + kSlots; // [kSlots] slot consumed by the MMAs
    static constexpr int kBarS = kBarEmpty + kSlots;    // [2] S_t written (and PV_t before it done)
    static constexpr int kBarP = kBarS + 2;             // [2] P_t written (128 arrivals)
    static constexpr int kBarO = kBarP + 2;             // [2] last PV_t done
    static constexpr int kBarVfix = kBarO + 2;          // V of the last key tile landed
    static constexpr int kBarDone = kBarVfix + 1;       // every MMA of the CTA done
    static constexpr int kNumBars = kBarDone + 1;
    static constexpr int kOffMisc = kOffBar + kNumBars * 8;
    // dual-key mode: tile b's (max, normaliser) of each row, for the merge
    static constexpr int kOffXchg = (kOffMisc + 32 + 15) & ~15;
    static constexpr int kSmemBytes = kOffXchg + kPrefillRows * 8 + 1024;  // + alignment slack
    static constexpr uint32_t kTmemCols = 512;
    static constexpr uint32_t kColS = 0;    // S_t (fp32) at 128 t; P_t (bf16 pairs) over its first 64
    static constexpr uint32_t kColO = 256;  // O_t (fp32) at 256 + 128 t
    static constexpr uint32_t kIdescQK = mma_idesc_bf16(128, kPrefillKeys, false);
    static constexpr uint32_t kIdescPV = mma_idesc_bf16(128, D, true);
    static_assert(kSmemBytes <= 232448, "shared memory");
    static_assert(kOffXchg % 16 == 0 && kOffRing % 1024 == 0 && kOffBar % 8 == 0, "alignment");
    static_assert(kPrefillQTiles == 2, "two query tiles per CTA");
};

struct Smem {
    uint32_t base;  // shared address of the 1024-aligned region
    uint8_t* ptr;
    template <int D>
    __device__ uint32_t bar(int i) const {
        return base + PreCfg<D>::kOffBar + 8 * i;
    }
};

// Bits 0 .. x of a word (x < 0: none; x >= 31: all).
__device__ __forceinline__ uint32_t low_bits_through(int x) {
    return x >= 31 ? 0xffffffffu : (x < 0 ? 0u : ((2u << x) - 1u));
}

// Order of the K and V loads of a CTA's T key tiles, load u into ring slot
// u mod kSlots.  Normally key tile by key tile: u = 2 j is K_j, u = 2 j + 1
// is V_j.  In dual-key mode (tile a takes the even key tiles, tile b the odd
// ones) the loads follow the order in which the MMA warp consumes them, so
// that no tile waits in the ring for a later one: K_0, K_1, then V_j and
// K_{j+2} in turn, and the last two V tiles.
__device__ __forceinline__ void load_of(int u, int T, bool dual, int& j, int& kv) {
    if (!dual) {
        j = u >> 1;
        kv = u & 1;
    } else if (u < 2) {
        j = u;
        kv = 0;
    } else if (u >= 2 * T - 2) {
        j = u - T;
        kv = 1;
    } else {
        j = ((u - 2) >> 1) + ((u & 1) ? 2 : 0);
        kv = (u & 1) ? 0 : 1;
    }
}
// The loads of K_j and V_j in dual-key mode (T >= 2).
__device__ __forceinline__ int dual_load_k(int j) { return j < 2 ? j : 2 * j - 1; }
__device__ __forceinline__ int dual_load_v(int j, int T) { return j < T - 1 ? 2 * j + 2 : 2 * T - 1; }

// The producer warp: the query tiles once, then the K and V tiles of every key
// tile into the ring in the order of load_of, two loads at a time: the whole
// warp waits for both slots, then lanes 0 and 1 arm their barriers and issue
// their copies together, so that the shared-memory round trips of the two
// overlap.  What a tile's copies need, {first key, page of box 0, page of box
// 1}, is held in
// registers: lane l has the record of the window's key tile j = l (mod 32),
// batches of 16 tiles alternating between the lower and the upper half-warp;
// a batch is read from global memory about ten tiles before its first use and
// moved into place a few tiles before it.  Boxes past the second (pages of
// fewer than 64 tokens) take their page from global memory.
template <int D>
__device__ void prefill_produce(const CUtensorMap* pool_map, const CUtensorMap* qmap,
                                const PrefillArgs& a, const Smem& sm, int g, int pos_lo, int t0,
                                int T, bool two, bool dual, volatile int* abort_flag, int lane) {
    using C = PreCfg<D>;
    if (lane == 0) {
        prefetch_tmap(pool_map);
        prefetch_tmap(qmap);
        const int nq = two ? 2 : 1;  // tile b is loaded only when it holds queries
        mbar_arrive_expect_tx(sm.bar<D>(C::kBarQ), nq * C::kColBlocks * a.BP * a.G * 128);
        for (int t = 0; t < nq; ++t)
            for (int cb = 0; cb < C::kColBlocks; ++cb)
                tma_load_3d(sm.base + C::kOffQ + t * C::kQBytes + cb * C::kBlockBytes, qmap,
                            sm.bar<D>(C::kBarQ), cb * 64, g * a.G, pos_lo + t * a.BP);
    }
    const int br = a.P < 64 ? a.P : 64;  // rows of one TMA box
    const int n_pieces = a.n_pieces;      // <= 16
    constexpr int kBatch = 16;
    // {first key of each half, page of box 0, page of box 1} of key tile
    // tb + lane % 16 (x = key0, y = page 0, z = page 1, w = key0b)
    auto load_rec = [&](int tb) {
        int4 r = make_int4(0, -1, -1, kPrefillNoKeys);
        const int jj = tb + (lane & (kBatch - 1));
        if (jj < T) {
            const size_t t = (size_t)(t0 + jj);
            r.x = __ldg(&a.tiles[t].key0);
            r.w = __ldg(&a.tiles[t].key0b);
            r.y = __ldg(&a.tile_pages[t * n_pieces]);
            if (n_pieces > 1) r.z = __ldg(&a.tile_pages[t * n_pieces + 1]);
        }
        return r;
    };
    int4 rec = make_int4(0, -1, -1, kPrefillNoKeys), pend = rec;
    if (lane < kBatch) rec = load_rec(0);
    int fill_b = 1;    // the next batch to read
    int merge_b = -1;  // the batch read into `pend`, not yet in place
    const int n_units = 2 * T;
    int issued = 0;
    int tail_u = -1;          // the load that used the fix-up barrier
    bool tail_done = false;   // ... and was handed over on its slot's barrier
    for (int u0 = 0; u0 < n_units; u0 += 2) {  // n_units is even
        int j0, kv0, j1, kv1;
        load_of(u0, T, dual, j0, kv0);
        load_of(u0 + 1, T, dual, j1, kv1);
        const int jmax = j0 > j1 ? j0 : j1;
        if (merge_b >= 0 && jmax + 4 >= kBatch * merge_b) {
            if ((lane >> 4) == (merge_b & 1)) rec = pend;
            merge_b = -1;
        }
        if (merge_b < 0 && fill_b * kBatch < T && jmax + 10 >= kBatch * fill_b) {
            if ((lane >> 4) == (fill_b & 1)) pend = load_rec(fill_b * kBatch);
            merge_b = fill_b++;
        }
        const int u = u0 + (lane & 1);  // lanes 0 and 1 issue
        const int j = (lane & 1) ? j1 : j0, kv = (lane & 1) ? kv1 : kv0;
        const int key0 = __shfl_sync(0xffffffffu, rec.x, j & 31);
        const int pg0 = __shfl_sync(0xffffffffu, rec.y, j & 31);
        const int pg1 = __shfl_sync(0xffffffffu, rec.z, j & 31);
        const int key0b = __shfl_sync(0xffffffffu, rec.w, j & 31);
        // rows of the tile inside the sequence (only the last tile has fewer
        // than 128): the lower half's, then the upper half's
        const int rows_b = key0b < a.n ? min(64, a.n - key0b) : 0;
        const int rows = rows_b > 0 ? 64 + rows_b : min(64, a.n - key0);
        const int slot = u % C::kSlots;
        const bool vfix = lane < 2 && kv == 1 && rows < kPrefillKeys;
        // every lane polls both slots' barriers in turn: warp-uniform waits,
        // so no lane waits at the vote below for two polling lanes
        bool ok = true;
        if (u0 >= C::kSlots)
            ok = mbar_wait(sm.bar<D>(C::kBarEmpty + u0 % C::kSlots), (u0 / C::kSlots - 1) & 1,
                           abort_flag);
        if (ok && u0 + 1 >= C::kSlots)
            ok = mbar_wait(sm.bar<D>(C::kBarEmpty + (u0 + 1) % C::kSlots),
                           ((u0 + 1) / C::kSlots - 1) & 1, abort_flag);
        // both slots free, or neither load is issued
        if (!__all_sync(0xffffffffu, ok)) {
            if (lane == 0) {
                set_error(a.err, kErrTimeout);
                *abort_flag = 1;
            }
            break;
        }
        if (lane < 2) {
            const int nv = (rows + br - 1) / br;  // boxes inside the sequence (a prefix)
            const uint32_t fb = vfix ? sm.bar<D>(C::kBarVfix) : sm.bar<D>(C::kBarFull + slot);
            mbar_arrive_expect_tx(fb, (uint32_t)nv * br * 128 * C::kColBlocks);
            const uint32_t dst = sm.base + C::kOffRing + slot * C::kSlotBytes;
            const int head_row = (kv ? a.Hkv + g : g) * a.P;
#pragma unroll 1
            for (int i = 0; i < nv; ++i) {
                int32_t page =
                    i == 0 ? pg0
                           : (i == 1 ? pg1
                                     : __ldg(&a.tile_pages[(size_t)(t0 + j) * n_pieces + i]));
                if ((uint32_t)page >= (uint32_t)a.num_pages) {
                    // a page outside the pool: flagged; the box is read from
                    // page 0 so that the barrier's byte count still completes
                    set_error(a.err, kErrBounds);
                    page = 0;
                }
                const int half = n_pieces / 2;
                const int key = i < half ? key0 + i * br : key0b + (i - half) * br;
#pragma unroll
                for (int cb = 0; cb < C::kColBlocks; ++cb)
                    tma_load_4d(dst + cb * C::kBlockBytes + i * br * 128, pool_map, fb, cb * 64,
                                head_row + key % a.P, page, a.layer);
            }
        }
        issued = u0 + 2;
        const uint32_t fix = __ballot_sync(0xffffffffu, vfix);
        if (fix) {
            // V of the last key tile: its rows past the sequence's end hold
            // stale or never-written data.  Their weights are zero, but 0 * NaN
            // is not, so zero those rows before the MMAs read the slot.
            const int src = __ffs(fix) - 1;
            const int fslot = __shfl_sync(0xffffffffu, slot, src);
            const int frows = __shfl_sync(0xffffffffu, rows, src);
            tail_u = u0 + src;
            if (lane == 0) ok = mbar_wait(sm.bar<D>(C::kBarVfix), 0, abort_flag);
            if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) {
                if (lane == 0) {
                    set_error(a.err, kErrTimeout);
                    *abort_flag = 1;
                }
                break;
            }
            const int r0 = frows;  // 1 .. 127
            const int chunks = (kPrefillKeys - r0) * 8;
            uint8_t* vsp = sm.ptr + C::kOffRing + fslot * C::kSlotBytes;
            for (int cb = 0; cb < C::kColBlocks; ++cb)
                for (int c = lane; c < chunks; c += 32)
                    *reinterpret_cast<uint4*>(vsp + cb * C::kBlockBytes + (r0 + (c >> 3)) * 128 +
                                              (c & 7) * 16) = make_uint4(0, 0, 0, 0);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(sm.bar<D>(C::kBarFull + fslot));
            tail_done = true;
        }
    }
    // Drain: every copy this CTA issued lands before the CTA exits (immediate
    // unless a consumer gave up early).
    if (lane == 0) {
        mbar_wait(sm.bar<D>(C::kBarQ), 0);
        for (int u = issued > C::kSlots ? issued - C::kSlots : 0; u < issued; ++u) {
            if (u == tail_u && !tail_done) mbar_wait(sm.bar<D>(C::kBarVfix), 0);
            else mbar_wait(sm.bar<D>(C::kBarFull + u % C::kSlots), (u / C::kSlots) & 1);
        }
    }
}

// S_t = Q_q K^T for the K tile in `slot`, into TMEM columns 128 t (q = t
// except in dual-key mode, where both tiles use query tile 0).
template <int D>
__device__ __forceinline__ void issue_qk(const Smem& sm, uint32_t tmem, int t, int slot, int q = -1) {
    using C = PreCfg<D>;
    const uint32_t qa = sm.base + C::kOffQ + (q < 0 ? t : q) * C::kQBytes;
    const uint32_t ka = sm.base + C::kOffRing + slot * C::kSlotBytes;
    const uint32_t dt = tmem + C::kColS + (uint32_t)t * kPrefillKeys;
    // descriptors built once and stepped per K step: the address field holds
    // address / 16 in 14 bits and every address here is below 2^18 bytes, so
    // adding offset / 16 cannot carry out of it
    const uint64_t qd = smem_desc_sw128(qa, 16, 1024), kd = smem_desc_sw128(ka, 16, 1024);
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
        const uint32_t off = ((ks >> 2) * C::kBlockBytes + (ks & 3) * 32) >> 4;
        mma_bf16_ss(dt, qd + off, kd + off, C::kIdescQK, ks > 0);
    }
}

// O_t += P_t V for the V tile in `slot`; P_t from TMEM over the first half of S_t.
template <int D>
__device__ __forceinline__ void issue_pv(const Smem& sm, uint32_t tmem, int t, int slot,
                                         bool first) {
    using C = PreCfg<D>;
    const uint32_t pa = tmem + C::kColS + (uint32_t)t * kPrefillKeys;
    const uint32_t va = sm.base + C::kOffRing + slot * C::kSlotBytes;
    const uint64_t vd = smem_desc_sw128(va, C::kBlockBytes, 1024);
#pragma unroll
    for (int ks = 0; ks < kPrefillKeys / 16; ++ks)
        mma_bf16_ts(tmem + C::kColO + (uint32_t)t * 128, pa + ks * 8, vd + (uint64_t)(ks * 128),
                    C::kIdescPV, (!first || ks > 0) ? 1u : 0u);
}

// Dual-key mode (every query of the CTA tile fits in tile a): both tiles
// hold tile a's queries; tile a takes key tiles 0, 2, 4, ... and tile b the
// odd ones, and the two results are merged at the end.  Key tile j's PV and
// the QK of key tile j + 2 (into the same S columns) are issued in the order
// of the loads, each as soon as its tile has landed.
template <int D>
__device__ bool prefill_mma_dual(const Smem& sm, uint32_t tmem, int T, volatile int* abort_flag) {
    using C = PreCfg<D>;
    bool ok = true;
    for (int t = 0; t < 2 && ok; ++t) {
        // S_t = Q_a K_t
        const int u = dual_load_k(t), slot = u % C::kSlots;
        if (!(ok = mbar_wait(sm.bar<D>(C::kBarFull + slot), (u / C::kSlots) & 1, abort_flag))) break;
        issue_qk<D>(sm, tmem, t, slot, 0);
        mma_commit(sm.bar<D>(C::kBarS + t));
        mma_commit(sm.bar<D>(C::kBarEmpty + slot));
    }
    for (int j = 0; ok && j < T; ++j) {
        const int t = j & 1, i = j >> 1;
        const int uv = dual_load_v(j, T), vslot = uv % C::kSlots;
        if (!(ok = mbar_wait(sm.bar<D>(C::kBarFull + vslot), (uv / C::kSlots) & 1, abort_flag)))
            break;
        if (!(ok = mbar_wait(sm.bar<D>(C::kBarP + t), i & 1, abort_flag))) break;
        tc_fence_after();
        issue_pv<D>(sm, tmem, t, vslot, i == 0);
        mma_commit(sm.bar<D>(C::kBarEmpty + vslot));
        if (j + 2 >= T) {  // the last key tile of tile t
            mma_commit(sm.bar<D>(C::kBarO + t));
            continue;
        }
        const int uk = dual_load_k(j + 2), kslot = uk % C::kSlots;
        if (!(ok = mbar_wait(sm.bar<D>(C::kBarFull + kslot), (uk / C::kSlots) & 1, abort_flag)))
            break;
        issue_qk<D>(sm, tmem, t, kslot, 0);
        mma_commit(sm.bar<D>(C::kBarS + t));
        mma_commit(sm.bar<D>(C::kBarEmpty + kslot));
    }
    return ok;
}

// `two`: tile b holds query rows (false for short query blocks, whose rows
// all fit in tile a; tile b's products are then skipped, or, with `dual`, it
// takes every other key tile).
template <int D>
__device__ void prefill_mma(const PrefillArgs& a, const Smem& sm, uint32_t tmem, int T, bool two,
                            bool dual, volatile int* abort_flag) {
    using C = PreCfg<D>;
    bool ok = mbar_wait(sm.bar<D>(C::kBarQ), 0, abort_flag);
    bool any = false;
    if (ok && T > 0 && dual) {
        tc_fence_after();
        any = true;
        ok = prefill_mma_dual<D>(sm, tmem, T, abort_flag);
    } else if (ok && T > 0) {
        tc_fence_after();
        const int k0 = 0;
        ok = mbar_wait(sm.bar<D>(C::kBarFull + k0), 0, abort_flag);
        if (ok) {
            any = true;
            issue_qk<D>(sm, tmem, 0, k0);
            mma_commit(sm.bar<D>(C::kBarS + 0));
            if (two) {
                issue_qk<D>(sm, tmem, 1, k0);
                mma_commit(sm.bar<D>(C::kBarS + 1));
            }
            mma_commit(sm.bar<D>(C::kBarEmpty + k0));
        }
        for (int j = 0; ok && j < T; ++j) {
            const int uv = 2 * j + 1, vslot = uv % C::kSlots;
            const int uk = 2 * j + 2, kslot = uk % C::kSlots;
            const bool more = j + 1 < T;
            // V_j and K_{j+1} have normally landed long ago; checking them before
            // P_a keeps these barrier reads off the path from P_a to the MMAs
            if (!(ok = mbar_wait(sm.bar<D>(C::kBarFull + vslot), (uv / C::kSlots) & 1, abort_flag)))
                break;
            if (more && !(ok = mbar_wait(sm.bar<D>(C::kBarFull + kslot), (uk / C::kSlots) & 1,
                                         abort_flag)))
                break;
            // tile a: O_a += P_a V_j, then S_a for the next key tile
            if (!(ok = mbar_wait(sm.bar<D>(C::kBarP + 0), j & 1, abort_flag))) break;
            tc_fence_after();
            issue_pv<D>(sm, tmem, 0, vslot, j == 0);
            if (!more) mma_commit(sm.bar<D>(C::kBarO + 0));
            if (!two) mma_commit(sm.bar<D>(C::kBarEmpty + vslot));
            if (more) {
                issue_qk<D>(sm, tmem, 0, kslot);
                mma_commit(sm.bar<D>(C::kBarS + 0));
                if (!two) mma_commit(sm.bar<D>(C::kBarEmpty + kslot));
            }
            if (!two) continue;
            // tile b
            if (!(ok = mbar_wait(sm.bar<D>(C::kBarP + 1), j & 1, abort_flag))) break;
            tc_fence_after();
            issue_pv<D>(sm, tmem, 1, vslot, j == 0);
            mma_commit(sm.bar<D>(C::kBarEmpty + vslot));
            if (!more) mma_commit(sm.bar<D>(C::kBarO + 1));
            if (more) {
                issue_qk<D>(sm, tmem, 1, kslot);
                mma_commit(sm.bar<D>(C::kBarS + 1));
                mma_commit(sm.bar<D>(C::kBarEmpty + kslot));
            }
        }
    }
    if (!ok) {
        set_error(a.err, kErrTimeout);
        *abort_flag = 1;
    }
    if (any) {
        // every MMA issued here completes before TMEM is released
        mma_commit(sm.bar<D>(C::kBarDone));
        mbar_wait(sm.bar<D>(C::kBarDone), 0);
    }
}

// Packed fp32 pair helpers (sm_100 family): d = a * b + c on two lanes at once.
__device__ __forceinline__ uint64_t f2pack(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2unpack(uint64_t v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
// lo += the low bf16 of w, hi += its high bf16 (mixed-precision adds: the
// bf16 operands are exact in fp32).
__device__ __forceinline__ void add_bf16x2_f32(uint32_t w, float& lo, float& hi) {
    asm("{\n\t.reg .b16 l16, h16;\n\tmov.b32 {l16, h16}, %2;\n\t"
        "add.rn.f32.bf16 %0, l16, %0;\n\tadd.rn.f32.bf16 %1, h16, %1;\n\t}"
        : "+f"(lo), "+f"(hi)
        : "r"(w));
}
// 2^x as the single PTX instruction ex2.approx.ftz (relative error about
// 2^-22).  Results below 2^-126 flush to zero: every row holds a weight of at
// least 1 (its running maximum's), so they change its sums by under 2^-119.
__device__ __forceinline__ float ex2_ftz(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Every lane of the warp polls the barrier (one instruction for the warp,
// no hand-on from a polling lane: a softmax warp sees its S ready sooner);
// returns the warp-uniform result.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, const volatile int* abort) {
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

// Softmax warpgroup of query tile t (one row per thread) and its epilogue.
template <int D>
__device__ void prefill_softmax(const PrefillArgs& a, const Smem& sm, uint32_t tmem, int t, int g,
                                int pos_lo, int t0, int T_cta, bool dual, volatile int* abort_flag,
                                int warp, int lane) {
    using C = PreCfg<D>;
    const int wq = warp & 3;
    const int row = wq * 32 + lane;
    // dual-key mode: both tiles hold tile a's queries, tile t takes key tiles
    // t, t + 2, t + 4, ... of the CTA's range
    const int qi = pos_lo + (dual ? 0 : t) * a.BP + row / a.G;
    const bool valid = row < a.BP * a.G && qi < a.n_q;
    const int T = dual ? (T_cta + 1 - t) / 2 : T_cta;
    const int kstep = dual ? 2 : 1, kfirst = dual ? t : 0;
    float* xchg = reinterpret_cast<float*>(sm.ptr + C::kOffXchg);
    // A warp none of whose rows is a query only keeps the barrier count: it
    // waits for each S and signals its P without computing (its rows of P
    // and O are never read back).
    if (!__any_sync(0xffffffffu, valid)) {
        bool wok = true;
        for (int j = 0; j < T; ++j) {
            if (wok) wok = warp_wait(sm.bar<D>(C::kBarS + t), j & 1, abort_flag);
            tc_fence_before();
            mbar_arrive(sm.bar<D>(C::kBarP + t));
        }
        if (!wok && lane == 0) {
            set_error(a.err, kErrTimeout);
            *abort_flag = 1;
        }
        // the merge of the two tiles' results meets all 256 threads, whatever happened
        if (dual) named_bar_sync(3, 256);
        return;
    }
    const int p_row = a.n - a.n_q + qi;
    const uint32_t tl = tmem + ((uint32_t)(wq * 32) << 16);
    const uint32_t col_s = C::kColS + (uint32_t)t * kPrefillKeys;
    const uint32_t col_o = C::kColO + (uint32_t)t * 128;
    const float sc = a.scale_log2;  // > 0 (the host raises a zero scale to a tiny one)
    float m_run = -INFINITY, l = 0.f;
    bool ok = true;
    int4 n0 = make_int4(0, 0, 0, 0), n1 = n0;
    if (T > 0) {
        const int4* tp = reinterpret_cast<const int4*>(a.tiles + t0 + kfirst);
        n0 = __ldg(tp);
        n1 = __ldg(tp + 1);
    }
    for (int j = 0; j < T; ++j) {
        // this tile's record; the next one is fetched while this tile is worked on
        const int4 w0 = n0, w1 = n1;
        if (j + 1 < T) {
            const int4* tp =
                reinterpret_cast<const int4*>(a.tiles + t0 + kfirst + (j + 1) * kstep);
            n0 = __ldg(tp);
            n1 = __ldg(tp + 1);
        }
        const int key0 = w0.x;
        const uint32_t vis[4] = {(uint32_t)w0.z, (uint32_t)w0.w, (uint32_t)w1.x, (uint32_t)w1.y};
        ok = warp_wait(sm.bar<D>(C::kBarS + t), j & 1, abort_flag);
        if (!ok) break;
        tc_fence_after();
        // Raw logits q.k (the scale is applied inside the exponent; it is > 0),
        // taken 64 columns at a time to keep registers low: one pass for the
        // row maximum, one for the weights.
        // keys key0 + c (lower half) and key0b + c (upper half) with c <= lim,
        // c <= limb are causal
        const int lim = p_row - key0, limb = p_row - w1.z;
        const bool unmasked = valid && (w0.y & kPrefillTileFull) && lim >= 63 && limb >= 63;
        // Weights 2^(s * scale - m) with the running maximum m, two arguments
        // at a time with a packed FMA, rounded to bf16 into wt (32 words per
        // 64 keys).  The normaliser sums the same rounded weights that the PV
        // product takes (eight fp32 chains), so the output is a convex
        // combination of the V rows whatever the rounding.
        // Nothing is stored: S stays intact until the weights are accepted.
        const uint64_t sc2 = f2pack(sc, sc);
        uint32_t wt[2][32];
        auto weights = [&](float m, float& tile_sum) {
            const float nmu = m == -INFINITY ? 0.f : -m;
            const uint64_t nmu2 = f2pack(nmu, nmu);
            float ls[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                uint32_t x[64];
                tmem_ld32(tl + col_s + 64 * hh, *reinterpret_cast<uint32_t(*)[32]>(&x[0]));
                tmem_ld32(tl + col_s + 64 * hh + 32, *reinterpret_cast<uint32_t(*)[32]>(&x[32]));
                tmem_wait_ld();
                if (!unmasked) {
#pragma unroll
                    for (int w = 0; w < 2; ++w) {
                        const int ww = 2 * hh + w;
                        const uint32_t mw =
                            valid ? (vis[ww] & low_bits_through((ww < 2 ? lim : limb) - 32 * (ww & 1))) : 0u;
#pragma unroll
                        for (int c = 0; c < 32; ++c)
                            if (!((mw >> c) & 1u)) x[32 * w + c] = 0xff800000u;  // -inf
                    }
                }
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float x0 = __uint_as_float(x[2 * i]), x1 = __uint_as_float(x[2 * i + 1]);
                    float a0, a1;
                    f2unpack(ffma2(f2pack(x0, x1), sc2, nmu2), a0, a1);
                    const __nv_bfloat162 hb = __floats2bfloat162_rn(ex2_ftz(a0), ex2_ftz(a1));
                    wt[hh][i] = *reinterpret_cast<const uint32_t*>(&hb);
                    add_bf16x2_f32(wt[hh][i], ls[2 * (i & 3)], ls[2 * (i & 3) + 1]);
                }
            }
            tile_sum = ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
        };
        // The maximum is raised lazily, so most tiles keep it: take the
        // weights with the current maximum and accept them when no row's sum
        // exceeds 2^16, which bounds every weight; no maximum is needed for
        // that.  Otherwise (or when a row has seen no key yet) find the tile's
        // maximum and redo the tile with it wherever it exceeds the running
        // one by more than 2^8.
        float mt = -INFINITY, tsum = 0.f;
        bool done = false;
        if (__all_sync(0xffffffffu, m_run != -INFINITY)) {
            weights(m_run, tsum);
            done = !__any_sync(0xffffffffu, tsum > 65536.f);
        }
        if (!done) {
            // row maximum: three-input max over four independent chains
            float mx[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) mx[c] = -INFINITY;
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                uint32_t x[64];
                tmem_ld32(tl + col_s + 64 * hh, *reinterpret_cast<uint32_t(*)[32]>(&x[0]));
                tmem_ld32(tl + col_s + 64 * hh + 32, *reinterpret_cast<uint32_t(*)[32]>(&x[32]));
                tmem_wait_ld();
                if (!unmasked) {
#pragma unroll
                    for (int w = 0; w < 2; ++w) {
                        const int ww = 2 * hh + w;
                        const uint32_t mw =
                            valid ? (vis[ww] & low_bits_through((ww < 2 ? lim : limb) - 32 * (ww & 1))) : 0u;
#pragma unroll
                        for (int c = 0; c < 32; ++c)
                            if (!((mw >> c) & 1u)) x[32 * w + c] = 0xff800000u;  // -inf
                    }
                }
#pragma unroll
                for (int c = 0; c < 64; c += 8) {
                    mx[0] = fmax3(mx[0], __uint_as_float(x[c]), __uint_as_float(x[c + 1]));
                    mx[1] = fmax3(mx[1], __uint_as_float(x[c + 2]), __uint_as_float(x[c + 3]));
                    mx[2] = fmax3(mx[2], __uint_as_float(x[c + 4]), __uint_as_float(x[c + 5]));
                    mx[3] = fmax3(mx[3], __uint_as_float(x[c + 6]), __uint_as_float(x[c + 7]));
                }
            }
            mt = fmaxf(fmax3(mx[0], mx[1], mx[2]), mx[3]) * sc;
        }
        if (done) {
            l += tsum;
        } else {
            const bool need = mt > m_run + 8.f;
            float alpha = 1.f;
            if (need) {
                alpha = exp2f(m_run - mt);
                m_run = mt;
                l *= alpha;
            }
            if (j > 0 && __any_sync(0xffffffffu, need)) {
                // O_t holds the products up to key tile j - 1 (complete: S_t(j)
                // was issued after them): rescale it in place
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t o[32];
                    tmem_ld32(tl + col_o + c * 32, o);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tmem_st32(tl + col_o + c * 32, o);
                }
            }
            weights(m_run, tsum);
            l += tsum;
        }
        // P_t over the first half of S_t: keys 64 hh .. +63 to columns 32 hh .. +31
        tmem_st32(tl + col_s, wt[0]);
        tmem_st32(tl + col_s + 32, wt[1]);
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(sm.bar<D>(C::kBarP + t));
    }
    if (ok && T > 0) ok = warp_wait(sm.bar<D>(C::kBarO + t), 0, abort_flag);
    // dual-key mode: tile b hands its (max, normaliser) to tile a, which
    // merges the two partial results of each row (weights 2^(m_t - max))
    float wa = 1.f, wb = 0.f;
    if (dual) {
        if (t == 1) {
            xchg[2 * row] = m_run;
            xchg[2 * row + 1] = l;
        }
        named_bar_sync(3, 256);
        if (t == 1) {
            if (!ok && lane == 0) {
                set_error(a.err, kErrTimeout);
                *abort_flag = 1;
            }
            return;
        }
        if (ok) ok = warp_wait(sm.bar<D>(C::kBarO + 1), 0, abort_flag);
        const float mb = xchg[2 * row], lb = xchg[2 * row + 1];
        const float M = fmaxf(m_run, mb);
        wa = m_run == -INFINITY ? 0.f : exp2f(m_run - M);
        wb = mb == -INFINITY ? 0.f : exp2f(mb - M);
        l = l * wa + lb * wb;
        m_run = M;
    }
    if (!ok) {
        if (lane == 0) {
            set_error(a.err, kErrTimeout);
            *abort_flag = 1;
        }
        return;
    }
    tc_fence_after();
    const float inv = l > 0.f ? 1.f / l : 0.f;
    const float lse2 = l > 0.f ? m_run + __log2f(l) : -INFINITY;
    const int h = g * a.G + row % a.G;
    float* part_row = nullptr;
    uint8_t* out_row = nullptr;
    if (a.n_split > 1) {
        const size_t pr = ((size_t)blockIdx.x * kPrefillQTiles + t) * kPrefillRows + row;
        part_row = a.part_o + pr * D;
        if (valid) a.part_ml[pr] = lse2;
    } else {
        out_row = reinterpret_cast<uint8_t*>(a.out) +
                  ((size_t)qi * a.Hq + h) * D * (a.out_f32 ? 4 : 2);
        if (valid && a.lse) a.lse[(size_t)qi * a.Hq + h] = lse2 * 0.69314718055994531f;
    }
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        if (T > 0) {
            tmem_ld32(tl + col_o + c * 32, o);
            tmem_wait_ld();
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = 0u;
        }
        float f[32];
        if (dual) {
            uint32_t ob[32];
            tmem_ld32(tl + C::kColO + 128 + c * 32, ob);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i)
                f[i] = (__uint_as_float(o[i]) * wa + __uint_as_float(ob[i]) * wb) * inv;
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) f[i] = __uint_as_float(o[i]) * inv;
        }
        if (!valid) continue;
        if (part_row || a.out_f32) {
            float4* dst = reinterpret_cast<float4*>(part_row ? part_row + c * 32
                                                             : reinterpret_cast<float*>(out_row) + c * 32);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                dst[i] = make_float4(f[4 * i], f[4 * i + 1], f[4 * i + 2], f[4 * i + 3]);
        } else {
            uint4* dst = reinterpret_cast<uint4*>(out_row + c * 64);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 hb = __floats2bfloat162_rn(f[8 * i + 2 * e], f[8 * i + 2 * e + 1]);
                    w[e] = *reinterpret_cast<const uint32_t*>(&hb);
                }
                dst[i] = make_uint4(w[0], w[1], w[2], w[3]);
            }
        }
    }
}

template <int D>
__global__ void __launch_bounds__(320, 1)
    sq_prefill_kernel(const __grid_constant__ CUtensorMap pool_map,
                      const __grid_constant__ CUtensorMap qmap, const PrefillArgs a) {
    using C = PreCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    Smem sm;
    sm.ptr = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                        ~static_cast<uintptr_t>(1023));
    sm.base = smem_addr(sm.ptr);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm.ptr + C::kOffMisc);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm.ptr + C::kOffMisc + 4);
    int* sched = reinterpret_cast<int*>(sm.ptr + C::kOffMisc + 8);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the split-merging kernel that follows may be scheduled from here on
    grid_launch_dependents();
    // heaviest CTA tiles (latest positions) first
    const int split = blockIdx.x % a.n_split;
    const int rest = blockIdx.x / a.n_split;
    const int g = rest % a.Hkv;
    const int qt = a.n_qt - 1 - rest / a.Hkv;
    const int pos_lo = qt * kPrefillQTiles * a.BP;
    if (threadIdx.x == 0) {
        mbar_init(sm.bar<D>(C::kBarQ), 1);
        for (int s = 0; s < C::kSlots; ++s) {
            mbar_init(sm.bar<D>(C::kBarFull + s), 1);
            mbar_init(sm.bar<D>(C::kBarEmpty + s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(sm.bar<D>(C::kBarS + b), 1);
            mbar_init(sm.bar<D>(C::kBarP + b), 128);
            mbar_init(sm.bar<D>(C::kBarO + b), 1);
        }
        mbar_init(sm.bar<D>(C::kBarVfix), 1);
        mbar_init(sm.bar<D>(C::kBarDone), 1);
        fence_mbar_init();
        *abort_flag = 0;
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
        tmem_relinquish();
    }
    // Launched as a programmatic dependent: the set-up above overlapped the
    // preceding kernel's tail; the plan, the queries and the pool are read
    // only from here on.
    grid_dependency_wait();
    if (threadIdx.x == 0) {
        // key tiles up to the CTA tile's last query position, split evenly
        const int lo = __ldg(&a.qt_tiles[qt]);
        const int t0 = (int)((int64_t)lo * split / a.n_split);
        sched[0] = t0;
        sched[1] = (int)((int64_t)lo * (split + 1) / a.n_split) - t0;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int t0 = sched[0], T = sched[1];
    // tile b is empty when every query of the CTA tile fits in tile a; it then
    // takes every other key tile of tile a's queries (dual-key mode)
    const bool two = pos_lo + a.BP < a.n_q;
    const bool dual = !two && T >= 2;
    if (warp == 0) {
        prefill_produce<D>(&pool_map, &qmap, a, sm, g, pos_lo, t0, T, two, dual, abort_flag, lane);
    } else if (warp == 1) {
        if (lane == 0) prefill_mma<D>(a, sm, tmem, T, two, dual, abort_flag);
        __syncwarp();
    } else if (warp < 6 || two || dual) {
        prefill_softmax<D>(a, sm, tmem, (warp - 2) >> 2, g, pos_lo, t0, T, dual, abort_flag, warp,
                           lane);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

// Merges the key-range splits of each query row: weights 2^(lse_s - max).
// One warp per (CTA tile, query tile, row); the lanes take the splits' log-sum-
// exps (up to 64 splits).  The partial outputs of the first 24 splits are
// loaded together with them, so a row of up to 24 splits costs one round trip;
// an empty split's partial (never written) is read but selected away.
template <int D>
__global__ void __launch_bounds__(256) sq_prefill_combine_kernel(const PrefillCombineArgs a) {
    constexpr int V = D / 32;  // output elements per lane
    constexpr int U = 24;      // splits per batch of loads
    // programmatic dependent of the prefill kernel: wait for its partials;
    // the next layer's prefill may then be scheduled
    grid_dependency_wait();
    grid_launch_dependents();
    const int gw = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    const int units = a.n_qt * a.Hkv;
    constexpr int kRowsPerUnit = kPrefillQTiles * kPrefillRows;
    if (gw >= units * kRowsPerUnit) return;
    const int rest = gw / kRowsPerUnit, tr = gw % kRowsPerUnit;
    const int t = tr / kPrefillRows, row = tr % kPrefillRows;
    const int g = rest % a.Hkv, qt = a.n_qt - 1 - rest / a.Hkv;
    const int qi = (qt * kPrefillQTiles + t) * a.BP + row / a.G;
    if (row >= a.BP * a.G || qi >= a.n_q) return;
    const int h = g * a.G + row % a.G;
    // partial row of split s: part0 + s * kRowsPerUnit
    const size_t part0 = ((size_t)rest * a.n_split * kPrefillQTiles + t) * kPrefillRows + row;
    const float ml0 = lane < a.n_split ? a.part_ml[part0 + (size_t)lane * kRowsPerUnit] : -INFINITY;
    const float ml1 =
        lane + 32 < a.n_split ? a.part_ml[part0 + (size_t)(lane + 32) * kRowsPerUnit] : -INFINITY;
    float vals[U][V];
    auto load = [&](int s0) {
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int s = s0 + u;  // the same in every lane
#pragma unroll
            for (int e = 0; e < V; ++e) vals[u][e] = 0.f;
            if (s < a.n_split) {
                const float* po = a.part_o + (part0 + (size_t)s * kRowsPerUnit) * D + lane * V;
                if constexpr (V == 4) {
                    const float4 v = *reinterpret_cast<const float4*>(po);
                    vals[u][0] = v.x; vals[u][1] = v.y; vals[u][2] = v.z; vals[u][3] = v.w;
                } else {
                    const float2 v = *reinterpret_cast<const float2*>(po);
                    vals[u][0] = v.x; vals[u][1] = v.y;
                }
            }
        }
    };
    load(0);
    float M = fmaxf(ml0, ml1);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float w0 = 0.f, w1 = 0.f;
    if (M != -INFINITY) {
        if (ml0 != -INFINITY) w0 = exp2f(ml0 - M);
        if (ml1 != -INFINITY) w1 = exp2f(ml1 - M);
    }
    float W = w0 + w1;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) W += __shfl_xor_sync(0xffffffffu, W, off);
    float acc[V];
#pragma unroll
    for (int e = 0; e < V; ++e) acc[e] = 0.f;
    for (int s0 = 0; W > 0.f && s0 < a.n_split; s0 += U) {
        if (s0 > 0) load(s0);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int s = s0 + u;
            const float ws = __shfl_sync(0xffffffffu, s < 32 ? w0 : w1, s & 31);
            if (s < a.n_split && ws > 0.f) {
#pragma unroll
                for (int e = 0; e < V; ++e) acc[e] += ws * vals[u][e];
            }
        }
    }
    const float inv = W > 0.f ? 1.f / W : 0.f;
    const size_t o = ((size_t)qi * a.Hq + h) * D + lane * V;
    if (a.out_f32) {
        float* out = reinterpret_cast<float*>(a.out) + o;
        if constexpr (V == 4)
            *reinterpret_cast<float4*>(out) =
                make_float4(acc[0] * inv, acc[1] * inv, acc[2] * inv, acc[3] * inv);
        else
            *reinterpret_cast<float2*>(out) = make_float2(acc[0] * inv, acc[1] * inv);
    } else {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out) + o;
        if constexpr (V == 4) {
            uint2 u;
            u.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
            u.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
            *reinterpret_cast<uint2*>(out) = u;
        } else {
            *reinterpret_cast<uint32_t*>(out) = pack_bf16x2(acc[0] * inv, acc[1] * inv);
        }
    }
    if (lane == 0 && a.lse)
        a.lse[(size_t)qi * a.Hq + h] = W > 0.f ? (M + __log2f(W)) * 0.69314718055994531f : -INFINITY;
}

}  // namespace
}  // namespace dev

int prefill_smem_bytes(int D) {
    return D == 128 ? dev::PreCfg<128>::kSmemBytes : dev::PreCfg<64>::kSmemBytes;
}

cudaError_t prefill_prepare(int D) {
    if (D == 128)
        return cudaFuncSetAttribute(dev::sq_prefill_kernel<128>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    dev::PreCfg<128>::kSmemBytes);
    return cudaFuncSetAttribute(dev::sq_prefill_kernel<64>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                dev::PreCfg<64>::kSmemBytes);
}

cudaError_t launch_prefill(const CUtensorMap& pool_map, const CUtensorMap& qmap,
                           const PrefillArgs& a, int D, cudaStream_t st) {
    const unsigned grid = (unsigned)(a.n_qt * a.Hkv * a.n_split);
    if (grid == 0) return cudaSuccess;
    // a programmatic dependent of whatever precedes it: its barrier and tensor
    // memory set-up overlaps that work's tail (it waits before any read)
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.stream = st;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    if (D == 128) {
        cfg.blockDim = dim3(dev::PreCfg<128>::kThreads);
        cfg.dynamicSmemBytes = dev::PreCfg<128>::kSmemBytes;
        return cudaLaunchKernelEx(&cfg, dev::sq_prefill_kernel<128>, pool_map, qmap, a);
    }
    cfg.blockDim = dim3(dev::PreCfg<64>::kThreads);
    cfg.dynamicSmemBytes = dev::PreCfg<64>::kSmemBytes;
    return cudaLaunchKernelEx(&cfg, dev::sq_prefill_kernel<64>, pool_map, qmap, a);
}

cudaError_t launch_prefill_combine(const PrefillCombineArgs& a, int D, cudaStream_t st) {
    const int64_t warps = (int64_t)a.n_qt * a.Hkv * kPrefillQTiles * kPrefillRows;
    const unsigned grid = (unsigned)((warps * 32 + 255) / 256);
    if (grid == 0) return cudaSuccess;
    // scheduled while the prefill kernel's last CTAs run; waits for them
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    if (D == 128) return cudaLaunchKernelEx(&cfg, dev::sq_prefill_combine_kernel<128>, a);
    return cudaLaunchKernelEx(&cfg, dev::sq_prefill_combine_kernel<64>, a);
}

}  // namespace sq
