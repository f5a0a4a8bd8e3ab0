// Split-K flash-decoding over the paged bf16 KV pool, with the log-sum-exp
// merge of its partial results in the same kernel.
//
// What is computed (Sec. 1 and Sec. 3.4: for every generated token,
// attention reads the whole KV cache of the context; Sec. 2.1: in
// grouped-query attention a K/V head serves G query heads): for sequence i,
// query head h and KV head g = h / G,
//     out[i][h] = sum_t softmax_t(sm_scale * q[i][h] . K_g[t]) V_g[t].
//
// Work decomposition (host planner, core.cpp): every run of pages that a
// group of sequences holds in common (a main thread and its forked auxiliary
// threads, Sec. 3.4) is one segment; a (segment, KV head) pair is a list of
// 64-token stages; the stages of all pairs are dealt evenly to persistent
// CTAs.  Each CTA streams its stages through a TMA + mbarrier ring in shared
// memory; each of four consumer warps owns 16 tokens of a stage and keeps an
// online-softmax partial (max, sum, unnormalised output) for up to 16 query
// rows — the G heads of every sequence in the group, so a shared page is read
// from HBM once for all of them.
//
// Merge: an item leaves one partial (max, sum, unnormalised output) per group
// member, in that (sequence, KV head)'s contiguous run of entries; a member
// whose run is this one item gets its normalised output directly.  After its
// last item a CTA counts its arrivals on each (sequence, KV head) it touched;
// the CTA that brings a count to the number of entries merges that run
// (max of the maxima, weights 2^(m - M)) and writes the normalised output.
// Counts are zero in every uploaded plan and the completing arrival resets
// its count, so every call starts from zero.
//
// Start-up: the kernel is a programmatic dependent of whatever precedes it.
// When the plan was already on the device (a reused plan), the producer reads
// its item range and first stages into registers and prefetches those stages
// into L2 before the dependency wait; the K/V rows themselves reach shared
// memory only after the wait, through L2, which holds whatever the preceding
// kernel wrote to them.
//
// Page fills: after a ragged eviction a page may hold fewer rows than it has
// slots (its rows first, then zeros or rows once appended).  Stages are in
// slot space (page index x P + slot); the plan then carries every page's
// fill, and the rows past a page's fill get no weight.
//
// Tensor cores: S = Q K^T and O += P V are m16n8k16 bf16 mma.sync with fp32
// accumulation; rows = query rows (<= 16), columns = tokens / head dims.  The
// contraction is tiny (G x d per token) and the kernel is HBM-bound, so the
// warp-level mma is the right size: the point is to keep HBM busy.
#include <math.h>

#include "launch.hpp"
#include "ptx.cuh"

namespace sq {
namespace {

using namespace dev;

template <int D>
struct DecCfg {
    static constexpr int kColBlocks = D / 64;                    // 128-byte column blocks
    static constexpr int kBlockBytes = kStageTokens * 128;       // one column block of a tile
    static constexpr int kTileBytes = kColBlocks * kBlockBytes;  // K (or V) of one stage
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kStages = (D == 128) ? 3 : 6;
    static constexpr int kThreads = (kDecodeConsumerWarps + 1) * 32;
    // item-end merge of the four consumer warps: per-warp row max / sum,
    // and one 16-row output tile
    static constexpr int kMergeStride = D + 8;  // floats per merge row (padded: fewer bank conflicts)
    static constexpr int kMergeBytes = 2 * kDecodeConsumerWarps * kRowsPerTile * 4 +
                                       kRowsPerTile * kMergeStride * 4 + kRowsPerTile * 4;
    // + 1024 alignment slack + 256 for the mbarriers and flags
    static constexpr int kSmemBytes = kStages * kStageBytes + kMergeBytes + 1024 + 256;
    static constexpr int kNT = D / 8;   // 8-wide output column tiles
    static constexpr int kKS = D / 16;  // 16-deep contraction steps
};

__device__ __forceinline__ uint32_t ld_u32(const __nv_bfloat16* p) {
    return *reinterpret_cast<const uint32_t*>(p);
}

// Sum of the two bf16 halves of a packed pair, in fp32.
__device__ __forceinline__ float bf16x2_sum(uint32_t v) {
    return __uint_as_float(v << 16) + __uint_as_float(v & 0xffff0000u);
}

// ---- start-up work before the grid-dependency wait --------------------------
constexpr int kPrefetchStages = 4;  // stages prefetched into L2
constexpr int kFastStages = 3;      // stages whose coordinates are kept in registers

// The coordinates of a CTA's first stages (whole-page stages only, P >= 64):
// the producer issues their loads right after the wait, without re-reading the
// plan there.
struct FastStart {
    int n;                       // stages read (0: none)
    int early;                   // of them, issued before the grid-dependency wait
    int it, s;                   // where the producer continues
    int32_t row[kFastStages];    // K row coordinate head * P + row0 (V: + Hkv * P)
    int32_t pid[kFastStages];
};

__device__ __forceinline__ void fast_start(const DecodeArgs& a, int it0, int it1, FastStart& fs) {
    const int P = a.P;
    int it = it0, s = 0, s1 = 0, head = 0, page_off = 0;
    if (it < it1) {
        const DecodeItem* item = a.items + it;
        s = item->s0;
        s1 = item->s1;
        head = item->head;
        page_off = a.segs[item->seg].page_off;
    }
    fs.n = 0;
#pragma unroll
    for (int k = 0; k < kFastStages; ++k) {
        while (it < it1 && s >= s1) {
            if (++it < it1) {
                const DecodeItem* item = a.items + it;
                s = item->s0;
                s1 = item->s1;
                head = item->head;
                page_off = a.segs[item->seg].page_off;
            }
        }
        if (it < it1) {
            const int tok0 = s * kStageTokens;
            fs.pid[k] = a.page_ids[page_off + tok0 / P];
            fs.row[k] = head * P + tok0 % P;
            fs.n = k + 1;
            ++s;
        }
    }
    fs.it = it;
    fs.s = s;
}

template <int D>
__device__ void prefetch_first_stages(const CUtensorMap* tmap, const DecodeArgs& a, int it0,
                                      int it1) {
    const int P = a.P;
    const int pages_per_stage = P < kStageTokens ? kStageTokens / P : 1;
    int n = 0;
    for (int it = it0; it < it1 && n < kPrefetchStages; ++it) {
        const DecodeItem* item = a.items + it;
        const int head = item->head, s1 = item->s1;
        const DecodeSeg* seg = a.segs + item->seg;
        const int page_off = seg->page_off, n_pages = seg->n_pages;
        for (int s = item->s0; s < s1 && n < kPrefetchStages; ++s, ++n) {
            const int tok0 = s * kStageTokens;
            const int pi0 = tok0 / P;
            const int row0 = P > kStageTokens ? (tok0 % P) : 0;
            const int np = P >= kStageTokens ? 1 : min(pages_per_stage, n_pages - pi0);
            for (int k = 0; k < np; ++k) {
                const int32_t p = a.page_ids[page_off + pi0 + k];
                if ((uint32_t)p >= (uint32_t)a.num_pages) continue;  // reported by the producer
                for (int cb = 0; cb < DecCfg<D>::kColBlocks; ++cb) {
                    tma_prefetch_l2_4d(tmap, cb * 64, head * P + row0, p, a.layer);
                    tma_prefetch_l2_4d(tmap, cb * 64, (a.Hkv + head) * P + row0, p, a.layer);
                }
            }
        }
    }
}

// ---- producer: one thread issues the TMA loads of every stage -------------
// Issues the loads of fast stage k (whole-page stage, ring slot k).
template <int D>
__device__ __forceinline__ void issue_fast_stage(const CUtensorMap* tmap, const DecodeArgs& a,
                                                 const FastStart& fs, int k, uint8_t* smem,
                                                 uint64_t* bars) {
    using C = DecCfg<D>;
    const uint32_t bytes = (uint32_t)kStageTokens * 128u * C::kColBlocks * 2u;
    const uint32_t full = smem_addr(&bars[k]);
    const int32_t p = fs.pid[k];
    if ((uint32_t)p < (uint32_t)a.num_pages) {
        mbar_arrive_expect_tx(full, bytes);
        const uint32_t dk = smem_addr(smem + k * C::kStageBytes);
#pragma unroll
        for (int cb = 0; cb < C::kColBlocks; ++cb) {
            tma_load_4d(dk + cb * C::kBlockBytes, tmap, full, cb * 64, fs.row[k], p, a.layer);
            tma_load_4d(dk + cb * C::kBlockBytes + C::kTileBytes, tmap, full, cb * 64,
                        fs.row[k] + a.Hkv * a.P, p, a.layer);
        }
    } else {
        set_error(a.err, kErrBounds);
        mbar_arrive(full);
    }
}

template <int D>
__device__ void produce(const CUtensorMap* tmap, const DecodeArgs& a, int it0, int it1,
                        const FastStart& fs, uint8_t* smem, uint64_t* bars,
                        volatile int* abort_flag) {
    using C = DecCfg<D>;
    const int P = a.P;
    const int box_rows = P < kStageTokens ? P : kStageTokens;
    const int pages_per_stage = P < kStageTokens ? kStageTokens / P : 1;
    const uint32_t box_bytes = (uint32_t)box_rows * 128u;
    int slot = 0;
    uint32_t phase = 0;
    uint32_t issued = 0, issued_phase = 0;  // per-slot bits of the last issue
    bool ok = true;
    int it_start = it0, s_start = -1;       // -1: the item's first stage
    if (fs.n > 0) {
        // the first stages, from registers (whole-page stages; fresh slots);
        // the first fs.early of them were issued before the dependency wait
#pragma unroll
        for (int k = 0; k < kFastStages; ++k) {
            if (k < fs.n) {
                if (k >= fs.early) issue_fast_stage<D>(tmap, a, fs, k, smem, bars);
                issued |= 1u << k;
            }
        }
        slot = fs.n;
        if (slot == C::kStages) {
            slot = 0;
            phase = 1;
        }
        it_start = fs.it;
        s_start = fs.s;
    }
    for (int it = it_start; it < it1 && ok; ++it) {
        const DecodeItem item = a.items[it];
        const DecodeSeg* seg = a.segs + item.seg;
        const int page_off = seg->page_off, n_pages = seg->n_pages;
        for (int s = (it == it_start && s_start >= 0) ? s_start : item.s0; s < item.s1; ++s) {
            const uint32_t full = smem_addr(&bars[slot]);
            const uint32_t empty = smem_addr(&bars[C::kStages + slot]);
            if (!mbar_wait(empty, phase ^ 1, abort_flag)) {
                if (!*abort_flag) set_error(a.err, kErrTimeout);
                *abort_flag = 1;
                ok = false;
                break;
            }
            if (*abort_flag) {
                ok = false;
                break;
            }
            if ((int)blockIdx.x == a.debug_drop_cta && it == it0 && s == item.s0) {
                // test hook: leave this stage unsignalled (the consumers'
                // bounded wait runs out; nothing is in flight for it)
                if (++slot == C::kStages) {
                    slot = 0;
                    phase ^= 1;
                }
                continue;
            }
            const int tok0 = s * kStageTokens;
            const int pi0 = tok0 / P;
            const int row0 = P > kStageTokens ? (tok0 % P) : 0;
            const int np = P >= kStageTokens ? 1 : min(pages_per_stage, n_pages - pi0);
            int32_t pid[kStageTokens / 8];
            uint32_t vmask = 0;
            for (int k = 0; k < np; ++k) {
                const int32_t p = a.page_ids[page_off + pi0 + k];
                pid[k] = p;
                if ((uint32_t)p < (uint32_t)a.num_pages) vmask |= 1u << k;
                else set_error(a.err, kErrBounds);
            }
            const uint32_t bytes = (uint32_t)__popc(vmask) * box_bytes * C::kColBlocks * 2u;
            uint8_t* stage = smem + slot * C::kStageBytes;
            if (bytes == 0) {
                mbar_arrive(full);
            } else {
                mbar_arrive_expect_tx(full, bytes);
                for (int k = 0; k < np; ++k) {
                    if (!((vmask >> k) & 1u)) continue;
                    for (int cb = 0; cb < C::kColBlocks; ++cb) {
                        const uint32_t dk =
                            smem_addr(stage + cb * C::kBlockBytes + k * box_rows * 128);
                        tma_load_4d(dk, tmap, full, cb * 64, item.head * P + row0, pid[k],
                                    a.layer);
                        tma_load_4d(dk + C::kTileBytes, tmap, full, cb * 64,
                                    (a.Hkv + item.head) * P + row0, pid[k], a.layer);
                    }
                }
            }
            issued |= 1u << slot;
            issued_phase = (issued_phase & ~(1u << slot)) | (phase << slot);
            if (++slot == C::kStages) {
                slot = 0;
                phase ^= 1;
            }
        }
    }
    if (!ok) {
        // Leave only after every copy already issued has landed (bounded).
        for (int sl = 0; sl < C::kStages; ++sl)
            if ((issued >> sl) & 1u)
                mbar_wait(smem_addr(&bars[sl]), (issued_phase >> sl) & 1u);
    }
}

// ---- consumers: four warps, 16 tokens of every stage each ------------------
// Every consumer warp runs every item and every stage and reaches every
// named barrier of every item, also after a wait ran out (it then skips the
// work only), so the barriers never miss a participant.
template <int D>
__device__ void consume(const DecodeArgs& a, int it0, int it1, uint8_t* smem, uint64_t* bars,
                        volatile int* abort_flag, float* merge, int warp, int lane) {
    using C = DecCfg<D>;
    const int gid = lane >> 2, tig = lane & 3;
    const int r0 = gid, r1 = gid + 8;
    const int mi = lane >> 3, rr = lane & 7;
    float* red_m = merge;                                          // [4][16]
    float* red_l = merge + kDecodeConsumerWarps * kRowsPerTile;    // [4][16]
    float* red_o = merge + 2 * kDecodeConsumerWarps * kRowsPerTile;  // [16][kMergeStride]
    float* red_sum = red_o + kRowsPerTile * C::kMergeStride;          // [16] merged row sums
    int slot = 0;
    uint32_t phase = 0;
    bool dead = false;  // warp-uniform: a wait ran out or the CTA aborted
    for (int it = it0; it < it1; ++it) {
        const DecodeItem item = a.items[it];
        const DecodeSeg* seg = a.segs + item.seg;
        const int G = a.G;
        const int n_grp = seg->n_grp;
        const int j0 = r0 / G, j1 = r1 / G;
        const bool v0 = j0 < n_grp, v1 = j1 < n_grp;
        const int lim0 = v0 ? seg->grp_lim[j0] : 0;
        const int lim1 = v1 ? seg->grp_lim[j1] : 0;
        const int n_tok = seg->n_tok;

        uint32_t qa[C::kKS][4];
        {
            const __nv_bfloat16* q0 =
                a.q + ((size_t)(v0 ? seg->grp_seq[j0] : 0) * a.Hq + item.head * G + r0 % G) * D;
            const __nv_bfloat16* q1 =
                a.q + ((size_t)(v1 ? seg->grp_seq[j1] : 0) * a.Hq + item.head * G + r1 % G) * D;
#pragma unroll
            for (int kk = 0; kk < C::kKS; ++kk) {
                const int c = kk * 16 + tig * 2;
                qa[kk][0] = v0 ? ld_u32(q0 + c) : 0u;
                qa[kk][1] = v1 ? ld_u32(q1 + c) : 0u;
                qa[kk][2] = v0 ? ld_u32(q0 + c + 8) : 0u;
                qa[kk][3] = v1 ? ld_u32(q1 + c + 8) : 0u;
            }
        }
        float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
        float o[C::kNT][4];
#pragma unroll
        for (int nd = 0; nd < C::kNT; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;

        for (int s = item.s0; s < item.s1; ++s) {
            const uint32_t full = smem_addr(&bars[slot]);
            const uint32_t empty = smem_addr(&bars[C::kStages + slot]);
            // Pages a ragged eviction left partial: bit r of vm says whether
            // row r of this warp's 16 holds a row of its page (read before
            // the wait, off the critical path).  The unused slots hold zeros
            // or rows once appended, so only their scores are masked.
            uint32_t vm = 0xffffu;
            if (a.page_fill) {
                // P is a power of two >= 8 and the 16 rows start at a multiple
                // of 16: one page holds them all (P >= 16), or two (P = 8)
                const int P = a.P;
                const int t0 = s * kStageTokens + warp * 16;  // segment slot position
                const int pq = t0 >> (__ffs(P) - 1);
                const int f0 = pq < seg->n_pages ? __ldg(&a.page_fill[seg->page_off + pq]) : 0;
                if (P >= 16) {
                    const int v = min(max(f0 - (t0 & (P - 1)), 0), 16);
                    vm = (uint32_t)((1u << v) - 1u);   // v = 16 gives 0xffff
                } else {
                    const int f1 =
                        pq + 1 < seg->n_pages ? __ldg(&a.page_fill[seg->page_off + pq + 1]) : 0;
                    vm = ((1u << min(f0, 8)) - 1u) | (((1u << min(f1, 8)) - 1u) << 8);
                }
            }
            if (!dead) {
                const bool ok = mbar_wait(full, phase, abort_flag);
                if (!__all_sync(0xffffffffu, ok)) {
                    if (lane == 0 && !*abort_flag) set_error(a.err, kErrTimeout);
                    *abort_flag = 1;
                    dead = true;
                }
            }
            if (!dead) {
                const uint32_t kb = smem_addr(smem + slot * C::kStageBytes);
                const uint32_t vb = kb + C::kTileBytes;
                const int tbase = s * kStageTokens + warp * 16;  // segment-relative

                // S = Q K^T over this warp's 16 tokens (two n8 tiles)
                float sc[2][4];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
                {
                    const int t = warp * 16 + (mi >> 1) * 8 + rr;
                    const uint32_t row = kb + t * 128;
                    const int sw = t & 7;
#pragma unroll
                    for (int kk = 0; kk < C::kKS; ++kk) {
                        const int d0 = kk * 16 + (mi & 1) * 8;
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(row + (d0 >> 6) * C::kBlockBytes + ((((d0 & 63) >> 3) ^ sw) << 4), b0,
                                b1, b2, b3);
                        mma_bf16(sc[0], qa[kk], b0, b1);
                        mma_bf16(sc[1], qa[kk], b2, b3);
                    }
                }

                // masking, scaling, online softmax (log2 domain)
                float x[2][4];
                float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int tk = tbase + nt * 8 + tig * 2 + e;
                        const bool rv = (vm >> (nt * 8 + tig * 2 + e)) & 1u;
                        x[nt][e] = tk < lim0 && rv ? sc[nt][e] * a.scale_log2 : -INFINITY;
                        x[nt][2 + e] = tk < lim1 && rv ? sc[nt][2 + e] * a.scale_log2 : -INFINITY;
                        mx0 = fmaxf(mx0, x[nt][e]);
                        mx1 = fmaxf(mx1, x[nt][2 + e]);
                    }
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
                const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
                const float ms0 = mn0 == -INFINITY ? 0.f : mn0;
                const float ms1 = mn1 == -INFINITY ? 0.f : mn1;
                const float al0 = exp2f(m0 - ms0), al1 = exp2f(m1 - ms1);
                m0 = mn0;
                m1 = mn1;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        x[nt][e] = exp2f(x[nt][e] - ms0);
                        x[nt][2 + e] = exp2f(x[nt][2 + e] - ms1);
                    }
                // P in bf16 for the PV product; the normaliser sums the same
                // rounded weights, so the output is an exact convex combination
                uint32_t pa[4];
                pa[0] = pack_bf16x2(x[0][0], x[0][1]);
                pa[1] = pack_bf16x2(x[0][2], x[0][3]);
                pa[2] = pack_bf16x2(x[1][0], x[1][1]);
                pa[3] = pack_bf16x2(x[1][2], x[1][3]);
                const float ps0 = bf16x2_sum(pa[0]) + bf16x2_sum(pa[2]);
                const float ps1 = bf16x2_sum(pa[1]) + bf16x2_sum(pa[3]);
                l0 = l0 * al0 + ps0;
                l1 = l1 * al1 + ps1;
#pragma unroll
                for (int nd = 0; nd < C::kNT; ++nd) {
                    o[nd][0] *= al0;
                    o[nd][1] *= al0;
                    o[nd][2] *= al1;
                    o[nd][3] *= al1;
                }

                // Rows past the last valid token hold stale or never-written
                // shared memory: zero this warp's such V rows so 0 * V stays 0.
                const bool tail = tbase + 16 > n_tok;
                if (tail) {
                    const int first = max(0, n_tok - tbase);
                    const int per_row = C::kColBlocks * 8;  // 16-byte chunks per row
                    const int total = (16 - first) * per_row;
                    uint8_t* vgen = smem + slot * C::kStageBytes + C::kTileBytes;
                    for (int idx = lane; idx < total; idx += 32) {
                        const int row = warp * 16 + first + idx / per_row;
                        const int rem = idx % per_row;
                        *reinterpret_cast<uint4*>(vgen + (rem >> 3) * C::kBlockBytes + row * 128 +
                                                  (rem & 7) * 16) = make_uint4(0, 0, 0, 0);
                    }
                    __syncwarp();
                }

                // O += P V (V^T fragments through ldmatrix.trans)
                {
                    const int t = warp * 16 + (mi & 1) * 8 + rr;
                    const uint32_t row = vb + t * 128;
                    const int sw = t & 7;
#pragma unroll
                    for (int nd2 = 0; nd2 < C::kKS; ++nd2) {
                        const int d0 = nd2 * 16 + (mi >> 1) * 8;
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4_trans(row + (d0 >> 6) * C::kBlockBytes + ((((d0 & 63) >> 3) ^ sw) << 4),
                                      b0, b1, b2, b3);
                        mma_bf16(o[2 * nd2], pa, b0, b1);
                        mma_bf16(o[2 * nd2 + 1], pa, b2, b3);
                    }
                }
                if (tail) fence_proxy_async_smem();  // generic writes before the next TMA fill
                __syncwarp();
                if (lane == 0) mbar_arrive(empty);
            }
            if (++slot == C::kStages) {
                slot = 0;
                phase ^= 1;
            }
        }

        // close the item: merge the four warps' (m, l, o) in shared memory,
        // then write one partial (unnormalised o, m, l) for the item
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
        if (tig == 0) {
            red_m[warp * kRowsPerTile + r0] = dead ? -INFINITY : m0;
            red_m[warp * kRowsPerTile + r1] = dead ? -INFINITY : m1;
            red_l[warp * kRowsPerTile + r0] = dead ? 0.f : l0;
            red_l[warp * kRowsPerTile + r1] = dead ? 0.f : l1;
        }
        named_bar_sync(1, kDecodeConsumerWarps * 32);
        float M0 = -INFINITY, M1 = -INFINITY;
#pragma unroll
        for (int w = 0; w < kDecodeConsumerWarps; ++w) {
            M0 = fmaxf(M0, red_m[w * kRowsPerTile + r0]);
            M1 = fmaxf(M1, red_m[w * kRowsPerTile + r1]);
        }
        const float Ms0 = M0 == -INFINITY ? 0.f : M0, Ms1 = M1 == -INFINITY ? 0.f : M1;
        const float f0 = dead ? 0.f : exp2f(m0 - Ms0), f1 = dead ? 0.f : exp2f(m1 - Ms1);
        // the merged tile: member j's G rows, plus their (M, L), go to its
        // partial entry; a member whose run is this item alone gets its
        // normalised output instead
        const int rows = n_grp * G;
        const int32_t* ent = a.items[it].ent;
        const int sole = a.items[it].sole;
        constexpr int kVecRow = D / 4;  // float4 per row
        if (threadIdx.x < rows) {
            const int r = threadIdx.x;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kDecodeConsumerWarps; ++w) M = fmaxf(M, red_m[w * kRowsPerTile + r]);
            const float Ms = M == -INFINITY ? 0.f : M;
            float L = 0.f;
#pragma unroll
            for (int w = 0; w < kDecodeConsumerWarps; ++w)
                L += red_l[w * kRowsPerTile + r] * exp2f(red_m[w * kRowsPerTile + r] - Ms);
            red_sum[r] = L;
            if (!((sole >> (r / G)) & 1))
                *reinterpret_cast<float4*>(a.part_ml + ((size_t)ent[r / G] * G + r % G) * 4) =
                    make_float4(M, L, 0.f, 0.f);
        }
        // one row's float4 of the merged tile to its destination (read after
        // a barrier that follows the red_sum writes)
        auto put = [&](int r, int c4, float4 v) {
            const int j = r / G;
            if ((sole >> j) & 1) {
                const float inv = 1.f / red_sum[r];
                const size_t ob =
                    ((size_t)seg->grp_seq[j] * a.Hq + item.head * G + r % G) * D + c4 * 4;
                if (a.out_f32) {
                    *reinterpret_cast<float4*>(reinterpret_cast<float*>(a.out) + ob) =
                        make_float4(v.x * inv, v.y * inv, v.z * inv, v.w * inv);
                } else {
                    uint2 u;
                    u.x = pack_bf16x2(v.x * inv, v.y * inv);
                    u.y = pack_bf16x2(v.z * inv, v.w * inv);
                    *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(a.out) + ob) = u;
                }
            } else {
                float* po = a.part_o + ((size_t)ent[j] * G + r % G) * D;
                reinterpret_cast<float4*>(po)[c4] = v;
            }
        };
        if (it + 1 == it1) {
            // The CTA's last item: every warp is past its last stage (the
            // barrier above) and no copy is pending, so the ring is free.
            // Each warp leaves its rows there; all threads add the four.
            float* wo = reinterpret_cast<float*>(smem) + warp * kRowsPerTile * C::kMergeStride;
#pragma unroll
            for (int nd = 0; nd < C::kNT; ++nd) {
                *reinterpret_cast<float2*>(wo + r0 * C::kMergeStride + nd * 8 + tig * 2) =
                    dead ? make_float2(0.f, 0.f) : make_float2(o[nd][0] * f0, o[nd][1] * f0);
                *reinterpret_cast<float2*>(wo + r1 * C::kMergeStride + nd * 8 + tig * 2) =
                    dead ? make_float2(0.f, 0.f) : make_float2(o[nd][2] * f1, o[nd][3] * f1);
            }
            named_bar_sync(1, kDecodeConsumerWarps * 32);
            const float* ro = reinterpret_cast<const float*>(smem);
            for (int v = threadIdx.x; v < rows * kVecRow; v += kDecodeConsumerWarps * 32) {
                const int r = v / kVecRow, c4 = v % kVecRow;
                float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int w = 0; w < kDecodeConsumerWarps; ++w) {
                    const float4 x = *reinterpret_cast<const float4*>(
                        ro + (w * kRowsPerTile + r) * C::kMergeStride + c4 * 4);
                    sum.x += x.x; sum.y += x.y; sum.z += x.z; sum.w += x.w;
                }
                put(r, c4, sum);
            }
        } else {
            // the ring is still in use: the four warps add in turn into one tile
            for (int w = 0; w < kDecodeConsumerWarps; ++w) {
                if (w == warp) {
#pragma unroll
                    for (int nd = 0; nd < C::kNT; ++nd) {
                        float2* p0 = reinterpret_cast<float2*>(red_o + r0 * C::kMergeStride + nd * 8 + tig * 2);
                        float2* p1 = reinterpret_cast<float2*>(red_o + r1 * C::kMergeStride + nd * 8 + tig * 2);
                        float2 a0 = dead ? make_float2(0.f, 0.f) : make_float2(o[nd][0] * f0, o[nd][1] * f0);
                        float2 a1 = dead ? make_float2(0.f, 0.f) : make_float2(o[nd][2] * f1, o[nd][3] * f1);
                        if (w > 0) {
                            const float2 b0 = *p0, b1 = *p1;
                            a0.x += b0.x; a0.y += b0.y;
                            a1.x += b1.x; a1.y += b1.y;
                        }
                        *p0 = a0;
                        *p1 = a1;
                    }
                }
                named_bar_sync(1, kDecodeConsumerWarps * 32);
            }
            for (int v = threadIdx.x; v < rows * kVecRow; v += kDecodeConsumerWarps * 32) {
                const int r = v / kVecRow, c4 = v % kVecRow;
                put(r, c4, *reinterpret_cast<const float4*>(red_o + r * C::kMergeStride + c4 * 4));
            }
        }
        // the merge buffers are rewritten by the next item only after every
        // warp has copied them out
        named_bar_sync(1, kDecodeConsumerWarps * 32);
    }
}

// ---- arrivals and the merge of finished (sequence, KV head) runs -----------
// The arrival word of a run holds two counts.  Its low half counts the items
// that finished (a relaxed add, the claim); the claim that brings it to the
// run's length makes its CTA the merger.  Every other CTA then publishes its
// partial with a release add to the high half, and the merger, instead of
// releasing its own partial first (a GPU-scope fence on its critical path),
// waits with acquire loads until the high half counts the other entries; its
// own partial it reads back within the CTA.  The merger sets the word back to
// zero.  Every CTA claims once per (item, group member), also after a wait ran
// out, so every call leaves every word at zero, and a plan upload writes
// zeros; the word therefore always starts a call at zero.  A run holds at
// most 65,535 entries (the planner's limit), so the halves never carry.

// GPU-scope atomics of the arrival protocol.
__device__ __forceinline__ unsigned atom_add_relaxed_gpu(unsigned* p, unsigned v) {
    unsigned old;
    asm volatile("atom.relaxed.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
__device__ __forceinline__ void red_add_release_gpu(unsigned* p, unsigned v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Up to 4 output float4 per thread per round; a round stages whole runs
// (several when they fit) or one chunk of a long run.
constexpr int kMergeOuts = 4;

// Stages entries [c0, c0 + cn) of run r (first entry e0) at `dst`:
// [cn][G][D] outputs, then [cn][G] (m, l, -, -) records.
template <int D>
__device__ __forceinline__ void stage_run(const DecodeArgs& a, uint32_t dst, int e0, int c0, int cn,
                                          int tid) {
    const int G = a.G;
    const int nv_o = cn * G * (D / 4);
    const float* so = a.part_o + (size_t)(e0 + c0) * G * D;
    for (int v = tid; v < nv_o; v += kDecodeConsumerWarps * 32) cp_async_16(dst + v * 16, so + v * 4);
    const float* sm = a.part_ml + (size_t)(e0 + c0) * G * 4;
    const uint32_t dm = dst + nv_o * 16;
    for (int v = tid; v < cn * G; v += kDecodeConsumerWarps * 32) cp_async_16(dm + v * 16, sm + v * 4);
}

template <int D>
__device__ void arrive_and_merge(const DecodeArgs& a, int it0, int it1, uint8_t* ring, int* smem_i,
                                 int warp) {
    using C = DecCfg<D>;
    constexpr int kT = kDecodeConsumerWarps * 32;
    constexpr int kVec = D / 4;                       // float4 per output row
    const int tid = threadIdx.x;
    const int G = a.G;
    const int outs_run = G * kVec;                    // output float4 of one run (<= 512)
    const int ent_bytes = G * (D * 4 + 16);           // one staged entry
    const int cap = C::kStages * C::kStageBytes / ent_bytes;  // entries per round (>= 11)
    const uint32_t ring_s = smem_addr(ring);
    int* n_last = smem_i;
    int* l_key = smem_i + 1;        // completed runs: key, first entry, entries
    int* l_e0 = l_key + kT;
    int* l_n = l_e0 + kT;
    int total = 0;
    for (int it = it0; it < it1; ++it) total += a.segs[a.items[it].seg].n_grp;
    for (int rb = 0; rb < total; rb += kT) {
        if (tid == 0) *n_last = 0;
        named_bar_sync(1, kT);
        int key = -1;
        for (int it = it0, p = 0; it < it1 && p <= rb + tid; ++it) {
            const DecodeItem* item = a.items + it;
            const DecodeSeg* seg = a.segs + item->seg;
            const int j = rb + tid - p;
            if (j < seg->n_grp && !((item->sole >> j) & 1)) key = seg->grp_seq[j] * a.Hkv + item->head;
            p += seg->n_grp;
        }
        if (key >= 0) {
            const int e0 = a.comb_off[key], n = a.comb_off[key + 1] - e0;
            // claim; a CTA that does not complete the run releases its
            // partials (written before the barrier above) to the merger, which
            // acquires every other entry's before its reads (its own were
            // written within the CTA)
            const unsigned old = atom_add_relaxed_gpu(a.arrive + key, 1u);
            const bool merger = (old & 0xffffu) + 1u == (unsigned)n;
            if (!merger) {
                red_add_release_gpu(a.arrive + key, 0x10000u);
            } else {
                const uint64_t t0 = globaltimer_ns();
                for (uint32_t spin = 1;; ++spin) {
                    if ((ld_acquire_gpu(a.arrive + key) >> 16) == (unsigned)(n - 1)) break;
                    if ((spin & 31) == 0 && globaltimer_ns() - t0 > kWaitLimitNs) {
                        set_error(a.err, kErrTimeout);
                        break;
                    }
                }
            }
            if (merger) {
                a.arrive[key] = 0u;
                const int k = atomicAdd(n_last, 1);
                l_key[k] = key;
                l_e0[k] = e0;
                l_n[k] = n;
            }
        }
        named_bar_sync(1, kT);
        const int nl = *reinterpret_cast<volatile int*>(n_last);
        for (int k = 0; k < nl;) {
            // whole runs while they fit, else chunks of the one run
            int k1 = k, ents = 0;
            while (k1 < nl && ents + l_n[k1] <= cap && (k1 - k + 1) * outs_run <= kMergeOuts * kT)
                ents += l_n[k1++];
            const bool chunked = k1 == k;
            if (chunked) k1 = k + 1;
            const int n_chunk = chunked ? l_n[k] : 0;
            float Mr[kMergeOuts], Lr[kMergeOuts], acc[kMergeOuts][4];
#pragma unroll
            for (int r = 0; r < kMergeOuts; ++r) {
                Mr[r] = -INFINITY;
                Lr[r] = 0.f;
                acc[r][0] = acc[r][1] = acc[r][2] = acc[r][3] = 0.f;
            }
            for (int c0 = 0; c0 < (chunked ? n_chunk : 1); c0 += cap) {
                const int cn_chunk = chunked ? min(cap, n_chunk - c0) : 0;
                // stage
                uint32_t off = 0;
                for (int q = k; q < k1; ++q) {
                    const int cn = chunked ? cn_chunk : l_n[q];
                    stage_run<D>(a, ring_s + off, l_e0[q], chunked ? c0 : 0, cn, tid);
                    off += cn * ent_bytes;
                }
                cp_async_commit();
                cp_async_wait<0>();
                named_bar_sync(1, kT);
                // merge this thread's outputs
#pragma unroll
                for (int r = 0; r < kMergeOuts; ++r) {
                    const int o = tid + r * kT;
                    if (o >= (k1 - k) * outs_run) continue;
                    const int q = k + o / outs_run;
                    const int row = (o % outs_run) / kVec, c4 = o % kVec;
                    uint32_t base = 0;
                    for (int t = k; t < q; ++t) base += l_n[t] * ent_bytes;
                    const int cn = chunked ? cn_chunk : l_n[q];
                    const float4* so = reinterpret_cast<const float4*>(ring + base);
                    const float4* sm = so + cn * G * kVec;
                    float bm = Mr[r];
#pragma unroll 4
                    for (int e = 0; e < cn; ++e) bm = fmaxf(bm, sm[e * G + row].x);
                    const float bs = bm == -INFINITY ? 0.f : bm;
                    const float sc = exp2f(Mr[r] - bs);
                    Lr[r] *= sc;
                    acc[r][0] *= sc; acc[r][1] *= sc; acc[r][2] *= sc; acc[r][3] *= sc;
#pragma unroll 4
                    for (int e = 0; e < cn; ++e) {
                        const float4 ml = sm[e * G + row];
                        const float w = exp2f(ml.x - bs);
                        Lr[r] += w * ml.y;
                        const float4 v = so[(e * G + row) * kVec + c4];
                        acc[r][0] += w * v.x; acc[r][1] += w * v.y;
                        acc[r][2] += w * v.z; acc[r][3] += w * v.w;
                    }
                    Mr[r] = bm;
                }
                named_bar_sync(1, kT);  // the staging is rewritten by the next round
            }
            // normalised outputs
#pragma unroll
            for (int r = 0; r < kMergeOuts; ++r) {
                const int o = tid + r * kT;
                if (o >= (k1 - k) * outs_run) continue;
                const int q = k + o / outs_run;
                const int row = (o % outs_run) / kVec, c4 = o % kVec;
                const int rk = l_key[q];
                const int i = rk / a.Hkv, h = (rk % a.Hkv) * G + row;
                const float inv = 1.f / Lr[r];
                const size_t ob = ((size_t)i * a.Hq + h) * D + c4 * 4;
                if (a.out_f32) {
                    *reinterpret_cast<float4*>(reinterpret_cast<float*>(a.out) + ob) = make_float4(
                        acc[r][0] * inv, acc[r][1] * inv, acc[r][2] * inv, acc[r][3] * inv);
                } else {
                    uint2 u;
                    u.x = pack_bf16x2(acc[r][0] * inv, acc[r][1] * inv);
                    u.y = pack_bf16x2(acc[r][2] * inv, acc[r][3] * inv);
                    *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(a.out) + ob) = u;
                }
            }
            k = k1;
        }
        named_bar_sync(1, kT);  // the list is rewritten by the next batch of arrivals
    }
}

template <int D>
__global__ void __launch_bounds__(DecCfg<D>::kThreads, 2)
    sq_decode_splitk_kernel(const __grid_constant__ CUtensorMap tmap, const DecodeArgs a) {
    using C = DecCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * C::kStages);
    float* merge = reinterpret_cast<float*>(smem + C::kStages * C::kStageBytes + 256);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_addr(&bars[s]), 1);
            mbar_init(smem_addr(&bars[C::kStages + s]), kDecodeConsumerWarps);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    // A reused plan is read before the wait: the producer keeps its item range
    // and first stages in registers and warms L2 with the first stages' rows.
    FastStart fs;
    fs.n = 0;
    fs.early = 0;
    int p_it0 = 0, p_it1 = 0;
    if (warp == kDecodeConsumerWarps && lane == 0) {
        prefetch_tmap(&tmap);
        if (a.plan_ready) {
            p_it0 = a.cta_begin[blockIdx.x];
            p_it1 = a.cta_begin[blockIdx.x + 1];
            if (a.P >= kStageTokens && (int)blockIdx.x != a.debug_drop_cta)
                fast_start(a, p_it0, p_it1, fs);
            prefetch_first_stages<D>(&tmap, a, p_it0, p_it1);
        }
    }
    __syncthreads();
    // Pages no in-flight work writes (the host checked every library write to
    // them is complete; the kernels before this one write no other pool
    // memory) may be loaded before the wait: the first stages stream in while
    // the previous kernel finishes.  Stop at the first stage in a page that
    // may still be written; the rest go out after the wait, in order.
    if (warp == kDecodeConsumerWarps && lane == 0 && a.kv_early && fs.n > 0) {
        for (int k = 0; k < fs.n; ++k) {
            bool unsafe = false;
            for (int u = 0; u < a.n_unsafe; ++u) unsafe |= a.unsafe[u] == fs.pid[k];
            if (unsafe) break;
            issue_fast_stage<D>(&tmap, a, fs, k, smem, bars);
            fs.early = k + 1;
        }
    }
    // Launched as a programmatic dependent: the set-up above overlapped the
    // previous kernel's tail; nothing else it may have written is read before here.
    grid_dependency_wait();
    grid_launch_dependents();  // the next kernel may be scheduled as CTAs retire
    if (warp == kDecodeConsumerWarps) {
        if (lane == 0) {
            if (!a.plan_ready) {
                p_it0 = a.cta_begin[blockIdx.x];
                p_it1 = a.cta_begin[blockIdx.x + 1];
            }
            produce<D>(&tmap, a, p_it0, p_it1, fs, smem, bars, abort_flag);
        }
        return;
    }
    const int it0 = a.cta_begin[blockIdx.x], it1 = a.cta_begin[blockIdx.x + 1];
    consume<D>(a, it0, it1, smem, bars, abort_flag, merge, warp, lane);
    // the ring and the merge buffers are free again (every stage consumed, the
    // last item ended on a barrier)
    arrive_and_merge<D>(a, it0, it1, smem, reinterpret_cast<int*>(merge), warp);
}

}  // namespace

int64_t decode_partial_bytes(int32_t n_ent, int32_t G, int32_t D) {
    return (int64_t)n_ent * G * (D + 4) * (int64_t)sizeof(float);
}

template <int D>
static cudaError_t prepare_one() {
    cudaError_t e = cudaFuncSetAttribute(sq_decode_splitk_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         DecCfg<D>::kSmemBytes);
    if (e != cudaSuccess) return e;
    // the largest shared-memory carveout, so that two CTAs fit on an SM
    return cudaFuncSetAttribute(sq_decode_splitk_kernel<D>,
                                cudaFuncAttributePreferredSharedMemoryCarveout,
                                cudaSharedmemCarveoutMaxShared);
}

cudaError_t decode_prepare(int D) { return D == 128 ? prepare_one<128>() : prepare_one<64>(); }

int decode_ctas_per_sm(int D) {
    int n = 0;
    cudaError_t e;
    if (D == 128)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, sq_decode_splitk_kernel<128>,
                                                          DecCfg<128>::kThreads,
                                                          DecCfg<128>::kSmemBytes);
    else
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, sq_decode_splitk_kernel<64>,
                                                          DecCfg<64>::kThreads,
                                                          DecCfg<64>::kSmemBytes);
    if (e != cudaSuccess || n < 1) return 1;
    return n;
}

// The kernel is launched as a programmatic dependent of whatever precedes it
// on the stream: it waits (griddepcontrol.wait) before it reads anything the
// preceding work may write, so its launch and set-up overlap that work's tail.
static cudaLaunchAttribute pdl_attr() {
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    return at;
}

cudaError_t launch_decode(const CUtensorMap& tmap, const DecodeArgs& a, int n_ctas, int D,
                          cudaStream_t st) {
    cudaLaunchAttribute at = pdl_attr();
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n_ctas);
    cfg.stream = st;
    cfg.attrs = &at;
    cfg.numAttrs = 1;
    if (D == 128) {
        cfg.blockDim = dim3(DecCfg<128>::kThreads);
        cfg.dynamicSmemBytes = DecCfg<128>::kSmemBytes;
        return cudaLaunchKernelEx(&cfg, sq_decode_splitk_kernel<128>, tmap, a);
    }
    cfg.blockDim = dim3(DecCfg<64>::kThreads);
    cfg.dynamicSmemBytes = DecCfg<64>::kSmemBytes;
    return cudaLaunchKernelEx(&cfg, sq_decode_splitk_kernel<64>, tmap, a);
}

}  // namespace sq
