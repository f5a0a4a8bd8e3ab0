// K/V row movement in the paged pool: append, copy-on-write of a partial
// page, and in-place span-eviction compaction.
//
// Pool layout: [L][num_pages][2 (K, V)][Hkv][P][D] bf16, so the rows of one
// (layer, page, K/V, head) are P*D contiguous elements and one token row is
// D*2 bytes.  All movement is in 16-byte vectors, coalesced along rows.
#include "launch.hpp"
#include "ptx.cuh"

namespace sq {
namespace {

using namespace dev;

__device__ __forceinline__ int64_t row_offset(int64_t num_pages, int Hkv, int P, int D, int layer,
                                              int page, int kv, int head, int slot) {
    return (((((int64_t)layer * num_pages + page) * 2 + kv) * Hkv + head) * P + slot) * (int64_t)D;
}

// ---- append (Algorithm 1: C <- C + R, C <- C + O) ---------------------------
__global__ void __launch_bounds__(256) sq_append_kv_kernel(const AppendArgs a) {
    const int vpr = a.D / 8;  // 16-byte vectors per row
    const int64_t total = (int64_t)a.L * a.n_tok * 2 * a.Hkv * vpr;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = idx;
        const int vc = (int)(r % vpr); r /= vpr;
        const int head = (int)(r % a.Hkv); r /= a.Hkv;
        const int kv = (int)(r % 2); r /= 2;
        const int t = (int)(r % a.n_tok);
        const int layer = (int)(r / a.n_tok);
        const __nv_bfloat16* src = (kv ? a.v : a.k) +
            (((int64_t)layer * a.n_total + a.tok_begin + t) * a.Hkv + head) * a.D + vc * 8;
        const int pos = a.pos0 + t;
        const int pi = pos / a.P - a.page_index0;
        if (pi < 0 || pi >= a.n_pages) { set_error(a.err, kErrBounds); continue; }
        const int page = a.pages[pi];
        if ((uint32_t)page >= (uint64_t)a.num_pages) { set_error(a.err, kErrBounds); continue; }
        __nv_bfloat16* dst = a.pool +
            row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, page, kv, head, pos % a.P) + vc * 8;
        *reinterpret_cast<uint4*>(dst) = __ldg(reinterpret_cast<const uint4*>(src));
    }
}

// ---- copy-on-write of the first `rows` rows of a page, every plane ----------
__global__ void __launch_bounds__(256) sq_cow_copy_kernel(const CowArgs a) {
    const int vpr = a.D / 8;
    const int64_t total = (int64_t)a.L * 2 * a.Hkv * a.rows * vpr;
    if ((uint64_t)a.src_page >= (uint64_t)a.num_pages || (uint64_t)a.dst_page >= (uint64_t)a.num_pages) {
        if (blockIdx.x == 0 && threadIdx.x == 0) set_error(a.err, kErrBounds);
        return;
    }
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = idx;
        const int vc = (int)(r % vpr); r /= vpr;
        const int slot = (int)(r % a.rows); r /= a.rows;
        const int head = (int)(r % a.Hkv); r /= a.Hkv;
        const int kv = (int)(r % 2);
        const int layer = (int)(r / 2);
        const int64_t so = row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, a.src_page, kv, head, slot);
        const int64_t d_o = row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, a.dst_page, kv, head, slot);
        *reinterpret_cast<uint4*>(a.pool + d_o + vc * 8) =
            *reinterpret_cast<const uint4*>(a.pool + so + vc * 8);
    }
}

// ---- span eviction: in-place compaction ---------------------------------------
//
// Algorithm 1, C.clear_kv(Delta_ids): the j-th kept row moves to position j.
// Since the kept positions increase, the source of destination row j is at
// position >= j.  One CTA owns one (layer, K/V, head) plane (or a column
// piece of it) and walks its destination tiles left to right.  The sources
// of tile t sit at positions >= t*R, so
//   * writes of tile t (positions in [t*R, (t+1)*R)) can only clobber sources
//     of tiles <= t; all of tile t's sources are in shared memory (cp.async
//     waited, then a CTA barrier) before any of its writes;
//   * loads of later tiles (positions >= (t+1)*R) never overlap writes of
//     tile t, so they are issued ahead (a 3-stage cp.async ring).
// Destination pages that were copied on write are fresh pages that hold no
// source row, so all their rows are written; other destination rows are
// skipped when they do not move.
constexpr int kEvictThreads = 128;
constexpr int kEvictVecsPerThread = 4;
constexpr int kEvictTileVecs = kEvictThreads * kEvictVecsPerThread;  // 8 KB per stage
constexpr int kEvictStages = 3;

__device__ __forceinline__ int kept_source(const int32_t* run_dst, const int32_t* run_src,
                                           int n_runs, int j) {
    int lo = 0, hi = n_runs - 1;  // last run with run_dst <= j
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(run_dst + mid) <= j) lo = mid;
        else hi = mid - 1;
    }
    return __ldg(run_src + lo) + (j - __ldg(run_dst + lo));
}

__global__ void __launch_bounds__(kEvictThreads) sq_evict_compact_kernel(const EvictArgs a) {
    __shared__ __align__(16) uint8_t buf[kEvictStages][kEvictTileVecs * 16];
    const int plane = blockIdx.x / a.col_split;
    const int piece = blockIdx.x % a.col_split;
    const int head = plane % a.Hkv;
    const int kv = (plane / a.Hkv) % 2;
    const int layer = plane / (2 * a.Hkv);
    const int vpr = a.D / 8 / a.col_split;       // vectors per row piece
    const int rows_per_tile = kEvictTileVecs / vpr;
    const int col0 = piece * vpr * 8;            // first element of the piece
    const int tid = threadIdx.x;
    const int vc = tid % vpr;
    const int row_lane = tid / vpr;
    const int row_step = kEvictThreads / vpr;

    const int t_first = a.first_row / rows_per_tile;
    const int t_end = (a.n_new + rows_per_tile - 1) / rows_per_tile;
    if (t_first >= t_end) return;

    // destination element offset per (stage, vector), -1 = nothing to write
    int64_t dst_off[kEvictStages][kEvictVecsPerThread];

    auto issue = [&](int t, int st) {
#pragma unroll
        for (int k = 0; k < kEvictVecsPerThread; ++k) {
            dst_off[st][k] = -1;
            const int j = t * rows_per_tile + row_lane + k * row_step;
            if (j < a.first_row || j >= a.n_new) continue;
            const int q = j / a.P;
            const int dpage = __ldg(a.new_pt + q);
            const bool fresh = dpage != __ldg(a.old_pt + q);
            const int src = kept_source(a.run_dst, a.run_src, a.n_runs, j);
            if (!fresh && src == j) continue;
            const int sq_ = src / a.P;
            if (sq_ >= a.n_old_pages) { set_error(a.err, kErrBounds); continue; }
            const int spage = __ldg(a.old_pt + sq_);
            if ((uint64_t)spage >= (uint64_t)a.num_pages || (uint64_t)dpage >= (uint64_t)a.num_pages) {
                set_error(a.err, kErrBounds);
                continue;
            }
            const int64_t so = row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, spage, kv, head,
                                          src % a.P) + col0 + vc * 8;
            dst_off[st][k] = row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, dpage, kv, head,
                                        j % a.P) + col0 + vc * 8;
            cp_async_16(smem_addr(&buf[st][(tid + k * kEvictThreads) * 16]), a.pool + so);
        }
        cp_async_commit();
    };

    // prologue: tiles t_first, t_first + 1
#pragma unroll
    for (int s = 0; s < kEvictStages - 1; ++s) {
        if (t_first + s < t_end) issue(t_first + s, s);
        else cp_async_commit();
    }
    int st = 0;
    for (int t = t_first; t < t_end; ++t) {
        const int ahead = t + kEvictStages - 1;
        const int st_ahead = (st + kEvictStages - 1) % kEvictStages;
        if (ahead < t_end) issue(ahead, st_ahead);
        else cp_async_commit();
        cp_async_wait<kEvictStages - 1>();  // tile t has landed (this thread's part)
        __syncthreads();                    // ... and every thread's part
#pragma unroll
        for (int k = 0; k < kEvictVecsPerThread; ++k) {
            if (dst_off[st][k] < 0) continue;
            *reinterpret_cast<uint4*>(a.pool + dst_off[st][k]) =
                *reinterpret_cast<const uint4*>(&buf[st][(tid + k * kEvictThreads) * 16]);
        }
        st = (st + 1) % kEvictStages;
    }
    cp_async_wait<0>();
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, int num_sms, cudaStream_t st) {
    const int64_t total = (int64_t)a.L * a.n_tok * 2 * a.Hkv * (a.D / 8);
    if (total == 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    const int64_t cap = (int64_t)num_sms * 8;
    if (blocks > cap) blocks = cap;
    sq_append_kv_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_cow_copy(const CowArgs& a, int num_sms, cudaStream_t st) {
    const int64_t total = (int64_t)a.L * 2 * a.Hkv * a.rows * (a.D / 8);
    if (total == 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    const int64_t cap = (int64_t)num_sms * 8;
    if (blocks > cap) blocks = cap;
    sq_cow_copy_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

int evict_ctas_per_sm() {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, sq_evict_compact_kernel, kEvictThreads, 0) !=
            cudaSuccess || n < 1)
        return 1;
    return n;
}

cudaError_t launch_evict(const EvictArgs& a, cudaStream_t st) {
    const int blocks = a.L * 2 * a.Hkv * a.col_split;
    if (blocks == 0 || a.first_row >= a.n_new) return cudaSuccess;
    sq_evict_compact_kernel<<<blocks, kEvictThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace sq
