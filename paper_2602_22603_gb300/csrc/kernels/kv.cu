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

// The new lengths of the appended sequences, into the cached decode plans
// that stay valid (block 0; read by later kernels of the stream).
__device__ __forceinline__ void write_lens(const AppendLens& l) {
    if (blockIdx.x == 0 && threadIdx.x < l.n) *l.ptr[threadIdx.x] = l.val[threadIdx.x];
}

// ---- append (Algorithm 1: C <- C + R, C <- C + O) ---------------------------
__global__ void __launch_bounds__(256) sq_append_kv_kernel(const AppendArgs a) {
    write_lens(a.lens);
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

// ---- one new token for each of a batch of sequences --------------------------
__global__ void __launch_bounds__(256) sq_append_kv_batch_kernel(const AppendBatchArgs a) {
    write_lens(a.lens);
    const int vpr = a.D / 8;
    const int64_t total = (int64_t)a.L * a.n * 2 * a.Hkv * vpr;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = idx;
        const int vc = (int)(r % vpr); r /= vpr;
        const int head = (int)(r % a.Hkv); r /= a.Hkv;
        const int kv = (int)(r % 2); r /= 2;
        const int i = (int)(r % a.n);
        const int layer = (int)(r / a.n);
        const int page = a.page[i], slot = a.slot[i];
        if ((uint64_t)page >= (uint64_t)a.num_pages || slot < 0 || slot >= a.P) {
            set_error(a.err, kErrBounds);
            continue;
        }
        const __nv_bfloat16* src = (kv ? a.v : a.k) +
            (((int64_t)layer * a.n_total + a.row0 + i) * a.Hkv + head) * a.D + vc * 8;
        __nv_bfloat16* dst = a.pool +
            row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, page, kv, head, slot) + vc * 8;
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
// position >= j.  The host splits the rows that change into destination
// tiles (contiguous rows of one page, increasing logical order) and each tile
// into contiguous source pieces; the list is the same for every
// (layer, K/V, head) plane.  One CTA owns one plane; one thread drives it
// with 1-D bulk copies (TMA):
//   * bulk loads of tile t's pieces land in a shared-memory slot, tracked by
//     an mbarrier (expect-tx);
//   * after the barrier completes, one bulk store writes the tile back;
//   * the slot is refilled (tile t + S - 1) once that store has read it.
// All sources of tile t sit at positions >= its first destination row, so
// (a) every source a store of tile t could overwrite belongs to tile t or an
// earlier tile, whose loads have all completed before the store is issued,
// and (b) the loads issued ahead for later tiles read positions past every
// row written so far.  Copy-on-write destination pages are fresh pages that
// hold no source row.  No inter-CTA wait is needed.
//
// A ragged eviction's windows share no page, so the tile list is cut at
// window starts into chunks that separate CTAs of one plane run in parallel;
// each chunk keeps the in-order rule above.  A tile without pieces writes
// zeros: the unused slots of a page that a ragged eviction leaves partial.  Its store reads a zero tile that the
// CTA's warp clears once; it writes only past the rows its window kept, and
// later tiles read only later windows' pages.
template <int S>  // ring slots
__global__ void __launch_bounds__(32) sq_evict_compact_kernel(const EvictArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
    const uint32_t row_bytes = (uint32_t)a.D * 2u;
    const uint32_t tile_bytes = (uint32_t)a.tile_rows * row_bytes;
    uint8_t* zero = smem + S * tile_bytes;   // the zero tile (a.zero_tiles only)
    if (a.zero_tiles) {
        for (uint32_t i = threadIdx.x * 16u; i < tile_bytes; i += blockDim.x * 16u)
            *reinterpret_cast<uint4*>(zero + i) = make_uint4(0, 0, 0, 0);
        fence_proxy_async_smem();  // the bulk stores read it through the async proxy
        __syncwarp();
    }
    if (threadIdx.x != 0) return;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (S + (a.zero_tiles ? 1 : 0)) * tile_bytes);
    // CTA = (chunk of independent windows, plane); tiles [tb, te) of the list
    const int planes = a.L * 2 * a.Hkv;
    const int plane = blockIdx.x % planes;
    const int ch = blockIdx.x / planes;
    const int tb = a.chunk ? __ldg(&a.chunk[ch]) : 0;
    const int te = a.chunk ? __ldg(&a.chunk[ch + 1]) : a.n_tiles;
    if (tb < 0 || te > a.n_tiles || tb > te) {
        set_error(a.err, kErrBounds);
        return;
    }
    const int head = plane % a.Hkv;
    const int kv = (plane / a.Hkv) % 2;
    const int layer = plane / (2 * a.Hkv);
    uint8_t* base = reinterpret_cast<uint8_t*>(a.pool) +
                    row_offset(a.num_pages, a.Hkv, a.P, a.D, layer, 0, kv, head, 0) * 2;
    const int64_t page_stride = (int64_t)2 * a.Hkv * a.P * row_bytes;  // bytes between pages
    for (int s = 0; s < S; ++s) mbar_init(smem_addr(&full[s]), 1);
    fence_mbar_init();

    auto issue_loads = [&](int t) {   // t: index in the chunk
        const int slot = t % S;
        const int g = tb + t;
        const uint32_t bar = smem_addr(&full[slot]);
        const uint32_t dst0 = smem_addr(smem + slot * tile_bytes);
        const int pb = __ldg(&a.tiles[g].piece_begin);
        const int pe = g + 1 < a.n_tiles ? __ldg(&a.tiles[g + 1].piece_begin) : a.n_pieces;
        uint32_t bytes = 0;
        for (int k = pb; k < pe; ++k) {
            const EvictPiece pc = a.pieces[k];
            if ((uint64_t)pc.src_page >= (uint64_t)a.num_pages || pc.src_slot < 0 ||
                pc.n_rows <= 0 || pc.src_slot + pc.n_rows > a.P || pc.dst_row < 0 ||
                pc.dst_row + pc.n_rows > a.tile_rows)
                continue;
            bytes += (uint32_t)pc.n_rows * row_bytes;
        }
        if (bytes == 0) {
            mbar_arrive(bar);
        } else {
            mbar_arrive_expect_tx(bar, bytes);
        }
        for (int k = pb; k < pe; ++k) {
            const EvictPiece pc = a.pieces[k];
            if ((uint64_t)pc.src_page >= (uint64_t)a.num_pages || pc.src_slot < 0 ||
                pc.n_rows <= 0 || pc.src_slot + pc.n_rows > a.P || pc.dst_row < 0 ||
                pc.dst_row + pc.n_rows > a.tile_rows) {
                set_error(a.err, kErrBounds);
                continue;
            }
            bulk_load(dst0 + (uint32_t)pc.dst_row * row_bytes,
                      base + pc.src_page * page_stride + (int64_t)pc.src_slot * row_bytes,
                      (uint32_t)pc.n_rows * row_bytes, bar);
        }
    };

    const int T = te - tb;
    for (int t = 0; t < S - 1 && t < T; ++t) issue_loads(t);
    int t = 0;
    for (; t < T; ++t) {
        const int slot = t % S;
        if (!mbar_wait(smem_addr(&full[slot]), (uint32_t)(t / S) & 1u)) {
            set_error(a.err, kErrTimeout);
            break;
        }
        fence_proxy_async_smem();
        const int g = tb + t;
        const EvictTile tl = a.tiles[g];
        const int pe = g + 1 < a.n_tiles ? __ldg(&a.tiles[g + 1].piece_begin) : a.n_pieces;
        const bool zeros = tl.piece_begin == pe;  // no pieces: a tile of zeros
        if ((uint64_t)tl.dst_page < (uint64_t)a.num_pages && tl.dst_slot >= 0 && tl.n_rows > 0 &&
            tl.n_rows <= a.tile_rows && tl.dst_slot + tl.n_rows <= a.P && (!zeros || a.zero_tiles)) {
            bulk_store(base + tl.dst_page * page_stride + (int64_t)tl.dst_slot * row_bytes,
                       smem_addr(zeros ? zero : smem + slot * tile_bytes),
                       (uint32_t)tl.n_rows * row_bytes);
        } else {
            set_error(a.err, kErrBounds);
        }
        bulk_commit();
        const int tn = t + S - 1;
        if (tn < T) {
            bulk_wait_read<1>();  // the store of tile t - 1 has read its slot
            issue_loads(tn);
        }
    }
    if (t < T) {
        // timed out: let the loads already issued land (bounded) before leaving
        for (int u = t + 1; u < T && u < t + S - 1; ++u)
            mbar_wait(smem_addr(&full[u % S]), (uint32_t)(u / S) & 1u);
    }
    bulk_wait<0>();
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

cudaError_t launch_append_batch(const AppendBatchArgs& a, int num_sms, cudaStream_t st) {
    const int64_t total = (int64_t)a.L * a.n * 2 * a.Hkv * (a.D / 8);
    if (total == 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    const int64_t cap = (int64_t)num_sms * 8;
    if (blocks > cap) blocks = cap;
    sq_append_kv_batch_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
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

int evict_smem_bytes(int tile_rows, int D, int stages, bool zero_tiles) {
    return (stages + (zero_tiles ? 1 : 0)) * tile_rows * D * 2 + stages * 8 + 128;
}

// The ring depths built: 3, 4 and 6 slots (the host's choices).
template <typename F>
static cudaError_t with_evict_kernel(int stages, F f) {
    switch (stages) {
        case 3: return f(sq_evict_compact_kernel<3>);
        case 4: return f(sq_evict_compact_kernel<4>);
        case 6: return f(sq_evict_compact_kernel<6>);
        default: return cudaErrorInvalidValue;
    }
}

int evict_ctas_per_sm(int tile_rows, int D, int stages) {
    int n = 0;
    const cudaError_t e = with_evict_kernel(stages, [&](auto kernel) {
        return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, 32,
                                                             evict_smem_bytes(tile_rows, D, stages));
    });
    return e != cudaSuccess || n < 1 ? 1 : n;
}

cudaError_t evict_prepare() {
    for (int stages : {3, 4, 6}) {
        const cudaError_t e = with_evict_kernel(stages, [&](auto kernel) {
            return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        evict_smem_bytes(kStageTokens, 128, stages, true));
        });
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_evict(const EvictArgs& a, cudaStream_t st) {
    const int blocks = a.L * 2 * a.Hkv * (a.chunk ? a.n_chunks : 1);
    if (blocks == 0 || a.n_tiles == 0) return cudaSuccess;
    const int smem = evict_smem_bytes(a.tile_rows, a.D, a.stages, a.zero_tiles != 0);
    const cudaError_t e = with_evict_kernel(a.stages, [&](auto kernel) {
        kernel<<<blocks, 32, smem, st>>>(a);
        return cudaSuccess;
    });
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace sq
