// libsq C ABI: validation, transactional host state, plan upload, launches.
// See include/sq.h for the contract of every call.
#include "sq.h"

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cstddef>
#include <cstring>
#include <deque>
#include <memory>
#include <new>
#include <unordered_map>
#include <vector>

#include "../host/core.hpp"
#include "../kernels/launch.hpp"
#include "../kernels/noalloc.hpp"

using namespace sq;

namespace {

// An NVTX range around every C-ABI call, so that a timeline tool shows the
// library's calls next to their kernels (no cost without an attached tool).
struct TraceRange {
    explicit TraceRange(const char* name) { nvtxRangePushA(name); }
    ~TraceRange() { nvtxRangePop(); }
};

constexpr int kPlanCacheEntries = 8;
constexpr int kUploadSlots = 8;

struct PlanEntry {
    bool valid = false;
    int32_t n_ctas = 0;
    std::vector<int32_t> handles;
    std::vector<uint64_t> versions;
    DecodePlanLayout lay{};
    int64_t unique_tokens = 0, logical_tokens = 0;
    int32_t first_busy_cta = 0;  // lowest CTA with work (target of the test hook)
    // write tickets of the plan's pages (fixed while the plan is valid: a
    // write to a page changes the version of every sequence holding it): the
    // kDecodeMaxUnsafe newest (ticket, page) pairs and the newest ticket of
    // all other pages
    std::vector<std::pair<uint64_t, int32_t>> tick_top;
    uint64_t tick_rest = 0;
    // per call-local sequence: the segment holding its last page when that
    // segment has it alone (else -1), the slot-space start of that run, and
    // the last page's entry in page_fill (plans with page fills)
    std::vector<int32_t> tail_seg, tail_base, tail_fill;
    uint8_t* d_plan = nullptr;
    size_t plan_cap = 0;
    float* d_part = nullptr;
    size_t part_cap = 0;
    cudaEvent_t ev = nullptr;   // recorded after the last launch that used it
    bool ev_recorded = false;
    cudaStream_t ev_stream = nullptr;  // ... on this stream (work on it is ordered after anyway)
    uint64_t last_use = 0;
};

// Prefill plans, reused while the sequence (its version), the query count,
// the spans and the CTA target stay the same: the layers of one step share
// one plan, planned and uploaded once.
constexpr int kPrefillPlanEntries = 4;
struct PrefillPlanEntry {
    bool valid = false;
    int32_t seq = 0;
    uint64_t version = 0;
    int32_t n_q = 0;
    int32_t target = 0;
    std::vector<int32_t> spans;  // start, end pairs as passed
    size_t tb = 0, qb = 0;       // bytes of the tile records, of the per-CTA-tile counts
    int32_t n_tiles = 0, n_pieces = 0, BP = 0, n_qt = 0, n_split = 0;
    int64_t visible_pairs = 0;
    uint8_t* d = nullptr;  // [tiles][qt_tiles][tile_pages]
    size_t cap = 0;
    cudaEvent_t ev = nullptr;  // recorded after the last launch that used it
    bool ev_recorded = false;
    cudaStream_t ev_stream = nullptr;  // ... on this stream
    uint64_t last_use = 0;
};

struct UploadSlot {
    uint8_t* d = nullptr;
    size_t cap = 0;
    cudaEvent_t ev = nullptr;
    bool ev_recorded = false;
    cudaStream_t ev_stream = nullptr;
};

// Pinned host staging for uploads: a copy from pageable memory may wait for
// the stream's earlier work (draining the GPU between calls); from pinned
// memory it is a plain asynchronous DMA.  A buffer is refilled only after the
// copy that last used it has run.
constexpr int kPinnedSlots = 8;
// Capacity the cache gives each upload buffer (device) and each pinned staging
// buffer when it is created, so that the first eviction or plan upload of its
// life allocates nothing on its path (measured: a first 32k-token eviction
// spent ~170 us more in the call than later ones).  Larger uploads still grow
// a buffer.
constexpr size_t kUploadInitBytes = 256 << 10;
constexpr size_t kPinnedInitBytes = 256 << 10;
// Pinned staging of sq_decode_attention_noalloc's plans, allocated with the
// cache: two slots of 2 MiB (a decode plan of 16 sequences of 2^17 tokens is
// ~0.2 MiB); a larger plan is copied from pageable memory instead.
constexpr int kNoallocPinnedSlots = 2;
constexpr size_t kNoallocPinnedBytes = 2u << 20;
struct PinnedSlot {
    uint8_t* h = nullptr;
    size_t cap = 0;
    cudaEvent_t ev = nullptr;
    bool ev_recorded = false;
};

}  // namespace

struct sq_cache {
    Geometry g;
    std::unique_ptr<HostCache> host;
    int device = 0;
    int num_sms = 0;
    int decode_ctas = 0;
    int evict_tile_rows = 0;
    int evict_stages = 0;
    int64_t evict_resident = 0;  // eviction CTAs resident on the device at once
    __nv_bfloat16* pool = nullptr;
    bool own_pool = false;
    size_t pool_bytes = 0;
    CUtensorMap tmap;
    void* encode_fn = nullptr;  // cuTensorMapEncodeTiled
    int* d_err = nullptr;
    // prefill split-K partials, reused by every call (grown on demand)
    float* pre_part = nullptr;
    size_t pre_part_cap = 0;
    cudaEvent_t pre_ev = nullptr;
    bool pre_ev_recorded = false;
    cudaStream_t pre_ev_stream = nullptr;
    PlanEntry plans[kPlanCacheEntries];
    PrefillPlanEntry pre_plans[kPrefillPlanEntries];
    uint64_t use_clock = 0;
    UploadSlot slots[kUploadSlots];
    int next_slot = 0;
    PinnedSlot pinned[kPinnedSlots];
    int next_pinned = 0;
    std::vector<uint8_t> staging;
    // sq_decode_attention_noalloc: the device address of the library's fixed
    // scratch on this cache's device (resolved at creation; null if that
    // failed, with the status kept), and pinned staging for its plan uploads,
    // allocated at creation too
    uint8_t* noalloc_base = nullptr;
    int noalloc_status = SQ_OK;
    PinnedSlot noalloc_pinned[kNoallocPinnedSlots];
    int next_noalloc_pinned = 0;
    // pages freed by work on a stream become reusable elsewhere only after
    // that work: the stream that freed each free page, and one event per
    // stream recorded after its latest freeing operation
    std::vector<void*> freed_on;
    std::vector<uint8_t> fenced;
    std::unordered_map<void*, cudaEvent_t> free_event;
    // Writes to the pool by the library's kernels: every append, copy-on-write
    // and eviction takes a ticket, stamps the pages it writes and records an
    // event; write_done is the newest ticket whose work, and all before it,
    // is known complete.
    uint64_t write_seq = 0, write_done = 0;
    bool early_ok = true;
    std::vector<uint64_t> page_ticket;
    std::deque<std::pair<uint64_t, cudaEvent_t>> write_pending;
    std::vector<cudaEvent_t> write_events;  // recycled
    int32_t debug_flags = 0;
    sq_stats_t stats;
};

namespace {

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

int cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return SQ_OK;
    if (e == cudaErrorMemoryAllocation) return SQ_ERR_NO_MEMORY;
    return SQ_ERR_CUDA;
}

int geometry_from(const sq_config* cfg, Geometry* g) {
    if (!cfg) return SQ_ERR_INVALID_ARG;
    g->L = cfg->num_layers;
    g->Hq = cfg->num_q_heads;
    g->Hkv = cfg->num_kv_heads;
    g->D = cfg->head_dim;
    g->P = cfg->page_size;
    g->num_pages = cfg->num_pages;
    g->max_seqs = cfg->max_seqs;
    g->max_pages_per_seq = cfg->max_pages_per_seq;
    return check_geometry(*g);
}

size_t pool_bytes_of(const Geometry& g) {
    return (size_t)g.L * g.num_pages * 2 * g.Hkv * g.P * g.D * sizeof(__nv_bfloat16);
}

int make_tensor_map(sq_cache* c) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
        return SQ_ERR_CUDA;
    c->encode_fn = fn;
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    const Geometry& g = c->g;
    // dims, innermost first: head dim, row within a (layer, page) block
    // ((kv * Hkv + head) * P + slot), page, layer
    cuuint64_t dims[4] = {(cuuint64_t)g.D, (cuuint64_t)2 * g.Hkv * g.P, (cuuint64_t)g.num_pages,
                          (cuuint64_t)g.L};
    cuuint64_t strides[3] = {(cuuint64_t)g.D * 2, (cuuint64_t)2 * g.Hkv * g.P * g.D * 2,
                             (cuuint64_t)g.num_pages * 2 * g.Hkv * g.P * g.D * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)std::min(g.P, kStageTokens), 1, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = encode(&c->tmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, c->pool, dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? SQ_OK : SQ_ERR_UNSUPPORTED;
}

// Before `stream` writes pages taken from the free list, wait for the work
// that freed them on other streams.
int fence_taken_pages(sq_cache* c, const std::vector<int32_t>& taken, void* stream) {
    void* waited[8];
    int n_waited = 0;
    for (int32_t p : taken) {
        if (!c->fenced[p]) continue;
        c->fenced[p] = 0;
        void* s = c->freed_on[p];
        if (s == stream) continue;
        bool seen = false;
        for (int i = 0; i < n_waited; ++i) seen |= waited[i] == s;
        if (seen) continue;
        auto it = c->free_event.find(s);
        if (it == c->free_event.end()) continue;
        cudaError_t e = cudaStreamWaitEvent(as_stream(stream), it->second, 0);
        if (e != cudaSuccess) return cuda_status(e);
        if (n_waited < 8) waited[n_waited++] = s;
    }
    return SQ_OK;
}

// Marks pages freed by the work enqueued on `stream` so far.
int record_freed(sq_cache* c, const std::vector<int32_t>& freed, void* stream) {
    if (freed.empty()) return SQ_OK;
    auto it = c->free_event.find(stream);
    if (it == c->free_event.end()) {
        cudaEvent_t ev;
        cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_status(e);
        it = c->free_event.emplace(stream, ev).first;
    }
    cudaError_t e = cudaEventRecord(it->second, as_stream(stream));
    if (e != cudaSuccess) return cuda_status(e);
    for (int32_t p : freed) {
        c->freed_on[p] = stream;
        c->fenced[p] = 1;
    }
    return SQ_OK;
}

// Stamps the pages a pool-writing launch just enqueued on `stream` writes.
// If the event cannot be recorded, decode stops loading anything before its
// dependency wait for the rest of the cache's life.
void note_writes(sq_cache* c, const int32_t* pages, size_t n, void* stream) {
    if (n == 0 || !c->early_ok) return;
    const uint64_t t = ++c->write_seq;
    for (size_t i = 0; i < n; ++i)
        if (pages[i] >= 0 && pages[i] < c->g.num_pages) c->page_ticket[pages[i]] = t;
    cudaEvent_t ev;
    if (!c->write_events.empty()) {
        ev = c->write_events.back();
        c->write_events.pop_back();
    } else if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        c->early_ok = false;
        return;
    }
    if (cudaEventRecord(ev, as_stream(stream)) != cudaSuccess) {
        cudaGetLastError();
        c->write_events.push_back(ev);
        c->early_ok = false;
        return;
    }
    c->write_pending.push_back({t, ev});
}

// Advances write_done over the writes whose events have completed, in
// ticket order (a write still running holds back every later ticket).
void poll_writes(sq_cache* c) {
    while (!c->write_pending.empty()) {
        const cudaError_t q = cudaEventQuery(c->write_pending.front().second);
        if (q == cudaErrorNotReady) break;
        if (q != cudaSuccess) {   // leave the ticket pending; the error surfaces elsewhere
            cudaGetLastError();
            break;
        }
        c->write_done = c->write_pending.front().first;
        c->write_events.push_back(c->write_pending.front().second);
        c->write_pending.pop_front();
    }
}

// Asynchronous host -> device copy of `bytes` from `src` through a pinned
// staging buffer; `src` may be reused as soon as this returns.
int staged_copy(sq_cache* c, void* dst, const void* src, size_t bytes, void* stream) {
    PinnedSlot& p = c->pinned[c->next_pinned];
    c->next_pinned = (c->next_pinned + 1) % kPinnedSlots;
    cudaError_t e;
    if (!p.ev) {
        e = cudaEventCreateWithFlags(&p.ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_status(e);
    }
    if (p.ev_recorded) {
        e = cudaEventSynchronize(p.ev);
        if (e != cudaSuccess) return cuda_status(e);
    }
    if (bytes > p.cap) {
        if (p.h) cudaFreeHost(p.h);
        p.h = nullptr;
        p.cap = 0;
        const size_t cap = std::max<size_t>(bytes * 5 / 4, 64 << 10);
        e = cudaHostAlloc(reinterpret_cast<void**>(&p.h), cap, cudaHostAllocDefault);
        if (e != cudaSuccess) return cuda_status(e);
        p.cap = cap;
    }
    std::memcpy(p.h, src, bytes);
    e = cudaMemcpyAsync(dst, p.h, bytes, cudaMemcpyHostToDevice, as_stream(stream));
    if (e != cudaSuccess) return cuda_status(e);
    e = cudaEventRecord(p.ev, as_stream(stream));
    if (e != cudaSuccess) return cuda_status(e);
    p.ev_recorded = true;
    return SQ_OK;
}

int upload(sq_cache* c, UploadSlot& s, const void* src, size_t bytes, void* stream) {
    if (bytes > s.cap) {
        if (s.d) {
            if (s.ev_recorded) cudaEventSynchronize(s.ev);
            cudaFree(s.d);
            s.d = nullptr;
            s.cap = 0;
        }
        size_t cap = std::max<size_t>(bytes, 4096);
        cudaError_t e = cudaMalloc(&s.d, cap);
        if (e != cudaSuccess) return cuda_status(e);
        s.cap = cap;
        s.ev_recorded = false;
    }
    // work on the stream that recorded the event is ordered after it already
    if (s.ev_recorded && s.ev_stream != as_stream(stream)) {
        cudaError_t e = cudaStreamWaitEvent(as_stream(stream), s.ev, 0);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return staged_copy(c, s.d, src, bytes, stream);
}

void free_entry(PlanEntry& p) {
    if (p.d_plan) cudaFree(p.d_plan);
    if (p.d_part) cudaFree(p.d_part);
    if (p.ev) cudaEventDestroy(p.ev);
    p = PlanEntry();
}

// Eviction CTA shape (evict_tile_rows_for, evict_stages_for) and the CTAs
// of it resident on the device at once.
void choose_evict_shape(sq_cache* c) {
    const int64_t planes = (int64_t)c->g.L * 2 * c->g.Hkv;
    c->evict_tile_rows = evict_tile_rows_for(c->g.P, c->g.D);
    c->evict_stages = evict_stages_for(planes, c->num_sms);
    c->evict_resident =
        (int64_t)c->num_sms * evict_ctas_per_sm(c->evict_tile_rows, c->g.D, c->evict_stages);
}

}  // namespace

extern "C" {

const char* sq_strerror(int code) {
    switch (code) {
        case SQ_OK: return "SQ_OK";
        case SQ_ERR_INVALID_ARG: return "SQ_ERR_INVALID_ARG";
        case SQ_ERR_BAD_HANDLE: return "SQ_ERR_BAD_HANDLE";
        case SQ_ERR_NO_PAGES: return "SQ_ERR_NO_PAGES";
        case SQ_ERR_CAPACITY: return "SQ_ERR_CAPACITY";
        case SQ_ERR_CUDA: return "SQ_ERR_CUDA";
        case SQ_ERR_DEVICE: return "SQ_ERR_DEVICE";
        case SQ_ERR_DEVICE_TIMEOUT: return "SQ_ERR_DEVICE_TIMEOUT";
        case SQ_ERR_UNSUPPORTED: return "SQ_ERR_UNSUPPORTED";
        case SQ_ERR_NO_MEMORY: return "SQ_ERR_NO_MEMORY";
        default: return "SQ_ERR_UNKNOWN";
    }
}

size_t sq_pool_bytes(const sq_config* cfg) {
    Geometry g;
    if (geometry_from(cfg, &g) != SQ_OK) return 0;
    return pool_bytes_of(g);
}

int sq_cache_create(const sq_config* cfg, sq_cache** out) {
    TraceRange trace_("sq_cache_create");
    if (!out) return SQ_ERR_INVALID_ARG;
    *out = nullptr;
    Geometry g;
    int rc = geometry_from(cfg, &g);
    if (rc != SQ_OK) return rc;
    if (cfg->decode_ctas < 0) return SQ_ERR_INVALID_ARG;
    if (cfg->kv_pool && (reinterpret_cast<uintptr_t>(cfg->kv_pool) & 255)) return SQ_ERR_INVALID_ARG;
    std::unique_ptr<sq_cache> c(new (std::nothrow) sq_cache());
    if (!c) return SQ_ERR_NO_MEMORY;
    c->g = g;
    c->host.reset(new (std::nothrow) HostCache(g));
    if (!c->host) return SQ_ERR_NO_MEMORY;
    c->freed_on.assign(g.num_pages, nullptr);
    c->fenced.assign(g.num_pages, 0);
    c->page_ticket.assign(g.num_pages, 0);
    std::memset(&c->stats, 0, sizeof c->stats);
    cudaError_t e = cudaGetDevice(&c->device);
    if (e != cudaSuccess) return cuda_status(e);
    e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) return cuda_status(e);
    e = decode_prepare(g.D);
    if (e != cudaSuccess) return cuda_status(e);
    c->decode_ctas = cfg->decode_ctas > 0 ? cfg->decode_ctas : c->num_sms * decode_ctas_per_sm(g.D);
    e = evict_prepare();
    if (e != cudaSuccess) return cuda_status(e);
    e = prefill_prepare(g.D);
    if (e != cudaSuccess) return cuda_status(e);
    choose_evict_shape(c.get());
    c->pool_bytes = pool_bytes_of(g);
    if (cfg->kv_pool) {
        c->pool = reinterpret_cast<__nv_bfloat16*>(cfg->kv_pool);
    } else {
        e = cudaMalloc(&c->pool, c->pool_bytes);
        if (e != cudaSuccess) return cuda_status(e);
        c->own_pool = true;
        e = cudaMemset(c->pool, 0, c->pool_bytes);
        if (e != cudaSuccess) {
            cudaFree(c->pool);
            return cuda_status(e);
        }
    }
    auto fail = [&](int code) {
        if (c->own_pool) cudaFree(c->pool);
        if (c->d_err) cudaFree(c->d_err);
        for (auto& s : c->slots) {
            if (s.d) cudaFree(s.d);
            s.d = nullptr;
        }
        for (auto& p : c->pinned) {
            if (p.h) cudaFreeHost(p.h);
            p.h = nullptr;
        }
        for (auto& p : c->noalloc_pinned) {
            if (p.h) cudaFreeHost(p.h);
            if (p.ev) cudaEventDestroy(p.ev);
        }
        return code;
    };
    // [0] device error word, [1] sink of the read probe
    e = cudaMalloc(&c->d_err, 4 * sizeof(int));
    if (e != cudaSuccess) return fail(cuda_status(e));
    e = cudaMemset(c->d_err, 0, 4 * sizeof(int));
    if (e != cudaSuccess) return fail(cuda_status(e));
    rc = make_tensor_map(c.get());
    if (rc != SQ_OK) return fail(rc);
    for (auto& s : c->slots) {
        e = cudaEventCreateWithFlags(&s.ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return fail(cuda_status(e));
        e = cudaMalloc(&s.d, kUploadInitBytes);
        if (e != cudaSuccess) return fail(cuda_status(e));
        s.cap = kUploadInitBytes;
    }
    for (auto& p : c->pinned) {
        e = cudaHostAlloc(reinterpret_cast<void**>(&p.h), kPinnedInitBytes, cudaHostAllocDefault);
        if (e != cudaSuccess) return fail(cuda_status(e));
        p.cap = kPinnedInitBytes;
    }
    // The no-alloc decode's scratch: looking its address up loads its module
    // on this device now, so that the decode call itself loads and allocates
    // nothing.  A failure here only disables that call.
    {
        void* base = nullptr;
        c->noalloc_status = noalloc_scratch(&base);
        c->noalloc_base = static_cast<uint8_t*>(base);
        if (c->noalloc_status != SQ_OK) cudaGetLastError();
        for (auto& p : c->noalloc_pinned) {
            if (c->noalloc_status != SQ_OK) break;
            e = cudaEventCreateWithFlags(&p.ev, cudaEventDisableTiming);
            if (e == cudaSuccess)
                e = cudaHostAlloc(reinterpret_cast<void**>(&p.h), kNoallocPinnedBytes,
                                  cudaHostAllocDefault);
            if (e != cudaSuccess) {
                cudaGetLastError();
                c->noalloc_status = cuda_status(e);
                break;
            }
            p.cap = kNoallocPinnedBytes;
        }
    }
    e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return fail(cuda_status(e));
    *out = c.release();
    return SQ_OK;
}

int sq_cache_destroy(sq_cache* c) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    cudaDeviceSynchronize();
    for (auto& p : c->plans) free_entry(p);
    for (auto& p : c->pre_plans) {
        if (p.d) cudaFree(p.d);
        if (p.ev) cudaEventDestroy(p.ev);
    }
    for (auto& s : c->slots) {
        if (s.d) cudaFree(s.d);
        if (s.ev) cudaEventDestroy(s.ev);
    }
    for (auto& p : c->pinned) {
        if (p.h) cudaFreeHost(p.h);
        if (p.ev) cudaEventDestroy(p.ev);
    }
    for (auto& p : c->noalloc_pinned) {
        if (p.h) cudaFreeHost(p.h);
        if (p.ev) cudaEventDestroy(p.ev);
    }
    for (auto& kv : c->free_event) cudaEventDestroy(kv.second);
    for (auto& w : c->write_pending) cudaEventDestroy(w.second);
    for (cudaEvent_t ev : c->write_events) cudaEventDestroy(ev);
    if (c->pre_part) cudaFree(c->pre_part);
    if (c->pre_ev) cudaEventDestroy(c->pre_ev);
    if (c->d_err) cudaFree(c->d_err);
    if (c->own_pool) cudaFree(c->pool);
    delete c;
    return SQ_OK;
}

int sq_seq_new(sq_cache* c, sq_seq* out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!out) return SQ_ERR_INVALID_ARG;
    return c->host->seq_new(out);
}

int sq_fork_aux(sq_cache* c, sq_seq parent, sq_seq* child_out) {
    TraceRange trace_("sq_fork_aux");
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!child_out) return SQ_ERR_INVALID_ARG;
    return c->host->fork(parent, child_out);
}

// Cached decode plans an append leaves valid.  An append that stays inside
// a sequence's last page (no new page, no copy-on-write) and inside its last
// 64-token stage changes, for a plan holding that sequence, only the row
// limit of the run holding that page: the stages, the CTA split and every
// page stay as they were.  The page is the sequence's alone (else it would
// have been copied on write), so that run's segment has it as its one member
// and the limit is two words of the segment (its token count and the member's
// limit).  The append kernel rewrites them, after the plan's last decode on
// the same stream, and the plan takes the sequence's new version; a plan
// with page fills also gets the last page's new fill.  Plans last used on
// another stream, and pages of fewer than 64 tokens (a stage spans pages),
// are rebuilt instead.
struct LenUpdate {
    PlanEntry* e;
    int32_t i;     // call-local index of the sequence in the plan
    int32_t val;   // the new row limit of its last run (end in slot space - run start)
    int32_t fill;  // the new fill of its last page
};

static void plan_len_updates(sq_cache* c, sq_seq seq, const AppendPlan& ap, uint64_t old_version,
                             cudaStream_t st, std::vector<LenUpdate>* out) {
    if (c->g.P % kStageTokens != 0 || ap.cow || !ap.taken.empty() || ap.n_new < 1) return;
    const int64_t e0 = ap.pos0, e1 = (int64_t)ap.pos0 + ap.n_new;
    if ((e0 + kStageTokens - 1) / kStageTokens != (e1 + kStageTokens - 1) / kStageTokens) return;
    const int32_t fill = (int32_t)(e1 - (int64_t)ap.first_page_index * c->g.P);
    for (auto& e : c->plans) {
        if (!e.valid || !e.ev_recorded || e.ev_stream != st) continue;
        for (size_t i = 0; i < e.handles.size(); ++i)
            if (e.handles[i] == seq && e.versions[i] == old_version && e.tail_seg[i] >= 0)
                out->push_back({&e, (int32_t)i, (int32_t)(e1 - e.tail_base[i]), fill});
    }
}

// Words the kernel rewrites for one update: the run's token count, its one
// member's limit, and (plans with page fills) the last page's fill.
static int update_words(const LenUpdate& u) { return u.e->lay.page_fill >= 0 ? 3 : 2; }

// The kernel's writes for `ups` (from index `from`), as many updates as fit
// whole; returns how many were taken.
static size_t fill_lens(const std::vector<LenUpdate>& ups, size_t from, AppendLens* l) {
    l->n = 0;
    size_t k = from;
    for (; k < ups.size() && l->n + update_words(ups[k]) <= kAppendLenMax; ++k) {
        const LenUpdate& u = ups[k];
        uint8_t* seg = u.e->d_plan + u.e->lay.segs + sizeof(DecodeSeg) * u.e->tail_seg[u.i];
        l->ptr[l->n] = reinterpret_cast<int32_t*>(seg + offsetof(DecodeSeg, n_tok));
        l->val[l->n++] = u.val;
        l->ptr[l->n] = reinterpret_cast<int32_t*>(seg + offsetof(DecodeSeg, grp_lim));
        l->val[l->n++] = u.val;
        if (u.e->lay.page_fill >= 0) {
            l->ptr[l->n] = reinterpret_cast<int32_t*>(u.e->d_plan + u.e->lay.page_fill) +
                           u.e->tail_fill[u.i];
            l->val[l->n++] = u.fill;
        }
    }
    return k - from;
}

// After the append's launches: the updated plans take the sequence's new
// version, count its new rows, list the written page among their newest
// writes, and count the append as their last use on the stream.
static void plan_len_apply(sq_cache* c, const LenUpdate& u, uint64_t new_version, int32_t n_new,
                           int32_t page, cudaStream_t st) {
    PlanEntry& e = *u.e;
    e.versions[u.i] = new_version;
    e.unique_tokens += n_new;
    e.logical_tokens += n_new;
    const uint64_t t = c->page_ticket[page];
    bool found = false;
    for (auto& tp : e.tick_top)
        if (tp.second == page) {
            tp.first = std::max(tp.first, t);
            found = true;
        }
    if (!found) {
        e.tick_top.push_back({t, page});
        if (e.tick_top.size() > (size_t)kDecodeMaxUnsafe) {
            auto oldest = std::min_element(
                e.tick_top.begin(), e.tick_top.end(),
                [](const std::pair<uint64_t, int32_t>& x, const std::pair<uint64_t, int32_t>& y) {
                    return x.first < y.first;
                });
            e.tick_rest = std::max(e.tick_rest, oldest->first);
            e.tick_top.erase(oldest);
        }
    }
    // the plan's buffer is written by this append: it is reused (or replaced)
    // only after it
    if (cudaEventRecord(e.ev, st) != cudaSuccess) {
        cudaGetLastError();
        e.valid = false;
    }
}

int sq_append_kv(sq_cache* c, sq_seq seq, int32_t n_tokens, const void* k, const void* v,
                 void* stream) {
    TraceRange trace_("sq_append_kv");
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!c->host->seq(seq)) return SQ_ERR_BAD_HANDLE;
    if (n_tokens < 0) return SQ_ERR_INVALID_ARG;
    if (n_tokens == 0) return SQ_OK;
    if (!k || !v || (reinterpret_cast<uintptr_t>(k) & 15) || (reinterpret_cast<uintptr_t>(v) & 15))
        return SQ_ERR_INVALID_ARG;
    AppendPlan plan;
    const uint64_t old_version = c->host->seq(seq)->version;
    int rc = c->host->append(seq, n_tokens, &plan);
    if (rc != SQ_OK) return rc;
    const Geometry& g = c->g;
    cudaStream_t st = as_stream(stream);
    auto undo = [&](int code) {
        c->host->undo_append(seq, plan);
        return code;
    };
    std::vector<LenUpdate> ups;
    plan_len_updates(c, seq, plan, old_version, st, &ups);
    size_t n_ups = 0;  // of them, passed to the kernel
    rc = fence_taken_pages(c, plan.taken, stream);
    if (rc != SQ_OK) return undo(rc);
    if (plan.cow) {
        CowArgs ca;
        ca.pool = c->pool;
        ca.num_pages = g.num_pages;
        ca.L = g.L; ca.Hkv = g.Hkv; ca.P = g.P; ca.D = g.D;
        ca.src_page = plan.cow_old;
        ca.dst_page = plan.cow_new;
        ca.rows = plan.cow_rows;
        ca.err = c->d_err;
        cudaError_t e = launch_cow_copy(ca, c->num_sms, st);
        if (e != cudaSuccess) return undo(cuda_status(e));
    }
    // rows go to slot-space positions pos0 .. pos0 + n - 1 (the last page's
    // free slots, then the fresh pages)
    const int64_t end = (int64_t)plan.pos0 + plan.n_new;
    for (size_t b = 0; b < plan.pages.size(); b += kAppendMaxPages) {
        AppendArgs a;
        a.pool = c->pool;
        a.k = reinterpret_cast<const __nv_bfloat16*>(k);
        a.v = reinterpret_cast<const __nv_bfloat16*>(v);
        a.num_pages = g.num_pages;
        a.L = g.L; a.Hkv = g.Hkv; a.P = g.P; a.D = g.D;
        a.n_total = n_tokens;
        a.page_index0 = plan.first_page_index + (int32_t)b;
        a.n_pages = (int32_t)std::min<size_t>(kAppendMaxPages, plan.pages.size() - b);
        for (int i = 0; i < a.n_pages; ++i) a.pages[i] = plan.pages[b + i];
        const int64_t pb = std::max<int64_t>(plan.pos0, (int64_t)a.page_index0 * g.P);
        const int64_t pe = std::min<int64_t>(end, (int64_t)(a.page_index0 + a.n_pages) * g.P);
        if (pe <= pb) continue;
        a.pos0 = (int32_t)pb;
        a.tok_begin = (int32_t)(pb - plan.pos0);
        a.n_tok = (int32_t)(pe - pb);
        a.lens.n = 0;
        if (b == 0) n_ups = fill_lens(ups, 0, &a.lens);  // an in-page append is one launch
        a.err = c->d_err;
        cudaError_t e = launch_append(a, c->num_sms, st);
        if (e != cudaSuccess) return undo(cuda_status(e));
    }
    note_writes(c, plan.pages.data(), plan.pages.size(), stream);
    {
        const uint64_t nv = c->host->seq(seq)->version;
        for (size_t k = 0; k < n_ups; ++k) plan_len_apply(c, ups[k], nv, plan.n_new, plan.pages[0], st);
    }
    c->host->seq_mut(seq)->last_stream = stream;
    c->stats.appended_tokens += n_tokens;
    if (plan.cow) c->stats.cow_pages += 1;
    return SQ_OK;
}

int sq_append_kv_batch(sq_cache* c, const sq_seq* seqs, int32_t n_seqs, const void* k,
                       const void* v, void* stream) {
    TraceRange trace_("sq_append_kv_batch");
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (n_seqs < 0 || (n_seqs > 0 && !seqs)) return SQ_ERR_INVALID_ARG;
    if (n_seqs == 0) return SQ_OK;
    if (!k || !v || (reinterpret_cast<uintptr_t>(k) & 15) || (reinterpret_cast<uintptr_t>(v) & 15))
        return SQ_ERR_INVALID_ARG;
    for (int32_t i = 0; i < n_seqs; ++i) {
        if (!c->host->seq(seqs[i])) return SQ_ERR_BAD_HANDLE;
        for (int32_t j = 0; j < i; ++j)
            if (seqs[j] == seqs[i]) return SQ_ERR_INVALID_ARG;
    }
    const Geometry& g = c->g;
    std::vector<AppendPlan> plans(n_seqs);
    auto undo = [&](int32_t upto, int code) {
        for (int32_t j = upto - 1; j >= 0; --j) c->host->undo_append(seqs[j], plans[j]);
        return code;
    };
    std::vector<int32_t> taken;
    std::vector<uint64_t> old_versions(n_seqs);
    for (int32_t i = 0; i < n_seqs; ++i) {
        old_versions[i] = c->host->seq(seqs[i])->version;
        int rc = c->host->append(seqs[i], 1, &plans[i]);
        if (rc != SQ_OK) return undo(i, rc);
        taken.insert(taken.end(), plans[i].taken.begin(), plans[i].taken.end());
    }
    cudaStream_t st = as_stream(stream);
    // the plans each sequence's append leaves valid, and which of them the
    // launch writing that sequence's row could take
    std::vector<std::vector<LenUpdate>> ups(n_seqs);
    std::vector<size_t> n_ups(n_seqs, 0);
    for (int32_t i = 0; i < n_seqs; ++i)
        plan_len_updates(c, seqs[i], plans[i], old_versions[i], st, &ups[i]);
    int rc = fence_taken_pages(c, taken, stream);
    if (rc != SQ_OK) return undo(n_seqs, rc);
    for (int32_t i = 0; i < n_seqs; ++i) {
        if (!plans[i].cow) continue;
        CowArgs ca;
        ca.pool = c->pool;
        ca.num_pages = g.num_pages;
        ca.L = g.L; ca.Hkv = g.Hkv; ca.P = g.P; ca.D = g.D;
        ca.src_page = plans[i].cow_old;
        ca.dst_page = plans[i].cow_new;
        ca.rows = plans[i].cow_rows;
        ca.err = c->d_err;
        cudaError_t e = launch_cow_copy(ca, c->num_sms, st);
        if (e != cudaSuccess) return undo(n_seqs, cuda_status(e));
    }
    for (int32_t b = 0; b < n_seqs; b += kAppendBatchMax) {
        AppendBatchArgs a;
        a.pool = c->pool;
        a.k = reinterpret_cast<const __nv_bfloat16*>(k);
        a.v = reinterpret_cast<const __nv_bfloat16*>(v);
        a.num_pages = g.num_pages;
        a.L = g.L; a.Hkv = g.Hkv; a.P = g.P; a.D = g.D;
        a.n_total = n_seqs;
        a.row0 = b;
        a.n = std::min(kAppendBatchMax, n_seqs - b);
        AppendLens& l = a.lens;
        l.n = 0;
        for (int32_t i = 0; i < a.n; ++i) {
            const AppendPlan& pl = plans[b + i];
            a.page[i] = pl.pages[0];                 // the page holding slot position pos0
            a.slot[i] = pl.pos0 % g.P;
            // a sequence's plan updates go all into this launch, or none do
            int words = 0;
            for (const LenUpdate& u : ups[b + i]) words += update_words(u);
            if (l.n + words <= kAppendLenMax) {
                AppendLens part;
                n_ups[b + i] = fill_lens(ups[b + i], 0, &part);
                for (int32_t k = 0; k < part.n; ++k) {
                    l.ptr[l.n] = part.ptr[k];
                    l.val[l.n] = part.val[k];
                    ++l.n;
                }
            }
        }
        a.err = c->d_err;
        cudaError_t e = launch_append_batch(a, c->num_sms, st);
        if (e != cudaSuccess) return undo(n_seqs, cuda_status(e));
    }
    {
        std::vector<int32_t> written(n_seqs);
        for (int32_t i = 0; i < n_seqs; ++i) written[i] = plans[i].pages[0];
        note_writes(c, written.data(), written.size(), stream);
    }
    for (int32_t i = 0; i < n_seqs; ++i) {
        const uint64_t nv = c->host->seq(seqs[i])->version;
        for (size_t k = 0; k < n_ups[i]; ++k)
            plan_len_apply(c, ups[i][k], nv, 1, plans[i].pages[0], st);
    }
    for (int32_t i = 0; i < n_seqs; ++i) {
        c->host->seq_mut(seqs[i])->last_stream = stream;
        if (plans[i].cow) c->stats.cow_pages += 1;
    }
    c->stats.appended_tokens += n_seqs;
    return SQ_OK;
}

// True when the byte ranges [a, a + na) and [b, b + nb) share a byte.  The
// attention calls write outputs while other CTAs still read the queries, so
// an output that overlaps the queries (or the log-sum-exps either) is refused.
static bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return na > 0 && nb > 0 && x < y + nb && y < x + na;
}

int sq_decode_attention(sq_cache* c, const sq_seq* seqs, int32_t n_seqs, int32_t layer,
                        const void* q, void* out, int32_t out_dtype, float sm_scale,
                        void* stream) {
    TraceRange trace_("sq_decode_attention");
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Geometry& g = c->g;
    if (!seqs || n_seqs < 1 || n_seqs > g.max_seqs || !q || !out) return SQ_ERR_INVALID_ARG;
    if (layer < 0 || layer >= g.L) return SQ_ERR_INVALID_ARG;
    if (out_dtype != SQ_OUT_BF16 && out_dtype != SQ_OUT_F32) return SQ_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(q) & 15) || (reinterpret_cast<uintptr_t>(out) & 15))
        return SQ_ERR_INVALID_ARG;
    if (!(sm_scale == sm_scale)) return SQ_ERR_INVALID_ARG;
    {
        const size_t rows = (size_t)n_seqs * g.Hq * g.D;
        if (overlaps(q, rows * 2, out, rows * (out_dtype == SQ_OUT_F32 ? 4 : 2)))
            return SQ_ERR_INVALID_ARG;
    }
    for (int32_t i = 0; i < n_seqs; ++i) {
        const Seq* s = c->host->seq(seqs[i]);
        if (!s) return SQ_ERR_BAD_HANDLE;
        if (s->n < 1) return SQ_ERR_INVALID_ARG;
    }
    // plan cache lookup: same handles, same versions, same CTA count
    PlanEntry* hit = nullptr;
    for (auto& p : c->plans) {
        if (!p.valid || p.n_ctas != c->decode_ctas || (int32_t)p.handles.size() != n_seqs) continue;
        bool same = true;
        for (int32_t i = 0; i < n_seqs && same; ++i)
            same = p.handles[i] == seqs[i] && p.versions[i] == c->host->seq(seqs[i])->version;
        if (same) {
            hit = &p;
            break;
        }
    }
    cudaStream_t st = as_stream(stream);
    cudaError_t e;
    // a reused plan that needs no cross-stream wait was on the device before
    // anything this call enqueues: the kernel may read it before its
    // grid-dependency wait
    bool plan_ready = false;
    if (!hit) {
        DecodePlanHost plan;
        int rc = plan_decode(*c->host, seqs, n_seqs, c->decode_ctas, &plan);
        if (rc != SQ_OK) return rc;
        DecodePlanLayout lay = plan_layout(plan, n_seqs, g.Hkv);
        // least recently used entry
        PlanEntry* victim = &c->plans[0];
        for (auto& p : c->plans)
            if (!p.valid || p.last_use < victim->last_use) victim = &p;
        const size_t part_bytes = (size_t)decode_partial_bytes(lay.n_comb_ent, g.G(), g.D);
        if ((size_t)lay.total > victim->plan_cap || part_bytes > victim->part_cap) {
            if (victim->ev_recorded) cudaEventSynchronize(victim->ev);
            if ((size_t)lay.total > victim->plan_cap) {
                if (victim->d_plan) cudaFree(victim->d_plan);
                victim->d_plan = nullptr;
                victim->plan_cap = 0;
                size_t cap = (size_t)lay.total * 5 / 4 + 4096;
                e = cudaMalloc(&victim->d_plan, cap);
                if (e != cudaSuccess) { victim->valid = false; return cuda_status(e); }
                victim->plan_cap = cap;
            }
            if (part_bytes > victim->part_cap) {
                if (victim->d_part) cudaFree(victim->d_part);
                victim->d_part = nullptr;
                victim->part_cap = 0;
                size_t cap = part_bytes * 5 / 4 + 4096;
                e = cudaMalloc(&victim->d_part, cap);
                if (e != cudaSuccess) { victim->valid = false; return cuda_status(e); }
                victim->part_cap = cap;
            }
        }
        if (!victim->ev) {
            e = cudaEventCreateWithFlags(&victim->ev, cudaEventDisableTiming);
            if (e != cudaSuccess) return cuda_status(e);
        }
        if (victim->ev_recorded && victim->ev_stream != st) {
            e = cudaStreamWaitEvent(st, victim->ev, 0);
            if (e != cudaSuccess) return cuda_status(e);
        }
        if (c->staging.size() < (size_t)lay.total) c->staging.resize(lay.total);
        plan_serialize(plan, lay, c->staging.data());
        int urc = staged_copy(c, victim->d_plan, c->staging.data(), lay.total, stream);
        if (urc != SQ_OK) { victim->valid = false; return urc; }
        c->stats.decode_plans_built += 1;
        victim->valid = true;
        victim->n_ctas = c->decode_ctas;
        victim->handles.assign(seqs, seqs + n_seqs);
        victim->versions.resize(n_seqs);
        for (int32_t i = 0; i < n_seqs; ++i) victim->versions[i] = c->host->seq(seqs[i])->version;
        victim->lay = lay;
        victim->unique_tokens = plan.unique_tokens;
        victim->logical_tokens = plan.logical_tokens;
        victim->tail_seg.assign(n_seqs, -1);
        victim->tail_base.assign(n_seqs, 0);
        victim->tail_fill.assign(n_seqs, 0);
        for (size_t s = 0; s < plan.segs.size(); ++s) {
            const DecodeSeg& sg = plan.segs[s];
            if (sg.n_grp == 1 && (sg.tail & 1)) {
                victim->tail_seg[sg.grp_seq[0]] = (int32_t)s;
                victim->tail_base[sg.grp_seq[0]] = sg.q0 * g.P;
                victim->tail_fill[sg.grp_seq[0]] = sg.page_off + sg.n_pages - 1;
            }
        }
        victim->first_busy_cta = 0;
        while (victim->first_busy_cta + 1 < (int32_t)plan.cta_begin.size() &&
               plan.cta_begin[victim->first_busy_cta + 1] == plan.cta_begin[victim->first_busy_cta])
            ++victim->first_busy_cta;
        {
            std::vector<std::pair<uint64_t, int32_t>> tk(plan.page_ids.size());
            for (size_t i = 0; i < tk.size(); ++i)
                tk[i] = {c->page_ticket[plan.page_ids[i]], plan.page_ids[i]};
            const size_t top = std::min<size_t>(kDecodeMaxUnsafe, tk.size());
            std::partial_sort(tk.begin(), tk.begin() + top, tk.end(),
                              [](const std::pair<uint64_t, int32_t>& x,
                                 const std::pair<uint64_t, int32_t>& y) { return x.first > y.first; });
            victim->tick_top.assign(tk.begin(), tk.begin() + top);
            victim->tick_rest = 0;
            for (size_t i = top; i < tk.size(); ++i) victim->tick_rest = std::max(victim->tick_rest, tk[i].first);
        }
        hit = victim;
    } else if (hit->ev_recorded && hit->ev_stream != st) {
        e = cudaStreamWaitEvent(st, hit->ev, 0);
        if (e != cudaSuccess) return cuda_status(e);
    } else {
        plan_ready = true;
    }
    hit->last_use = ++c->use_clock;
    const DecodePlanLayout& L = hit->lay;
    float* part_o = hit->d_part;
    float* part_ml = part_o + (size_t)L.n_comb_ent * g.G() * g.D;

    DecodeArgs a;
    a.segs = reinterpret_cast<const DecodeSeg*>(hit->d_plan + L.segs);
    a.items = reinterpret_cast<const DecodeItem*>(hit->d_plan + L.items);
    a.cta_begin = reinterpret_cast<const int32_t*>(hit->d_plan + L.cta_begin);
    a.page_ids = reinterpret_cast<const int32_t*>(hit->d_plan + L.page_ids);
    a.comb_off = reinterpret_cast<const int32_t*>(hit->d_plan + L.comb_off);
    a.arrive = reinterpret_cast<unsigned int*>(hit->d_plan + L.arrive);
    a.page_fill = L.page_fill >= 0 ? reinterpret_cast<const int32_t*>(hit->d_plan + L.page_fill)
                                   : nullptr;
    a.q = reinterpret_cast<const __nv_bfloat16*>(q);
    a.out = out;
    a.part_o = part_o;
    a.part_ml = part_ml;
    a.out_f32 = out_dtype == SQ_OUT_F32;
    a.plan_ready = plan_ready ? 1 : 0;
    a.layer = layer;
    a.Hq = g.Hq;
    a.Hkv = g.Hkv;
    a.G = g.G();
    a.P = g.P;
    a.num_pages = g.num_pages;
    a.scale_log2 = sm_scale * 1.4426950408889634f;
    a.debug_drop_cta = (c->debug_flags & SQ_DEBUG_DROP_DECODE_STAGE) ? hit->first_busy_cta : -1;
    a.kv_early = 0;
    a.n_unsafe = 0;
    if (plan_ready && c->early_ok) {
        // every write to the plan's pages outside its newest few is complete:
        // the kernel may load its first stages before its dependency wait,
        // except from the pages whose writes may still be running
        poll_writes(c);
        if (hit->tick_rest <= c->write_done) {
            a.kv_early = 1;
            for (const auto& tp : hit->tick_top)
                if (tp.first > c->write_done) a.unsafe[a.n_unsafe++] = tp.second;
            c->stats.decode_early_calls += 1;
            c->stats.decode_early_held += a.n_unsafe;
        }
    }
    c->debug_flags &= ~SQ_DEBUG_DROP_DECODE_STAGE;
    a.err = c->d_err;
    e = launch_decode(c->tmap, a, L.n_ctas, g.D, st);
    if (e != cudaSuccess) { hit->valid = false; return cuda_status(e); }
    e = cudaEventRecord(hit->ev, st);
    if (e != cudaSuccess) return cuda_status(e);
    hit->ev_recorded = true;
    hit->ev_stream = st;
    for (int32_t i = 0; i < n_seqs; ++i) c->host->seq_mut(seqs[i])->last_stream = stream;
    c->stats.decode_calls += 1;
    c->stats.decode_logical_bytes += hit->logical_tokens * g.token_layer_bytes();
    c->stats.decode_unique_bytes += hit->unique_tokens * g.token_layer_bytes();
    return SQ_OK;
}

}  // extern "C"

namespace {

int evict_impl(sq_cache* c, sq_seq seq, const sq_span* spans, int32_t n_spans, void* stream,
               bool ragged) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!c->host->seq(seq)) return SQ_ERR_BAD_HANDLE;
    if (n_spans < 0 || (n_spans > 0 && !spans)) return SQ_ERR_INVALID_ARG;
    if (n_spans == 0) return SQ_OK;
    std::vector<int32_t> a(n_spans), b(n_spans);
    for (int32_t i = 0; i < n_spans; ++i) {
        a[i] = spans[i].start;
        b[i] = spans[i].end;
    }
    EvictPlan plan;
    int rc = c->host->evict(seq, a.data(), b.data(), n_spans, &plan, ragged);
    if (rc != SQ_OK) return rc;
    const Geometry& g = c->g;
    cudaStream_t st = as_stream(stream);
    auto undo = [&](int code) {
        c->host->undo_evict(seq, plan);
        return code;
    };
    rc = fence_taken_pages(c, plan.cow_pages, stream);
    if (rc != SQ_OK) return undo(rc);
    if (!plan.moves.empty()) {
        std::vector<EvictTile> tiles;
        std::vector<EvictPiece> pieces;
        std::vector<int32_t> window_tile, chunk;
        evict_tiles(plan, c->evict_tile_rows, &tiles, &pieces, &window_tile);
        // Independent windows (ragged eviction) run as chunks in parallel
        // CTAs, up to about four waves of resident CTAs over all planes
        const int64_t planes = (int64_t)g.L * 2 * g.Hkv;
        const int64_t resident = c->evict_resident;
        const int32_t max_chunks = (int32_t)std::max<int64_t>(1, 4 * resident / planes);
        evict_chunks(window_tile, (int32_t)tiles.size(), max_chunks, 4, &chunk);
        const size_t tb = tiles.size() * sizeof(EvictTile);
        const size_t pcb = pieces.size() * sizeof(EvictPiece);
        std::vector<uint8_t> buf(tb + pcb + chunk.size() * sizeof(int32_t));
        std::memcpy(buf.data(), tiles.data(), tb);
        std::memcpy(buf.data() + tb, pieces.data(), pcb);
        std::memcpy(buf.data() + tb + pcb, chunk.data(), chunk.size() * sizeof(int32_t));
        UploadSlot& s = c->slots[c->next_slot];
        c->next_slot = (c->next_slot + 1) % kUploadSlots;
        rc = upload(c, s, buf.data(), buf.size(), stream);
        if (rc != SQ_OK) return undo(rc);
        EvictArgs ea;
        ea.pool = c->pool;
        ea.num_pages = g.num_pages;
        ea.L = g.L; ea.Hkv = g.Hkv; ea.P = g.P; ea.D = g.D;
        ea.tiles = reinterpret_cast<const EvictTile*>(s.d);
        ea.pieces = reinterpret_cast<const EvictPiece*>(s.d + tb);
        ea.n_tiles = (int32_t)tiles.size();
        ea.n_pieces = (int32_t)pieces.size();
        ea.tile_rows = c->evict_tile_rows;
        ea.stages = c->evict_stages;
        ea.zero_tiles = plan.zeroed_rows > 0 ? 1 : 0;
        ea.n_chunks = (int32_t)chunk.size() - 1;
        ea.chunk = ea.n_chunks > 1 ? reinterpret_cast<const int32_t*>(s.d + tb + pcb) : nullptr;
        ea.err = c->d_err;
        cudaError_t e = launch_evict(ea, st);
        if (e != cudaSuccess) return undo(cuda_status(e));
        e = cudaEventRecord(s.ev, st);
        if (e != cudaSuccess) return cuda_status(e);
        s.ev_recorded = true;
        s.ev_stream = st;
        std::vector<int32_t> written;
        for (const EvictMove& m : plan.moves)
            if (written.empty() || written.back() != m.dst_page) written.push_back(m.dst_page);
        note_writes(c, written.data(), written.size(), stream);
    }
    rc = record_freed(c, plan.freed, stream);
    if (rc != SQ_OK) return rc;
    c->host->seq_mut(seq)->last_stream = stream;
    c->stats.evict_calls += 1;
    c->stats.evicted_tokens += plan.evicted;
    c->stats.evict_moved_rows += plan.moved_rows;
    // rows copied are read and written, zeroed rows only written
    c->stats.evict_bytes += (2 * plan.moved_rows + plan.zeroed_rows) * g.L * g.token_layer_bytes();
    c->stats.cow_pages += (int64_t)plan.cow_pages.size();
    return SQ_OK;
}

}  // namespace

extern "C" {

int sq_evict_spans(sq_cache* c, sq_seq seq, const sq_span* spans, int32_t n_spans, void* stream) {
    TraceRange trace_("sq_evict_spans");
    return evict_impl(c, seq, spans, n_spans, stream, false);
}

int sq_evict_spans_ragged(sq_cache* c, sq_seq seq, const sq_span* spans, int32_t n_spans,
                          void* stream) {
    TraceRange trace_("sq_evict_spans_ragged");
    return evict_impl(c, seq, spans, n_spans, stream, true);
}

int sq_prefill_attention(sq_cache* c, sq_seq seq, int32_t layer, int32_t n_q, const void* q,
                         void* out, int32_t out_dtype, float* lse, float sm_scale,
                         const sq_span* spans, int32_t n_spans, void* stream) {
    TraceRange trace_("sq_prefill_attention");
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    const Geometry& g = c->g;
    if (layer < 0 || layer >= g.L || n_q < 1 || n_q > s->n || !q || !out)
        return SQ_ERR_INVALID_ARG;
    if (out_dtype != SQ_OUT_BF16 && out_dtype != SQ_OUT_F32) return SQ_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(q) & 15) || (reinterpret_cast<uintptr_t>(out) & 15) ||
        (reinterpret_cast<uintptr_t>(lse) & 3))
        return SQ_ERR_INVALID_ARG;
    if (!(sm_scale >= 0.f) || sm_scale > 3.0e38f) return SQ_ERR_INVALID_ARG;
    {
        const size_t rows = (size_t)n_q * g.Hq;
        const size_t qb = rows * g.D * 2, ob = rows * g.D * (out_dtype == SQ_OUT_F32 ? 4 : 2);
        const size_t lb = lse ? rows * 4 : 0;
        if (overlaps(q, qb, out, ob) || overlaps(q, qb, lse, lb) || overlaps(out, ob, lse, lb))
            return SQ_ERR_INVALID_ARG;
    }
    if (n_spans < 0 || (n_spans > 0 && !spans)) return SQ_ERR_INVALID_ARG;
    std::vector<int32_t> key(2 * (size_t)n_spans);
    for (int32_t i = 0; i < n_spans; ++i) {
        key[2 * i] = spans[i].start;
        key[2 * i + 1] = spans[i].end;
    }
    cudaStream_t st = as_stream(stream);
    cudaError_t e;
    PrefillPlanEntry* hit = nullptr;
    for (auto& p : c->pre_plans)
        if (p.valid && p.seq == seq && p.version == s->version && p.n_q == n_q &&
            p.target == c->num_sms && p.spans == key) {
            hit = &p;
            break;
        }
    if (!hit) {
        std::vector<int32_t> sa(n_spans), sb(n_spans);
        for (int32_t i = 0; i < n_spans; ++i) {
            sa[i] = key[2 * i];
            sb[i] = key[2 * i + 1];
        }
        PrefillPlanHost plan;
        int rc;
        if (has_partial_pages(*s, g.P)) {
            // slot space: the spans mapped through the page fills, plus the
            // unused slots of the partial pages
            std::vector<int32_t> xa, xb;
            int32_t n_slots = 0;
            rc = prefill_slot_spans(*s, g.P, n_q, sa.data(), sb.data(), n_spans, &xa, &xb,
                                    &n_slots);
            if (rc != SQ_OK) return rc;
            rc = plan_prefill(g, n_slots, n_q, xa.data(), xb.data(), (int32_t)xa.size(),
                              c->num_sms, &plan, s->pages.data());
        } else {
            rc = plan_prefill(g, s->n, n_q, sa.data(), sb.data(), n_spans, c->num_sms, &plan,
                              s->pages.data());
        }
        if (rc != SQ_OK) return rc;
        // upload: key tiles, per-CTA-tile counts, then the page of every piece
        const size_t tb = plan.tiles.size() * sizeof(PrefillTile);
        const size_t qb = plan.qt_tiles.size() * sizeof(int32_t);
        const size_t pb = plan.tile_pages.size() * sizeof(int32_t);
        // least recently used entry
        PrefillPlanEntry* victim = &c->pre_plans[0];
        for (auto& p : c->pre_plans)
            if (!p.valid || p.last_use < victim->last_use) victim = &p;
        victim->valid = false;
        if (!victim->ev) {
            e = cudaEventCreateWithFlags(&victim->ev, cudaEventDisableTiming);
            if (e != cudaSuccess) return cuda_status(e);
        }
        if (tb + qb + pb > victim->cap) {
            if (victim->ev_recorded) cudaEventSynchronize(victim->ev);
            if (victim->d) cudaFree(victim->d);
            victim->d = nullptr;
            victim->cap = 0;
            victim->ev_recorded = false;
            const size_t cap = std::max<size_t>((tb + qb + pb) * 5 / 4, 4096);
            e = cudaMalloc(&victim->d, cap);
            if (e != cudaSuccess) return cuda_status(e);
            victim->cap = cap;
        }
        if (victim->ev_recorded && victim->ev_stream != st) {
            // the launches that read the old plan run before it is overwritten
            e = cudaStreamWaitEvent(st, victim->ev, 0);
            if (e != cudaSuccess) return cuda_status(e);
        }
        if (c->staging.size() < tb + qb + pb) c->staging.resize(tb + qb + pb);
        if (tb) std::memcpy(c->staging.data(), plan.tiles.data(), tb);
        std::memcpy(c->staging.data() + tb, plan.qt_tiles.data(), qb);
        if (pb) std::memcpy(c->staging.data() + tb + qb, plan.tile_pages.data(), pb);
        rc = staged_copy(c, victim->d, c->staging.data(), tb + qb + pb, stream);
        if (rc != SQ_OK) return rc;
        victim->seq = seq;
        victim->version = s->version;
        victim->n_q = n_q;
        victim->target = c->num_sms;
        victim->spans = key;
        victim->tb = tb;
        victim->qb = qb;
        victim->n_tiles = (int32_t)plan.tiles.size();
        victim->n_pieces = plan.n_pieces;
        victim->BP = plan.BP;
        victim->n_qt = plan.n_qt;
        victim->n_split = plan.n_split;
        victim->visible_pairs = plan.visible_pairs;
        victim->valid = true;
        hit = victim;
    } else if (hit->ev_recorded && hit->ev_stream != st) {
        // its upload ran on the stream of the call that planned it
        e = cudaStreamWaitEvent(st, hit->ev, 0);
        if (e != cudaSuccess) return cuda_status(e);
    }
    hit->last_use = ++c->use_clock;
    const PrefillPlanEntry& plan = *hit;
    const int64_t grid = (int64_t)plan.n_qt * g.Hkv * plan.n_split;
    if (plan.n_split > 1) {
        const size_t need =
            (size_t)grid * kPrefillQTiles * kPrefillRows * (g.D + 1) * sizeof(float);
        if (!c->pre_ev) {
            e = cudaEventCreateWithFlags(&c->pre_ev, cudaEventDisableTiming);
            if (e != cudaSuccess) return cuda_status(e);
        }
        if (need > c->pre_part_cap) {
            if (c->pre_ev_recorded) cudaEventSynchronize(c->pre_ev);
            if (c->pre_part) cudaFree(c->pre_part);
            c->pre_part = nullptr;
            c->pre_part_cap = 0;
            e = cudaMalloc(&c->pre_part, need * 5 / 4);
            if (e != cudaSuccess) return cuda_status(e);
            c->pre_part_cap = need * 5 / 4;
            c->pre_ev_recorded = false;
        }
        if (c->pre_ev_recorded && c->pre_ev_stream != st) {
            e = cudaStreamWaitEvent(st, c->pre_ev, 0);
            if (e != cudaSuccess) return cuda_status(e);
        }
    }
    // queries: {D, Hq, n_q}, one box = the G heads of a KV head x BP positions
    CUtensorMap qmap;
    {
        auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(c->encode_fn);
        cuuint64_t dims[3] = {(cuuint64_t)g.D, (cuuint64_t)g.Hq, (cuuint64_t)n_q};
        cuuint64_t strides[2] = {(cuuint64_t)g.D * 2, (cuuint64_t)g.Hq * g.D * 2};
        cuuint32_t box[3] = {64, (cuuint32_t)g.G(), (cuuint32_t)plan.BP};
        cuuint32_t estr[3] = {1, 1, 1};
        CUresult r = encode(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims,
                            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return SQ_ERR_INVALID_ARG;
    }
    PrefillArgs a;
    a.tiles = reinterpret_cast<const PrefillTile*>(plan.d);
    a.qt_tiles = reinterpret_cast<const int32_t*>(plan.d + plan.tb);
    a.tile_pages = reinterpret_cast<const int32_t*>(plan.d + plan.tb + plan.qb);
    a.n_pieces = plan.n_pieces;
    a.n_tiles = plan.n_tiles;
    a.n = slot_end(*s, g.P);   // the slot-space end (s->n when every page but the last is full)
    a.n_q = n_q;
    a.layer = layer;
    a.Hq = g.Hq;
    a.Hkv = g.Hkv;
    a.G = g.G();
    a.P = g.P;
    a.num_pages = g.num_pages;
    a.BP = plan.BP;
    a.n_qt = plan.n_qt;
    a.n_split = plan.n_split;
    // the kernel keeps the scale inside the exponent (s * scale - m); a zero
    // scale runs as 1e-30, whose weights 2^(s * 1e-30 - m) are exactly 1
    a.scale_log2 = std::max(sm_scale * 1.4426950408889634f, 1e-30f);
    a.out = out;
    a.out_f32 = out_dtype == SQ_OUT_F32;
    a.lse = lse;
    a.part_o = c->pre_part;
    a.part_ml = c->pre_part
                    ? c->pre_part + (size_t)grid * kPrefillQTiles * kPrefillRows * g.D
                    : nullptr;
    a.err = c->d_err;
    e = launch_prefill(c->tmap, qmap, a, g.D, st);
    if (e != cudaSuccess) return cuda_status(e);
    if (plan.n_split > 1) {
        PrefillCombineArgs ca;
        ca.part_o = a.part_o;
        ca.part_ml = a.part_ml;
        ca.out = out;
        ca.out_f32 = a.out_f32;
        ca.lse = lse;
        ca.n_q = n_q;
        ca.Hq = g.Hq;
        ca.Hkv = g.Hkv;
        ca.G = g.G();
        ca.BP = plan.BP;
        ca.n_qt = plan.n_qt;
        ca.n_split = plan.n_split;
        e = launch_prefill_combine(ca, g.D, st);
        if (e != cudaSuccess) return cuda_status(e);
        e = cudaEventRecord(c->pre_ev, st);
        if (e != cudaSuccess) return cuda_status(e);
        c->pre_ev_recorded = true;
        c->pre_ev_stream = st;
    }
    e = cudaEventRecord(hit->ev, st);
    if (e != cudaSuccess) return cuda_status(e);
    hit->ev_recorded = true;
    hit->ev_stream = st;
    c->host->seq_mut(seq)->last_stream = stream;
    c->stats.prefill_calls += 1;
    c->stats.prefill_pairs += plan.visible_pairs;
    return SQ_OK;
}

int sq_release(sq_cache* c, sq_seq seq, void* stream) {
    TraceRange trace_("sq_release");
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    void* last = s->last_stream;
    if (last && last != stream) {
        // make `stream` follow the sequence's last work before the pages go
        cudaEvent_t ev;
        cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_status(e);
        e = cudaEventRecord(ev, as_stream(last));
        if (e == cudaSuccess) e = cudaStreamWaitEvent(as_stream(stream), ev, 0);
        cudaEventDestroy(ev);
        if (e != cudaSuccess) return cuda_status(e);
    }
    std::vector<int32_t> freed;
    int rc = c->host->release(seq, &freed);
    if (rc != SQ_OK) return rc;
    return record_freed(c, freed, stream);
}

int sq_seq_info(sq_cache* c, sq_seq seq, int32_t* n_tokens, int32_t* n_pages) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    if (n_tokens) *n_tokens = s->n;
    if (n_pages) *n_pages = (int32_t)s->pages.size();
    return SQ_OK;
}

int sq_seq_next_pos(sq_cache* c, sq_seq seq, int64_t* out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    if (!out) return SQ_ERR_INVALID_ARG;
    *out = s->next_pos;
    return SQ_OK;
}

int sq_get_page_table(sq_cache* c, sq_seq seq, int32_t* host_out, int32_t cap, int32_t* n_out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    const int32_t n = (int32_t)s->pages.size();
    if (n_out) *n_out = n;
    if (n > 0 && (!host_out || cap < n)) return SQ_ERR_INVALID_ARG;
    if (n > 0) std::memcpy(host_out, s->pages.data(), sizeof(int32_t) * n);
    return SQ_OK;
}

int sq_get_page_fill(sq_cache* c, sq_seq seq, int32_t* host_out, int32_t cap, int32_t* n_out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Seq* s = c->host->seq(seq);
    if (!s) return SQ_ERR_BAD_HANDLE;
    const int32_t n = (int32_t)s->fill.size();
    if (n_out) *n_out = n;
    if (n > 0 && (!host_out || cap < n)) return SQ_ERR_INVALID_ARG;
    if (n > 0) std::memcpy(host_out, s->fill.data(), sizeof(int32_t) * n);
    return SQ_OK;
}

int sq_page_refcount(sq_cache* c, int32_t page, int32_t* out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!out || page < 0 || page >= c->g.num_pages) return SQ_ERR_INVALID_ARG;
    *out = c->host->alloc().refcount(page);
    return SQ_OK;
}

int sq_free_pages(sq_cache* c, int32_t* out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!out) return SQ_ERR_INVALID_ARG;
    *out = c->host->alloc().free_count();
    return SQ_OK;
}

int sq_pool_ptr(sq_cache* c, void** out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!out) return SQ_ERR_INVALID_ARG;
    *out = c->pool;
    return SQ_OK;
}

int sq_stats(sq_cache* c, sq_stats_t* out) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!out) return SQ_ERR_INVALID_ARG;
    *out = c->stats;
    out->live_pages = c->host->live_pages();
    out->peak_live_pages = c->host->peak_live_pages();
    return SQ_OK;
}

int sq_probe_read(sq_cache* c, const void* buf, size_t bytes, void* stream) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (!buf || bytes == 0 || (bytes & 15) || (reinterpret_cast<uintptr_t>(buf) & 15))
        return SQ_ERR_INVALID_ARG;
    cudaError_t e = launch_read_probe(buf, bytes, reinterpret_cast<unsigned int*>(c->d_err) + 1,
                                      c->num_sms, as_stream(stream));
    return cuda_status(e);
}

int sq_debug_set(sq_cache* c, int32_t flags) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    if (flags & ~SQ_DEBUG_DROP_DECODE_STAGE) return SQ_ERR_INVALID_ARG;
    c->debug_flags = flags;
    return SQ_OK;
}

int sq_sync_status(sq_cache* c, void* stream) {
    if (!c) return SQ_ERR_BAD_HANDLE;
    cudaError_t e = cudaStreamSynchronize(as_stream(stream));
    if (e != cudaSuccess) return SQ_ERR_CUDA;
    int err = 0;
    e = cudaMemcpy(&err, c->d_err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return SQ_ERR_CUDA;
    if (err) {
        e = cudaMemset(c->d_err, 0, sizeof(int));
        if (e != cudaSuccess) return SQ_ERR_CUDA;
    }
    if (err & 2) return SQ_ERR_DEVICE_TIMEOUT;
    if (err & 1) return SQ_ERR_DEVICE;
    return SQ_OK;
}

int sq_decode_attention_noalloc(sq_cache* c, const sq_seq* seqs, int32_t n_seqs, int32_t layer,
                                const void* q, void* out, int32_t out_dtype, float sm_scale,
                                void* stream) {
    TraceRange trace_("sq_decode_attention_noalloc");
    if (!c) return SQ_ERR_BAD_HANDLE;
    const Geometry& g = c->g;
    if (!seqs || n_seqs < 1 || n_seqs > g.max_seqs || !q || !out) return SQ_ERR_INVALID_ARG;
    if (layer < 0 || layer >= g.L) return SQ_ERR_INVALID_ARG;
    if (out_dtype != SQ_OUT_BF16 && out_dtype != SQ_OUT_F32) return SQ_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(q) & 15) || (reinterpret_cast<uintptr_t>(out) & 15))
        return SQ_ERR_INVALID_ARG;
    if (!(sm_scale == sm_scale)) return SQ_ERR_INVALID_ARG;
    {
        const size_t rows = (size_t)n_seqs * g.Hq * g.D;
        if (overlaps(q, rows * 2, out, rows * (out_dtype == SQ_OUT_F32 ? 4 : 2)))
            return SQ_ERR_INVALID_ARG;
    }
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return SQ_ERR_CUDA;
    if (dev != c->device) return SQ_ERR_INVALID_ARG;
    if (c->noalloc_status != SQ_OK) return c->noalloc_status;
    DecodePlanHost plan;
    int rc = plan_decode(*c->host, seqs, n_seqs, c->decode_ctas, &plan);
    if (rc != SQ_OK) return rc;
    const DecodePlanLayout L = plan_layout(plan, n_seqs, g.Hkv);
    // scratch = [plan (with zeroed arrival words) | partial outputs | partial (max, sum)]
    const size_t part_off = ((size_t)L.total + 255) & ~size_t(255);
    const size_t need = part_off + (size_t)decode_partial_bytes(L.n_comb_ent, g.G(), g.D);
    if (need > (size_t)SQ_NOALLOC_SCRATCH_BYTES) return SQ_ERR_CAPACITY;
    uint8_t* scratch = c->noalloc_base;

    // The plan goes up from one of the cache's two pinned slots (an
    // asynchronous copy; the slot is refilled only after its previous copy
    // ran), or, if it is larger than a slot, from pageable memory.
    cudaStream_t st = as_stream(stream);
    cudaError_t e;
    if ((size_t)L.total <= kNoallocPinnedBytes) {
        PinnedSlot& ps = c->noalloc_pinned[c->next_noalloc_pinned];
        c->next_noalloc_pinned = (c->next_noalloc_pinned + 1) % kNoallocPinnedSlots;
        if (ps.ev_recorded) {
            e = cudaEventSynchronize(ps.ev);
            if (e != cudaSuccess) return cuda_status(e);
        }
        plan_serialize(plan, L, ps.h);
        e = cudaMemcpyAsync(scratch, ps.h, L.total, cudaMemcpyHostToDevice, st);
        if (e != cudaSuccess) return cuda_status(e);
        e = cudaEventRecord(ps.ev, st);
        if (e != cudaSuccess) return cuda_status(e);
        ps.ev_recorded = true;
    } else {
        // (a copy from pageable memory has taken its source when it returns)
        std::vector<uint8_t> host(L.total);
        plan_serialize(plan, L, host.data());
        e = cudaMemcpyAsync(scratch, host.data(), L.total, cudaMemcpyHostToDevice, st);
        if (e != cudaSuccess) return cuda_status(e);
    }
    float* part_o = reinterpret_cast<float*>(scratch + part_off);
    float* part_ml = part_o + (size_t)L.n_comb_ent * g.G() * g.D;

    DecodeArgs a;
    a.segs = reinterpret_cast<const DecodeSeg*>(scratch + L.segs);
    a.items = reinterpret_cast<const DecodeItem*>(scratch + L.items);
    a.cta_begin = reinterpret_cast<const int32_t*>(scratch + L.cta_begin);
    a.page_ids = reinterpret_cast<const int32_t*>(scratch + L.page_ids);
    a.comb_off = reinterpret_cast<const int32_t*>(scratch + L.comb_off);
    a.arrive = reinterpret_cast<unsigned int*>(scratch + L.arrive);
    a.page_fill = L.page_fill >= 0 ? reinterpret_cast<const int32_t*>(scratch + L.page_fill)
                                   : nullptr;
    a.q = reinterpret_cast<const __nv_bfloat16*>(q);
    a.out = out;
    a.part_o = part_o;
    a.part_ml = part_ml;
    a.out_f32 = out_dtype == SQ_OUT_F32;
    a.plan_ready = 0;  // uploaded just now
    a.layer = layer;
    a.Hq = g.Hq;
    a.Hkv = g.Hkv;
    a.G = g.G();
    a.P = g.P;
    a.num_pages = g.num_pages;
    a.scale_log2 = sm_scale * 1.4426950408889634f;
    int32_t busy = 0;
    while (busy + 1 < (int32_t)plan.cta_begin.size() && plan.cta_begin[busy + 1] == plan.cta_begin[busy])
        ++busy;
    a.debug_drop_cta = (c->debug_flags & SQ_DEBUG_DROP_DECODE_STAGE) ? busy : -1;
    a.kv_early = 0;   // the plan was uploaded just now (read after the wait)
    a.n_unsafe = 0;
    c->debug_flags &= ~SQ_DEBUG_DROP_DECODE_STAGE;
    a.err = c->d_err;
    e = launch_decode(c->tmap, a, L.n_ctas, g.D, st);
    if (e != cudaSuccess) return cuda_status(e);
    for (int32_t i = 0; i < n_seqs; ++i) c->host->seq_mut(seqs[i])->last_stream = stream;
    c->stats.decode_calls += 1;
    c->stats.decode_logical_bytes += plan.logical_tokens * g.token_layer_bytes();
    c->stats.decode_unique_bytes += plan.unique_tokens * g.token_layer_bytes();
    return SQ_OK;
}

}  // extern "C"
