// Fixed device scratch for sq_decode_attention_noalloc.
//
// Some callers cannot allocate GPU memory at decode time: a serving runtime
// that reserves the whole device up front for its KV pool and forbids
// allocations on its hot path, an embedding process whose allocator is owned
// by a host framework that is not reachable from C, or code running where a
// cudaMalloc could block on a device-wide synchronisation.  For them the
// split-K plan and partial results of one decode call live in this
// file-scope array instead of in buffers the library would allocate.
//
// The array is part of the library's device image: every GPU that loads the
// library holds its SQ_NOALLOC_SCRATCH_BYTES until the process exits.  Host
// code cannot use the symbol itself (on the host it names a stand-in, not a
// device address), so its device address is looked up once per device with
// cudaGetSymbolAddress, with that device current, and handed to the kernels.
#include <cuda_runtime.h>

#include <mutex>

#include "noalloc.hpp"
#include "sq.h"

namespace sq {
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SQ_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {};

}  // namespace

int noalloc_scratch(int device, void** ptr) {
    if (device < 0 || device >= kMaxDevices) return SQ_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_addr[device]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) return SQ_ERR_CUDA;
        g_addr[device] = p;
    }
    *ptr = g_addr[device];
    return SQ_OK;
}

}  // namespace sq
