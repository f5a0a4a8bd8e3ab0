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
// The array belongs to this file's device module.  With lazy module loading
// (the CUDA default) the module, and with it the array's
// SQ_NOALLOC_SCRATCH_BYTES, is loaded on a device the first time anything in
// it is used there, and then stays until the process exits.  Host code
// cannot use the symbol itself (on the host it names a stand-in, not a
// device address), so sq_cache_create looks its device address up with
// cudaGetSymbolAddress, with the cache's device current, which is the
// first use: the decode call itself then loads and allocates nothing.
#include <cuda_runtime.h>

#include "noalloc.hpp"
#include "sq.h"

namespace sq {
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SQ_NOALLOC_SCRATCH_BYTES];

}  // namespace

int noalloc_scratch(void** ptr) {
    *ptr = nullptr;
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) return SQ_ERR_CUDA;
    *ptr = p;
    return SQ_OK;
}

}  // namespace sq
