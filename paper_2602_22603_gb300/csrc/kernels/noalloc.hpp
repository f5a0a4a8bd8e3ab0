// Device address of the fixed scratch used by sq_decode_attention_noalloc.
#pragma once

namespace sq {

// Looks up the device address of the library's static scratch array on the
// current device (loading its module there if it is not loaded yet).
// Returns SQ_OK or SQ_ERR_CUDA.
int noalloc_scratch(void** ptr);

}  // namespace sq
