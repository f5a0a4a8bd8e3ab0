// Device address of the fixed scratch used by sq_decode_attention_noalloc.
#pragma once

namespace sq {

// Looks up (once per device; the device must be current) the device address
// of the library's static scratch array.  Returns SQ_OK or SQ_ERR_CUDA /
// SQ_ERR_UNSUPPORTED.  Allocates nothing.
int noalloc_scratch(int device, void** ptr);

}  // namespace sq
