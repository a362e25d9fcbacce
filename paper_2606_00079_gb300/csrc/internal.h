// Library-internal declarations shared by the host packer and the CUDA side.
#pragma once
#include <stddef.h>
#include <stdint.h>

#include <vector>

#include "../../include/bitsmoe.h"
#include "format.h"

namespace bmoe {

// Build the packed image of a host layer. Returns BITSMOE_OK or an error code.
int build_image(const bitsmoe_layer_host* src, std::vector<uint8_t>& img);

// Check a packed image before it is trusted (offsets, counts, unit indices).
int validate_image(const uint8_t* img, size_t bytes);

// Rebuild host arrays from a (validated) image.
int unpack_image(const uint8_t* img, size_t bytes, bitsmoe_layer_host_out* dst);

inline const ImageHeader* header_of(const uint8_t* img) {
  return reinterpret_cast<const ImageHeader*>(img);
}
inline const ExpertDesc* desc_of(const uint8_t* img) {
  return reinterpret_cast<const ExpertDesc*>(img + header_of(img)->off_desc);
}

// Keep a failed CUDA call's error for bitsmoe_last_cuda_error (on this host
// thread) and return BITSMOE_ERR_CUDA.
int record_cuda_error(int cuda_error);

// Supported quantisation groups and their checks.
inline bool group_ok(int g) { return g == 32 || g == 64 || g == 128 || g == 256; }
inline bool bits_ok(int b) {
  return b == 0 || b == 1 || b == 2 || b == 3 || b == 4 || b == 6 || b == 8 || b == 16;
}

}  // namespace bmoe
