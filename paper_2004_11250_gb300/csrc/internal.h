// Internal declarations shared by the library's translation units.
#pragma once

#include <cstdint>
#include <vector>

#include "ppconv.h"

// The compact pattern-grouped storage of a layer (Section 3, "Sparse model
// storage" and "Matrix reorder"); field meanings are documented at
// pp_pack_layer in ppconv.h.
struct pp_packed {
  int Co = 0, Ci = 0, P = 0;
  std::vector<uint8_t> taps;   // [P][4]
  std::vector<int32_t> perm;   // [Co]
  std::vector<int32_t> kptr;   // [Co + 1]
  std::vector<int32_t> kidx;   // [nk]
  std::vector<uint8_t> kpat;   // [nk]
  std::vector<float> kw;       // [nk][4]
};

namespace ppc {

// Maximum filter slots handled by one warp of the conv kernel.
constexpr int kSlots = 16;
// Input channels staged in shared memory per pipeline step.
constexpr int kChunk = 16;

// Tap-set identifiers.  A pattern's taps are encoded as a 9-bit mask; the
// kernels specialise on the fixed ring set of 8 centre-based patterns and fall
// back to a per-tap dispatch for any other set.
uint16_t tap_mask(const uint8_t* taps4);

}  // namespace ppc
