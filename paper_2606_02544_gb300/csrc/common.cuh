// common.cuh -- constants and small device helpers shared by the kernels.
#pragma once
#include <cstdint>

#include "../../include/simsd.h"

namespace simsd {

constexpr uint8_t kSectData = SIMSD_SECT_DATA;
constexpr uint8_t kSectMask = SIMSD_SECT_MASK;
constexpr uint8_t kSectPad = SIMSD_SECT_PAD;

__device__ __forceinline__ void raise_error(int32_t* err_word, uint32_t bit) {
  if (err_word) atomicOr(reinterpret_cast<int*>(err_word), static_cast<int>(bit));
}

// Eq. (1) in one comparison.  Row slot i (section si, label ti) sees new
// column slot j (sj, tj) iff both are real slots and
//   (j is a data slot) == (tj < ti + [i is a data slot]).
// Data row: data columns with tj <= ti, mask columns with tj > ti.
// Mask row: data columns with tj < ti, mask columns with tj >= ti.
__host__ __device__ __forceinline__ bool temporal_visible(uint8_t si, int ti, uint8_t sj, int tj) {
  if (si == kSectPad || sj == kSectPad) return false;
  const int bias = (si == kSectData) ? 1 : 0;
  return (sj == kSectData) == (tj < ti + bias);
}

}  // namespace simsd
