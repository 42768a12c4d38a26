// mask.cu -- per-slot metadata of the verification input (Sec. 3.1 "Temporal
// Attention Mask", Eq. (1); "Position Encoding Alignment").
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace simsd {

// One CTA per sequence, one thread per slot (blockDim = 64 >= 2*gamma).
__global__ void __launch_bounds__(64) build_mask_kernel(const int32_t* __restrict__ step_map,
                                                        const int32_t* __restrict__ prefix_len, int gamma,
                                                        int32_t* __restrict__ tau, uint8_t* __restrict__ section,
                                                        int32_t* __restrict__ rope_pos,
                                                        unsigned long long* __restrict__ mask_bits,
                                                        int32_t* err_word) {
  __shared__ int mu[32];
  __shared__ int map_ok;
  __shared__ int s_tau[64];
  __shared__ uint8_t s_sect[64];
  const int b = blockIdx.x, i = threadIdx.x, S = 2 * gamma;
  pdl_wait();
  pdl_launch_next();
  if (i == 0) map_ok = 1;
  if (i < gamma) mu[i] = step_map ? step_map[static_cast<size_t>(b) * gamma + i] : i + 1;
  __syncthreads();
  // the drafted labels must be distinct values in 1..gamma; the other
  // entries are 0 (padding), SIMSD_STEP_UNDRAFTED or SIMSD_STEP_DECODED
  if (i < gamma) {
    const int v = mu[i];
    bool bad = v < SIMSD_STEP_DECODED || v > gamma;
    if (!bad && v > 0)
      for (int k = 0; k < i; ++k) bad |= (mu[k] == v);
    if (bad) map_ok = 0;
  }
  __syncthreads();
  if (i == 0 && !map_ok) raise_error(err_word, SIMSD_EW_STEP_MAP);
  if (i < S) {
    const bool is_data = i < gamma;
    const int k = is_data ? i : i - gamma;
    const int v = map_ok ? mu[k] : 0;
    // drafted: both slots at tau = v; undrafted: a mask placeholder after
    // every draft step; decoded: a data token known before every step
    int t = 0;
    uint8_t sec = kSectPad;
    if (v > 0) {
      t = v;
      sec = is_data ? kSectData : kSectMask;
    } else if (v == SIMSD_STEP_UNDRAFTED && !is_data) {
      t = gamma + 1;
      sec = kSectMask;
    } else if (v == SIMSD_STEP_DECODED && is_data) {
      t = 0;
      sec = kSectData;
    }
    s_tau[i] = t;
    s_sect[i] = sec;
    const size_t o = static_cast<size_t>(b) * S + i;
    tau[o] = t;
    section[o] = sec;
    // RoPE copy: D~_k reuses the position of D_k, which is n_b + k
    rope_pos[o] = prefix_len[b] + k;
  }
  __syncthreads();
  if (mask_bits && i < S) {
    unsigned long long bits = 0;
    for (int j = 0; j < S; ++j)
      if (temporal_visible(s_sect[i], s_tau[i], s_sect[j], s_tau[j])) bits |= 1ull << j;
    mask_bits[static_cast<size_t>(b) * S + i] = bits;
  }
}

cudaError_t launch_build_mask(const int32_t* step_map, const int32_t* prefix_len, int Bt, int gamma, int32_t* tau,
                              uint8_t* section, int32_t* rope_pos, uint64_t* mask_bits, int32_t* err_word,
                              cudaStream_t stream) {
  return launch_overlapped(build_mask_kernel, dim3(Bt), dim3(64), 0, stream, 1, step_map, prefix_len, gamma, tau,
                           section, rope_pos, reinterpret_cast<unsigned long long*>(mask_bits), err_word);
}

}  // namespace simsd
