// common.cuh -- constants and small device helpers shared by the kernels.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>
#include <utility>

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

// ---- programmatic dependent launch.  Every kernel of the library is
// launched so that it may start (set-up only) while the previous kernel on
// the stream finishes: it calls pdl_wait() before it reads or writes any
// memory that earlier work may touch, and pdl_launch_next() to let the next
// kernel be scheduled (one thread per CTA is enough).  The wait returns once
// the previous grid has completed and its memory operations are visible.
// Short kernels trigger at once; the attention and acceptance kernels only
// after their main loop, since CTAs of the next kernel that wait beside a
// long-running one slowed it down.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_next() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Host side: launches kern with the attribute that allows the overlap above
// (and a cluster dimension when cluster > 1).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_overlapped(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                     unsigned cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  unsigned na = 0;
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (cluster > 1) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = cluster;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// ---- rotary position embedding (Su et al., RoFormer), rotate-half layout:
// for i < d/2 the pair (x_i, x_{i+d/2}) turns by the angle pos * theta^(-2i/d).
// The per-pair frequencies theta^(-2i/d) come in a RopeTable (kernels.h).

// sin and cos of pos * f for 0 <= pos < 2^24.  The product is kept in
// float-float (the rounding error of p * hi comes back exactly from an FMA)
// and reduced to [-pi, pi] by Cody-Waite subtraction of k * 2pi, with 2pi
// split into three floats of which the first has 8 significant bits, so the
// first subtraction is exact; the reduced angle is good to ~2e-7 rad up to
// pos = 2^20.
__device__ __forceinline__ void rope_sincos(int pos, float2 f, float* sn, float* cs) {
  constexpr float kTwoPiA = 6.28125f;
  constexpr float kTwoPiB = 1.9353071693331003e-03f;
  constexpr float kTwoPiC = 1.0253131677018246e-11f;
  constexpr float kInvTwoPi = 0.15915493667125702f;
  const float p = static_cast<float>(pos);
  const float a = p * f.x;
  const float b = fmaf(p, f.y, fmaf(p, f.x, -a));
  const float k = rintf(a * kInvTwoPi);
  float r = fmaf(-k, kTwoPiA, a);
  r = fmaf(-k, kTwoPiB, r);
  r = fmaf(-k, kTwoPiC, r);
  sincosf(r + b, sn, cs);
}

// Rotates one pair in place.
__device__ __forceinline__ void rope_pair(float& x, float& y, float sn, float cs) {
  const float x2 = x * cs - y * sn;
  const float y2 = fmaf(x, sn, y * cs);
  x = x2;
  y = y2;
}

}  // namespace simsd
