// attention_f32.cu -- fp32 verification attention on CUDA cores (the paper's
// own runs are fp32, Sec. 4.1).  One warp per query row; lanes split the
// head dimension; online softmax over the visible keys: the paged prefix,
// then the new slots admitted by Eq. (1).
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace simsd {

constexpr int kF32Warps = 4;

template <int DPL>  // head-dim elements per lane (d = 32 * DPL)
__global__ void __launch_bounds__(kF32Warps * 32) attention_f32_kernel(AttnF32Args a) {
  const int lane = threadIdx.x & 31;
  const long long row = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int S = 2 * a.gamma, g = a.Hq / a.Hkv, d = 32 * DPL;
  const long long rows = static_cast<long long>(a.Bt) * S * a.Hq;
  if (row >= rows) return;
  const int h = static_cast<int>(row % a.Hq);
  const int s = static_cast<int>((row / a.Hq) % S);
  const int b = static_cast<int>(row / (static_cast<long long>(a.Hq) * S));
  const int kvh = h / g;
  float* o = a.out + row * d;

  const int n = a.prefix_len[b];
  bool ok = n >= 0 && static_cast<long long>(n) <= static_cast<long long>(a.max_pages) * a.page_size;
  if (!ok && lane == 0 && s == 0 && h == 0) raise_error(a.err_word, SIMSD_EW_PREFIX_LEN);
  if (ok) {
    const int npages = (n + a.page_size - 1) / a.page_size;
    bool bad = false;
    for (int p = lane; p < npages; p += 32) {
      const int pg = a.block_table[static_cast<size_t>(b) * a.max_pages + p];
      bad |= (pg < 0 || pg >= a.num_pages);
    }
    if (__any_sync(0xffffffffu, bad)) {
      ok = false;
      if (lane == 0 && s == 0 && h == 0) raise_error(a.err_word, SIMSD_EW_PAGE);
    }
  }
  const uint8_t si = a.section[static_cast<size_t>(b) * S + s];
  if (!ok || si == kSectPad) {
#pragma unroll
    for (int c = 0; c < DPL; ++c) o[lane + 32 * c] = 0.f;
    return;
  }
  const int ti = a.tau[static_cast<size_t>(b) * S + s];
  float qv[DPL], acc[DPL];
#pragma unroll
  for (int c = 0; c < DPL; ++c) {
    qv[c] = a.q[row * d + lane + 32 * c];
    acc[c] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  auto visit = [&](const float* kr, const float* vr) {
    float dot = 0.f;
#pragma unroll
    for (int c = 0; c < DPL; ++c) dot = fmaf(qv[c], kr[lane + 32 * c], dot);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    const float sc = dot * a.scale;
    const float m_new = fmaxf(m, sc);
    const float corr = expf(m - m_new);
    const float pr = expf(sc - m_new);
    l = l * corr + pr;
#pragma unroll
    for (int c = 0; c < DPL; ++c) acc[c] = fmaf(acc[c], corr, pr * vr[lane + 32 * c]);
    m = m_new;
  };
  for (int p = 0; p < n; ++p) {
    const int pg = a.block_table[static_cast<size_t>(b) * a.max_pages + p / a.page_size];
    const size_t off = ((static_cast<size_t>(pg) * a.Hkv + kvh) * a.page_size + (p % a.page_size)) * d;
    visit(a.k_cache + off, a.v_cache + off);
  }
  for (int t = 0; t < S; ++t) {
    const uint8_t sj = a.section[static_cast<size_t>(b) * S + t];
    const int tj = a.tau[static_cast<size_t>(b) * S + t];
    if (!temporal_visible(si, ti, sj, tj)) continue;
    const size_t off = ((static_cast<size_t>(b) * S + t) * a.Hkv + kvh) * d;
    visit(a.k_new + off, a.v_new + off);
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
  for (int c = 0; c < DPL; ++c) o[lane + 32 * c] = acc[c] * inv;
}

cudaError_t launch_attention_f32(const AttnF32Args& a, cudaStream_t stream) {
  const long long rows = static_cast<long long>(a.Bt) * 2 * a.gamma * a.Hq;
  const unsigned blocks = static_cast<unsigned>((rows + kF32Warps - 1) / kF32Warps);
  if (a.d == 64)
    attention_f32_kernel<2><<<blocks, kF32Warps * 32, 0, stream>>>(a);
  else
    attention_f32_kernel<4><<<blocks, kF32Warps * 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace simsd
