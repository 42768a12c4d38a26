// attention_f32.cu -- fp32 verification attention on CUDA cores (the paper's
// own runs are fp32, Sec. 4.1).  One CTA per query row; its warps split the
// keys in chunks of 32 (chunk c goes to warp c mod kF32Warps): the paged
// prefix rows, then the new slots admitted by Eq. (1).  Each lane scores
// one key of the chunk, the warp folds the chunk into its running max / sum
// (online softmax) and accumulates V with lanes over the head dimension; the
// warps' partial (max, sum, accumulator) are merged through shared memory at
// the end.  When the inputs are not rotated yet (Sec. 3.1 RoPE copy), the
// query row is rotated once in shared memory and each new key on the fly
// while it is scored; cached keys are stored rotated.
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace simsd {

constexpr int kF32Warps = 4;

template <int DPL>  // head-dim elements per lane (d = 32 * DPL)
__global__ void __launch_bounds__(kF32Warps * 32) attention_f32_kernel(const __grid_constant__ AttnF32Args a) {
  constexpr int d = 32 * DPL;
  __shared__ __align__(16) float q_s[d];
  __shared__ float acc_s[kF32Warps][d];
  __shared__ float m_s[kF32Warps], l_s[kF32Warps];
  __shared__ int ok_s;
  pdl_wait();
  pdl_launch_next();
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const long long row = blockIdx.x;
  const int S = 2 * a.gamma, g = a.Hq / a.Hkv;
  const int h = static_cast<int>(row % a.Hq);
  const int s = static_cast<int>((row / a.Hq) % S);
  const int b = static_cast<int>(row / (static_cast<long long>(a.Hq) * S));
  const int kvh = h / g;
  float* o = a.out + row * d;

  const int n = a.prefix_len[b];
  const uint8_t si = a.section[static_cast<size_t>(b) * S + s];
  const int ti = a.tau[static_cast<size_t>(b) * S + s];
  // the page id of this lane's key in the warp's first chunk, loaded beside
  // n (entries past the prefix are read but not used)
  const int pi0 = (32 * wib + lane) / a.page_size;
  const int pg0 = pi0 < a.max_pages ? a.block_table[static_cast<size_t>(b) * a.max_pages + pi0] : -1;
  if (wib == 0) {
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
    if (lane == 0) ok_s = ok && si != kSectPad;
  }
  for (int c = threadIdx.x; c < d; c += blockDim.x) q_s[c] = a.q[row * d + c];
  __syncthreads();
  if (!ok_s) {
    for (int c = threadIdx.x; c < d; c += blockDim.x) o[c] = 0.f;
    return;
  }
  if (a.rope_pos) {
    const int pos = a.rope_pos[static_cast<size_t>(b) * S + s];
    for (int i = threadIdx.x; i < d / 2; i += blockDim.x) {
      float sn, cs;
      rope_sincos(pos, a.rope.f[i], &sn, &cs);
      rope_pair(q_s[i], q_s[i + d / 2], sn, cs);
    }
    __syncthreads();
  }
  float acc[DPL];
#pragma unroll
  for (int c = 0; c < DPL; ++c) acc[c] = 0.f;
  float m = -INFINITY, l = 0.f;
  // keys 0..n-1 are the prefix rows, keys n..n+S-1 the new slots; lane j of
  // a chunk of 32 scores key base+j, then the warp folds the chunk in
  const int nkeys = n + S;
  for (int base = 32 * wib; base < nkeys; base += 32 * kF32Warps) {
    const int j = base + lane;
    const float* kr = nullptr;
    long long voff = -1;
    bool from_cache = false;
    if (j < n) {
      const int pg = base == 32 * wib ? pg0 : a.block_table[static_cast<size_t>(b) * a.max_pages + j / a.page_size];
      voff = ((static_cast<long long>(pg) * a.Hkv + kvh) * a.page_size + (j % a.page_size)) * d;
      kr = a.k_cache + voff;
      from_cache = true;
    } else if (j < nkeys) {
      const int t = j - n;
      const size_t st_i = static_cast<size_t>(b) * S + t;
      if (temporal_visible(si, ti, a.section[st_i], a.tau[st_i])) {
        voff = ((static_cast<long long>(b) * S + t) * a.Hkv + kvh) * d;
        kr = a.k_new + voff;
      }
    }
    float sc = -INFINITY;
    if (kr) {
      float dot = 0.f;
      const float4* k4 = reinterpret_cast<const float4*>(kr);
      const float4* q4 = reinterpret_cast<const float4*>(q_s);
      if (!from_cache && a.rope_pos) {
        // new key: rotate each (i, i + d/2) pair at its slot's position
        const int pos = a.rope_pos[static_cast<size_t>(b) * S + (j - n)];
        constexpr int hc = d / 8;  // float4 chunks per half
#pragma unroll 2
        for (int c = 0; c < hc; ++c) {
          const float4 kl = __ldg(k4 + c), kh = __ldg(k4 + c + hc);
          const float4 ql = q4[c], qh = q4[c + hc];
          float kx[4] = {kl.x, kl.y, kl.z, kl.w}, ky[4] = {kh.x, kh.y, kh.z, kh.w};
          const float qx[4] = {ql.x, ql.y, ql.z, ql.w}, qy[4] = {qh.x, qh.y, qh.z, qh.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            float sn, cs;
            rope_sincos(pos, a.rope.f[4 * c + e], &sn, &cs);
            rope_pair(kx[e], ky[e], sn, cs);
            dot = fmaf(qx[e], kx[e], dot);
            dot = fmaf(qy[e], ky[e], dot);
          }
        }
      } else {
#pragma unroll 8
        for (int c = 0; c < d / 4; ++c) {
          const float4 kv = __ldg(k4 + c);
          const float4 qv = q4[c];
          dot = fmaf(qv.x, kv.x, dot);
          dot = fmaf(qv.y, kv.y, dot);
          dot = fmaf(qv.z, kv.z, dot);
          dot = fmaf(qv.w, kv.w, dot);
        }
      }
      sc = dot * a.scale;
    }
    float mc = sc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, off));
    const float m_new = fmaxf(m, mc);
    if (m_new == -INFINITY) continue;  // nothing visible yet
    const float corr = expf(m - m_new);
    const float pr = kr ? expf(sc - m_new) : 0.f;
    float ps = pr;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
    l = l * corr + ps;
#pragma unroll
    for (int c = 0; c < DPL; ++c) acc[c] *= corr;
    // P.V of the chunk, kRound keys at a time so that their V loads are in
    // flight together (read cold, each round costs a DRAM round trip): all 32
    // at d = 64, 8 at d = 128 (more would spill); the FMAs run in key order
    constexpr int kRound = DPL <= 2 ? 32 : 8;
    const float* vrow = kr ? (from_cache ? a.v_cache : a.v_new) + voff : a.v_new;
#pragma unroll 1
    for (int j0 = 0; j0 < 32; j0 += kRound) {
      float vv[kRound][DPL], pj[kRound];
      bool use[kRound];
#pragma unroll
      for (int u = 0; u < kRound; ++u) {
        const float* vr = reinterpret_cast<const float*>(
            __shfl_sync(0xffffffffu, reinterpret_cast<uintptr_t>(vrow), j0 + u));
        pj[u] = __shfl_sync(0xffffffffu, pr, j0 + u);
        use[u] = __shfl_sync(0xffffffffu, kr != nullptr, j0 + u);
#pragma unroll
        for (int c = 0; c < DPL; ++c) vv[u][c] = use[u] ? __ldg(vr + lane + 32 * c) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kRound; ++u)
#pragma unroll
        for (int c = 0; c < DPL; ++c) acc[c] = use[u] ? fmaf(pj[u], vv[u][c], acc[c]) : acc[c];
    }
    m = m_new;
  }
  // merge the warps: O = sum_w e^(m_w - M) acc_w / sum_w e^(m_w - M) l_w
  if (lane == 0) {
    m_s[wib] = m;
    l_s[wib] = l;
  }
#pragma unroll
  for (int c = 0; c < DPL; ++c) acc_s[wib][lane + 32 * c] = acc[c];
  __syncthreads();
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kF32Warps; ++w) M = fmaxf(M, m_s[w]);
  float L = 0.f, f[kF32Warps];
#pragma unroll
  for (int w = 0; w < kF32Warps; ++w) {
    f[w] = m_s[w] == -INFINITY ? 0.f : expf(m_s[w] - M);
    L = fmaf(f[w], l_s[w], L);
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kF32Warps; ++w) v = fmaf(f[w], acc_s[w][c], v);
    o[c] = v * inv;
  }
}

cudaError_t launch_attention_f32(const AttnF32Args& a, cudaStream_t stream) {
  const long long rows = static_cast<long long>(a.Bt) * 2 * a.gamma * a.Hq;
  const unsigned blocks = static_cast<unsigned>(rows);  // one CTA per query row
  if (a.d == 64) return launch_overlapped(attention_f32_kernel<2>, dim3(blocks), dim3(kF32Warps * 32), 0, stream, 1, a);
  return launch_overlapped(attention_f32_kernel<4>, dim3(blocks), dim3(kF32Warps * 32), 0, stream, 1, a);
}

}  // namespace simsd
