// accept_sampled.cu -- stochastic acceptance of the drafts (Sec. 3.2, Eq. (2)):
// draft r is accepted iff u_r < alpha_r = min(1, p_theta(x_r) / p_phi(x_r)),
// p = softmax(logits / T), along the draft order up to the first rejection a;
// the token at position a is drawn from the residual max(0, p_theta - p_phi)
// (renormalised) or, when every draft is accepted, from p_theta of the extra
// target row, by inverse CDF with a given uniform u_sample.
//
// One thread-block cluster per sequence.  Phase 1: the sequence's gamma+1
// target rows and gamma draft rows are laid end to end, each row padded to a
// multiple of 32 units (a unit is 4 or 1 floats), and the CTAs take
// contiguous spans of warp-aligned units, so the 32 lanes of a warp are always
// on the same row.  Each lane keeps the running maximum m of z = x*log2(e)/T
// and s = sum 2^(z - m) of the row it is on; when the warp moves to the next
// row it merges its lanes by shuffles and stores the pair in a per-warp slot
// (no atomics).  CTA 0 merges the warps' and the CTAs' pairs (distributed
// shared memory), forms alpha_r from the drafts' own logits and the accepted
// length a, and broadcasts a.  Phase 2: each CTA takes a column range of row
// a and each thread a contiguous run of it; the thread sums the weights of
// its run.  CTA 0 forms the threshold u_sample * total and names the CTA
// whose range holds it; that CTA scans its threads' sums, and the one thread
// whose run holds the threshold walks it.  Row a is read a second time (2 of
// the 2*gamma+1 rows); no global scratch memory is used.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace simsd {
namespace {

constexpr int kSampThreads = 512;
constexpr int kSampWarps = kSampThreads / 32;
constexpr int kSampUnroll = 8;
constexpr int kSampMaxRows = 65;  // 2*gamma+1 <= 65
constexpr float kLog2e = 1.4426950408889634f;
// A residual whose total is at most this is empty: p_theta and p_phi agree
// to fp32 precision (each probability carries a relative error of a few
// units of 2^-24, the row sums about 1e-6), so what is left is rounding.
constexpr float kResidFloor = 1.0f / 65536.0f;

// Merges two (m, s) pairs of a base-2 log-sum-exp: s = s1 2^(m1 - M) +
// s2 2^(m2 - M), M = max; m = -inf stands for an empty set.
__device__ __forceinline__ void ms_merge(float& m, float& s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = s * exp2f(m - M) + s2 * exp2f(m2 - M);
  m = M;
}

__device__ __forceinline__ float4 ld_stream_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

// Row `row` of the combined row space: target rows 0..gamma, then draft rows.
__device__ __forceinline__ const float* row_ptr(const float* tgt, const float* drf, int b, int gamma, int vocab,
                                                int row) {
  return row <= gamma ? tgt + (static_cast<size_t>(b) * (gamma + 1) + row) * vocab
                      : drf + (static_cast<size_t>(b) * gamma + (row - gamma - 1)) * vocab;
}

__global__ void __launch_bounds__(kSampThreads, 2) accept_sampled_kernel(
    const float* __restrict__ tgt, const float* __restrict__ drf, const int32_t* __restrict__ draft,
    const float* __restrict__ u_accept, const float* __restrict__ u_sample, float zscale, int gamma, int vocab,
    int vec4, int32_t* __restrict__ accepted_len, int32_t* __restrict__ out_tokens, int32_t* err_word) {
  __shared__ float2 part[kSampWarps][kSampMaxRows];  // per warp (m, s) of each row
  __shared__ float2 cta_ms[kSampMaxRows];            // this CTA's (m, s) of each row
  __shared__ float row_m[kSampMaxRows], row_s[kSampMaxRows];
  __shared__ float tsum[kSampThreads];               // phase 2: each thread's run total
  __shared__ float warp_tot[kSampWarps];
  __shared__ int a_sh;
  __shared__ float w_cta;          // this CTA's weight of row a
  __shared__ float w_off, w_thr;   // the owner's offset and threshold (-1 elsewhere), set by CTA 0
  __shared__ int w_state;          // 1: the total weight was positive (set by CTA 0)
  __shared__ int pick_t, last_t;   // phase 2 owner thread
  pdl_wait();
  pdl_launch_next();
  cg::cluster_group cluster = cg::this_cluster();
  const int CL = static_cast<int>(cluster.num_blocks());
  const int c = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.x / CL;
  const int rows = 2 * gamma + 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned full = 0xffffffffu;
  for (int i = tid; i < kSampWarps * kSampMaxRows; i += kSampThreads)
    part[i / kSampMaxRows][i % kSampMaxRows] = make_float2(-INFINITY, 0.f);
  __syncthreads();

  // ---- phase 1: per-row (m, s) over this CTA's span of warp-aligned units
  {
    const int W = vec4 ? (vocab >> 2) : vocab;  // units per row
    const int Wp = (W + 31) & ~31;              // padded: a warp never straddles two rows
    const long long G = static_cast<long long>(rows) * (Wp >> 5);  // groups of 32 units
    const long long per = (G + CL - 1) / CL;
    const long long f0 = 32 * min(G, c * per), f1 = 32 * min(G, c * per + per);
    long long f = f0 + tid;
    int row = static_cast<int>(f / Wp);
    int col = static_cast<int>(f - static_cast<long long>(row) * Wp);
    int cur = row;
    float m = -INFINITY, s = 0.f;
    // merges the warp's lanes (all on row `cur`) into its slot
    auto flush = [&]() {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(full, m, o), s2 = __shfl_xor_sync(full, s, o);
        ms_merge(m, s, m2, s2);
      }
      if (lane == 0) {
        float2 p = part[warp][cur];
        ms_merge(p.x, p.y, m, s);
        part[warp][cur] = p;
      }
    };
    // f, f0, f1 and Wp are multiples of 32 at the warp's first lane, so every
    // test below is the same for the 32 lanes of a warp
    for (; f < f1; f += static_cast<long long>(kSampThreads) * kSampUnroll) {
      float4 v[kSampUnroll];
      int vr[kSampUnroll];
#pragma unroll
      for (int u = 0; u < kSampUnroll; ++u) {
        vr[u] = -1;
        if (f + static_cast<long long>(u) * kSampThreads < f1) {
          vr[u] = row;
          v[u] = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
          if (col < W) {
            const float* rp = row_ptr(tgt, drf, b, gamma, vocab, row);
            if (vec4)
              v[u] = ld_stream_f4(rp + 4 * col);
            else
              v[u].x = __ldg(rp + col);
          }
        }
        col += kSampThreads;
        if (col >= Wp) {
          row += col / Wp;
          col %= Wp;
        }
      }
#pragma unroll
      for (int u = 0; u < kSampUnroll; ++u) {
        if (vr[u] < 0) break;
        if (vr[u] != cur) {
          flush();
          cur = vr[u];
          m = -INFINITY;
          s = 0.f;
        }
        const float z0 = v[u].x * zscale, z1 = v[u].y * zscale, z2 = v[u].z * zscale, z3 = v[u].w * zscale;
        const float mz = fmaxf(fmaxf(z0, z1), fmaxf(z2, z3));
        if (mz > m) {
          s = (m == -INFINITY) ? 0.f : s * exp2f(m - mz);
          m = mz;
        }
        // a logit of -inf has weight 0: while m is still -inf the exponent
        // is taken against 0, so that -inf - -inf never occurs
        const float mr = m == -INFINITY ? 0.f : m;
        s += exp2f(z0 - mr) + exp2f(z1 - mr) + exp2f(z2 - mr) + exp2f(z3 - mr);
      }
    }
    if (f0 + 32 * warp < f1) flush();
  }
  __syncthreads();
  for (int r = tid; r < rows; r += kSampThreads) {
    float m = -INFINITY, s = 0.f;
    for (int w = 0; w < kSampWarps; ++w) ms_merge(m, s, part[w][r].x, part[w][r].y);
    cta_ms[r] = make_float2(m, s);
  }
  cluster.sync();

  // ---- CTA 0: merge the CTAs, alpha_r, accepted length
  if (c == 0) {
    for (int r = tid; r < rows; r += kSampThreads) {
      float m = -INFINITY, s = 0.f;
      for (int peer = 0; peer < CL; ++peer) {
        const float2 v = *cluster.map_shared_rank(&cta_ms[r], peer);
        ms_merge(m, s, v.x, v.y);
      }
      row_m[r] = m;
      row_s[r] = s;
    }
    __syncthreads();
    if (warp == 0) {
      bool acc = false, bad = false;
      if (lane < gamma) {
        const int x = draft[static_cast<size_t>(b) * gamma + lane];
        if (x < 0 || x >= vocab) {
          bad = true;
        } else {
          // log2 of p_theta(x) / p_phi(x)
          const float zt = __ldg(tgt + (static_cast<size_t>(b) * (gamma + 1) + lane) * vocab + x) * zscale;
          const float zd = __ldg(drf + (static_cast<size_t>(b) * gamma + lane) * vocab + x) * zscale;
          const int rd = gamma + 1 + lane;
          const float lr = (zt - row_m[lane] - log2f(row_s[lane])) - (zd - row_m[rd] - log2f(row_s[rd]));
          const float alpha = lr >= 0.f ? 1.f : exp2f(lr);
          acc = u_accept[static_cast<size_t>(b) * gamma + lane] < alpha;
        }
      }
      const unsigned rej = __ballot_sync(full, lane < gamma && !acc);
      if (__any_sync(full, bad) && lane == 0) raise_error(err_word, SIMSD_EW_DRAFT);
      const int a = rej ? __ffs(rej) - 1 : gamma;
      if (lane == 0) {
        accepted_len[b] = a;
        for (int peer = 0; peer < CL; ++peer) *cluster.map_shared_rank(&a_sh, peer) = a;
      }
      int32_t* ot = out_tokens + static_cast<size_t>(b) * (gamma + 1);
      for (int r = lane; r <= gamma; r += 32)
        if (r != a) ot[r] = r < a ? draft[static_cast<size_t>(b) * gamma + r] : -1;
      // the merged (m, s) of the rows phase 2 needs, for every CTA
      if (lane < 2) {
        const int rr = lane == 0 ? a : gamma + 1 + a;
        if (lane == 0 || a < gamma)
          for (int peer = 0; peer < CL; ++peer) {
            *cluster.map_shared_rank(&row_m[rr], peer) = row_m[rr];
            *cluster.map_shared_rank(&row_s[rr], peer) = row_s[rr];
          }
      }
    }
  }
  cluster.sync();

  // ---- phase 2: weights of row a; CTA c takes a column range, each thread a
  // contiguous run of it
  const int a = a_sh;
  bool resid = a < gamma;
  const float* trow = tgt + (static_cast<size_t>(b) * (gamma + 1) + a) * vocab;
  const float* drow = a < gamma ? drf + (static_cast<size_t>(b) * gamma + a) * vocab : nullptr;
  const float mt = row_m[a], it = 1.f / row_s[a];
  const float md = a < gamma ? row_m[gamma + 1 + a] : 0.f, id = a < gamma ? 1.f / row_s[gamma + 1 + a] : 0.f;
  const int per = (vocab + CL - 1) / CL;
  const int v0 = min(vocab, c * per), v1 = min(vocab, v0 + per);
  const int q = (v1 - v0 + kSampThreads - 1) / kSampThreads;
  const int r0 = min(v1, v0 + tid * q), r1 = min(v1, r0 + q);
  auto weight = [&](int v) -> float {
    const float pt = exp2f(__ldg(trow + v) * zscale - mt) * it;
    if (!resid) return pt;
    const float pd = exp2f(__ldg(drow + v) * zscale - md) * id;
    return fmaxf(0.f, pt - pd);
  };
  // an empty residual (p_theta = p_phi to fp32 precision) cannot reject:
  // the draw then falls back to p_theta (second pass)
  float ts = 0.f;
  for (int pass = 0; pass < 2; ++pass) {
    ts = 0.f;
#pragma unroll 4
    for (int v = r0; v < r1; ++v) ts += weight(v);
    float ws = ts;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ws += __shfl_xor_sync(full, ws, o);
    if (lane == 0) warp_tot[warp] = ws;
    __syncthreads();
    if (tid == 0) {
      float t = 0.f;
      for (int w = 0; w < kSampWarps; ++w) t += warp_tot[w];
      w_cta = t;
    }
    cluster.sync();
    if (c == 0 && tid == 0) {
      // the threshold and the CTA whose range holds it: the first with
      // positive weight whose range ends past it, else (rounding) the last
      // with positive weight
      float wc[16];
      float total = 0.f;
      for (int peer = 0; peer < CL; ++peer) {
        wc[peer] = *cluster.map_shared_rank(&w_cta, peer);
        total += wc[peer];
      }
      const float thr = u_sample[b] * total;
      int owner = -1, last = -1;
      float off = 0.f, own_off = 0.f, last_off = 0.f;
      for (int peer = 0; peer < CL; ++peer) {
        if (wc[peer] > 0.f) {
          if (owner < 0 && thr < off + wc[peer]) {
            owner = peer;
            own_off = off;
          }
          last = peer;
          last_off = off;
        }
        off += wc[peer];
      }
      if (owner < 0) {
        owner = last;
        own_off = last_off;
      }
      for (int peer = 0; peer < CL; ++peer) {
        *cluster.map_shared_rank(&w_state, peer) = total > (resid ? kResidFloor : 0.f) ? 1 : 0;
        *cluster.map_shared_rank(&w_thr, peer) = peer == owner ? thr : -1.f;
        *cluster.map_shared_rank(&w_off, peer) = own_off;
      }
    }
    cluster.sync();
    if (w_state || !resid) break;
    resid = false;
  }
  // no positive weight at all (non-finite logits): no token can be drawn
  if (!w_state && c == 0 && tid == 0) out_tokens[static_cast<size_t>(b) * (gamma + 1) + a] = -1;
  const float thr = w_thr;
  if (thr >= 0.f) {
    // exclusive prefix of the threads' run totals, in thread order
    if (tid == 0) {
      pick_t = 0x7fffffff;
      last_t = -1;
    }
    float x = ts;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(full, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    float lo = w_off + x - ts;
    for (int w = 0; w < warp; ++w) lo += warp_tot[w];
    // the first thread of positive weight whose run ends past the threshold,
    // else (rounding) the last thread of positive weight
    if (ts > 0.f) {
      if (thr < lo + ts) atomicMin(&pick_t, tid);
      atomicMax(&last_t, tid);
    }
    __syncthreads();
    const int owner_t = pick_t != 0x7fffffff ? pick_t : last_t;
    if (tid == owner_t) {
      int tok = -1, last_pos = -1;
      float cum = lo;
      for (int v = r0; v < r1; ++v) {
        const float w = weight(v);
        if (w > 0.f) {
          last_pos = v;
          if (cum + w > thr) {
            tok = v;
            break;
          }
        }
        cum += w;
      }
      out_tokens[static_cast<size_t>(b) * (gamma + 1) + a] = tok >= 0 ? tok : last_pos;
    }
  }
  cluster.sync();  // peers stay resident until every remote access is done
}

struct SampCapacity {
  bool ready = false;
  int resident[17] = {};
};

cudaError_t samp_capacity(const SampCapacity** out) {
  static std::mutex mu;
  static SampCapacity cap[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  SampCapacity& cp = cap[dev];
  if (!cp.ready) {
    e = cudaFuncSetAttribute(accept_sampled_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    for (int cl = 1; cl <= 16; ++cl) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(static_cast<unsigned>(cl));
      cfg.blockDim = dim3(kSampThreads);
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = static_cast<unsigned>(cl);
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      e = cudaOccupancyMaxActiveClusters(&n, accept_sampled_kernel, &cfg);
      if (e != cudaSuccess) return e;
      cp.resident[cl] = n;
    }
    cp.ready = true;
  }
  *out = &cp;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_accept_sampled(const float* target_logits, const float* draft_logits, const int32_t* draft,
                                  const float* u_accept, const float* u_sample, float temperature, int Bt,
                                  int gamma, int vocab, int32_t* accepted_len, int32_t* out_tokens,
                                  int32_t* err_word, cudaStream_t stream) {
  const SampCapacity* cap = nullptr;
  cudaError_t e = samp_capacity(&cap);
  if (e != cudaSuccess) return e;
  int CL = 1;
  for (int cl = 16; cl >= 1; cl >>= 1)
    if (cap->resident[cl] >= Bt) {
      CL = cl;
      break;
    }
  const int vec4 = (vocab % 4 == 0) && ((reinterpret_cast<uintptr_t>(target_logits) & 15u) == 0) &&
                   ((reinterpret_cast<uintptr_t>(draft_logits) & 15u) == 0);
  return launch_overlapped(accept_sampled_kernel, dim3(static_cast<unsigned>(Bt) * CL), dim3(kSampThreads), 0,
                           stream, static_cast<unsigned>(CL), target_logits, draft_logits, draft, u_accept, u_sample,
                           kLog2e / temperature, gamma, vocab, vec4, accepted_len, out_tokens, err_word);
}

}  // namespace simsd
