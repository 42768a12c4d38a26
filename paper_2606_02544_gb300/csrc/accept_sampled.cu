// accept_sampled.cu -- stochastic acceptance of the drafts (Sec. 3.2, Eq. (2)):
// draft r is accepted iff u_r < alpha_r = min(1, p_theta(x_r) / p_phi(x_r)),
// p = softmax(logits / T), along the draft order up to the first rejection a;
// the token at position a is drawn from the residual max(0, p_theta - p_phi)
// (renormalised) or, when every draft is accepted, from p_theta of the extra
// target row, by inverse CDF with a given uniform u_sample.
//
// One thread-block cluster per sequence.  Phase 1: the sequence's gamma+1
// target rows and gamma draft rows are laid end to end, each row padded to a
// multiple of 32 units (a unit is 4 floats, or 1 when rows are not 16-byte
// aligned), and the CTAs take contiguous spans of warp-aligned units, so the
// 32 lanes of a warp are always on the same row.  Each lane keeps the running maximum m of
// z = x*log2(e)/T and s = sum 2^(z - m) of its row; when the warp moves to
// the next row it merges its lanes by shuffles into a per-warp slot (no
// atomics).  CTA 0 merges the warps' and the CTAs' pairs (distributed
// shared memory), forms alpha_r from the drafts' own logits (fetched at the
// start, while phase 1 streams) and the accepted length a, and broadcasts a.
// Phase 2: each CTA takes a range of row a and each warp a contiguous part
// of that, which it sums in coalesced steps of 32 units, keeping the sums of
// up to 64 macro-steps.  CTA 0 forms the threshold u_sample * total and names
// the CTA whose range holds it; there the warp whose part holds it finds the
// macro-step by a scan of the kept sums and walks only that one.  Row a is read a second time (2 of the
// 2*gamma+1 rows); no global scratch memory is used.
//
// Few sequences with a caller workspace: phase 1 is split over many CTAs
// that need not be resident together (samp_part_kernel, per-part (m, s) of
// every row), then samp_resid_kernel, one CTA per (sequence, part), merges
// the (m, s), takes a, sums its span of row a and lets the last CTA of the
// sequence draw the token: no cluster and no CTA waiting for another.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cfloat>
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace simsd {
namespace {

constexpr int kSampThreads = 512;
constexpr int kSampWarps = kSampThreads / 32;
constexpr int kSampMaxRows = 65;  // 2*gamma+1 <= 65
constexpr int kSampMaxCluster = 16;
constexpr int kSampMacros = 64;  // phase 2: macro-steps kept per warp
constexpr float kLog2e = 1.4426950408889634f;
// The running maximum starts at -FLT_MAX rather than -inf: 2^(z - m) is then
// 0 for z = -inf (a masked logit) without a special case, and merging two
// empty pairs gives an empty pair (s = 0).
constexpr float kEmpty = -FLT_MAX;
// A residual whose total is at most this is empty: p_theta and p_phi agree
// to fp32 precision (each probability carries a relative error of a few
// units of 2^-22, the row sums about 1e-6), so what is left is rounding.
constexpr float kResidFloor = 1.0f / 65536.0f;

// 2^x by the PTX approximation (relative error about 2^-22; results below
// 2^-126 flush to 0, far below any weight that matters in a row whose
// largest weight is 1).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Merges two (m, s) pairs of a base-2 log-sum-exp: s = s1 2^(m1 - M) +
// s2 2^(m2 - M), M = max(m1, m2).
__device__ __forceinline__ void ms_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  s = s * ex2(m - M) + s2 * ex2(m2 - M);
  m = M;
}

__device__ __forceinline__ float4 ld_stream_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
  const unsigned sa = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(sa), "l"(gmem) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Row `row` of the combined row space: target rows 0..gamma, then draft rows.
__device__ __forceinline__ const float* row_ptr(const float* tgt, const float* drf, int b, int gamma, int vocab,
                                                int row) {
  return row <= gamma ? tgt + (static_cast<size_t>(b) * (gamma + 1) + row) * vocab
                      : drf + (static_cast<size_t>(b) * gamma + (row - gamma - 1)) * vocab;
}

// the same through L1 (phase 2 re-reads a thread's lines)
template <bool VEC>
__device__ __forceinline__ float4 load_unit_cached(const float* rp, int col) {
  if constexpr (VEC) {
    return __ldg(reinterpret_cast<const float4*>(rp) + col);
  } else {
    return make_float4(__ldg(rp + col), -INFINITY, -INFINITY, -INFINITY);
  }
}

template <bool VEC>
__device__ __forceinline__ float4 load_unit(const float* rp, int col) {
  if constexpr (VEC) {
    return ld_stream_f4(rp + 4 * col);
  } else {
    return make_float4(__ldg(rp + col), -INFINITY, -INFINITY, -INFINITY);
  }
}

// The accepted length of sequence b (one warp, lane r taking draft r): with
// the rows' base-2 log-sum-exp (m, s) in row_m / row_s and the drafts' own
// logits zt / zd, draft r is accepted iff u_r < alpha_r = min(1,
// p_theta(x_r) / p_phi(x_r)); a is the first rejection (gamma when there is
// none).  A draft token out of range is rejected and flagged.  With `write`
// set, lane 0 stores a and the lanes the tokens of every position but a
// (accepted drafts, then -1).
__device__ __forceinline__ int accept_walk(int b, int gamma, int vocab, float zscale, const float* row_m,
                                           const float* row_s, float zt, float zd, float ua, bool bad,
                                           const int32_t* __restrict__ draft, int32_t* __restrict__ accepted_len,
                                           int32_t* __restrict__ out_tokens, int32_t* err_word, bool write) {
  const int lane = threadIdx.x & 31;
  const unsigned full = 0xffffffffu;
  bool acc = false;
  if (lane < gamma && !bad) {
    // log2 of p_theta(x) / p_phi(x)
    const int rd = gamma + 1 + lane;
    const float lr = (zt * zscale - row_m[lane] - log2f(row_s[lane])) - (zd * zscale - row_m[rd] - log2f(row_s[rd]));
    const float alpha = lr >= 0.f ? 1.f : exp2f(lr);
    acc = ua < alpha;
  }
  const unsigned rej = __ballot_sync(full, lane < gamma && !acc);
  const int a = rej ? __ffs(rej) - 1 : gamma;
  if (write) {
    if (__any_sync(full, bad) && lane == 0) raise_error(err_word, SIMSD_EW_DRAFT);
    if (lane == 0) accepted_len[b] = a;
    int32_t* ot = out_tokens + static_cast<size_t>(b) * (gamma + 1);
    for (int r = lane; r <= gamma; r += 32)
      if (r != a) ot[r] = r < a ? draft[static_cast<size_t>(b) * gamma + r] : -1;
  }
  (void)vocab;
  return a;
}

// Phase 1 of one CTA: the running (m, s) of z = x log2(e) / T over span c
// of CL equal spans of the sequence's rows (target rows 0..gamma, then
// draft rows), merged per warp into part[warp][row].
template <bool VEC, int UNROLL>
__device__ __forceinline__ void phase1_span(const float* __restrict__ tgt, const float* __restrict__ drf, int b,
                                            int gamma, int vocab, float zscale, int c, int CL,
                                            float2 (*part)[kSampMaxRows]) {
  const int rows = 2 * gamma + 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned full = 0xffffffffu;
  const int W = VEC ? (vocab >> 2) : vocab;  // units per row
  const int Wp = (W + 31) & ~31;             // padded: a warp never straddles two rows
  const int G = rows * (Wp >> 5);            // groups of 32 units
  const int per = (G + CL - 1) / CL;
  const int f0 = 32 * min(G, c * per), f1 = 32 * min(G, c * per + per);
  constexpr int kStep = kSampThreads;
  int f = f0 + tid;
  int row = f / Wp;
  int col = f - row * Wp;
  const float* rp = row_ptr(tgt, drf, b, gamma, vocab, min(row, rows - 1));
  int cur = row;
  float m = kEmpty, s = 0.f;
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
  auto advance = [&](int by) {
    col += by;
    if (col >= Wp) {
      do {
        col -= Wp;
        ++row;
      } while (col >= Wp);
      rp = row_ptr(tgt, drf, b, gamma, vocab, min(row, rows - 1));
    }
  };
  // Loads of H units.  f0, f1, Wp and the f and col of a warp's first lane
  // are multiples of 32, so every test here is the same for the 32 lanes
  // of a warp.  vr[u] is the unit's row, -1 past the span.
  constexpr int H = UNROLL == 16 ? 8 : UNROLL;
  auto fetch = [&](float4(&v)[H], int(&vr)[H]) {
    if (f - lane + kStep * (H - 1) < f1 && col - lane + kStep * (H - 1) + 31 < W) {
      // the common case: every unit valid, on one row, inside the row
#pragma unroll
      for (int u = 0; u < H; ++u) {
        v[u] = load_unit<VEC>(rp, col + u * kStep);
        vr[u] = row;
      }
      advance(kStep * H);
    } else {
#pragma unroll
      for (int u = 0; u < H; ++u) {
        vr[u] = -1;
        if (f + u * kStep < f1) {
          vr[u] = row;
          v[u] = col < W ? load_unit<VEC>(rp, col) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        }
        advance(kStep);
      }
    }
    f += kStep * H;
  };
  auto consume = [&](const float4(&v)[H], const int(&vr)[H]) {
#pragma unroll
    for (int u = 0; u < H; ++u) {
      if (vr[u] < 0) break;
      if (vr[u] != cur) {
        flush();
        cur = vr[u];
        m = kEmpty;
        s = 0.f;
      }
      const float mz = fmaxf(fmaxf(v[u].x, v[u].y), fmaxf(v[u].z, v[u].w)) * zscale;
      if (mz > m) {
        s *= ex2(m - mz);
        m = mz;
      }
      const float nm = -m;
      s += ex2(fmaf(v[u].x, zscale, nm)) + ex2(fmaf(v[u].y, zscale, nm)) + ex2(fmaf(v[u].z, zscale, nm)) +
           ex2(fmaf(v[u].w, zscale, nm));
    }
  };
  if constexpr (UNROLL == 16) {
    // one CTA per SM: two batches of 8, the next one's loads in flight
    // while the current one is summed
    float4 va[H], vb[H];
    int ra[H], rb[H];
    fetch(va, ra);
    while (ra[0] >= 0) {
      fetch(vb, rb);
      consume(va, ra);
      if (rb[0] < 0) break;
      fetch(va, ra);
      consume(vb, rb);
    }
  } else {
    float4 v[H];
    int vr[H];
    for (;;) {
      fetch(v, vr);
      if (vr[0] < 0) break;
      consume(v, vr);
    }
  }
  if (f0 + 32 * warp < f1) flush();
}

// Units in flight per thread in phase 1: UNROLL 8 with two CTAs per SM;
// UNROLL 16 when the grid has at most one CTA per SM (small batches), where
// the CTA's bytes in flight set its bandwidth: two batches of 8, one loading
// while the other is summed.
template <bool VEC, int UNROLL>
__global__ void __launch_bounds__(kSampThreads, UNROLL == 8 ? 2 : 1) accept_sampled_kernel(
    const float* __restrict__ tgt, const float* __restrict__ drf, const int32_t* __restrict__ draft,
    const float* __restrict__ u_accept, const float* __restrict__ u_sample, float zscale, int gamma, int vocab,
    int32_t* __restrict__ accepted_len, int32_t* __restrict__ out_tokens, int32_t* err_word) {
  __shared__ float2 part[kSampWarps][kSampMaxRows];  // per warp (m, s) of each row
  __shared__ float2 cta_ms[kSampMaxRows];            // this CTA's (m, s) of each row
  __shared__ float row_m[kSampMaxRows], row_s[kSampMaxRows];
  __shared__ float warp_tot[kSampWarps];
  __shared__ float zt_sh[32], zd_sh[32], ua_sh[32];  // CTA 0: the drafts' logits and u_accept
  __shared__ float us_sh;                            // CTA 0: u_sample
  __shared__ int a_sh;
  __shared__ float w_cta;          // this CTA's weight of row a
  __shared__ float w_off, w_thr;   // the owner's offset and threshold (-1 elsewhere), set by CTA 0
  __shared__ int w_state;          // 1: the total weight was positive (set by CTA 0)
  __shared__ float mac[kSampWarps][kSampMacros];     // phase 2: weight of each macro-step
  pdl_wait();
  cg::cluster_group cluster = cg::this_cluster();
  const int CL = static_cast<int>(cluster.num_blocks());
  const int c = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.x / CL;
  const int rows = 2 * gamma + 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned full = 0xffffffffu;
  for (int i = tid; i < kSampWarps * kSampMaxRows; i += kSampThreads)
    part[i / kSampMaxRows][i % kSampMaxRows] = make_float2(kEmpty, 0.f);
  // CTA 0, warp 0: the drafts, their two logits and the uniforms, fetched now
  // so that their latency hides behind phase 1
  bool bad = false;
  if (c == 0 && warp == 0) {
    if (lane < gamma) {
      const int x = draft[static_cast<size_t>(b) * gamma + lane];
      ua_sh[lane] = u_accept[static_cast<size_t>(b) * gamma + lane];
      bad = x < 0 || x >= vocab;
      if (!bad) {
        cp_async4(&zt_sh[lane], tgt + (static_cast<size_t>(b) * (gamma + 1) + lane) * vocab + x);
        cp_async4(&zd_sh[lane], drf + (static_cast<size_t>(b) * gamma + lane) * vocab + x);
      }
    }
    if (lane == 31) us_sh = u_sample[b];
  }
  __syncthreads();

  // ---- phase 1: per-row (m, s) over this CTA's span of warp-aligned units
  phase1_span<VEC, UNROLL>(tgt, drf, b, gamma, vocab, zscale, c, CL, part);
  // the next kernel may be scheduled once the logits have streamed through
  pdl_launch_next();
  __syncthreads();
  for (int r = tid; r < rows; r += kSampThreads) {
    float m = kEmpty, s = 0.f;
#pragma unroll
    for (int w = 0; w < kSampWarps; ++w) ms_merge(m, s, part[w][r].x, part[w][r].y);
    cta_ms[r] = make_float2(m, s);
  }
  cluster.sync();

  // ---- CTA 0: merge the CTAs, alpha_r, accepted length
  if (c == 0) {
    // warp w merges rows w, w+16, ...; lane p reads CTA p's pair
    constexpr int kRowsPerWarp = (kSampMaxRows + kSampWarps - 1) / kSampWarps;
    float2 pv[kRowsPerWarp];
#pragma unroll
    for (int j = 0; j < kRowsPerWarp; ++j) {
      const int r = warp + kSampWarps * j;
      pv[j] = (r < rows && lane < CL) ? *cluster.map_shared_rank(&cta_ms[r], lane) : make_float2(kEmpty, 0.f);
    }
#pragma unroll
    for (int j = 0; j < kRowsPerWarp; ++j) {
      const int r = warp + kSampWarps * j;
      if (r < rows) {  // the same for the whole warp
        float m = pv[j].x, s = pv[j].y;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float m2 = __shfl_xor_sync(full, m, o), s2 = __shfl_xor_sync(full, s, o);
          ms_merge(m, s, m2, s2);
        }
        if (lane == 0) {
          row_m[r] = m;
          row_s[r] = s;
        }
      }
    }
    __syncthreads();
    if (warp == 0) {
      cp_async_wait_all();
      __syncwarp();
      const bool lb = lane < gamma;
      const int a = accept_walk(b, gamma, vocab, zscale, row_m, row_s, lb ? zt_sh[lane] : 0.f,
                                lb ? zd_sh[lane] : 0.f, lb ? ua_sh[lane] : 0.f, bad, draft, accepted_len, out_tokens,
                                err_word, true);
      // a and the merged (m, s) of the rows phase 2 needs, to every CTA
      if (lane < CL) {
        const int rd = gamma + 1 + a;
        *cluster.map_shared_rank(&a_sh, lane) = a;
        *cluster.map_shared_rank(&row_m[a], lane) = row_m[a];
        *cluster.map_shared_rank(&row_s[a], lane) = row_s[a];
        if (a < gamma) {
          *cluster.map_shared_rank(&row_m[rd], lane) = row_m[rd];
          *cluster.map_shared_rank(&row_s[rd], lane) = row_s[rd];
        }
      }
    }
  }
  cluster.sync();

  // ---- phase 2: weights of row a.  CTA c takes a range of units of the
  // row and warp w a contiguous part of that, in steps of 32 units (one per
  // lane, coalesced); the warp keeps the weight of every macro-step of M
  // steps, at most kSampMacros of them, so that the draw walks one macro.
  const int a = a_sh;
  bool resid = a < gamma;
  const float* trow = tgt + (static_cast<size_t>(b) * (gamma + 1) + a) * vocab;
  const float* drow = a < gamma ? drf + (static_cast<size_t>(b) * gamma + a) * vocab : trow;
  const float nmt = -row_m[a], it = 1.f / row_s[a];
  const float nmd = a < gamma ? -row_m[gamma + 1 + a] : 0.f, id = a < gamma ? 1.f / row_s[gamma + 1 + a] : 0.f;
  const int W = VEC ? (vocab >> 2) : vocab;
  const int per_c = (W + CL - 1) / CL;
  const int c0 = min(W, c * per_c), c1 = min(W, c0 + per_c);
  const int per_w = (((c1 - c0 + kSampWarps - 1) / kSampWarps) + 31) & ~31;
  const int w0 = min(c1, c0 + warp * per_w), w1 = min(c1, w0 + per_w);
  const int nsteps = (w1 - w0 + 31) >> 5;
  const int M = max(1, (nsteps + kSampMacros - 1) / kSampMacros);
  const int nmac = (nsteps + M - 1) / M;
  // the four weights of a unit (the scalar layout has one column per unit)
  auto weights = [&](const float4& xt, const float4& xd) -> float4 {
    float4 w = make_float4(ex2(fmaf(xt.x, zscale, nmt)) * it, ex2(fmaf(xt.y, zscale, nmt)) * it,
                           ex2(fmaf(xt.z, zscale, nmt)) * it, ex2(fmaf(xt.w, zscale, nmt)) * it);
    if (resid) {
      w.x = fmaxf(0.f, w.x - ex2(fmaf(xd.x, zscale, nmd)) * id);
      w.y = fmaxf(0.f, w.y - ex2(fmaf(xd.y, zscale, nmd)) * id);
      w.z = fmaxf(0.f, w.z - ex2(fmaf(xd.z, zscale, nmd)) * id);
      w.w = fmaxf(0.f, w.w - ex2(fmaf(xd.w, zscale, nmd)) * id);
    }
    return w;
  };
  const float4 kNone = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  // loads of 4 steps from step i0 (units past the part give weight 0)
  auto load4 = [&](int i0, float4(&xt)[4], float4(&xd)[4]) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int u = w0 + 32 * (i0 + j) + lane;
      const bool ok = u < w1;
      xt[j] = ok ? load_unit_cached<VEC>(trow, u) : kNone;
      xd[j] = ok && resid ? load_unit_cached<VEC>(drow, u) : kNone;
    }
  };
  // an empty residual (p_theta = p_phi to fp32 precision) cannot reject:
  // the draw then falls back to p_theta (second pass)
  for (int pass = 0; pass < 2; ++pass) {
    float acc = 0.f, wt = 0.f;
    for (int i0 = 0; i0 < nsteps; i0 += 4) {
      float4 xt[4], xd[4];
      load4(i0, xt, xd);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = i0 + j;
        if (i >= nsteps) break;
        const float4 w = weights(xt[j], xd[j]);
        acc += (w.x + w.y) + (w.z + w.w);
        if ((i + 1) % M == 0 || i + 1 == nsteps) {
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(full, acc, o);
          if (lane == 0) mac[warp][i / M] = acc;
          wt += acc;
          acc = 0.f;
        }
      }
    }
    if (lane == 0) warp_tot[warp] = wt;
    __syncthreads();
    if (tid == 0) {
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < kSampWarps; ++w) t += warp_tot[w];
      w_cta = t;
    }
    cluster.sync();
    if (c == 0 && warp == 0) {
      // lane p holds CTA p's weight; the threshold and the CTA whose range
      // holds it: the first with positive weight whose range ends past it,
      // else (rounding) the last with positive weight
      const float wc = lane < CL ? *cluster.map_shared_rank(&w_cta, lane) : 0.f;
      float incl = wc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(full, incl, o);
        if (lane >= o) incl += y;
      }
      const float total = __shfl_sync(full, incl, 31);
      const float thr = us_sh * total;
      const unsigned hold = __ballot_sync(full, wc > 0.f && thr < incl);
      const unsigned pos = __ballot_sync(full, wc > 0.f);
      const int owner = hold ? __ffs(hold) - 1 : (pos ? 31 - __clz(pos) : -1);
      const float own_off = __shfl_sync(full, incl - wc, owner < 0 ? 0 : owner);
      if (lane < CL) {
        *cluster.map_shared_rank(&w_state, lane) = total > (resid ? kResidFloor : 0.f) ? 1 : 0;
        *cluster.map_shared_rank(&w_thr, lane) = lane == owner ? thr : -1.f;
        *cluster.map_shared_rank(&w_off, lane) = own_off;
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
    // the warp whose part holds the threshold: the first of positive weight
    // whose part ends past it, else (rounding) the last of positive weight
    float lo = w_off;
    int owner_w = -1, last_w = -1;
    float last_lo = lo;
    for (int w = 0; w < kSampWarps; ++w) {
      const float t = warp_tot[w];
      if (t > 0.f) {
        if (thr < lo + t) {
          owner_w = w;
          break;
        }
        last_w = w;
        last_lo = lo;
      }
      lo += t;
    }
    if (owner_w < 0) {
      owner_w = last_w;
      lo = last_lo;
    }
    if (warp == owner_w) {
      // the macro-step that holds the threshold, by a scan of the macro
      // weights (lane k holds macros k and 32 + k), with the same fallback
      const float ma = lane < nmac ? mac[warp][lane] : 0.f;
      const float mb = lane + 32 < nmac ? mac[warp][lane + 32] : 0.f;
      float ia = ma, ib = mb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float ya = __shfl_up_sync(full, ia, o), yb = __shfl_up_sync(full, ib, o);
        if (lane >= o) {
          ia += ya;
          ib += yb;
        }
      }
      ib += __shfl_sync(full, ia, 31);
      const unsigned ha = __ballot_sync(full, ma > 0.f && thr < lo + ia);
      const unsigned hb = __ballot_sync(full, mb > 0.f && thr < lo + ib);
      const unsigned pa = __ballot_sync(full, ma > 0.f), pb = __ballot_sync(full, mb > 0.f);
      int k = ha ? __ffs(ha) - 1 : hb ? 32 + __ffs(hb) - 1 : pb ? 63 - __clz(pb) : pa ? 31 - __clz(pa) : 0;
      float base = lo + __shfl_sync(full, k < 32 ? ia - ma : ib - mb, k & 31);
      // walk the macro's steps in order: lane sums, a warp scan, and the
      // first lane whose cumulative weight passes the threshold
      int tok = -1, last_pos = -1;
      const int s_end = min(nsteps, (k + 1) * M);
      for (int i0 = k * M; i0 < s_end && tok < 0; i0 += 4) {
        float4 xt[4], xd[4];
        load4(i0, xt, xd);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (tok >= 0 || i0 + j >= s_end) break;
          const int u = w0 + 32 * (i0 + j) + lane;
          const float4 w = weights(xt[j], xd[j]);
          const float w4[4] = {w.x, w.y, w.z, w.w};
          const float ls = (w4[0] + w4[1]) + (w4[2] + w4[3]);
          float incl = ls;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const float y = __shfl_up_sync(full, incl, o);
            if (lane >= o) incl += y;
          }
          // this lane's first column passing the threshold, and its last
          // column of positive weight
          int hit_col = -1, pos_col = -1;
          float cum = base + incl - ls;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            if (w4[e] > 0.f) {
              if (hit_col < 0 && cum + w4[e] > thr) hit_col = VEC ? 4 * u + e : u;
              pos_col = VEC ? 4 * u + e : u;
            }
            cum += w4[e];
          }
          const unsigned hit = __ballot_sync(full, hit_col >= 0);
          const unsigned pos = __ballot_sync(full, pos_col >= 0);
          if (hit) tok = __shfl_sync(full, hit_col, __ffs(hit) - 1);
          if (pos) last_pos = __shfl_sync(full, pos_col, 31 - __clz(pos));
          base += __shfl_sync(full, incl, 31);
        }
      }
      if (lane == 0) out_tokens[static_cast<size_t>(b) * (gamma + 1) + a] = tok >= 0 ? tok : last_pos;
    }
  }
  cluster.sync();  // peers stay resident until every remote access is done
}

// Few sequences: phase 1 of each sequence split over `parts` CTAs that need
// not be resident together; each merges its warps' pairs and writes the
// (m, s) of every row to pre[b][part][row] (rows outside its span get the
// empty pair).  accept_sampled_kernel then merges these instead of
// streaming the logits itself.
template <bool VEC>
__global__ void __launch_bounds__(kSampThreads, 2) samp_part_kernel(const float* __restrict__ tgt,
                                                                    const float* __restrict__ drf, float zscale,
                                                                    int gamma, int vocab, int parts,
                                                                    float2* __restrict__ pre,
                                                                    unsigned* __restrict__ arrivals) {
  __shared__ float2 part[kSampWarps][kSampMaxRows];
  const int b = blockIdx.x / parts, c = blockIdx.x - b * parts;
  const int rows = 2 * gamma + 1;
  const int tid = threadIdx.x;
  for (int i = tid; i < kSampWarps * kSampMaxRows; i += kSampThreads)
    part[i / kSampMaxRows][i % kSampMaxRows] = make_float2(kEmpty, 0.f);
  pdl_wait();
  // the arrival count samp_resid_kernel uses for this sequence starts at 0
  if (c == 0 && tid == 0) arrivals[b] = 0u;
  __syncthreads();
  phase1_span<VEC, 8>(tgt, drf, b, gamma, vocab, zscale, c, parts, part);
  __syncthreads();
  for (int r = tid; r < rows; r += kSampThreads) {
    float m = kEmpty, s = 0.f;
#pragma unroll
    for (int w = 0; w < kSampWarps; ++w) ms_merge(m, s, part[w][r].x, part[w][r].y);
    pre[(static_cast<size_t>(b) * parts + c) * rows + r] = make_float2(m, s);
  }
  pdl_launch_next();
}

// Row a's weights at one unit of 4 columns (1 in the scalar layout, the
// other three 0): p_theta = 2^(z_t - m_t) / s_t and the residual
// max(0, p_theta - p_phi) (p_theta again when there is no draft row).
struct RowW {
  const float* trow;
  const float* drow;
  float zscale, nmt, it, nmd, id;
  bool resid;
};
struct UnitW {
  float4 t, r;
};
template <bool VEC>
__device__ __forceinline__ UnitW unit_weights(const RowW& w, int u) {
  const float4 xt = load_unit_cached<VEC>(w.trow, u);
  UnitW o;
  o.t = make_float4(ex2(fmaf(xt.x, w.zscale, w.nmt)) * w.it, ex2(fmaf(xt.y, w.zscale, w.nmt)) * w.it,
                    ex2(fmaf(xt.z, w.zscale, w.nmt)) * w.it, ex2(fmaf(xt.w, w.zscale, w.nmt)) * w.it);
  if (w.resid) {
    const float4 xd = load_unit_cached<VEC>(w.drow, u);
    o.r = make_float4(fmaxf(0.f, o.t.x - ex2(fmaf(xd.x, w.zscale, w.nmd)) * w.id),
                      fmaxf(0.f, o.t.y - ex2(fmaf(xd.y, w.zscale, w.nmd)) * w.id),
                      fmaxf(0.f, o.t.z - ex2(fmaf(xd.z, w.zscale, w.nmd)) * w.id),
                      fmaxf(0.f, o.t.w - ex2(fmaf(xd.w, w.zscale, w.nmd)) * w.id));
  } else {
    o.r = o.t;
  }
  return o;
}

// Sum of a value over the CTA (every thread gets it).
__device__ __forceinline__ float cta_sum(float v, float* red) {
  const unsigned full = 0xffffffffu;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(full, v, o);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kSampWarps; ++w) t += red[w];
  return t;
}

// Few sequences, after samp_part_kernel: one CTA per (sequence b, span c of
// row a; rparts spans).  Every CTA merges the parts' (m, s) of every row
// (over the parts whose spans overlap the row) and takes the accepted
// length a itself (part 0 stores the outputs); then it sums the weights of
// its span c of row a's units, both the residual max(0, p_theta -
// p_phi) and p_theta (the fallback when the residual is empty), and
// counts itself in.  The last CTA of the sequence to arrive draws the token
// by inverse CDF with u_sample: the spans in order of the vocabulary give
// the one that holds the threshold (the first of positive weight whose end
// passes it, else, by rounding, the last of positive weight), and a scan of
// that span the token (the first of positive weight whose cumulative weight
// passes it, else the last of positive weight).  No CTA waits for another.
template <bool VEC>
__global__ void __launch_bounds__(kSampThreads, 2) samp_resid_kernel(
    const float* __restrict__ tgt, const float* __restrict__ drf, const int32_t* __restrict__ draft,
    const float* __restrict__ u_accept, const float* __restrict__ u_sample, float zscale, int gamma, int vocab,
    int32_t* __restrict__ accepted_len, int32_t* __restrict__ out_tokens, int32_t* err_word,
    const float2* __restrict__ pre, int parts, int rparts, float2* __restrict__ sums,
    unsigned* __restrict__ arrivals) {
  __shared__ float row_m[kSampMaxRows], row_s[kSampMaxRows];
  __shared__ float red[kSampWarps], red2[kSampWarps];
  __shared__ int a_sh, last_sh, tok_sh, pos_sh;
  __shared__ float thr_sh, base_sh;
  __shared__ int owner_sh, mode_sh;  // mode: 0 residual, 1 p_theta, -1 no positive weight
  const int b = blockIdx.x / rparts, c = blockIdx.x - b * rparts;
  const int rows = 2 * gamma + 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned full = 0xffffffffu;
  pdl_wait();
  float zt = 0.f, zd = 0.f, ua = 0.f;
  bool bad = false;
  if (warp == 0 && lane < gamma) {
    const int x = draft[static_cast<size_t>(b) * gamma + lane];
    ua = u_accept[static_cast<size_t>(b) * gamma + lane];
    bad = x < 0 || x >= vocab;
    if (!bad) {
      zt = __ldg(tgt + (static_cast<size_t>(b) * (gamma + 1) + lane) * vocab + x);
      zd = __ldg(drf + (static_cast<size_t>(b) * gamma + lane) * vocab + x);
    }
  }
  // the rows' (m, s): warp w merges rows w, w + 16, ... (at most
  // kRowsPerWarp), lanes over the parts.  samp_part_kernel cut the rows'
  // groups of 32 units into parts of `per` groups, so row r's pair is
  // non-empty only in parts r*Wg/per .. ((r+1)*Wg - 1)/per (the others hold
  // the empty pair, which a merge leaves unchanged); a lane loads one pair
  // of each of the warp's rows per round, all before any is merged
  {
    constexpr int kRowsPerWarp = (kSampMaxRows + kSampWarps - 1) / kSampWarps;
    const int Wg = ((VEC ? (vocab >> 2) : vocab) + 31) >> 5;  // groups per row
    const int per = (rows * Wg + parts - 1) / parts;
    float m[kRowsPerWarp], sm[kRowsPerWarp];
    int q_lo[kRowsPerWarp], q_n[kRowsPerWarp];
    int most = 0;
#pragma unroll
    for (int i = 0; i < kRowsPerWarp; ++i) {
      const int r = warp + kSampWarps * i;
      m[i] = kEmpty;
      sm[i] = 0.f;
      q_lo[i] = r < rows ? r * Wg / per : 0;
      q_n[i] = r < rows ? min(parts - 1, ((r + 1) * Wg - 1) / per) - q_lo[i] + 1 : 0;
      most = max(most, q_n[i]);
    }
    for (int k0 = 0; k0 < most; k0 += 32) {
      float2 v[kRowsPerWarp];
#pragma unroll
      for (int i = 0; i < kRowsPerWarp; ++i) {
        const int k = k0 + lane, r = warp + kSampWarps * i;
        v[i] = k < q_n[i] ? pre[(static_cast<size_t>(b) * parts + q_lo[i] + k) * rows + r] : make_float2(kEmpty, 0.f);
      }
#pragma unroll
      for (int i = 0; i < kRowsPerWarp; ++i)
        if (warp + kSampWarps * i < rows) ms_merge(m[i], sm[i], v[i].x, v[i].y);
    }
#pragma unroll
    for (int i = 0; i < kRowsPerWarp; ++i) {
      const int r = warp + kSampWarps * i;
      if (r >= rows) continue;  // (the same for the whole warp)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(full, m[i], o), s2 = __shfl_xor_sync(full, sm[i], o);
        ms_merge(m[i], sm[i], m2, s2);
      }
      if (lane == 0) {
        row_m[r] = m[i];
        row_s[r] = sm[i];
      }
    }
  }
  __syncthreads();
  if (warp == 0) {
    const int a = accept_walk(b, gamma, vocab, zscale, row_m, row_s, zt, zd, ua, bad, draft, accepted_len,
                              out_tokens, err_word, c == 0);
    if (lane == 0) a_sh = a;
  }
  __syncthreads();
  // ---- the weights of row a over this part's span of units
  const int a = a_sh;
  const bool resid = a < gamma;
  const float* trow = tgt + (static_cast<size_t>(b) * (gamma + 1) + a) * vocab;
  const float* drow = resid ? drf + (static_cast<size_t>(b) * gamma + a) * vocab : trow;
  const float nmt = -row_m[a], it = 1.f / row_s[a];
  const float nmd = resid ? -row_m[gamma + 1 + a] : 0.f, id = resid ? 1.f / row_s[gamma + 1 + a] : 0.f;
  const int W = VEC ? (vocab >> 2) : vocab;
  const int per = (W + rparts - 1) / rparts;
  const RowW rw{trow, drow, zscale, nmt, it, nmd, id, resid};
  {
    const int u0 = min(W, c * per), u1 = min(W, u0 + per);
    float st = 0.f, sr = 0.f;
    for (int u = u0 + tid; u < u1; u += kSampThreads) {
      const UnitW w = unit_weights<VEC>(rw, u);
      st += (w.t.x + w.t.y) + (w.t.z + w.t.w);
      sr += (w.r.x + w.r.y) + (w.r.z + w.r.w);
    }
    st = cta_sum(st, red);
    sr = cta_sum(sr, red2);
    if (tid == 0) {
      sums[static_cast<size_t>(b) * rparts + c] = make_float2(sr, st);
      __threadfence();
      last_sh = atomicAdd(arrivals + b, 1u) == static_cast<unsigned>(rparts - 1);
    }
  }
  pdl_launch_next();
  __syncthreads();
  if (!last_sh) return;
  __threadfence();
  // ---- the last CTA of the sequence: which span holds the threshold
  if (warp == 0) {
    // the other CTAs' sums, read past L1 (they were written by other SMs)
    const volatile float* vs = reinterpret_cast<const volatile float*>(sums + static_cast<size_t>(b) * rparts);
    float tr = 0.f, tt = 0.f;
    for (int q = lane; q < rparts; q += 32) {
      tr += vs[2 * q];
      tt += vs[2 * q + 1];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      tr += __shfl_xor_sync(full, tr, o);
      tt += __shfl_xor_sync(full, tt, o);
    }
    // an empty residual (p_theta = p_phi to fp32 precision) cannot reject:
    // the draw falls back to p_theta
    int mode = (resid && tr > kResidFloor) || (!resid && tr > 0.f) ? 0 : (tt > 0.f ? 1 : -1);
    const float total = mode == 0 ? tr : tt;
    const float thr = u_sample[b] * total;
    int owner = -1, last_pos = -1;
    float base = 0.f, last_base = 0.f, run = 0.f;
    for (int q0 = 0; q0 < rparts && mode >= 0 && owner < 0; q0 += 32) {
      const int q = q0 + lane;
      const float wq = q < rparts ? vs[2 * q + (mode == 0 ? 0 : 1)] : 0.f;
      float incl = wq;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(full, incl, o);
        if (lane >= o) incl += y;
      }
      incl += run;
      const unsigned hold = __ballot_sync(full, wq > 0.f && thr < incl);
      const unsigned pos = __ballot_sync(full, wq > 0.f);
      if (hold) {
        const int l = __ffs(hold) - 1;
        owner = q0 + l;
        base = __shfl_sync(full, incl - wq, l);
      } else if (pos) {
        const int l = 31 - __clz(pos);
        last_pos = q0 + l;
        last_base = __shfl_sync(full, incl - wq, l);
      }
      run = __shfl_sync(full, incl, 31);
    }
    if (owner < 0 && mode >= 0) {
      owner = last_pos;
      base = last_base;
    }
    if (lane == 0) {
      mode_sh = owner < 0 ? -1 : mode;
      owner_sh = owner;
      thr_sh = thr;
      base_sh = base;
      tok_sh = 0x7fffffff;
      pos_sh = -1;
    }
  }
  __syncthreads();
  const int mode = mode_sh;
  if (mode < 0) {
    if (tid == 0) out_tokens[static_cast<size_t>(b) * (gamma + 1) + a] = -1;
    return;
  }
  // ---- the owner span: thread t takes k consecutive units, a scan over the
  // threads, then each thread walks its own units in order
  const int u0 = min(W, owner_sh * per), u1 = min(W, u0 + per);
  const int k = (u1 - u0 + kSampThreads - 1) / kSampThreads;
  const int t0 = min(u1, u0 + tid * k), t1 = min(u1, t0 + k);
  float mine = 0.f;
  for (int u = t0; u < t1; ++u) {
    const UnitW uw = unit_weights<VEC>(rw, u);
    const float4 w = mode == 0 ? uw.r : uw.t;
    mine += (w.x + w.y) + (w.z + w.w);
  }
  // exclusive scan of the threads' sums (in thread order = vocabulary order)
  float incl = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(full, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) red[warp] = incl;
  __syncthreads();
  float before = 0.f;
  for (int w = 0; w < warp; ++w) before += red[w];
  float cum = base_sh + before + incl - mine;
  const float thr = thr_sh;
  int hit = -1, lastp = -1;
  // one column: its weight, then the cumulative weight past it
  auto step = [&](float w, int col) {
    if (w > 0.f) {
      if (hit < 0 && cum + w > thr) hit = col;
      lastp = col;
    }
    cum += w;
  };
  for (int u = t0; u < t1 && hit < 0; ++u) {
    const UnitW uw = unit_weights<VEC>(rw, u);
    const float4 w = mode == 0 ? uw.r : uw.t;
    const int col = VEC ? 4 * u : u;  // (the scalar layout's other three weights are 0)
    step(w.x, col);
    step(w.y, col + 1);
    step(w.z, col + 2);
    step(w.w, col + 3);
  }
  if (hit >= 0) atomicMin(&tok_sh, hit);
  if (lastp >= 0) atomicMax(&pos_sh, lastp);
  __syncthreads();
  if (tid == 0) out_tokens[static_cast<size_t>(b) * (gamma + 1) + a] = tok_sh != 0x7fffffff ? tok_sh : pos_sh;
}

struct SampCapacity {
  bool ready = false;
  int resident8[kSampMaxCluster + 1] = {};   // clusters resident at once, UNROLL 8
  int resident16[kSampMaxCluster + 1] = {};  // UNROLL 16
};

template <bool VEC, int UNROLL>
cudaError_t max_clusters(int cl, int* n) {
  auto kern = accept_sampled_kernel<VEC, UNROLL>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
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
  return cudaOccupancyMaxActiveClusters(n, kern, &cfg);
}

template <int UNROLL>
cudaError_t min_clusters(int cl, int* n) {
  int n1 = 0, n2 = 0;
  cudaError_t e = max_clusters<true, UNROLL>(cl, &n1);
  if (e != cudaSuccess) return e;
  e = max_clusters<false, UNROLL>(cl, &n2);
  *n = n1 < n2 ? n1 : n2;
  return e;
}

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
    for (int cl = 1; cl <= kSampMaxCluster; cl <<= 1) {
      e = min_clusters<8>(cl, &cp.resident8[cl]);
      if (e != cudaSuccess) return e;
      e = min_clusters<16>(cl, &cp.resident16[cl]);
      if (e != cudaSuccess) return e;
    }
    cp.ready = true;
  }
  *out = &cp;
  return cudaSuccess;
}

template <bool VEC, int UNROLL>
cudaError_t launch_samp(dim3 grid, unsigned CL, cudaStream_t stream, const float* tl, const float* dl,
                        const int32_t* draft, const float* ua, const float* us, float zscale, int gamma, int vocab,
                        int32_t* accepted_len, int32_t* out_tokens, int32_t* err_word) {
  return launch_overlapped(accept_sampled_kernel<VEC, UNROLL>, grid, dim3(kSampThreads), 0, stream, CL, tl, dl,
                           draft, ua, us, zscale, gamma, vocab, accepted_len, out_tokens, err_word);
}

}  // namespace

int samp_parts(int Bt, int gamma, int vocab, int num_sms) {
  // as for greedy acceptance: few sequences, each with at least 6 MiB of
  // logits (target and draft rows), about 8 units of 16 bytes per thread
  if (static_cast<long long>(Bt) * kSampMaxCluster > num_sms) return 0;
  const long long rows = 2LL * gamma + 1;
  // at least 3 MiB of logits a sequence (measured with the current second
  // launch, L2 flushed: 1 x 9 rows 23.2 -> 19.6 us, 8 x 17 rows 37.5 -> 34.4
  // us; 4 x 9 rows even)
  if (rows * vocab * 4 < (3LL << 20)) return 0;
  const long long units = rows * ((vocab + 3) / 4);
  // at most two CTAs per SM in all: one wave
  const long long parts = std::min(units / (8LL * kSampThreads), 2LL * num_sms / Bt);
  return parts > kSampMaxCluster ? static_cast<int>(parts) : 0;
}

// Spans of row a in samp_resid_kernel: about 1024 units (16 KB of each of
// the two rows) a CTA, at most the parts of phase 1.
int samp_resid_parts(int parts, int vocab) {
  const int units = (vocab + 3) / 4;
  return std::max(1, std::min(parts, (units + 1023) / 1024));
}

// Workspace of the split path: the parts' (m, s) [Bt][parts][rows] (float2),
// the spans' weight sums of row a [Bt][rparts <= parts] (float2: residual,
// p_theta), then an arrival count per sequence (uint32).
size_t samp_workspace_bytes(int Bt, int gamma, int vocab, int num_sms) {
  const int parts = samp_parts(Bt, gamma, vocab, num_sms);
  if (!parts) return 0;
  const size_t n = static_cast<size_t>(Bt) * parts;
  return n * (2 * gamma + 1) * sizeof(float2) + n * sizeof(float2) + ((static_cast<size_t>(Bt) * 4 + 7) & ~size_t{7});
}

cudaError_t launch_accept_sampled(const float* target_logits, const float* draft_logits, const int32_t* draft,
                                  const float* u_accept, const float* u_sample, float temperature, int Bt,
                                  int gamma, int vocab, int32_t* accepted_len, int32_t* out_tokens,
                                  int32_t* err_word, cudaStream_t stream, void* workspace, int num_sms) {
  const bool vec4 = (vocab % 4 == 0) && ((reinterpret_cast<uintptr_t>(target_logits) & 15u) == 0) &&
                    ((reinterpret_cast<uintptr_t>(draft_logits) & 15u) == 0);
  const float zscale = kLog2e / temperature;
  // with a workspace and few sequences: the log-sum-exp pass split over many
  // CTAs (samp_part_kernel), then samp_resid_kernel over the same CTAs
  const int parts = workspace ? samp_parts(Bt, gamma, vocab, num_sms) : 0;
  if (parts) {
    const size_t n = static_cast<size_t>(Bt) * parts;
    float2* pre = static_cast<float2*>(workspace);
    float2* sums = pre + n * (2 * gamma + 1);
    unsigned* arrivals = reinterpret_cast<unsigned*>(sums + n);
    const dim3 pgrid(static_cast<unsigned>(n));
    const int rparts = samp_resid_parts(parts, vocab);
    const dim3 rgrid(static_cast<unsigned>(Bt) * rparts);
    cudaError_t e = vec4 ? launch_overlapped(samp_part_kernel<true>, pgrid, dim3(kSampThreads), 0, stream, 1u,
                                             target_logits, draft_logits, zscale, gamma, vocab, parts, pre, arrivals)
                         : launch_overlapped(samp_part_kernel<false>, pgrid, dim3(kSampThreads), 0, stream, 1u,
                                             target_logits, draft_logits, zscale, gamma, vocab, parts, pre, arrivals);
    if (e != cudaSuccess) return e;
    return vec4 ? launch_overlapped(samp_resid_kernel<true>, rgrid, dim3(kSampThreads), 0, stream, 1u, target_logits,
                                    draft_logits, draft, u_accept, u_sample, zscale, gamma, vocab, accepted_len,
                                    out_tokens, err_word, static_cast<const float2*>(pre), parts, rparts, sums,
                                    arrivals)
                : launch_overlapped(samp_resid_kernel<false>, rgrid, dim3(kSampThreads), 0, stream, 1u,
                                    target_logits, draft_logits, draft, u_accept, u_sample, zscale, gamma, vocab,
                                    accepted_len, out_tokens, err_word, static_cast<const float2*>(pre), parts, rparts,
                                    sums, arrivals);
  }
  const SampCapacity* cap = nullptr;
  cudaError_t e = samp_capacity(&cap);
  if (e != cudaSuccess) return e;
  // the largest cluster with which the whole batch is resident at once; the
  // deeper unroll when that still holds with one CTA per SM
  int CL = 1;
  for (int cl = kSampMaxCluster; cl >= 1; cl >>= 1)
    if (cap->resident8[cl] >= Bt) {
      CL = cl;
      break;
    }
  const bool deep = cap->resident16[CL] >= Bt;
  const dim3 grid(static_cast<unsigned>(Bt) * CL);
  const unsigned ucl = static_cast<unsigned>(CL);
  if (vec4)
    return deep ? launch_samp<true, 16>(grid, ucl, stream, target_logits, draft_logits, draft, u_accept, u_sample,
                                        zscale, gamma, vocab, accepted_len, out_tokens, err_word)
                : launch_samp<true, 8>(grid, ucl, stream, target_logits, draft_logits, draft, u_accept, u_sample,
                                       zscale, gamma, vocab, accepted_len, out_tokens, err_word);
  return deep ? launch_samp<false, 16>(grid, ucl, stream, target_logits, draft_logits, draft, u_accept, u_sample,
                                       zscale, gamma, vocab, accepted_len, out_tokens, err_word)
              : launch_samp<false, 8>(grid, ucl, stream, target_logits, draft_logits, draft, u_accept, u_sample,
                                      zscale, gamma, vocab, accepted_len, out_tokens, err_word);
}

}  // namespace simsd
