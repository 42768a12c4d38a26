// accept.cu -- greedy longest-prefix acceptance (Sec. 3.2, Eq. (2) at
// temperature 0: the r-th draft is accepted iff it equals the argmax of the
// target's distribution at its verification slot).
//
// One thread-block cluster per sequence.  The CTAs of a cluster split the
// sequence's [gamma+1][vocab] block into contiguous spans; each thread
// streams 16-byte loads (8 or 16 in flight), keeps a running (value, index) per
// row with plain float compares, and folds it into a 64-bit key per row in
// shared memory when its row changes.
// Each CTA then writes its keys into CTA 0's shared memory (distributed
// shared memory) and arrives on an mbarrier there, and exits; CTA 0 waits for
// the CL arrivals, takes the maximum per row and walks the draft order.  No
// global scratch memory is used.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace cg = cooperative_groups;

namespace simsd {

constexpr int kAcceptThreads = 512;
constexpr int kMaxRows = 33;  // gamma + 1 <= 33
constexpr int kMaxCluster = 16;  // CTAs per sequence (non-portable cluster size)

// Total order used by the argmax: larger key = better.  NaN ranks above every
// number, -0.0 equals +0.0, and among equal values the lower index wins
// (the index is stored complemented in the low half).
__device__ __forceinline__ unsigned long long argmax_key(float x, uint32_t idx) {
  uint32_t u = __float_as_uint(x);
  uint32_t k;
  if (x != x) {
    k = 0xFFFFFFFFu;
  } else {
    if (u == 0x80000000u) u = 0u;
    k = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  }
  return (static_cast<unsigned long long>(k) << 32) | static_cast<unsigned long long>(~idx);
}

__device__ __forceinline__ float4 ld_stream_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

// Running argmax of one thread over the elements it visits in increasing
// index order within one row: the strict '>' keeps the first of equal
// values (and treats -0.0 as +0.0); NaNs are tracked apart (first one wins).
struct RowBest {
  float v;
  uint32_t i;
  uint32_t nan_i;
  __device__ __forceinline__ void reset(uint32_t first) {
    v = -INFINITY;
    i = first;
    nan_i = 0xFFFFFFFFu;
  }
  __device__ __forceinline__ void see(float x, uint32_t e) {
    const bool gt = x > v;
    v = gt ? x : v;
    i = gt ? e : i;
  }
  __device__ __forceinline__ unsigned long long key() const {
    return nan_i != 0xFFFFFFFFu ? argmax_key(__int_as_float(0x7fc00000), nan_i) : argmax_key(v, i);
  }
};

// Span c of CL equal spans of one sequence's [rows][vocab] block (in 16-byte
// units when rows are 16-byte aligned): each thread streams its elements
// and folds a running (value, index) per row into best[row] (shared memory,
// 64-bit keys, atomicMax) when its row changes.
template <int UNROLL>
__device__ __forceinline__ void scan_span(const float* __restrict__ base, int rows, int vocab, int vec4, int c, int CL,
                                          unsigned long long* best) {
  const int tid = threadIdx.x;
  const int W = vec4 ? (vocab >> 2) : vocab;   // units per row
  const long long F = static_cast<long long>(rows) * W;
  const long long per = (F + CL - 1) / CL;
  const long long f0 = min(F, c * per), f1 = min(F, f0 + per);
  long long f = f0 + tid;
  int row = static_cast<int>(f / W);
  int col = static_cast<int>(f - static_cast<long long>(row) * W);
  int cur = row;
  RowBest rb;
  rb.reset(vec4 ? 4u * col : static_cast<uint32_t>(col));
  constexpr int kStride = kAcceptThreads;
  if (vec4) {
    const float4* b4 = reinterpret_cast<const float4*>(base);
    for (; f < f1; f += static_cast<long long>(kStride) * UNROLL) {
      float4 v[UNROLL];
#pragma unroll
      for (int u = 0; u < UNROLL; ++u) {
        const long long fu = f + static_cast<long long>(u) * kStride;
        if (fu < f1) v[u] = ld_stream_f4(reinterpret_cast<const float*>(b4 + fu));
      }
#pragma unroll
      for (int u = 0; u < UNROLL; ++u) {
        if (f + static_cast<long long>(u) * kStride >= f1) break;
        if (row != cur) {
          atomicMax(&best[cur], rb.key());
          cur = row;
          rb.reset(4u * col);
        }
        const uint32_t e = 4u * static_cast<uint32_t>(col);
        if (isnan(v[u].x) | isnan(v[u].y) | isnan(v[u].z) | isnan(v[u].w)) {
          if (rb.nan_i == 0xFFFFFFFFu)
            rb.nan_i = isnan(v[u].x) ? e : isnan(v[u].y) ? e + 1 : isnan(v[u].z) ? e + 2 : e + 3;
        }
        rb.see(v[u].x, e);
        rb.see(v[u].y, e + 1);
        rb.see(v[u].z, e + 2);
        rb.see(v[u].w, e + 3);
        col += kStride;
        if (col >= W) {
          row += col / W;
          col %= W;
        }
      }
    }
  } else {
    for (; f < f1; f += kStride) {
      const float x = __ldg(base + f);
      if (row != cur) {
        atomicMax(&best[cur], rb.key());
        cur = row;
        rb.reset(col);
      }
      if (isnan(x) && rb.nan_i == 0xFFFFFFFFu) rb.nan_i = col;
      rb.see(x, static_cast<uint32_t>(col));
      col += kStride;
      if (col >= W) {
        row += col / W;
        col %= W;
      }
    }
  }
  if (f0 + tid < f1) atomicMax(&best[cur], rb.key());
}

// One warp of sequence b, after am[r] (shared memory) holds the argmax of
// every row: the accepted length (drafts in tau order, lane r checks draft
// r; gamma <= 32) and the output tokens.
__device__ __forceinline__ void walk_drafts(const int* am, int dr_lane, int b, int gamma, int vocab,
                                            int32_t* __restrict__ accepted_len, int32_t* __restrict__ out_tokens,
                                            int32_t* __restrict__ row_argmax, int32_t* err_word) {
  const int lane = threadIdx.x & 31;
  const int rows = gamma + 1;
  if (row_argmax)
    for (int r = lane; r < rows; r += 32) row_argmax[static_cast<size_t>(b) * rows + r] = am[r];
  bool in_range = true, match = false;
  if (lane < gamma) {
    in_range = dr_lane >= 0 && dr_lane < vocab;
    match = in_range && dr_lane == am[lane];
  }
  const unsigned bad = __ballot_sync(0xffffffffu, !in_range);
  const unsigned miss = __ballot_sync(0xffffffffu, lane < gamma && !match);
  const int a = miss ? (__ffs(miss) - 1) : gamma;
  if (lane == 0) {
    if (bad) raise_error(err_word, SIMSD_EW_DRAFT);
    accepted_len[b] = a;
  }
  int32_t* ot = out_tokens + static_cast<size_t>(b) * rows;
  for (int r = lane; r < rows; r += 32) ot[r] = r < a ? dr_lane : (r == a ? am[a] : -1);
}

// UNROLL 16-byte loads are in flight per thread: 8 in general, 16 when the
// grid leaves SMs idle (then each CTA has the SM to itself).
template <int UNROLL>
__global__ void __launch_bounds__(kAcceptThreads) accept_kernel(const float* __restrict__ logits,
                                                                const int32_t* __restrict__ draft, int gamma,
                                                                int vocab, int vec4, int32_t* __restrict__ accepted_len,
                                                                int32_t* __restrict__ out_tokens,
                                                                int32_t* __restrict__ row_argmax, int32_t* err_word,
                                                                uint32_t extra_arrivals, unsigned long long wait_ns) {
  __shared__ unsigned long long best[kMaxRows];
  __shared__ unsigned long long gath[kMaxCluster][kMaxRows];  // CTA 0: every CTA's keys
  __shared__ __align__(8) unsigned long long gbar;              // CTA 0: one arrival per CTA
  __shared__ int am[kMaxRows];
  cg::cluster_group cluster = cg::this_cluster();
  const int c = static_cast<int>(cluster.block_rank());
  const int CL = static_cast<int>(cluster.num_blocks());
  const int b = blockIdx.x / CL;
  const int rows = gamma + 1;
  const int tid = threadIdx.x;
  for (int r = tid; r < rows; r += kAcceptThreads) best[r] = 0ull;
  if (c == 0 && tid == 0) {
    mbar_init(smem_u32(&gbar), static_cast<uint32_t>(CL) + extra_arrivals);
    fence_mbar_init();
  }
  // CTA 0's barrier must be initialised before any CTA arrives on it: every
  // thread arrives here and waits just before its first remote write
  cluster_arrive_relaxed();
  pdl_wait();
  // the drafts are needed only at the end; their load is issued now
  const int dr_lane = (c == 0 && tid < gamma) ? draft[static_cast<size_t>(b) * gamma + tid] : 0;
  __syncthreads();

  // This CTA owns one contiguous span of the sequence's [rows][vocab] block
  // (in 16-byte units when rows are 16-byte aligned).
  scan_span<UNROLL>(logits + static_cast<size_t>(b) * rows * vocab, rows, vocab, vec4, c, CL, best);
  // the next kernel may be scheduled once the stream of logits is done
  // (earlier, its waiting CTAs would sit beside this one's)
  pdl_launch_next();
  __syncthreads();
  cluster_wait();
  if (tid < 32) {
    // warp 0 pushes this CTA's keys into CTA 0 and arrives there (release:
    // the pushes of all lanes, ordered by the __syncwarp, go with it)
    unsigned long long* dst = cluster.map_shared_rank(&gath[c][0], 0);
    for (int r = tid; r < rows; r += 32) dst[r] = best[r];
    __syncwarp();
    if (tid == 0) mbar_arrive_cluster(smem_u32(&gbar), 0);
  }
  // Nothing reads this CTA's shared memory: every CTA but CTA 0 is done.
  if (c != 0 || tid >= 32) return;

  // CTA 0, warp 0: lane r takes row r (and row 32 on lane 0)
  const int lane = tid;
  if (!mbar_wait_cluster_warp(smem_u32(&gbar), 0, wait_ns)) {
    if (lane == 0) raise_error(err_word, SIMSD_EW_TIMEOUT);
    return;
  }
  for (int r = lane; r < rows; r += 32) {
    unsigned long long k = 0ull;
    for (int p = 0; p < CL; ++p) k = gath[p][r] > k ? gath[p][r] : k;
    am[r] = static_cast<int>(~static_cast<uint32_t>(k & 0xFFFFFFFFull));
  }
  __syncwarp();
  walk_drafts(am, dr_lane, b, gamma, vocab, accepted_len, out_tokens, row_argmax, err_word);
}


// Few sequences: the block of each sequence is split over `parts` CTAs that
// need not be resident together (no cluster).  Each writes its 64-bit key
// per row to keys[b][row][part]; accept_merge_kernel then takes the maximum
// per row and walks the drafts.  The merge launch is let in as soon as this
// grid has started, so that its launch latency hides behind the streaming
// (its blocks, one per sequence, only wait for this grid to complete).
__global__ void __launch_bounds__(kAcceptThreads) accept_part_kernel(const float* __restrict__ logits, int gamma,
                                                                     int vocab, int vec4, int parts,
                                                                     unsigned long long* __restrict__ keys) {
  __shared__ unsigned long long best[kMaxRows];
  const int b = blockIdx.x / parts, c = blockIdx.x - b * parts;
  const int rows = gamma + 1;
  for (int r = threadIdx.x; r < rows; r += kAcceptThreads) best[r] = 0ull;
  pdl_wait();
  pdl_launch_next();
  __syncthreads();
  scan_span<8>(logits + static_cast<size_t>(b) * rows * vocab, rows, vocab, vec4, c, parts, best);
  __syncthreads();
  for (int r = threadIdx.x; r < rows; r += kAcceptThreads)
    keys[(static_cast<size_t>(b) * rows + r) * parts + c] = best[r];
}

// One block per sequence: warp w takes rows w and w + 32 (the maximum key
// over the parts, lanes over the parts: coalesced loads of
// keys[b][row][part]), then warp 0 walks the drafts.  A lane's keys of both
// rows, up to kMergePer each (the parts of a one-wave grid on up to 160
// SMs), are loaded before any is compared, so that a warp waits for one
// round trip however many rows and parts it has; more parts take further
// rounds.
constexpr int kMergeThreads = 1024;
constexpr int kMergePer = 10;
__global__ void __launch_bounds__(kMergeThreads) accept_merge_kernel(const unsigned long long* __restrict__ keys,
                                                                     int parts, const int32_t* __restrict__ draft,
                                                                     int gamma, int vocab,
                                                                     int32_t* __restrict__ accepted_len,
                                                                     int32_t* __restrict__ out_tokens,
                                                                     int32_t* __restrict__ row_argmax,
                                                                     int32_t* err_word) {
  __shared__ int am[kMaxRows];
  const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int rows = gamma + 1;
  const unsigned full = 0xffffffffu;
  pdl_wait();
  const int dr_lane = (warp == 0 && lane < gamma) ? draft[static_cast<size_t>(b) * gamma + lane] : 0;
  static_assert(kMaxRows <= 2 * (kMergeThreads / 32), "two rows a warp at most");
  const int r0 = warp, r1 = warp + kMergeThreads / 32;
  const bool has0 = r0 < rows, has1 = r1 < rows;
  const unsigned long long* k0 = keys + (static_cast<size_t>(b) * rows + (has0 ? r0 : 0)) * parts;
  const unsigned long long* k1 = keys + (static_cast<size_t>(b) * rows + (has1 ? r1 : 0)) * parts;
  unsigned long long m0 = 0ull, m1 = 0ull;
  for (int p0 = 0; has0 && p0 < parts; p0 += 32 * kMergePer) {
    unsigned long long v0[kMergePer], v1[kMergePer];
#pragma unroll
    for (int j = 0; j < kMergePer; ++j) {
      const int p = p0 + 32 * j + lane;
      v0[j] = p < parts ? k0[p] : 0ull;
      v1[j] = has1 && p < parts ? k1[p] : 0ull;
    }
#pragma unroll
    for (int j = 0; j < kMergePer; ++j) {
      m0 = v0[j] > m0 ? v0[j] : m0;
      m1 = v1[j] > m1 ? v1[j] : m1;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long u0 = __shfl_xor_sync(full, m0, o), u1 = __shfl_xor_sync(full, m1, o);
    m0 = u0 > m0 ? u0 : m0;
    m1 = u1 > m1 ? u1 : m1;
  }
  if (lane == 0 && has0) am[r0] = static_cast<int>(~static_cast<uint32_t>(m0 & 0xFFFFFFFFull));
  if (lane == 0 && has1) am[r1] = static_cast<int>(~static_cast<uint32_t>(m1 & 0xFFFFFFFFull));
  __syncthreads();
  pdl_launch_next();
  if (warp == 0) walk_drafts(am, dr_lane, b, gamma, vocab, accepted_len, out_tokens, row_argmax, err_word);
}

namespace {

// How many clusters of each size (1..16) the device keeps resident at once,
// asked once per device from the occupancy calculator (clusters must fit in
// one GPC, so this is less than SMs x CTAs per SM / size).
struct ClusterCapacity {
  bool ready = false;
  int resident[kMaxCluster + 1] = {};
};

template <int UNROLL>
cudaError_t cluster_capacity(const ClusterCapacity** out) {
  static std::mutex mu;
  static ClusterCapacity cap[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  ClusterCapacity& c = cap[dev];
  if (!c.ready) {
    e = cudaFuncSetAttribute(accept_kernel<UNROLL>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    for (int cl = 1; cl <= kMaxCluster; ++cl) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(static_cast<unsigned>(cl));
      cfg.blockDim = dim3(kAcceptThreads);
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = static_cast<unsigned>(cl);
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      e = cudaOccupancyMaxActiveClusters(&n, accept_kernel<UNROLL>, &cfg);
      if (e != cudaSuccess) return e;
      c.resident[cl] = n;
    }
    c.ready = true;
  }
  *out = &c;
  return cudaSuccess;
}

}  // namespace

int accept_parts(int Bt, int gamma, int vocab, int num_sms) {
  // few sequences only: one 16-CTA cluster each leaves SMs idle
  if (static_cast<long long>(Bt) * kMaxCluster > num_sms) return 0;
  // and at least 4 MiB of logits per sequence: below that the cluster's 16
  // CTAs stream it about as fast as the split, which pays a second launch
  // (measured, L2 flushed: 3 MB per sequence 15.0 us cluster against 15.5
  // us split at 8 sequences; 5.5 MB 21.2 against 18.1 us, 10 MB 23.2
  // against 14.0 us at one sequence)
  if (static_cast<long long>(gamma + 1) * vocab * 4 < (4LL << 20)) return 0;
  // about 8 units of 16 bytes per thread of a part, at most two parts per SM
  const long long units = static_cast<long long>(gamma + 1) * ((vocab + 3) / 4);
  const long long by_work = units / (8LL * kAcceptThreads);
  const long long by_sms = 2LL * num_sms / Bt;  // one wave of two CTAs per SM
  const long long parts = std::min(by_work, by_sms);
  return parts > kMaxCluster ? static_cast<int>(parts) : 0;
}

size_t accept_workspace_bytes(int Bt, int gamma, int vocab, int num_sms) {
  const int parts = accept_parts(Bt, gamma, vocab, num_sms);
  return parts ? static_cast<size_t>(Bt) * parts * (gamma + 1) * sizeof(unsigned long long) : 0;
}

cudaError_t launch_accept_parts(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab,
                                int32_t* accepted_len, int32_t* out_tokens, int32_t* row_argmax, void* workspace,
                                int32_t* err_word, int num_sms, cudaStream_t stream) {
  const int parts = accept_parts(Bt, gamma, vocab, num_sms);
  const int vec4 = (vocab % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15u) == 0);
  auto* keys = static_cast<unsigned long long*>(workspace);
  cudaError_t e = launch_overlapped(accept_part_kernel, dim3(static_cast<unsigned>(Bt) * parts), dim3(kAcceptThreads),
                                    0, stream, 1u, logits, gamma, vocab, vec4, parts, keys);
  if (e != cudaSuccess) return e;
  return launch_overlapped(accept_merge_kernel, dim3(static_cast<unsigned>(Bt)), dim3(kMergeThreads), 0, stream, 1u,
                           static_cast<const unsigned long long*>(keys), parts, draft, gamma, vocab, accepted_len,
                           out_tokens, row_argmax, err_word);
}

cudaError_t launch_accept(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab,
                          int32_t* accepted_len, int32_t* out_tokens, int32_t* row_argmax, int32_t* err_word,
                          int num_sms, cudaStream_t stream, const WaitFault& fault) {
  const unsigned long long wait_ns = fault.wait_ns ? fault.wait_ns : kWaitLimitNs;
  const int vec4 = (vocab % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15u) == 0);
  const ClusterCapacity* cap = nullptr;
  // few sequences: the largest clusters still leave SMs idle, so each CTA
  // keeps twice as many loads in flight
  if (Bt * kMaxCluster <= num_sms) {
    cudaError_t e = cluster_capacity<16>(&cap);
    if (e != cudaSuccess) return e;
    if (cap->resident[kMaxCluster] >= Bt) {
      if (fault.extra) return cudaErrorNotSupported;
      return launch_overlapped(accept_kernel<16>, dim3(static_cast<unsigned>(Bt) * kMaxCluster),
                               dim3(kAcceptThreads), 0, stream, static_cast<unsigned>(kMaxCluster), logits, draft,
                               gamma, vocab, vec4, accepted_len, out_tokens, row_argmax, err_word, 0u, wait_ns);
    }
  }
  cudaError_t e = cluster_capacity<8>(&cap);
  if (e != cudaSuccess) return e;
  // the largest cluster for which one cluster per sequence still fits in a
  // single wave: more CTAs keep more loads in flight
  int CL = 1;
  for (int cl = kMaxCluster; cl >= 1; --cl) {
    if (cap->resident[cl] >= Bt) {
      CL = cl;
      break;
    }
  }
  if (fault.extra && CL > 1) return cudaErrorNotSupported;
  return launch_overlapped(accept_kernel<8>, dim3(static_cast<unsigned>(Bt) * CL), dim3(kAcceptThreads), 0, stream,
                           static_cast<unsigned>(CL), logits, draft, gamma, vocab, vec4, accepted_len, out_tokens,
                           row_argmax, err_word, fault.extra, wait_ns);
}

}  // namespace simsd
