// commit.cu -- append the accepted drafts' K/V to the paged cache (Sec. 3.2:
// the accepted prefix is committed to the block; Sec. 3.3: later steps reuse
// the cached K/V).  Row r < a_b of sequence b takes the data-slot K/V whose
// temporal label is r+1 and lands in cache row n_b + r.  When the new keys
// are not rotated yet, each committed key is rotated at its slot's RoPE
// position (Sec. 3.1) so that the cache holds rotated keys.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace simsd {

constexpr int kCommitWarps = 8;

// rotation of committed keys (null pos: the keys are rotated already)
struct CommitRope {
  const int32_t* pos;  // [Bt][2*gamma] or null
  RopeTable table;
};

// One thread-block cluster per sequence.  Every thread reads n_b and a_b and
// arrives on the cluster barrier; the cluster's warps then share the
// sequence's accepted rows.  Without RoPE a warp copies one (layer, accepted
// row) at a time: the KV heads of that row are adjacent in K_new/V_new, and
// each lane keeps several 16-byte chunks in flight.  With RoPE a warp
// rotates one (layer, accepted row, KV head) row at a time.  After every
// thread of the cluster has arrived, thread 0 of CTA 0 writes n_b + a_b (no
// thread reads n_b after that).
__global__ void __launch_bounds__(kCommitWarps * 32) kv_commit_kernel(
    const uint8_t* __restrict__ k_new, const uint8_t* __restrict__ v_new, int L, const int32_t* __restrict__ tau,
    const uint8_t* __restrict__ section, const int32_t* __restrict__ accepted_len, uint8_t* __restrict__ k_cache,
    uint8_t* __restrict__ v_cache, int num_pages, const int32_t* __restrict__ block_table, int max_pages,
    int page_size, int32_t* __restrict__ prefix_len, int gamma, int Hkv, int row_bytes, int elem_bytes,
    const __grid_constant__ CommitRope rope, int32_t* err_word) {
  pdl_wait();
  pdl_launch_next();
  cg::cluster_group cluster = cg::this_cluster();
  const int CL = static_cast<int>(cluster.num_blocks());
  const int rank = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.x / CL;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int S = 2 * gamma;
  const int a = accepted_len[b];
  const int n = prefix_len[b];
  // the labels of the data slots (lane k: slot k) do not depend on a or n:
  // their loads go out together with those two
  const bool lane_data = lane < gamma && section[static_cast<size_t>(b) * S + lane] == kSectData;
  const int lane_tau = lane < gamma ? tau[static_cast<size_t>(b) * S + lane] : 0;
  const int32_t* bt = block_table + static_cast<size_t>(b) * max_pages;
  // page ids of a 32-page window (lane i: page win + i) that holds every
  // destination row n_b .. n_b + a_b - 1 (a_b <= 32): the first 32 pages,
  // loaded beside n_b and a_b, or, when the rows lie beyond them, the 32
  // pages from the first destination page.  With no layer there is no row
  // to place, and the caller may pass no block table at all.
  int win = 0;
  int lane_pg = (L > 0 && lane < max_pages) ? bt[lane] : -1;
  // "n_b has been read"
  asm volatile("barrier.cluster.arrive.release;" ::: "memory");
  const bool ok = a >= 0 && a <= gamma && n >= 0;
  if (ok && a > 0 && L > 0) {
    const int last_page = (n + a - 1) / page_size;
    if (last_page >= 32) {
      win = n / page_size;
      lane_pg = win + lane < max_pages ? bt[win + lane] : -1;
    }
    const size_t Bt = gridDim.x / CL;
    const int chunks = row_bytes >> 4;  // 16-byte chunks of one KV head's row
    const int rows = rope.pos ? a * L * Hkv : a * L;
    for (int row = rank * kCommitWarps + warp; row < rows; row += CL * kCommitWarps) {
      const int kvh = rope.pos ? row % Hkv : 0;
      const int q = rope.pos ? row / Hkv : row;  // (layer, accepted row)
      const int r = q % a, l = q / a;
      // source: the data slot whose label is r+1
      const bool hit = lane_data && lane_tau == r + 1;
      const unsigned m = __ballot_sync(0xffffffffu, hit);
      if (!m) {
        if (lane == 0) raise_error(err_word, SIMSD_EW_STEP_MAP);
        continue;
      }
      const int src = __ffs(m) - 1;
      const int dst_row = n + r;
      const int pidx = dst_row / page_size;
      if (pidx >= max_pages) {
        if (lane == 0) raise_error(err_word, SIMSD_EW_PAGE);
        continue;
      }
      const int pg = __shfl_sync(0xffffffffu, lane_pg, pidx - win);
      if (pg < 0 || pg >= num_pages) {
        if (lane == 0) raise_error(err_word, SIMSD_EW_PAGE);
        continue;
      }
      const int off = dst_row - pidx * page_size;
      // row indices (in rows of row_bytes): K_new/V_new [L][Bt][S][Hkv],
      // the pools [L][num_pages][Hkv][page_size]
      const size_t s_row = ((static_cast<size_t>(l) * Bt + b) * S + src) * Hkv + kvh;
      const size_t d_row = ((static_cast<size_t>(l) * num_pages + pg) * Hkv + kvh) * page_size + off;
      const uint4* ks = reinterpret_cast<const uint4*>(k_new + s_row * row_bytes);
      const uint4* vs = reinterpret_cast<const uint4*>(v_new + s_row * row_bytes);
      uint4* kd = reinterpret_cast<uint4*>(k_cache + d_row * row_bytes);
      uint4* vd = reinterpret_cast<uint4*>(v_cache + d_row * row_bytes);
      if (rope.pos) {
        const int pos = rope.pos[static_cast<size_t>(b) * S + src];
        const int d = row_bytes / elem_bytes, half = d / 2;
        for (int i = lane; i < half; i += 32) {
          float sn, cs;
          rope_sincos(pos, rope.table.f[i], &sn, &cs);
          if (elem_bytes == 4) {
            const float* kf = reinterpret_cast<const float*>(ks);
            float* kdf = reinterpret_cast<float*>(kd);
            float x = kf[i], y = kf[i + half];
            rope_pair(x, y, sn, cs);
            kdf[i] = x;
            kdf[i + half] = y;
          } else {
            const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(ks);
            __nv_bfloat16* kdb = reinterpret_cast<__nv_bfloat16*>(kd);
            float x = __bfloat162float(kb[i]), y = __bfloat162float(kb[i + half]);
            rope_pair(x, y, sn, cs);
            kdb[i] = __float2bfloat16_rn(x);
            kdb[i + half] = __float2bfloat16_rn(y);
          }
        }
        for (int c = lane; c < chunks; c += 32) vd[c] = vs[c];
      } else {
        // every KV head of the row: chunk c of the Hkv * chunks source
        // chunks (contiguous) lands in head c / chunks, page_size rows apart
        const int total = Hkv * chunks;
        const size_t head_step = static_cast<size_t>(page_size) * chunks;
        for (int c0 = 0; c0 < total; c0 += 128) {
          uint4 kx[4], vx[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int c = c0 + 32 * j + lane;
            if (c < total) {
              kx[j] = ks[c];
              vx[j] = vs[c];
            }
          }
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int c = c0 + 32 * j + lane;
            if (c < total) {
              const int h = c / chunks;
              const size_t dc = h * head_step + (c - h * chunks);
              kd[dc] = kx[j];
              vd[dc] = vx[j];
            }
          }
        }
      }
    }
  }
  // every thread of the cluster has read n_b once this returns
  asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
  if (rank == 0 && threadIdx.x == 0) {
    if (a < 0 || a > gamma)
      raise_error(err_word, SIMSD_EW_ACCEPT_LEN);
    else if (n < 0)
      raise_error(err_word, SIMSD_EW_PREFIX_LEN);
    else
      prefix_len[b] = n + a;
  }
}

cudaError_t launch_kv_commit(int elem_bytes, const void* k_new, const void* v_new, int L, const int32_t* tau,
                             const uint8_t* section, const int32_t* accepted_len, void* k_cache, void* v_cache,
                             int num_pages, const int32_t* block_table, int max_pages, int page_size,
                             int32_t* prefix_len, int Bt, int gamma, int Hkv, int d, const int32_t* rope_pos,
                             const RopeTable& rope_table, int32_t* err_word, cudaStream_t stream) {
  // about two CTAs per SM in all, at most 8 per sequence (a power of two)
  int CL = 8;
  while (CL > 1 && static_cast<long long>(Bt) * CL > 320) CL >>= 1;
  return launch_overlapped(kv_commit_kernel, dim3(static_cast<unsigned>(Bt) * CL), dim3(kCommitWarps * 32), 0, stream,
                           static_cast<unsigned>(CL), static_cast<const uint8_t*>(k_new),
                           static_cast<const uint8_t*>(v_new), L, tau, section, accepted_len,
                           static_cast<uint8_t*>(k_cache), static_cast<uint8_t*>(v_cache), num_pages, block_table,
                           max_pages, page_size, prefix_len, gamma, Hkv, d * elem_bytes, elem_bytes,
                           CommitRope{rope_pos, rope_table}, err_word);
}

}  // namespace simsd
