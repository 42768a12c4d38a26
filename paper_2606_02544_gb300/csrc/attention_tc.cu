// attention_tc.cu -- bf16 verification attention on the sm_103a tensor cores
// (Sec. 3.2 "Target Model Verification", Sec. 3.3 KV cache; the extra cost
// of the paired layout is linear in the prefix, Eqs. (4)-(5)).
//
// Work unit: (sequence b, KV head, row block, prefix split).  The query rows
// of one unit are the g = Hq/Hkv heads x 2*gamma slots that share the KV
// head ("GQA packing"), up to 128 rows, so QK^T and PV are M = 128 MMAs.
// Keys stream in tiles of 64: first the cached prefix pages (read through
// the page table with TMA), then one tile with the 2*gamma new slots, whose
// Eq. (1) visibility is evaluated on the fly from (section, tau).
//
// Warp roles (320 threads):
//   warps 0-3, 4-7  two softmax warpgroups.  Group w takes the unit's tiles
//              w, w+2, w+4, ... with its own S, P and O in TMEM and its own
//              running max / sum; thread i of a group owns query row i (TMEM
//              lane i).  Two groups keep two tiles in flight through the
//              softmax, so the shared-memory ring recycles twice as fast.
//              At the end group 1 hands its (m, l, O) rows to group 0 through
//              shared memory and group 0 writes the merged result.
//   warp 8     TMA producer (one thread): Q once, then K/V tiles into a
//              STAGES-deep shared-memory ring.
//   warp 9     MMA issuer (one thread) and TMEM owner.  It polls both
//              groups and issues whatever is ready: S_i = Q K_i^T (SS MMA,
//              128x64x128) or O_w += P_i V_i (TS MMA, P in TMEM, V MN-major in
//              shared memory, 128x128x64).
// TMEM (512 columns): group w owns [256w, 256w+256): S [0,64) fp32, P in two
// buffers [64,96) and [96,128) (bf16 pairs), O [128,256) fp32.
//
// Every mbarrier wait is bounded; a wait that expires sets SIMSD_EW_TIMEOUT
// and makes the whole CTA stop, drain its async work and free its TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

// Scratch of simsd_verify_attention_noalloc: the split partials live in this
// file-scope array instead of caller memory.  Every device that loads the
// library holds it until the process exits.  Host code must not use the
// symbol's address directly (on the host it is only a stand-in); it asks
// the runtime for the device address once per device (below).
static __device__ __align__(256) unsigned char g_noalloc_scratch[12u << 20];

namespace simsd {
namespace {

constexpr int kTile = 64;            // keys per tile
constexpr int kD = 128;              // head dimension
constexpr int kRows = 128;           // MMA M (query rows per CTA)
constexpr int kGroups = 2;           // softmax warpgroups
constexpr int kThreads = 32 * (4 * kGroups + 2);
constexpr int kWarpProducer = 4 * kGroups;
constexpr int kWarpMma = 4 * kGroups + 1;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kGroupCols = 256;
constexpr uint32_t kColS = 0, kColP = 64, kColO = 128;
constexpr int kQHalfBytes = kRows * 128;    // 128 rows x 64 bf16
constexpr int kKvHalfBytes = kTile * 128;   // 64 rows x 64 bf16
constexpr float kRescaleThreshold = 8.0f;   // log2 units: rescale when the max grows by > 2^8

struct TcParams {
  const int32_t* block_table;
  const int32_t* prefix_len;
  const int32_t* tau;
  const uint8_t* section;
  __nv_bfloat16* out;
  float* ws;  // partials: O [units*nsplit][rows_blk][128] then (m, l) [units*nsplit][rows_blk][2]
  int32_t* err_word;
  int max_pages, page_size, num_pages;
  int Bt, gamma, S, Hq, Hkv, g, rb, rows_blk, s_blk, nsplit;
  float scale_log2;
};

template <int STAGES>
struct alignas(1024) Smem {
  uint8_t q[2][kQHalfBytes];                // [d half][row][64]
  uint8_t kv[STAGES][4][kKvHalfBytes];      // [stage][K0, K1, V0, V1][key][64]
  uint64_t bar_q;
  uint64_t bar_k[STAGES], bar_v[STAGES], bar_empty[STAGES];
  uint64_t bar_s_full[kGroups], bar_s_free[kGroups], bar_p[kGroups][2], bar_o[kGroups];
  uint64_t bar_ofinal, bar_drain;
  uint32_t tmem_base;
  int abort_flag;
  int seq_bad;
  int b_sel;
  int32_t tau[64];
  uint8_t sect[64];
};

template <int STAGES>
constexpr size_t smem_bytes() {
  return sizeof(Smem<STAGES>) + 1024;
}
static_assert(smem_bytes<6>() <= 232448, "shared memory budget of one CTA");

template <int STAGES>
__device__ __forceinline__ void signal_abort(Smem<STAGES>& sm, int32_t* err_word) {
  raise_error(err_word, SIMSD_EW_TIMEOUT);
  *reinterpret_cast<volatile int*>(&sm.abort_flag) = 1;
}

template <int STAGES>
__global__ void __launch_bounds__(kThreads, 1)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kn,
                        const __grid_constant__ CUtensorMap tm_vn, const __grid_constant__ CUtensorMap tm_kc,
                        const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem<STAGES>& sm =
      *reinterpret_cast<Smem<STAGES>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  volatile int* abort_flag = &sm.abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // ---- which unit this CTA computes; sequences go longest prefix first
  const int per_seq = p.nsplit * p.Hkv * p.rb;
  const int rank = blockIdx.x / per_seq;
  int rem = blockIdx.x - rank * per_seq;
  const int split = rem / (p.Hkv * p.rb);
  rem -= split * p.Hkv * p.rb;
  const int kvh = rem / p.rb;
  const int rblk = rem - kvh * p.rb;

  if (tid == 0) {
    sm.abort_flag = 0;
    sm.seq_bad = 0;
    sm.b_sel = rank;
  }
  // prefix lengths, staged in the (still unused) K/V ring for the ranking
  int32_t* nval = reinterpret_cast<int32_t*>(sm.kv[0][0]);
  const bool sort = p.Bt <= 256;
  if (sort)
    for (int i = tid; i < p.Bt; i += kThreads) nval[i] = p.prefix_len[i];
  __syncthreads();
  if (sort) {
    for (int i = tid; i < p.Bt; i += kThreads) {
      const int ni = nval[i];
      int r = 0;
      for (int j = 0; j < p.Bt; ++j) {
        const int nj = nval[j];
        r += (nj > ni) || (nj == ni && j < i);
      }
      if (r == rank) sm.b_sel = i;
    }
  }
  __syncthreads();
  const int b = sm.b_sel;
  const int n = p.prefix_len[b];
  const bool n_bad = n < 0 || static_cast<long long>(n) > static_cast<long long>(p.max_pages) * p.page_size;
  if (n_bad) {
    if (tid == 0) {
      sm.seq_bad = 1;
      raise_error(p.err_word, SIMSD_EW_PREFIX_LEN);
    }
  } else {
    const int npages = (n + p.page_size - 1) / p.page_size;
    for (int i = tid; i < npages; i += kThreads) {
      const int pg = p.block_table[static_cast<size_t>(b) * p.max_pages + i];
      if (pg < 0 || pg >= p.num_pages) {
        sm.seq_bad = 1;
        raise_error(p.err_word, SIMSD_EW_PAGE);
      }
    }
  }
  for (int i = tid; i < p.S; i += kThreads) {
    sm.tau[i] = p.tau[static_cast<size_t>(b) * p.S + i];
    sm.sect[i] = p.section[static_cast<size_t>(b) * p.S + i];
  }
  if (tid == 0) {
    mbar_init(smem_u32(&sm.bar_q), 1);
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&sm.bar_k[s]), 1);
      mbar_init(smem_u32(&sm.bar_v[s]), 1);
      mbar_init(smem_u32(&sm.bar_empty[s]), 1);
    }
    for (int w = 0; w < kGroups; ++w) {
      mbar_init(smem_u32(&sm.bar_s_full[w]), 1);
      mbar_init(smem_u32(&sm.bar_s_free[w]), 4);
      mbar_init(smem_u32(&sm.bar_p[w][0]), 4);
      mbar_init(smem_u32(&sm.bar_p[w][1]), 4);
      mbar_init(smem_u32(&sm.bar_o[w]), 1);
    }
    mbar_init(smem_u32(&sm.bar_ofinal), 1);
    mbar_init(smem_u32(&sm.bar_drain), 1);
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  const bool seq_bad = sm.seq_bad != 0;
  const int T = seq_bad ? 0 : (n + kTile - 1) / kTile;  // prefix tiles
  const int T_all = seq_bad ? 0 : T + 1;                 // + the tile of new slots
  const int t0 = static_cast<int>(static_cast<long long>(split) * T_all / p.nsplit);
  const int t1 = static_cast<int>(static_cast<long long>(split + 1) * T_all / p.nsplit);
  const int ntiles = t1 - t0;

  if (warp == kWarpProducer) {
    // ------------------------------------------------------------ producer
    if (lane == 0 && ntiles > 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_kc);
      tma_prefetch_desc(&tm_vc);
      const uint32_t q_bytes = 2u * static_cast<uint32_t>(p.g * p.s_blk) * 128u;
      mbar_arrive_expect_tx(smem_u32(&sm.bar_q), q_bytes);
      const int qz = b * p.S + rblk * p.s_blk;
      tma_load_3d(smem_u32(sm.q[0]), &tm_q, smem_u32(&sm.bar_q), 0, kvh * p.g, qz);
      tma_load_3d(smem_u32(sm.q[1]), &tm_q, smem_u32(&sm.bar_q), 64, kvh * p.g, qz);
      const int P = p.page_size;
      int issued = 0;
      for (int i = 0; i < ntiles; ++i) {
        const int t = t0 + i, st = i % STAGES;
        if (i >= STAGES && !mbar_wait(smem_u32(&sm.bar_empty[st]), ((i / STAGES) - 1) & 1, abort_flag)) {
          signal_abort(sm, p.err_word);
          break;
        }
        const uint32_t bk = smem_u32(&sm.bar_k[st]), bv = smem_u32(&sm.bar_v[st]);
        const uint32_t k0 = smem_u32(sm.kv[st][0]), k1 = smem_u32(sm.kv[st][1]);
        const uint32_t v0 = smem_u32(sm.kv[st][2]), v1 = smem_u32(sm.kv[st][3]);
        if (t < T) {
          const int key0 = t * kTile;
          const int valid = min(kTile, n - key0);
          const int32_t* bt = p.block_table + static_cast<size_t>(b) * p.max_pages;
          if (P >= kTile) {
            const int row = (bt[key0 / P] * p.Hkv + kvh) * P + (key0 % P);
            mbar_arrive_expect_tx(bk, 2u * kKvHalfBytes);
            tma_load_2d(k0, &tm_kc, bk, 0, row);
            tma_load_2d(k1, &tm_kc, bk, 64, row);
            mbar_arrive_expect_tx(bv, 2u * kKvHalfBytes);
            tma_load_2d(v0, &tm_vc, bv, 0, row);
            tma_load_2d(v1, &tm_vc, bv, 64, row);
          } else {
            const int nsub = (valid + P - 1) / P;
            const uint32_t sub_bytes = static_cast<uint32_t>(P) * 128u;
            mbar_arrive_expect_tx(bk, 2u * nsub * sub_bytes);
            for (int sb = 0; sb < nsub; ++sb) {
              const int row = (bt[(key0 + sb * P) / P] * p.Hkv + kvh) * P;
              tma_load_2d(k0 + sb * sub_bytes, &tm_kc, bk, 0, row);
              tma_load_2d(k1 + sb * sub_bytes, &tm_kc, bk, 64, row);
            }
            mbar_arrive_expect_tx(bv, 2u * nsub * sub_bytes);
            for (int sb = 0; sb < nsub; ++sb) {
              const int row = (bt[(key0 + sb * P) / P] * p.Hkv + kvh) * P;
              tma_load_2d(v0 + sb * sub_bytes, &tm_vc, bv, 0, row);
              tma_load_2d(v1 + sb * sub_bytes, &tm_vc, bv, 64, row);
            }
          }
        } else {
          const uint32_t new_bytes = static_cast<uint32_t>(p.S) * 128u;
          mbar_arrive_expect_tx(bk, 2u * new_bytes);
          tma_load_3d(k0, &tm_kn, bk, 0, kvh, b * p.S);
          tma_load_3d(k1, &tm_kn, bk, 64, kvh, b * p.S);
          mbar_arrive_expect_tx(bv, 2u * new_bytes);
          tma_load_3d(v0, &tm_vn, bv, 0, kvh, b * p.S);
          tma_load_3d(v1, &tm_vn, bv, 64, kvh, b * p.S);
        }
        ++issued;
      }
      // Drain: every issued load must have landed before the CTA may exit.
      // In a normal run these phases completed long ago.
      for (int i = max(0, issued - STAGES); i < issued; ++i) {
        const int st = i % STAGES;
        mbar_wait(smem_u32(&sm.bar_k[st]), (i / STAGES) & 1, nullptr);
        mbar_wait(smem_u32(&sm.bar_v[st]), (i / STAGES) & 1, nullptr);
      }
      mbar_wait(smem_u32(&sm.bar_q), 0, nullptr);
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // ----------------------------------------------------------- MMA issuer
    // Tile i belongs to group w = i & 1 as its j = i >> 1-th tile.
    //   QK_i needs K_i and S_w free (group w has read S of tile i-2), and,
    //   because P_w is double-buffered, PV_{i-4} already issued.
    //   PV_i needs P_i and V_i; PVs go in tile order.
    if (lane == 0 && ntiles > 0) {
      constexpr uint32_t kIdescQK = idesc_bf16_f32(kRows, kTile, 0, 0);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(kRows, kD, 0, 1);
      bool ok = mbar_wait(smem_u32(&sm.bar_q), 0, abort_flag);
      tc_fence_after();
      const uint32_t q0 = smem_u32(sm.q[0]), q1 = smem_u32(sm.q[1]);
      int next_qk = 0, next_pv = 0;
      unsigned long long t_idle = 0;
      uint32_t spins = 0;
      while (ok && next_pv < ntiles) {
        bool progressed = false;
        if (next_qk < ntiles && next_qk - 4 < next_pv) {
          const int i = next_qk, w = i & 1, j = i >> 1, st = i % STAGES;
          if (mbar_try_wait(smem_u32(&sm.bar_k[st]), (i / STAGES) & 1) &&
              (j == 0 || mbar_try_wait(smem_u32(&sm.bar_s_free[w]), (j - 1) & 1))) {
            tc_fence_after();
            const uint32_t kb0 = smem_u32(sm.kv[st][0]), kb1 = smem_u32(sm.kv[st][1]);
            const uint32_t d_s = tmem + w * kGroupCols + kColS;
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
              const uint32_t qa = (kk < 4 ? q0 : q1) + (kk & 3) * 32;
              const uint32_t ka = (kk < 4 ? kb0 : kb1) + (kk & 3) * 32;
              tc_mma_ss(d_s, sdesc_sw128(qa, 16, 1024), sdesc_sw128(ka, 16, 1024), kIdescQK, kk > 0);
            }
            tc_commit(smem_u32(&sm.bar_s_full[w]));
            ++next_qk;
            progressed = true;
          }
        }
        if (next_pv < next_qk) {
          const int i = next_pv, w = i & 1, j = i >> 1, st = i % STAGES;
          if (mbar_try_wait(smem_u32(&sm.bar_p[w][j & 1]), (j >> 1) & 1) &&
              mbar_try_wait(smem_u32(&sm.bar_v[st]), (i / STAGES) & 1)) {
            tc_fence_after();
            const uint32_t vb = smem_u32(sm.kv[st][2]);
            const uint32_t gbase = tmem + w * kGroupCols;
#pragma unroll
            for (int kk = 0; kk < kTile / 16; ++kk) {
              tc_mma_ts(gbase + kColO, gbase + kColP + 32 * (j & 1) + 8 * kk,
                        sdesc_sw128(vb + kk * 2048, kKvHalfBytes, 1024), kIdescPV, (j > 0 || kk > 0) ? 1u : 0u);
            }
            tc_commit(smem_u32(&sm.bar_empty[st]));
            tc_commit(smem_u32(&sm.bar_o[w]));
            ++next_pv;
            progressed = true;
          }
        }
        if (progressed) {
          spins = 0;
        } else if ((++spins & 63u) == 0) {
          const unsigned long long now = globaltimer_ns();
          if (spins == 64) t_idle = now;
          if (*abort_flag || now - t_idle > kWaitLimitNs) ok = false;
        }
      }
      if (!ok) signal_abort(sm, p.err_word);
      tc_commit(smem_u32(&sm.bar_ofinal));
      // every MMA issued by this thread has completed once this fires
      tc_commit(smem_u32(&sm.bar_drain));
      mbar_wait(smem_u32(&sm.bar_drain), 0, nullptr);
    }
    __syncwarp();
  } else {
    // -------------------------------------------------------------- softmax
    const int grp = warp >> 2;                 // 0 or 1
    const int row = tid & (kRows - 1);         // TMEM lane / query row
    const int wq = warp & 3;                   // lane quadrant of this warp
    const int s = rblk * p.s_blk + row / p.g;
    const int hl = row % p.g;
    const bool row_exists = row < p.rows_blk && s < p.S;
    const bool active = row_exists && !seq_bad && sm.sect[s] != kSectPad;
    unsigned long long vis = 0ull;
    if (active) {
      const uint8_t si = sm.sect[s];
      const int ti = sm.tau[s];
      for (int t = 0; t < p.S; ++t)
        if (temporal_visible(si, ti, sm.sect[t], sm.tau[t])) vis |= 1ull << t;
    }
    const uint32_t lane_tmem = tmem + grp * kGroupCols + (static_cast<uint32_t>(wq * 32) << 16);
    float m_ref = -INFINITY, l_sum = 0.f;
    bool ok = true;
    int j = 0;
    for (int i = grp; i < ntiles; i += kGroups, ++j) {
      const int t = t0 + i, st = i % STAGES;
      if (!mbar_wait_warp(smem_u32(&sm.bar_s_full[grp]), j & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sa[32], sb[32];
      tmem_ld32(lane_tmem + kColS, sa);
      tmem_ld32(lane_tmem + kColS + 32, sb);
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&sm.bar_s_free[grp]));

      const bool is_new = (t == T);
      const int valid = is_new ? p.S : min(kTile, n - t * kTile);
      float x[kTile];
#pragma unroll
      for (int c = 0; c < kTile; ++c) x[c] = __uint_as_float(c < 32 ? sa[c] : sb[c - 32]);
      if (is_new || valid < kTile) {
        // partial prefix tile or the tile of new slots: hide what the row may not see
#pragma unroll
        for (int c = 0; c < kTile; ++c) {
          const bool see = c < valid && (!is_new || ((vis >> c) & 1ull));
          x[c] = see ? x[c] : -INFINITY;
        }
      }
      // raw-score maximum (pairwise tree); scale_log2 > 0 commutes with max
      float mx;
      {
        float r[kTile / 2];
#pragma unroll
        for (int c = 0; c < kTile / 2; ++c) r[c] = fmaxf(x[2 * c], x[2 * c + 1]);
#pragma unroll
        for (int w2 = kTile / 4; w2 >= 1; w2 >>= 1)
#pragma unroll
          for (int c = 0; c < w2; ++c) r[c] = fmaxf(r[c], r[c + w2]);
        mx = active ? r[0] * p.scale_log2 : -INFINITY;
      }
      bool need = false;
      if (active && mx != -INFINITY) {
        if (m_ref == -INFINITY)
          m_ref = mx;
        else if (mx > m_ref + kRescaleThreshold)
          need = true;
      }
      if (__any_sync(0xffffffffu, need)) {
        // O_grp holds this group's earlier tiles: wait for the PV of its
        // previous tile, then rescale
        if (!mbar_wait_warp(smem_u32(&sm.bar_o[grp]), (j - 1) & 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const float f = need ? fast_exp2(m_ref - mx) : 1.0f;
        if (need) {
          l_sum *= f;
          m_ref = mx;
        }
#pragma unroll 1
        for (int ch = 0; ch < kD / 32; ++ch) {
          uint32_t o[32];
          tmem_ld32(lane_tmem + kColO + 32 * ch, o);
          tmem_wait_ld();
#pragma unroll
          for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * f);
          tmem_st32(lane_tmem + kColO + 32 * ch, o);
        }
        tmem_wait_st();
      }
      // p = 2^(s*scale*log2e - m): one FFMA and one MUFU.EX2 per score.  Rows
      // that are not active leave garbage in their own P/O rows only (MMA rows
      // are independent) and write zeros at the end.
      const float neg_m = (active && m_ref != -INFINITY) ? -m_ref : 0.f;
      uint32_t pk[32];
      float ps[kTile / 2];
#pragma unroll
      for (int c = 0; c < kTile / 2; ++c) {
        const float p0 = fast_exp2(fmaf(x[2 * c], p.scale_log2, neg_m));
        const float p1 = fast_exp2(fmaf(x[2 * c + 1], p.scale_log2, neg_m));
        ps[c] = p0 + p1;
        pk[c] = pack_bf16x2(p0, p1);
      }
#pragma unroll
      for (int w2 = kTile / 4; w2 >= 1; w2 >>= 1)
#pragma unroll
        for (int c = 0; c < w2; ++c) ps[c] += ps[c + w2];
      l_sum += ps[0];
      tmem_st32(lane_tmem + kColP + 32 * (j & 1), pk);
      tmem_wait_st();
      if (wq < 2 && (valid < kTile || is_new)) {
        // rows of V that no query may use are zeroed so that 0 * (stale or
        // non-finite data) cannot reach O
        if (!mbar_wait_warp(smem_u32(&sm.bar_v[st]), (i / STAGES) & 1, abort_flag)) {
          ok = false;
          break;
        }
        const int kr = row;
        const bool zero = kr >= valid || (is_new && sm.sect[kr] == kSectPad);
        if (zero) {
          const uint4 z = make_uint4(0u, 0u, 0u, 0u);
          uint4* r0 = reinterpret_cast<uint4*>(sm.kv[st][2] + kr * 128);
          uint4* r1 = reinterpret_cast<uint4*>(sm.kv[st][3] + kr * 128);
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            r0[c] = z;
            r1[c] = z;
          }
        }
        fence_proxy_async_smem();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&sm.bar_p[grp][j & 1]));
    }
    if (!ok && lane == 0) signal_abort(sm, p.err_word);
    // ---- epilogue: group 1 hands (m, l, O) to group 0, which merges
    const bool have_o = ok && ntiles > 0 && mbar_wait_warp(smem_u32(&sm.bar_ofinal), 0, abort_flag);
    if (have_o) tc_fence_after();
    const bool live = have_o && active && j > 0;   // this group saw at least one tile
    // the ring is idle once every MMA has completed: reuse it for the hand-off
    float* xo = reinterpret_cast<float*>(sm.kv[0][0]);          // [128 rows][132]
    constexpr int kXStride = kD + 4;
    if (grp == 1) {
#pragma unroll 1
      for (int ch = 0; ch < kD / 32; ++ch) {
        uint32_t o[32];
        if (have_o) {
          tmem_ld32(lane_tmem + kColO + 32 * ch, o);
          tmem_wait_ld();
        }
        float4* dst = reinterpret_cast<float4*>(xo + row * kXStride + 32 * ch);
#pragma unroll
        for (int c = 0; c < 8; ++c)
          dst[c] = live ? make_float4(__uint_as_float(o[4 * c]), __uint_as_float(o[4 * c + 1]),
                                      __uint_as_float(o[4 * c + 2]), __uint_as_float(o[4 * c + 3]))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
      }
      xo[row * kXStride + kD] = live ? m_ref : -INFINITY;
      xo[row * kXStride + kD + 1] = live ? l_sum : 0.f;
    }
    asm volatile("bar.sync 1, %0;" ::"r"(4 * kGroups * 32) : "memory");
    if (grp == 0) {
      // merge the two groups' partial softmax states of this row
      const float m1 = xo[row * kXStride + kD], l1 = xo[row * kXStride + kD + 1];
      const float m0 = live ? m_ref : -INFINITY, l0 = live ? l_sum : 0.f;
      const float M = fmaxf(m0, m1);
      const float a0 = (M == -INFINITY || m0 == -INFINITY) ? 0.f : fast_exp2(m0 - M);
      const float a1 = (M == -INFINITY || m1 == -INFINITY) ? 0.f : fast_exp2(m1 - M);
      const float L = a0 * l0 + a1 * l1;
      const bool any = active && have_o && L > 0.f;
      const int h = kvh * p.g + hl;
      if (p.nsplit == 1) {
        const float inv = any ? 1.0f / L : 0.f;
        __nv_bfloat16* orow = p.out + ((static_cast<size_t>(b) * p.S + s) * p.Hq + h) * kD;
#pragma unroll 1
        for (int ch = 0; ch < kD / 32; ++ch) {
          uint32_t o[32];
          if (have_o) {
            tmem_ld32(lane_tmem + kColO + 32 * ch, o);
            tmem_wait_ld();
          }
          if (row_exists) {
            const float* o1 = xo + row * kXStride + 32 * ch;
            uint4 pkd[4];
            uint32_t* wv = reinterpret_cast<uint32_t*>(pkd);
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              const float v0 = live ? __uint_as_float(o[2 * c]) : 0.f;
              const float v1 = live ? __uint_as_float(o[2 * c + 1]) : 0.f;
              const float r0 = any ? (a0 * v0 + a1 * o1[2 * c]) * inv : 0.f;
              const float r1 = any ? (a0 * v1 + a1 * o1[2 * c + 1]) * inv : 0.f;
              wv[c] = pack_bf16x2(r0, r1);
            }
            uint4* dst = reinterpret_cast<uint4*>(orow + 32 * ch);
#pragma unroll
            for (int c = 0; c < 4; ++c) dst[c] = pkd[c];
          }
        }
      } else {
        const size_t unit = ((static_cast<size_t>(b) * p.Hkv + kvh) * p.rb + rblk) * p.nsplit + split;
        const size_t nunits = static_cast<size_t>(p.Bt) * p.Hkv * p.rb * p.nsplit;
        float* wo = p.ws + (unit * p.rows_blk + row) * kD;
        float* wml = p.ws + nunits * p.rows_blk * kD + (unit * p.rows_blk + row) * 2;
#pragma unroll 1
        for (int ch = 0; ch < kD / 32; ++ch) {
          uint32_t o[32];
          if (have_o) {
            tmem_ld32(lane_tmem + kColO + 32 * ch, o);
            tmem_wait_ld();
          }
          if (row < p.rows_blk) {
            const float* o1 = xo + row * kXStride + 32 * ch;
            float4* dst = reinterpret_cast<float4*>(wo + 32 * ch);
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              float4 v;
              v.x = any ? a0 * (live ? __uint_as_float(o[4 * c]) : 0.f) + a1 * o1[4 * c] : 0.f;
              v.y = any ? a0 * (live ? __uint_as_float(o[4 * c + 1]) : 0.f) + a1 * o1[4 * c + 1] : 0.f;
              v.z = any ? a0 * (live ? __uint_as_float(o[4 * c + 2]) : 0.f) + a1 * o1[4 * c + 2] : 0.f;
              v.w = any ? a0 * (live ? __uint_as_float(o[4 * c + 3]) : 0.f) + a1 * o1[4 * c + 3] : 0.f;
              dst[c] = v;
            }
          }
        }
        if (row < p.rows_blk) {
          wml[0] = any ? M : -INFINITY;
          wml[1] = any ? L : 0.f;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merges the prefix splits of every (sequence, KV head, row block):
// O = sum_i 2^(m_i - M) O_i / sum_i 2^(m_i - M) l_i.  One warp per row.
__global__ void __launch_bounds__(128) combine_kernel(const TcParams p) {
  const int lane = threadIdx.x & 31;
  const long long wid = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long units = static_cast<long long>(p.Bt) * p.Hkv * p.rb;
  if (wid >= units * p.rows_blk) return;
  const int row = static_cast<int>(wid % p.rows_blk);
  const long long u = wid / p.rows_blk;
  const int rblk = static_cast<int>(u % p.rb);
  const int kvh = static_cast<int>((u / p.rb) % p.Hkv);
  const int b = static_cast<int>(u / (static_cast<long long>(p.rb) * p.Hkv));
  const int s = rblk * p.s_blk + row / p.g;
  if (s >= p.S) return;
  const int h = kvh * p.g + row % p.g;
  const size_t nunits = static_cast<size_t>(units) * p.nsplit;
  const float* wml = p.ws + nunits * p.rows_blk * kD;
  float M = -INFINITY;
  for (int i = 0; i < p.nsplit; ++i) {
    const size_t e = (static_cast<size_t>(u) * p.nsplit + i) * p.rows_blk + row;
    if (wml[2 * e + 1] > 0.f) M = fmaxf(M, wml[2 * e]);
  }
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float L = 0.f;
  if (M != -INFINITY) {
    for (int i = 0; i < p.nsplit; ++i) {
      const size_t e = (static_cast<size_t>(u) * p.nsplit + i) * p.rows_blk + row;
      const float li = wml[2 * e + 1];
      if (!(li > 0.f)) continue;
      const float w = exp2f(wml[2 * e] - M);
      L += w * li;
      const float4 o = reinterpret_cast<const float4*>(p.ws + e * kD)[lane];
      acc.x += w * o.x;
      acc.y += w * o.y;
      acc.z += w * o.z;
      acc.w += w * o.w;
    }
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  __nv_bfloat16* orow = p.out + ((static_cast<size_t>(b) * p.S + s) * p.Hq + h) * kD;
  uint2 v;
  v.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  v.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  reinterpret_cast<uint2*>(orow)[lane] = v;
}

constexpr int kStages = 6;

cudaError_t ensure_smem_attr() {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(attention_tc_kernel<kStages>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem_bytes<kStages>()));
  if (e == cudaSuccess) done = true;
  return e;
}

int occupancy_per_sm() {
  static int occ = -1;
  if (occ < 0) {
    int o = 0;
    ensure_smem_attr();
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, attention_tc_kernel<kStages>, kThreads,
                                                      smem_bytes<kStages>()) != cudaSuccess ||
        o < 1)
      o = 1;
    occ = o;
  }
  return occ;
}

bool make_map(EncodeTiledFn encode, CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims,
              const cuuint64_t* strides, const cuuint32_t* box) {
  cuuint32_t es[3] = {1, 1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool plan_attention_tc(int Bt, int gamma, int Hq, int Hkv, int max_pages, int page_size, int num_sms,
                       AttnTcPlan* plan) {
  const int S = 2 * gamma, g = Hq / Hkv;
  const int R = g * S;
  AttnTcPlan pl{};
  if (R <= kRows) {
    pl.rb = 1;
    pl.s_blk = S;
  } else {
    if (kRows % g != 0) return false;
    pl.s_blk = kRows / g;
    pl.rb = (S + pl.s_blk - 1) / pl.s_blk;
  }
  pl.rows_blk = g * pl.s_blk;
  if (pl.rows_blk > kRows || g > 256 || pl.s_blk > 256) return false;
  // split the prefix only when the units alone cannot fill the GPU
  const long long units = static_cast<long long>(Bt) * Hkv * pl.rb;
  const long long slots = static_cast<long long>(num_sms) * occupancy_per_sm();
  const long long max_tiles = (static_cast<long long>(max_pages) * page_size + kTile - 1) / kTile + 1;
  int ns = 1;
  if (units < slots) {
    // as many splits as keep every CTA in one wave
    ns = static_cast<int>(std::max<long long>(1, slots / units));
    ns = static_cast<int>(std::min<long long>(ns, std::max<long long>(1, max_tiles / 2)));
    ns = std::min(ns, 64);
  }
  pl.nsplit = ns;
  pl.ws_bytes = ns > 1 ? static_cast<size_t>(units) * ns * pl.rows_blk * (kD + 2) * sizeof(float) : 0;
  *plan = pl;
  return true;
}

cudaError_t launch_attention_tc(const AttnTcArgs& a, const AttnTcPlan& pl, EncodeTiledFn encode,
                                cudaStream_t stream) {
  const int S = 2 * a.gamma, g = a.Hq / a.Hkv;
  CUtensorMap tq, tkn, tvn, tkc, tvc;
  {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.Hq),
                                static_cast<cuuint64_t>(a.Bt) * S};
    const cuuint64_t strides[2] = {kD * 2ull, static_cast<cuuint64_t>(a.Hq) * kD * 2ull};
    const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(g), static_cast<cuuint32_t>(pl.s_blk)};
    if (!make_map(encode, &tq, a.q, 3, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.Hkv),
                                static_cast<cuuint64_t>(a.Bt) * S};
    const cuuint64_t strides[2] = {kD * 2ull, static_cast<cuuint64_t>(a.Hkv) * kD * 2ull};
    const cuuint32_t box[3] = {64u, 1u, static_cast<cuuint32_t>(S)};
    if (!make_map(encode, &tkn, a.k_new, 3, dims, strides, box)) return cudaErrorInvalidValue;
    if (!make_map(encode, &tvn, a.v_new, 3, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    // a pool without pages is described by a one-row map that is never read
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(kD),
                                std::max<cuuint64_t>(1, static_cast<cuuint64_t>(a.num_pages) * a.Hkv * a.page_size)};
    const cuuint64_t strides[1] = {kD * 2ull};
    const cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(std::min(a.page_size, kTile))};
    if (!make_map(encode, &tkc, a.k_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
    if (!make_map(encode, &tvc, a.v_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
  }
  TcParams p{};
  p.block_table = a.block_table;
  p.prefix_len = a.prefix_len;
  p.tau = a.tau;
  p.section = a.section;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ws = static_cast<float*>(a.workspace);
  p.err_word = a.err_word;
  p.max_pages = a.max_pages;
  p.page_size = a.page_size;
  p.num_pages = a.num_pages;
  p.Bt = a.Bt;
  p.gamma = a.gamma;
  p.S = S;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.g = g;
  p.rb = pl.rb;
  p.rows_blk = pl.rows_blk;
  p.s_blk = pl.s_blk;
  p.nsplit = pl.nsplit;
  p.scale_log2 = a.scale * 1.4426950408889634f;

  {
    cudaError_t e = ensure_smem_attr();
    if (e != cudaSuccess) return e;
  }
  const long long grid = static_cast<long long>(a.Bt) * pl.nsplit * a.Hkv * pl.rb;
  attention_tc_kernel<kStages><<<static_cast<unsigned>(grid), kThreads, smem_bytes<kStages>(), stream>>>(
      tq, tkn, tvn, tkc, tvc, p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || pl.nsplit == 1) return e;
  const long long warps = static_cast<long long>(a.Bt) * a.Hkv * pl.rb * pl.rows_blk;
  combine_kernel<<<static_cast<unsigned>((warps + 3) / 4), 128, 0, stream>>>(p);
  return cudaGetLastError();
}

size_t noalloc_scratch_capacity() { return sizeof(g_noalloc_scratch); }

cudaError_t noalloc_scratch_pointer(void** out) {
  // Set-up, once per device and with that device current: the device
  // address of the static scratch array.
  static std::mutex mu;
  static void* ptr[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  if (!ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    ptr[dev] = p;
  }
  *out = ptr[dev];
  return cudaSuccess;
}

}  // namespace simsd
