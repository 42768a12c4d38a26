// attention_tc.cu -- bf16 verification attention on the sm_103a tensor cores
// (Sec. 3.2 "Target Model Verification", Sec. 3.3 KV cache; the extra cost
// of the paired layout is linear in the prefix, Eqs. (4)-(5)).
//
// Work unit: (sequence b, KV head, row block, prefix split).  The query rows
// of one unit are the g = Hq/Hkv heads x 2*gamma slots that share the KV
// head ("GQA packing"), up to 128 rows, so QK^T and PV are M = 128 MMAs.
// Keys stream in tiles of 64: first one tile with the 2*gamma new slots, whose
// Eq. (1) visibility is evaluated on the fly from (section, tau), then the
// cached prefix pages (read through the page table with TMA).  When the
// inputs are not rotated yet (Sec. 3.1 RoPE copy), the softmax warps rotate
// Q while moving it into TMEM and rotate the new keys in shared memory before
// the first S is computed; cached keys are stored rotated.
//
// Two CTAs share each SM (96 KB of shared memory, 256 TMEM columns and 192
// threads apiece), so one CTA's set-up, first loads and epilogue overlap the
// other's streaming, and the two rings together keep the same bytes in
// flight as one large ring.
//
// Warp roles (192 threads):
//   warps 0-3  softmax; thread i owns query row i (TMEM lane i).  They first
//              move the Q tile from shared memory into TMEM, then per key
//              tile read S, update the running max / sum, write P (bf16)
//              over the first half of S and hand it to the MMA issuer.
//   warp 4     TMA producer (one thread): Q, then K/V tiles into a 3-deep
//              ring of 32 KB slots (Q uses the first slot once).
//   warp 5     MMA issuer (one thread) and TMEM owner.  Per tile:
//              S = Q K^T (TS MMA: Q in TMEM, K in shared memory) and, once P
//              is written, O += P V (TS MMA: P in TMEM, V MN-major in shared
//              memory).  The next S overwrites P, so it waits for that PV.
// TMEM (256 columns): Q [0,64) as bf16 pairs, S [64,128) fp32 with P in its
// first 32 columns, O [128,256) fp32.
//
// Every mbarrier wait is bounded; a wait that expires sets SIMSD_EW_TIMEOUT
// and makes the whole CTA stop, drain its async work and free its TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cooperative_groups.h>
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

namespace cg = cooperative_groups;

namespace simsd {
namespace {

constexpr int kTile = 64;            // keys per tile
constexpr int kD = 128;              // head dimension
constexpr int kRows = 128;           // MMA M (query rows per CTA)
constexpr int kStages = 3;           // ring slots of one CTA
constexpr int kThreads = 192;
constexpr int kCtasPerSm = 2;        // shared-memory budget of one CTA
// Registers per thread: at most 128, so that two CTAs fit one SM by the
// per-scheduler register file (each CTA's warps 0, 1, 4, 5 share two of the
// four schedulers).  With more, the block scheduler counts one CTA per SM: a
// launch still starts two per SM, but a freed slot is refilled only once its
// SM is empty, which left SMs idle for tens of microseconds on ragged
// prefixes.
constexpr int kMaxRegs = 128;
constexpr int kWarpProducer = 4;
constexpr int kWarpMma = 5;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColQ = 0, kColS = 64, kColO = 128;
constexpr int kHalfBytes = kTile * 128;     // 64 rows x 64 bf16 (one d-half of K or V)
// Split merge in place (fused): per-row partials in the ring, padded rows
constexpr int kMaxSplitFuse = 8;            // cluster of at most 8 splits
constexpr int kPartStride = kD + 4;         // floats per partial row (no bank conflicts)
constexpr int kPartMl = kRows * kPartStride;              // (m, l) per row
constexpr int kPartWts = kPartMl + 2 * kRows;             // merge weights [row][split]
constexpr int kSlotBytes = 4 * kHalfBytes;  // K0 K1 V0 V1, or Q0 Q1 (16 KB each)
constexpr int kPageCache = 512;             // page ids of one sequence kept in shared memory
constexpr float kRescaleThreshold = 8.0f;   // log2 units: rescale when the max grows by > 2^8

struct TcParams {
  const int32_t* block_table;
  const int32_t* prefix_len;
  const int32_t* tau;
  const uint8_t* section;
  const int32_t* rope_pos;  // [Bt][2*gamma] or null (inputs rotated already)
  __nv_bfloat16* out;
  float* ws;  // partials: O [units*nsplit][rows_blk][128] then (m, l) [units*nsplit][rows_blk][2]
  int32_t* err_word;
  int max_pages, page_size, num_pages;
  int Bt, gamma, S, Hq, Hkv, g, rb, rows_blk, s_blk, nsplit;
  int sort;  // order sequences longest prefix first (grids of more than one wave)
  int slots;  // CTAs resident at once: blocks past this start in a later wave
  int fuse;   // the prefix splits of a unit form a cluster and merge in shared memory
  float scale_log2;
  // bounded waits: time limit and extra arrivals expected on bar_p (0 in
  // normal use; a test arms one launch so that a wait runs out)
  unsigned long long wait_ns;
  uint32_t extra_p;
  RopeTable rope;
};

struct alignas(1024) Smem {
  uint8_t ring[kStages][kSlotBytes];
  uint64_t bar_k[kStages], bar_v[kStages], bar_empty[kStages];
  uint64_t bar_qt, bar_s_full, bar_p, bar_pv, bar_drain;
  uint32_t tmem_base;
  int abort_flag;
  int seq_bad;
  int b_sel, n_sel;
  int32_t tau[64];
  uint8_t sect[64];
  int32_t pages[kPageCache];
};

constexpr size_t smem_bytes() { return sizeof(Smem) + 1024; }
static_assert(kCtasPerSm * (smem_bytes() + 1024) <= 233472, "two CTAs per SM");
static_assert((kPartWts + (kRows / 2) * kMaxSplitFuse) * sizeof(float) <= sizeof(Smem::ring),
              "the fused split merge fits in the ring");

__device__ __forceinline__ void signal_abort(Smem& sm, int32_t* err_word) {
  raise_error(err_word, SIMSD_EW_TIMEOUT);
  *reinterpret_cast<volatile int*>(&sm.abort_flag) = 1;
}

// Row r of a 128-byte-swizzled tile: 16-byte chunk c sits at chunk c ^ (r & 7).
__device__ __forceinline__ uint4 ld_sw128_chunk(const uint8_t* half, int r, int c) {
  return *reinterpret_cast<const uint4*>(half + r * 128 + ((c ^ (r & 7)) << 4));
}

// kFuse: the prefix splits of a unit form a cluster and merge their partials
// in shared memory (a separate instantiation, so that the unclustered kernel
// carries no cluster barriers).
template <bool kFuse>
__global__ void __maxnreg__(kMaxRegs)
    attention_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kn,
                        const __grid_constant__ CUtensorMap tm_vn, const __grid_constant__ CUtensorMap tm_kc,
                        const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  volatile int* abort_flag = &sm.abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // ---- which unit this CTA computes; sequences go longest prefix first.
  // Merged in place, the splits of a unit are adjacent (one cluster);
  // otherwise the splits of a sequence follow one another.
  const int per_seq = p.nsplit * p.Hkv * p.rb;
  const int rank = blockIdx.x / per_seq;
  int rem = blockIdx.x - rank * per_seq;
  int split;
  if (kFuse) {
    split = rem % p.nsplit;
    rem /= p.nsplit;
  } else {
    split = rem / (p.Hkv * p.rb);
    rem -= split * p.Hkv * p.rb;
  }
  const int kvh = rem / p.rb;
  const int rblk = rem - kvh * p.rb;

  if (tid == 0) {
    sm.abort_flag = 0;
    sm.seq_bad = 0;
    sm.b_sel = rank;
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&sm.bar_k[s]), 1);
      mbar_init(smem_u32(&sm.bar_v[s]), 1);
      mbar_init(smem_u32(&sm.bar_empty[s]), 1);
    }
    mbar_init(smem_u32(&sm.bar_qt), 1);
    mbar_init(smem_u32(&sm.bar_s_full), 1);
    mbar_init(smem_u32(&sm.bar_p), 4 + p.extra_p);
    mbar_init(smem_u32(&sm.bar_pv), 1);
    mbar_init(smem_u32(&sm.bar_drain), 1);
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpProducer && lane == 0) {
    // the tensor maps are kernel parameters, not results of earlier work
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kn);
    tma_prefetch_desc(&tm_vn);
    tma_prefetch_desc(&tm_kc);
    tma_prefetch_desc(&tm_vc);
  }
  // the set-up above touches no global memory; from here on the previous
  // kernel's results are needed
  pdl_wait();
  // A CTA of a later wave lets the next kernel in at once: the next grid can
  // then fill the slots this grid's last wave leaves idle (consecutive
  // layers).  First-wave CTAs let it in after their tile loop (below), so
  // that in a single-wave grid no waiting CTA of the next kernel sits beside
  // this one for its whole run (that cost up to 30 us with 32 sequences of
  // 4096-token prefixes).
  if (static_cast<int>(blockIdx.x) >= p.slots) pdl_launch_next();
  // the barriers and flags set by thread 0 above must be in place before the
  // producer (another warp) issues its first load on them
  __syncthreads();
  // When the grid takes more than one wave, the sequences go longest prefix
  // first: the prefix lengths are staged in the (still unused) ring and
  // ranked.  In a single wave every CTA is resident at once and the order
  // does not matter, so the CTA reads its own sequence's length only.
  int b, n = 0;
  if (p.sort) {
    int32_t* nval = reinterpret_cast<int32_t*>(sm.ring[0]);
    for (int i = tid; i < p.Bt; i += kThreads) nval[i] = p.prefix_len[i];
    __syncthreads();
    for (int i = tid; i < p.Bt; i += kThreads) {
      const int ni = nval[i];
      int r = 0;
      for (int j = 0; j < p.Bt; ++j) {
        const int nj = nval[j];
        r += (nj > ni) || (nj == ni && j < i);
      }
      if (r == rank) {
        sm.b_sel = i;
        sm.n_sel = ni;
      }
    }
    // the staging area is overwritten by TMA later
    fence_proxy_async_smem();
    __syncthreads();
    b = sm.b_sel;
    n = sm.n_sel;
  } else {
    b = rank;
  }
  const int32_t* bt = p.block_table + static_cast<size_t>(b) * p.max_pages;

  // ---- TMA issue of ring items (producer thread only): item 0 is Q, item
  // i + 1 is the i-th key tile of this unit (tile 0: new slots, 1..T: prefix)
  auto issue_q = [&]() {
    const uint32_t q_bytes = 2u * static_cast<uint32_t>(p.g * p.s_blk) * 128u;
    const int qz = b * p.S + rblk * p.s_blk;
    const uint32_t q0 = smem_u32(sm.ring[0]);
    mbar_arrive_expect_tx(smem_u32(&sm.bar_k[0]), q_bytes);
    tma_load_3d(q0, &tm_q, smem_u32(&sm.bar_k[0]), 0, kvh * p.g, qz);
    tma_load_3d(q0 + 2 * kHalfBytes, &tm_q, smem_u32(&sm.bar_k[0]), 64, kvh * p.g, qz);
    mbar_arrive(smem_u32(&sm.bar_v[0]));  // keeps the two barriers of slot 0 in step
  };
  auto issue_tile = [&](int it, int t) {
    const int P = p.page_size;
    const int st = it % kStages;
    const uint32_t bk = smem_u32(&sm.bar_k[st]), bv = smem_u32(&sm.bar_v[st]);
    const uint32_t k0 = smem_u32(sm.ring[st]), k1 = k0 + kHalfBytes;
    const uint32_t v0 = k0 + 2 * kHalfBytes, v1 = k0 + 3 * kHalfBytes;
    if (t > 0) {
      const int key0 = (t - 1) * kTile;
      const int valid = min(kTile, n - key0);
      if (P >= kTile) {
        const int pi = key0 / P;
        const int pg = pi < kPageCache ? sm.pages[pi] : bt[pi];
        const int row = (pg * p.Hkv + kvh) * P + (key0 % P);
        mbar_arrive_expect_tx(bk, 2u * kHalfBytes);
        tma_load_2d(k0, &tm_kc, bk, 0, row);
        tma_load_2d(k1, &tm_kc, bk, 64, row);
        mbar_arrive_expect_tx(bv, 2u * kHalfBytes);
        tma_load_2d(v0, &tm_vc, bv, 0, row);
        tma_load_2d(v1, &tm_vc, bv, 64, row);
      } else {
        const int nsub = (valid + P - 1) / P;
        const uint32_t sub_bytes = static_cast<uint32_t>(P) * 128u;
        mbar_arrive_expect_tx(bk, 2u * nsub * sub_bytes);
        for (int sb = 0; sb < nsub; ++sb) {
          const int pi = (key0 + sb * P) / P;
          const int pg = pi < kPageCache ? sm.pages[pi] : bt[pi];
          const int row = (pg * p.Hkv + kvh) * P;
          tma_load_2d(k0 + sb * sub_bytes, &tm_kc, bk, 0, row);
          tma_load_2d(k1 + sb * sub_bytes, &tm_kc, bk, 64, row);
        }
        mbar_arrive_expect_tx(bv, 2u * nsub * sub_bytes);
        for (int sb = 0; sb < nsub; ++sb) {
          const int pi = (key0 + sb * P) / P;
          const int pg = pi < kPageCache ? sm.pages[pi] : bt[pi];
          const int row = (pg * p.Hkv + kvh) * P;
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
  };
  // Q, and in split 0 the tile of new slots, need neither the prefix length
  // nor a page id: they go out first.  If the sequence turns out to be
  // invalid they are drained unused.
  int early = 0;
  if (warp == kWarpProducer && lane == 0) {
    issue_q();
    early = 1;
    if (split == 0) {
      issue_tile(1, 0);
      early = 2;
    }
  }
  // The prefix length, the sequence's page ids (up to the page cache) and
  // its slot labels are read together: one memory latency instead of a
  // chain.  Page ids past the prefix are loaded but not used.
  if (!p.sort) n = p.prefix_len[b];
  constexpr int kPgRegs = (kPageCache + kThreads - 1) / kThreads;
  int pg_reg[kPgRegs];
  const int pg_lim = min(p.max_pages, kPageCache);
#pragma unroll
  for (int j = 0; j < kPgRegs; ++j) {
    const int i = tid + j * kThreads;
    pg_reg[j] = i < pg_lim ? bt[i] : -1;
  }
  for (int i = tid; i < p.S; i += kThreads) {
    sm.tau[i] = p.tau[static_cast<size_t>(b) * p.S + i];
    sm.sect[i] = p.section[static_cast<size_t>(b) * p.S + i];
  }
  const bool n_bad = n < 0 || static_cast<long long>(n) > static_cast<long long>(p.max_pages) * p.page_size;
  if (n_bad) {
    if (tid == 0) {
      sm.seq_bad = 1;
      raise_error(p.err_word, SIMSD_EW_PREFIX_LEN);
    }
  } else {
    const int npages = (n + p.page_size - 1) / p.page_size;
#pragma unroll
    for (int j = 0; j < kPgRegs; ++j) {
      const int i = tid + j * kThreads;
      if (i < npages && i < kPageCache) {
        const int pg = pg_reg[j];
        sm.pages[i] = pg;
        if (pg < 0 || pg >= p.num_pages) {
          sm.seq_bad = 1;
          raise_error(p.err_word, SIMSD_EW_PAGE);
        }
      }
    }
    for (int i = kPageCache + tid; i < npages; i += kThreads) {
      const int pg = bt[i];
      if (pg < 0 || pg >= p.num_pages) {
        sm.seq_bad = 1;
        raise_error(p.err_word, SIMSD_EW_PAGE);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  const bool seq_bad = sm.seq_bad != 0;
  const int T = seq_bad ? 0 : (n + kTile - 1) / kTile;  // prefix tiles
  const int T_all = seq_bad ? 0 : T + 1;                 // tile 0: new slots, tiles 1..T: prefix
  // Split 0 always holds tile 0 (issued above).  Split i takes tiles
  // [ceil(i T_all / nsplit), ceil((i + 1) T_all / nsplit)); merged in a
  // cluster, where the slowest split sets the pace, split 0 instead holds
  // tile 0, the costliest (the Eq. (1) mask, zeroed V rows), plus tiles up
  // to floor(T_all / nsplit) in all, and splits 1.. share the rest evenly,
  // so the extra tiles of an uneven split go to splits without tile 0.
  int t0, t1;
  if (kFuse) {
    const int first = T_all == 0 ? 0 : max(1, T_all / p.nsplit);
    t0 = 0;
    t1 = first;
    if (split > 0) {
      const long long rest = T_all - first, ns1 = p.nsplit - 1;
      t0 = first + static_cast<int>(((split - 1) * rest + ns1 - 1) / ns1);
      t1 = first + static_cast<int>((split * rest + ns1 - 1) / ns1);
    }
  } else {
    t0 = static_cast<int>((static_cast<long long>(split) * T_all + p.nsplit - 1) / p.nsplit);
    t1 = static_cast<int>((static_cast<long long>(split + 1) * T_all + p.nsplit - 1) / p.nsplit);
  }
  const int ntiles = t1 - t0;

  // fused split merge: what the softmax thread of this row hands over
  bool fz_any = false, fz_have = false;
  float fz_m = -INFINITY, fz_l = 0.f;

  if (warp == kWarpProducer) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int issued = early;
      if (ntiles > 0) {
        // Q (and in split 0 the tile of new slots) went out already
        for (int i = issued - 1; i < ntiles; ++i) {
          const int it = i + 1, st = it % kStages;
          if (it >= kStages &&
              !mbar_wait(smem_u32(&sm.bar_empty[st]), ((it / kStages) - 1) & 1, abort_flag, p.wait_ns)) {
            signal_abort(sm, p.err_word);
            break;
          }
          issue_tile(it, t0 + i);
          ++issued;
        }
      }
      // Drain: every issued load must have landed before the CTA may exit.
      // In a normal run these phases completed long ago.  These waits keep
      // the full limit even when a test shortens the others.
      for (int it = max(0, issued - kStages); it < issued; ++it) {
        const int st = it % kStages;
        mbar_wait(smem_u32(&sm.bar_k[st]), (it / kStages) & 1, nullptr);
        mbar_wait(smem_u32(&sm.bar_v[st]), (it / kStages) & 1, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // ----------------------------------------------------------- MMA issuer
    if (lane == 0 && ntiles > 0) {
      constexpr uint32_t kIdescQK = idesc_bf16_f32(kRows, kTile, 0, 0);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(kRows, kD, 0, 1);
      bool ok = mbar_wait(smem_u32(&sm.bar_qt), 0, abort_flag, p.wait_ns);
      for (int i = 0; ok && i < ntiles; ++i) {
        const int it = i + 1, st = it % kStages;
        const uint32_t par = (it / kStages) & 1;
        // S overwrites P of the previous tile; tcgen05.mma ops issued by one
        // thread run in issue order, so that PV has read P before this S lands
        if (!mbar_wait(smem_u32(&sm.bar_k[st]), par, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t kb0 = smem_u32(sm.ring[st]), kb1 = kb0 + kHalfBytes;
#pragma unroll
        for (int kk = 0; kk < kD / 16; ++kk) {
          const uint32_t ka = (kk < 4 ? kb0 : kb1) + (kk & 3) * 32;
          tc_mma_ts(tmem + kColS, tmem + kColQ + 8 * kk, sdesc_sw128(ka, 16, 1024), kIdescQK, kk > 0);
        }
        tc_commit(smem_u32(&sm.bar_s_full));
        if (!mbar_wait(smem_u32(&sm.bar_p), i & 1, abort_flag, p.wait_ns) ||
            !mbar_wait(smem_u32(&sm.bar_v[st]), par, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t vb = kb0 + 2 * kHalfBytes;
#pragma unroll
        for (int kk = 0; kk < kTile / 16; ++kk) {
          tc_mma_ts(tmem + kColO, tmem + kColS + 8 * kk, sdesc_sw128(vb + kk * 2048, kHalfBytes, 1024),
                    kIdescPV, (i > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(smem_u32(&sm.bar_empty[st]));
        tc_commit(smem_u32(&sm.bar_pv));
      }
      if (!ok) signal_abort(sm, p.err_word);
      // every MMA issued by this thread has completed once this fires
      tc_commit(smem_u32(&sm.bar_drain));
      mbar_wait(smem_u32(&sm.bar_drain), 0, nullptr);
    }
    __syncwarp();
  } else {
    // -------------------------------------------------------------- softmax
    const int row = tid;                       // TMEM lane / query row
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
    const uint32_t lane_tmem = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    float m_ref = -INFINITY, l_sum = 0.f;
    bool ok = true;

    // ---- Q: shared memory (ring slot 0) -> TMEM columns [0, 64)
    if (ntiles > 0) {
      const int pos = p.rope_pos ? p.rope_pos[static_cast<size_t>(b) * p.S + (s < p.S ? s : 0)] : 0;
      ok = mbar_wait_warp(smem_u32(&sm.bar_k[0]), 0, abort_flag, p.wait_ns);
      if (ok && p.rope_pos) {
        // rotate this row's query at its slot's position on the way
        const uint8_t* h0 = sm.ring[0];
        const uint8_t* h1 = sm.ring[0] + 2 * kHalfBytes;
        uint32_t q0r[32], q1r[32];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 va = ld_sw128_chunk(h0, row, c), vb = ld_sw128_chunk(h1, row, c);
          const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            float x0 = __uint_as_float(wa[w] << 16), x1 = __uint_as_float(wa[w] & 0xffff0000u);
            float y0 = __uint_as_float(wb[w] << 16), y1 = __uint_as_float(wb[w] & 0xffff0000u);
            float sn, cs;
            rope_sincos(pos, p.rope.f[8 * c + 2 * w], &sn, &cs);
            rope_pair(x0, y0, sn, cs);
            rope_sincos(pos, p.rope.f[8 * c + 2 * w + 1], &sn, &cs);
            rope_pair(x1, y1, sn, cs);
            q0r[4 * c + w] = pack_bf16x2(x0, x1);
            q1r[4 * c + w] = pack_bf16x2(y0, y1);
          }
        }
        tmem_st32(lane_tmem + kColQ, q0r);
        tmem_st32(lane_tmem + kColQ + 32, q1r);
        tmem_wait_st();
      } else if (ok) {
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const uint8_t* half = sm.ring[0] + h * 2 * kHalfBytes;
          uint32_t qr[32];
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 v = ld_sw128_chunk(half, row, c);
            qr[4 * c] = v.x;
            qr[4 * c + 1] = v.y;
            qr[4 * c + 2] = v.z;
            qr[4 * c + 3] = v.w;
          }
          tmem_st32(lane_tmem + kColQ + 32 * h, qr);
        }
        tmem_wait_st();
      }
      if (ok && p.rope_pos && t0 == 0) {
        // the new keys (ring item 1, the unit's first tile) are rotated in
        // place before the first S = Q K^T reads them
        constexpr int st1 = 1 % kStages;
        ok = mbar_wait_warp(smem_u32(&sm.bar_k[st1]), 0, abort_flag, p.wait_ns);
        if (ok) {
          uint8_t* h0 = sm.ring[st1];
          uint8_t* h1 = sm.ring[st1] + kHalfBytes;
          for (int task = tid; task < p.S * 8; task += 128) {
            const int r = task >> 3, c = task & 7;
            const int pos = p.rope_pos[static_cast<size_t>(b) * p.S + r];
            uint4* pa = reinterpret_cast<uint4*>(h0 + r * 128 + ((c ^ (r & 7)) << 4));
            uint4* pb = reinterpret_cast<uint4*>(h1 + r * 128 + ((c ^ (r & 7)) << 4));
            const uint4 va = *pa, vb = *pb;
            uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
            for (int w = 0; w < 4; ++w) {
              float x0 = __uint_as_float(wa[w] << 16), x1 = __uint_as_float(wa[w] & 0xffff0000u);
              float y0 = __uint_as_float(wb[w] << 16), y1 = __uint_as_float(wb[w] & 0xffff0000u);
              float sn, cs;
              rope_sincos(pos, p.rope.f[8 * c + 2 * w], &sn, &cs);
              rope_pair(x0, y0, sn, cs);
              rope_sincos(pos, p.rope.f[8 * c + 2 * w + 1], &sn, &cs);
              rope_pair(x1, y1, sn, cs);
              wa[w] = pack_bf16x2(x0, x1);
              wb[w] = pack_bf16x2(y0, y1);
            }
            *pa = make_uint4(wa[0], wa[1], wa[2], wa[3]);
            *pb = make_uint4(wb[0], wb[1], wb[2], wb[3]);
          }
          fence_proxy_async_smem();
        }
      }
      tc_fence_before();
      asm volatile("bar.sync 1, 128;" ::: "memory");
      if (tid == 0 && ok && !*abort_flag) {
        mbar_arrive(smem_u32(&sm.bar_qt));
        mbar_arrive(smem_u32(&sm.bar_empty[0]));
      }
    }

    for (int i = 0; ok && i < ntiles; ++i) {
      const int it = i + 1, st = it % kStages;
      const int t = t0 + i;
      if (!mbar_wait_warp(smem_u32(&sm.bar_s_full), i & 1, abort_flag, p.wait_ns)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sa[32], sb[32];
      tmem_ld32(lane_tmem + kColS, sa);
      tmem_ld32(lane_tmem + kColS + 32, sb);
      tmem_wait_ld();

      const bool is_new = (t == 0);
      const int valid = is_new ? p.S : min(kTile, n - (t - 1) * kTile);
      float x[kTile];
#pragma unroll
      for (int c = 0; c < kTile; ++c) x[c] = __uint_as_float(c < 32 ? sa[c] : sb[c - 32]);
      if (is_new || valid < kTile) {
        // partial prefix tile or the tile of new slots: hide what the row may
        // not see.  One bit word per row and a select per column: the rows of
        // a warp see different new slots, so a per-column branch would
        // diverge (it cost microseconds on the first tile).
        const unsigned long long keep = is_new ? vis : (valid >= kTile ? ~0ull : ((1ull << valid) - 1ull));
        const uint32_t klo = static_cast<uint32_t>(keep), khi = static_cast<uint32_t>(keep >> 32);
#pragma unroll
        for (int c = 0; c < kTile; ++c) {
          const uint32_t bit = ((c < 32 ? klo : khi) >> (c & 31)) & 1u;
          x[c] = bit ? x[c] : -INFINITY;
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
        // O holds the earlier tiles; their PVs completed before this S was
        // computed (the S MMA waited for the last one)
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
      tmem_st32(lane_tmem + kColS, pk);
      tmem_wait_st();
      if (warp < 2 && (valid < kTile || is_new)) {
        // rows of V that no query may use are zeroed so that 0 * (stale or
        // non-finite data) cannot reach O
        if (!mbar_wait_warp(smem_u32(&sm.bar_v[st]), (it / kStages) & 1, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        const int kr = row;
        const bool zero = kr >= valid || (is_new && sm.sect[kr] == kSectPad);
        if (zero) {
          const uint4 z = make_uint4(0u, 0u, 0u, 0u);
          uint4* r0 = reinterpret_cast<uint4*>(sm.ring[st] + 2 * kHalfBytes + kr * 128);
          uint4* r1 = reinterpret_cast<uint4*>(sm.ring[st] + 3 * kHalfBytes + kr * 128);
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
      if (lane == 0) mbar_arrive(smem_u32(&sm.bar_p));
    }
    if (!ok && lane == 0) signal_abort(sm, p.err_word);
    // the next kernel on the stream may be scheduled now (its CTAs wait for
    // this grid to finish anyway).  A clustered grid lets it in only when
    // its CTAs exit: next-kernel CTAs placed beside clusters still merging
    // cost more than they gain (measured at 8 sequences, 4 splits each).
    if (!kFuse) pdl_launch_next();
    // ---- epilogue: O of the last PV, scaled by 1/l
    const bool have_o =
        ok && ntiles > 0 && mbar_wait_warp(smem_u32(&sm.bar_pv), (ntiles - 1) & 1, abort_flag, p.wait_ns);
    if (have_o) tc_fence_after();
    const bool any = have_o && active && l_sum > 0.f;
    const int h = kvh * p.g + hl;
    if (kFuse) {
      // written to the ring after the whole CTA is done with it (below)
      fz_any = any;
      fz_have = have_o;
      fz_m = m_ref;
      fz_l = l_sum;
    } else if (p.nsplit == 1) {
      const float inv = any ? 1.0f / l_sum : 0.f;
      __nv_bfloat16* orow = p.out + ((static_cast<size_t>(b) * p.S + s) * p.Hq + h) * kD;
#pragma unroll 1
      for (int ch = 0; ch < kD / 32; ++ch) {
        uint32_t o[32];
        if (have_o) {
          tmem_ld32(lane_tmem + kColO + 32 * ch, o);
          tmem_wait_ld();
        }
        if (row_exists) {
          uint4 pkd[4];
          uint32_t* wv = reinterpret_cast<uint32_t*>(pkd);
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const float r0 = any ? __uint_as_float(o[2 * c]) * inv : 0.f;
            const float r1 = any ? __uint_as_float(o[2 * c + 1]) * inv : 0.f;
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
          float4* dst = reinterpret_cast<float4*>(wo + 32 * ch);
#pragma unroll
          for (int c = 0; c < 8; ++c)
            dst[c] = any ? make_float4(__uint_as_float(o[4 * c]), __uint_as_float(o[4 * c + 1]),
                                       __uint_as_float(o[4 * c + 2]), __uint_as_float(o[4 * c + 3]))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      if (row < p.rows_blk) {
        wml[0] = any ? m_ref : -INFINITY;
        wml[1] = any ? l_sum : 0.f;
      }
    }
  }

  if (kFuse) {
    // Merge of the splits of this unit, O = sum_i 2^(m_i - M) O_i / sum_i
    // 2^(m_i - M) l_i: CTA c of the cluster takes rows c, c + nsplit, ...,
    // reading every split's partials through distributed shared memory.
    // First this CTA's partial O (unnormalised) and (m, l) of each row go
    // into the ring, once every load and MMA of the CTA has completed.
    cg::cluster_group cluster = cg::this_cluster();
    float* part = reinterpret_cast<float*>(sm.ring[0]);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp < 4) {
      const int row = tid;
      const uint32_t lane_tmem = tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll 1
      for (int ch = 0; ch < kD / 32; ++ch) {
        uint32_t o[32];
        if (fz_have) {
          tmem_ld32(lane_tmem + kColO + 32 * ch, o);
          tmem_wait_ld();
        }
        if (row < p.rows_blk) {
          float4* dst = reinterpret_cast<float4*>(part + row * kPartStride + 32 * ch);
#pragma unroll
          for (int c = 0; c < 8; ++c)
            dst[c] = fz_any ? make_float4(__uint_as_float(o[4 * c]), __uint_as_float(o[4 * c + 1]),
                                          __uint_as_float(o[4 * c + 2]), __uint_as_float(o[4 * c + 3]))
                            : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      if (row < p.rows_blk) {
        part[kPartMl + 2 * row] = fz_any ? fz_m : -INFINITY;
        part[kPartMl + 2 * row + 1] = fz_any ? fz_l : 0.f;
      }
    }
    cluster.sync();  // every split's partials are in place
    if (warp < 4) {
      // Every remote load of a step is issued before its first use, so one
      // round trip through distributed shared memory serves all splits.
      const int nsp = p.nsplit;
      float* wts = part + kPartWts;  // [row of this CTA][split]
      const int nrows = (p.rows_blk - split + nsp - 1) / nsp;
      for (int k = tid; k < nrows; k += 128) {
        const int r = split + k * nsp;
        float2 ml[kMaxSplitFuse];
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i)
          ml[i] = i < nsp ? *reinterpret_cast<const float2*>(cluster.map_shared_rank(part, i) + kPartMl + 2 * r)
                          : make_float2(-INFINITY, 0.f);
        float M = -INFINITY;
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i)
          if (ml[i].y > 0.f) M = fmaxf(M, ml[i].x);
        float w[kMaxSplitFuse], L = 0.f;
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i) {
          w[i] = (M != -INFINITY && ml[i].y > 0.f) ? exp2f(ml[i].x - M) : 0.f;
          L = fmaf(w[i], ml[i].y, L);
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i) wts[k * kMaxSplitFuse + i] = w[i] * inv;
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      constexpr int kVec = kD / 4;
      for (int e = tid; e < nrows * kVec; e += 128) {
        const int k = e / kVec, c4 = e - k * kVec;
        const int r = split + k * nsp;
        float4 x[kMaxSplitFuse];
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i)
          if (i < nsp) x[i] = *reinterpret_cast<const float4*>(cluster.map_shared_rank(part, i) + r * kPartStride + 4 * c4);
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int i = 0; i < kMaxSplitFuse; ++i) {
          if (i < nsp) {
            const float wi = wts[k * kMaxSplitFuse + i];
            v.x = fmaf(wi, x[i].x, v.x);
            v.y = fmaf(wi, x[i].y, v.y);
            v.z = fmaf(wi, x[i].z, v.z);
            v.w = fmaf(wi, x[i].w, v.w);
          }
        }
        const int sr = rblk * p.s_blk + r / p.g;
        if (sr < p.S) {
          const int hr = kvh * p.g + r % p.g;
          uint2 pk;
          pk.x = pack_bf16x2(v.x, v.y);
          pk.y = pack_bf16x2(v.z, v.w);
          *reinterpret_cast<uint2*>(p.out + ((static_cast<size_t>(b) * p.S + sr) * p.Hq + hr) * kD + 4 * c4) = pk;
        }
      }
    }
    cluster.sync();  // no CTA leaves while a peer may still read its partials
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merges the prefix splits of every (sequence, KV head, row block):
// O = sum_i 2^(m_i - M) O_i / sum_i 2^(m_i - M) l_i.  One warp per row; the
// lanes take the splits' (m, l) in parallel, then sum the partial O rows with
// lanes over the head dimension (independent loads, several in flight).
// kBatch: splits whose partials a lane loads before adding any (see
// launch_combine for the choice)
template <int kBatch>
__global__ void __launch_bounds__(128) combine_kernel(const __grid_constant__ TcParams p) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const unsigned full = 0xffffffffu;
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
  const size_t e0 = static_cast<size_t>(u) * p.nsplit;
  float M = -INFINITY;
  for (int i = lane; i < p.nsplit; i += 32) {
    const size_t e = (e0 + i) * p.rows_blk + row;
    if (wml[2 * e + 1] > 0.f) M = fmaxf(M, wml[2 * e]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(full, M, o));
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float L = 0.f;
  if (M != -INFINITY) {
    for (int c0 = 0; c0 < p.nsplit; c0 += 32) {
      // lane j holds the weight of split c0 + j
      float wj = 0.f;
      if (c0 + lane < p.nsplit) {
        const size_t e = (e0 + c0 + lane) * p.rows_blk + row;
        const float lj = wml[2 * e + 1];
        if (lj > 0.f) {
          wj = exp2f(wml[2 * e] - M);
          L = fmaf(wj, lj, L);
        }
      }
      const int cnt = min(32, p.nsplit - c0);
      // the partials of kBatch splits are loaded before any is added (one
      // round trip per batch; the sum keeps the split order)
      const float4* ob = reinterpret_cast<const float4*>(p.ws + ((e0 + c0) * p.rows_blk + row) * kD) + lane;
      const size_t split4 = static_cast<size_t>(p.rows_blk) * (kD / 4);  // float4s from one split to the next
      for (int j0 = 0; j0 < cnt; j0 += kBatch) {
        float4 o[kBatch];
#pragma unroll
        for (int j = 0; j < kBatch; ++j)
          o[j] = j0 + j < cnt ? ob[(j0 + j) * split4] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < kBatch; ++j) {
          if (j0 + j < cnt) {  // (the same for the whole warp)
            const float w = __shfl_sync(full, wj, j0 + j);
            acc.x = fmaf(w, o[j].x, acc.x);
            acc.y = fmaf(w, o[j].y, acc.y);
            acc.z = fmaf(w, o[j].z, acc.z);
            acc.w = fmaf(w, o[j].w, acc.w);
          }
        }
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(full, L, o);
  const float inv = L > 0.f ? 1.f / L : 0.f;
  __nv_bfloat16* orow = p.out + ((static_cast<size_t>(b) * p.S + s) * p.Hq + h) * kD;
  uint2 v;
  v.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  v.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  reinterpret_cast<uint2*>(orow)[lane] = v;
  // the next kernel is let in only as this grid's blocks finish: launched
  // at the start, its CTAs took SMs that thousands of these small blocks
  // still needed
  pdl_launch_next();
}

// The kernels' shared-memory attributes, set once per device (function
// attributes apply to the current device only).
cudaError_t ensure_smem_attr() {
  static std::mutex mu;
  static bool done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(mu);
  if (done[dev]) return cudaSuccess;
  for (auto kern : {attention_tc_kernel<false>, attention_tc_kernel<true>}) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem_bytes()));
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
  }
  done[dev] = true;
  return cudaSuccess;
}

bool make_map(EncodeTiledFn encode, CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims,
              const cuuint64_t* strides, const cuuint32_t* box) {
  return make_bf16_map(encode, m, base, rank, dims, strides, box);
}

}  // namespace

bool make_bf16_map(EncodeTiledFn encode, CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims,
                   const cuuint64_t* strides, const cuuint32_t* box) {
  cuuint32_t es[3] = {1, 1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool plan_attention_tc(int Bt, int gamma, int Hq, int Hkv, int max_pages, int page_size, int num_sms,
                       AttnTcPlan* plan, bool allow_streamk) {
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
  pl.num_sms = num_sms;
  const long long max_tiles = (static_cast<long long>(max_pages) * page_size + kTile - 1) / kTile + 1;
  if (const int ns256 = tc256_splits(Bt, Hkv, pl.rb, max_tiles, num_sms)) {
    // two row blocks share one CTA and its K/V stream; with fewer units
    // than SMs each unit's key tiles are split into ranges whose partials
    // the combine kernel merges
    pl.kind = 1;
    pl.streamk = allow_streamk ? tc256_streamk(Bt, Hkv, max_tiles, ns256, num_sms) : 0;
    pl.nsplit = pl.streamk ? 1 : ns256;
    pl.sort = 0;
    pl.fuse = 0;
    pl.slots = num_sms;
    pl.ws_bytes = pl.streamk ? tc256_streamk_bytes(num_sms)
                  : pl.nsplit > 1
                      ? static_cast<size_t>(Bt) * Hkv * pl.rb * pl.nsplit * pl.rows_blk * (kD + 2) * sizeof(float)
                      : 0;
    *plan = pl;
    return true;
  }
  // split the prefix only when the units alone cannot fill the GPU (the
  // occupancy calculator reports one CTA per SM for this kernel although two
  // are resident, so the budget the kernel is built for is used instead)
  const long long units = static_cast<long long>(Bt) * Hkv * pl.rb;
  const long long slots = static_cast<long long>(num_sms) * kCtasPerSm;
  int ns = 1;
  if (units < slots) {
    // as many splits as keep every CTA in one wave
    ns = static_cast<int>(std::max<long long>(1, slots / units));
    ns = static_cast<int>(std::min<long long>(ns, std::max<long long>(1, max_tiles / 2)));
    ns = std::min(ns, 64);
  }
  pl.nsplit = ns;
  pl.sort = (units * ns > slots && Bt <= 256) ? 1 : 0;
  // up to 8 splits merge in place (a cluster per unit), more through the
  // workspace and combine_kernel
  pl.fuse = (ns >= 2 && ns <= kMaxSplitFuse) ? 1 : 0;
  pl.slots = static_cast<int>(slots);
  pl.ws_bytes = (ns > 1 && !pl.fuse) ? static_cast<size_t>(units) * ns * pl.rows_blk * (kD + 2) * sizeof(float) : 0;
  *plan = pl;
  return true;
}

// The combine launch, a warp per row.  With many splits a row (a small
// batch) a lane loads 16 splits' partials at once: 128 registers, four
// blocks per SM, which pays while the grid fits in one wave of those.
// Otherwise four at a time (about 56 registers): a large grid merging a
// few splits a row needs its blocks resident more than wide loads.
cudaError_t launch_combine(const TcParams& p, long long warps, int num_sms, cudaStream_t stream) {
  const long long blocks = (warps + 3) / 4;
  const bool wide = p.nsplit > 4 && blocks <= 4LL * num_sms;
  return wide ? launch_overlapped(combine_kernel<16>, dim3(static_cast<unsigned>(blocks)), dim3(128), 0, stream, 1, p)
              : launch_overlapped(combine_kernel<4>, dim3(static_cast<unsigned>(blocks)), dim3(128), 0, stream, 1, p);
}

cudaError_t launch_attention_combine(const AttnTcArgs& a, const AttnTcPlan& pl, cudaStream_t stream) {
  TcParams p{};
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ws = static_cast<float*>(a.workspace);
  p.Bt = a.Bt;
  p.gamma = a.gamma;
  p.S = 2 * a.gamma;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.g = a.Hq / a.Hkv;
  p.rb = pl.rb;
  p.rows_blk = pl.rows_blk;
  p.s_blk = pl.s_blk;
  p.nsplit = pl.nsplit;
  const long long warps = static_cast<long long>(a.Bt) * a.Hkv * pl.rb * pl.rows_blk;
  return launch_combine(p, warps, pl.num_sms, stream);
}

cudaError_t launch_attention_tc(const AttnTcArgs& a, const AttnTcPlan& pl, EncodeTiledFn encode,
                                cudaStream_t stream) {
  if (pl.kind == 1) return launch_attention_tc256(a, pl, encode, stream);
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
  p.rope_pos = a.rope_pos;
  p.rope = a.rope;
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
  p.sort = pl.sort;
  p.fuse = pl.fuse;
  p.slots = pl.slots;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.wait_ns = a.fault.wait_ns ? a.fault.wait_ns : kWaitLimitNs;
  p.extra_p = a.fault.extra;

  {
    cudaError_t e = ensure_smem_attr();
    if (e != cudaSuccess) return e;
  }
  const long long grid = static_cast<long long>(a.Bt) * pl.nsplit * a.Hkv * pl.rb;
  cudaError_t e = pl.fuse ? launch_overlapped(attention_tc_kernel<true>, dim3(static_cast<unsigned>(grid)),
                                               dim3(kThreads), smem_bytes(), stream,
                                               static_cast<unsigned>(pl.nsplit), tq, tkn, tvn, tkc, tvc, p)
                          : launch_overlapped(attention_tc_kernel<false>, dim3(static_cast<unsigned>(grid)),
                                              dim3(kThreads), smem_bytes(), stream, 1u, tq, tkn, tvn, tkc, tvc, p);
  if (e != cudaSuccess || pl.nsplit == 1 || pl.fuse) return e;
  const long long warps = static_cast<long long>(a.Bt) * a.Hkv * pl.rb * pl.rows_blk;
  return launch_combine(p, warps, pl.num_sms, stream);
}

size_t noalloc_scratch_capacity() { return sizeof(g_noalloc_scratch); }

cudaError_t noalloc_scratch_pointer(void** out) {
  // Set-up, once per device and with that device current: the device
  // address of the static scratch array.  It is kept for the life of the
  // process (a device reset, which would move the array, is not supported).
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
