// attention_tc256.cu -- bf16 verification attention for units of 256 query
// rows on the sm_103a tensor cores (Sec. 3.2 "Target Model Verification",
// Sec. 3.3 KV cache; cost Eqs. (4)-(5)).
//
// A unit is (sequence b, KV head) when its g = Hq/Hkv heads x 2*gamma slots
// make two row blocks of 128 (32 drafts with g = 4, 16 with g = 8).  One CTA
// owns both row blocks, so every K/V tile crosses HBM and L2 once and feeds
// four MMAs: S_A = Q_A K^T, S_B = Q_B K^T, O_A += P_A V, O_B += P_B V.  At
// this intensity (about 256 flop per K/V byte, the ridge of the GPU) the
// tensor pipe must stay busy while the softmax runs, so S is double-buffered
// per row block: the MMAs of tile i+1 run while the softmax works on tile i.
//
// The kernel is persistent: one CTA per SM (512 TMEM columns, ~227 KB of
// shared memory) walks pieces of units.  Tensor memory, barriers and the
// K/V ring carry over from piece to piece; the producer loads the next
// piece's Q and tiles while the softmax warps finish the previous one.  Two
// walks:
//   ranges: units (or, with fewer units than SMs, equal key-tile ranges of
//     every unit) blockIdx.x, blockIdx.x + gridDim.x, ... in
//     longest-prefix-first order;
//   stream-K: the key tiles of all units, end to end, cut into gridDim.x
//     runs of equal length; a CTA takes the pieces of the units its run
//     overlaps.  Every SM then streams the same number of tiles, where whole
//     units would leave some SMs with one unit more than others (256 units
//     on 152 SMs: 104 take two, 48 one).  A unit cut by run boundaries
//     leaves partial results that streamk_combine_kernel merges.
//
// Warp roles (512 threads):
//   warps 0-3  softmax of row block A, warps 4-7 of row block B; thread i of
//              a block owns query row i (TMEM lane i).  Per tile: read S,
//              update the running max / sum, write P (bf16) over the first
//              half of its S buffer, hand it to the MMA issuer.  Per unit:
//              O / l to the output.
//   warp 8     TMA producer of Q (both blocks, into a region of its own, per
//              unit) and of the K half of every tile; warp 11 of the V
//              half.  The ring has 5 slots of 32 KB whose halves are
//              refilled apart: K is free once the tile's S MMAs are done, a
//              softmax before V.  Each producer's lanes hold a window of 32
//              page ids.
//   warps 9, 10, 12, 13  MMA issuers, one thread each: S of row block A, S
//              of B, PV of A, PV of B (a thread that issues a tcgen05.mma
//              is held about as long as the MMA runs, so a thread serving
//              two of these streams delays one behind the other); warp 9
//              owns TMEM.
// TMEM (512 columns): S_A[2] [0,128), S_B[2] [128,256), O_A [256,384),
// O_B [384,512); S buffers hold fp32 scores, P overwrites their first 32
// columns.
//
// Every mbarrier wait is bounded; after a wait expires the CTA raises
// SIMSD_EW_TIMEOUT, every role leaves its loops (the softmax warps still
// meet at their named barriers), drains its copies and MMAs and frees TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace simsd {
namespace {

constexpr int kTile = 64;        // keys per tile
constexpr int kD = 128;          // head dimension
constexpr int kRows = 128;       // query rows per row block (MMA M)
constexpr int kStages = 5;       // K/V ring slots
constexpr int kThreads = 512;  // warps 14-15 only meet the final barrier
constexpr int kSoftmaxThreads = 256;
constexpr int kWarpProducer = 8;
constexpr int kWarpMma = 9;  // S issuer of row block A and TMEM owner; warp 10: S of block B
constexpr int kWarpPv = 12;  // PV issuer of row block A; warp 13: PV of block B
constexpr int kWarpProducerV = 11;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;    // S of block X, buffer u: kColS + 64 * (2X + u)
constexpr uint32_t kColO = 256;  // O of block X: kColO + 128 X
constexpr int kHalfBytes = kTile * 128;      // 64 rows x 64 bf16 (one d-half of K or V)
constexpr int kSlotBytes = 4 * kHalfBytes;   // K0 K1 V0 V1
constexpr int kQHalfBytes = kRows * 128;     // 128 rows x 64 bf16
constexpr int kQBlockBytes = 2 * kQHalfBytes;
constexpr int kMaxSort = 256;                // sequences ranked by prefix length (longest first)
constexpr int kMaxStreamK = kMaxSort - 1;    // stream-K: tile offsets of Bt + 1 sequences in `order`
constexpr float kRescaleThreshold = 8.0f;    // log2 units: rescale when the max grows by > 2^8
static_assert(kTile == 64, "the softmax reductions are written out for 64 keys");

struct Tc256Params {
  const int32_t* block_table;
  const int32_t* prefix_len;
  const int32_t* tau;
  const uint8_t* section;
  const int32_t* rope_pos;  // [Bt][2*gamma] or null (inputs rotated already)
  __nv_bfloat16* out;
  int32_t* err_word;
  int max_pages, page_size, num_pages;
  int Bt, S, Hq, Hkv, g, s_blk;
  int units;   // Bt * Hkv
  int nsplit;  // key-tile ranges per unit (work items = units * nsplit)
  int items;
  int streamk;  // 1: equal runs of the global key-tile sequence per CTA (Bt <= kMaxStreamK)
  int ctas;     // grid size (stream-K partial slots: 2 per CTA)
  float* ws;    // partial O, (m, l) of split units (layouts at partial_entry)
  int sort;     // rank sequences by prefix length (Bt <= kMaxSort)
  float scale_log2;
  unsigned long long wait_ns;
  uint32_t extra_p;  // planted extra arrivals on bar_p (a test of the bounded waits)
  RopeTable rope;
};

struct alignas(1024) Smem256 {
  uint8_t ring[kStages][kSlotBytes];
  uint8_t q[2][kQBlockBytes];
  // K and V of a slot are released apart: K once the tile's S MMAs have
  // completed, V once its PV MMAs have
  uint64_t bar_k[kStages], bar_v[kStages], bar_kfree[kStages], bar_vfree[kStages];
  uint64_t bar_q, bar_qr, bar_qfree;
  uint64_t bar_s[2][2], bar_p[2][2], bar_ofree[2];
  // PV_X of the tiles that use S buffer u have completed (one phase per PV)
  uint64_t bar_pvs[2][2];
  uint64_t bar_drain[4];
  uint32_t tmem_base;
  int abort_flag;
  int bad[2];           // per unit parity: a needed page id is out of range
  int32_t tau[2][64];   // per unit parity: slot labels of the unit's sequence
  uint8_t sect[2][64];
  int32_t order[kMaxSort];  // ranking, or (stream-K) tile offsets of the sequences
};

constexpr size_t smem_bytes() { return sizeof(Smem256) + 1024; }
static_assert(smem_bytes() <= 232448, "one CTA per SM");

__device__ __forceinline__ void signal_abort(Smem256& sm, int32_t* err_word) {
  raise_error(err_word, SIMSD_EW_TIMEOUT);
  *reinterpret_cast<volatile int*>(&sm.abort_flag) = 1;
}

// Row r of a 128-byte-swizzled tile: 16-byte chunk c sits at chunk c ^ (r & 7).
__device__ __forceinline__ uint4* sw128_chunk(uint8_t* half, int r, int c) {
  return reinterpret_cast<uint4*>(half + r * 128 + ((c ^ (r & 7)) << 4));
}

// Rotates the pairs (x_i, x_{i+64}) held in chunk c of two d-halves in place.
__device__ __forceinline__ void rope_chunk_pair(uint4* pa, uint4* pb, int pos, int c, const RopeTable& rope) {
  const uint4 va = *pa, vb = *pb;
  uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    float x0 = __uint_as_float(wa[w] << 16), x1 = __uint_as_float(wa[w] & 0xffff0000u);
    float y0 = __uint_as_float(wb[w] << 16), y1 = __uint_as_float(wb[w] & 0xffff0000u);
    float sn, cs;
    rope_sincos(pos, rope.f[8 * c + 2 * w], &sn, &cs);
    rope_pair(x0, y0, sn, cs);
    rope_sincos(pos, rope.f[8 * c + 2 * w + 1], &sn, &cs);
    rope_pair(x1, y1, sn, cs);
    wa[w] = pack_bf16x2(x0, x1);
    wb[w] = pack_bf16x2(y0, y1);
  }
  *pa = make_uint4(wa[0], wa[1], wa[2], wa[3]);
  *pb = make_uint4(wb[0], wb[1], wb[2], wb[3]);
}

// Tiles of a unit of a sequence with prefix length n: ceil(n / 64) + 1 (tile
// 0: the new slots); stream-K counts one for a length out of range (a piece
// that only zeroes the unit's rows).
__device__ __forceinline__ bool prefix_bad(const Tc256Params& p, int n) {
  return n < 0 || static_cast<long long>(n) > static_cast<long long>(p.max_pages) * p.page_size;
}
__device__ __forceinline__ int streamk_tiles(const Tc256Params& p, int n) {
  return prefix_bad(p, n) ? 1 : (n + kTile - 1) / kTile + 1;
}

// The work item at position U of the walk: key-tile range `split` of the
// unit (sequence b, KV head), sequences longest prefix first when ranked.
// A unit has T = ceil(n / 64) + 1 tiles (tile 0: the new slots, 1..: the
// prefix; none when the prefix length is out of range); range i holds tiles
// [ceil(i T / nsplit), ceil((i + 1) T / nsplit)), so range 0 holds tile 0.
struct Unit {
  int b, kvh, n, split, t0, tiles;
  bool n_bad;
  bool lead;  // the piece that raises the unit's error bits (range 0, or the one with tile 0)
  bool part;  // writes partial results instead of the output
  int slot;   // stream-K: 0 for the piece at the start of the CTA's run, else 1
  bool last;  // the CTA's last piece
};

__device__ __forceinline__ Unit unit_at(const Tc256Params& p, const Smem256& sm, int U) {
  Unit u;
  const int unit = U / p.nsplit;
  u.split = U - unit * p.nsplit;
  const int rank = unit / p.Hkv;
  u.kvh = unit - rank * p.Hkv;
  u.b = p.sort ? sm.order[rank] : rank;
  u.n = p.prefix_len[u.b];
  u.n_bad = prefix_bad(p, u.n);
  // T < 2^25 and split < 64: the products fit 32 bits
  const unsigned T = u.n_bad ? 0u : static_cast<unsigned>((u.n + kTile - 1) / kTile + 1);
  const unsigned ns = static_cast<unsigned>(p.nsplit), sp = static_cast<unsigned>(u.split);
  u.t0 = static_cast<int>((sp * T + ns - 1) / ns);
  u.tiles = static_cast<int>(((sp + 1) * T + ns - 1) / ns) - u.t0;
  return u;
}

// cum[b] = key tiles of the units of sequences 0 .. b-1 (Hkv units each),
// cum[Bt] = all of them (below 2^30, as the planner checks).  Called by
// every thread of the block; Bt <= 255.
__device__ void streamk_offsets(const Tc256Params& p, int32_t* cum) {
  for (int b = threadIdx.x; b < p.Bt; b += blockDim.x) cum[b + 1] = p.Hkv * streamk_tiles(p, p.prefix_len[b]);
  __syncthreads();
  if (threadIdx.x < 32) {
    // lane l scans entries 8l + 1 .. 8l + 8
    const int lane = threadIdx.x;
    int v[8], sum = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int i = 8 * lane + j + 1;
      v[j] = i <= p.Bt ? cum[i] : 0;
      sum += v[j];
    }
    int inc = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    int run = inc - sum;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int i = 8 * lane + j + 1;
      run += v[j];
      if (i <= p.Bt) cum[i] = run;
    }
    if (lane == 0) cum[0] = 0;
  }
  __syncthreads();
}

// The sequence whose units hold global tile G: cum[b] <= G < cum[b + 1]
// (every sequence holds at least Hkv tiles, so b is unique).
__device__ __forceinline__ int streamk_seq(const int32_t* cum, int Bt, int G) {
  int lo = 0, hi = Bt - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (cum[mid] <= G)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

// A CTA's walk: the next item of the ranges walk, or the next tile of its
// stream-K run [R0, R1).  The run is walked from H, the first unit start in
// it, to R1, and then [R0, H): the piece cut at the run's start comes last,
// so that both pieces of a unit cut by a boundary are written near the end
// of the launch (and stay in L2 for the merge).
struct Walk {
  int U;  // ranges: the next item; stream-K: the phase (0: [H, R1), 1: [R0, H))
  int G, R0, R1, H;
};

__device__ __forceinline__ Walk walk_begin(const Tc256Params& p, const Smem256& sm) {
  Walk w;
  w.U = blockIdx.x;
  w.G = w.R0 = w.R1 = w.H = 0;
  if (p.streamk) {
    w.U = 0;
    const int total = sm.order[p.Bt];
    const int W = (total + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x);
    w.R0 = static_cast<int>(min(static_cast<long long>(total), static_cast<long long>(blockIdx.x) * W));
    w.R1 = min(total, w.R0 + W);
    w.H = w.R0;
    if (w.R0 < w.R1) {
      const int b = streamk_seq(sm.order, p.Bt, w.R0);
      const int T = streamk_tiles(p, p.prefix_len[b]);
      const int t = (w.R0 - sm.order[b]) % T;
      if (t > 0) w.H = min(w.R1, w.R0 - t + T);
    }
    w.G = w.H;
  }
  return w;
}

// The CTA's next piece; false when its walk is done.  Every role walks the
// same pieces in the same order.
__device__ __forceinline__ bool walk_next(const Tc256Params& p, const Smem256& sm, Walk& w, Unit& u) {
  if (!p.streamk) {
    if (w.U >= p.items) return false;
    u = unit_at(p, sm, w.U);
    w.U += gridDim.x;
    u.lead = u.split == 0;
    u.part = p.nsplit > 1;
    u.slot = 0;
    u.last = w.U >= p.items;
    return true;
  }
  if (w.U == 0 && w.G >= w.R1) {
    w.U = 1;  // then the piece cut at the run's start
    w.G = w.R0;
  }
  if (w.U == 1 && w.G >= w.H) return false;
  const int end = w.U == 0 ? w.R1 : w.H;
  const int b = streamk_seq(sm.order, p.Bt, w.G);
  u.b = b;
  u.n = p.prefix_len[b];
  u.n_bad = prefix_bad(p, u.n);
  const int T = u.n_bad ? 1 : (u.n + kTile - 1) / kTile + 1;
  const int off = w.G - sm.order[b];
  u.kvh = off / T;
  u.t0 = off - u.kvh * T;
  const int take = min(T - u.t0, end - w.G);
  u.split = 0;
  u.tiles = u.n_bad ? 0 : take;
  u.lead = u.t0 == 0;
  u.part = take < T;
  u.slot = w.G == w.R0 ? 0 : 1;
  w.G += take;
  u.last = w.U == 1 ? w.G >= w.H : (w.G >= w.R1 && w.H == w.R0);
  return true;
}

// Partial results of a split unit: O (unnormalised, fp32) [entries][128][d],
// then (m, l) [entries][128][2], row `row` of block x; m is the row's
// reference maximum in log2 units.  Ranges walk (the combine kernel's
// layout): entries = units * 2 * nsplit, entry ((b Hkv + kvh) 2 + x) nsplit
// + split.  Stream-K: entries = ctas * 4, entry (cta * 2 + slot) * 2 + x.
__device__ __forceinline__ size_t partial_entries(const Tc256Params& p) {
  return p.streamk ? static_cast<size_t>(p.ctas) * 4 : static_cast<size_t>(p.units) * 2 * p.nsplit;
}
__device__ __forceinline__ size_t partial_entry(const Tc256Params& p, const Unit& u, int x) {
  if (p.streamk) return (static_cast<size_t>(blockIdx.x) * 2 + u.slot) * 2 + x;
  return ((static_cast<size_t>(u.b) * p.Hkv + u.kvh) * 2 + x) * p.nsplit + u.split;
}
__device__ __forceinline__ float* partial_o(const Tc256Params& p, const Unit& u, int x, int row) {
  return p.ws + (partial_entry(p, u, x) * kRows + row) * kD;
}
__device__ __forceinline__ float* partial_ml(const Tc256Params& p, const Unit& u, int x, int row) {
  return p.ws + partial_entries(p) * kRows * kD + (partial_entry(p, u, x) * kRows + row) * 2;
}
// Stream-K: after the partials, one record per run boundary c (int4): the
// unit that boundary c is the first to cut (b Hkv + kvh, or -1), the CTAs
// c0 .. c1 holding its pieces and the slot of CTA c0's piece.
__device__ __forceinline__ int4* streamk_records(const Tc256Params& p) {
  return reinterpret_cast<int4*>(p.ws + partial_entries(p) * kRows * (kD + 2));
}

__global__ void __launch_bounds__(kThreads, 1)
    attention_tc256_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kn,
                           const __grid_constant__ CUtensorMap tm_vn, const __grid_constant__ CUtensorMap tm_kc,
                           const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ Tc256Params p) {
  extern __shared__ uint8_t smem_raw[];
  Smem256& sm =
      *reinterpret_cast<Smem256*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  volatile int* abort_flag = &sm.abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    sm.abort_flag = 0;
    sm.bad[0] = sm.bad[1] = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&sm.bar_k[s]), 1);
      mbar_init(smem_u32(&sm.bar_v[s]), 1);
      mbar_init(smem_u32(&sm.bar_kfree[s]), 2);  // one commit per MMA issuer
      mbar_init(smem_u32(&sm.bar_vfree[s]), 2);
    }
    mbar_init(smem_u32(&sm.bar_q), 1);
    mbar_init(smem_u32(&sm.bar_qr), 1);
    mbar_init(smem_u32(&sm.bar_qfree), 2);  // one commit per S issuer
    for (int x = 0; x < 2; ++x) {
      for (int u = 0; u < 2; ++u) {
        mbar_init(smem_u32(&sm.bar_s[x][u]), 1);
        mbar_init(smem_u32(&sm.bar_p[x][u]), 4 + p.extra_p);
        mbar_init(smem_u32(&sm.bar_pvs[x][u]), 1);
      }
      mbar_init(smem_u32(&sm.bar_ofree[x]), 4);
    }
    for (int d = 0; d < 4; ++d) mbar_init(smem_u32(&sm.bar_drain[d]), 1);
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpProducer && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kn);
    tma_prefetch_desc(&tm_vn);
    tma_prefetch_desc(&tm_kc);
    tma_prefetch_desc(&tm_vc);
  }
  // from here on the previous kernel's results (prefix lengths, labels) are read
  pdl_wait();
  if (p.sort) {
    // rank sequences by prefix length, longest first (ties: lower index first)
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
      sm.order[r] = i;
    }
    // the staging area is overwritten by TMA later
    fence_proxy_async_smem();
  }
  if (p.streamk) streamk_offsets(p, sm.order);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  // Register split (setmaxnreg, per warpgroup): the two softmax warpgroups
  // take 200 registers a thread, the two control warpgroups give theirs
  // down to 56 (2 x 128 x 200 + 2 x 128 x 56 = 65,536, the 512 x 128 the
  // block is launched with).
  if (warp >= 8) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 56;");
    if (warp == kWarpProducer || warp == kWarpProducerV) {
      // ----------------------------------------------------------- producers
      // warp 8 loads Q and the K half of every tile, warp 11 the V half; each
      // refills a slot's half as soon as that half is released, so K runs
      // ahead of V (K is consumed a softmax earlier than V)
      const int kv = warp == kWarpProducer ? 0 : 1;
      uint32_t g = 0, jq = 0;  // tiles and pieces (with tiles) issued so far
      bool ok = true;
      Walk w = walk_begin(p, sm);
      Unit u;
      while (ok && walk_next(p, sm, w, u)) {
        if (u.tiles == 0) continue;
        if (kv == 0) {
          if (lane == 0 && jq > 0 && !mbar_wait(smem_u32(&sm.bar_qfree), (jq - 1) & 1, abort_flag, p.wait_ns))
            ok = false;
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;
          if (lane == 0) {
            const uint32_t bq = smem_u32(&sm.bar_q);
            const int z = u.b * p.S;
            mbar_arrive_expect_tx(bq, 2u * kQBlockBytes);
            tma_load_3d(smem_u32(sm.q[0]), &tm_q, bq, 0, u.kvh * p.g, z);
            tma_load_3d(smem_u32(sm.q[0]) + kQHalfBytes, &tm_q, bq, 64, u.kvh * p.g, z);
            tma_load_3d(smem_u32(sm.q[1]), &tm_q, bq, 0, u.kvh * p.g, z + p.s_blk);
            tma_load_3d(smem_u32(sm.q[1]) + kQHalfBytes, &tm_q, bq, 64, u.kvh * p.g, z + p.s_blk);
          }
          ++jq;
        }
        const int32_t* bt = p.block_table + static_cast<size_t>(u.b) * p.max_pages;
        const int P = p.page_size;
        int win_base = -(1 << 30), win = -1;  // lane i holds the page id of page win_base + i
        for (int t = u.t0; t < u.t0 + u.tiles; ++t) {
          const int st = g % kStages;
          // page ids this tile needs (prefix tiles), loaded by the whole warp
          int pi0 = 0, nsub = 0, key0 = 0, valid = 0;
          if (t > 0) {
            key0 = (t - 1) * kTile;
            valid = min(kTile, u.n - key0);
            pi0 = key0 / P;
            nsub = P >= kTile ? 1 : (valid + P - 1) / P;
            if (pi0 < win_base || pi0 + nsub > win_base + 32) {
              win_base = pi0;
              const int pi = win_base + lane;
              win = pi < p.max_pages ? bt[pi] : -1;
            }
          }
          int pgs[kTile / 8];
  #pragma unroll
          for (int sb = 0; sb < kTile / 8; ++sb) {
            const int pg = __shfl_sync(0xffffffffu, win, (pi0 + sb - win_base) & 31);
            // a page id out of range is replaced by page 0 (the softmax warps
            // zero that sequence's output and the error bit is set there)
            pgs[sb] = (pg < 0 || pg >= p.num_pages) ? 0 : pg;
          }
          if (lane == 0) {
            const uint64_t* freed = kv == 0 ? &sm.bar_kfree[st] : &sm.bar_vfree[st];
            if (g >= static_cast<uint32_t>(kStages) &&
                !mbar_wait(smem_u32(freed), ((g / kStages) - 1) & 1, abort_flag, p.wait_ns)) {
              ok = false;
            } else {
              const uint32_t bar = smem_u32(kv == 0 ? &sm.bar_k[st] : &sm.bar_v[st]);
              const uint32_t d0 = smem_u32(sm.ring[st]) + 2 * kv * kHalfBytes, d1 = d0 + kHalfBytes;
              if (t == 0) {
                const CUtensorMap* m = kv == 0 ? &tm_kn : &tm_vn;
                mbar_arrive_expect_tx(bar, 2u * static_cast<uint32_t>(p.S) * 128u);
                tma_load_3d(d0, m, bar, 0, u.kvh, u.b * p.S);
                tma_load_3d(d1, m, bar, 64, u.kvh, u.b * p.S);
              } else {
                const CUtensorMap* m = kv == 0 ? &tm_kc : &tm_vc;
                if (P >= kTile) {
                  const int row = (pgs[0] * p.Hkv + u.kvh) * P + (key0 % P);
                  mbar_arrive_expect_tx(bar, 2u * kHalfBytes);
                  tma_load_2d(d0, m, bar, 0, row);
                  tma_load_2d(d1, m, bar, 64, row);
                } else {
                  const uint32_t sub_bytes = static_cast<uint32_t>(P) * 128u;
                  mbar_arrive_expect_tx(bar, 2u * nsub * sub_bytes);
  #pragma unroll
                  for (int sb = 0; sb < kTile / 8; ++sb) {
                    if (sb < nsub) {  // (a constant index keeps pgs in registers)
                      const int row = (pgs[sb] * p.Hkv + u.kvh) * P;
                      tma_load_2d(d0 + sb * sub_bytes, m, bar, 0, row);
                      tma_load_2d(d1 + sb * sub_bytes, m, bar, 64, row);
                    }
                  }
                }
              }
            }
          }
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;  // nothing was issued for tile g
          ++g;
        }
      }
      if (!ok && lane == 0) signal_abort(sm, p.err_word);
      // Drain: every issued load of this warp must have landed before the CTA
      // may exit (full limit, whatever the other waits use).
      if (lane == 0) {
        for (uint32_t it = g > static_cast<uint32_t>(kStages) ? g - kStages : 0; it < g; ++it) {
          const int st = it % kStages;
          mbar_wait(smem_u32(kv == 0 ? &sm.bar_k[st] : &sm.bar_v[st]), (it / kStages) & 1, nullptr);
        }
        if (kv == 0 && jq > 0) mbar_wait(smem_u32(&sm.bar_q), (jq - 1) & 1, nullptr);
      }
      __syncwarp();
    } else if (warp >= kWarpMma && warp <= kWarpPv + 1) {
      // ---------------------------------------------------------- MMA issuers
      // four threads: the S MMAs of row block A (warp 9) and B (warp 10), the
      // PV MMAs of A (warp 12) and B (warp 13).  A thread that issues a
      // tcgen05.mma is held about as long as the MMA runs, so a thread that
      // served two of these streams kept a request of one waiting behind the
      // MMAs of the other (a written P behind the next tile's S, or one
      // block's P behind the other's PV).  Each thread waits on one barrier
      // at a time, polling it with test_wait (a try_wait that suspends the
      // thread woke it later; ~1% slower at 32 drafts).
      const bool is_s = warp < kWarpProducerV;
      const int x = is_s ? warp - kWarpMma : warp - kWarpPv;
      if (lane == 0) {
        constexpr uint32_t kIdescQK = idesc_bf16_f32(kRows, kTile, 0, 0);
        constexpr uint32_t kIdescPV = idesc_bf16_f32(kRows, kD, 0, 1);
        const uint32_t qb0 = smem_u32(sm.q[x]), qb1 = qb0 + kQHalfBytes;
        const uint32_t ocol = tmem + kColO + 128u * x;
        uint32_t g = 0, jq = 0;
        bool ok = true;
        Walk w = walk_begin(p, sm);
        Unit u;
        while (ok && walk_next(p, sm, w, u)) {
          if (u.tiles == 0) continue;
          ++jq;
          const uint32_t g0 = g, g_end = g + u.tiles;
          if (is_s) {
            // Q landed (rotated by the softmax warps when RoPE is applied here)
            ok = mbar_wait(smem_u32(p.rope_pos ? &sm.bar_qr : &sm.bar_q), (jq - 1) & 1, abort_flag, p.wait_ns);
            for (uint32_t gg = g0; ok && gg < g_end; ++gg) {
              // S_X(t) needs K(t) and the completion of PV_X(t - 2), which read
              // the P held in the same S buffer
              const int st = gg % kStages;
              ok = mbar_wait_poll(smem_u32(&sm.bar_k[st]), (gg / kStages) & 1, abort_flag, p.wait_ns) &&
                   (gg < 2 || mbar_wait_poll(smem_u32(&sm.bar_pvs[x][gg & 1]), ((gg - 2) >> 1) & 1, abort_flag, p.wait_ns));
              if (!ok) break;
              tc_fence_after();
              const uint32_t kb0 = smem_u32(sm.ring[st]), kb1 = kb0 + kHalfBytes;
              const uint32_t scol = tmem + kColS + 64u * (2 * x + (gg & 1));
  #pragma unroll
              for (int kk = 0; kk < kD / 16; ++kk) {
                const uint32_t off = (kk & 3) * 32;
                tc_mma_ss(scol, sdesc_sw128((kk < 4 ? qb0 : qb1) + off, 16, 1024),
                          sdesc_sw128((kk < 4 ? kb0 : kb1) + off, 16, 1024), kIdescQK, kk > 0);
              }
              tc_commit(smem_u32(&sm.bar_s[x][gg & 1]));
              // K of this slot may be replaced once both blocks' S have completed
              tc_commit(smem_u32(&sm.bar_kfree[st]));
            }
            // the unit's last S MMAs: Q may be replaced once both blocks' have completed
            if (ok) tc_commit(smem_u32(&sm.bar_qfree));
          } else {
            for (uint32_t gg = g0; ok && gg < g_end; ++gg) {
              // PV_X(t) needs P_X(t), V(t) and, for the unit's first tile, the
              // previous unit's O_X read out by the epilogue
              const int st = gg % kStages;
              const bool first = gg == g0;
              ok = mbar_wait_poll(smem_u32(&sm.bar_p[x][gg & 1]), (gg >> 1) & 1, abort_flag, p.wait_ns) &&
                   (!first || jq <= 1 || mbar_wait_poll(smem_u32(&sm.bar_ofree[x]), (jq - 2) & 1, abort_flag, p.wait_ns)) &&
                   mbar_wait_poll(smem_u32(&sm.bar_v[st]), (gg / kStages) & 1, abort_flag, p.wait_ns);
              if (!ok) break;
              tc_fence_after();
              const uint32_t vb = smem_u32(sm.ring[st]) + 2 * kHalfBytes;
              const uint32_t pcol = tmem + kColS + 64u * (2 * x + (gg & 1));
  #pragma unroll
              for (int kk = 0; kk < kTile / 16; ++kk)
                tc_mma_ts(ocol, pcol + 8 * kk, sdesc_sw128(vb + kk * 2048, kHalfBytes, 1024), kIdescPV,
                          (first && kk == 0) ? 0u : 1u);
              tc_commit(smem_u32(&sm.bar_pvs[x][gg & 1]));
              tc_commit(smem_u32(&sm.bar_vfree[st]));
            }
          }
          g = g_end;
        }
        if (!ok) signal_abort(sm, p.err_word);
        // every MMA issued by this thread has completed once this fires
        const int d = (is_s ? 0 : 2) + x;
        tc_commit(smem_u32(&sm.bar_drain[d]));
        mbar_wait(smem_u32(&sm.bar_drain[d]), 0, nullptr);
      }
      __syncwarp();
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 200;");
    // -------------------------------------------------------------- softmax
    const int x = warp >> 2;          // row block
    const int row = tid & (kRows - 1);  // TMEM lane / query row of the block
    const int hl = row % p.g;
    const uint32_t lane_tmem = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t o_tmem = lane_tmem + kColO + 128u * x;
    uint32_t g = 0, jq = 0, mu = 0;
    bool ok = true;
    Walk w = walk_begin(p, sm);
    Unit u;
    for (; walk_next(p, sm, w, u); ++mu) {
      const int par = mu & 1;  // metadata buffer of this piece
      // every softmax thread is done with the previous unit: its flag
      // (the other buffer) is cleared for the next one
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (tid == 0) sm.bad[par ^ 1] = 0;
      if (tid < p.S) {
        sm.tau[par][tid] = p.tau[static_cast<size_t>(u.b) * p.S + tid];
        sm.sect[par][tid] = p.section[static_cast<size_t>(u.b) * p.S + tid];
      }
      if (u.n_bad) {
        if (tid == 0 && u.kvh == 0 && u.lead) raise_error(p.err_word, SIMSD_EW_PREFIX_LEN);
      } else {
        const int npages = (u.n + p.page_size - 1) / p.page_size;
        const int32_t* bt = p.block_table + static_cast<size_t>(u.b) * p.max_pages;
        bool bad = false;
        for (int i = tid; i < npages; i += kSoftmaxThreads) {
          const int pg = bt[i];
          bad |= pg < 0 || pg >= p.num_pages;
        }
        if (bad) {
          atomicOr(&sm.bad[par], 1);
          if (u.kvh == 0 && u.lead) raise_error(p.err_word, SIMSD_EW_PAGE);
        }
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
      const bool seq_bad = u.n_bad || sm.bad[par] != 0;
      const int s = x * p.s_blk + row / p.g;
      const bool row_exists = s < p.S;
      const bool active = row_exists && !seq_bad && sm.sect[par][s] != kSectPad;
      unsigned long long vis = 0ull;
      if (active) {
        const uint8_t si = sm.sect[par][s];
        const int ti = sm.tau[par][s];
        for (int t = 0; t < p.S; ++t)
          if (temporal_visible(si, ti, sm.sect[par][t], sm.tau[par][t])) vis |= 1ull << t;
      }
      float m_ref = -INFINITY, l_sum = 0.f;
      if (u.tiles > 0) {
        ++jq;
        if (p.rope_pos) {
          // Q of both blocks and, in range 0, the new keys (its first tile)
          // are rotated in shared memory before the first S reads them
          const int pos = p.rope_pos[static_cast<size_t>(u.b) * p.S + (row_exists ? s : 0)];
          if (ok) ok = mbar_wait_warp(smem_u32(&sm.bar_q), (jq - 1) & 1, abort_flag, p.wait_ns);
          if (ok) {
            uint8_t* h0 = sm.q[x];
            uint8_t* h1 = sm.q[x] + kQHalfBytes;
#pragma unroll 1
            for (int c = 0; c < 8; ++c) rope_chunk_pair(sw128_chunk(h0, row, c), sw128_chunk(h1, row, c), pos, c, p.rope);
          }
          const int st0 = g % kStages;
          if (ok && u.t0 == 0) ok = mbar_wait_warp(smem_u32(&sm.bar_k[st0]), (g / kStages) & 1, abort_flag, p.wait_ns);
          if (ok && u.t0 == 0) {
            uint8_t* h0 = sm.ring[st0];
            uint8_t* h1 = sm.ring[st0] + kHalfBytes;
            for (int task = tid; task < p.S * 8; task += kSoftmaxThreads) {
              const int r = task >> 3, c = task & 7;
              const int kpos = p.rope_pos[static_cast<size_t>(u.b) * p.S + r];
              rope_chunk_pair(sw128_chunk(h0, r, c), sw128_chunk(h1, r, c), kpos, c, p.rope);
            }
          }
          fence_proxy_async_smem();
          asm volatile("bar.sync 1, 256;" ::: "memory");
          if (tid == 0 && !*abort_flag) mbar_arrive(smem_u32(&sm.bar_qr));
        }
        for (int i = 0; ok && i < u.tiles; ++i) {
          const uint32_t gg = g + i;
          const int st = gg % kStages;
          const uint32_t buf = gg & 1;
          const uint32_t s_tmem = lane_tmem + kColS + 64u * (2 * x + buf);
          if (!mbar_wait_warp(smem_u32(&sm.bar_s[x][buf]), (gg >> 1) & 1, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          uint32_t sa[32], sb[32];
          tmem_ld32(s_tmem, sa);
          tmem_ld32(s_tmem + 32, sb);
          tmem_wait_ld();
          const int t = u.t0 + i;  // tile of the unit
          const bool is_new = (t == 0);
          const int valid = is_new ? p.S : min(kTile, u.n - (t - 1) * kTile);
          float xs[kTile];
#pragma unroll
          for (int c = 0; c < kTile; ++c) xs[c] = __uint_as_float(c < 32 ? sa[c] : sb[c - 32]);
          if (is_new || valid < kTile) {
            // one bit word per row and a select per column (no divergence)
            const unsigned long long keep = is_new ? vis : ((1ull << valid) - 1ull);
            const uint32_t klo = static_cast<uint32_t>(keep), khi = static_cast<uint32_t>(keep >> 32);
#pragma unroll
            for (int c = 0; c < kTile; ++c) {
              const uint32_t bit = ((c < 32 ? klo : khi) >> (c & 31)) & 1u;
              xs[c] = bit ? xs[c] : -INFINITY;
            }
          }
          float mx;
          {
            // 64 -> 22 -> 8 -> 3 -> 1 with three-input maxima
            float r[22], r2[8];
#pragma unroll
            for (int c = 0; c < 21; ++c) r[c] = fmax3(xs[3 * c], xs[3 * c + 1], xs[3 * c + 2]);
            r[21] = xs[63];
#pragma unroll
            for (int c = 0; c < 7; ++c) r2[c] = fmax3(r[3 * c], r[3 * c + 1], r[3 * c + 2]);
            r2[7] = r[21];
            const float m3 = fmax3(fmax3(r2[0], r2[1], r2[2]), fmax3(r2[3], r2[4], r2[5]), fmaxf(r2[6], r2[7]));
            mx = active ? m3 * p.scale_log2 : -INFINITY;
          }
          bool need = false;
          if (active && mx != -INFINITY) {
            if (m_ref == -INFINITY)
              m_ref = mx;
            else if (mx > m_ref + kRescaleThreshold)
              need = true;
          }
          if (__any_sync(0xffffffffu, need)) {
            // O holds the unit's earlier tiles: wait until the last PV of
            // this block has completed, then scale it
            if (i > 0 && !mbar_wait_warp(smem_u32(&sm.bar_pvs[x][(gg - 1) & 1]), ((gg - 1) >> 1) & 1, abort_flag,
                                         p.wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const float f = need ? fast_exp2(m_ref - mx) : 1.0f;
            if (need) {
              l_sum *= f;
              m_ref = mx;
            }
            if (i > 0) {
#pragma unroll 1
              for (int ch = 0; ch < kD / 32; ++ch) {
                uint32_t o[32];
                tmem_ld32(o_tmem + 32 * ch, o);
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * f);
                tmem_st32(o_tmem + 32 * ch, o);
              }
            }
          }
          const float neg_m = (active && m_ref != -INFINITY) ? -m_ref : 0.f;
          uint32_t pk[32];
          unsigned long long ps[kTile / 2];
          {
            const unsigned long long sc2 = f32x2(p.scale_log2, p.scale_log2), nm2 = f32x2(neg_m, neg_m);
#pragma unroll
            for (int c = 0; c < kTile / 2; ++c) {
              float e0, e1;
              f32x2_split(fma_f32x2(f32x2(xs[2 * c], xs[2 * c + 1]), sc2, nm2), e0, e1);
              const float p0 = fast_exp2(e0), p1 = fast_exp2(e1);
              ps[c] = f32x2(p0, p1);
              pk[c] = pack_bf16x2(p0, p1);
            }
          }
#pragma unroll
          for (int w2 = kTile / 4; w2 >= 1; w2 >>= 1)
#pragma unroll
            for (int c = 0; c < w2; ++c) ps[c] = add_f32x2(ps[c], ps[c + w2]);
          {
            float s0, s1;
            f32x2_split(ps[0], s0, s1);
            l_sum += s0 + s1;
          }
          tmem_st32(s_tmem, pk);
          tmem_wait_st();
          if ((warp & 3) < 2 && (valid < kTile || is_new)) {
            // rows of V that no query may use are zeroed so that 0 * (stale
            // or non-finite data) cannot reach O.  The first two warps of
            // each block zero them (writing the same zeros), so that each
            // block's PV, which waits only for its own P, sees them zeroed.
            if (!mbar_wait_warp(smem_u32(&sm.bar_v[st]), (gg / kStages) & 1, abort_flag, p.wait_ns)) {
              ok = false;
              break;
            }
            const bool zero = row >= valid || (is_new && sm.sect[par][row] == kSectPad);
            if (zero) {
              const uint4 z = make_uint4(0u, 0u, 0u, 0u);
              uint4* r0 = reinterpret_cast<uint4*>(sm.ring[st] + 2 * kHalfBytes + row * 128);
              uint4* r1 = reinterpret_cast<uint4*>(sm.ring[st] + 3 * kHalfBytes + row * 128);
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
          if (lane == 0) mbar_arrive(smem_u32(&sm.bar_p[x][buf]));
        }
        if (u.last) pdl_launch_next();
        // ---- epilogue: O of the unit's last PV, scaled by 1/l.  The S of
        // the last tile implies that the PV two tiles back has completed,
        // not the one just before, so the PVs of the last two tiles are
        // awaited, each on the barrier of its S buffer: neither barrier can
        // complete a later phase before this epilogue has ended (their next
        // PVs need P of the next unit), so no parity wait can be misread.
        const uint32_t last = g + u.tiles - 1;
        bool have_o = ok;
        if (have_o && u.tiles >= 2)
          have_o = mbar_wait_warp(smem_u32(&sm.bar_pvs[x][(last - 1) & 1]), ((last - 1) >> 1) & 1, abort_flag,
                                  p.wait_ns);
        if (have_o)
          have_o = mbar_wait_warp(smem_u32(&sm.bar_pvs[x][last & 1]), (last >> 1) & 1, abort_flag, p.wait_ns);
        if (!have_o) ok = false;
        if (have_o) tc_fence_after();
        const bool any = have_o && active && l_sum > 0.f;
        const float inv = any ? 1.0f / l_sum : 0.f;
        const int h = u.kvh * p.g + hl;
        __nv_bfloat16* orow = p.out + ((static_cast<size_t>(u.b) * p.S + (row_exists ? s : 0)) * p.Hq + h) * kD;
        // a split unit leaves its partial O (fp32) and (m, l) to the combine
        const bool part = u.part;
        float* wo = part ? partial_o(p, u, x, row) : nullptr;
#pragma unroll 1
        for (int ch = 0; ch < kD / 32; ++ch) {
          uint32_t o[32];
          if (have_o) {
            tmem_ld32(o_tmem + 32 * ch, o);
            tmem_wait_ld();
          }
          if (row_exists && part) {
            float4* dst = reinterpret_cast<float4*>(wo + 32 * ch);
#pragma unroll
            for (int c = 0; c < 8; ++c)
              dst[c] = any ? make_float4(__uint_as_float(o[4 * c]), __uint_as_float(o[4 * c + 1]),
                                         __uint_as_float(o[4 * c + 2]), __uint_as_float(o[4 * c + 3]))
                           : make_float4(0.f, 0.f, 0.f, 0.f);
          } else if (row_exists) {
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
        if (row_exists && part) {
          float* wml = partial_ml(p, u, x, row);
          wml[0] = any ? m_ref : -INFINITY;
          wml[1] = any ? l_sum : 0.f;
        }
        // O_X may be overwritten by the next unit's first PV
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&sm.bar_ofree[x]));
        g += u.tiles;
      } else if (u.part) {
        // an empty tile range (or a prefix length out of range): an empty
        // partial, which the combine skips
        if (u.last) pdl_launch_next();
        if (row_exists) {
          float4* dst = reinterpret_cast<float4*>(partial_o(p, u, x, row));
#pragma unroll 4
          for (int c = 0; c < kD / 4; ++c) dst[c] = make_float4(0.f, 0.f, 0.f, 0.f);
          float* wml = partial_ml(p, u, x, row);
          wml[0] = -INFINITY;
          wml[1] = 0.f;
        }
      } else {
        // a prefix length out of range: this unit's rows are zero
        if (u.last) pdl_launch_next();
        if (row_exists) {
          const int h = u.kvh * p.g + hl;
          uint4* dst = reinterpret_cast<uint4*>(p.out + ((static_cast<size_t>(u.b) * p.S + s) * p.Hq + h) * kD);
#pragma unroll
          for (int c = 0; c < kD / 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    if (!ok && lane == 0) signal_abort(sm, p.err_word);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  // stream-K: the record of run boundary blockIdx.x for the merge (written
  // last, so that it is still in L2 when the merge reads it)
  if (p.streamk && tid == 0 && blockIdx.x > 0) {
    int4 rec = make_int4(-1, 0, 0, 0);
    const int total = sm.order[p.Bt];
    const int W = (total + static_cast<int>(gridDim.x) - 1) / static_cast<int>(gridDim.x);
    const long long G = static_cast<long long>(blockIdx.x) * W;
    if (G < total) {
      const int b = streamk_seq(sm.order, p.Bt, static_cast<int>(G));
      const int T = streamk_tiles(p, p.prefix_len[b]);
      const int off = static_cast<int>(G) - sm.order[b];
      const int kvh = off / T, t = off - kvh * T;
      const int start = static_cast<int>(G) - t, c0 = start / W;
      if (t > 0 && c0 + 1 == static_cast<int>(blockIdx.x))
        rec = make_int4(b * p.Hkv + kvh, c0, (start + T - 1) / W, start != c0 * W ? 1 : 0);
    }
    streamk_records(p)[blockIdx.x] = rec;
  }
}

// Stream-K merge.  Blocks (c - 1, x, z) take run boundary c, row block x,
// rows 16z .. 16z + 15 (four per warp, lanes over the head dimension).  The
// boundary's record names the unit it is the first to cut and its pieces:
// those of CTAs c0 .. c1 (CTA c0's in the record's slot, the others' in
// slot 0).  Per row: O = sum_i 2^(m_i - M) O_i / sum_i 2^(m_i - M) l_i, M =
// max m_i over the pieces that saw a key (l_i > 0); none gives a zero row.
// A unit cut once (two pieces, the usual case) is merged from loads that
// are all issued together; more pieces take the general loop.
constexpr int kMergeRows = 4;  // rows per warp
__global__ void __launch_bounds__(128) streamk_combine_kernel(const __grid_constant__ Tc256Params p) {
  pdl_wait();
  const int c = static_cast<int>(blockIdx.x) + 1, x = static_cast<int>(blockIdx.y);
  const int4 rec = streamk_records(p)[c];
  if (rec.x >= 0) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int b = rec.x / p.Hkv, kvh = rec.x - b * p.Hkv, c0 = rec.y, np = rec.z - rec.y + 1;
    const int row0 = static_cast<int>(blockIdx.z) * 16 + warp * kMergeRows;
    const size_t entries = static_cast<size_t>(p.ctas) * 4;
    const float2* wml = reinterpret_cast<const float2*>(p.ws + entries * kRows * kD);
    auto entry = [&](int j) { return (static_cast<size_t>(c0 + j) * 2 + (j == 0 ? rec.w : 0)) * 2 + x; };
    float M[kMergeRows], L[kMergeRows];
    float4 acc[kMergeRows];
#pragma unroll
    for (int k = 0; k < kMergeRows; ++k) {
      M[k] = -INFINITY;
      L[k] = 0.f;
      acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (np == 2) {
      const size_t e0 = entry(0), e1 = entry(1);
      const float4* o0 = reinterpret_cast<const float4*>(p.ws + (e0 * kRows + row0) * kD);
      const float4* o1 = reinterpret_cast<const float4*>(p.ws + (e1 * kRows + row0) * kD);
      float4 va[kMergeRows], vb[kMergeRows];
      float2 ma[kMergeRows], mb[kMergeRows];
#pragma unroll
      for (int k = 0; k < kMergeRows; ++k) {
        va[k] = o0[k * (kD / 4) + lane];
        vb[k] = o1[k * (kD / 4) + lane];
        ma[k] = wml[e0 * kRows + row0 + k];
        mb[k] = wml[e1 * kRows + row0 + k];
      }
#pragma unroll
      for (int k = 0; k < kMergeRows; ++k) {
        const bool ha = ma[k].y > 0.f, hb = mb[k].y > 0.f;
        M[k] = fmaxf(ha ? ma[k].x : -INFINITY, hb ? mb[k].x : -INFINITY);
        const float wa = ha ? exp2f(ma[k].x - M[k]) : 0.f, wb = hb ? exp2f(mb[k].x - M[k]) : 0.f;
        L[k] = fmaf(wa, ma[k].y, wb * mb[k].y);
        acc[k] = make_float4(fmaf(wa, va[k].x, wb * vb[k].x), fmaf(wa, va[k].y, wb * vb[k].y),
                             fmaf(wa, va[k].z, wb * vb[k].z), fmaf(wa, va[k].w, wb * vb[k].w));
      }
    } else {
      // lane j of a chunk of 32 pieces holds piece j0 + j
      for (int j0 = 0; j0 < np; j0 += 32) {
        if (j0 + lane < np) {
          const size_t e = entry(j0 + lane);
#pragma unroll
          for (int k = 0; k < kMergeRows; ++k) {
            const float2 ml = wml[e * kRows + row0 + k];
            if (ml.y > 0.f) M[k] = fmaxf(M[k], ml.x);
          }
        }
      }
#pragma unroll
      for (int k = 0; k < kMergeRows; ++k)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) M[k] = fmaxf(M[k], __shfl_xor_sync(full, M[k], o));
      for (int j0 = 0; j0 < np; j0 += 32) {
        float wj[kMergeRows];
#pragma unroll
        for (int k = 0; k < kMergeRows; ++k) wj[k] = 0.f;
        if (j0 + lane < np) {
          const size_t e = entry(j0 + lane);
#pragma unroll
          for (int k = 0; k < kMergeRows; ++k) {
            const float2 ml = wml[e * kRows + row0 + k];
            if (ml.y > 0.f && M[k] != -INFINITY) {
              wj[k] = exp2f(ml.x - M[k]);
              L[k] = fmaf(wj[k], ml.y, L[k]);
            }
          }
        }
        const int cnt = min(32, np - j0);
        for (int i = 0; i < cnt; ++i) {
          const float4* o = reinterpret_cast<const float4*>(p.ws + (entry(j0 + i) * kRows + row0) * kD);
          float4 v[kMergeRows];
#pragma unroll
          for (int k = 0; k < kMergeRows; ++k) v[k] = o[k * (kD / 4) + lane];
#pragma unroll
          for (int k = 0; k < kMergeRows; ++k) {
            const float w = __shfl_sync(full, wj[k], i);
            acc[k].x = fmaf(w, v[k].x, acc[k].x);
            acc[k].y = fmaf(w, v[k].y, acc[k].y);
            acc[k].z = fmaf(w, v[k].z, acc[k].z);
            acc[k].w = fmaf(w, v[k].w, acc[k].w);
          }
        }
      }
#pragma unroll
      for (int k = 0; k < kMergeRows; ++k)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) L[k] += __shfl_xor_sync(full, L[k], o);
    }
#pragma unroll
    for (int k = 0; k < kMergeRows; ++k) {
      const int row = row0 + k, s = x * p.s_blk + row / p.g;
      if (s < p.S) {
        const float inv = L[k] > 0.f ? 1.f / L[k] : 0.f;
        const int h = kvh * p.g + row % p.g;
        uint2 w2;
        w2.x = pack_bf16x2(acc[k].x * inv, acc[k].y * inv);
        w2.y = pack_bf16x2(acc[k].z * inv, acc[k].w * inv);
        reinterpret_cast<uint2*>(p.out + ((static_cast<size_t>(b) * p.S + s) * p.Hq + h) * kD)[lane] = w2;
      }
    }
  }
  pdl_launch_next();
}

}  // namespace

int tc256_splits(int Bt, int Hkv, int rb, long long max_tiles, int num_sms) {
  if (rb != 2) return 0;
  const long long units = static_cast<long long>(Bt) * Hkv;
  if (units >= num_sms) return 1;
  // short units (under 16 key tiles) that would need splitting stay with
  // the one-row-block kernel, whose splits merge in a cluster (at 512 keys
  // it was ~3.5% faster per step)
  if (max_tiles < 16) return 0;
  // Fewer units than SMs: split each unit's key tiles into ns ranges (at
  // least two tiles each).  A CTA walks ceil(units ns / SMs) items, each
  // costing its tiles plus a fixed ~14 tiles (Q, the pipeline refill, the
  // partial write); ns minimises that product (measured at 8 sequences x 8
  // KV heads: ~0.9 us per tile, ~13 us per item).
  const long long kItemCost = 14;
  const long long ns_max = std::min<long long>(64, std::max<long long>(1, max_tiles / 2));
  long long best = 1, best_cost = -1;
  for (long long ns = 1; ns <= ns_max; ++ns) {
    const long long per_cta = (units * ns + num_sms - 1) / num_sms;
    const long long cost = per_cta * ((max_tiles + ns - 1) / ns + kItemCost);
    if (best_cost < 0 || cost < best_cost) {
      best = ns;
      best_cost = cost;
    }
  }
  return static_cast<int>(best);
}

int tc256_streamk(int Bt, int Hkv, long long max_tiles, int nsplit, int num_sms) {
  const long long units = static_cast<long long>(Bt) * Hkv;
  if (nsplit < 1 || Bt > kMaxStreamK || units * max_tiles >= (1ll << 30)) return 0;
  // Costs in key tiles of the busiest CTA, T = max_tiles.  The walk of
  // tc256_splits (whole units when nsplit is 1): ceil(units ns / SMs) items
  // of ceil(T / ns) tiles plus ~14 each (Q, the pipeline refill, the
  // output).  Equal runs of W = ceil(units T / SMs) tiles: a run overlaps
  // at most ceil(W / T) + 1 units, ~14 each again, and the merge launch
  // costs ~10 more.  Stream-K is taken when it saves at least 3% (measured
  // at 32 drafts, 32 sequences: 512 keys 42.9 us whole against 67.3 us in
  // runs, 8192 keys 260 against 256 us, 32768 keys 955 against 849 us).
  const long long kItemCost = 14, kMergeCost = 10;
  const long long T = max_tiles, ns = nsplit;
  const long long ranges = (units * ns + num_sms - 1) / num_sms * ((T + ns - 1) / ns + kItemCost);
  const long long W = (units * T + num_sms - 1) / num_sms;
  const long long runs = W + ((W + T - 1) / T + 1) * kItemCost + kMergeCost;
  return runs * 100 < ranges * 97 ? 1 : 0;
}

size_t tc256_streamk_bytes(int num_sms) {
  // two partial pieces per CTA, two row blocks each: O and (m, l) of 128
  // rows; then a 16-byte record per run boundary
  return static_cast<size_t>(num_sms) * (4 * kRows * (kD + 2) * sizeof(float) + sizeof(int4));
}

cudaError_t launch_attention_tc256(const AttnTcArgs& a, const AttnTcPlan& pl, EncodeTiledFn encode,
                                   cudaStream_t stream) {
  const int S = 2 * a.gamma, g = a.Hq / a.Hkv, s_blk = pl.s_blk;
  CUtensorMap tq, tkn, tvn, tkc, tvc;
  {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.Hq),
                                static_cast<cuuint64_t>(a.Bt) * S};
    const cuuint64_t strides[2] = {kD * 2ull, static_cast<cuuint64_t>(a.Hq) * kD * 2ull};
    const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(g), static_cast<cuuint32_t>(s_blk)};
    if (!make_bf16_map(encode, &tq, a.q, 3, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kD), static_cast<cuuint64_t>(a.Hkv),
                                static_cast<cuuint64_t>(a.Bt) * S};
    const cuuint64_t strides[2] = {kD * 2ull, static_cast<cuuint64_t>(a.Hkv) * kD * 2ull};
    const cuuint32_t box[3] = {64u, 1u, static_cast<cuuint32_t>(S)};
    if (!make_bf16_map(encode, &tkn, a.k_new, 3, dims, strides, box)) return cudaErrorInvalidValue;
    if (!make_bf16_map(encode, &tvn, a.v_new, 3, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(kD),
                                std::max<cuuint64_t>(1, static_cast<cuuint64_t>(a.num_pages) * a.Hkv * a.page_size)};
    const cuuint64_t strides[1] = {kD * 2ull};
    const cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(std::min(a.page_size, kTile))};
    if (!make_bf16_map(encode, &tkc, a.k_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
    if (!make_bf16_map(encode, &tvc, a.v_cache, 2, dims, strides, box)) return cudaErrorInvalidValue;
  }
  Tc256Params p{};
  p.block_table = a.block_table;
  p.prefix_len = a.prefix_len;
  p.tau = a.tau;
  p.section = a.section;
  p.rope_pos = a.rope_pos;
  p.rope = a.rope;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.err_word = a.err_word;
  p.max_pages = a.max_pages;
  p.page_size = a.page_size;
  p.num_pages = a.num_pages;
  p.Bt = a.Bt;
  p.S = S;
  p.Hq = a.Hq;
  p.Hkv = a.Hkv;
  p.g = g;
  p.s_blk = s_blk;
  p.units = a.Bt * a.Hkv;
  p.nsplit = pl.nsplit;
  p.items = p.units * pl.nsplit;
  p.streamk = pl.streamk;
  p.ws = static_cast<float*>(a.workspace);
  p.sort = (!pl.streamk && a.Bt <= kMaxSort) ? 1 : 0;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.wait_ns = a.fault.wait_ns ? a.fault.wait_ns : kWaitLimitNs;
  p.extra_p = a.fault.extra;
  {
    // the shared-memory attribute, once per device (function attributes
    // apply to the current device only)
    static std::mutex mu;
    static bool done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(mu);
    if (!done[dev]) {
      e = cudaFuncSetAttribute(attention_tc256_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem_bytes()));
      if (e != cudaSuccess) return e;
      done[dev] = true;
    }
  }
  const int grid = pl.streamk ? pl.num_sms : std::min(p.items, pl.num_sms);
  p.ctas = grid;
  cudaError_t e = launch_overlapped(attention_tc256_kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads),
                                    smem_bytes(), stream, 1u, tq, tkn, tvn, tkc, tvc, p);
  if (e != cudaSuccess) return e;
  if (pl.streamk)
    return grid > 1 ? launch_overlapped(streamk_combine_kernel, dim3(static_cast<unsigned>(grid - 1), 2u, kRows / 16),
                                        dim3(128), 0, stream, 1u, p)
                    : cudaSuccess;
  if (pl.nsplit == 1) return e;
  return launch_attention_combine(a, pl, stream);
}

}  // namespace simsd
