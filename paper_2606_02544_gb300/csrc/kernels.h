// kernels.h -- internal launch functions behind the C ABI (not exported).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace simsd {

// Rotary embedding frequencies theta^(-2i/d), i < d/2 <= 64, each as an
// unevaluated sum f.x + f.y of two floats (rounded from double).
struct RopeTable {
  float2 f[64];
};
RopeTable make_rope_table(double theta, int d);

// A planted wait expiry for one launch (tests of failure detection): the
// kernel expects `extra` more arrivals than ever come on one of its
// barriers and its waits give up after wait_ns.  {0, 0}: normal launch.
struct WaitFault {
  uint32_t extra = 0;
  unsigned long long wait_ns = 0;
};

cudaError_t launch_build_mask(const int32_t* step_map, const int32_t* prefix_len, int Bt, int gamma, int32_t* tau,
                              uint8_t* section, int32_t* rope_pos, uint64_t* mask_bits, int32_t* err_word,
                              cudaStream_t stream);

// fault.extra > 0 is applied only when every sequence runs as a single
// CTA (no other CTA then writes into the waiting CTA's shared memory);
// otherwise cudaErrorNotSupported.
cudaError_t launch_accept(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab,
                          int32_t* accepted_len, int32_t* out_tokens, int32_t* row_argmax, int32_t* err_word,
                          int num_sms, cudaStream_t stream, const WaitFault& fault = WaitFault{});

// Few sequences with a caller workspace: each sequence's logits split over
// accept_parts() CTAs (0: the shape takes the cluster kernel), their
// per-row keys merged by a second launch.
int accept_parts(int Bt, int gamma, int vocab, int num_sms);
size_t accept_workspace_bytes(int Bt, int gamma, int vocab, int num_sms);
cudaError_t launch_accept_parts(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab,
                                int32_t* accepted_len, int32_t* out_tokens, int32_t* row_argmax, void* workspace,
                                int32_t* err_word, int num_sms, cudaStream_t stream);

// workspace (may be null): with samp_workspace_bytes() > 0 bytes, phase 1
// of few sequences is split over many CTAs (samp_part_kernel) first.
int samp_parts(int Bt, int gamma, int vocab, int num_sms);
size_t samp_workspace_bytes(int Bt, int gamma, int vocab, int num_sms);
cudaError_t launch_accept_sampled(const float* target_logits, const float* draft_logits, const int32_t* draft,
                                  const float* u_accept, const float* u_sample, float temperature, int Bt,
                                  int gamma, int vocab, int32_t* accepted_len, int32_t* out_tokens,
                                  int32_t* err_word, cudaStream_t stream, void* workspace, int num_sms);

cudaError_t launch_kv_commit(int elem_bytes, const void* k_new, const void* v_new, int L, const int32_t* tau,
                             const uint8_t* section, const int32_t* accepted_len, void* k_cache, void* v_cache,
                             int num_pages, const int32_t* block_table, int max_pages, int page_size,
                             int32_t* prefix_len, int Bt, int gamma, int Hkv, int d, const int32_t* rope_pos,
                             const RopeTable& rope, int32_t* err_word, cudaStream_t stream);

struct AttnF32Args {
  const float *q, *k_new, *v_new, *k_cache, *v_cache;
  const int32_t *block_table, *prefix_len, *tau;
  const uint8_t* section;
  const int32_t* rope_pos;  // null: inputs rotated already
  RopeTable rope;
  float* out;
  int32_t* err_word;
  int num_pages, max_pages, page_size, Bt, gamma, Hq, Hkv, d;
  float scale;
};
cudaError_t launch_attention_f32(const AttnF32Args& a, cudaStream_t stream);

// bf16 tensor-core path
struct AttnTcPlan {
  int nsplit;       // prefix splits per (sequence, KV head, row block)
  int rb;           // row blocks of 128 query rows
  int rows_blk;     // query rows per row block (<= 128)
  int s_blk;        // slots per row block
  int sort;         // more CTAs than resident slots: longest prefix first
  int slots;        // CTAs resident at once (SMs x CTAs per SM)
  int fuse;         // 2..8 splits merge in place (cluster per unit), no workspace
  int kind;         // 0: one row block per CTA; 1: 256-row units, one persistent CTA per SM
  int streamk;      // kind 1: equal runs of the key tiles of all units per CTA, cut units merged after
  int num_sms;
  size_t ws_bytes;  // workspace bytes for the split partials (0 if nsplit == 1)
};
// Returns false if the shape is not supported by the tensor-core kernel.
// allow_streamk = false keeps the 256-row kernel on whole units or ranges.
bool plan_attention_tc(int Bt, int gamma, int Hq, int Hkv, int max_pages, int page_size, int num_sms,
                       AttnTcPlan* plan, bool allow_streamk = true);

struct AttnTcArgs {
  const void *q, *k_new, *v_new, *k_cache, *v_cache;
  const int32_t *block_table, *prefix_len, *tau;
  const uint8_t* section;
  const int32_t* rope_pos;  // null: inputs rotated already
  RopeTable rope;
  void* out;
  void* workspace;
  int32_t* err_word;
  int num_pages, max_pages, page_size, Bt, gamma, Hq, Hkv;
  float scale;
  WaitFault fault;
};
// The tensor-map encoder is the driver's cuTensorMapEncodeTiled.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
cudaError_t launch_attention_tc(const AttnTcArgs& a, const AttnTcPlan& plan, EncodeTiledFn encode,
                                cudaStream_t stream);

// bf16 tensor map with the 128-byte swizzle (shared by the attention kernels)
bool make_bf16_map(EncodeTiledFn encode, CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims,
                   const cuuint64_t* strides, const cuuint32_t* box);

// 256-row units (two row blocks per KV head) on one persistent CTA per SM.
// tc256_splits: 0 if the kernel does not take the shape (not two row
// blocks, or fewer units than SMs with under 16 key tiles each), else the
// key-tile ranges per unit (1 when there are at least as many units as SMs).
int tc256_splits(int Bt, int Hkv, int rb, long long max_tiles, int num_sms);
// 1 when the kernel walks stream-K runs instead of the nsplit ranges (or
// whole units) that tc256_splits chose: Bt <= 255 and a cost model in key
// tiles favours equal runs by at least 3%; its partial workspace is
// tc256_streamk_bytes.
int tc256_streamk(int Bt, int Hkv, long long max_tiles, int nsplit, int num_sms);
size_t tc256_streamk_bytes(int num_sms);
cudaError_t launch_attention_tc256(const AttnTcArgs& a, const AttnTcPlan& pl, EncodeTiledFn encode,
                                   cudaStream_t stream);
// Merge of split partials (workspace layout of the plan) into the output.
cudaError_t launch_attention_combine(const AttnTcArgs& a, const AttnTcPlan& pl, cudaStream_t stream);

// Static device scratch of simsd_verify_attention_noalloc.
size_t noalloc_scratch_capacity();
cudaError_t noalloc_scratch_pointer(void** out);

}  // namespace simsd
