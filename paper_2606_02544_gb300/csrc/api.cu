// api.cu -- the extern "C" entry points of libsimsd.so (declared in
// include/simsd.h): argument checks on the host, then kernel launches on the
// caller's stream.  No call allocates memory or synchronises, except
// simsd_check_error.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "../../include/simsd.h"
#include "kernels.h"

namespace {

thread_local char g_last_error[256] = "";

// Planted wait expiry armed by simsd_debug_expire_next_wait for the next
// launch of one kernel on this thread (index: SIMSD_DEBUG_WAIT_*).
thread_local simsd::WaitFault g_armed[3];

simsd::WaitFault take_armed(int which) {
  const simsd::WaitFault f = g_armed[which];
  g_armed[which] = simsd::WaitFault{};
  return f;
}

int cuda_fail(cudaError_t e, const char* where) {
  std::snprintf(g_last_error, sizeof(g_last_error), "%s: %s", where, cudaGetErrorString(e));
  return SIMSD_ERR_CUDA;
}

int arg_fail(const char* what) {
  std::snprintf(g_last_error, sizeof(g_last_error), "invalid argument: %s", what);
  return SIMSD_ERR_INVALID_ARG;
}

int unsupported(const char* what) {
  std::snprintf(g_last_error, sizeof(g_last_error), "unsupported: %s", what);
  return SIMSD_ERR_UNSUPPORTED;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct DeviceInfo {
  int num_sms = 0;
  int major = 0, minor = 0;
};

// Per-device properties, queried once per device.
int device_info(DeviceInfo* out) {
  static std::mutex mu;
  static DeviceInfo cache[64];
  static bool have[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) return unsupported("device ordinal >= 64");
  std::lock_guard<std::mutex> lk(mu);
  if (!have[dev]) {
    DeviceInfo d;
    if ((e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    cache[dev] = d;
    have[dev] = true;
  }
  *out = cache[dev];
  return SIMSD_OK;
}

int require_sm103(DeviceInfo* info) {
  int rc = device_info(info);
  if (rc != SIMSD_OK) return rc;
  if (info->major != 10 || info->minor != 3) return unsupported("this library is built for sm_103a only");
  return SIMSD_OK;
}

simsd::EncodeTiledFn encoder() {
  static simsd::EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<simsd::EncodeTiledFn>(p);
  });
  return fn;
}

cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

// Shared body of the two attention entry points.  static_scratch: the
// split partials go to the library's static array instead of the caller's
// workspace.
int verify_attention_impl(int dtype, const void* q, const void* k_new, const void* v_new, const void* k_cache,
                          const void* v_cache, int num_pages, const int32_t* block_table, int max_pages,
                          int page_size, const int32_t* prefix_len, const int32_t* tau, const uint8_t* section,
                          const int32_t* rope_pos, float rope_theta, int Bt, int gamma, int Hq, int Hkv, int d,
                          float softmax_scale, void* out, void* workspace, size_t workspace_bytes,
                          bool static_scratch, const simsd::WaitFault& fault, int32_t* err_word, void* stream) {
  if (Bt < 0) return arg_fail("Bt < 0");
  if (gamma < 1 || gamma > 32) return arg_fail("gamma must be in [1, 32]");
  if (Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0) return arg_fail("Hq must be a positive multiple of Hkv");
  if (num_pages < 0 || max_pages < 0) return arg_fail("negative page count");
  if (page_size < 8 || !((page_size % 64 == 0) || (64 % page_size == 0)))
    return unsupported("page_size must be a multiple of 64 or a divisor of 64 (>= 8)");
  if (rope_pos && (!(rope_theta > 0.f) || std::isinf(rope_theta)))
    return arg_fail("rope_theta must be positive and finite when rope_pos is given");
  if (!(softmax_scale >= 0.f) || std::isinf(softmax_scale)) return arg_fail("softmax_scale");
  if (Bt == 0) return SIMSD_OK;
  if (!q || !k_new || !v_new || !prefix_len || !tau || !section || !out) return arg_fail("null pointer");
  if (max_pages > 0 && (!block_table || !k_cache || !v_cache || num_pages == 0))
    return arg_fail("null cache or block table");
  if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out) ||
      (k_cache && !aligned16(k_cache)) || (v_cache && !aligned16(v_cache)))
    return arg_fail("tensor pointers must be 16-byte aligned");
  DeviceInfo info;
  int rc = require_sm103(&info);
  if (rc != SIMSD_OK) return rc;
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(d));
  cudaStream_t s = as_stream(stream);
  if (dtype == SIMSD_F32) {
    // the fp32 path uses no scratch
    if (d != 64 && d != 128) return unsupported("fp32 path needs d in {64, 128}");
    simsd::AttnF32Args a{};
    a.q = static_cast<const float*>(q);
    a.k_new = static_cast<const float*>(k_new);
    a.v_new = static_cast<const float*>(v_new);
    a.k_cache = static_cast<const float*>(k_cache);
    a.v_cache = static_cast<const float*>(v_cache);
    a.block_table = block_table;
    a.prefix_len = prefix_len;
    a.tau = tau;
    a.section = section;
    a.rope_pos = rope_pos;
    if (rope_pos) a.rope = simsd::make_rope_table(rope_theta, d);
    a.out = static_cast<float*>(out);
    a.err_word = err_word;
    a.num_pages = num_pages;
    a.max_pages = max_pages;
    a.page_size = page_size;
    a.Bt = Bt;
    a.gamma = gamma;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.d = d;
    a.scale = scale;
    cudaError_t e = simsd::launch_attention_f32(a, s);
    return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "attention_f32 launch");
  }
  if (dtype != SIMSD_BF16) return unsupported("dtype");
  if (d != 128) return unsupported("bf16 path needs d = 128");
  if (static_cast<long long>(num_pages) * Hkv * page_size >= (1ll << 31))
    return unsupported("page pool too large for 32-bit TMA row coordinates");
  if (static_cast<long long>(Bt) * 2 * gamma * Hq >= (1ll << 31)) return unsupported("too many query rows");
  simsd::AttnTcPlan plan;
  if (!simsd::plan_attention_tc(Bt, gamma, Hq, Hkv, max_pages, page_size, info.num_sms, &plan, !static_scratch))
    return unsupported("query rows per KV head: need 2*gamma*Hq/Hkv <= 128 or 128 % (Hq/Hkv) == 0");
  if (static_scratch) {
    // (stream-K runs are not used here: their partials would outgrow the array)
    if (plan.ws_bytes > simsd::noalloc_scratch_capacity()) {
      std::snprintf(g_last_error, sizeof(g_last_error),
                    "unsupported: these sizes need %zu bytes of scratch, more than the %zu-byte static array; "
                    "use simsd_verify_attention with a caller workspace",
                    plan.ws_bytes, simsd::noalloc_scratch_capacity());
      return SIMSD_ERR_UNSUPPORTED;
    }
    workspace = nullptr;
    if (plan.ws_bytes > 0) {
      cudaError_t e = simsd::noalloc_scratch_pointer(&workspace);
      if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the static scratch");
    }
  } else if (plan.ws_bytes > 0 && (!workspace || workspace_bytes < plan.ws_bytes || !aligned16(workspace))) {
    return arg_fail("workspace smaller than simsd_verify_workspace_bytes()");
  }
  simsd::EncodeTiledFn enc = encoder();
  if (!enc) return cuda_fail(cudaErrorNotSupported, "cuTensorMapEncodeTiled entry point");
  simsd::AttnTcArgs a{};
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  // a pool with no pages is still described by a valid (never read) map
  a.k_cache = k_cache ? k_cache : q;
  a.v_cache = v_cache ? v_cache : q;
  a.block_table = block_table;
  a.prefix_len = prefix_len;
  a.tau = tau;
  a.section = section;
  a.rope_pos = rope_pos;
  if (rope_pos) a.rope = simsd::make_rope_table(rope_theta, d);
  a.out = out;
  a.workspace = workspace;
  a.err_word = err_word;
  a.num_pages = num_pages > 0 ? num_pages : 1;
  a.max_pages = max_pages;
  a.page_size = page_size;
  a.Bt = Bt;
  a.gamma = gamma;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.scale = scale;
  a.fault = fault;
  if (num_pages == 0) {
    a.max_pages = 0;
    a.num_pages = 0;
  }
  cudaError_t e = simsd::launch_attention_tc(a, plan, enc, s);
  return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "attention_tc launch");
}

}  // namespace

namespace simsd {

RopeTable make_rope_table(double theta, int d) {
  RopeTable t{};
  for (int i = 0; i < d / 2 && i < 64; ++i) {
    const double f = std::pow(theta, -2.0 * i / d);
    const float hi = static_cast<float>(f);
    t.f[i] = make_float2(hi, static_cast<float>(f - static_cast<double>(hi)));
  }
  return t;
}

}  // namespace simsd

extern "C" {

int simsd_version(void) { return 1 * 10000 + 1 * 100 + 0; }

const char* simsd_last_error(void) { return g_last_error; }

int simsd_build_mask(const int32_t* step_map, const int32_t* prefix_len, int Bt, int gamma, int32_t* tau,
                     uint8_t* section, int32_t* rope_pos, uint64_t* mask_bits, int32_t* err_word, void* stream) {
  if (Bt < 0) return arg_fail("Bt < 0");
  if (gamma < 1 || gamma > 32) return arg_fail("gamma must be in [1, 32]");
  if (Bt == 0) return SIMSD_OK;
  if (!prefix_len || !tau || !section || !rope_pos) return arg_fail("null pointer");
  DeviceInfo info;
  int rc = require_sm103(&info);
  if (rc != SIMSD_OK) return rc;
  cudaError_t e = simsd::launch_build_mask(step_map, prefix_len, Bt, gamma, tau, section, rope_pos, mask_bits,
                                           err_word, as_stream(stream));
  return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "build_mask launch");
}

size_t simsd_verify_workspace_bytes(int dtype, int Bt, int gamma, int Hq, int Hkv, int d, int max_pages,
                                    int page_size) {
  if (dtype != SIMSD_BF16 || Bt <= 0 || gamma < 1 || gamma > 32 || Hkv <= 0 || Hq % Hkv != 0 || d != 128 ||
      max_pages < 0 || page_size <= 0)
    return 0;
  DeviceInfo info;
  if (device_info(&info) != SIMSD_OK) return 0;
  simsd::AttnTcPlan plan;
  if (!simsd::plan_attention_tc(Bt, gamma, Hq, Hkv, max_pages, page_size, info.num_sms, &plan)) return 0;
  return plan.ws_bytes;
}

int simsd_verify_attention(int dtype, const void* q, const void* k_new, const void* v_new, const void* k_cache,
                           const void* v_cache, int num_pages, const int32_t* block_table, int max_pages,
                           int page_size, const int32_t* prefix_len, const int32_t* tau, const uint8_t* section,
                           const int32_t* rope_pos, float rope_theta, int Bt, int gamma, int Hq, int Hkv, int d,
                           float softmax_scale, void* out, void* workspace, size_t workspace_bytes,
                           int32_t* err_word, void* stream) {
  // an armed wait expiry is consumed by this call whatever its outcome
  const simsd::WaitFault fault = take_armed(SIMSD_DEBUG_WAIT_ATTENTION);
  return verify_attention_impl(dtype, q, k_new, v_new, k_cache, v_cache, num_pages, block_table, max_pages,
                               page_size, prefix_len, tau, section, rope_pos, rope_theta, Bt, gamma, Hq, Hkv, d,
                               softmax_scale, out, workspace, workspace_bytes, false, fault, err_word, stream);
}

int simsd_verify_attention_noalloc(int dtype, const void* q, const void* k_new, const void* v_new,
                                   const void* k_cache, const void* v_cache, int num_pages,
                                   const int32_t* block_table, int max_pages, int page_size,
                                   const int32_t* prefix_len, const int32_t* tau, const uint8_t* section,
                                   const int32_t* rope_pos, float rope_theta, int Bt, int gamma, int Hq, int Hkv,
                                   int d, float softmax_scale, void* out, int32_t* err_word, void* stream) {
  return verify_attention_impl(dtype, q, k_new, v_new, k_cache, v_cache, num_pages, block_table, max_pages,
                               page_size, prefix_len, tau, section, rope_pos, rope_theta, Bt, gamma, Hq, Hkv, d,
                               softmax_scale, out, nullptr, 0, true, simsd::WaitFault{}, err_word, stream);
}

namespace {

// Greedy acceptance: the cluster kernel, or with a workspace (ws_ok) the
// split over many CTAs when the shape takes it.
int accept_impl(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab, int32_t* accepted_len,
                int32_t* out_tokens, int32_t* row_argmax, bool ws_ok, void* workspace, size_t workspace_bytes,
                int32_t* err_word, void* stream) {
  // an armed wait expiry is consumed by this call whatever its outcome
  const simsd::WaitFault fault = take_armed(SIMSD_DEBUG_WAIT_ACCEPT);
  if (Bt < 0) return arg_fail("Bt < 0");
  if (gamma < 1 || gamma > 32) return arg_fail("gamma must be in [1, 32]");
  if (vocab < 1 || vocab > (1 << 28)) return arg_fail("vocab must be in [1, 2^28]");
  if (Bt == 0) return SIMSD_OK;
  if (!logits || !draft || !accepted_len || !out_tokens) return arg_fail("null pointer");
  DeviceInfo info;
  int rc = require_sm103(&info);
  if (rc != SIMSD_OK) return rc;
  const size_t need = ws_ok ? simsd::accept_workspace_bytes(Bt, gamma, vocab, info.num_sms) : 0;
  cudaError_t e;
  if (need > 0) {
    if (!workspace || workspace_bytes < need) return arg_fail("workspace smaller than simsd_accept_workspace_bytes()");
    if ((reinterpret_cast<uintptr_t>(workspace) & 7u) != 0) return arg_fail("workspace not 8-byte aligned");
    if (fault.extra) return unsupported("a planted wait expiry needs the cluster kernel (this path has no wait)");
    e = simsd::launch_accept_parts(logits, draft, Bt, gamma, vocab, accepted_len, out_tokens, row_argmax, workspace,
                                   err_word, info.num_sms, as_stream(stream));
  } else {
    e = simsd::launch_accept(logits, draft, Bt, gamma, vocab, accepted_len, out_tokens, row_argmax, err_word,
                             info.num_sms, as_stream(stream), fault);
    if (e == cudaErrorNotSupported && fault.extra)
      return unsupported("a planted wait expiry needs one CTA per sequence (a batch too large for clusters)");
  }
  return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "accept launch");
}

}  // namespace

int simsd_accept(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab, int32_t* accepted_len,
                 int32_t* out_tokens, int32_t* row_argmax, int32_t* err_word, void* stream) {
  return accept_impl(logits, draft, Bt, gamma, vocab, accepted_len, out_tokens, row_argmax, false, nullptr, 0,
                     err_word, stream);
}

size_t simsd_accept_workspace_bytes(int Bt, int gamma, int vocab) {
  if (Bt <= 0 || gamma < 1 || gamma > 32 || vocab < 1 || vocab > (1 << 28)) return 0;
  DeviceInfo info;
  if (require_sm103(&info) != SIMSD_OK) return 0;
  return simsd::accept_workspace_bytes(Bt, gamma, vocab, info.num_sms);
}

int simsd_accept_ws(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab, int32_t* accepted_len,
                    int32_t* out_tokens, int32_t* row_argmax, void* workspace, size_t workspace_bytes,
                    int32_t* err_word, void* stream) {
  return accept_impl(logits, draft, Bt, gamma, vocab, accepted_len, out_tokens, row_argmax, true, workspace,
                     workspace_bytes, err_word, stream);
}

namespace {

int accept_sampled_impl(const float* target_logits, const float* draft_logits, const int32_t* draft,
                        const float* u_accept, const float* u_sample, float temperature, int Bt, int gamma, int vocab,
                        int32_t* accepted_len, int32_t* out_tokens, bool ws_ok, void* workspace,
                        size_t workspace_bytes, int32_t* err_word, void* stream) {
  if (Bt < 0) return arg_fail("Bt < 0");
  if (gamma < 1 || gamma > 32) return arg_fail("gamma must be in [1, 32]");
  if (vocab < 1 || vocab > (1 << 24)) return arg_fail("vocab must be in [1, 2^24]");
  if (!(temperature > 0.f) || std::isinf(temperature)) return arg_fail("temperature must be positive and finite");
  if (Bt == 0) return SIMSD_OK;
  if (!target_logits || !draft_logits || !draft || !u_accept || !u_sample || !accepted_len || !out_tokens)
    return arg_fail("null pointer");
  DeviceInfo info;
  int rc = require_sm103(&info);
  if (rc != SIMSD_OK) return rc;
  const size_t need = ws_ok ? simsd::samp_workspace_bytes(Bt, gamma, vocab, info.num_sms) : 0;
  if (need > 0) {
    if (!workspace || workspace_bytes < need)
      return arg_fail("workspace smaller than simsd_accept_sampled_workspace_bytes()");
    if ((reinterpret_cast<uintptr_t>(workspace) & 7u) != 0) return arg_fail("workspace not 8-byte aligned");
  }
  cudaError_t e = simsd::launch_accept_sampled(target_logits, draft_logits, draft, u_accept, u_sample, temperature,
                                               Bt, gamma, vocab, accepted_len, out_tokens, err_word,
                                               as_stream(stream), need > 0 ? workspace : nullptr, info.num_sms);
  return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "accept_sampled launch");
}

}  // namespace

int simsd_accept_sampled(const float* target_logits, const float* draft_logits, const int32_t* draft,
                         const float* u_accept, const float* u_sample, float temperature, int Bt, int gamma,
                         int vocab, int32_t* accepted_len, int32_t* out_tokens, int32_t* err_word, void* stream) {
  return accept_sampled_impl(target_logits, draft_logits, draft, u_accept, u_sample, temperature, Bt, gamma, vocab,
                             accepted_len, out_tokens, false, nullptr, 0, err_word, stream);
}

size_t simsd_accept_sampled_workspace_bytes(int Bt, int gamma, int vocab) {
  if (Bt <= 0 || gamma < 1 || gamma > 32 || vocab < 1 || vocab > (1 << 24)) return 0;
  DeviceInfo info;
  if (require_sm103(&info) != SIMSD_OK) return 0;
  return simsd::samp_workspace_bytes(Bt, gamma, vocab, info.num_sms);
}

int simsd_plan_attention(int dtype, int Bt, int gamma, int Hq, int Hkv, int d, int max_pages, int page_size,
                         int num_sms, int32_t* plan, size_t* ws_bytes) {
  if (!plan || !ws_bytes || num_sms < 1) return arg_fail("null output or num_sms < 1");
  if (Bt < 0 || gamma < 1 || gamma > 32 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || max_pages < 0 ||
      page_size <= 0)
    return arg_fail("sizes out of range");
  for (int i = 0; i < 5; ++i) plan[i] = 0;
  *ws_bytes = 0;
  if (dtype == SIMSD_F32) {
    if (d != 64 && d != 128) return unsupported("fp32 path needs d = 64 or 128");
    plan[0] = 2;
    plan[1] = 1;
    plan[3] = 2 * gamma * (Hq / Hkv);
    return SIMSD_OK;
  }
  if (dtype != SIMSD_BF16) return unsupported("dtype");
  if (d != 128) return unsupported("bf16 path needs d = 128");
  simsd::AttnTcPlan pl;
  if (!simsd::plan_attention_tc(Bt > 0 ? Bt : 1, gamma, Hq, Hkv, max_pages, page_size, num_sms, &pl))
    return unsupported("query rows per KV head: need 2*gamma*Hq/Hkv <= 128 or 128 % (Hq/Hkv) == 0");
  plan[0] = pl.kind;
  plan[1] = pl.nsplit;
  plan[2] = pl.streamk;
  plan[3] = pl.rows_blk;
  plan[4] = pl.fuse;
  *ws_bytes = Bt > 0 ? pl.ws_bytes : 0;
  return SIMSD_OK;
}

int simsd_plan_accept(int sampled, int Bt, int gamma, int vocab, int num_sms, int32_t* parts, size_t* ws_bytes) {
  if (!parts || !ws_bytes || num_sms < 1) return arg_fail("null output or num_sms < 1");
  if (Bt < 0 || gamma < 1 || gamma > 32 || vocab < 1 || vocab > (sampled ? (1 << 24) : (1 << 28)))
    return arg_fail("sizes out of range");
  *parts = 0;
  *ws_bytes = 0;
  if (Bt == 0) return SIMSD_OK;
  *parts = sampled ? simsd::samp_parts(Bt, gamma, vocab, num_sms) : simsd::accept_parts(Bt, gamma, vocab, num_sms);
  *ws_bytes = sampled ? simsd::samp_workspace_bytes(Bt, gamma, vocab, num_sms)
                      : simsd::accept_workspace_bytes(Bt, gamma, vocab, num_sms);
  return SIMSD_OK;
}

int simsd_accept_sampled_ws(const float* target_logits, const float* draft_logits, const int32_t* draft,
                            const float* u_accept, const float* u_sample, float temperature, int Bt, int gamma,
                            int vocab, int32_t* accepted_len, int32_t* out_tokens, void* workspace,
                            size_t workspace_bytes, int32_t* err_word, void* stream) {
  return accept_sampled_impl(target_logits, draft_logits, draft, u_accept, u_sample, temperature, Bt, gamma, vocab,
                             accepted_len, out_tokens, true, workspace, workspace_bytes, err_word, stream);
}

int simsd_kv_commit(int dtype, const void* k_new, const void* v_new, int L, const int32_t* tau,
                    const uint8_t* section, const int32_t* rope_pos, float rope_theta, const int32_t* accepted_len,
                    void* k_cache, void* v_cache, int num_pages, const int32_t* block_table, int max_pages,
                    int page_size, int32_t* prefix_len, int Bt, int gamma, int Hkv, int d, int32_t* err_word,
                    void* stream) {
  if (Bt < 0 || L < 0) return arg_fail("Bt < 0 or L < 0");
  if (gamma < 1 || gamma > 32) return arg_fail("gamma must be in [1, 32]");
  if (Hkv <= 0 || page_size <= 0 || num_pages < 0 || max_pages < 0) return arg_fail("sizes");
  if (dtype != SIMSD_F32 && dtype != SIMSD_BF16) return unsupported("dtype");
  const int eb = dtype == SIMSD_F32 ? 4 : 2;
  if (d <= 0 || (d * eb) % 16 != 0) return arg_fail("d * element size must be a multiple of 16 bytes");
  if (rope_pos && (!(rope_theta > 0.f) || std::isinf(rope_theta) || d > 128 || d % 2 != 0))
    return arg_fail("rope needs a positive finite rope_theta and an even d <= 128");
  if (Bt == 0) return SIMSD_OK;
  if (!tau || !section || !accepted_len || !prefix_len) return arg_fail("null pointer");
  if (L > 0 && (!k_new || !v_new || !k_cache || !v_cache || !block_table)) return arg_fail("null pointer");
  if ((k_new && !aligned16(k_new)) || (v_new && !aligned16(v_new)) || (k_cache && !aligned16(k_cache)) ||
      (v_cache && !aligned16(v_cache)))
    return arg_fail("tensor pointers must be 16-byte aligned");
  DeviceInfo info;
  int rc = require_sm103(&info);
  if (rc != SIMSD_OK) return rc;
  const simsd::RopeTable table = rope_pos ? simsd::make_rope_table(rope_theta, d) : simsd::RopeTable{};
  cudaError_t e = simsd::launch_kv_commit(eb, k_new, v_new, L, tau, section, accepted_len, k_cache, v_cache,
                                          num_pages, block_table, max_pages, page_size, prefix_len, Bt, gamma, Hkv,
                                          d, rope_pos, table, err_word, as_stream(stream));
  return e == cudaSuccess ? SIMSD_OK : cuda_fail(e, "kv_commit launch");
}

int simsd_debug_expire_next_wait(int which, unsigned int limit_us) {
  if (which != SIMSD_DEBUG_WAIT_ATTENTION && which != SIMSD_DEBUG_WAIT_ACCEPT) return arg_fail("which");
  if (limit_us < 10 || limit_us > 1000000) return arg_fail("limit_us must be in [10, 10^6]");
  g_armed[which].extra = 1;
  g_armed[which].wait_ns = 1000ull * limit_us;
  return SIMSD_OK;
}

int simsd_check_error(const int32_t* err_word, int32_t* host_word, void* stream) {
  if (!err_word) return arg_fail("null error word");
  int32_t w = 0;
  cudaError_t e = cudaMemcpyAsync(&w, err_word, sizeof(w), cudaMemcpyDeviceToHost, as_stream(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "check_error");
  if (host_word) *host_word = w;
  return w ? SIMSD_ERR_DEVICE : SIMSD_OK;
}

}  // extern "C"
