/*
 * simsd.h -- C ABI of libsimsd.so: the verification forward of SimSD
 * speculative decoding for block-diffusion language models, on one GB300
 * (sm_103a).
 *
 * Paper: "SimSD: Simple Speculative Decoding in Diffusion Language Models".
 * One speculative step drafts gamma tokens, then the target verifies them in
 * a single forward pass over a paired layout: a data section D holding the
 * drafted (reference) tokens and a mask section D~ of prediction slots
 * (Sec. 3.1 "Input Layout Prepare", Sec. 3.2 "Target Model Verification").
 * A token-level temporal mask, Eq. (1), decides what each slot sees; the
 * prefix (prompt and earlier blocks) is read from a KV cache (Sec. 3.3).
 * The drafts are accepted along the draft order up to the first rejection
 * (Sec. 3.2, Eq. (2)), and the accepted drafts' K/V are appended to the
 * cache.
 *
 * Conventions shared by every call
 *   - Slot layout of one sequence: S = 2*gamma slots; slot k in [0,gamma)
 *     is the data slot D_k, slot gamma+k is the mask slot D~_k of the same
 *     block position k.  Row r of the acceptance logits and entry r of the
 *     draft array belong to the draft with temporal label tau = r+1.
 *   - Every pointer is caller-owned device memory unless stated otherwise;
 *     the library keeps no allocation of its own.  Arrays are dense,
 *     row-major, 16-byte aligned.
 *   - Every compute call is asynchronous on `stream` (a cudaStream_t passed
 *     as void*; NULL = the legacy default stream) and never synchronises.
 *   - Every call returns one of the SIMSD_* status codes.  Argument errors
 *     are detected on the host before anything is launched.  Errors that
 *     depend on device data (a bad step map, prefix length, page id, draft
 *     id or accepted length) are OR-ed into the caller's int32 error word
 *     (may be NULL) as SIMSD_EW_* bits, and the affected outputs are
 *     defined below; read the word with simsd_check_error.
 *   - dtype selects the storage and compute type of Q/K/V/O:
 *     SIMSD_BF16 (tensor cores, fp32 accumulation and softmax) or
 *     SIMSD_F32 (CUDA cores, fp32 throughout).
 */
#ifndef SIMSD_H_
#define SIMSD_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SIMSD_API __attribute__((visibility("default")))
#else
#define SIMSD_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* status codes */
#define SIMSD_OK 0
#define SIMSD_ERR_INVALID_ARG 1 /* null pointer, bad size, misaligned pointer */
#define SIMSD_ERR_UNSUPPORTED 2 /* dtype, head size or device not supported */
#define SIMSD_ERR_CUDA 3        /* a CUDA call failed; see simsd_last_error() */
#define SIMSD_ERR_DEVICE 4      /* simsd_check_error: the error word is non-zero */

/* dtypes */
#define SIMSD_F32 0
#define SIMSD_BF16 1

/* slot sections */
#define SIMSD_SECT_DATA 0 /* D: reference (drafted) token */
#define SIMSD_SECT_MASK 1 /* D~: prediction slot */
#define SIMSD_SECT_PAD 255 /* padding: row outputs zero, column never visible */

/* step-map codes besides the drafted labels 1..gamma and 0 (padding).
 * Sec. 3.2 verifies only the drafted positions of a block and has the target
 * complete the block itself when fewer than gamma positions remain; these
 * codes put the block's other positions into the same layout. */
#define SIMSD_STEP_UNDRAFTED (-1) /* stays [MASK]: mask slot only, tau = gamma+1 */
#define SIMSD_STEP_DECODED (-2)   /* decoded earlier in the block: data slot only, tau = 0 */

/* device error-word bits */
#define SIMSD_EW_STEP_MAP 1u    /* step map entry outside the codes above, or a repeated label */
#define SIMSD_EW_PREFIX_LEN 2u  /* prefix length < 0 or beyond the block table */
#define SIMSD_EW_PAGE 4u        /* a needed page id is outside [0, num_pages) */
#define SIMSD_EW_DRAFT 8u       /* a draft id is outside [0, vocab) */
#define SIMSD_EW_TIMEOUT 16u    /* a bounded on-device wait expired */
#define SIMSD_EW_ACCEPT_LEN 32u /* an accepted length is outside [0, gamma] */

/*
 * simsd_build_mask -- per-slot metadata of the verification input.
 * Sec. 3.1 "Temporal Attention Mask" and Eq. (1); "Position Encoding
 * Alignment" (RoPE copy); Sec. 3.2 (the slot of the r-th draft gets tau=r).
 *
 *   step_map   [Bt][gamma] int32: mu_k in 1..gamma for a drafted position
 *              (distinct labels), 0 for padding, SIMSD_STEP_UNDRAFTED or
 *              SIMSD_STEP_DECODED; NULL means the identity mu_k = k+1.  A
 *              map of undrafted and decoded entries only is the target's own
 *              block decoding: every real slot sees every other.
 *   prefix_len [Bt] int32, cached prefix length n_b.
 *   tau        [Bt][2gamma] int32 out: tau of D_k and D~_k is mu_k for a
 *              drafted position; gamma+1 for an undrafted mask slot, 0 for
 *              a decoded data slot and for padding.
 *   section    [Bt][2gamma] uint8 out: SIMSD_SECT_DATA / _MASK / _PAD.
 *   rope_pos   [Bt][2gamma] int32 out: n_b + k for both D_k and D~_k.
 *   mask_bits  [Bt][2gamma] uint64 out or NULL: bit j of row i is A_ij of
 *              Eq. (1) over the new slots (prefix columns are always visible).
 *   1 <= gamma <= 32.  A step map row with an entry outside these codes or a
 *   repeated label sets SIMSD_EW_STEP_MAP and turns every slot of that
 *   sequence into padding.
 */
SIMSD_API int simsd_build_mask(const int32_t* step_map, const int32_t* prefix_len, int Bt, int gamma,
                     int32_t* tau, uint8_t* section, int32_t* rope_pos, uint64_t* mask_bits,
                     int32_t* err_word, void* stream);

/*
 * simsd_verify_workspace_bytes -- bytes of scratch simsd_verify_attention
 * needs for these sizes on the current device: partial results of units
 * whose prefix is split over several CTAs (0 when nothing is split).
 * max_pages*page_size bounds every prefix length.  Shapes with 129..256
 * query rows per KV head (for example 32 drafts with 32/8 heads) and at
 * most 255 sequences whose units (sequence, KV head) would load the SMs
 * unevenly enough that equal shares pay for their extra pieces and merge
 * (long prefixes: a cost model in key tiles) give every CTA an equal share
 * of all key tiles and need about 266 KB per SM (40 MB on 152 SMs).
 */
SIMSD_API size_t simsd_verify_workspace_bytes(int dtype, int Bt, int gamma, int Hq, int Hkv, int d, int max_pages,
                                    int page_size);

/*
 * simsd_verify_attention -- the masked attention of the verification
 * forward (Sec. 3.2 "Target Model Verification"; Sec. 3.3 KV cache; cost of
 * the paired layout linear in the prefix, Eqs. (4)-(5)).
 *
 * For each sequence b, slot s and query head h (KV head h/(Hq/Hkv)):
 *   out[b][s][h] = softmax_j(scale * q.k_j) v_j over the keys j that the
 *   slot sees: all n_b cached prefix rows (visible to every response
 *   position) and each new slot t with A_st = 1 under Eq. (1), evaluated on
 *   the fly from tau/section.
 *
 *   q, out       [Bt][2gamma][Hq][d]   dtype
 *   k_new, v_new [Bt][2gamma][Hkv][d]  dtype (K/V of the new slots)
 *   k_cache, v_cache [num_pages][Hkv][page_size][d] dtype; prefix row p of
 *                sequence b is row p % page_size of page
 *                block_table[b][p / page_size].  Rows past n_b are never used.
 *   block_table  [Bt][max_pages] int32; entries past the prefix are ignored.
 *   tau, section [Bt][2gamma] from simsd_build_mask.
 *   rope_pos     NULL: q and k_new arrive rotated already.  Otherwise
 *                [Bt][2gamma] int32 positions, normally the RoPE-copy
 *                positions of simsd_build_mask (Sec. 3.1 "Position Encoding
 *                Alignment": D~_k reuses n_b + k of D_k); any other positions
 *                (e.g. the physical ones of the Table 4 ablation) may be
 *                given.  Each q row of slot s and each k_new row of slot t
 *                is then rotated at rope_pos[b][s] / rope_pos[b][t] before
 *                use (rotary embedding of RoFormer, rotate-half layout: the
 *                pair (x_i, x_{i+d/2}) turns by pos * rope_theta^(-2i/d));
 *                cached keys must be stored rotated.  Positions in [0, 2^20).
 *   rope_theta   RoPE base, > 0 when rope_pos is given (ignored otherwise).
 *   softmax_scale 0 selects 1/sqrt(d).
 *   workspace    scratch of simsd_verify_workspace_bytes() bytes (NULL if 0).
 * Supported: SIMSD_BF16 with d = 128 and Hq/Hkv*2gamma <= 128 or
 * 128 % (Hq/Hkv) == 0; SIMSD_F32 with d in {64, 128}; page_size a multiple
 * of 64 or a divisor of 64 (>= 8).
 * A sequence with a bad prefix length or page id gets all-zero output rows
 * and sets SIMSD_EW_PREFIX_LEN / SIMSD_EW_PAGE; padding rows are zero.
 */
SIMSD_API int simsd_verify_attention(int dtype, const void* q, const void* k_new, const void* v_new, const void* k_cache,
                           const void* v_cache, int num_pages, const int32_t* block_table, int max_pages,
                           int page_size, const int32_t* prefix_len, const int32_t* tau, const uint8_t* section,
                           const int32_t* rope_pos, float rope_theta, int Bt, int gamma, int Hq, int Hkv, int d,
                           float softmax_scale, void* out, void* workspace, size_t workspace_bytes,
                           int32_t* err_word, void* stream);

/*
 * simsd_verify_attention_noalloc -- simsd_verify_attention for callers that
 * cannot allocate device memory.  The paper has no counterpart; this is a
 * deployment convenience.
 *
 * Some callers cannot call cudaMalloc: an engine that hands all device
 * memory to its own pool at start-up and must not stall on the allocator
 * (cudaMalloc may synchronise the device), or a process under a memory
 * budget that forbids further device allocation.  This entry point takes
 * the same arguments minus the workspace: the scratch for the split
 * partials comes from a 12 MiB array in device memory that the library owns
 * (every GPU that loads libsimsd.so holds it until the process exits).  It
 * allocates nothing and calls no allocating routine.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) and keeps it for the life of the process; make
 *     that first call before any stream capture.  Because the address is
 *     kept, a cudaDeviceReset between calls is not supported.
 *   - Where simsd_verify_attention would give every CTA an equal share of
 *     all key tiles (scratch beyond 12 MiB), this entry point keeps units
 *     whole or splits them into equal ranges as it would without that
 *     option; results may differ from simsd_verify_attention's in the last
 *     bits (another order of summation).
 *   - Sizes whose scratch would exceed 12 MiB are rejected with
 *     SIMSD_ERR_UNSUPPORTED (see simsd_last_error); use
 *     simsd_verify_attention with a caller workspace for those.
 *   - All calls share the one array: calls that overlap on the GPU (on
 *     different streams, or different threads) race and give wrong results.
 *     Nothing in the array has to start at zero; each call overwrites what it
 *     reads.
 */
SIMSD_API int simsd_verify_attention_noalloc(int dtype, const void* q, const void* k_new, const void* v_new,
                                             const void* k_cache, const void* v_cache, int num_pages,
                                             const int32_t* block_table, int max_pages, int page_size,
                                             const int32_t* prefix_len, const int32_t* tau, const uint8_t* section,
                                             const int32_t* rope_pos, float rope_theta, int Bt, int gamma, int Hq,
                                             int Hkv, int d, float softmax_scale, void* out, int32_t* err_word,
                                             void* stream);

/*
 * simsd_accept -- greedy longest-prefix acceptance (Sec. 3.2, Eq. (2) with
 * temperature 0: accept the r-th draft iff it equals the target argmax).
 *
 *   logits      [Bt][gamma+1][vocab] fp32; row r scores the draft with
 *               tau = r+1, row gamma gives the next token when every draft
 *               is accepted.
 *   draft       [Bt][gamma] int32, in tau order.
 *   accepted_len[Bt] int32 out: a_b = leading drafts equal to their row argmax.
 *   out_tokens  [Bt][gamma+1] int32 out: the a_b accepted drafts, the argmax of
 *               row a_b (the target's token at the first rejected position),
 *               then -1.
 *   row_argmax  [Bt][gamma+1] int32 out or NULL.
 * Argmax ties go to the lowest index; NaN ranks above every number (the
 * first NaN wins); -0.0 equals +0.0.  A draft id outside [0, vocab) sets
 * SIMSD_EW_DRAFT and never matches.  No scratch memory is used.
 */
SIMSD_API int simsd_accept(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab, int32_t* accepted_len,
                 int32_t* out_tokens, int32_t* row_argmax, int32_t* err_word, void* stream);

/*
 * simsd_accept_workspace_bytes -- bytes of scratch simsd_accept_ws uses for
 * these sizes on the current device: 0 when the shape keeps the
 * scratch-free kernel of simsd_accept (more than num_SMs / 16 sequences, or
 * too few logits per sequence to split), else Bt x parts x (gamma+1) x 8.
 * Returns 0 for invalid sizes or when no sm_103a device is current.
 *
 * simsd_accept_ws -- simsd_accept (same arguments, outputs and error rules)
 * with a caller workspace.  For few sequences each sequence's logits are
 * split over more CTAs than one thread-block cluster holds: a first launch
 * writes one 64-bit argmax key per (sequence, part, row) to the workspace,
 * a second takes the maximum per row and walks the drafts.  The results are
 * identical to simsd_accept's (the argmax is a total order).
 *   workspace   device memory of at least simsd_accept_workspace_bytes()
 *               bytes, 8-byte aligned, owned by the caller; its contents
 *               need no initial value and are overwritten.  NULL/0 is
 *               accepted when that size is 0.
 * A workspace smaller than needed returns SIMSD_ERR_INVALID_ARG before any
 * launch.  Two calls that share a workspace must not overlap on the GPU.
 */
SIMSD_API size_t simsd_accept_workspace_bytes(int Bt, int gamma, int vocab);
SIMSD_API int simsd_accept_ws(const float* logits, const int32_t* draft, int Bt, int gamma, int vocab,
                              int32_t* accepted_len, int32_t* out_tokens, int32_t* row_argmax, void* workspace,
                              size_t workspace_bytes, int32_t* err_word, void* stream);

/*
 * simsd_accept_sampled -- stochastic acceptance (Sec. 3.2, Eq. (2)): with
 * p = softmax(logits / temperature), the r-th draft x_r is accepted iff
 * u_accept[b][r] < alpha_r = min(1, p_theta^(r)(x_r) / p_phi^(r)(x_r)),
 * along the draft order up to the first rejection.  The token at the first
 * rejected position a is drawn from the residual max(0, p_theta^(a) -
 * p_phi^(a)) renormalised (the rejection-sampling correction that keeps the
 * target distribution; p_theta^(a) itself if the residual is empty to float
 * precision); when every draft is accepted it is drawn from p_theta of row
 * gamma.  The draw is an inverse CDF: the smallest token whose cumulative
 * weight exceeds u_sample[b] times the total.
 *
 *   target_logits [Bt][gamma+1][vocab] fp32 (rows in tau order, as for
 *                 simsd_accept)
 *   draft_logits  [Bt][gamma][vocab] fp32: the draft model's logits that x_r
 *                 was drawn from
 *   draft         [Bt][gamma] int32, in tau order
 *   u_accept      [Bt][gamma] fp32 uniform draws in [0, 1)
 *   u_sample      [Bt] fp32 uniform draws in [0, 1)
 *   temperature   > 0;  vocab in [1, 2^24]
 *   accepted_len  [Bt] int32 out; out_tokens [Bt][gamma+1] int32 out: the
 *                 accepted drafts, the drawn token, then -1.
 * Probabilities are formed in fp32 from one pass over the logits (row a is
 * read once more); a draft id outside [0, vocab) sets SIMSD_EW_DRAFT and is
 * rejected.  No scratch memory is used.
 */
SIMSD_API int simsd_accept_sampled(const float* target_logits, const float* draft_logits, const int32_t* draft,
                                   const float* u_accept, const float* u_sample, float temperature, int Bt, int gamma,
                                   int vocab, int32_t* accepted_len, int32_t* out_tokens, int32_t* err_word,
                                   void* stream);

/*
 * simsd_accept_sampled_workspace_bytes / simsd_accept_sampled_ws -- the same
 * stochastic acceptance with a caller workspace.  For few sequences (at most
 * num_SMs / 16) holding at least 3 MiB of logits each (target and draft
 * rows), the log-sum-exp pass over every row is split over more CTAs than
 * one cluster per sequence holds: a first launch writes per-row (max, sum)
 * pairs of each part to the workspace; a second, over spans of row a,
 * merges them, forms alpha_r, sums the residual weights of its span and
 * lets the last CTA of each sequence draw the token by the same inverse CDF
 * as simsd_accept_sampled (per-sequence arrival counts in the workspace,
 * reset by the first launch of every call, so the workspace need not start
 * zeroed).
 * The workspace bytes are 0 for other shapes (then the call is
 * simsd_accept_sampled).  The pairs are merged in another order than the
 * cluster kernel's, so probabilities can differ in the last fp32 bits (the
 * same rounding as between any two summation orders).
 *   workspace  device memory of at least the returned bytes, 8-byte
 *              aligned, owned by the caller; no initial value needed.
 * A workspace smaller than needed returns SIMSD_ERR_INVALID_ARG before any
 * launch.  Two calls that share a workspace must not overlap on the GPU.
 */
SIMSD_API size_t simsd_accept_sampled_workspace_bytes(int Bt, int gamma, int vocab);
SIMSD_API int simsd_accept_sampled_ws(const float* target_logits, const float* draft_logits, const int32_t* draft,
                                      const float* u_accept, const float* u_sample, float temperature, int Bt,
                                      int gamma, int vocab, int32_t* accepted_len, int32_t* out_tokens,
                                      void* workspace, size_t workspace_bytes, int32_t* err_word, void* stream);

/*
 * simsd_kv_commit -- append the accepted drafts' K/V to the paged cache of
 * every layer (Sec. 3.2: accepted tokens are committed; Sec. 3.3: the cache
 * is reused by later steps).
 *
 * For each layer l, sequence b, r < accepted_len[b] and KV head: the
 * data-slot row whose tau is r+1 is copied to cache row prefix_len[b] + r;
 * then prefix_len[b] += accepted_len[b] (in place).
 *   k_new, v_new [L][Bt][2gamma][Hkv][d] dtype
 *   rope_pos     NULL: k_new is rotated already.  Otherwise [Bt][2gamma]
 *                positions as for simsd_verify_attention: the copied key of
 *                data slot k is rotated at rope_pos[b][k] (rope_theta > 0,
 *                even d <= 128) and rounded to dtype, so that the cache
 *                holds rotated keys; values are copied unchanged.
 *   k_cache, v_cache [L][num_pages][Hkv][page_size][d] dtype
 * A destination page outside the table or pool sets SIMSD_EW_PAGE and that
 * row is skipped; a missing source slot sets SIMSD_EW_STEP_MAP and that row
 * is skipped; a negative prefix length (SIMSD_EW_PREFIX_LEN) or an accepted
 * length outside [0, gamma] (SIMSD_EW_ACCEPT_LEN) leaves the sequence
 * untouched.
 */
SIMSD_API int simsd_kv_commit(int dtype, const void* k_new, const void* v_new, int L, const int32_t* tau,
                              const uint8_t* section, const int32_t* rope_pos, float rope_theta,
                              const int32_t* accepted_len, void* k_cache, void* v_cache, int num_pages,
                              const int32_t* block_table, int max_pages, int page_size, int32_t* prefix_len, int Bt,
                              int gamma, int Hkv, int d, int32_t* err_word, void* stream);

/*
 * simsd_check_error -- synchronises `stream`, copies the device error word
 * to *host_word (may be NULL) and returns SIMSD_ERR_DEVICE if it is
 * non-zero, SIMSD_OK otherwise.  The only call that synchronises.
 */
SIMSD_API int simsd_check_error(const int32_t* err_word, int32_t* host_word, void* stream);

/*
 * simsd_plan_attention -- the work decomposition simsd_verify_attention
 * takes for these sizes on a GPU with num_sms SMs (a diagnostic for host
 * code and tests; the paper has no counterpart).  Pure host arithmetic: no
 * device is touched, so it works without a GPU.
 *   plan[5]   int32, written: [0] kernel (0 bf16 one row block per CTA,
 *             1 bf16 256-row units, 2 fp32 CUDA cores); [1] key-tile
 *             ranges per unit (1: whole units); [2] 1 when the 256-row
 *             kernel walks stream-K runs; [3] query rows per row block;
 *             [4] 1 when 2..8 ranges merge in a cluster (no workspace).
 *   ws_bytes  written: the workspace simsd_verify_attention needs on such a
 *             device (what simsd_verify_workspace_bytes returns there).
 * Bt = 0 is accepted (an empty batch: no workspace).  Returns SIMSD_OK,
 * SIMSD_ERR_INVALID_ARG (null outputs, num_sms < 1, sizes out of range) or
 * SIMSD_ERR_UNSUPPORTED (a shape the kernels do not take).
 *
 * simsd_plan_accept -- the same for simsd_accept_ws (sampled = 0) and
 * simsd_accept_sampled_ws (sampled = 1): *parts CTAs per sequence for the
 * streaming pass (0: the cluster kernel, no workspace) and *ws_bytes of
 * workspace.  Returns SIMSD_OK or SIMSD_ERR_INVALID_ARG.
 */
SIMSD_API int simsd_plan_attention(int dtype, int Bt, int gamma, int Hq, int Hkv, int d, int max_pages,
                                   int page_size, int num_sms, int32_t* plan, size_t* ws_bytes);
SIMSD_API int simsd_plan_accept(int sampled, int Bt, int gamma, int vocab, int num_sms, int32_t* parts,
                                size_t* ws_bytes);

/*
 * simsd_debug_expire_next_wait -- test hook for failure detection; the paper
 * has no counterpart.  Arms the next bf16 simsd_verify_attention
 * (which = SIMSD_DEBUG_WAIT_ATTENTION) or simsd_accept
 * (which = SIMSD_DEBUG_WAIT_ACCEPT) call made by this host thread so that
 * one of its on-device barriers expects one arrival more than ever comes
 * and its waits give up after limit_us microseconds (10..10^6) instead of
 * 1 s.  The wait then runs out: the kernel sets SIMSD_EW_TIMEOUT, stops
 * every warp, waits (with the full limit) for its own copies and MMAs in
 * flight, frees its tensor memory and returns; the outputs of that call are
 * undefined and the context stays usable.  Attention: the softmax warps'
 * hand-off of P to the MMA issuer.  Acceptance: CTA 0's wait for the
 * per-CTA row maxima; armed only where every sequence runs as a single CTA
 * (a batch too large for one cluster per sequence to be resident), else the
 * call returns SIMSD_ERR_UNSUPPORTED.  The arm is consumed by that call.
 */
#define SIMSD_DEBUG_WAIT_ATTENTION 1
#define SIMSD_DEBUG_WAIT_ACCEPT 2
SIMSD_API int simsd_debug_expire_next_wait(int which, unsigned int limit_us);

/* Text of the last CUDA error seen by this thread (empty if none). */
SIMSD_API const char* simsd_last_error(void);

/* Library version: major*10000 + minor*100 + patch. */
SIMSD_API int simsd_version(void);

#ifdef __cplusplus
}
#endif
#endif /* SIMSD_H_ */
