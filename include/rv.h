/*
 * rv.h -- C ABI of the GB300 (sm_103a) verify step of Reflective Verification
 * (arXiv 2505.18629, "Think Before You Accept").
 *
 * The target model verifies gamma draft tokens x_1..x_gamma in ONE forward pass
 * over the packed block (Eq. 1, Alg. 1)
 *
 *     [x_1..x_gamma | template | x_1..x_gamma],   template = prompt || prefix,
 *
 * of length Lb = 2*gamma + R (R = |template|).  The first segment yields the
 * original logits o_1..o_{gamma+1}, the copy after the template yields the
 * reflective logits o_m..o_{m+gamma}, m = gamma + R + 1 (Alg. 1).  They are
 * fused as p_i = softmax((1-alpha) o_i + alpha o_{m+i-1}) (Eq. 2) and the
 * drafts are checked by exact match against the greedy choice of p_i (Alg. 2),
 * keeping the longest accepted prefix.
 *
 * Conventions for every entry point
 *   - Tensor arguments are DEVICE pointers to caller-owned, contiguous,
 *     row-major memory on the handle's device, unless the name ends in _host.
 *     bf16 tensors hold IEEE bfloat16 bit patterns; with RV_DTYPE_F32 the same
 *     arguments hold float32.  Ids and lengths are int32.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Calls only enqueue work on it: they never synchronize (except the
 *     functions documented as synchronous) and are safe to capture in a CUDA
 *     graph.
 *   - The handle owns only its scratch workspace (allocated once in rv_create).
 *     Calls that share a handle must be ordered on one stream.
 *   - Return 0 (RV_OK) on success or a negative RV_ERR_* code; the message is
 *     available from rv_last_error().  Arguments are validated on the host
 *     before anything is launched.  Values that live in device memory
 *     (ctx_lens, draft ids) are checked by the kernels: an out-of-range value
 *     is skipped (never dereferenced) and raises a bit in the device status
 *     word read by rv_read_status().  No kernel traps or asserts.
 */
#ifndef RV_H_
#define RV_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define RV_API __attribute__((visibility("default")))
#else
#define RV_API
#endif

/* ---- status codes ------------------------------------------------------- */
#define RV_OK 0
#define RV_ERR_INVALID_ARG (-1)     /* NULL pointer, bad enum, alpha not finite */
#define RV_ERR_SHAPE (-2)           /* sizes inconsistent with the config */
#define RV_ERR_CAPACITY (-3)        /* batch / gamma / template above the config maxima */
#define RV_ERR_CUDA (-4)            /* a CUDA runtime call or launch failed */
#define RV_ERR_NOT_IMPLEMENTED (-5) /* combination not built (e.g. head_dim) */
#define RV_ERR_UNSUPPORTED (-6)     /* device is not sm_103 / lacks resources */
#define RV_ERR_DEVICE (-7)          /* rv_read_status found a device-side error bit */

/* ---- device status bits (rv_read_status) -------------------------------- */
#define RV_DEV_CTX_RANGE 1u     /* ctx_len < 0 or ctx_len + Lb > max_ctx: sequence skipped */
#define RV_DEV_DRAFT_RANGE 2u   /* draft id outside [0, vocab): treated as rejected */
#define RV_DEV_TIMEOUT 4u       /* a pipeline wait in a kernel gave up (no hang) */

/* ---- data types ---------------------------------------------------------- */
#define RV_DTYPE_BF16 0         /* bf16 storage, fp32 accumulation (tensor cores) */
#define RV_DTYPE_F32 1          /* fp32 storage and accumulation (CUDA cores) */

/* ---- per-position scores written by rv_verify_head ---------------------- */
#define RV_NSCORES 7
#define RV_SCORE_LSE_ORIG 0     /* logsumexp_v o_i[v]                         */
#define RV_SCORE_LSE_REFL 1     /* logsumexp_v o_{m+i-1}[v]                   */
#define RV_SCORE_LSE_FUSED 2    /* logsumexp_v z_i[v], z_i = (1-a)o_i + a o'_i */
#define RV_SCORE_LOGP_FUSED 3   /* log p_i(x_i) = z_i[x_i] - lse_fused (NaN at i = gamma+1) */
#define RV_SCORE_LOGP_ORIG 4    /* o_i[x_i] - lse_orig                        */
#define RV_SCORE_LOGP_REFL 5    /* o'_i[x_i] - lse_refl                       */
#define RV_SCORE_ENT_ORIG 6     /* H(softmax(o_i)): entropy (nats) of the unfused original
                                   distribution, for the typical acceptance of Alg. 3 */

/* Acceptance rules (rv_set_acceptance). */
#define RV_ACCEPT_EXACT 0       /* exact match with the greedy choice (Alg. 2)               */
#define RV_ACCEPT_TYPICAL 1     /* entropy-based threshold of typical acceptance (Alg. 3)     */
#define RV_ACCEPT_SPECULATIVE 2 /* speculative sampling with residual resampling (Alg. 1)     */
#define RV_ACCEPT_SAMPLED 3     /* exact match with target tokens sampled at temperature T (Alg. 2) */
#define RV_ACCEPT_TYPICAL_SAMPLED 4 /* typical acceptance (Alg. 3), t ~ p_{n+1} at temperature T */

/* LM-head variants (rv_set_head_mode). */
#define RV_HEAD_FUSED_LOGITS 0  /* o_i and o_{m+i-1} from their own rows, fused (Eq. 2)      */
#define RV_HEAD_PREBLENDED 1    /* z_i = W b_i from the blended hidden state (linearity)      */
#define RV_HEAD_STANDARD 2      /* standard speculative verification: no reflection           */

/* Model / capacity description fixed at creation. */
typedef struct rv_config {
    int32_t hidden;       /* H: hidden size (multiple of 8)                     */
    int32_t vocab;        /* V: LM-head rows                                    */
    int32_t n_q_heads;    /* Hq                                                 */
    int32_t n_kv_heads;   /* Hkv (Hq % Hkv == 0; query head h uses h / (Hq/Hkv)) */
    int32_t head_dim;     /* D: 64 or 128 for bf16; multiple of 32, <= 256 for f32 */
    int32_t max_batch;    /* largest B of any call                               */
    int32_t max_gamma;    /* largest gamma                                        */
    int32_t max_template; /* largest R = |template|                               */
    int32_t max_ctx;      /* KV-cache capacity Cmax (positions per sequence)      */
    int32_t dtype;        /* RV_DTYPE_BF16 or RV_DTYPE_F32                        */
} rv_config;

typedef struct rv_handle rv_handle;

/* Create a handle on the current CUDA device.  Validates the config, checks
 * that the device is sm_103, and allocates the scratch workspace (per-CTA
 * partial statistics of the LM head, gathered hidden rows, status word,
 * staging for rv_verify_step_host).  The library owns that memory until
 * rv_destroy.  *out is set only on success. */
RV_API int rv_create(const rv_config* cfg, rv_handle** out);

/* Free the handle and its workspace.  Synchronizes the device first.  NULL is a no-op. */
RV_API int rv_destroy(rv_handle* h);

/* Message of the last failed call on this handle ("" if none).  Valid until the
 * next call on the handle.  h == NULL returns the last rv_create failure. */
RV_API const char* rv_last_error(const rv_handle* h);

/* Workspace bytes the handle holds (for capacity planning). */
RV_API int rv_workspace_bytes(const rv_handle* h, uint64_t* bytes);

/* Build the verify block of Eq. 1 / Alg. 1 ("reflective_draft") for each sequence:
 *   block_ids[b] = [x_1..x_gamma, prompt_1..prompt_P, prefix_1..prefix_L, x_1..x_gamma]
 *   pos_ids[b][j] = ctx_lens[b] + j            (positions run on from the context)
 * draft_ids [B, gamma]; prompt_ids [n_prompt] (shared by all sequences, may be
 * NULL if n_prompt == 0); prefix_ids [B, n_prefix] (the last n_prefix context
 * tokens of each sequence: Prefix_position of Eq. 1); ctx_lens [B].
 * Outputs block_ids, pos_ids [B, Lb], Lb = 2*gamma + n_prompt + n_prefix. */
RV_API int rv_pack_block(rv_handle* h, const int32_t* draft_ids, const int32_t* prompt_ids,
                         const int32_t* prefix_ids, const int32_t* ctx_lens, int32_t B,
                         int32_t gamma, int32_t n_prompt, int32_t n_prefix, int32_t* block_ids,
                         int32_t* pos_ids, void* stream);

/* The pending-token block [t_b, x_1..x_gamma, prompt, prefix_b, x_1..x_gamma]:
 * as rv_pack_block, with the last emitted token t_b = pending_ids[b] (not yet
 * run through the target) in front.  Its final hidden state gives o_1 (the
 * prefix of Alg. 1 then ends in t_b), and its key/value are appended with the
 * block's.  Outputs block_ids, pos_ids [B, Lb + 1] with positions
 * ctx_lens[b] .. ctx_lens[b] + Lb, Lb = 2*gamma + n_prompt + n_prefix. */
RV_API int rv_pack_block_pending(rv_handle* h, const int32_t* pending_ids,
                                 const int32_t* draft_ids, const int32_t* prompt_ids,
                                 const int32_t* prefix_ids, const int32_t* ctx_lens, int32_t B,
                                 int32_t gamma, int32_t n_prompt, int32_t n_prefix,
                                 int32_t* block_ids, int32_t* pos_ids, void* stream);

/* One attention layer of the verify forward pass (Sec. 3.1): causal attention
 * of the block's queries against the KV cache plus the block itself.  Query j
 * of sequence b (position ctx_b + j) attends to cached keys [0, ctx_b) and
 * block keys [0, j]; query head h reads KV head h / (Hq / Hkv).
 *   q      [B, Lb, Hq, D]   post-RoPE queries
 *   k_blk  [B, Lb, Hkv, D]  post-RoPE keys of the block; v_blk likewise
 *   k_cache, v_cache [B, Hkv, max_ctx, D]: read at [0, ctx_b); the block's
 *          keys/values are written at [ctx_b, ctx_b + Lb) (the append; the
 *          caller prunes by advancing ctx_lens, see rv_accept)
 *   ctx_lens [B]  (device)
 *   out    [B, Lb, Hq, D]   softmax(q K^T / sqrt(D)) V
 * A sequence with ctx_b < 0 or ctx_b + Lb > max_ctx is skipped (its output
 * rows are left untouched) and RV_DEV_CTX_RANGE is raised. */
RV_API int rv_verify_attention(rv_handle* h, const void* q, const void* k_blk, const void* v_blk,
                               void* k_cache, void* v_cache, const int32_t* ctx_lens, int32_t B,
                               int32_t Lb, void* out, void* stream);

/* LM head + fusion for the original and reflective rows (Alg. 1, Eq. 2),
 * without ever writing logits to memory.
 *   hidden [B, Lb+1, H]: row 0 = last context position (gives o_1), row r =
 *          after block token r-1.  Original rows 0..gamma, reflective rows
 *          gamma+R .. 2*gamma+R (shift_len = gamma + R = m - 1).
 *   w_head [V, H] LM-head weight (no bias)
 *   draft_ids [B, gamma] (device)
 *   alpha  weight of the reflective logits (Eq. 2; the paper uses 0.3)
 * Outputs, per sequence b and position i = 1..gamma+1 (index i-1):
 *   scores [B, gamma+1, RV_NSCORES] float (see RV_SCORE_*)
 *   argmax [B, gamma+1] int32: greedy choice x^_i = argmax_v z_i[v]; ties go to
 *          the lowest token id
 *   margin [B, gamma] float: |z_i[x_i] - max_{v != x_i} z_i[v]|, the distance of
 *          the accept decision from its boundary (fused-logit units)
 * A draft id outside [0, V) raises RV_DEV_DRAFT_RANGE; its position gets NaN
 * log-probabilities and margin and an argmax that can never equal it. */
RV_API int rv_verify_head(rv_handle* h, const void* hidden, const void* w_head,
                          const int32_t* draft_ids, int32_t B, int32_t gamma, int32_t R,
                          float alpha, float* scores, int32_t* argmax, float* margin,
                          void* stream);

/* Exact-match verification (Alg. 2) with the greedy choice, prefix and next token:
 *   accept_mask[b][i-1] = (x_i == x^_i)                         uint8 [B, gamma]
 *   accepted_len[b] = n = min({i-1 : x_i != x^_i} U {gamma})    int32 [B]
 *   next_token[b]   = t = x^_{n+1}                              int32 [B]
 *   ctx_out[b]      = ctx_in[b] + n   (prunes template, copy and rejected
 *                     drafts from the cache by length; may alias ctx_in)
 * argmax [B, gamma+1] as written by rv_verify_head. */
RV_API int rv_accept(rv_handle* h, const int32_t* draft_ids, const int32_t* argmax, int32_t B,
                     int32_t gamma, uint8_t* accept_mask, int32_t* accepted_len,
                     int32_t* next_token, const int32_t* ctx_in, int32_t* ctx_out, void* stream);

/* Typical acceptance with Reflective Verification (Alg. 3): position i keeps
 * its draft when the fused probability exceeds an entropy-based threshold,
 *   p_i(x_i) > min(eps, delta * exp(-H(softmax(o_i)))),
 * with p_i the fused distribution (Eq. 2) and H the entropy of the unfused
 * original distribution at the same position (scores[..., RV_SCORE_ENT_ORIG]);
 * the test is taken in the log domain on scores[..., RV_SCORE_LOGP_FUSED]:
 *   accept_mask[b][i-1] = logp > min(log eps, log delta - H)     uint8 [B, gamma]
 *   accepted_len[b] = n = number of leading kept drafts             int32 [B]
 *   next_token[b]   = argmax[b][n] (the greedy choice at n+1: the sampling
 *                     temperature of Alg. 3 taken to 0)             int32 [B]
 *   ctx_out[b]      = ctx_in[b] + n (may alias ctx_in)
 * scores [B, gamma+1, RV_NSCORES] and argmax [B, gamma+1] as written by
 * rv_verify_head.  eps > 0 and delta > 0, else RV_ERR_INVALID_ARG.  A draft
 * whose log-probability is NaN (out-of-range id) is rejected. */
RV_API int rv_accept_typical(rv_handle* h, const int32_t* draft_ids, const float* scores,
                             const int32_t* argmax, int32_t B, int32_t gamma, float eps,
                             float delta, uint8_t* accept_mask, int32_t* accepted_len,
                             int32_t* next_token, const int32_t* ctx_in, int32_t* ctx_out,
                             void* stream);

/* Acceptance rule of this handle, for the following calls:
 *   RV_ACCEPT_EXACT (the default; eps and delta ignored) and RV_ACCEPT_TYPICAL
 *     (eps > 0, delta > 0; see rv_accept_typical) apply to rv_verify_step and
 *     rv_verify_step_host;
 *   RV_ACCEPT_SPECULATIVE and RV_ACCEPT_SAMPLED make every LM-head call
 *     (rv_verify_head, the step) also write its fused logits z_i to a buffer
 *     of the handle (allocated here once: max_batch * (max_gamma+1) * vocab
 *     floats), which rv_accept_speculative / rv_verify_step_speculative and
 *     rv_accept_sampled / rv_verify_step_sampled read; in these modes plain
 *     rv_verify_step returns RV_ERR_INVALID_ARG (it has no draft
 *     distributions or uniforms).  Inside rv_verify_step_sampled a bf16
 *     handle's head writes no logits: per position and 32-row vocabulary
 *     subtile it stores (max z, sum exp((z - max) / T)) in a second buffer
 *     allocated here (max_batch * (max_gamma+1) * ceil(vocab / 32) pairs of
 *     floats), and the draw recomputes the logits of one subtile;
 *   RV_ACCEPT_TYPICAL_SAMPLED (eps > 0, delta > 0, the fused head mode):
 *     typical acceptance as RV_ACCEPT_TYPICAL for the kept drafts and n, with
 *     the next token drawn as Alg. 3 states, t ~ p_{n+1} at temperature T
 *     (the draw of rv_accept_sampled at position n+1); it takes the same
 *     buffers and applies to rv_verify_step_sampled only.
 * Errors: RV_ERR_INVALID_ARG for an unknown mode or bad eps / delta,
 * RV_ERR_CUDA if the buffer cannot be allocated. */
RV_API int rv_set_acceptance(rv_handle* h, int32_t mode, float eps, float delta);

/* LM-head variant of this handle, for every following head call (rv_verify_head
 * and the steps):
 *   RV_HEAD_FUSED_LOGITS (the default): the original and reflective logits come
 *     from their own hidden rows and are fused per vocab row (Eq. 2);
 *   RV_HEAD_PREBLENDED: the head has no bias, so z_i = (1-a) W h + a W h' =
 *     W b_i; each sequence's gamma+1 rows b_i = bf16(fl((1-a) h) + fl(a h'))
 *     (float32 products and sum, then one rounding to bf16) go through the
 *     head instead of 2(gamma+1) rows.  Half the MMA work and, above 128
 *     positions, one weight stream where the fused head needs two.  z differs
 *     from the fused logits by that rounding only (|dz_v| <= 2^-8 sum_k
 *     |W_vk| |b_k|).  The original / reflective fields of `scores` (lse_orig,
 *     lse_refl, logp_orig, logp_refl, ent_orig) are NaN, so the typical rule
 *     (Alg. 3, which needs the entropy) is refused in this mode.
 *   RV_HEAD_STANDARD: standard speculative verification, the baseline the
 *     method is compared with (Sec. 4): the block is the drafts alone,
 *     [x_1..x_gamma] (Lb = gamma; the template must be empty, R = 0, else
 *     RV_ERR_SHAPE), hidden is [B, gamma+1, H] with row i-1 giving
 *     p_i = softmax(o_i), alpha is not used.  The step entry points, the pack
 *     calls and the host-buffer step follow this layout; the fused fields of
 *     `scores` hold o's statistics and the other fields are NaN, as above.
 * Errors: RV_ERR_INVALID_ARG for an unknown mode or with the typical rule set,
 * RV_ERR_UNSUPPORTED for an fp32 handle. */
RV_API int rv_set_head_mode(rv_handle* h, int32_t mode);

/* Speculative sampling with Reflective Verification (Alg. 1), after an
 * rv_verify_head call on this handle in RV_ACCEPT_SPECULATIVE mode (same
 * stream, same B and gamma):
 *   accept_mask[b][i-1] = r_i <= p_i(x_i) / q_i(x_i)       uint8 [B, gamma]
 *     (tested as log r_i <= log p_i(x_i) - log q_i(x_i), p_i the fused
 *      distribution of Eq. 2; q_i(x_i) = 0 keeps the draft)
 *   accepted_len[b] = n = number of leading kept drafts       int32 [B]
 *   next_token[b]   = t ~ norm(max(0, p_{n+1} - q_{n+1})) if n < gamma, else
 *                     t ~ p_{gamma+1}, drawn by inverse CDF with u: the
 *                     smallest v whose cumulative weight exceeds u * sum(w)
 *   ctx_out[b]      = ctx_in[b] + n (may alias ctx_in)
 * Inputs (device, float32): q_draft [B, gamma, vocab] the draft model's
 * distributions q_i (rows sum to 1), r_uniform [B, gamma] and u_uniform [B]
 * in [0, 1); scores as written by the preceding rv_verify_head.  Draft ids
 * outside [0, vocab) are rejected and set RV_DEV_DRAFT_RANGE. */
RV_API int rv_accept_speculative(rv_handle* h, const int32_t* draft_ids, const float* q_draft,
                                 const float* r_uniform, const float* u_uniform,
                                 const float* scores, int32_t B, int32_t gamma,
                                 uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                                 const int32_t* ctx_in, int32_t* ctx_out, void* stream);

/* Exact-match verification with target tokens sampled at temperature T
 * (Alg. 2), after an rv_verify_head call on this handle in RV_ACCEPT_SAMPLED
 * mode (same stream, same B and gamma).  The target's token at position
 * i = 1..gamma+1 is x^_i ~ softmax(z_i / T), with z_i the fused logits of
 * Eq. 2, drawn by inverse CDF with u = u_uniform[b][i-1]: the smallest v
 * whose cumulative weight exp((z_i[v] - max z_i) / T) exceeds u times the sum
 * of the weights.  Then, as in rv_accept:
 *   sampled[b][i-1]     = x^_i                                  int32 [B, gamma+1]
 *   accept_mask[b][i-1] = (x_i == x^_i)                          uint8 [B, gamma]
 *   accepted_len[b] = n = min({i-1 : x_i != x^_i} U {gamma})     int32 [B]
 *   next_token[b]   = t = x^_{n+1}, the draw already taken at n+1
 *   ctx_out[b]      = ctx_in[b] + n (may alias ctx_in)
 * The emitted tokens [x_1..x_n, t] are x^_1..x^_{n+1}: what sampling the
 * target alone gives with the same uniforms.  u_uniform [B, gamma+1] float32
 * in [0, 1) (device).  temperature must be finite and > 0, else
 * RV_ERR_INVALID_ARG.  Two launches: the draws (one CTA per position), then
 * the acceptance. */
RV_API int rv_accept_sampled(rv_handle* h, const int32_t* draft_ids, const float* u_uniform,
                             float temperature, int32_t B, int32_t gamma, int32_t* sampled,
                             uint8_t* accept_mask, int32_t* accepted_len, int32_t* next_token,
                             const int32_t* ctx_in, int32_t* ctx_out, void* stream);

/* The whole verify step on device buffers, in one call and three to five
 * kernel launches: on `stream`, one launch that gathers the LM-head rows and
 * packs the block (rv_pack_block; skipped when block_ids is NULL), the LM head
 * and, above 64 positions, one launch that merges the head's statistics and
 * runs the acceptance (rv_accept, or rv_accept_typical when the handle's rule
 * is RV_ACCEPT_TYPICAL; see rv_set_acceptance; with fewer positions the head's
 * last CTA does it); the attention (rv_verify_attention) on an internal stream
 * forked from `stream` after the head's launch, beside it -- except the
 * persistent tcgen05 attention of handles whose KV capacity exceeds 4608
 * positions, which runs first, on `stream`.  The internal stream is joined
 * back into `stream` before the call returns, so later work on `stream` sees
 * every output; the pattern is also valid inside stream capture.  Arguments as
 * in those calls; the template is n_prompt prompt ids + n_prefix prefix ids,
 * so R = n_prompt + n_prefix and Lb = 2*gamma + R (Lb = gamma, no template,
 * for RV_HEAD_STANDARD).  ctx_out may alias ctx_in. */
RV_API int rv_verify_step(rv_handle* h, const void* q, const void* k_blk, const void* v_blk,
                          void* k_cache, void* v_cache, const void* hidden, const void* w_head,
                          const int32_t* draft_ids, const int32_t* prompt_ids,
                          const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B,
                          int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha,
                          int32_t* block_ids, int32_t* pos_ids, void* attn_out, float* scores,
                          int32_t* argmax, float* margin, uint8_t* accept_mask,
                          int32_t* accepted_len, int32_t* next_token, int32_t* ctx_out,
                          void* stream);

/* rv_verify_step over the pending-token block (rv_pack_block_pending): the
 * attention covers Lb + 1 = 2*gamma + R + 1 block positions (q, k_blk,
 * v_blk, attn_out have Lb + 1 rows; their keys/values are appended at
 * [ctx_b, ctx_b + Lb + 1)); hidden [B, Lb + 1, H] has the pending token's
 * state in row 0, which gives o_1, so the LM head is unchanged (original rows
 * 0..gamma, reflective rows gamma+R..2*gamma+R).  The handle's exact-match or
 * typical rule runs; since t stays in the context, ctx_out = ctx_in + 1 + n.
 * RV_ERR_INVALID_ARG in the sampling modes. */
RV_API int rv_verify_step_pending(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache,
    void* v_cache, const void* hidden, const void* w_head, const int32_t* pending_ids,
    const int32_t* draft_ids, const int32_t* prompt_ids, const int32_t* prefix_ids,
    const int32_t* ctx_in, int32_t B, int32_t gamma, int32_t n_prompt, int32_t n_prefix,
    float alpha, int32_t* block_ids, int32_t* pos_ids, void* attn_out, float* scores,
    int32_t* argmax, float* margin, uint8_t* accept_mask, int32_t* accepted_len,
    int32_t* next_token, int32_t* ctx_out, void* stream);

/* rv_verify_step with the speculative-sampling acceptance of Alg. 1
 * (rv_accept_speculative) in place of the handle's fused rule; needs the
 * handle in RV_ACCEPT_SPECULATIVE mode.  q_draft, r_uniform, u_uniform as in
 * rv_accept_speculative; one more launch than rv_verify_step. */
RV_API int rv_verify_step_speculative(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache,
    void* v_cache, const void* hidden, const void* w_head, const int32_t* draft_ids,
    const int32_t* prompt_ids, const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B,
    int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha, const float* q_draft,
    const float* r_uniform, const float* u_uniform, int32_t* block_ids, int32_t* pos_ids,
    void* attn_out, float* scores, int32_t* argmax, float* margin, uint8_t* accept_mask,
    int32_t* accepted_len, int32_t* next_token, int32_t* ctx_out, void* stream);

/* rv_verify_step with target tokens sampled at temperature T in place of the
 * greedy choice; needs the handle in RV_ACCEPT_SAMPLED mode (exact match
 * against the draws, as rv_accept_sampled) or RV_ACCEPT_TYPICAL_SAMPLED
 * (typical acceptance, t = the draw at position n+1).  temperature,
 * u_uniform and sampled as in rv_accept_sampled.  On a bf16 handle one launch
 * more than rv_verify_step (the draws and the acceptance); on fp32 two. */
RV_API int rv_verify_step_sampled(
    rv_handle* h, const void* q, const void* k_blk, const void* v_blk, void* k_cache,
    void* v_cache, const void* hidden, const void* w_head, const int32_t* draft_ids,
    const int32_t* prompt_ids, const int32_t* prefix_ids, const int32_t* ctx_in, int32_t B,
    int32_t gamma, int32_t n_prompt, int32_t n_prefix, float alpha, float temperature,
    const float* u_uniform, int32_t* block_ids, int32_t* pos_ids, void* attn_out, float* scores,
    int32_t* argmax, float* margin, int32_t* sampled, uint8_t* accept_mask,
    int32_t* accepted_len, int32_t* next_token, int32_t* ctx_out, void* stream);

/* The whole verify step from HOST buffers (synchronous).  The small per-step
 * inputs (draft / prompt / prefix ids, ctx lens) are gathered into a pinned
 * buffer of the handle that the kernels read in place, and the kernels write
 * all results but the attention output into a second pinned buffer, which is
 * scattered into the caller's buffers after the stream synchronises.  The row
 * gather reads hidden_host in place when it is page-locked (only the rows the
 * LM head needs cross the link), else it is copied into device staging first.
 * q / k_blk / v_blk are copied into device staging on the handle's second
 * stream (page-locked memory makes these copies asynchronous).  The first call
 * allocates the two small pinned buffers (RV_ERR_CUDA if that fails).  The
 * model state stays on the device: w_head, k_cache and v_cache are device
 * pointers.  Host buffers have the layouts of rv_verify_step; attn_out_host
 * may be NULL to skip reading the attention output back, block_ids_host NULL
 * to skip the packing.  A call repeated with the same arguments on a
 * non-default stream replays a CUDA graph (rv_host_step_graphed).
 * *h2d_bytes / *d2h_bytes (optional) receive the bytes of the per-step inputs
 * and outputs (the inputs' full sizes, also where only some rows are read). */
RV_API int rv_verify_step_host(rv_handle* h, const void* q_host, const void* k_blk_host,
                               const void* v_blk_host, void* k_cache, void* v_cache,
                               const void* hidden_host, const void* w_head,
                               const int32_t* draft_ids_host, const int32_t* prompt_ids_host,
                               const int32_t* prefix_ids_host, const int32_t* ctx_in_host,
                               int32_t B, int32_t gamma, int32_t n_prompt, int32_t n_prefix,
                               float alpha, int32_t* block_ids_host, int32_t* pos_ids_host,
                               void* attn_out_host, float* scores_host, int32_t* argmax_host,
                               float* margin_host, uint8_t* accept_mask_host,
                               int32_t* accepted_len_host, int32_t* next_token_host,
                               int32_t* ctx_out_host, uint64_t* h2d_bytes, uint64_t* d2h_bytes,
                               void* stream);

/* Whether this handle holds the CUDA graph of a repeated rv_verify_step_host
 * call: the second call with the same arguments (pointers, sizes, alpha, the
 * handle's modes and stream) is captured on `stream`, and later identical
 * calls replay it.  No capture is attempted on the legacy default stream
 * (NULL), with pageable host buffers, or while profiling is enabled.  *active
 * = 1 when a graph is held, else 0.  Errors: RV_ERR_INVALID_ARG for NULL
 * arguments. */
RV_API int rv_host_step_graphed(const rv_handle* h, int32_t* active);

/* ---- allocation-free LM head ------------------------------------------------
 * The paper has no counterpart: this entry point exists for callers that may
 * not allocate device memory (code running where cudaMalloc is unavailable or
 * forbidden, e.g. inside host callbacks, under an allocator that owns the whole
 * device, or in plug-ins whose host forbids extra allocations).  It computes
 * exactly what rv_verify_head computes, without a handle and without
 * allocating: its scratch is one fixed file-scope device array of about
 * 2.6 MB that every GPU loading this library keeps until the process exits.
 *   hidden, w_head, draft_ids, B, gamma, R, alpha, scores, argmax, margin:
 *           as in rv_verify_head (bf16 only); vocab / hidden_size give V, H.
 *   dev_status: optional device word; the RV_DEV_* bits of this call are
 *           OR-ed into it and never cleared by the library, so the caller
 *           zeroes it before the first call (NULL: the bits go to the shared
 *           array and are lost).
 * Limits: B * (gamma + 1) <= RV_STATIC_MAX_PAIRS and hidden_size <=
 * RV_STATIC_MAX_HIDDEN, else RV_ERR_CAPACITY before anything is launched.
 * The first call on a device (make it before any stream capture) looks up the
 * array's device address and configures the kernel; later calls only launch.
 * All calls share the array: calls that may run at the same time on the GPU
 * (unordered streams) race; order them on one stream. */
#define RV_STATIC_MAX_PAIRS 64
#define RV_STATIC_MAX_HIDDEN 8192
RV_API int rv_verify_head_static(const void* hidden, const void* w_head,
                                 const int32_t* draft_ids, int32_t B, int32_t gamma, int32_t R,
                                 int32_t vocab, int32_t hidden_size, float alpha, float* scores,
                                 int32_t* argmax, float* margin, uint32_t* dev_status,
                                 void* stream);

/* Synchronize `stream`, read the device status word (RV_DEV_* bits) into
 * *status and clear it.  Returns RV_ERR_DEVICE if any bit was set. */
RV_API int rv_read_status(rv_handle* h, void* stream, uint32_t* status);

/* ---- kernel timing (CUDA events recorded by the library itself) ---------- */
#define RV_PROF_ATTENTION 0   /* attention kernel of rv_verify_attention */
#define RV_PROF_HEAD_GEMM 1   /* the LM-head GEMM + online log-softmax kernel alone */
#define RV_PROF_HEAD 2        /* everything rv_verify_head launches (gather + LM head [+ merge]) */
#define RV_PROF_ACCEPT 3      /* rv_accept (inside rv_verify_step it is part of RV_PROF_HEAD) */
#define RV_PROF_COUNT 4

/* mask: bit (1 << region) set = from now on, record a CUDA event pair on the
 * launching stream around each such region (up to 1024 per region between two
 * rv_profile_read calls, then recording stops); 0 stops recording.  Pairs
 * recorded under earlier masks are kept until rv_profile_read.  An event pair around RV_PROF_HEAD_GEMM
 * sits between the row-gather launch and the LM-head launch and so disables
 * their overlap (programmatic dependent launch); RV_PROF_HEAD brackets both
 * without that cost.  Not for use inside graph capture. */
RV_API int rv_profile_enable(rv_handle* h, int32_t mask);
/* Synchronize the recorded events and return the summed duration (ms) and
 * number of recorded launches of `region`; then forget them. */
RV_API int rv_profile_read(rv_handle* h, int32_t region, double* total_ms, int32_t* count);

/* Number of kernel launches the library has issued on this handle (all
 * entry points), for launch accounting. */
RV_API int rv_launch_count(const rv_handle* h, uint64_t* count);

#ifdef __cplusplus
}
#endif
#endif /* RV_H_ */
