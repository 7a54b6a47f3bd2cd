/*
 * cdsl.h -- C ABI of the GB300 CDSL lookahead step.
 *
 * Constrained Decoding with Speculative Lookaheads (CDSL, arXiv 2412.10418): a small draft
 * model M_q rolls out d greedy lookahead tokens (Sec. 3.2.1), a large target model M_p
 * verifies them in one forward pass (Sec. 3.2.2, "Validation by M_p"), a task reward R scores
 * them ("Validation by R") and a state machine over the acceptance score a and the reward r
 * decides what is emitted (Sec. 3.2.3, Algorithm 1).
 *
 * This library runs the batched "CDSL-k" step on one GPU: for each of B prompts, the top-k
 * target candidates c_1..c_k (the beams of Algorithm 2) each get a d-token draft rollout over
 * a shared-prefix paged KV cache; the target verifies all B*k*(d+1) rows [c_b, x_b1..x_bd] in
 * one pass; a fused epilogue computes log-softmax / argmax / the hard-rejection count n_b,
 * a_b = n_b/d, the rewards, the chosen beam b* (largest r^full, first on ties) and the state:
 *   S1  (a_b* >= a_t and r^acc_b* >= r_t): emit c_b*, x_b*,1..n       (Sec. 3.2.3, S1)
 *   S2/S3 (a < a_t), S4 (a >= a_t, r < r_t): emit c_b* only, i.e. the one CDLH-appx token of
 *   Algorithm 1's fallback (Step-2); with a Step-1 budget b >= 1 (cdsl_run_cfg.step1_budget),
 *   S2/S3 first tries M_p's greedy tokens: c_1 if r^full_1 >= r_t, and with b = 2 then
 *   c_1, x' (x' = M_p's argmax after c_1) if the reward of x''s own lookahead reaches r_t
 *   (state 3).
 *
 * Conventions
 *  - Every compute call is asynchronous on the stream given to cdsl_init (a cudaStream_t
 *    passed as void*; NULL = the legacy default stream). Pointers prefixed d_ are device
 *    pointers, h_ host pointers. All index outputs are int32, all real outputs float32.
 *  - Ownership: weights, the workspace and every output buffer belong to the caller and must
 *    outlive the context; the context only borrows them. The context owns its host metadata.
 *  - Errors: each call returns a cdsl_status. Argument and call-order errors are detected
 *    on the host before anything is launched. Errors found on the device (a bounded wait
 *    that expired, a non-finite logit row, the KV page pool running out) are latched in a
 *    device status word that cdsl_get_status reads. cdsl_last_error gives a message.
 *  - Any d_ output pointer may be NULL: that output is then not written.
 *  - Weights: matrices are [out_features, in_features] row-major (y = x W^T), in the model's
 *    dtype (float32 or bfloat16); RMSNorm gains are vectors of d_model in the same dtype.
 */
#ifndef CDSL_H
#define CDSL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define CDSL_API __attribute__((visibility("default")))
#else
#define CDSL_API
#endif

typedef enum cdsl_status {
  CDSL_OK = 0,
  CDSL_EINVAL = 1,     /* invalid argument or configuration */
  CDSL_ENOMEM = 2,     /* workspace smaller than cdsl_workspace_size */
  CDSL_ECUDA = 3,      /* a CUDA runtime or driver call failed */
  CDSL_ETIMEOUT = 4,   /* device: a bounded wait in a kernel gave up */
  CDSL_ENONFINITE = 5, /* device: a logits row held NaN or Inf */
  CDSL_ESTATE = 6,     /* calls made out of order (e.g. cdsl_verify before cdsl_lookahead) */
  CDSL_ERANGE = 7      /* device: KV page pool exhausted or a position beyond the limits */
} cdsl_status;

enum { CDSL_DTYPE_F32 = 0, CDSL_DTYPE_BF16 = 1 };

/* Pre-norm decoder: RMSNorm, GQA attention with rotate-half RoPE, SwiGLU FFN, untied LM head
 * (the draft and target models of Sec. 2.2 / Sec. 3; Llama-style shapes for the synthetic
 * workloads). head_dim must be 64 or 128 and n_heads a multiple of n_kv_heads. */
typedef struct cdsl_model_cfg {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t d_ffn;
  int32_t vocab;
  int32_t dtype;       /* CDSL_DTYPE_F32 or CDSL_DTYPE_BF16 */
  float rope_theta;    /* e.g. 10000 */
  float norm_eps;      /* e.g. 1e-5 */
} cdsl_model_cfg;

/* Decoding parameters, Algorithm 1 inputs (d, l_m, k, r_t, a_t) plus batch and reward. */
typedef struct cdsl_run_cfg {
  int32_t batch;        /* B prompts decoded side by side (each its own CDSL state) */
  int32_t k;            /* beams = top-k target candidates, 1..16 */
  int32_t d;            /* lookahead length, 1..16 */
  int32_t max_prompt;   /* longest prompt, tokens */
  int32_t max_new;      /* l_m: tokens generated per prompt */
  int32_t n_keywords;   /* keyword ids per prompt for the coverage reward, 1..32 */
  float a_t;            /* acceptance threshold */
  float r_t;            /* reward threshold */
  int32_t reward_head;  /* 0: R = coverage; 1: R = 0.5 coverage + 0.5 sigmoid(w . h_last) */
  int32_t page_size;    /* KV page size in tokens (power of two, 16..256); 0 = 64 */
  int32_t max_chunk;    /* rows per prefill forward pass; 0 = 256 (the tensor-core GEMM maximum) */
  /* Validation of the lookahead by M_p (Sec. 3.2.2):
   *   0: hard rejection: x_j is accepted while argmax p_j == x_j;
   *   1: speculative sampling: x_j is accepted while u_j <= min(1, p_j(x_j) / q_j(x_j)),
   *      tested as log(u_j) <= log p_j(x_j) - log q_j(x_j) in float32. The rejected position's
   *      resampled token is never emitted (CDSL keeps only accepted drafts, Sec. 3.2.2), so
   *      only the count n_b is used.
   * u_j = (SplitMix64 output number c of the generator seeded with `seed`) >> 40, times 2^-24,
   * where c = ((step * batch + b) * k + beam) * d + (j - 1) and step counts the completed
   * steps of the context (SplitMix64: Steele, Lea, Flood, OOPSLA 2014). */
  int32_t acceptance;
  uint32_t seed;
  /* Step-1 budget b of Alg. 1's S2/S3 branch (Sec. 3.2.3), 0, 1 or 2. With b >= 1,
   * a step in S2/S3 (a < a_t) first tries M_p's greedy token, the root c_1, whose draft
   * lookahead and reward r_1^full the step already has: if r_1^full >= r_t it emits c_1
   * (state 3) instead of the CDLH-appx token c_{b*} of Step-2. With b = 2, when that fails,
   * round 2 takes x' = argmax M_p(pfx + c_1) (verify row (b, 1, 0)), runs d greedy draft
   * calls from pfx + c_1 + x' (lookahead lh) and one target pass over [x', c_1, lh] (for
   * M_p(pfx + c_1 + x'), the reward head at lh_d and the K/V of c_1, x'), and emits c_1, x'
   * (state 3) if R(T + c_1 + x' + lh) >= r_t. The round runs every step for every prompt
   * (d extra draft calls and one extra target pass per step); only prompts whose round 1
   * failed in S2/S3 use it. cdsl_get_step1 returns its tokens and rewards. */
  int32_t step1_budget;
} cdsl_run_cfg;

typedef struct cdsl_ctx cdsl_ctx;

/* Number of weight pointers a model takes:
 *   [0] embed [vocab, d_model]
 *   per layer l (base 1 + 9 l): attn_norm [d_model], wq [n_heads*hd, d_model],
 *       wk [n_kv_heads*hd, d_model], wv [n_kv_heads*hd, d_model], wo [d_model, n_heads*hd],
 *       ffn_norm [d_model], w_gate [d_ffn, d_model], w_up [d_ffn, d_model],
 *       w_down [d_model, d_ffn]
 *   [1 + 9 L] final_norm [d_model], [2 + 9 L] lm_head [vocab, d_model]
 * Every pointer must be 16-byte aligned. Returns -1 for an invalid configuration. */
CDSL_API int32_t cdsl_num_weights(const cdsl_model_cfg* cfg);

/* Bytes of device workspace cdsl_init needs for these configurations (KV page pools for
 * B * (max_prompt + max_new + 1) positions of both models, the per-beam KV tails, activation
 * and logits buffers for the largest pass, decoding state). */
CDSL_API int32_t cdsl_workspace_size(const cdsl_model_cfg* target, const cdsl_model_cfg* draft,
                            const cdsl_run_cfg* run, size_t* bytes);

/* Validate the configurations, borrow the weights (arrays of cdsl_num_weights device
 * pointers each), carve the caller's workspace (256-byte aligned, at least
 * cdsl_workspace_size bytes) and bind the stream. d_reward_head: the linear reward head w
 * [target d_model] float32 (may be NULL when run->reward_head == 0). The target and draft
 * must share the vocabulary (Sec. 4.2). Launches only memsets and table set-up kernels. */
CDSL_API int32_t cdsl_init(const cdsl_model_cfg* target, const void* const* h_target_weights,
                  const cdsl_model_cfg* draft, const void* const* h_draft_weights,
                  const cdsl_run_cfg* run, const float* d_reward_head,
                  void* d_workspace, size_t workspace_bytes, void* stream, cdsl_ctx** out);

/* Start decoding: reset the state, run both models over the prompts (writing their KV into
 * the prefix pages) and take the top-k of M_p(pfx) as the first beams.
 * d_prompts [B, max_prompt] token ids, row b valid for h_prompt_lens[b] tokens (1..max_prompt);
 * d_keywords [B, n_keywords] distinct keyword ids per prompt. */
CDSL_API int32_t cdsl_prefill(cdsl_ctx* ctx, const int32_t* d_prompts, const int32_t* h_prompt_lens,
                     const int32_t* d_keywords);

/* Lookahead generation (Sec. 3.2.1; Alg. 2 lookahead with M_q): d greedy draft decode calls
 * over the B*k beam rows. Outputs d_roots [B, k] (the beams' first tokens c_b, descending
 * target logit, ties to the lower id), d_draft_tok [B, k, d] x_b,j and d_logq [B, k, d]
 * log q_j(x_b,j). */
CDSL_API int32_t cdsl_lookahead(cdsl_ctx* ctx, int32_t* d_roots, int32_t* d_draft_tok, float* d_logq);

/* Validation by M_p (Sec. 3.2.2, hard rejection): one target pass over the B*k*(d+1) rows
 * [c_b, x_b,1..x_b,d]. Row j of beam b gives p_b,j+1. Outputs d_logp [B, k, d]
 * log p_b,j(x_b,j), d_argmax [B, k, d+1] argmax of every row (ties to the lower id),
 * d_n_accept [B, k] n_b, and optionally d_logits [B, k, d+1, vocab] (the raw logits, for
 * inspection). Requires a preceding cdsl_lookahead. */
CDSL_API int32_t cdsl_verify(cdsl_ctx* ctx, float* d_logp, int32_t* d_argmax, int32_t* d_n_accept,
                    float* d_logits);

/* Acceptance decision and commit (Sec. 3.2.3, Algorithm 1 with b = 0, 1 or 2): rewards
 * d_reward [B, k, 2] = (r^full, r^acc) per beam, d_beam [B] the beam whose tokens are
 * emitted (b*, or 0 for a Step-1 token), d_state [B] 1 (S1), 2 (S2/S3), 3 (S2/S3 resolved by
 * Step-1) or 4 (S4), d_emitted [B, d+1] the emitted tokens (-1 padded), d_n_emitted [B]
 * (0 for prompts that already hold l_m tokens). Emission is cut at l_m. Then the winner's KV
 * rows are committed to the prefix pages and the next beams are taken from the winner's
 * verify row (after a round-2 Step-1 emission: from M_p(pfx + c_1 + x')). With budget 2 the
 * call also runs the Step-1 round (see cdsl_run_cfg.step1_budget). Requires a preceding
 * cdsl_verify. */
CDSL_API int32_t cdsl_select(cdsl_ctx* ctx, int32_t* d_beam, int32_t* d_state, int32_t* d_emitted,
                    int32_t* d_n_emitted, float* d_reward);

/* One whole CDSL-k step: cdsl_lookahead + cdsl_verify + cdsl_select, launched as one
 * CUDA graph after its first call (control stays on the device; nothing is read back).
 * Same outputs as cdsl_select. */
CDSL_API int32_t cdsl_step(cdsl_ctx* ctx, int32_t* d_beam, int32_t* d_state, int32_t* d_emitted,
                  int32_t* d_n_emitted, float* d_reward);

/* Copy the decoded state: d_tokens [B, max_prompt + max_new] (prompt then generated tokens,
 * -1 padded), d_lengths [B] prompt + generated length. Either may be NULL. */
CDSL_API int32_t cdsl_get_tokens(cdsl_ctx* ctx, int32_t* d_tokens, int32_t* d_lengths);

/* Counters since cdsl_prefill, host int64[8]: [0] steps, [1] draft forward passes, [2] target
 * forward passes, [3] tokens emitted (all prompts), [4] S1 decisions, [5] prompt-steps
 * decided, [6] kernel launches in one cdsl_step (0 before the first cdsl_step), [7] 0.
 * Synchronizes the stream. [1]-[3] give the paper's "LLM calls per token" (Sec. 4.3,
 * Table 6): per step each beam's lookahead is d draft calls and its verification one target
 * call. */
CDSL_API int32_t cdsl_get_counters(cdsl_ctx* ctx, int64_t* h_counters);

/* Kernel timing (a measurement aid; the paper has no counterpart). cdsl_profile(ctx, mode):
 *   0: off.
 *   1: every kernel launch of the following calls is bracketed by CUDA events on the
 *      context's stream, and cdsl_step launches its kernels directly instead of through its
 *      graph (per-launch durations without the overlap of programmatic dependent launch).
 *   2: in-graph timing. cdsl_step replays a second graph whose GEMM, attention and row
 *      statistics kernels stamp their first block's entry and last block's exit on the device
 *      clock (%globaltimer); after each step the call synchronizes the stream and charges
 *      every stamped launch, in stream order, from its entry (or the previous stamped exit,
 *      whichever is later) to its exit. The charged intervals are disjoint, so their sum
 *      never exceeds the step. The attention kernel also counts its own algorithmic bytes
 *      (K and V of every key once per prompt and KV head, queries and outputs once).
 * cdsl_get_profile synchronizes the stream and returns, for kernel class `impl`
 * (0 = CUDA-core tiled GEMM, 1 = weight-streaming GEMV, 2 = tcgen05 tensor-core GEMM,
 * 3 = attention, 4 = RMSNorm, 5 = logits row statistics, 6 = embedding, 7 = plans, decision
 * and commit; in mode 2 also 8 = the stamped steps: {steps, milliseconds from the first
 * stamped entry to the last stamped exit, 0, 0}),
 * h_out[4] = {launches, total milliseconds, algorithmic bytes (weights read once, activations
 * read, outputs written; attention as counted by the kernel), flops} over the launches
 * recorded since cdsl_profile was last called (each call clears the record). In mode 2 the
 * classes 4, 6 and 7 are not stamped and report 0 milliseconds. */
CDSL_API int32_t cdsl_profile(cdsl_ctx* ctx, int32_t enable);
CDSL_API int32_t cdsl_get_profile(cdsl_ctx* ctx, int32_t impl, double* h_out);
/* Per-launch form of the same record: for each of the first h_capacity recorded launches,
 * in launch order, four doubles {class, milliseconds, algorithmic bytes, flops} at h_out
 * [4 * i] (mode 2: one record per launch of the stamped step, milliseconds and bytes
 * averaged over the stamped steps); returns the number of records written (>= 0) or a
 * negative status. Synchronizes the stream. */
CDSL_API int32_t cdsl_get_profile_launches(cdsl_ctx* ctx, double* h_out, int32_t h_capacity);

/* Step-1 round 2 of the last cdsl_select / cdsl_step (budget 2; Alg. 1, S2/S3 Step-1): d_need [B]
 * 1 where round 1 failed in S2/S3 so that round 2 decided the step, d_tokens [B, d+1] the
 * round's x' and lookahead lh_1..lh_d, d_reward [B] R(T + c_1 + x' + lh) (meaningful where
 * d_need = 1). Any pointer may be NULL. CDSL_EINVAL with a smaller budget. */
CDSL_API int32_t cdsl_get_step1(cdsl_ctx* ctx, int32_t* d_need, int32_t* d_tokens, float* d_reward);

/* Limit of the tensor-core kernels' bounded waits on another agent's progress (a pipeline
 * stage, an accumulator, an MMA result), in nanoseconds of device wall time; 2 s after
 * cdsl_init. A wait that runs out latches CDSL_ETIMEOUT in the device status word; the block
 * then skips the rest of its work, waits (with a fixed 2 s limit) for its own copies and
 * MMAs in flight, meets its cluster barriers and exits, so the launch ends and the CUDA
 * context stays usable. The context's results are undefined after CDSL_ETIMEOUT: destroy it
 * (a new context on the same device works). A short limit exercises that failure path
 * without a fault (0: every wait not already satisfied gives up). Synchronizes the stream;
 * the next cdsl_step captures its graph again. */
CDSL_API int32_t cdsl_set_wait_limit(cdsl_ctx* ctx, uint64_t ns);

/* Synchronize the stream and return the device status word (a cdsl_status; CDSL_OK when no
 * device-side error was latched) in *h_device_status. Clears nothing. */
CDSL_API int32_t cdsl_get_status(cdsl_ctx* ctx, int32_t* h_device_status);

/* Weight-streaming GEMM that allocates nothing (the paper has no counterpart). It serves
 * callers of this library that cannot allocate device memory: host frameworks whose own
 * caching allocator has already reserved the GPU's memory, real-time loops that must not
 * block on cudaMalloc / cudaFree, and runtimes that forbid device allocation after start-up.
 * y[R, N] = x[R, K] W^T with fp32 accumulation, computed by the library's CUDA-core split-K
 * GEMV (x is split into bf16 hi and lo planes, so the result is within about 1e-5 relative
 * of the exact product): d_w [N, K] bfloat16 row-major, d_x [R, K] float32, d_y [R, N]
 * float32, all device pointers on the current device, contiguous and 16-byte aligned; stream
 * is a cudaStream_t (NULL: the legacy stream).
 * Limits: 1 <= R <= 8, 8 <= K <= 8192 with K % 8 == 0, 1 <= N <= 32768; anything beyond them
 * returns CDSL_EINVAL without launching. Its scratch (split-K partials, arrival counters and
 * the hi/lo activation planes, 8.3 MiB) is one fixed array inside the library, which every
 * GPU that loads the library holds until the process exits; no call allocates or frees.
 * Set-up: the first call in each CUDA context looks up that array's device address (and
 * clears its counters) with the context current. Only contexts that stay alive are
 * supported: after a device reset the array's address may be stale. Every call shares the
 * array: calls that overlap on a GPU (other streams or threads) race, and the caller must
 * order them. Asynchronous on `stream`; errors via cdsl_last_error(NULL). */
CDSL_API int32_t cdsl_gemv_noalloc(const void* d_w, int32_t N, int32_t K, const float* d_x,
                                   int32_t R, float* d_y, void* stream);

/* Message of the last error on this context (never NULL; "" when none). With ctx == NULL,
 * the message of the last failed context-free call (cdsl_init, cdsl_workspace_size,
 * cdsl_gemv_noalloc) on this thread. */
CDSL_API const char* cdsl_last_error(const cdsl_ctx* ctx);

/* Release the context's host metadata and CUDA graph. Does not free borrowed memory. */
CDSL_API void cdsl_destroy(cdsl_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* CDSL_H */
