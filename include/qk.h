/*
 * qk.h -- C ABI of libqk: the forward pass of a Qwen3-architecture decoder on
 * one GB300 (sm_103a), for rollout decode and teacher-forced log-prob scoring.
 *
 * What it computes.  The policy forward pass whose per-token log-probability
 * log pi_theta(y_t | x, y_<t) enters the SFT objective (Eq. sft, Sec. "Task
 * Serialization and SFT Objective") and the PPO-clipped GRPO objective (Eq. ppo,
 * Sec. "GRPO Optimization": the ratio rho_t and the KL term), and whose
 * autoregressive decode produces the rollouts of the RL loop (Sec.
 * "Implementation Components").  The paper cites the Qwen3 architecture without
 * restating it; the layer definition used here is:
 *     x = E[token];  per layer: u = RMSNorm(x)*g1; q,k,v = W_q u, W_k u, W_v u;
 *     per head RMSNorm of q and k (gains of length head_dim) then rotate-half
 *     RoPE (theta from the config); causal GQA attention (kv head = q head /
 *     (n_q/n_kv), scale 1/sqrt(head_dim)); x += W_o o; u = RMSNorm(x)*g2;
 *     x += W_down(silu(W_gate u) * W_up u);
 *     logits = W_lm (RMSNorm(x)*g_final); log p = logit - logsumexp(logits).
 * RMSNorm is x / sqrt(mean(x^2) + eps).
 *
 * Conventions (every entry point):
 *  - Memory.  The library never allocates device memory.  Every device buffer
 *    (packed weights, KV cache, workspace, inputs, outputs) is allocated by the
 *    caller and borrowed for the duration of the call (the packed-weight buffer
 *    for the model's lifetime).  Pointers documented "dev" are device pointers.
 *  - Streams.  `stream` is a cudaStream_t passed as void*; NULL means the
 *    legacy default stream.  Every compute call is asynchronous on that stream
 *    and performs no host synchronisation; it can be captured in a CUDA graph.
 *  - Errors.  Every int-returning call returns QK_OK (0) or a negative QK_E*
 *    code and leaves a message for qk_last_error() (thread-local).  Arguments
 *    are validated on the host before any launch; a call that returns an error
 *    has launched nothing.  Data-dependent faults found on the device (a token
 *    id outside [0, vocab), a position outside the cache, a bounded wait that
 *    expired) set bits of the model's device status word instead; the kernels
 *    then substitute a safe value (token 0, position clamped, page 0 for a page
 *    id outside the pool) rather than read out of bounds.  qk_check_status() reads and clears that word.
 *  - dtype.  QK_DTYPE_BF16 models keep weights, activations and KV cache in
 *    bf16 with fp32 accumulation, an fp32 residual stream and fp32 softmax /
 *    log-softmax statistics.  QK_DTYPE_F32 models are fp32 end to end (no TF32).
 */
#ifndef QK_H
#define QK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define QK_OK 0
#define QK_EINVAL (-1)   /* null pointer, bad enum, unknown preset            */
#define QK_ESHAPE (-2)   /* size out of range: B > max_batch, T too long, ... */
#define QK_EDTYPE (-3)   /* unsupported dtype / head_dim / grouping           */
#define QK_ECUDA (-4)    /* a CUDA runtime / driver call failed               */
#define QK_ETIMEOUT (-5) /* a device-side bounded wait expired (qk_check_status) */
#define QK_EDEVICE (-6)  /* device status word had a fault bit set            */
#define QK_ENOSPACE (-7) /* caller buffer smaller than the size query returns */

#define QK_DTYPE_BF16 0
#define QK_DTYPE_F32 1

/* Bits of the device status word (qk_check_status). */
#define QK_STATUS_BAD_TOKEN 1u    /* token id outside [0, vocab) (an input id, or no
                                     drawable token: non-finite logits); 0 was used */
#define QK_STATUS_BAD_POS 2u      /* position outside [0, max_seq); it was clamped */
#define QK_STATUS_TIMEOUT 4u      /* a bounded device wait gave up                 */
#define QK_STATUS_BAD_PAGE 8u     /* page-table entry outside [0, n_pages); page 0  */
                                  /* was used in its place                         */

/* Kinds of call for qk_workspace_bytes. */
#define QK_CALL_DECODE 0   /* qk_decode_step / qk_decode_layer: B tokens          */
#define QK_CALL_PREFILL 1  /* qk_prefill: B x T tokens                             */
#define QK_CALL_SCORE 2    /* qk_score_logprobs: B x T tokens, no KV cache         */
#define QK_CALL_ROLLOUT 3  /* qk_rollout_teacher_forced: prefill B x T then decode */
#define QK_CALL_BACKWARD 4 /* qk_backward_logprob: B x T tokens (max_seq ignored)     */

typedef struct qk_config {
    int32_t n_layers;      /* decoder layers                                  */
    int32_t hidden;        /* H, multiple of 64                               */
    int32_t n_q_heads;     /* query heads                                     */
    int32_t n_kv_heads;    /* key/value heads; n_q_heads % n_kv_heads == 0    */
    int32_t head_dim;      /* d: 64 or 128                                    */
    int32_t intermediate;  /* SwiGLU width I, multiple of 128                 */
    int32_t vocab;         /* V                                               */
    int32_t dtype;         /* QK_DTYPE_BF16 or QK_DTYPE_F32                   */
    int32_t max_positions; /* length of the RoPE table (largest position + 1) */
    int32_t reserved;      /* must be 0                                       */
    double rms_eps;        /* RMSNorm epsilon (inside the square root)        */
    double rope_theta;     /* RoPE base                                       */
} qk_config;

typedef struct qk_model qk_model;

/* Fill *out with a named preset: "tiny_fp32" (2 layers, H 256, 4/2 heads, d 64,
 * I 768, V 4096, fp32), "q8b" (36 layers, H 4096, 32/8 heads, d 128, I 12288,
 * V 151936, bf16), "q8b_layer" (one q8b layer).  eps 1e-6, theta 1e6,
 * max_positions 8192.  Returns QK_EINVAL for an unknown name.
 * Source: the policy is Qwen3-8B(-Instruct) (Sec. "Training Configuration" and
 * the hyperparameter table of Sec. "Hyperparameters": sequence lengths 8K / 16K);
 * the paper does not restate the architecture, so its dimensions, eps and theta
 * here are the public Qwen3-8B values, and max_positions 8192 covers the 8K
 * sequences of the HIP runs. */
int qk_config_preset(const char* name, qk_config* out);

/* Number of weight tensors of a config, in the canonical order used by
 * qk_model_load: embed [V,H]; then per layer attn_norm [H], wq [nq*d,H],
 * wk [nkv*d,H], wv [nkv*d,H], q_norm [d], k_norm [d], wo [H,nq*d],
 * mlp_norm [H], wg [I,H], wu [I,H], wd [H,I]; then final_norm [H],
 * lm_head [V,H].  Matrices are row-major [out, in].  (The tensors of the Qwen3
 * layer definition in the file header; the paper cites the architecture only.) */
int qk_weight_count(const qk_config* cfg, int* n_tensors);

/* Bytes of the packed device buffer qk_model_load needs for this config (a
 * service call: the library never allocates, so it reports sizes). */
int qk_model_packed_bytes(const qk_config* cfg, size_t* bytes);

/* Build a model: the Qwen3-8B policy whose forward pass the paper trains with
 * SFT and GRPO (Sec. "Agentic Integration": one Qwen3-8B policy serves every
 * agent role), here with caller-supplied (random-init) weights; the paper
 * publishes no trained checkpoint.
 * `tensors` is a host array of n_tensors device pointers in the
 * canonical order above, each holding the tensor in the config's dtype.  They
 * are read (repacked into `packed`, which must hold qk_model_packed_bytes bytes
 * and be 256-byte aligned) on `stream` and may be freed once the stream has
 * passed this call.  `packed` is borrowed for the model's lifetime.  *out
 * receives a host object owned by the library; release it with qk_model_free. */
int qk_model_load(const qk_config* cfg, const void* const* tensors, int n_tensors, void* packed,
                  size_t packed_bytes, void* stream, qk_model** out);
void qk_model_free(qk_model* m);

/* KV cache bytes for max_batch rows of max_seq positions: per layer K then V,
 * each [max_batch, n_kv, max_seq, d] in the model dtype, contiguous.  The cache
 * holds the keys and values of every earlier position of a rollout, so that a
 * decode step of the autoregressive rollout loop (Sec. "Implementation
 * Components": the policy generates candidates for up to T = 3 turns) attends to
 * them without recomputing the prefix.  Sized for the paper's RL batches (64
 * prompts x G = 8 rollouts, sequences up to 8K / 16K tokens, hyperparameter
 * table). */
int qk_kv_bytes(const qk_model* m, int max_batch, int max_seq, size_t* bytes);

/* Workspace bytes for one call of the given kind (QK_CALL_*) with batch B and
 * T tokens per row (T = 1 for decode; T = prompt length for a rollout) against
 * a cache of max_seq positions.  (A service call; the paper has no counterpart.) */
int qk_workspace_bytes(const qk_model* m, int kind, int B, int T, int max_seq, size_t* bytes);

/* Prefill: the prompt pass of a rollout (Sec. "Execution-Aware Reinforcement
 * Learning": each candidate is generated from the task prompt; Sec.
 * "Implementation Components": the rollout loop samples prompts and the policy
 * generates from them).
 * Prefill T tokens per row at positions start_pos .. start_pos+T-1 (causal
 * attention over cache positions 0 .. p), writing their K and V into the cache.
 * tokens: dev int32 [B, T].  The cache rows b < B must already hold positions
 * < start_pos.  Outputs for the last position of each row (any may be NULL):
 * last_logits dev fp32 [B, V]; logprobs dev fp32 [B] = log p(targets[b]) with
 * targets dev int32 [B] (required when logprobs is given); argmax dev int32 [B]
 * (lowest index among equal maxima).  QK_ESHAPE if B > max_batch or
 * start_pos + T > max_seq. */
int qk_prefill(qk_model* m, void* kv, int max_batch, int max_seq, const int32_t* tokens, int B,
               int T, int start_pos, float* last_logits, const int32_t* targets, float* logprobs,
               int32_t* argmax, void* workspace, size_t ws_bytes, void* stream);

/* One decode step of the autoregressive rollout (Sec. "Execution-Aware
 * Reinforcement Learning" and the rollout loop of Sec. "Implementation
 * Components": the policy generates each candidate token by token; its
 * log-probability log pi_theta(y_t | x, y_<t) is the quantity of Eq. sft and
 * of the ratio in Eq. ppo).
 * Row b consumes tokens[b] at position pos[b] (dev int32 [B]
 * each), writes its K and V at pos[b] and attends positions 0 .. pos[b].
 * Outputs as in qk_prefill, for the B new positions. */
int qk_decode_step(qk_model* m, void* kv, int max_batch, int max_seq, const int32_t* tokens,
                   const int32_t* pos, int B, float* logits, const int32_t* targets,
                   float* logprobs, int32_t* argmax, void* workspace, size_t ws_bytes,
                   void* stream);

/* One decoder layer of a decode step (the unit of the rollout decode above, on
 * its own for per-layer parity and timing) on a given residual stream: x dev fp32
 * [B, H] is updated in place; the new K and V go to the layer's cache at
 * pos[b] (dev int32 [B]) and attention covers 0 .. pos[b]. */
int qk_decode_layer(qk_model* m, int layer, void* kv, int max_batch, int max_seq, float* x,
                    const int32_t* pos, int B, void* workspace, size_t ws_bytes, void* stream);

/* Append a turn to rows that sit at different positions (multi-turn rollouts,
 * Sec. "Multi-Turn On-Policy Reflection": feedback appended to each rollout).
 * Row b appends tokens[b, 0 .. len[b]-1] (dev int32 [B, T], row stride T) at
 * positions start[b] .. start[b] + len[b] - 1 (start, len dev int32 [B];
 * len NULL = T; 1 <= len[b] <= T and start[b] + T <= max_seq are required: a
 * position outside the cache sets QK_STATUS_BAD_POS and is clamped).  The
 * entries t >= len[b] of a row are padding: they are computed and written at
 * positions start[b] + len[b] .. start[b] + T - 1, which the row's next tokens
 * overwrite and which no earlier position attends.  last_logits dev fp32 [B, V]
 * or NULL: the logits after each row's last appended token.  Workspace:
 * qk_workspace_bytes(QK_CALL_PREFILL, B, T, max_seq). */
int qk_prefill_rows(qk_model* m, void* kv, int max_batch, int max_seq, const int32_t* tokens,
                    int B, int T, const int32_t* start, const int32_t* len, float* last_logits,
                    void* workspace, size_t ws_bytes, void* stream);

/* Paged KV cache.  The rollouts of one RL batch (Sec. "Execution-Aware
 * Reinforcement Learning": G = 8 rollouts per prompt) and their appended turns
 * (Sec. "Multi-Turn On-Policy Reflection") end at different lengths, so a
 * dense cache that reserves max_seq positions for every row holds mostly
 * unused positions.  A paged cache holds, per layer, a K pool then a V pool of
 * n_pages pages, each [n_kv, page_size, d] in the model dtype (per layer
 * 2 x n_pages x n_kv x page_size x d elements, layers contiguous: the bytes of
 * qk_kv_bytes with max_batch = n_pages, max_seq = page_size; qk_kv_pages_bytes
 * returns them).  Position p of row b lives at offset p % page_size of page
 * table[b * per_row + p / page_size].  table: dev int32 [B, per_row], owned by
 * the caller, read by every paged call and never written; an entry a call
 * reaches (row b's pages up to its last position) must lie in [0, n_pages):
 * one outside sets QK_STATUS_BAD_PAGE and page 0 is used in its place; entries
 * beyond a row's last position are not read.  Rows may share a page that
 * holds a common prefix (its positions written once, through one row), as long
 * as no call writes positions of that page through another row.  A row holds per_row x page_size positions,
 * which plays the part of max_seq (<= max_positions; workspace sizes:
 * qk_workspace_bytes with max_seq = per_row x page_size).  page_size is a
 * multiple of 128 (one tensor-core key tile never straddles two pages).  (A
 * memory layout of this library; the paper does not describe cache memory.) */
typedef struct qk_kv_pages {
    const int32_t* table; /* dev int32 [B, per_row] page ids                  */
    int per_row;          /* table entries per row                            */
    int n_pages;          /* pages in each layer's K pool (and in its V pool) */
    int page_size;        /* positions per page, a multiple of 128            */
} qk_kv_pages;

/* Bytes of a paged cache of n_pages pages of page_size positions (all layers).
 * QK_ESHAPE unless n_pages >= 1 and page_size is a positive multiple of 128. */
int qk_kv_pages_bytes(const qk_model* m, int n_pages, int page_size, size_t* bytes);

/* qk_decode_step over a paged cache (same tokens, pos, outputs and workspace as
 * qk_decode_step with max_seq = per_row x page_size; pos[b] < per_row x
 * page_size, else QK_STATUS_BAD_POS and clamping). */
int qk_decode_step_paged(qk_model* m, void* kv, const qk_kv_pages* pages, const int32_t* tokens,
                         const int32_t* pos, int B, float* logits, const int32_t* targets,
                         float* logprobs, int32_t* argmax, void* workspace, size_t ws_bytes,
                         void* stream);

/* qk_prefill_rows over a paged cache: prompts (start[b] = 0) and appended turns
 * at per-row positions, the same arguments and rules as qk_prefill_rows with
 * max_seq = per_row x page_size. */
int qk_prefill_rows_paged(qk_model* m, void* kv, const qk_kv_pages* pages, const int32_t* tokens,
                          int B, int T, const int32_t* start, const int32_t* len, float* last_logits,
                          void* workspace, size_t ws_bytes, void* stream);

/* qk_rollout_teacher_forced and qk_rollout_sampled over a paged cache: the same
 * arguments, outputs, workspace (max_seq = per_row x page_size) and graph replay
 * (the replayed graph is cached per cache base, page layout, table pointer and
 * the call's buffers).  P + N <= per_row x page_size. */
int qk_rollout_teacher_forced_paged(qk_model* m, void* kv, const qk_kv_pages* pages,
                                    const int32_t* seq, int B, int P, int N, float* logprobs,
                                    int32_t* argmax, void* workspace, size_t ws_bytes, void* stream);
int qk_rollout_sampled_paged(qk_model* m, void* kv, const qk_kv_pages* pages, const int32_t* prompt,
                             int B, int P, int N, float tau, uint64_t seed, int32_t* tokens,
                             float* logprobs, void* workspace, size_t ws_bytes, void* stream);

/* Teacher-forced scoring (Eq. sft / Eq. ppo inputs): tokens dev int32 [B, T],
 * T >= 2.  logprobs dev fp32 [B, T-1]: logprobs[b, t] = log p(tokens[b, t+1] |
 * tokens[b, <= t]).  argmax dev int32 [B, T-1] or NULL.  Positions start at 0;
 * no KV cache is kept. */
int qk_score_logprobs(qk_model* m, const int32_t* tokens, int B, int T, float* logprobs,
                      int32_t* argmax, void* workspace, size_t ws_bytes, void* stream);

/* ---- GRPO token loss (Sec. "GRPO Optimization", Eq. advantage and Eq. ppo) --
 * Advantage of row b (Eq. advantage, no variance normalisation):
 *   A_b = rewards[b] - mean(rewards[g0 .. g0 + group - 1]),  g0 = b - b % group.
 * Per response token (Eq. ppo), rho = exp(lp - lp_old):
 *   loss_tok = -min(rho A_b, clip(rho, 1 - eps_low, 1 + eps_high) A_b) + beta * k3,
 *   k3 = exp(lp_ref - lp) - (lp_ref - lp) - 1  (the KL estimator is a reading:
 *   the paper does not name one).
 * loss_mean = sum(mask * loss_tok) / sum(mask) over the batch (0 for an empty
 * mask).  Every [B, T] array is dev fp32, row-major with row stride ld >= T;
 * mask dev uint8 (1 = response token) or NULL for all ones; lp_ref may be NULL
 * only when beta == 0; rewards dev fp32 [B] with B % group == 0.  loss_tok
 * receives all T entries of each row (masked ones included); loss_mean is dev
 * fp32 [1] or NULL.  Sums run in a fixed order (deterministic).  workspace:
 * qk_grpo_workspace_bytes(B) bytes of device scratch. */
int qk_grpo_workspace_bytes(int B, size_t* bytes);
int qk_grpo_token_loss(const float* lp, const float* lp_old, const float* lp_ref, int B, int T,
                       int ld, const float* rewards, int group, const uint8_t* mask,
                       float eps_low, float eps_high, float beta, float* loss_tok,
                       float* loss_mean, void* workspace, size_t ws_bytes, void* stream);

/* Scoring with the GRPO loss in its log-prob epilogue: as qk_score_logprobs for
 * tokens [B, T] (logprobs dev fp32 [B, T-1]), and where each log-prob is formed
 * its token loss as in qk_grpo_token_loss with ld = T-1 (lp_old, lp_ref, mask,
 * loss_tok [B, T-1]).  workspace: qk_workspace_bytes(QK_CALL_SCORE, B, T, T)
 * plus qk_grpo_workspace_bytes(B) bytes (the GRPO scratch follows the scoring
 * scratch, 256-byte aligned). */
int qk_score_grpo(qk_model* m, const int32_t* tokens, int B, int T, const float* lp_old,
                  const float* lp_ref, const float* rewards, int group, const uint8_t* mask,
                  float eps_low, float eps_high, float beta, float* logprobs, float* loss_tok,
                  float* loss_mean, void* workspace, size_t ws_bytes, void* stream);

/* Per-token coefficients of the GRPO gradient (Sec. "GRPO Optimization", Eq. ppo):
 * with loss_mean = sum(mask * loss_tok) / sum(mask) as in qk_grpo_token_loss,
 *   coef[b, t] = -mask[b, t] * (d loss_tok[b, t] / d lp[b, t]) / sum(mask),
 * so that qk_backward_logprob with these coefficients returns d loss_mean / d theta
 * (the chain rule through the log-probs; lp_old, lp_ref and the advantages are
 * constants).  d loss_tok / d lp = -rho A where rho A <= clip(rho) A (the unclipped
 * term is the minimum), 0 elsewhere (the clipped term is constant there), plus
 * beta (1 - exp(lp_ref - lp)).  Arguments and workspace as qk_grpo_token_loss
 * (loss_tok and loss_mean are written too); coef dev fp32 [B, ld], entries t < T.
 * All zero for an empty mask. */
int qk_grpo_coef(const float* lp, const float* lp_old, const float* lp_ref, int B, int T, int ld,
                 const float* rewards, int group, const uint8_t* mask, float eps_low, float eps_high,
                 float beta, float* coef, float* loss_tok, float* loss_mean, void* workspace,
                 size_t ws_bytes, void* stream);

/* ---- Backward pass (gradient of the token log-likelihood) -------------------
 * The SFT objective (Sec. "Task Serialization and SFT Objective", Eq. sft)
 * maximises log pi_theta(y* | x) over the target tokens; the GRPO objective
 * (Eq. ppo) depends on theta only through the same per-token log-probs.  Both
 * gradients are therefore the gradient of
 *   loss = sum_{b, t < T-1} coef[b, t] * (-log p(tokens[b, t+1] | tokens[b, <= t]))
 * for per-token coefficients coef (SFT: mask / number of target tokens; GRPO:
 * qk_grpo_coef).  tokens dev int32 [B, T], T >= 2, positions 0 .. T-1; coef dev
 * fp32 [B, T-1].  grads: host array of n_grads = qk_weight_count() device fp32
 * pointers, one per weight tensor in the canonical order and shape of
 * qk_model_load (row-major [out, in]), each 16-byte aligned; each receives
 * d loss / d tensor (accumulate == 0: overwritten; else added to).  loss dev fp32
 * [1] or NULL receives the loss.  workspace: qk_workspace_bytes(QK_CALL_BACKWARD,
 * B, T, 0), 256-byte aligned (it keeps every layer's forward activations, about
 * 1.1 GB per layer per 8192 tokens at Qwen3-8B size, the attention probabilities of
 * one layer and a [min(B T, 4096), V] block of logit gradients).  bf16 models
 * need head_dim 128 and vocab, hidden % 64 == 0 (QK_ESHAPE otherwise) and run each
 * row padded to a multiple of 128 positions inside the workspace (zero
 * coefficients after the row's end: causal attention keeps the padding invisible
 * to the real positions, so the result is that of the unpadded rows); fp32 models
 * take any shape.  Activations are rounded to
 * the model dtype where the forward pass rounds them (and the logit and attention
 * gradients, which are tensor-core operands, likewise); accumulation, norms,
 * softmax statistics, the residual gradient and every weight gradient are fp32.
 * Gain gradients sum in a fixed order; embedding rows that share a token are
 * added with fp32 atomics, and on bf16 models the attention's query gradient is
 * summed over key tiles by reductions in memory: both round in an order that can
 * differ between calls (a few 1e-3 of a gradient's norm after bf16 operands relay
 * it).  A token id outside
 * [0, V) sets QK_STATUS_BAD_TOKEN and counts as 0. */
int qk_backward_logprob(qk_model* m, const int32_t* tokens, int B, int T, const float* coef,
                        float* const* grads, int n_grads, int accumulate, float* loss,
                        void* workspace, size_t ws_bytes, void* stream);

/* Teacher-forced rollout: seq dev int32 [B, P+N+1] = prompt (P tokens) ++
 * c[0..N].  Prefill over the prompt scores c[0]; decode step j (0 <= j < N)
 * consumes c[j] at position P+j and scores c[j+1].  logprobs dev fp32 [B, N+1],
 * argmax dev int32 [B, N+1] or NULL.  The cache ends holding P+N positions;
 * P + N <= max_seq. */
int qk_rollout_teacher_forced(qk_model* m, void* kv, int max_batch, int max_seq,
                              const int32_t* seq, int B, int P, int N, float* logprobs,
                              int32_t* argmax, void* workspace, size_t ws_bytes, void* stream);

/* Sampled rollout at temperature tau > 0 (the paper samples at 1.0): prompt dev
 * int32 [B, P].  The prefill's last logits draw c[0]; decode step j (0 <= j < N)
 * consumes c[j] at position P+j and draws c[j+1].  A draw from softmax(z / tau)
 * is the Gumbel-max rule c = argmax_v (z_v / tau - log(-log u_v)) (lowest index on
 * ties), u_v the 24-bit uniform (floor(x / 2^40) + 1/2) / 2^24 of output
 * i = b 2^40 + j 2^18 + v of the SplitMix64 stream seeded with `seed` (row b,
 * step j, token v; needs B < 2^24, N < 2^22, vocab <= 2^18).  tokens dev int32
 * [B, N+1] receives c[0..N]; logprobs dev fp32 [B, N+1] receives
 * log softmax(z_j / tau)[c[j]].  Workspace and cache as qk_rollout_teacher_forced. */
int qk_rollout_sampled(qk_model* m, void* kv, int max_batch, int max_seq, const int32_t* prompt,
                       int B, int P, int N, float tau, uint64_t seed, int32_t* tokens,
                       float* logprobs, void* workspace, size_t ws_bytes, void* stream);

/* Synchronise `stream`, read the device status word into *flags (QK_STATUS_*
 * bits) and clear it.  Returns QK_ETIMEOUT if QK_STATUS_TIMEOUT was set (a
 * bounded device wait gave up; other bits may be set too and are in *flags),
 * else QK_EDEVICE if any other bit was set, QK_OK otherwise.  (A service call of
 * the library; the paper has no counterpart.) */
int qk_check_status(qk_model* m, void* stream, uint32_t* flags);

/* ---- measurement ----------------------------------------------------------
 * Kernel classes that qk_profile_begin can bracket with CUDA events.  Only the
 * launches made by decode steps (qk_decode_step, the decode phase of
 * qk_rollout_teacher_forced, qk_decode_layer) are bracketed. */
#define QK_PROF_QKV 0      /* RMSNorm'd input x W_qkv                     */
#define QK_PROF_O 1        /* attention output x W_o + residual           */
#define QK_PROF_GATE_UP 2  /* x W_gate, x W_up (with SwiGLU when fused)    */
#define QK_PROF_DOWN 3     /* h x W_down + residual                       */
#define QK_PROF_ATTN 4     /* decode attention (all its kernels)          */
#define QK_PROF_LM_HEAD 5  /* final RMSNorm'd x W_lm (logits)             */

/* Start bracketing up to max_launches launches of kernel class `kind` with
 * CUDA events recorded on the launching stream.  Creates 2*max_launches
 * events (host objects; no device allocation).  Replaces any active session. */
int qk_profile_begin(qk_model* m, int kind, int max_launches);
/* End the session: synchronise on its last event and return the summed
 * event-to-event time (ms) and the number of bracketed launches. */
int qk_profile_end(qk_model* m, float* total_ms, int* launches);

/* Number of kernels libqk has launched in this process (all models; a service
 * call for measurement, no counterpart in the paper). */
uint64_t qk_launch_count(void);

/* Message of the last failed call on this thread ("" if none; service call). */
const char* qk_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* QK_H */
