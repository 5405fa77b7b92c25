/*
 * grpo.h — C ABI of the GB300 (sm_103a) GRPO hot-path library (libgrpo.so).
 *
 * The library computes the data-parallel part of a GRPO policy update
 * (Section 3.3, Eq. 1 and Eq. 2): group-relative advantages, per-token
 * log-probabilities of sampled tokens through the LM head, the clipped-ratio
 * objective with a KL penalty, and the backward pass of that loss to the final
 * hidden states H and the LM-head weight W.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every array pointer is a DEVICE pointer owned by the caller; the library
 *   never frees or keeps it.  bf16 arrays are passed as their 16-bit patterns
 *   (uint16_t).  All matrices are row-major and densely packed.
 * - One exception: the hidden states H may also be page-locked host memory
 *   registered with CUDA (cudaHostAlloc, cudaMallocHost, cudaHostRegister).
 *   The row gather then reads the unmasked rows over the host link (the
 *   masked rows never cross it) instead of the caller copying every row to
 *   the device first.  As with an asynchronous copy, H must stay unchanged
 *   and allocated until the call's work on the stream has completed.
 *   Pageable host memory is GRPO_ERR_INVALID_ARG.
 * - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is
 *   enqueued on it; no entry point synchronises the stream except
 *   grpo_check_device_status.  Nothing is allocated: scratch space comes from
 *   the caller's workspace `ws` of `ws_bytes` bytes (see grpo_workspace_bytes).
 * - Errors the host can see (null pointers, bad sizes, misalignment, a
 *   workspace that is too small) return a status at once and enqueue nothing.
 *   Data-dependent problems found on the device (a target outside [0, V) on an
 *   unmasked row, a pipeline wait that timed out, a non-finite log-sum-exp)
 *   set bits of a status word inside the workspace; the affected rows' outputs
 *   are 0.  grpo_check_device_status reports that word.
 * - Outputs are overwritten, never accumulated into.  Results are
 *   deterministic: the one floating-point accumulation across launches (dH
 *   over vocabulary chunks, in the workspace) adds each chunk's value to each
 *   element once, in stream order, so the rounding order is fixed; nothing
 *   else uses atomics on floating-point values.
 * - One workspace must not be used by two calls that can run concurrently.
 */
#ifndef GRPO_H_
#define GRPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  GRPO_OK = 0,
  GRPO_ERR_INVALID_ARG = 1,   /* null pointer, bad size or alignment */
  GRPO_ERR_WORKSPACE = 2,     /* ws missing, misaligned or smaller than grpo_workspace_bytes */
  GRPO_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed */
  GRPO_ERR_DEVICE_CHECK = 4,  /* device found a bad target index or a non-finite value */
  GRPO_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up; outputs are invalid */
  GRPO_ERR_UNSUPPORTED = 6,   /* device is not sm_103 / sm_100 class, or shape beyond limits */
  GRPO_ERR_CAPACITY = 7       /* more unmasked rows than the workspace was sized for
                                 (grpo_workspace_bytes_rows); outputs are invalid */
} grpo_status;

/*
 * Which call a workspace is sized for (grpo_workspace_bytes `which`).
 * GRPO_WS_LOSS sizes the loss workspace of the default backward, which
 * recomputes each vocabulary chunk of the logits with a second GEMM: nothing
 * of [tokens x vocabulary] size is ever stored.  GRPO_WS_LOSS_LOGITS is an
 * opt-in: a loss workspace that also keeps the fp32 logits of the forward
 * ([rows x V], 4 bytes each: 12.2 GB for 19,572 unmasked rows at V 155136) so
 * that the backward forms dZ from them with an HBM-bound pass instead of
 * recomputing the logits GEMM.  A loss call keeps the logits only when its
 * ws_bytes is exactly such a size; see grpo_loss_plan.
 */
enum {
  GRPO_WS_LOGPROBS = 0,
  GRPO_WS_LOSS = 1,
  GRPO_WS_LOGPROBS_HEADS = 2,
  GRPO_WS_SAMPLE = 3,
  GRPO_WS_LOSS_LOGITS = 4,
  GRPO_WS_SAMPLE_TOP_P = 5
};

/* Most LM heads grpo_token_logprobs_heads sweeps in one call. */
enum { GRPO_MAX_HEADS = 4 };

/* Loss aggregation (grpo_loss_fwd_bwd `agg_mode`). */
enum {
  GRPO_AGG_TOKEN_MEAN = 0,    /* sum_t mask_t l_t / N_valid over the whole batch */
  GRPO_AGG_SEQ_MEAN = 1       /* Eq. 1 as printed: (1/n_resp) sum_i (1/|o_i|) sum_t l_{i,t} */
};

/*
 * Group-relative advantage, Eq. 2 (Section 3.3):
 *   A_i = (r_i - mean_g(r)) / (std_g(r) + eps)
 * over each group g of G consecutive responses; std is the sample standard
 * deviation (divisor G - 1).  Computed in fp64, rounded once to fp32.
 *   rewards  [n_resp] fp32 device, one reward per response
 *   adv_out  [n_resp] fp32 device
 * Requires G >= 2, n_resp >= 0 and n_resp % G == 0, else GRPO_ERR_INVALID_ARG.
 */
grpo_status grpo_group_advantages(const float* rewards, int64_t n_resp, int32_t G, float eps,
                                  float* adv_out, void* stream);

/*
 * Per-token log-probability of the sampled token, the pi_theta(o_{i,t} | q, o_{i,<t})
 * of Eq. 1 (Section 3.3):  logp_t = z_{t,y_t} - log sum_v exp(z_{t,v}),  z_t = H_t W^T.
 * The [T x V] logits are never written to memory.
 *   H        [T x Hd] bf16 device (or page-locked host, see above), final hidden
 *            states (16-byte aligned)
 *   W        [V x Hd] bf16 device, LM-head weight (16-byte aligned)
 *   targets  [T] int32 device, sampled token ids, must lie in [0, V) where mask != 0
 *   mask     [T] uint8 device, 0 = padding row
 *   logp_out [T] fp32 device; padding rows get 0
 *   ws       device workspace of at least grpo_workspace_bytes(T, Hd, V, GRPO_WS_LOGPROBS)
 *            bytes, 256-byte aligned
 * Requires Hd % 64 == 0, 0 < V < 2^31, 0 <= T < 2^31.
 */
grpo_status grpo_token_logprobs(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                const uint8_t* mask, int64_t T, int32_t Hd, int64_t V,
                                float* logp_out, void* ws, size_t ws_bytes, void* stream);

/*
 * grpo_token_logprobs for n_heads LM heads at once: the log-probs of the same
 * sampled tokens under the current policy, the old policy (the pi_theta_old
 * of Eq. 1's ratio) and the reference policy (the pi_ref of Eq. 1's KL term),
 * as the rollout-scoring step of GRPO needs them.  The unmasked rows are
 * gathered once and every head is swept in one launch.
 *   W_heads   HOST array of n_heads device pointers, each a [V x Hd] bf16 head
 *             (16-byte aligned); 1 <= n_heads <= GRPO_MAX_HEADS
 *   logp_out  [n_heads x T] fp32 device: row h holds head h's log-probs,
 *             0 on padding rows
 *   ws        at least grpo_workspace_bytes(T, Hd, V, GRPO_WS_LOGPROBS_HEADS) bytes
 * Other arguments and limits as grpo_token_logprobs.
 */
grpo_status grpo_token_logprobs_heads(const uint16_t* H, const uint16_t* const* W_heads, int32_t n_heads,
                                      const int32_t* targets, const uint8_t* mask, int64_t T, int32_t Hd,
                                      int64_t V, float* logp_out, void* ws, size_t ws_bytes, void* stream);

/*
 * The rollout draw of Eq. 1, {o_i} ~ pi_theta_old: for every unmasked row t,
 * sample o_t from softmax(H_t W^T / temperature) by the Gumbel-max rule
 *   o_t = argmax_v  z_{t,v} / temperature + G_{t,v}   (lowest v on a tie)
 * with G = -log(-log U) and U = ((w >> 9) + 1/2) / 2^23, w = word (v mod 4) of
 * Philox4x32-10 at counter (v / 4, t, offset mod 2^32, offset / 2^32) and key
 * (seed mod 2^32, seed / 2^32).  The logits never reach memory.
 *   mask        [T] uint8 device: rows to sample (0: token -1, log-prob 0)
 *   tokens_out  [T] int32 device, the sampled token ids
 *   logp_out    [T] fp32 device, log softmax(z_t / temperature) at the sampled token
 *   ws          at least grpo_workspace_bytes(T, Hd, V, GRPO_WS_SAMPLE) bytes
 * temperature must be finite and > 0; the same (seed, offset) gives the same draw.
 * Other arguments and limits as grpo_token_logprobs.
 */
grpo_status grpo_sample_tokens(const uint16_t* H, const uint16_t* W, const uint8_t* mask, int64_t T, int32_t Hd,
                               int64_t V, float temperature, uint64_t seed, uint64_t offset, int32_t* tokens_out,
                               float* logp_out, void* ws, size_t ws_bytes, void* stream);

/*
 * grpo_sample_tokens restricted to the nucleus (top-p truncation; the rollout
 * draw before Eq. 1, Section 3.3; the paper names no sampling parameters, this
 * is the common nucleus rule of Holtzman et al., 2020): with y = z_t /
 * temperature and p = softmax(y), the nucleus is the shortest set of the most
 * probable tokens whose mass reaches top_p together with every token tied with
 * its least probable member, and
 *   o_t = argmax over v in the nucleus of  y_v + G_{t,v}   (lowest v on a tie)
 * with G exactly as grpo_sample_tokens defines it, which draws from p
 * renormalised on the nucleus; top_p = 1 draws the same tokens as
 * grpo_sample_tokens.  The forward GEMM stores the fp32 logits of the unmasked
 * rows in the workspace (4 * V bytes per row) and keeps each vocabulary
 * split's best perturbed score; a streaming pass lists the rows whose plain
 * winner may fall outside the nucleus, and only those are resolved exactly:
 * the threshold from masses in 2^-40 fixed point (so the result does not
 * depend on the order of the sums), then the argmax over the nucleus from the
 * splits' winners, walking only the splits whose winner falls outside.
 *   top_p       in (0, 1]
 *   logp_out    [T] fp32 device, log softmax(y) at the sampled token (the
 *               untruncated distribution; subtract log of the nucleus mass for
 *               the truncated one)
 *   ws          at least grpo_workspace_bytes(T, Hd, V, GRPO_WS_SAMPLE_TOP_P)
 *               bytes (or grpo_workspace_bytes_rows for fewer unmasked rows)
 * Other arguments, outputs and limits as grpo_sample_tokens.
 */
grpo_status grpo_sample_tokens_top_p(const uint16_t* H, const uint16_t* W, const uint8_t* mask, int64_t T,
                                     int32_t Hd, int64_t V, float temperature, float top_p, uint64_t seed,
                                     uint64_t offset, int32_t* tokens_out, float* logp_out, void* ws, size_t ws_bytes,
                                     void* stream);

/*
 * The noise grpo_sample_tokens adds, written out for checking the generator
 * and the logarithms (the draw of Eq. 1 has no other observable):
 *   out[(t - row0) * cols + v] = G_{t,v}  for row0 <= t < row0 + rows, 0 <= v < cols
 * with G, U and the Philox counter exactly as grpo_sample_tokens defines them
 * (t is the token position).  out is [rows x cols] fp32 device memory (4-byte
 * aligned); row0 >= 0, row0 + rows <= 2^32, cols < 2^31, rows * cols <= 2^40.
 * Asynchronous on `stream`.
 */
grpo_status grpo_gumbel_noise(uint64_t seed, uint64_t offset, int64_t row0, int64_t rows, int64_t cols,
                              float* out, void* stream);

/*
 * GRPO loss (the negated objective of Eq. 1, Section 3.3) and its gradient
 * with respect to H and W.  Per unmasked token t of response i = t / L:
 *   rho  = exp(logp_t - old_logp_t)
 *   s    = min(rho A_i, clip(rho, 1 - clip_eps, 1 + clip_eps) A_i)
 *   KL   = exp(ref_logp_t - logp_t) - (ref_logp_t - logp_t) - 1
 *   l_t  = -s + beta KL,     loss = sum_t w_t l_t
 * with w_t from agg_mode.  At the kink of min() the unclipped branch is taken.
 *   H, W, targets, mask  as for grpo_token_logprobs, with T = n_resp * L
 *   old_logp, ref_logp   [T] fp32 device: log-probs of the old and reference policies
 *   adv                  [n_resp] fp32 device (e.g. from grpo_group_advantages)
 *   loss_out             device pointer to one fp32
 *   dH                   [T x Hd] fp32 device; padding rows get 0
 *   dW                   [V x Hd] fp32 device
 *   ws                   at least grpo_workspace_bytes(T, Hd, V, GRPO_WS_LOSS) bytes:
 *                        the backward recomputes the logits chunk by chunk and
 *                        never stores them.  Opt-in: exactly
 *                        grpo_workspace_bytes(T, Hd, V, GRPO_WS_LOSS_LOGITS)
 *                        bytes keep the fp32 logits from the forward for the
 *                        backward (bit-identical results, see grpo_loss_plan)
 * Requires n_resp >= 1, L >= 1, clip_eps >= 0, agg_mode in {0, 1}, dH and dW
 * 16-byte aligned, and the limits of grpo_token_logprobs.
 */
grpo_status grpo_loss_fwd_bwd(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                              const uint8_t* mask, const float* old_logp, const float* ref_logp,
                              const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                              float clip_eps, float beta, int32_t agg_mode, float* loss_out,
                              float* dH, float* dW, void* ws, size_t ws_bytes, void* stream);

/*
 * grpo_loss_fwd_bwd with the normaliser of the aggregation given by the
 * caller, for data-parallel training where each rank holds a shard of the
 * batch (whole prompt groups) and the loss is normalised over the global
 * batch (Eq. 1's expectation over all prompts of the step):
 *   agg_mode 0: w_t = mask_t / norm        (norm = N_valid summed over ranks)
 *   agg_mode 1: w_t = mask_t / (norm |o_i|) (norm = n_resp summed over ranks)
 * norm == 0 uses the local count (this is exactly grpo_loss_fwd_bwd).  With
 * the global norm on every rank, the sum over ranks of loss, and of dW, is the
 * loss and dW of the whole batch.  norm must be finite and >= 0.
 */
grpo_status grpo_loss_fwd_bwd_norm(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                   const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                   const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                   float clip_eps, float beta, int32_t agg_mode, float norm,
                                   float* loss_out, float* dH, float* dW, void* ws, size_t ws_bytes,
                                   void* stream);

/*
 * grpo_loss_fwd_bwd_norm with a cap on the per-token KL value (Eq. 1's
 * D_KL term; the paper leaves the estimator open):
 *   KL_t = min(k3_t, kl_clamp),  k3_t = exp(ref_logp_t - logp_t) - (ref_logp_t - logp_t) - 1
 * A token whose k3 lies above the cap adds beta * kl_clamp to its loss term and
 * nothing to the gradient through the KL; a tie counts as below the cap.  This
 * bounds the penalty of the few tokens on which the reference and the policy
 * disagree by many nats.  kl_clamp must be >= 0 (not NaN); +infinity is
 * exactly grpo_loss_fwd_bwd_norm, and 0 removes the KL term (k3 >= 0).
 * Every other argument as grpo_loss_fwd_bwd_norm.
 */
grpo_status grpo_loss_fwd_bwd_kl_clamp(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                       const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                       const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                       float clip_eps, float beta, int32_t agg_mode, float norm, float kl_clamp,
                                       float* loss_out, float* dH, float* dW, void* ws, size_t ws_bytes,
                                       void* stream);

/*
 * Rows of dW (vocabulary ids) per backward chunk: chunk c of
 * grpo_loss_fwd_bwd* covers rows [c * cols, min(V, (c + 1) * cols)).  cols is
 * 16384, or the environment variable GRPO_VOCAB_CHUNK (rounded up to a
 * multiple of 256) when set, capped at V rounded up to 256; the loss calls read
 * the same variable, so query under the same environment.  0 for V <= 0.
 */
int64_t grpo_vocab_chunk_cols(int64_t V);

/*
 * grpo_loss_fwd_bwd_norm that also records chunk_events[c] on `stream` as
 * soon as chunk c's rows of dW are written (and *loss_out, computed before the
 * backward, is final from chunk_events[0] on).  A data-parallel caller makes
 * its communication stream wait on each event and starts that chunk's dW
 * all-reduce while the later chunks still compute: the one exchange step of
 * the data-parallel path (dW summed over ranks) then overlaps the backward.
 *   chunk_events  HOST array of n_events cudaEvent_t handles, created by the
 *                 caller on the current device; entries 0 .. chunks - 1 are
 *                 recorded, chunks = ceil(V / grpo_vocab_chunk_cols(V))
 *   n_events      >= chunks, else GRPO_ERR_INVALID_ARG (nothing launched)
 * Every other argument as grpo_loss_fwd_bwd_norm.
 */
grpo_status grpo_loss_fwd_bwd_events(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                     const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                     const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                     float clip_eps, float beta, int32_t agg_mode, float norm, float* loss_out,
                                     float* dH, float* dW, void* const* chunk_events, int32_t n_events, void* ws,
                                     size_t ws_bytes, void* stream);

/*
 * grpo_loss_fwd_bwd_norm for a caller that wants dW in host memory: each
 * vocabulary chunk of dW is copied to dW_host as soon as it is computed, on
 * an internal copy stream (created once per device), so the copy of the
 * 2.5 GB gradient of an 8B head overlaps the rest of the backward instead of
 * following it.  dW (device) is still written.  When `stream` reaches the end
 * of the call's work, dW_host holds dW.
 *   dW_host  [V x Hd] fp32 HOST memory, page-locked (cudaHostAlloc /
 *            cudaHostRegister), 16-byte aligned; must stay valid until then
 */
grpo_status grpo_loss_fwd_bwd_to_host(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                      const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                      const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                      float clip_eps, float beta, int32_t agg_mode, float norm, float* loss_out,
                                      float* dH, float* dW, float* dW_host, void* ws, size_t ws_bytes,
                                      void* stream);

/*
 * grpo_loss_fwd_bwd_norm followed by the actor's optimiser step on the LM
 * head, with the step fused into the dW GEMM: each dW tile is consumed in
 * place by one AdamW step (Adam with decoupled weight decay) and dW itself is
 * never written.  The paper sets the actor learning rate (1e-6, Section 4.1)
 * but not the optimiser; AdamW is the reading taken:
 *   m <- beta1 m + (1 - beta1) g,  v <- beta2 v + (1 - beta2) g^2,
 *   W_master <- W_master (1 - lr wd) - lr (m / (1 - beta1^step)) / (sqrt(v / (1 - beta2^step)) + eps)
 *   W_master, exp_avg, exp_avg_sq   [V x Hd] fp32 device, updated in place
 *   W_out                           [V x Hd] bf16 device, receives bf16(W_master);
 *                                   may be W itself (the rows of a vocabulary chunk are
 *                                   no longer read when its update runs)
 *   step >= 1 (bias correction), 0 <= beta1, beta2 < 1, eps > 0, lr >= 0, weight_decay >= 0.
 * Everything else as grpo_loss_fwd_bwd_norm (loss_out and dH are written).
 */
grpo_status grpo_loss_fwd_bwd_adamw(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                    const uint8_t* mask, const float* old_logp, const float* ref_logp,
                                    const float* adv, int64_t n_resp, int64_t L, int32_t Hd, int64_t V,
                                    float clip_eps, float beta, int32_t agg_mode, float norm, float lr,
                                    float beta1, float beta2, float eps, float weight_decay, int64_t step,
                                    float* W_master, float* exp_avg, float* exp_avg_sq, uint16_t* W_out,
                                    float* loss_out, float* dH, void* ws, size_t ws_bytes, void* stream);

/*
 * One AdamW step over n fp32 elements (the same update as
 * grpo_loss_fwd_bwd_adamw, as a separate bandwidth-bound pass over a stored
 * gradient, e.g. the dW of grpo_loss_fwd_bwd).  W_master, exp_avg,
 * exp_avg_sq are updated in place; W_out receives bf16(W_master).  All
 * pointers are device memory, 16-byte aligned; n % 4 == 0.  Hyper-parameter
 * limits as grpo_loss_fwd_bwd_adamw.
 */
grpo_status grpo_adamw_step(float* W_master, float* exp_avg, float* exp_avg_sq, const float* grad,
                            uint16_t* W_out, int64_t n, float lr, float beta1, float beta2, float eps,
                            float weight_decay, int64_t step, void* stream);

/*
 * grpo_token_logprobs without a workspace argument, for callers that cannot
 * allocate device memory themselves: code running where cudaMalloc is not
 * allowed or would stall the device (inside a stream capture, in a real-time
 * loop with a fixed memory budget), or a binding that has no device allocator.
 * The paper has no counterpart; this is a deployment convenience.
 *
 * Scratch space is a fixed 64 MiB array of device memory inside libgrpo.so,
 * held on every GPU that loads the library until the process exits.  The
 * call allocates nothing: no cudaMalloc, no cudaFree, no allocating library
 * routine.  Arguments, layout and results are those of grpo_token_logprobs.
 *   - Returns GRPO_ERR_WORKSPACE if grpo_workspace_bytes(T, Hd, V,
 *     GRPO_WS_LOGPROBS) exceeds 64 MiB (7,680 tokens at Hd 4096,
 *     V 155136), GRPO_ERR_INVALID_ARG for arguments grpo_token_logprobs rejects.
 *   - Every call looks up the array's device address in the current device's
 *     context (so a context made after cudaDeviceReset gets its own).  The
 *     first call on a device also loads the library's device code there; make
 *     that first call before any stream capture.
 *   - Every call uses the same array and leaves its contents behind; each call
 *     clears what it needs cleared.  Calls whose work can overlap on the GPU
 *     (different streams, or different host threads) race on the array and
 *     give wrong results: serialise them.
 *   - Device-side problems (a target outside [0, V), a non-finite log-sum-exp)
 *     give 0 for the affected rows as in grpo_token_logprobs and set the
 *     array's device status word: read it with grpo_noalloc_check_status.
 */
grpo_status grpo_token_logprobs_noalloc(const uint16_t* H, const uint16_t* W, const int32_t* targets,
                                        const uint8_t* mask, int64_t T, int32_t Hd, int64_t V,
                                        float* logp_out, void* stream);

/*
 * grpo_check_device_status for the fixed array of grpo_token_logprobs_noalloc
 * (the paper has no counterpart): synchronises `stream`, then reports the
 * device status word the last no-alloc call on the current device left
 * behind, as GRPO_OK, GRPO_ERR_DEVICE_CHECK, GRPO_ERR_TIMEOUT or
 * GRPO_ERR_CAPACITY (GRPO_ERR_CUDA if the array cannot be reached).  Allocates
 * nothing.  The word is cleared at the start of every no-alloc call, and a
 * no-alloc call still running on another stream may change it.
 */
grpo_status grpo_noalloc_check_status(void* stream);

/*
 * Bytes of workspace the call `which` (GRPO_WS_LOGPROBS, GRPO_WS_LOSS,
 * GRPO_WS_LOGPROBS_HEADS, GRPO_WS_SAMPLE, GRPO_WS_LOSS_LOGITS or
 * GRPO_WS_SAMPLE_TOP_P) needs for T tokens, hidden size Hd and vocabulary V.
 * Returns 0 for arguments the calls would reject.  Sized for the worst case
 * N_valid = T.
 */
size_t grpo_workspace_bytes(int64_t T, int32_t Hd, int64_t V, int32_t which);

/*
 * Bytes of workspace for the call `which` on batches of T padded tokens of
 * which at most max_valid are unmasked (e.g. a ragged rollout batch where most
 * rows are padding): the regions that hold one row per unmasked token (the
 * gathered hidden states and, for the loss, its transposed copy, the dZ chunk
 * and the compacted dH) are sized for max_valid rounded up to 256 rows instead
 * of T.  At the 1M-row ragged 8B batch (168k unmasked) the loss workspace
 * shrinks from 69 GB to about 11 GB.  Every call accepts such a smaller
 * workspace: it derives the row capacity from ws_bytes.  A batch with more
 * unmasked rows than the capacity is not an error the host can see (the count
 * is only known on the device): the device status becomes GRPO_ERR_CAPACITY,
 * rows past the capacity get no output (0 / token -1), and every other output
 * of that call is invalid.  Returns 0 for arguments the calls would reject
 * or a negative max_valid; max_valid >= T gives grpo_workspace_bytes.
 */
size_t grpo_workspace_bytes_rows(int64_t T, int64_t max_valid, int32_t Hd, int64_t V, int32_t which);

/*
 * How the loss calls (grpo_loss_fwd_bwd and its variants) use a workspace of
 * ws_bytes for T tokens, hidden size Hd and vocabulary V (no device work; the
 * paper has no counterpart).  Returns 1 when the forward keeps the fp32
 * logits for the backward, 0 when the backward recomputes them with a second
 * logits GEMM, -1 for arguments or a workspace the calls would reject; *rows
 * (if not null) gets the row capacity (unmasked rows the call can hold).
 * The logits are kept only when ws_bytes is exactly what grpo_workspace_bytes
 * or grpo_workspace_bytes_rows returns for GRPO_WS_LOSS_LOGITS (and not also
 * exactly the plain layout's size); the row capacity is then the one it was
 * sized for (max_valid rounded up to 256 rows).  Any other size, however
 * large, runs the recomputing backward with the largest plain capacity that
 * fits, so a caller who never asks for the logits never gets them stored.
 * Both ways give bit-identical loss, dH and dW: the two GEMMs accumulate the
 * same logits in the same order, and both form dZ with the same arithmetic.
 */
int32_t grpo_loss_plan(int64_t T, int32_t Hd, int64_t V, size_t ws_bytes, int64_t* rows);

/*
 * Synchronises `stream`, reads the device status word of workspace `ws`
 * (written by the last call that used it) and returns GRPO_OK,
 * GRPO_ERR_DEVICE_CHECK or GRPO_ERR_TIMEOUT.  The word is cleared at the
 * start of every compute call.
 */
grpo_status grpo_check_device_status(void* ws, void* stream);

/* Static, human-readable name of a status code. */
const char* grpo_status_string(grpo_status status);

/*
 * Launch tracing (profiling aid; the paper has no counterpart).
 * Kernel classes reported by grpo_trace_read:
 */
enum {
  GRPO_K_ADVANTAGES = 0,  /* Eq. 2 reduction */
  GRPO_K_COMPACT = 1,     /* mask scan / scatter and the gather of unmasked rows */
  GRPO_K_LSE_GEMM = 2,    /* logits GEMM + online log-sum-exp + target gather */
  GRPO_K_LOGP_MERGE = 3,  /* merge of vocabulary splits -> logp */
  GRPO_K_LOSS = 4,        /* merge + Eq. 1 terms, dloss/dlogp, loss reduction */
  GRPO_K_DZ_GEMM = 5,     /* recomputed logits -> dZ chunk (bf16) */
  GRPO_K_DH_GEMM = 6,     /* dH (+)= dZ_chunk W_chunk */
  GRPO_K_DW_GEMM = 7,     /* dW_chunk = dZ_chunk^T H */
  GRPO_K_DH_ROWS = 8,     /* dH rows from the compacted order to the padded one (padding rows 0) */
  GRPO_K_ADAMW = 9,       /* standalone AdamW step (grpo_adamw_step) */
  GRPO_K_SAMPLE_GEMM = 10, /* logits GEMM + log-sum-exp + Gumbel-max draw */
  GRPO_K_TRANSPOSE = 11,  /* K-major (transposed) copy of the gathered hidden states for dW */
  GRPO_K_DZ_LOGITS = 12,  /* kept logits -> dZ chunk (bf16), element-wise */
  GRPO_K_TOP_P = 13       /* nucleus threshold + Gumbel-max over the kept logits (per row) */
};

/*
 * enable != 0: from now on, every kernel launch of the compute calls (from
 * any host thread) is bracketed by two CUDA events recorded on its stream;
 * the record is cleared.  enable == 0 stops recording (the record is kept).
 * Events are created on first use and reused; tracing costs two event
 * records per launch and nothing when disabled.
 */
grpo_status grpo_trace_enable(int32_t enable);

/*
 * Waits for the traced launches to finish and writes up to max_records of
 * them, oldest first: kind[i] (GRPO_K_*), cols[i] (vocabulary columns the
 * launch covered, or 0) and ms[i] (device time between its two events).
 * Returns the total number of records (may exceed max_records), or -1 if an
 * event query failed.  Pointers are host memory; any may be NULL when
 * max_records is 0.
 */
int32_t grpo_trace_read(int32_t* kind, int64_t* cols, float* ms, int32_t max_records);

#ifdef __cplusplus
}
#endif

#endif /* GRPO_H_ */
