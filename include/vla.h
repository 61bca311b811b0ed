/*
 * vla.h — C ABI of the GB300 (sm_103a) rollout / re-scoring hot path of VLA-RL
 * (arXiv 2505.18719).
 *
 * The policy is an auto-regressive Llama-2-style decoder (paper §3.1: OpenVLA-7B, whose
 * core is Llama-2-7B).  A rollout step (Algorithm 1, rollout phase) feeds each environment's
 * state — projected visual embeddings h(o_t) followed by instruction ids v_t^in — and
 * generates the n = |A| = 7 action tokens v_t^out (§3.3), each one of the 256 action bins
 * (§3.1).  a_t = f(v_t^out) maps bins to continuous values; log π(a_t|·) is the sum of the
 * token log-probs (Eq. 1), which the learning phase re-computes for the PPO ratio (Eq. 2).
 * A trajectory is a multi-turn conversation (§3.3): each step appends to the same context.
 * The paper runs this path as large-batch decoding on one dedicated inference GPU (§3.5).
 *
 * Conventions for every call:
 *  - All device pointers are CUDA device memory on the handle's device, 16-byte aligned.
 *    Weights are BORROWED: the caller keeps them alive for the handle's life.  The four
 *    projection matrices (q|k|v, o, gate|up, down) are read once into an fp16 copy that the
 *    handle owns (vla_create; again at vla_sync_weights after the caller changed them, e.g.
 *    after a learner update); every other weight is read where it lies at each call.
 *    Output buffers are caller-allocated device memory.  The handle owns its KV cache,
 *    workspaces and the fp16 projection copy (allocated in vla_create, freed in vla_destroy).
 *  - Arithmetic: every projection runs on fp16 tensor-core operands with fp32 accumulation.
 *    Its input activation is carried as an fp16 pair hi + lo (~21 significant bits); the
 *    weight-streaming GEMMs (calls of at most 128 rows: decode steps of up to 128 envs)
 *    multiply both halves, the tile GEMMs (prefill, score, larger decode batches) both halves
 *    for q|k|v and hi alone for o, gate|up and down.  K/V are cached in fp16 plus a 4-bit
 *    residual per element (value = hi + (2c - 15) ulp(hi) / 32, within ulp(hi) / 32 of the
 *    computed key / value), and every attention reads both.  A finite
 *    activation beyond the fp16 range (|x| > 65504) is stored as +-65504 and raises
 *    VLA_STATUS_SATURATED in the status word (reported by the next vla_sync).
 *  - Calls are asynchronous on the handle's stream.  Host-checkable errors return at once,
 *    with no side effects.  Errors found on the device (token id out of range, non-finite
 *    logits, a pipeline wait that timed out) set a device status word; the next vla_sync
 *    returns VLA_ERR_DEVICE_STATUS and clears it.
 *  - One handle per stream; a handle is not thread-safe.
 *  - bf16 = IEEE bfloat16 bits (uint16); matrices are row-major, nn.Linear layout [out, in].
 */
#ifndef VLA_H_
#define VLA_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct vla_handle vla_handle;

typedef enum {
  VLA_OK = 0,
  VLA_ERR_ARG = -1,           /* bad argument (NULL, size, shape, temperature < 0 / NaN) */
  VLA_ERR_CAPACITY = -2,      /* KV capacity per env or tokens per call would be exceeded */
  VLA_ERR_STATE = -3,         /* decode / score before any prefill                         */
  VLA_ERR_CUDA = -4,          /* a CUDA runtime call failed (message in vla_last_error)    */
  VLA_ERR_OOM = -5,           /* device allocation failed in vla_create                    */
  VLA_ERR_DEVICE_STATUS = -6, /* a kernel flagged an error (see vla_last_error)            */
  VLA_ERR_UNSUPPORTED = -7    /* shape outside what the kernels implement                 */
} vla_status;

/* Device status bits (reported through vla_last_error after VLA_ERR_DEVICE_STATUS). */
#define VLA_STATUS_BAD_TOKEN 0x1u     /* token id outside [0, vocab) (id 0 used instead)  */
#define VLA_STATUS_NONFINITE 0x2u     /* a logit was NaN or infinite                       */
#define VLA_STATUS_TIMEOUT 0x4u       /* a pipeline wait in the GEMM exceeded its limit    */
#define VLA_STATUS_BAD_FORCED 0x8u    /* forced / scored token not an action-bin id        */
#define VLA_STATUS_SATURATED 0x10u    /* a finite GEMM input activation beyond the fp16 range
                                         (|x| > 65504) was stored as +-65504 (results of that
                                         call are not those of the model)                  */

/* Model and handle sizes.
 * Supported: head_dim in {64, 128}; n_heads * head_dim == d_model; d_model % 128 == 0;
 *   d_model <= 6400;
 * d_ffn % 8 == 0; n_action_bins == 256; 1 <= action_dim <= 16; vocab >= n_action_bins. */
typedef struct {
  int n_layers, d_model, n_heads, head_dim, d_ffn, vocab;
  int n_action_bins; /* 256: the last 256 vocabulary ids, bin k <-> id vocab-256+k       */
  int action_dim;    /* 7 (= |A|, Eq. 1)                                                   */
  int max_batch;     /* environments per handle                                            */
  int kv_capacity;   /* KV positions per environment                                       */
  int max_tokens;    /* max rows of one vla_prefill call (sum of chunk lengths) and >= 6*B */
  float rms_eps;     /* 1e-6                                                               */
  float rope_theta;  /* 1e4                                                                */
} vla_config;

/* Weight pointers (device bf16), per-layer arrays have n_layers entries (host arrays of
 * device pointers; the host arrays are copied in vla_create). */
typedef struct {
  const void* embed;             /* [vocab, d]                                  */
  const void* const* attn_norm;  /* [L] -> [d]                                  */
  const void* const* wqkv;       /* [L] -> [3d, d], rows q | k | v              */
  const void* const* wo;         /* [L] -> [d, d]                               */
  const void* const* ffn_norm;   /* [L] -> [d]                                  */
  const void* const* w_gate_up;  /* [L] -> [2F, d], rows gate | up              */
  const void* const* w_down;     /* [L] -> [d, F]                               */
  const void* final_norm;        /* [d]                                         */
  const void* lm_head;           /* [vocab, d]; only the last 256 rows are read */
} vla_weights;

/* Create a handle on the current CUDA device.  `cuda_stream` is a cudaStream_t (NULL =
 * the legacy default stream).  Allocates the KV cache
 * (n_layers * max_batch * 2 * d_model * kv_capacity fp16, and half a byte per element for its
 * residual codes), the fp16 copy of the projection
 * matrices (n_layers * (4 d^2 + 3 d_ffn d) fp16) and workspaces, then fills the copy from the
 * bf16 weights and waits for it.  A bf16 weight with 2^-14 <= |w| <= 65504 is exact in
 * fp16; a smaller one rounds to a multiple of 2^-24.
 * Returns VLA_ERR_ARG / VLA_ERR_UNSUPPORTED (also: a projection weight with |w| > 65504 or
 * not finite) / VLA_ERR_OOM / VLA_ERR_CUDA on failure, with *out = NULL. */
int vla_create(const vla_config* cfg, const vla_weights* w, void* cuda_stream, vla_handle** out);

/* Prefill (Algorithm 1: h(o_t) then π_θ over the state; §3.3 multi-turn append).
 * For env b in [0, batch): its chunk is
 *     [pending 7th action token of its previous turn, if any]
 *   ‖ visual[b, 0:n_visual, :]            (device bf16 [batch, n_visual, d])
 *   ‖ embed[token_ids[b, 0:lengths[b]]]   (device int32 [batch, max_len]; HOST lengths)
 * appended to env b's context at positions len_b, len_b+1, ...  Chunk rows run through all
 * layers; their K/V enter the cache.  The last row's hidden state is kept for the first
 * action token.  Envs >= batch are untouched.  Requires len_b + chunk_b + 6 <= kv_capacity
 * and sum_b chunk_b <= max_tokens (else VLA_ERR_CAPACITY), chunk_b >= 1.
 * Token ids outside [0, vocab) set VLA_STATUS_BAD_TOKEN and read row 0. */
int vla_prefill(vla_handle* h, int batch, const void* visual, int n_visual,
                const int32_t* token_ids, const int32_t* lengths, int max_len);

/* Decode the action tokens of the latest turn (Algorithm 1: π_θ generates, f extracts,
 * Eq. 1 log-probs) for the envs of the latest prefill (B = its batch).
 *   uniforms      device f32 [B, action_dim, 256], values in (0,1) (clamped to
 *                 [2^-24, 1-2^-24]); token i of env b uses uniforms[b, i, :].
 *   temperature   T > 0: Gumbel-max sample k = argmax(z/T - log(-log u)), log-probs of
 *                 softmax(z/T) over the 256 bins.  T == 0: greedy argmax z, T = 1 log-probs.
 *   forced_tokens device int32 [B, action_dim] or NULL.  When given, token i fed to step
 *                 i+1 is forced_tokens[b, i] (teacher forcing) and logprobs_out holds the
 *                 forced token's log-prob; tokens_out / actions_out still report the sample.
 *   tokens_out    device int32 [B, action_dim]: vocab id vocab-256+k.
 *   logprobs_out  device f32 [B, action_dim].
 *   actions_out   device f32 [B, action_dim]: bin centre -1 + (2k+1)/256 (exact).
 *   logits_out    device f32 [B, action_dim, 256] or NULL: the untempered bin logits z.
 * Ties in the argmax go to the lowest bin.  The last token stays pending: its K/V are
 * written as the first row of the next prefill.  Calling decode again re-decodes the same
 * turn from its prefill state.  VLA_ERR_STATE before any prefill. */
int vla_decode_actions(vla_handle* h, const float* uniforms, float temperature,
                       const int32_t* forced_tokens, int32_t* tokens_out, float* logprobs_out,
                       float* actions_out, float* logits_out);

/* Teacher-forced re-scoring of the latest turn (the PPO ratio pass, Eq. 2): log-probs of
 * the given action tokens (device int32 [B, action_dim], action-bin ids) under this
 * handle's weights, at `temperature` (same meaning as in decode; the log-probs of T = 0
 * are those of T = 1).  The turn's actions become the given tokens (their K/V replace any
 * decoded ones; the last one is pending).  logprobs_out device f32 [B, action_dim];
 * logits_out device f32 [B, action_dim, 256] or NULL.  Tokens outside the action bins set
 * VLA_STATUS_BAD_FORCED.  VLA_ERR_STATE before any prefill. */
int vla_score_actions(vla_handle* h, const int32_t* tokens, float temperature,
                      float* logprobs_out, float* logits_out);

/* Rollout entropy (the training-dynamics quantity of §4.2): H = -sum_k p_k log p_k of each
 * action token's 256-bin distribution in the latest vla_decode_actions or vla_score_actions
 * call on this handle, at that call's temperature (T == 0: the T = 1 distribution, as for
 * the log-probs).  entropy_out device f32 [B, action_dim]; asynchronous on the handle's
 * stream.  VLA_ERR_STATE if neither has run since the latest prefill. */
int vla_action_entropy(vla_handle* h, float* entropy_out);

/* Value-model estimate V_t of Algorithm 1 at each env's latest prefill (the step's state),
 * for a handle whose decoder is a homogeneous value model (the policy's architecture with
 * one scalar output): V_b = RMSNorm(h_b; final_norm) . w_value + bias, h_b the last
 * prefix row's final hidden state.  w_value device bf16 [d_model] (read during the call);
 * values_out device f32 [B].  VLA_ERR_STATE before any prefill. */
int vla_value(vla_handle* h, const void* w_value, float bias, float* values_out);

/* Generalised advantage estimation (Algorithm 1, "compute advantages"), all device f32:
 *   rewards [M, B], values [M + 1, B] (V_0 .. V_M; V_M bootstraps the unfinished tail),
 *   dones [M, B] (1 where the episode ended with step t, else 0);
 *   delta_t = r_t + gamma (1 - done_t) V_{t+1} - V_t,
 *   A_t = delta_t + gamma lam (1 - done_t) A_{t+1} (A_M = 0) -> adv_out [M, B];
 *   returns_out [M, B] = A_t + V_t, or NULL.
 * Needs M, B >= 1 and 0 <= gamma, lam <= 1 (else VLA_ERR_ARG).  Asynchronous on cuda_stream. */
int vla_gae(const float* rewards, const float* values, const float* dones, int M, int B,
            float gamma, float lam, float* adv_out, float* returns_out, void* cuda_stream);

/* The clipped PPO objective of Eq. 2 over N samples (env-steps), all device f32:
 *   lp_new, lp_old [N, A]: token log-probs under the current and the rollout policy; an
 *   action's log-prob is their sum over the A tokens (Eq. 1); adv [N];
 *   rho = exp(sum lp_new - sum lp_old);
 *   objective_out [1] = mean over samples of min(rho A, clip(rho, 1 - eps, 1 + eps) A)
 *   (to maximise; a loss is its negative); ratio_out [N] (rho) and clip_frac_out [1]
 *   (share of samples with |rho - 1| > eps) may be NULL.
 * One fixed-order reduction: repeated calls give identical results.  Needs N, A >= 1 and
 * eps >= 0 (else VLA_ERR_ARG).  Asynchronous on cuda_stream. */
int vla_ppo_clip(const float* lp_new, const float* lp_old, const float* adv, int N, int A,
                 float eps, float* objective_out, float* ratio_out, float* clip_frac_out,
                 void* cuda_stream);

/* Reset environments (episode end, Algorithm 1 terminal flags): env_mask HOST uint8
 * [max_batch], nonzero = reset; NULL = all.  A reset env has an empty context. */
int vla_reset(vla_handle* h, const uint8_t* env_mask);

/* Synchronise the handle's stream and read the device status word. */
int vla_sync(vla_handle* h);

/* Re-read the four projection matrices from the borrowed bf16 pointers given to vla_create
 * into the handle's fp16 copy (after the caller changed them in place, e.g. a PPO update of
 * θ between rollouts, Algorithm 1).  Runs on the handle's stream after all work queued before
 * it and waits for it; later calls see the new weights.  Norm gains, embeddings and lm_head
 * are read in place at every call and need no sync.  VLA_ERR_UNSUPPORTED if a weight is
 * outside the fp16 range (the copy then holds it clamped to +-65504). */
int vla_sync_weights(vla_handle* h);

/* Current context length of env b (host bookkeeping, no sync); -1 if out of range. */
int vla_context_length(const vla_handle* h, int env);

/* Message of the last error on this handle (or of the last failed vla_create when h is
 * NULL).  Valid until the next call on the handle. */
const char* vla_last_error(const vla_handle* h);

/* Free the handle and everything it owns (synchronises its stream first).  NULL is a
 * no-op. */
void vla_destroy(vla_handle* h);

/* ---- measurement -------------------------------------------------------------------
 * Kernel classes timed with CUDA events on the handle's stream when profiling is on. */
#define VLA_KCLASS_GEMM_PREFILL 0  /* tcgen05 GEMMs of prefill / score chunks         */
#define VLA_KCLASS_GEMM_DECODE 1   /* tcgen05 GEMMs of the decode forwards            */
#define VLA_KCLASS_ATTN_PREFILL 2
#define VLA_KCLASS_ATTN_DECODE 3
#define VLA_KCLASS_HEAD 4
#define VLA_KCLASS_OTHER 5         /* assemble, RMSNorm, split-K reductions           */
#define VLA_KCLASS_COUNT 6

/* Enable (class_mask bit c = class c) or disable (0) event timing; clears the counters. */
int vla_profile(vla_handle* h, uint32_t class_mask);

/* Per class: launches, summed event time (ms), algorithmic FLOPs and algorithmic DRAM bytes
 * of the launches timed since vla_profile.  Synchronises the stream.  Arrays have
 * VLA_KCLASS_COUNT entries; any may be NULL. */
int vla_profile_read(vla_handle* h, int64_t* launches, double* ms, double* flops,
                     double* bytes);

/* Number of kernels launched by this handle since creation (all classes). */
int64_t vla_launch_count(const vla_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* VLA_H_ */
