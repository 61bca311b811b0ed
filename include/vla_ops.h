/*
 * vla_ops.h — single-kernel entry points of libvla.so, for checking one operation of the
 * hot path at a time.  Same conventions as vla.h (device pointers, asynchronous on
 * `cuda_stream`, host-checkable errors returned at once); each returns a vla_status.
 *
 * Errors found on the device by the GEMM and RMSNorm entry points (VLA_STATUS_TIMEOUT: a
 * pipeline wait ran out and that CTA's output tile was not written; VLA_STATUS_SATURATED)
 * are OR-ed into one status word per device that the library owns; vla_op_read_status
 * returns and clears it.
 */
#ifndef VLA_OPS_H_
#define VLA_OPS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* C[M, N] (f32, row stride ldc) = (A + A_lo)[M, K] · W[N, K]^T with A, A_lo, W bf16
 * row-major (row strides lda, ldw elements, multiples of 8), fp32 accumulation on the tcgen05
 * tensor cores.  A_lo may be NULL (then C = A · W^T); otherwise the activation is the
 * unevaluated bf16 pair A + A_lo (the engine itself runs the fp16 form below).
 * This is the contraction of every projection of the decoder layer (§3.1: the Llama-2
 * backbone's q/k/v, o, gate/up and down projections).  `block_n` in {128, 256} is the output
 * tile width; `splits` >= 1 splits K across CTAs (partials in `workspace`, f32
 * [splits, M, N], required when splits > 1, then summed in a fixed order).
 * Requires M, N, K >= 1. */
int vla_op_gemm_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C,
                     int ldc, int M, int N, int K, int block_n, int splits, float* workspace,
                     void* cuda_stream);

/* vla_op_gemm_bf16 (C f32 = (A + A_lo) · W^T, A_lo may be NULL) on CTA pairs: each pair of
 * SMs computes 256 x 256 output tiles with 2-SM tcgen05 MMAs (cta_group::2), each SM loading
 * half of the A and B tiles.  Same arguments and results as vla_op_gemm_bf16 without
 * split-K; the prefill projections run this way. */
int vla_op_gemm_pair_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw,
                          float* C, int ldc, int M, int N, int K, void* cuda_stream);

/* The decode-step projection (§3.1 projections at decode batch sizes, Algorithm 1 rollout):
 * C[M, N] (f32) = (A + A_lo)[M, K] · W[N, K]^T for M <= 128 activation rows, bf16 operands,
 * A_lo required.  Streams W from HBM once: swap-AB tcgen05 MMAs (W rows are the MMA's M),
 * stream-K over the 128-row weight tiles, fp32 partials in `workspace` (at least
 * vla_op_gemm_decode_workspace_bytes(M, N, K) bytes), fixed-order reduction into C.
 * VLA_ERR_ARG for M > 128, NULL pointers or a short workspace. */
int vla_op_gemm_decode_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw,
                            float* C, int ldc, int M, int N, int K, float* workspace,
                            size_t workspace_bytes, void* cuda_stream);
size_t vla_op_gemm_decode_workspace_bytes(int M, int N, int K);

/* The same three contractions with fp16 operands: A, A_lo and W hold IEEE binary16 bits, the
 * form in which the engine runs every projection (each fp16 half keeps 11 significant bits,
 * so hi alone is 8x closer to the activation than a bf16 hi; the pair hi + lo keeps ~21).
 * Arguments, layouts, workspaces, errors and the fp32 accumulation are those of the bf16
 * entry points above. */
int vla_op_gemm_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C,
                    int ldc, int M, int N, int K, int block_n, int splits, float* workspace,
                    void* cuda_stream);
int vla_op_gemm_pair_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw,
                         float* C, int ldc, int M, int N, int K, void* cuda_stream);
int vla_op_gemm_decode_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw,
                           float* C, int ldc, int M, int N, int K, float* workspace,
                           size_t workspace_bytes, void* cuda_stream);

/* vla_op_gemm_bf16 without a caller workspace: the paper has no counterpart; this entry
 * point exists for callers that cannot allocate device memory (all device memory owned by
 * another allocator, or a loop that must not pay the synchronisation of cudaMalloc/cudaFree).
 * Same arguments and result as vla_op_gemm_bf16 (its C within the same tolerance), but the
 * split-K partials live in a file-scope 8 MiB device array inside libvla.so, which every
 * device that loads the library holds until the process exits.  It allocates nothing.
 *  - splits * M * N * 4 bytes must fit in 8 MiB, else VLA_ERR_CAPACITY and nothing runs.
 *  - The first call on each device looks up the array's device address (with that device
 *    current); make that first call before any stream capture.
 *  - All calls share the one array: calls that overlap on the GPU (other streams, other
 *    threads) race on it.  Serialise them, e.g. on one stream.
 *  - Nothing carries over between calls: every partial is rewritten before it is read.
 *  - A pipeline timeout is reported in the op status word (vla_op_read_status). */
int vla_op_gemm_bf16_noalloc(const void* A, const void* A_lo, int lda, const void* W, int ldw,
                             float* C, int ldc, int M, int N, int K, int block_n, int splits,
                             void* cuda_stream);

/* RMSNorm of the decoder layer (§3.1, the Llama-2 backbone) on M rows: y = h / sqrt(mean(h^2)
 * + eps) * w, h f32 [M, d] (row stride ldh, 16-byte aligned, ldh % 4 == 0), w bf16 [d], written
 * as the operand pair the projections read: y_hi / y_lo [M, d] (row stride d, 8-byte aligned),
 * fp16 halves when fp16 != 0 (the engine's form), else bf16.  d % 4 == 0.  In the fp16 form a
 * finite value beyond +-65504 is stored as +-65504 and sets VLA_STATUS_SATURATED in the op
 * status word (NaN and infinities pass through unchanged). */
int vla_op_rmsnorm(const float* h, int ldh, int M, int d, const void* w, float eps, void* y_hi,
                   void* y_lo, int fp16, void* cuda_stream);

/* Reads the op entry points' status word of the current device into *status_out (VLA_STATUS_*
 * bits) after all work queued on cuda_stream, then clears it; synchronises the stream. */
int vla_op_read_status(void* cuda_stream, uint32_t* status_out);

/* The fused action head (§3.1 action bins; Eq. 1 log-probs; Algorithm 1 f) on B given
 * hidden states h (f32 [B, d], row stride ldh): RMSNorm with final_norm (bf16 [d], eps),
 * logits z = y · head_rows^T (head_rows bf16 [256, d] = the last 256 lm_head rows), then the
 * sampler of vla_decode_actions with uniforms (f32 [B, 256]) at `temperature`.
 * forced (int32 [B] bin indices 0..255, or NULL) selects whose log-prob is returned.
 * Outputs (device, [B]): bins_out int32 (sampled bin k), logprobs_out f32, actions_out f32,
 * logits_out f32 [B, 256] (required: the logits are formed there before sampling).  status:
 * device uint32 word, OR-ed with VLA_STATUS_* bits.  h must be 16-byte aligned with ldh a
 * multiple of 4, head_rows 16-byte aligned, final_norm 8-byte aligned, d a multiple of 8 and
 * at most 6400 (else VLA_ERR_UNSUPPORTED). */
int vla_op_action_head(const float* h, int ldh, int B, int d, const void* final_norm,
                       const void* head_rows, float eps, const float* uniforms,
                       float temperature, const int32_t* forced, int32_t* bins_out,
                       float* logprobs_out, float* actions_out, float* logits_out,
                       uint32_t* status, void* cuda_stream);

/* Decode-step causal attention (§3.1 self-attention over the env's whole multi-turn context,
 * §3.3) for B single queries, flash-decoding over the fp16 KV cache:
 *   q         f32 [B, H, hd] (already rotated);
 *   kv        fp16 cache laid out [env][K,V][H][cap][hd] (one layer, max_env envs);
 *   env, pos  int32 [B] each: query b reads env env[b], keys 0..pos[b] (pos[b] < cap);
 *   max_keys_per_cta  longest key range one CTA handles (0 = the library's default, 320);
 *   out_hi / out_lo  bf16 [B, H*hd]: the output o as the pair hi + lo;
 *   workspace f32, at least vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx,
 *             max_keys_per_cta) bytes, max_ctx >= every pos[b] + 1.
 * hd in {64, 128}. */
int vla_op_attn_decode(const float* q, const void* kv, int max_env, int H, int hd, int cap,
                       const int32_t* env, const int32_t* pos, int B, int max_ctx,
                       int max_keys_per_cta, void* out_hi, void* out_lo, float* workspace,
                       size_t workspace_bytes, void* cuda_stream);
size_t vla_op_attn_decode_workspace_bytes(int B, int H, int hd, int max_ctx, int max_keys_per_cta);

/* The engine's decode attention: vla_op_attn_decode with the cache read at its stored
 * precision, each value hi + (2c - 15) ulp(hi) / 32 from its fp16 part hi in kv and its 4-bit
 * code c in kv_res (the layout of vla_op_attn_chunk_res); kv and kv_res 16-byte aligned.  Cache
 * positions past pos[b] may hold anything (NaN included): they do not reach the output.  Same
 * workspace as vla_op_attn_decode. */
int vla_op_attn_decode_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd,
                           int cap, const int32_t* env, const int32_t* pos, int B, int max_ctx,
                           int max_keys_per_cta, void* out_hi, void* out_lo, float* workspace,
                           size_t workspace_bytes, void* cuda_stream);

/* Chunk causal attention (§3.1 self-attention; a prefill or appended chunk of each env attends
 * to its whole cached context, §3.3), the prefill / score kernel on its own:
 *   q          f32 [rows, H*hd] (already rotated), rows packed chunk after chunk;
 *   kv         fp16 cache [env][K,V][H][cap][hd] (one layer, max_env envs), already holding
 *              the chunk's own K/V;
 *   tiles_host HOST int32 [n_tiles][4] = (env, row0, nrows, pos0): query rows row0 ..
 *              row0+nrows-1 at positions pos0 .. pos0+nrows-1 of env, keys 0 .. position;
 *              1 <= nrows <= 64, env < max_env, pos0 >= 0, pos0 + nrows <= cap,
 *              row0 + nrows <= rows (checked on the host: VLA_ERR_ARG, nothing runs);
 *   tiles_dev  device int32 [n_tiles][4] the tiles are copied to (the caller's scratch);
 *   out_hi / out_lo  bf16 [rows, H*hd]: the output as the pair hi + lo.
 * hd in {64, 128}. */
int vla_op_attn_chunk(const float* q, const void* kv, int max_env, int H, int hd, int cap,
                      const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev,
                      void* out_hi, void* out_lo, void* cuda_stream);

/* The engine's chunk attention (§3.1 self-attention over the env's whole multi-turn context,
 * §3.3; the prefill chunks and the PPO ratio pass of Eq. 2) on the tcgen05 tensor cores, with
 * the cache read at its full stored precision:
 *   q, tiles_host, tiles_dev, rows, out_hi / out_lo as vla_op_attn_chunk, but tiles of up to 128
 *   rows (1 <= nrows <= 128);
 *   kv       fp16 cache [env][K,V][H][cap][hd] (one layer, max_env envs), 16-byte aligned;
 *   kv_res   its 4-bit residual codes, one byte per element pair of the same layout (element 2i
 *            in the low nibble of byte i), 16-byte aligned: code c of value x with fp16 part
 *            hi = fp16(x) is c = 8 + clamp(floor((x - hi) / ulp(hi) * 16), -8, 7), and the value
 *            read is hi + (2c - 15) ulp(hi) / 32, ulp(hi) = 2^(e-25) for hi's biased exponent
 *            e >= 1, 2^-24 for e = 0.
 * Cache positions past a tile's last visible key may hold anything (NaN included): they do not
 * reach the output.  A pipeline wait that runs out sets VLA_STATUS_TIMEOUT in the op status
 * word.  hd in {64, 128}. */
int vla_op_attn_chunk_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd,
                          int cap, const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev,
                          void* out_hi, void* out_lo, void* cuda_stream);

/* The same attention for short tiles, the engine's kernel when every tile has at most 16 rows
 * (the PPO ratio pass of Eq. 2: A - 1 teacher-forced rows per env): arguments as
 * vla_op_attn_chunk_res, with 1 <= nrows <= 16 per tile (VLA_ERR_ARG otherwise, nothing runs).
 * mma.sync on one CTA per (tile, head): each cached byte is read once per tile and head, and no
 * MMA row past the 16th is spent; same results to fp32 rounding order. */
int vla_op_attn_rows_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd,
                         int cap, const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev,
                         void* out_hi, void* out_lo, void* cuda_stream);

/* Number of SMs the kernels size their persistent grids for (device property). */
int vla_op_num_sms(void);

/* ---- failure injection, for tests of the error paths (no GPU fault is involved) ----------
 * vla_test_inject_launch_error: the nth_launch-th kernel launch of the library from now on
 *   (counting every kernel of every entry point) returns cuda_error (a cudaError_t value,
 *   non-zero) without launching, as a failed launch would; the entry point then returns
 *   VLA_ERR_CUDA.  nth_launch == 0 disarms.  Process-wide; not for concurrent use.
 * vla_test_set_wait_limit_ns: limit of each bounded pipeline wait of the tcgen05 GEMMs
 *   launched from now on (0 restores the default, 1 s).  A wait that runs out sets
 *   VLA_STATUS_TIMEOUT, the CTA waits (within the same limit) for its own copies and MMAs,
 *   frees its tensor memory and exits without writing its output tile.
 * vla_test_stall_next_gemm: in the next single-CTA tile GEMM launch, CTA 0 leaves its first
 *   pipeline stage unfilled, so its MMA thread waits on a barrier that nothing completes until
 *   the limit runs out (then as above).  The other CTAs run normally. */
int vla_test_inject_launch_error(int64_t nth_launch, int cuda_error);
int vla_test_set_wait_limit_ns(uint64_t limit_ns);
int vla_test_stall_next_gemm(void);

#ifdef __cplusplus
}
#endif
#endif /* VLA_OPS_H_ */
