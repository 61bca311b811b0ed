// Internal interface of the row kernels (kernels_misc.cu) and the action head (action_head.cu).
#pragma once
#include "common.cuh"

namespace vla {

// h[r] (f32 [rows, d]) = source row of RowInfo r: visual (bf16 row idx), text (embed[ids[idx]])
// or token (embed[tokens[idx]]).  Ids outside [0, vocab) -> VLA_STATUS_BAD_TOKEN, row 0.
int assemble_launch(const RowInfo* rows, int n_rows, const bf16* visual, const int* ids,
                    const int* tokens, const bf16* embed, int d, int vocab, float* h,
                    uint32_t* status, cudaStream_t s);

// y[m] = h[m] / sqrt(mean(h[m]^2) + eps) * w, h f32 [M, d] (row stride ldh), written as the
// operand pair (y_hi, y_lo) [M, d] with y_hi + y_lo ~ y, fp16 if `fp16` else bf16; a finite
// value beyond the fp16 range is stored as +-65504 and sets VLA_STATUS_SATURATED in *status.
int rmsnorm_launch(const float* h, int ldh, const bf16* w, int M, int d, float eps, bf16* y_hi,
                   bf16* y_lo, cudaStream_t s, bool fp16, uint32_t* status);

// dst[i] = fp16(src[i]) for n bf16 values (n % 8 == 0, both 16-byte aligned).  A value outside
// the finite fp16 range (|x| > 65504, or not finite) is clamped to +-65504 and sets
// *out_of_range to 1.  A bf16 value (8 significant bits) with 2^-14 <= |x| <= 65504 is exact
// in fp16 (11); a smaller one rounds to a multiple of 2^-24, an absolute error <= 2^-25.
int bf16_to_f16_launch(const bf16* src, f16* dst, size_t n, int* out_of_range, int num_sms,
                       cudaStream_t s);

// dst[i] = src[idx[i]] rows of width d (f32).
int gather_rows_launch(const float* src, const int* idx, int n, int d, float* dst, cudaStream_t s);
// dst[didx[i]] = src[sidx[i]] rows of width d (f32), i < n.
int scatter_rows_launch(const float* src, const int* sidx, const int* didx, int n, int d, float* dst,
                        cudaStream_t s);

struct HeadArgs {
  const float* h = nullptr;   // input rows, row (b * n_pos + j) has stride ldh
  int ldh = 0;
  int B = 0, n_pos = 1;       // grid: B x n_pos
  int step = 0;               // action index of j = 0 (decode: current step; score: 0)
  int A = 7;                  // actions per env (row stride of the [B, A] outputs)
  const bf16* final_norm = nullptr;
  const bf16* head_rows = nullptr;  // [256, d]
  int d = 0;
  float eps = 1e-6f;
  float temperature = 1.f;
  const float* uniforms = nullptr;  // [B, A, 256] (sample mode) or null (score mode)
  const int* forced = nullptr;      // [B, A] ids whose log-prob is reported (null: the sample)
  int forced_base = 0;              // subtracted from forced ids to get bins (vocab-256 or 0)
  int token_base = 0;               // vocab - 256
  int* tokens_out = nullptr;        // [B, A] sampled ids
  int* bins_out = nullptr;          // [B, A] sampled bins
  float* lp_out = nullptr;          // [B, A]
  float* act_out = nullptr;         // [B, A]
  float* logits_out = nullptr;      // [B, A, 256]
  float* z = nullptr;               // scratch [B * n_pos, 256] logits (may alias logits_out
                                    // when A == n_pos and step == 0)
  int* fed_out = nullptr;           // [B, A] token fed to the next step (forced or sampled)
  float* entropy_out = nullptr;     // [B, A] entropy of each token's bin distribution
  uint32_t* status = nullptr;
};
int action_head_launch(const HeadArgs& a, cudaStream_t s);

// learning.cu
int value_head_launch(const float* h, int ldh, int B, int d, const bf16* gain, const bf16* w, float eps,
                      float bias, float* out, cudaStream_t s);
int gae_launch(const float* r, const float* v, const float* done, int M, int B, float gamma, float lam,
               float* adv, float* ret, cudaStream_t s);
int ppo_clip_launch(const float* lp_new, const float* lp_old, const float* adv, int N, int A, float eps,
                    float* objective, float* ratio, float* clip_frac, cudaStream_t s);

}  // namespace vla
