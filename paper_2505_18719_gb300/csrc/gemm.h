// Internal interface of the tcgen05 GEMM (gemm_tc.cu) used by the engine and the op API.
#pragma once
#include "common.cuh"

namespace vla {

// Epilogue of Y[M, N] = A[M, K] · B[N, K]^T (fp32 accumulator in TMEM).
enum EpiKind : int {
  EPI_F32 = 0,     // out_f32[m * ldo + n] = y
  EPI_RESID = 1,   // resid[m * ldr + n] += y               (O-proj, down-proj)
  EPI_SWIGLU = 2,  // u = silu(y_gate) * y_up, f < F = N / 2, stored as the operand pair
                   // out_hi / out_lo [m * ldo + f]
  EPI_QKV = 3,     // RoPE(q) -> out_q f32 [M, d]; RoPE(k), v -> fp16 KV cache
  EPI_PARTIAL = 4  // internal: split-K partial sums to the workspace
};

struct EpiArgs {
  int kind = EPI_F32;
  // Operand format of the whole call: false = bf16, true = fp16.  It applies to A, A_lo and B
  // (one tcgen05 kind::f16 MMA takes both operands in one type) and to the pair outputs
  // out_hi / out_lo and norm_hi / norm_lo, which feed the next projection.  The pointers are
  // typed bf16 but hold 2-byte elements of the chosen format.
  bool fp16 = false;
  float* out_f32 = nullptr;
  float* out_q = nullptr;
  bf16* out_hi = nullptr;
  bf16* out_lo = nullptr;
  int ldo = 0;
  float* resid = nullptr;
  int ldr = 0;
  const RowInfo* rows = nullptr;  // EPI_QKV: env / position of each row
  KVLayout kv{};
  int layer = 0;
  const float2* rope = nullptr;   // EPI_QKV: [cap][hd/2] (cos, sin)
  int d = 0, hd = 0;
  // EPI_RESID of the weight-streaming GEMM only: after the residual add, the row's RMSNorm
  // with weight norm_w (bf16, N elements) is written as the operand pair norm_hi / norm_lo
  // [m * ldn + n] in the same kernel.  The tile GEMM rejects it.
  const bf16* norm_w = nullptr;
  float norm_eps = 0.f;
  bf16* norm_hi = nullptr;
  bf16* norm_lo = nullptr;
  int ldn = 0;
  // EPI_RESID of the tile GEMMs with norm_w set and ss_out != nullptr: the row of the updated
  // residual times norm_w goes to norm_hi / norm_lo NOT normalised, and the sum of squares of
  // the row's columns in each BN-wide tile to ss_out[n_tile * M + m]; the consuming GEMM
  // applies the normalisation (row_ss).
  float* ss_out = nullptr;
  // EPI_QKV / EPI_SWIGLU of the tile GEMMs: row_ss != nullptr scales each output row by
  // rsqrt(sum_{t < row_ss_n} row_ss[t * M + m] / row_d + row_eps) first (the RMSNorm of an
  // input given unnormalised: the norm is a per-row scale, so it commutes with the product).
  const float* row_ss = nullptr;
  int row_ss_n = 0, row_d = 0;
  float row_eps = 0.f;
  uint32_t* status = nullptr;
};

struct GemmArgs {
  const bf16* A = nullptr;     // [M, K], row stride lda
  const bf16* A_lo = nullptr;  // optional low half of A (same layout): Y = (A + A_lo) · B^T
  int lda = 0;
  const bf16* B = nullptr;  // [N, K], row stride ldb (SwiGLU: [2F, K] rows gate | up, N = 2F)
  int ldb = 0;
  int M = 0, N = 0, K = 0;
  int block_n = 256;        // 128 or 256
  int splits = 1;           // split-K factor (> 1 needs workspace)
  bool pair = false;        // 2-SM tiles (256 x 256 per CTA pair); needs block_n 256, splits 1
  float* workspace = nullptr;
  size_t workspace_bytes = 0;
  EpiArgs epi;
};

// Algorithmic cost of one GEMM call (for the roofline report).
struct GemmCost {
  double flops, bytes;
};

// Effective split count (no empty split) for a requested one.
int gemm_effective_splits(int K, int splits);
// Workspace bytes the call needs (0 when splits == 1).
size_t gemm_workspace_bytes(const GemmArgs& a);
// Launch; returns VLA_OK or an error code (host checks only; kernels report via status).
int gemm_launch(const GemmArgs& a, cudaStream_t stream, int num_sms, GemmCost* cost);

// Weight-streaming (decode) GEMM for M <= 128 rows with a split A (A_lo required; operand
// format epi.fp16): swap-AB tcgen05 MMAs, stream-K over the weight tiles, partials in
// `workspace` (gemv_workspace_bytes), then the epilogue of `a.epi` in a fixed-order reduction
// (EPI_RESID with norm_w set: fused with the following RMSNorm).
size_t gemv_workspace_bytes(int M, int N, int K, int num_sms);

// 2-D tensor map of 2-byte elements (bf16, or fp16 when fp16) over [rows, cols] (row stride ld
// elements), box {64, box_rows}, 128-byte swizzle.
bool make_tensor_map_2d(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_rows,
                        bool fp16);

// Failure injection (test hook): in the next single-CTA tile GEMM launch, CTA 0 leaves its first
// pipeline stage unfilled; its bounded wait on that stage runs out (VLA_STATUS_TIMEOUT).
void gemm_stall_next_launch();
int gemv_launch(const GemmArgs& a, cudaStream_t stream, int num_sms, GemmCost* cost);

}  // namespace vla
