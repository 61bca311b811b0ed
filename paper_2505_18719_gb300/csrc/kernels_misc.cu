// Row kernels of the hot path: chunk assembly (Algorithm 1: the state h(o_t) ‖ v_t^in, plus
// the pending action token of the previous turn in a multi-turn trajectory, §3.3), RMSNorm
// of the Llama-2 backbone (§3.1; fp32 math, output as the operand hi/lo pair the GEMM reads),
// row gathers and the bf16 -> fp16 conversion of the projection weights.  All HBM-bound; one
// CTA per row, vector accesses.
#include "misc.h"

namespace vla {

int64_t g_launch_count = 0;
std::atomic<int64_t> g_inject_countdown{0};
std::atomic<int> g_inject_error{0};
std::atomic<uint64_t> g_wait_limit_ns{kDefaultWaitLimitNs};

namespace {

__global__ void __launch_bounds__(256) assemble_kernel(const RowInfo* __restrict__ rows,
                                                       const bf16* __restrict__ visual,
                                                       const int* __restrict__ ids,
                                                       const int* tokens,
                                                       const bf16* __restrict__ embed, int d,
                                                       int vocab, float* __restrict__ h,
                                                       uint32_t* status) {
  pdl_launch_dependents();
  pdl_wait();
  const RowInfo ri = rows[blockIdx.x];
  const bf16* src;
  if (ri.kind == ROW_VISUAL) {
    src = visual + static_cast<size_t>(ri.idx) * d;
  } else {
    int id = (ri.kind == ROW_TEXT) ? ids[ri.idx] : tokens[ri.idx];
    if (id < 0 || id >= vocab) {
      if (threadIdx.x == 0) atomicOr(status, VLA_STATUS_BAD_TOKEN);
      id = 0;
    }
    src = embed + static_cast<size_t>(id) * d;
  }
  float* dst = h + static_cast<size_t>(blockIdx.x) * d;
  for (int c = threadIdx.x * 8; c < d; c += blockDim.x * 8) {
    const uint4 v = *reinterpret_cast<const uint4*>(src + c);
    const float2 a = unpack_bf16x2(v.x), b = unpack_bf16x2(v.y);
    const float2 e = unpack_bf16x2(v.z), f = unpack_bf16x2(v.w);
    reinterpret_cast<float4*>(dst + c)[0] = make_float4(a.x, a.y, b.x, b.y);
    reinterpret_cast<float4*>(dst + c)[1] = make_float4(e.x, e.y, f.x, f.y);
  }
}

__global__ void __launch_bounds__(256) rmsnorm_kernel(const float* h, int ldh,
                                                      const bf16* __restrict__ w, int d,
                                                      float eps, bf16* __restrict__ y_hi,
                                                      bf16* __restrict__ y_lo, bool fp16,
                                                      uint32_t* status) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[8];
  const float* row = h + static_cast<size_t>(blockIdx.x) * ldh;
  float ss = 0.f;
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(row + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int i = 0; i < (blockDim.x >> 5); ++i) tot += red[i];
  const float r = rsqrtf(tot / static_cast<float>(d) + eps);
  const size_t off = static_cast<size_t>(blockIdx.x) * d;
  uint32_t sat = 0;
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(row + c);
    const uint2 ww = *reinterpret_cast<const uint2*>(w + c);
    const float2 w0 = unpack_bf16x2(ww.x), w1 = unpack_bf16x2(ww.y);
    uint2 hi, lo;
    split_pack2(v.x * r * w0.x, v.y * r * w0.y, hi.x, lo.x, fp16, sat);
    split_pack2(v.z * r * w1.x, v.w * r * w1.y, hi.y, lo.y, fp16, sat);
    *reinterpret_cast<uint2*>(y_hi + off + c) = hi;
    if (y_lo) *reinterpret_cast<uint2*>(y_lo + off + c) = lo;
  }
  report_saturation(status, sat);
}

__global__ void gather_rows_kernel(const float* src, const int* __restrict__ idx,
                                   int d, float* __restrict__ dst) {
  pdl_launch_dependents();
  pdl_wait();
  const float* s = src + static_cast<size_t>(idx[blockIdx.x]) * d;
  float* o = dst + static_cast<size_t>(blockIdx.x) * d;
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4)
    *reinterpret_cast<float4*>(o + c) = *reinterpret_cast<const float4*>(s + c);
}

__global__ void scatter_rows_kernel(const float* src, const int* __restrict__ sidx,
                                    const int* __restrict__ didx, int d, float* __restrict__ dst) {
  pdl_launch_dependents();
  pdl_wait();
  const float* s = src + static_cast<size_t>(sidx[blockIdx.x]) * d;
  float* o = dst + static_cast<size_t>(didx[blockIdx.x]) * d;
  for (int c = threadIdx.x * 4; c < d; c += blockDim.x * 4)
    *reinterpret_cast<float4*>(o + c) = *reinterpret_cast<const float4*>(s + c);
}

}  // namespace

int assemble_launch(const RowInfo* rows, int n_rows, const bf16* visual, const int* ids,
                    const int* tokens, const bf16* embed, int d, int vocab, float* h,
                    uint32_t* status, cudaStream_t s) {
  if (n_rows <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(assemble_kernel, dim3(n_rows), dim3(256), 0, s, rows, visual, ids, tokens,
                          embed, d, vocab, h, status));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int rmsnorm_launch(const float* h, int ldh, const bf16* w, int M, int d, float eps, bf16* y_hi,
                   bf16* y_lo, cudaStream_t s, bool fp16, uint32_t* status) {
  if (M <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(rmsnorm_kernel, dim3(M), dim3(256), 0, s, h, ldh, w, d, eps, y_hi, y_lo, fp16,
                          status));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int gather_rows_launch(const float* src, const int* idx, int n, int d, float* dst, cudaStream_t s) {
  if (n <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(gather_rows_kernel, dim3(n), dim3(256), 0, s, src, idx, d, dst));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla

namespace vla {
int scatter_rows_launch(const float* src, const int* sidx, const int* didx, int n, int d, float* dst,
                        cudaStream_t s) {
  if (n <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(scatter_rows_kernel, dim3(n), dim3(256), 0, s, src, sidx, didx, d, dst));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}
}  // namespace vla

namespace vla {
namespace {
// 8 elements per thread per step (16-byte loads and stores); n % 8 == 0, 16-byte aligned.
__global__ void __launch_bounds__(256) bf16_to_f16_kernel(const bf16* __restrict__ src,
                                                          f16* __restrict__ dst, size_t n8,
                                                          int* __restrict__ out_of_range) {
  bool bad = false;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n8;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const uint4 v = reinterpret_cast<const uint4*>(src)[i];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = unpack_bf16x2(w[j]);
      bad |= !(fabsf(f.x) <= 65504.f) || !(fabsf(f.y) <= 65504.f);
      o[j] = pack_f16x2(fminf(fmaxf(f.x, -65504.f), 65504.f), fminf(fmaxf(f.y, -65504.f), 65504.f));
    }
    reinterpret_cast<uint4*>(dst)[i] = make_uint4(o[0], o[1], o[2], o[3]);
  }
  if (bad) atomicOr(out_of_range, 1);
}
}  // namespace

int bf16_to_f16_launch(const bf16* src, f16* dst, size_t n, int* out_of_range, int num_sms,
                       cudaStream_t s) {
  if (n == 0) return VLA_OK;
  if ((n & 7) || (reinterpret_cast<uintptr_t>(src) & 15) || (reinterpret_cast<uintptr_t>(dst) & 15))
    return VLA_ERR_ARG;
  const size_t n8 = n / 8;
  const size_t want = (n8 + 255) / 256;
  const int grid = static_cast<int>(want < static_cast<size_t>(num_sms) * 8 ? want : static_cast<size_t>(num_sms) * 8);
  VLA_CUDA_TRY(injected_launch_error());
  bf16_to_f16_kernel<<<grid, 256, 0, s>>>(src, dst, n8, out_of_range);
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}
}  // namespace vla
