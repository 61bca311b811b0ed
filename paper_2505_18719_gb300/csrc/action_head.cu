// Action head: final RMSNorm -> the 256 action-bin logits -> logsumexp -> Gumbel-max
// sample -> log-prob and bin-centre action (paper §3.1: each action token is one discrete
// bin of one action dimension, a_t = f(v_out); Eq. 1: per-token log-probs; Table 2: the
// sampling temperature).  Only the last 256 rows of lm_head are ever read.
//
// Two kernels:
//  head_logits_kernel  one CTA per (32 bins, 8 rows): the 8 rows are normalised into shared
//                      memory (fp32), then warp w forms the dot products of bins 4w .. 4w+3
//                      with all 8 rows, so each 16-byte piece of a weight row loaded from L2
//                      serves 8 rows (the 2 MB of bin rows are read R/8 times in all, not R).
//  head_sample_kernel  one CTA (256 threads) per row: thread k owns bin k; the argmax (ties
//                      to the lowest bin) and the logsumexp are block reductions.
#include "misc.h"

namespace vla {

namespace {

struct ArgMax {
  float v;
  int i;
};
// Larger value wins; equal values -> lower index.  Callers map NaN scores to -inf first (a NaN
// held in `a` would otherwise never be replaced, since no comparison with NaN is true).
__device__ __forceinline__ ArgMax better(ArgMax a, ArgMax b) {
  if (b.v > a.v || (b.v == a.v && b.i < a.i)) return b;
  return a;
}

constexpr int kHeadRows = 8;   // rows per logits CTA
constexpr int kHeadBins = 32;  // bins per logits CTA (4 per warp)

__global__ void __launch_bounds__(256) head_logits_kernel(const HeadArgs a) {
  extern __shared__ float ys[];  // [kHeadRows][d] normalised rows
  pdl_launch_dependents();
  pdl_wait();
  const int R = a.B * a.n_pos;
  const int r0 = blockIdx.y * kHeadRows;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d = a.d;

  // RMSNorm (fp32) of row r0 + warp by warp `warp`; each lane rescales its own elements
  {
    const int r = r0 + warp;
    float* yr = ys + static_cast<size_t>(warp) * d;
    if (r < R) {
      const float* hrow = a.h + static_cast<size_t>(r) * a.ldh;
      float ss = 0.f;
      for (int c = lane * 4; c < d; c += 128) {
        const float4 v = *reinterpret_cast<const float4*>(hrow + c);
        *reinterpret_cast<float4*>(yr + c) = v;
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
      }
      ss = warp_sum(ss);
      const float rs = rsqrtf(ss / static_cast<float>(d) + a.eps);
      for (int c = lane * 4; c < d; c += 128) {
        float4 v = *reinterpret_cast<const float4*>(yr + c);
        const uint2 ww = *reinterpret_cast<const uint2*>(a.final_norm + c);
        const float2 w0 = unpack_bf16x2(ww.x), w1 = unpack_bf16x2(ww.y);
        v.x = v.x * rs * w0.x;
        v.y = v.y * rs * w0.y;
        v.z = v.z * rs * w1.x;
        v.w = v.w * rs * w1.y;
        *reinterpret_cast<float4*>(yr + c) = v;
      }
    } else {
      for (int c = lane * 4; c < d; c += 128)
        *reinterpret_cast<float4*>(yr + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  __syncthreads();

  // z[r][k] for bins k0 .. k0+3 and the CTA's 8 rows
  const int k0 = blockIdx.x * kHeadBins + warp * 4;
  float acc[4][kHeadRows];
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int rr = 0; rr < kHeadRows; ++rr) acc[q][rr] = 0.f;
  for (int c = lane * 8; c < d; c += 256) {
    float w[4][8];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint4 wv = *reinterpret_cast<const uint4*>(a.head_rows + static_cast<size_t>(k0 + q) * d + c);
      const float2 f0 = unpack_bf16x2(wv.x), f1 = unpack_bf16x2(wv.y);
      const float2 f2 = unpack_bf16x2(wv.z), f3 = unpack_bf16x2(wv.w);
      w[q][0] = f0.x;
      w[q][1] = f0.y;
      w[q][2] = f1.x;
      w[q][3] = f1.y;
      w[q][4] = f2.x;
      w[q][5] = f2.y;
      w[q][6] = f3.x;
      w[q][7] = f3.y;
    }
#pragma unroll
    for (int rr = 0; rr < kHeadRows; ++rr) {
      const float4 y0 = *reinterpret_cast<const float4*>(ys + static_cast<size_t>(rr) * d + c);
      const float4 y1 = *reinterpret_cast<const float4*>(ys + static_cast<size_t>(rr) * d + c + 4);
      const float y[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
#pragma unroll
      for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[q][rr] = fmaf(w[q][e], y[e], acc[q][rr]);
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int rr = 0; rr < kHeadRows; ++rr) {
      const float v = warp_sum(acc[q][rr]);
      if (lane == q * kHeadRows + rr && r0 + rr < R) a.z[static_cast<size_t>(r0 + rr) * 256 + k0 + q] = v;
    }
}

__global__ void __launch_bounds__(256) head_sample_kernel(const HeadArgs a) {
  __shared__ float z_s[256];
  __shared__ float red_f[8];
  __shared__ ArgMax red_a[8];
  __shared__ float red_m[8];

  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x, j = blockIdx.y;
  const int i_act = a.step + j;               // action index
  const int out_i = b * a.A + i_act;          // [B, A] output slot
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  z_s[tid] = a.z[static_cast<size_t>(b * a.n_pos + j) * 256 + tid];
  __syncthreads();

  // sampler: thread k owns bin k
  const int k = tid;
  const float z = z_s[k];
  const float T = a.temperature;
  const float zt = (T > 0.f) ? z / T : z;
  float s = zt;
  if (T > 0.f && a.uniforms) {
    float u = a.uniforms[static_cast<size_t>(out_i) * 256 + k];
    u = fminf(fmaxf(u, 5.9604644775390625e-8f), 0.99999994039535522f);  // [2^-24, 1-2^-24]
    s = zt - logf(-logf(u));
  }
  // A NaN score (from a NaN logit, which raises VLA_STATUS_NONFINITE below) loses to every bin.
  ArgMax am{isnan(s) ? -INFINITY : s, k};
  float mx = zt;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ArgMax other{__shfl_xor_sync(0xffffffffu, am.v, o), __shfl_xor_sync(0xffffffffu, am.i, o)};
    am = better(am, other);
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == 0) {
    red_a[warp] = am;
    red_m[warp] = mx;
  }
  __syncthreads();
  ArgMax best = red_a[0];
  float zmax = red_m[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) {
    best = better(best, red_a[w]);
    zmax = fmaxf(zmax, red_m[w]);
  }
  const float e = expf(zt - zmax);
  float se = warp_sum(e);
  float sez = warp_sum(e * (zt - zmax));  // for the entropy: sum_k p_k (zt_k - zmax) * sum_e
  __syncthreads();  // red_f reuse
  if (lane == 0) {
    red_f[warp] = se;
    red_m[warp] = sez;
  }
  __syncthreads();
  float sum_e = 0.f, sum_ez = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    sum_e += red_f[w];
    sum_ez += red_m[w];
  }
  const float lse = zmax + logf(sum_e);
  // rollout entropy of this token's bin distribution: H = lse - sum_k p_k zt_k
  if (tid == 0 && a.entropy_out) a.entropy_out[out_i] = logf(sum_e) - sum_ez / sum_e;

  if (a.logits_out) a.logits_out[static_cast<size_t>(out_i) * 256 + k] = z;
  if (!isfinite(z)) atomicOr(a.status, VLA_STATUS_NONFINITE);

  if (tid == 0) {
    const int ks = best.i;
    int kl = ks;  // bin whose log-prob is reported
    int fed = a.token_base + ks;
    if (a.forced) {
      int f = a.forced[out_i] - a.forced_base;
      if (f < 0 || f >= 256) {
        atomicOr(a.status, VLA_STATUS_BAD_FORCED);
        f = f < 0 ? 0 : 255;
      }
      kl = f;
      fed = a.token_base + f;
    }
    a.lp_out[out_i] = z_s[kl] / (T > 0.f ? T : 1.f) - lse;
    if (a.tokens_out) a.tokens_out[out_i] = a.token_base + ks;
    if (a.bins_out) a.bins_out[out_i] = ks;
    if (a.act_out) a.act_out[out_i] = static_cast<float>(2 * ks + 1 - 256) * (1.0f / 256.0f);
    if (a.fed_out) a.fed_out[out_i] = fed;
  }
}

}  // namespace

int action_head_launch(const HeadArgs& a, cudaStream_t s) {
  if (a.B <= 0) return VLA_OK;
  if (a.d % 8 || a.ldh % 4 || !a.z || (reinterpret_cast<uintptr_t>(a.h) & 15) ||
      (reinterpret_cast<uintptr_t>(a.head_rows) & 15) || (reinterpret_cast<uintptr_t>(a.final_norm) & 7))
    return VLA_ERR_UNSUPPORTED;
  const size_t smem = static_cast<size_t>(kHeadRows) * a.d * sizeof(float);
  if (smem > 200 * 1024) return VLA_ERR_UNSUPPORTED;
  if (smem > 48 * 1024) {
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(head_logits_kernel, 200 * 1024, attr_done));
  }
  const int R = a.B * a.n_pos;
  VLA_CUDA_TRY(launch_pdl(head_logits_kernel, dim3(256 / kHeadBins, (R + kHeadRows - 1) / kHeadRows),
                          dim3(256), smem, s, a));
  note_launch();
  VLA_CUDA_TRY(launch_pdl(head_sample_kernel, dim3(a.B, a.n_pos), dim3(256), 0, s, a));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
