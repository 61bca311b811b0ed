// Fused action head: final RMSNorm -> the 256 action-bin logits -> logsumexp -> Gumbel-max
// sample -> log-prob and bin-centre action (paper §3.1: each action token is one discrete
// bin of one action dimension, a_t = f(v_out); Eq. 1: per-token log-probs; Table 2: the
// sampling temperature).  Only the last 256 rows of lm_head are ever read.
//
// One CTA (256 threads, 8 warps) per (env, action position).  Warp w computes the logits of
// bins 32w .. 32w+31: for each bin the 32 lanes stream the 2*d-byte weight row in 16-byte
// pieces (coalesced) against the fp32 normalised hidden state held in shared memory, then
// reduce with shuffles.  Thread k then owns bin k for the sampler; the argmax (ties to the
// lowest bin) and the logsumexp are block reductions.
#include "misc.h"

namespace vla {

namespace {

struct ArgMax {
  float v;
  int i;
};
__device__ __forceinline__ ArgMax better(ArgMax a, ArgMax b) {
  // larger value wins; equal values -> lower index (NaN never wins)
  if (b.v > a.v || (b.v == a.v && b.i < a.i)) return b;
  return a;
}

__global__ void __launch_bounds__(256) action_head_kernel(const HeadArgs a) {
  extern __shared__ float y[];  // [d] normalised hidden state
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
  const int d = a.d;
  const float* hrow = a.h + static_cast<size_t>(b * a.n_pos + j) * a.ldh;

  // RMSNorm (fp32)
  float ss = 0.f;
  for (int c = tid; c < d; c += 256) {
    const float v = hrow[c];
    y[c] = v;
    ss += v * v;
  }
  ss = warp_sum(ss);
  if (lane == 0) red_f[warp] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += red_f[w];
  const float r = rsqrtf(tot / static_cast<float>(d) + a.eps);
  for (int c = tid; c < d; c += 256) y[c] = y[c] * r * bf2f(a.final_norm[c]);
  __syncthreads();

  // logits of bins 32*warp .. 32*warp+31
  for (int kk = 0; kk < 32; ++kk) {
    const int k = warp * 32 + kk;
    const bf16* wrow = a.head_rows + static_cast<size_t>(k) * d;
    float acc = 0.f;
    for (int c = lane * 8; c < d; c += 256) {
      const uint4 wv = *reinterpret_cast<const uint4*>(wrow + c);
      const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_bf16x2(ww[e]);
        acc = fmaf(f.x, y[c + 2 * e], acc);
        acc = fmaf(f.y, y[c + 2 * e + 1], acc);
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) z_s[k] = acc;
  }
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
  ArgMax am{s, k};
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
  __syncthreads();  // red_f reuse
  if (lane == 0) red_f[warp] = se;
  __syncthreads();
  float sum_e = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) sum_e += red_f[w];
  const float lse = zmax + logf(sum_e);

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
  if (a.d % 8) return VLA_ERR_UNSUPPORTED;
  const size_t smem = static_cast<size_t>(a.d) * sizeof(float);
  if (smem > 48 * 1024) {
    static bool set = false;
    if (!set) {
      VLA_CUDA_TRY(cudaFuncSetAttribute(action_head_kernel,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
      set = true;
    }
  }
  dim3 grid(a.B, a.n_pos);
  VLA_CUDA_TRY(launch_pdl(action_head_kernel, grid, dim3(256), smem, s, a));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
