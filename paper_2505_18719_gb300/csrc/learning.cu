// The value model's output and the learning-phase quantities of the method, on the device:
//  * value head: V(o_t, v_t^in) of Algorithm 1 for a homogeneous value model (the same decoder
//    as the policy): the final RMSNorm of each env's last prefix row, then one linear output;
//  * GAE (Algorithm 1, "compute advantages"; §3.3): the reverse recursion over M steps,
//    one thread per env;
//  * the clipped PPO objective of Eq. 2 with action log-probs as the sum of the 7 token
//    log-probs (Eq. 1): one CTA, a fixed-order reduction, so the result is deterministic.
#include "misc.h"

namespace vla {

namespace {

// One CTA (256 threads) per env: V_b = sum_c h_c r g_c w_c + bias, r = rsqrt(mean h^2 + eps).
__global__ void __launch_bounds__(256) value_head_kernel(const float* h, int ldh, int d,
                                                         const bf16* __restrict__ gain,
                                                         const bf16* __restrict__ w, float eps,
                                                         float bias, float* __restrict__ out) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[2][8];
  const float* row = h + static_cast<size_t>(blockIdx.x) * ldh;
  float ss = 0.f, dot = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float x = row[c];
    ss += x * x;
    dot += x * bf2f(gain[c]) * bf2f(w[c]);
  }
  ss = warp_sum(ss);
  dot = warp_sum(dot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red[0][warp] = ss;
    red[1][warp] = dot;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f, t = 0.f;
    for (int i = 0; i < 8; ++i) {
      s += red[0][i];
      t += red[1][i];
    }
    out[blockIdx.x] = t * rsqrtf(s / static_cast<float>(d) + eps) + bias;
  }
}

// One thread per env b: A_t = delta_t + gamma lam (1 - done_t) A_{t+1}, walking t = M-1 .. 0.
__global__ void gae_kernel(const float* r, const float* v,
                           const float* done, int M, int B, float gamma, float lam,
                           float* __restrict__ adv, float* __restrict__ ret) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  float next = 0.f;
  for (int t = M - 1; t >= 0; --t) {
    const size_t i = static_cast<size_t>(t) * B + b;
    const float live = 1.f - done[i];
    const float vt = v[i];
    const float delta = r[i] + gamma * live * v[i + B] - vt;
    next = delta + gamma * lam * live * next;
    adv[i] = next;
    if (ret) ret[i] = next + vt;
  }
}

// One CTA of 1024 threads: thread j sums samples j, j + 1024, ... in order; then a fixed tree.
__global__ void __launch_bounds__(1024) ppo_clip_kernel(const float* lp_new,
                                                        const float* lp_old,
                                                        const float* adv, int N, int A,
                                                        float eps, float* __restrict__ objective,
                                                        float* __restrict__ ratio,
                                                        float* __restrict__ clip_frac) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[2][32];
  float acc = 0.f, clipped = 0.f;
  for (int n = threadIdx.x; n < N; n += blockDim.x) {
    float dl = 0.f;
    for (int i = 0; i < A; ++i)
      dl += lp_new[static_cast<size_t>(n) * A + i] - lp_old[static_cast<size_t>(n) * A + i];
    const float rho = expf(dl);
    const float a = adv[n];
    const float rc = fminf(fmaxf(rho, 1.f - eps), 1.f + eps);
    acc += fminf(rho * a, rc * a);
    clipped += fabsf(rho - 1.f) > eps ? 1.f : 0.f;
    if (ratio) ratio[n] = rho;
  }
  acc = warp_sum(acc);
  clipped = warp_sum(clipped);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red[0][warp] = acc;
    red[1][warp] = clipped;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f, c = 0.f;
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) {
      s += red[0][i];
      c += red[1][i];
    }
    objective[0] = s / static_cast<float>(N);
    if (clip_frac) clip_frac[0] = c / static_cast<float>(N);
  }
}

}  // namespace

int value_head_launch(const float* h, int ldh, int B, int d, const bf16* gain, const bf16* w, float eps,
                      float bias, float* out, cudaStream_t s) {
  if (B <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(value_head_kernel, dim3(B), dim3(256), 0, s, h, ldh, d, gain, w, eps, bias, out));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int gae_launch(const float* r, const float* v, const float* done, int M, int B, float gamma, float lam,
               float* adv, float* ret, cudaStream_t s) {
  if (M <= 0 || B <= 0) return VLA_OK;
  VLA_CUDA_TRY(launch_pdl(gae_kernel, dim3((B + 127) / 128), dim3(128), 0, s, r, v, done, M, B, gamma, lam, adv, ret));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int ppo_clip_launch(const float* lp_new, const float* lp_old, const float* adv, int N, int A, float eps,
                    float* objective, float* ratio, float* clip_frac, cudaStream_t s) {
  if (N <= 0) return VLA_ERR_ARG;
  VLA_CUDA_TRY(launch_pdl(ppo_clip_kernel, dim3(1), dim3(1024), 0, s, lp_new, lp_old, adv, N, A, eps, objective,
                          ratio, clip_frac));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
