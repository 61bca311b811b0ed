// Causal attention over the per-environment KV cache (paper §3.1: the policy's Llama-2
// self-attention; §3.3: the whole trajectory is one context, so every chunk attends to all
// earlier turns).
//
//  * attn_chunk: query rows of one env at consecutive positions (a prefill chunk, or the
//    6 teacher-forced action rows of the score pass) against keys 0..pos of that env.
//    One CTA per (64-row tile, head); K/V blocks of 64 keys staged in shared memory; online
//    softmax in the exp2 domain; fp32 math on the fp32 queries and fp16 K/V; the output is
//    written as the bf16 hi/lo pair the O-projection GEMM reads.
//  * attn_decode: one query per env (the decode step) with the key range split across CTAs
//    (flash-decoding); each CTA writes its partial (max, sum, unnormalised output) and a
//    combine kernel merges the splits in a fixed order.  16 lanes x 16 bytes read one
//    128-element key row, so each warp streams two rows per instruction.
//
// Keys visible to a query at position p are positions 0..p (all of them are in the cache:
// chunk rows write their K/V in the QKV epilogue before attention runs).
#include "attention.h"

namespace vla {

namespace {

constexpr int kTileRows = 64;
constexpr int kKeyBlock = 64;

template <int HD>
__global__ void __launch_bounds__(256) attn_chunk_kernel(const float* __restrict__ q,
                                                         bf16* __restrict__ out_hi,
                                                         bf16* __restrict__ out_lo,
                                                         const AttnTile* __restrict__ tiles,
                                                         KVLayout kv, int layer, int H,
                                                         float scale_log2) {
  constexpr int PER_LANE = HD / 32;  // output dims per lane
  constexpr int KS = HD + 1;          // padded key row (conflict-free column reads)
  extern __shared__ float sm[];
  float* Qs = sm;                         // [64][HD]
  float* Ks = Qs + kTileRows * HD;        // [64][HD+1]
  float* Vs = Ks + kKeyBlock * KS;        // [64][HD]

  const AttnTile t = tiles[blockIdx.x];
  const int head = blockIdx.y;
  const int d = H * HD;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // Q tile, pre-scaled by log2(e)/sqrt(hd)
  for (int i = threadIdx.x; i < kTileRows * HD; i += blockDim.x) {
    const int r = i / HD, c = i - r * HD;
    float v = 0.f;
    if (r < t.nrows) v = q[static_cast<size_t>(t.row0 + r) * d + head * HD + c] * scale_log2;
    Qs[i] = v;
  }
  const f16* kbase = kv.base + static_cast<int64_t>(layer) * kv.layer_stride +
                     static_cast<int64_t>(t.env) * kv.env_stride +
                     static_cast<int64_t>(head) * kv.head_stride;
  const f16* vbase = kbase + kv.kv_stride;

  float m_i[8], l_i[8], o_i[8][PER_LANE];
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    m_i[r] = -INFINITY;
    l_i[r] = 0.f;
#pragma unroll
    for (int c = 0; c < PER_LANE; ++c) o_i[r][c] = 0.f;
  }

  const int n_keys = t.pos0 + t.nrows;  // keys 0 .. last query position
  for (int j0 = 0; j0 < n_keys; j0 += kKeyBlock) {
    __syncthreads();
    for (int i = threadIdx.x; i < kKeyBlock * (HD / 8); i += blockDim.x) {
      const int r = i / (HD / 8), c8 = (i - r * (HD / 8)) * 8;
      const int key = j0 + r;
      uint4 kk = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
      if (key < n_keys) {
        kk = *reinterpret_cast<const uint4*>(kbase + static_cast<int64_t>(key) * HD + c8);
        vv = *reinterpret_cast<const uint4*>(vbase + static_cast<int64_t>(key) * HD + c8);
      }
      const uint32_t kw[4] = {kk.x, kk.y, kk.z, kk.w};
      const uint32_t vw[4] = {vv.x, vv.y, vv.z, vv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 kf = unpack_f16x2(kw[e]);
        const float2 vf = unpack_f16x2(vw[e]);
        Ks[r * KS + c8 + 2 * e] = kf.x;
        Ks[r * KS + c8 + 2 * e + 1] = kf.y;
        Vs[r * HD + c8 + 2 * e] = vf.x;
        Vs[r * HD + c8 + 2 * e + 1] = vf.y;
      }
    }
    __syncthreads();
#pragma unroll
    for (int rr = 0; rr < 8; ++rr) {
      const int r = warp * 8 + rr;
      if (r >= t.nrows) continue;  // warp-uniform
      const int qpos = t.pos0 + r;
      if (j0 > qpos) continue;     // whole block in the future (warp-uniform)
      const float* qrow = Qs + r * HD;
      float s0 = 0.f, s1 = 0.f;
      const float* k0 = Ks + lane * KS;
      const float* k1 = Ks + (lane + 32) * KS;
#pragma unroll 8
      for (int c = 0; c < HD; ++c) {
        const float qv = qrow[c];
        s0 = fmaf(qv, k0[c], s0);
        s1 = fmaf(qv, k1[c], s1);
      }
      if (j0 + lane > qpos) s0 = -INFINITY;
      if (j0 + lane + 32 > qpos) s1 = -INFINITY;
      const float mx = warp_max(fmaxf(s0, s1));
      const float m_new = fmaxf(m_i[rr], mx);
      const float alpha = exp2f(m_i[rr] - m_new);
      const float p0 = exp2f(s0 - m_new), p1 = exp2f(s1 - m_new);
      l_i[rr] = l_i[rr] * alpha + warp_sum(p0 + p1);
      m_i[rr] = m_new;
#pragma unroll
      for (int c = 0; c < PER_LANE; ++c) o_i[rr][c] *= alpha;
      for (int jj = 0; jj < 32; ++jj) {
        const float pa = __shfl_sync(0xffffffffu, p0, jj);
        const float pb = __shfl_sync(0xffffffffu, p1, jj);
#pragma unroll
        for (int c = 0; c < PER_LANE; ++c) {
          o_i[rr][c] = fmaf(pa, Vs[jj * HD + lane + 32 * c], o_i[rr][c]);
          o_i[rr][c] = fmaf(pb, Vs[(jj + 32) * HD + lane + 32 * c], o_i[rr][c]);
        }
      }
    }
  }
#pragma unroll
  for (int rr = 0; rr < 8; ++rr) {
    const int r = warp * 8 + rr;
    if (r >= t.nrows) continue;
    const float inv = 1.f / l_i[rr];
    const size_t off = static_cast<size_t>(t.row0 + r) * d + head * HD;
#pragma unroll
    for (int c = 0; c < PER_LANE; ++c) {
      bf16 hi, lo;
      split_bf16(o_i[rr][c] * inv, hi, lo);
      out_hi[off + lane + 32 * c] = hi;
      out_lo[off + lane + 32 * c] = lo;
    }
  }
}

// ---------------------------------------------------------------------------------- decode
template <int HD>
__global__ void __launch_bounds__(128) attn_decode_kernel(const float* __restrict__ q,
                                                          const RowInfo* __restrict__ rows,
                                                          KVLayout kv, int layer, int H,
                                                          int chunk, int S, float scale_log2,
                                                          float* __restrict__ part_o,
                                                          float2* __restrict__ part_ml) {
  constexpr int LPK = HD / 8;     // lanes per key row (8 bf16 = 16 bytes per lane)
  constexpr int KPI = 32 / LPK;   // key rows per warp instruction
  __shared__ float s_m[4][KPI], s_l[4][KPI];
  __shared__ float s_o[4][KPI][HD];

  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane / LPK, part = lane - sub * LPK;
  const RowInfo ri = rows[b];
  const int d = H * HD;
  const int k_begin = split * chunk;
  const int k_end = min(k_begin + chunk, ri.pos + 1);

  float qv[8];
  {
    const float4* qp = reinterpret_cast<const float4*>(q + static_cast<size_t>(b) * d + head * HD + part * 8);
    const float4 q0 = qp[0], q1 = qp[1];
    qv[0] = q0.x * scale_log2;
    qv[1] = q0.y * scale_log2;
    qv[2] = q0.z * scale_log2;
    qv[3] = q0.w * scale_log2;
    qv[4] = q1.x * scale_log2;
    qv[5] = q1.y * scale_log2;
    qv[6] = q1.z * scale_log2;
    qv[7] = q1.w * scale_log2;
  }
  const f16* kbase = kv.base + static_cast<int64_t>(layer) * kv.layer_stride +
                     static_cast<int64_t>(ri.env) * kv.env_stride +
                     static_cast<int64_t>(head) * kv.head_stride;
  const f16* vbase = kbase + kv.kv_stride;

  float m = -INFINITY, l = 0.f, o[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) o[e] = 0.f;

  for (int key0 = k_begin + warp * KPI; key0 < k_end; key0 += 4 * KPI) {
    const int key = key0 + sub;
    const bool valid = key < k_end;
    float s = -INFINITY;
    uint4 vv = make_uint4(0, 0, 0, 0);
    if (valid) {
      const uint4 kk = *reinterpret_cast<const uint4*>(kbase + static_cast<int64_t>(key) * HD + part * 8);
      vv = *reinterpret_cast<const uint4*>(vbase + static_cast<int64_t>(key) * HD + part * 8);
      const uint32_t w[4] = {kk.x, kk.y, kk.z, kk.w};
      float acc = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_f16x2(w[e]);
        acc = fmaf(qv[2 * e], f.x, acc);
        acc = fmaf(qv[2 * e + 1], f.y, acc);
      }
      s = acc;
    }
    // reduce the dot product across the LPK lanes of this key row (all lanes take part)
    // (a key row's LPK lanes share `valid`, and the xor offsets stay inside the group)
#pragma unroll
    for (int off = LPK / 2; off > 0; off >>= 1) {
      const float other = __shfl_xor_sync(0xffffffffu, s, off);
      if (valid) s += other;
    }
    if (valid) {
      const float m_new = fmaxf(m, s);
      const float alpha = exp2f(m - m_new);
      const float p = exp2f(s - m_new);
      l = l * alpha + p;
      const uint32_t w[4] = {vv.x, vv.y, vv.z, vv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_f16x2(w[e]);
        o[2 * e] = fmaf(p, f.x, o[2 * e] * alpha);
        o[2 * e + 1] = fmaf(p, f.y, o[2 * e + 1] * alpha);
      }
      m = m_new;
    }
  }
  // per (warp, sub) partials -> shared memory
  if (part == 0) {
    s_m[warp][sub] = m;
    s_l[warp][sub] = l;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) s_o[warp][sub][part * 8 + e] = o[e];
  __syncthreads();
  // merge the 4 * KPI partial states in a fixed order
  float M = -INFINITY;
  for (int w = 0; w < 4; ++w)
    for (int k = 0; k < KPI; ++k) M = fmaxf(M, s_m[w][k]);
  const size_t slot = (static_cast<size_t>(b) * H + head) * S + split;
  for (int c = threadIdx.x; c < HD; c += blockDim.x) {
    float acc = 0.f;
    for (int w = 0; w < 4; ++w)
      for (int k = 0; k < KPI; ++k)
        if (s_m[w][k] != -INFINITY) acc += s_o[w][k][c] * exp2f(s_m[w][k] - M);
    part_o[slot * HD + c] = acc;
  }
  if (threadIdx.x == 0) {
    float L = 0.f;
    for (int w = 0; w < 4; ++w)
      for (int k = 0; k < KPI; ++k)
        if (s_m[w][k] != -INFINITY) L += s_l[w][k] * exp2f(s_m[w][k] - M);
    part_ml[slot] = make_float2(M, L);
  }
}

template <int HD>
__global__ void attn_combine_kernel(const float* __restrict__ part_o,
                                    const float2* __restrict__ part_ml, int H, int S,
                                    bf16* __restrict__ out_hi, bf16* __restrict__ out_lo) {
  const int bh = blockIdx.x;  // b * H + head
  const int c = threadIdx.x;
  float M = -INFINITY;
  for (int s = 0; s < S; ++s) M = fmaxf(M, part_ml[static_cast<size_t>(bh) * S + s].x);
  float L = 0.f, acc = 0.f;
  for (int s = 0; s < S; ++s) {
    const float2 ml = part_ml[static_cast<size_t>(bh) * S + s];
    if (ml.x == -INFINITY) continue;
    const float w = exp2f(ml.x - M);
    L += ml.y * w;
    acc += part_o[(static_cast<size_t>(bh) * S + s) * HD + c] * w;
  }
  const int b = bh / H, head = bh - b * H;
  bf16 hi, lo;
  split_bf16(acc / L, hi, lo);
  out_hi[static_cast<size_t>(b) * H * HD + head * HD + c] = hi;
  out_lo[static_cast<size_t>(b) * H * HD + head * HD + c] = lo;
}

}  // namespace

int attn_chunk_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles,
                      int n_tiles, KVLayout kv, int layer, int H, int hd, cudaStream_t stream) {
  if (n_tiles <= 0) return VLA_OK;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  dim3 grid(n_tiles, H);
  if (hd == 128) {
    const int smem = (kTileRows * 128 + kKeyBlock * 129 + kKeyBlock * 128) * 4;
    static bool set = false;
    if (!set) {
      VLA_CUDA_TRY(cudaFuncSetAttribute(attn_chunk_kernel<128>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
      set = true;
    }
    attn_chunk_kernel<128><<<grid, 256, smem, stream>>>(q, out_hi, out_lo, tiles, kv, layer, H, scale_log2);
  } else if (hd == 64) {
    const int smem = (kTileRows * 64 + kKeyBlock * 65 + kKeyBlock * 64) * 4;
    static bool set = false;
    if (!set) {
      VLA_CUDA_TRY(cudaFuncSetAttribute(attn_chunk_kernel<64>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
      set = true;
    }
    attn_chunk_kernel<64><<<grid, 256, smem, stream>>>(q, out_hi, out_lo, tiles, kv, layer, H, scale_log2);
  } else {
    return VLA_ERR_UNSUPPORTED;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int attn_decode_launch(const float* q, bf16* out_hi, bf16* out_lo, const RowInfo* rows, int B,
                       int max_ctx, KVLayout kv, int layer, int H, int hd, int chunk,
                       float* part_o, float2* part_ml, cudaStream_t stream) {
  if (B <= 0) return VLA_OK;
  const int S = (max_ctx + chunk - 1) / chunk;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  dim3 grid(S, H, B);
  if (hd == 128) {
    attn_decode_kernel<128><<<grid, 128, 0, stream>>>(q, rows, kv, layer, H, chunk, S,
                                                      scale_log2, part_o, part_ml);
    note_launch();
    attn_combine_kernel<128><<<B * H, 128, 0, stream>>>(part_o, part_ml, H, S, out_hi, out_lo);
  } else if (hd == 64) {
    attn_decode_kernel<64><<<grid, 128, 0, stream>>>(q, rows, kv, layer, H, chunk, S,
                                                     scale_log2, part_o, part_ml);
    note_launch();
    attn_combine_kernel<64><<<B * H, 64, 0, stream>>>(part_o, part_ml, H, S, out_hi, out_lo);
  } else {
    return VLA_ERR_UNSUPPORTED;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
