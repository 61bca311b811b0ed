// tcgen05 / TMEM / TMA GEMM for sm_103a with the decoder layer's fused epilogues.
//
// Y[M, N] = A[M, K] · B[N, K]^T, fp16 or bf16 operands (one format per launch, both K-major),
// fp32 accumulation in TMEM.  With a split A (the activation carried as a pair hi + lo), each
// K step issues two MMAs, hi·B and lo·B, into the same accumulator, so the product sees ~21
// (fp16) or ~16 (bf16) significant bits of the activation; the weights are one 2-byte value
// each.  The engine runs fp16 operands; the bf16 form serves the bf16 op entry points.
// This is every projection of the Llama-2 backbone of the policy (paper §3.1): q|k|v, o,
// gate|up and down.  Epilogues fuse what follows each projection in the layer: RoPE and
// the KV-cache write after q|k|v, the residual add after o and down, SwiGLU after gate|up.
//
// Kernel structure (one persistent CTA per SM, 192 threads):
//   warp 0      TMA producer: 128x64 A tile(s) + BNx64 B tile per stage, 128-byte swizzle,
//               STAGES-deep ring guarded by full/empty mbarriers.
//   warp 1      allocates 2*BN TMEM columns (two accumulators); lane 0 issues
//               tcgen05.mma.cta_group::1.kind::f16 (M=128, N=BN, K=16) and commits
//               stage releases / accumulator-ready to mbarriers.
//   warps 2-5   epilogue: tcgen05.ld 32x32b (one TMEM lane = one output row per thread),
//               fused math, global stores; releases the accumulator to the MMA warp so
//               the next tile's main loop overlaps this tile's epilogue.
// Work units (m-tile, n-tile, k-split) are rastered in groups of 16 m-tiles so that the
// tiles in flight share A and B in L2.  Every mbarrier wait is bounded (globaltimer): on
// timeout the CTA records VLA_STATUS_TIMEOUT, drains its own copies and MMAs, frees TMEM and
// exits.  No TMA multicast is used; the pair variant (gemm_tc2_kernel) runs on clusters of two
// CTAs issuing cta_group::2 MMAs on 256 x 256 tiles.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "gemm.h"
#include "ptx.cuh"

namespace vla {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes = one swizzle atom row
constexpr int kThreads = 192;
constexpr int kGroupM = 16;      // 128-row m-tiles per raster group (2048 rows)
constexpr int kGroupMPair = 8;   // 256-row m-tiles per raster group of the pair kernel

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of 128 bytes,
// 8-row core-matrix groups 1024 bytes apart (SBO); LBO unused for this layout.
__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(1) << 16;            // LBO (ignored for swizzled K-major)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;    // SBO
  d |= static_cast<uint64_t>(1) << 46;            // descriptor version (sm_100 family)
  d |= static_cast<uint64_t>(2) << 61;            // SWIZZLE_128B
  return d;
}

// Instruction descriptor, kind::f16: D f32, A/B bf16, both K-major, M = 128, N = BN.
template <int BN>
__device__ __forceinline__ constexpr uint32_t make_idesc() {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
         (static_cast<uint32_t>(BM >> 4) << 24);
}
// A and B format fields (bits 7-9, 10-12): 1 = bf16, 0 = fp16.
constexpr uint32_t kIdescBf16Operands = (1u << 7) | (1u << 10);
__device__ __forceinline__ uint32_t idesc_for(uint32_t bf16_desc, bool fp16) {
  return fp16 ? (bf16_desc & ~kIdescBf16Operands) : bf16_desc;
}

struct Params {
  int M, N, K;          // N: columns of B used (SwiGLU: 2F)
  int tiles_m, tiles_n, splits, kb_total, kb_per_split;
  int group_m;          // m-tiles per raster group
  EpiArgs epi;
  uint64_t wait_limit;  // ns per bounded mbarrier wait
  int stall;            // failure injection (test hook): CTA 0 never fills its first stage
};

__device__ __forceinline__ void unit_coords(const Params& p, int u, int& m_blk, int& n_blk,
                                            int& split) {
  const int ncols = p.tiles_n * p.splits;        // (n-tile, split) pairs
  const int per_group = p.group_m * ncols;
  const int g = u / per_group;
  const int r = u - g * per_group;
  const int first_m = g * p.group_m;
  const int gsize = min(p.group_m, p.tiles_m - first_m);
  m_blk = first_m + r % gsize;
  const int col = r / gsize;
  n_blk = col / p.splits;
  split = col - n_blk * p.splits;
}

// ----------------------------------------------------------------------------- epilogues
// 16 values as operand hi/lo pairs, fp16 if `fp16` else bf16 (two 32-byte stores each); the
// low half is not stored when lo_dst is null (a consumer that reads only the high half).
__device__ __forceinline__ void store_split16(bf16* hi_dst, bf16* lo_dst, const float (&v)[16],
                                              bool fp16, uint32_t& sat) {
  uint32_t h[8], l[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) split_pack2(v[2 * i], v[2 * i + 1], h[i], l[i], fp16, sat);
  reinterpret_cast<uint4*>(hi_dst)[0] = make_uint4(h[0], h[1], h[2], h[3]);
  reinterpret_cast<uint4*>(hi_dst)[1] = make_uint4(h[4], h[5], h[6], h[7]);
  if (!lo_dst) return;
  reinterpret_cast<uint4*>(lo_dst)[0] = make_uint4(l[0], l[1], l[2], l[3]);
  reinterpret_cast<uint4*>(lo_dst)[1] = make_uint4(l[4], l[5], l[6], l[7]);
}
// dst + off, or null when dst is null.
template <class T>
__device__ __forceinline__ T* opt_at(T* dst, size_t off) {
  return dst ? dst + off : nullptr;
}
__device__ __forceinline__ void store_f16x16(f16* dst, const float (&v)[16]) {
  uint4 a, b;
  a.x = pack_f16x2(v[0], v[1]);
  a.y = pack_f16x2(v[2], v[3]);
  a.z = pack_f16x2(v[4], v[5]);
  a.w = pack_f16x2(v[6], v[7]);
  b.x = pack_f16x2(v[8], v[9]);
  b.y = pack_f16x2(v[10], v[11]);
  b.z = pack_f16x2(v[12], v[13]);
  b.w = pack_f16x2(v[14], v[15]);
  reinterpret_cast<uint4*>(dst)[0] = a;
  reinterpret_cast<uint4*>(dst)[1] = b;
}
// 16 values as fp16 at dst and their 4-bit residual codes (8 bytes) at res, when res is set.
__device__ __forceinline__ void store_kv16(f16* dst, uint8_t* res, const float (&v)[16]) {
  store_f16x16(dst, v);
  if (!res) return;
  uint32_t w[2] = {0u, 0u};
#pragma unroll
  for (int i = 0; i < 16; ++i) w[i >> 3] |= kv_res_code(v[i], __float2half_rn(v[i])) << (4 * (i & 7));
  *reinterpret_cast<uint2*>(res) = make_uint2(w[0], w[1]);
}
// Stores the fp16 value of x at dst[i] and, when res is set, the residual byte of the element
// pair (i, i + 1) at res[i / 2]: lane l holds element i and lane l + 1 element i + 1 (i even on
// even lanes); every lane of the warp must call this together.
__device__ __forceinline__ void store_kv_pairlanes(f16* dst, uint8_t* res, int i, float x) {
  const f16 h = __float2half_rn(x);
  dst[i] = h;
  const uint32_t c = res ? kv_res_code(x, h) : 0u;
  const uint32_t c_next = __shfl_down_sync(0xffffffffu, c, 1);
  if (res && (i & 1) == 0) res[i >> 1] = static_cast<uint8_t>(c | (c_next << 4));
}
__device__ __forceinline__ void store_f32x16(float* dst, const float (&v)[16]) {
#pragma unroll
  for (int i = 0; i < 4; ++i)
    reinterpret_cast<float4*>(dst)[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}

__device__ __forceinline__ void ld16f(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  tmem_ld16(taddr, r);
  tmem_wait_ld();
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 1 / RMS of row m from the per-tile sums of squares (fixed order), or 1 without them.
__device__ __forceinline__ float row_scale(const Params& p, int m) {
  if (!p.epi.row_ss || m >= p.M) return 1.f;
  float ss = 0.f;
  for (int t = 0; t < p.epi.row_ss_n; ++t) ss += p.epi.row_ss[static_cast<size_t>(t) * p.M + m];
  return rsqrtf(ss / static_cast<float>(p.epi.row_d) + p.epi.row_eps);
}

// Plain epilogues: F32 / RESID / PARTIAL, 16 columns at a time.
template <int BN, int EPI>
__device__ __forceinline__ void epilogue_plain(const Params& p, uint32_t trow, int m, int n0,
                                               int split, uint32_t& sat) {
  const bool row_ok = m < p.M;
  // residual + the next RMSNorm's numerator (h * w) and this tile's sum of squares of h
  const bool norm_next = (EPI == EPI_RESID) && p.epi.ss_out != nullptr;
  float ss = 0.f;
#pragma unroll 1
  for (int c = 0; c < BN; c += 16) {
    float v[16];
    ld16f(trow + c, v);
    const int n = n0 + c;
    if (!row_ok || n >= p.N) continue;
    float* dst;
    int ld;
    if (EPI == EPI_F32) {
      dst = p.epi.out_f32 + static_cast<size_t>(m) * p.epi.ldo + n;
      ld = p.epi.ldo;
    } else if (EPI == EPI_RESID) {
      dst = p.epi.resid + static_cast<size_t>(m) * p.epi.ldr + n;
      ld = p.epi.ldr;
    } else {  // PARTIAL: workspace [splits][M][N]
      dst = p.epi.out_f32 + (static_cast<size_t>(split) * p.M + m) * p.N + n;
      ld = p.N;
    }
    const bool vec = (n + 16 <= p.N) && ((ld & 3) == 0) &&
                     ((reinterpret_cast<uintptr_t>(dst) & 15) == 0);
    if (vec) {
      float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float4 o;
        if (EPI == EPI_RESID) {
          o = d4[i];
          o.x += v[4 * i];
          o.y += v[4 * i + 1];
          o.z += v[4 * i + 2];
          o.w += v[4 * i + 3];
        } else {
          o = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
        d4[i] = o;
        if (norm_next) {
          v[4 * i] = o.x;
          v[4 * i + 1] = o.y;
          v[4 * i + 2] = o.z;
          v[4 * i + 3] = o.w;
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (n + i >= p.N) continue;
        if (EPI == EPI_RESID) {
          dst[i] += v[i];
          v[i] = dst[i];
        } else {
          dst[i] = v[i];
        }
      }
    }
    if (norm_next) {
      const int cnt = n + 16 <= p.N ? 16 : p.N - n;
      float y[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float hv = i < cnt ? v[i] : 0.f;
        ss += hv * hv;
        y[i] = i < cnt ? hv * bf2f(p.epi.norm_w[n + i]) : 0.f;
      }
      const size_t off = static_cast<size_t>(m) * p.epi.ldn + n;
      if (cnt == 16 && (p.epi.ldn & 7) == 0) {
        store_split16(p.epi.norm_hi + off, opt_at(p.epi.norm_lo, off), y, p.epi.fp16, sat);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          if (i >= cnt) continue;
          store_split1(p.epi.norm_hi, p.epi.norm_lo, off + i, y[i], p.epi.fp16, sat);
        }
      }
    }
  }
  if (norm_next && row_ok) p.epi.ss_out[static_cast<size_t>(n0 / BN) * p.M + m] = ss;
}

// SwiGLU: tile columns [0, BN/2) are gate features f0.., [BN/2, BN) the matching up features.
template <int BN>
__device__ __forceinline__ void epilogue_swiglu(const Params& p, uint32_t trow, int m, int f0,
                                                uint32_t& sat) {
  const int F = p.N >> 1;
  const bool row_ok = m < p.M;
  const float rs = row_scale(p, m);
#pragma unroll 1
  for (int j = 0; j < BN / 2; j += 16) {
    float g[16], u[16];
    ld16f(trow + j, g);
    ld16f(trow + BN / 2 + j, u);
    const int f = f0 + j;
    if (!row_ok || f >= F) continue;
    float o[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) o[i] = silu_f(g[i] * rs) * (u[i] * rs);
    const size_t off = static_cast<size_t>(m) * p.epi.ldo + f;
    if (f + 16 <= F && ((p.epi.ldo & 7) == 0)) {
      store_split16(p.epi.out_hi + off, opt_at(p.epi.out_lo, off), o, p.epi.fp16, sat);
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (f + i >= F) continue;
        store_split1(p.epi.out_hi, p.epi.out_lo, off + i, o[i], p.epi.fp16, sat);
      }
    }
  }
}

// q|k|v with RoPE (rotate-half: pair (i, i + hd/2) rotated by pos * theta^(-2i/hd)) and the
// KV-cache write.  q is stored fp32, K and V fp16 (cache).  The tile lies inside
// one of the q / k / v sections (BN divides d) and holds BN / hd whole heads.
template <int BN>
__device__ __forceinline__ void epilogue_qkv(const Params& p, uint32_t trow, int m, int n0) {
  const int d = p.epi.d, hd = p.epi.hd, half = hd >> 1;
  const int sec = n0 / d;              // 0 q, 1 k, 2 v
  const int head0 = (n0 - sec * d) / hd;
  const bool row_ok = m < p.M;
  const float rs = row_scale(p, m);
  RowInfo ri{0, 0, 0, 0};
  if (row_ok) ri = p.epi.rows[m];
  const KVLayout& kv = p.epi.kv;
  f16* kv_row = nullptr;
  if (row_ok && sec > 0) {
    kv_row = kv.base + static_cast<int64_t>(p.epi.layer) * kv.layer_stride +
             static_cast<int64_t>(ri.env) * kv.env_stride + (sec == 2 ? kv.kv_stride : 0) +
             static_cast<int64_t>(ri.pos) * hd;
  }
  const int heads = BN / hd;
#pragma unroll 1
  for (int hh = 0; hh < heads; ++hh) {
    const int head = head0 + hh;
    const uint32_t tcol = trow + hh * hd;
    if (sec == 2) {
      f16* dst = row_ok ? kv_row + static_cast<int64_t>(head) * kv.head_stride : nullptr;
      uint8_t* rdst = (row_ok && kv.res) ? kv.res + (dst - kv.base) / 2 : nullptr;
#pragma unroll 1
      for (int j = 0; j < hd; j += 16) {
        float v[16];
        ld16f(tcol + j, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] *= rs;
        if (row_ok) store_kv16(dst + j, rdst ? rdst + j / 2 : nullptr, v);
      }
    } else {
#pragma unroll 1
      for (int j = 0; j < half; j += 16) {
        float a[16], b[16];
        ld16f(tcol + j, a);
        ld16f(tcol + half + j, b);
        if (!row_ok) continue;
        const float2* cs = p.epi.rope + static_cast<size_t>(ri.pos) * half + j;
        float ra[16], rb[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float2 t = cs[i];
          const float ai = a[i] * rs, bi = b[i] * rs;
          ra[i] = ai * t.x - bi * t.y;
          rb[i] = bi * t.x + ai * t.y;
        }
        if (sec == 0) {
          float* dst = p.epi.out_q + static_cast<size_t>(m) * d + head * hd;
          store_f32x16(dst + j, ra);
          store_f32x16(dst + half + j, rb);
        } else {
          f16* dst = kv_row + static_cast<int64_t>(head) * kv.head_stride;
          uint8_t* rdst = kv.res ? kv.res + (dst - kv.base) / 2 : nullptr;
          store_kv16(dst + j, rdst ? rdst + j / 2 : nullptr, ra);
          store_kv16(dst + half + j, rdst ? rdst + (half + j) / 2 : nullptr, rb);
        }
      }
    }
  }
}

// ----------------------------------------------------------------------------- the kernel
template <int BN, int STAGES, int EPI, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                   const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmB2,
                   const Params p) {
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int A_TOTAL = SPLIT ? 2 * A_BYTES : A_BYTES;
  constexpr int B_BYTES = BN * BK * 2;
  constexpr int STAGE_BYTES = A_TOTAL + B_BYTES;
  constexpr uint32_t TMEM_COLS = 2 * BN;
  const uint32_t IDESC = idesc_for(make_idesc<BN>(), p.epi.fp16);
  constexpr bool SWIGLU = (EPI == EPI_SWIGLU);

  pdl_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  // bars: full[STAGES], empty[STAGES], tfull[2], tempty[2], drain
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t tfull0 = empty0 + 8 * STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain_bar = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 4);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    if (SPLIT)
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA2)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int units = p.tiles_m * p.tiles_n * p.splits;
  uint32_t* status = p.epi.status;
  const uint64_t limit = p.wait_limit;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      pdl_wait_async();  // everything this CTA reads or writes is ordered after this wait
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;
      bool ok = true;
      // Failure injection (test hook): CTA 0 leaves its first stage unfilled, so the MMA
      // thread's bounded wait on that stage is one that nothing completes.
      bool skip_stage = p.stall != 0 && blockIdx.x == 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        int m_blk, n_blk, split;
        unit_coords(p, u, m_blk, n_blk, split);
        const int kb0 = split * p.kb_per_split;
        const int kb1 = min(kb0 + p.kb_per_split, p.kb_total);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!wait_bounded(empty0 + 8 * stage, phase ^ 1u, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          if (skip_stage) {
            skip_stage = false;
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
            continue;
          }
          const uint32_t fb = full0 + 8 * stage;
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_TOTAL;
          mbar_arrive_expect_tx(fb, STAGE_BYTES);
          tma_load_2d(sa, &tmA, fb, kb * BK, m_blk * BM);
          if (SPLIT) tma_load_2d(sa + A_BYTES, &tmA2, fb, kb * BK, m_blk * BM);
          if (SWIGLU) {
            tma_load_2d(sb, &tmB, fb, kb * BK, n_blk * (BN / 2));
            tma_load_2d(sb + (BN / 2) * BK * 2, &tmB2, fb, kb * BK, n_blk * (BN / 2));
          } else {
            tma_load_2d(sb, &tmB, fb, kb * BK, n_blk * BN);
          }
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // Drain: every stage's last issued copy has landed before the CTA may exit.
      for (int s = 0; s < STAGES; ++s)
        if (issued & (1u << s)) wait_drain(full0 + 8 * s, (issued_phase >> s) & 1u, limit);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++it) {
        int m_blk, n_blk, split;
        unit_coords(p, u, m_blk, n_blk, split);
        const int kb0 = split * p.kb_per_split;
        const int kb1 = min(kb0 + p.kb_per_split, p.kb_total);
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!wait_bounded(tempty0 + 8 * acc, acc_phase ^ 1u, abort_flag, status, limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!wait_bounded(full0 + 8 * stage, phase, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_TOTAL;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t bdesc = make_sdesc(sb + k * 32);
            tc_mma(d_tmem, make_sdesc(sa + k * 32), bdesc, IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
            if (SPLIT) tc_mma(d_tmem, make_sdesc(sa + A_BYTES + k * 32), bdesc, IDESC, 1u);
          }
          tc_commit(empty0 + 8 * stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) tc_commit(tfull0 + 8 * acc);
      }
      // Drain: all MMAs issued by this thread have completed before TMEM is freed.
      tc_commit(drain_bar);
      wait_drain(drain_bar, 0, limit);
    }
  } else {
    // -------------------------------------------------------------- epilogue warps 2..5
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    uint32_t sat = 0;
    int it = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
      int m_blk, n_blk, split;
      unit_coords(p, u, m_blk, n_blk, split);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      int ok = 1;
      if (lane == 0) ok = wait_bounded(tfull0 + 8 * acc, acc_phase, abort_flag, status, limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int m = m_blk * BM + q * 32 + lane;
      const uint32_t trow = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * BN;
      if (EPI == EPI_SWIGLU)
        epilogue_swiglu<BN>(p, trow, m, n_blk * (BN / 2), sat);
      else if (EPI == EPI_QKV)
        epilogue_qkv<BN>(p, trow, m, n_blk * BN);
      else
        epilogue_plain<BN, EPI>(p, trow, m, n_blk * BN, split, sat);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
    report_saturation(status, sat);
  }

  // Lanes 1..31 of the producer and MMA warps got here long before their lane 0: reconverge
  // each warp first, since the CTA barrier counts whole converged warps.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

// ----------------------------------------------------------------------------- 2-SM GEMM
// The same GEMM on CTA pairs (clusters of 2 on one TPC): a pair computes a 256 x 256 output
// tile with tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 16).  Each CTA loads only its half
// of A (128 rows, hi and lo) and its half of B (128 rows of W; SwiGLU: the even CTA the gate
// rows, the odd CTA the matching up rows) into its own shared memory; the MMA of the pair reads
// both halves, so each SM fills 48 KB of operands per 64-wide k-block instead of 64 KB, for the
// same MMA work.  Each CTA's TMEM holds the pair's accumulator rows of that CTA (two 256-column
// accumulators), and each CTA runs the same epilogue on its rows.
//  * even CTA (leader): its producer posts the expected bytes of both CTAs on its full
//    barrier; its MMA thread issues all MMAs and commits stage releases and accumulator
//    readiness to the barriers of both CTAs (multicast commit);
//  * odd CTA: its producer's TMA loads complete on the leader's full barrier;
//  * both epilogues release an accumulator on the leader's tempty barrier (8 warp arrivals).
// All waits are bounded; a cluster barrier closes the kernel before TMEM is freed, so no CTA
// leaves while its partner's MMAs may still read its shared memory.
template <int STAGES, int EPI, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                    const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmB2,
                    const Params p) {
  constexpr int BN = 256;
  constexpr int A_BYTES = BM * BK * 2;            // 128 rows of A (one half of the pair's 256)
  constexpr int A_TOTAL = SPLIT ? 2 * A_BYTES : A_BYTES;
  constexpr int B_BYTES = (BN / 2) * BK * 2;      // this CTA's 128 rows of B
  constexpr int STAGE_BYTES = A_TOTAL + B_BYTES;
  constexpr uint32_t TMEM_COLS = 2 * BN;
  const uint32_t IDESC = idesc_for((1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BN >> 3) << 17) |
                                       (static_cast<uint32_t>(256 >> 4) << 24),
                                   p.epi.fp16);
  constexpr bool SWIGLU = (EPI == EPI_SWIGLU);

  pdl_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t tfull0 = empty0 + 8 * STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain_bar = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint32_t leader = rank & ~1u;
  const bool is_leader = rank == leader;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << leader);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 8);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers are initialised before either touches the other's
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int units = p.tiles_m * p.tiles_n;
  const int n_pairs = gridDim.x >> 1;
  const int pair = blockIdx.x >> 1;
  uint32_t* status = p.epi.status;
  const uint64_t limit = p.wait_limit;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer (both CTAs)
      pdl_wait_async();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;
      bool ok = true;
      for (int u = pair; u < units && ok; u += n_pairs) {
        int m_blk, n_blk, split;
        unit_coords(p, u, m_blk, n_blk, split);
        const int row_a = m_blk * 256 + static_cast<int>(rank - leader) * 128;
        for (int kb = 0; kb < p.kb_total; ++kb) {
          if (!wait_bounded(empty0 + 8 * stage, phase ^ 1u, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          const uint32_t fb = mapa_shared(full0 + 8 * stage, leader);
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_TOTAL;
          if (is_leader) mbar_arrive_expect_tx(full0 + 8 * stage, 2 * STAGE_BYTES);
          tma_load_2d_pair(sa, &tmA, fb, kb * BK, row_a);
          if (SPLIT) tma_load_2d_pair(sa + A_BYTES, &tmA2, fb, kb * BK, row_a);
          if (SWIGLU)
            tma_load_2d_pair(sb, rank == leader ? &tmB : &tmB2, fb, kb * BK, n_blk * (BN / 2));
          else
            tma_load_2d_pair(sb, &tmB, fb, kb * BK, n_blk * BN + static_cast<int>(rank - leader) * (BN / 2));
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      // Drain (leader only: the pair's loads complete on the leader's barriers).
      if (is_leader)
        for (int s = 0; s < STAGES; ++s)
          if (issued & (1u << s)) wait_drain(full0 + 8 * s, (issued_phase >> s) & 1u, limit);
    }
  } else if (warp == 1) {
    if (lane == 0 && is_leader) {
      // ------------------------------------------------------------ MMA issuer (leader)
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int u = pair; u < units && ok; u += n_pairs, ++it) {
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!wait_bounded(tempty0 + 8 * acc, acc_phase ^ 1u, abort_flag, status, limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < p.kb_total; ++kb) {
          if (!wait_bounded(full0 + 8 * stage, phase, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_TOTAL;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t bdesc = make_sdesc(sb + k * 32);
            tc_mma_pair(d_tmem, make_sdesc(sa + k * 32), bdesc, IDESC, (kb > 0 || k > 0) ? 1u : 0u);
            if (SPLIT) tc_mma_pair(d_tmem, make_sdesc(sa + A_BYTES + k * 32), bdesc, IDESC, 1u);
          }
          tc_commit_pair(empty0 + 8 * stage, pair_mask);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) tc_commit_pair(tfull0 + 8 * acc, pair_mask);
      }
      tc_commit_pair(drain_bar, static_cast<uint16_t>(1u << leader));
      wait_drain(drain_bar, 0, limit);
    }
  } else {
    // -------------------------------------------------------------- epilogue warps 2..5
    const int q = warp & 3;
    const uint32_t tempty_leader = mapa_shared(tempty0, leader);
    uint32_t sat = 0;
    int it = 0;
    for (int u = pair; u < units; u += n_pairs, ++it) {
      int m_blk, n_blk, split;
      unit_coords(p, u, m_blk, n_blk, split);
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      int ok = 1;
      if (lane == 0) ok = wait_bounded(tfull0 + 8 * acc, acc_phase, abort_flag, status, limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int m = m_blk * 256 + static_cast<int>(rank - leader) * 128 + q * 32 + lane;
      const uint32_t trow = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * BN;
      if (EPI == EPI_SWIGLU)
        epilogue_swiglu<BN>(p, trow, m, n_blk * (BN / 2), sat);
      else if (EPI == EPI_QKV)
        epilogue_qkv<BN>(p, trow, m, n_blk * BN);
      else
        epilogue_plain<BN, EPI>(p, trow, m, n_blk * BN, 0, sat);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty_leader + 8 * acc);
    }
    report_saturation(status, sat);
  }

  __syncwarp();  // reconverge the role warps before the CTA and cluster barriers
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the partner's MMAs have finished reading this CTA's shared memory
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                 : "memory");
  }
}

// ----------------------------------------------------------------------------- partial sums
// Partials of a split GEMM are summed in a fixed order, so results do not depend on the
// launch.  Two layouts:
//  SplitSrc   split-K of the tile GEMM: ws[s][M][N], s = 0 .. S-1.
//  StreamSrc  stream-K of the weight-streaming GEMM: ws[slot][BNX][256] (output row n of
//             tile t = n / 256 at column n % 256, batch row m at row m); the CTAs whose
//             iteration ranges cover tile t are c = t*KB / P .. ((t+1)*KB - 1) / P, and CTA c
//             keeps tile t in slot c * max_seg + t - (c * P) / KB.
struct SplitSrc {
  const float* ws;
  int S, M, N;
  static constexpr bool kBatchFastest = false;
  __device__ __forceinline__ float operator()(int m, int n) const {
    float a = 0.f;
    for (int s = 0; s < S; ++s) a += ws[(static_cast<size_t>(s) * M + m) * N + n];
    return a;
  }
};
struct StreamSrc {
  const float* ws;
  int BNX, KB, P, max_seg;
  static constexpr bool kBatchFastest = false;
  __device__ __forceinline__ float operator()(int m, int n) const {
    const int t = n >> 8, r = n & 255;
    const int c0 = (t * KB) / P, c1 = (t * KB + KB - 1) / P;
    float a = 0.f;
    for (int c = c0; c <= c1; ++c) {
      const int slot = c * max_seg + t - (c * P) / KB;
      a += ws[(static_cast<size_t>(slot) * BNX + m) * 256 + r];
    }
    return a;
  }
};

// Linear index -> (row m, rest r) with the layout-friendly order.
template <class Src>
__device__ __forceinline__ void split_index(int64_t i, int M, int64_t R, int& m, int64_t& r) {
  if (Src::kBatchFastest) {
    m = static_cast<int>(i % M);
    r = i / M;
  } else {
    m = static_cast<int>(i / R);
    r = i - static_cast<int64_t>(m) * R;
  }
}

template <class Src>
__global__ void reduce_f32_kernel(Src src, int M, int N, float* out, int ldo, int resid) {
  pdl_launch_dependents();
  pdl_wait();
  const int64_t total = static_cast<int64_t>(M) * N;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    int m;
    int64_t n;
    split_index<Src>(i, M, N, m, n);
    const float acc = src(m, static_cast<int>(n));
    float* o = out + static_cast<size_t>(m) * ldo + n;
    if (resid)
      *o += acc;
    else
      *o = acc;
  }
}

template <class Src>
__global__ void reduce_swiglu_kernel(Src src, int M, int F, bf16* out_hi, bf16* out_lo, int ldo,
                                     bool fp16, uint32_t* status) {
  pdl_launch_dependents();
  pdl_wait();
  uint32_t sat = 0;
  const int64_t total = static_cast<int64_t>(M) * F;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    int m;
    int64_t f;
    split_index<Src>(i, M, F, m, f);
    const float g = src(m, static_cast<int>(f));
    const float u = src(m, static_cast<int>(f) + F);
    store_split1(out_hi, out_lo, static_cast<size_t>(m) * ldo + f, silu_f(g) * u, fp16, sat);
  }
  report_saturation(status, sat);
}

// One thread per (row, q|k|v section, head, i < hd/2): sums the pair (i, i + hd/2).  Rotary
// index i runs along the lanes (hd/2 is a multiple of 32), so the residual byte of elements
// (i, i + 1) is assembled from two neighbouring lanes.
template <class Src>
__global__ void reduce_qkv_kernel(Src src, int M, EpiArgs e) {
  pdl_launch_dependents();
  pdl_wait();
  const int d = e.d, hd = e.hd, half = hd >> 1, H = d / hd;
  const int64_t R = 3LL * H * half;
  const int64_t total = static_cast<int64_t>(M) * R;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    int m;
    int64_t r;
    split_index<Src>(t, M, R, m, r);
    const int i = static_cast<int>(r % half);
    r /= half;
    const int head = static_cast<int>(r % H);
    const int sec = static_cast<int>(r / H);
    const int c = sec * d + head * hd + i;
    float a = src(m, c), b = src(m, c + half);
    const RowInfo ri = e.rows[m];
    if (sec < 2) {
      const float2 cs = e.rope[static_cast<size_t>(ri.pos) * half + i];
      const float ra = a * cs.x - b * cs.y;
      const float rb = b * cs.x + a * cs.y;
      a = ra;
      b = rb;
    }
    if (sec == 0) {
      float* dst = e.out_q + static_cast<size_t>(m) * d + head * hd;
      dst[i] = a;
      dst[i + half] = b;
    } else {
      f16* dst = e.kv.base + static_cast<int64_t>(e.layer) * e.kv.layer_stride +
                 static_cast<int64_t>(ri.env) * e.kv.env_stride + (sec == 2 ? e.kv.kv_stride : 0) +
                 static_cast<int64_t>(head) * e.kv.head_stride + static_cast<int64_t>(ri.pos) * hd;
      uint8_t* res = e.kv.res ? e.kv.res + (dst - e.kv.base) / 2 : nullptr;
      store_kv_pairlanes(dst, res, i, a);
      store_kv_pairlanes(dst, res, i + half, b);
    }
  }
}

// Stream-K reductions of the weight-streaming GEMM, per work item (x: 256-column tile of the
// product, y: chunk of kMR batch rows).  The CTAs whose ranges cover a tile are found once per
// thread and four CTAs' partials are loaded before their adds, which run in ascending CTA
// order as in StreamSrc.  One CTA per work item (a grid of at most two CTAs per SM, which
// would leave room for the next GEMM's CTAs, measured slower: the reduction is bound by
// the latency of its loads).
constexpr int kMR = 4;

struct TileSum {
  const float* base;  // ws + column r of the tile
  int c0, c1;
  int t, KB, P, max_seg, BNX;
  __device__ __forceinline__ TileSum(const StreamSrc& s, int n) {
    t = n >> 8;
    KB = s.KB;
    P = s.P;
    max_seg = s.max_seg;
    BNX = s.BNX;
    c0 = (t * KB) / P;
    c1 = (t * KB + KB - 1) / P;
    base = s.ws + (n & 255);
  }
  __device__ __forceinline__ const float* row(int c, int m) const {
    const int slot = c * max_seg + t - (c * P) / KB;
    return base + (static_cast<size_t>(slot) * BNX + m) * 256;
  }
  // acc[j] = sum over c of partial(c, row m0 + j), rows m0 + j < M only
  __device__ __forceinline__ void sum(int m0, int M, float (&acc)[kMR]) const {
#pragma unroll
    for (int j = 0; j < kMR; ++j) acc[j] = 0.f;
    for (int c = c0; c <= c1; c += 4) {
      float v[4][kMR];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float* src = row(c + u <= c1 ? c + u : c1, m0);
#pragma unroll
        for (int j = 0; j < kMR; ++j) v[u][j] = (c + u <= c1 && m0 + j < M) ? src[j * 256] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (c + u <= c1) {
#pragma unroll
          for (int j = 0; j < kMR; ++j) acc[j] += v[u][j];
        }
    }
  }
  // columns n .. n+3 (n % 4 == 0) of row m; six CTAs' partials in flight
  __device__ __forceinline__ float4 sum4(int m) const {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = c0; c <= c1; c += 6) {
      float4 v[6];
#pragma unroll
      for (int u = 0; u < 6; ++u)
        v[u] = (c + u <= c1) ? *reinterpret_cast<const float4*>(row(c + u, m)) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int u = 0; u < 6; ++u)
        if (c + u <= c1) {
          acc.x += v[u].x;
          acc.y += v[u].y;
          acc.z += v[u].z;
          acc.w += v[u].w;
        }
    }
    return acc;
  }
};

// Two columns' sums (each as TileSum::sum) with both columns' loads in flight together.
__device__ __forceinline__ void sum_pair(const TileSum& A, const TileSum& B, int m0, int M, float (&a)[kMR],
                                         float (&b)[kMR]) {
#pragma unroll
  for (int j = 0; j < kMR; ++j) a[j] = b[j] = 0.f;
  const int na = A.c1 - A.c0 + 1, nb = B.c1 - B.c0 + 1;
  const int n = na > nb ? na : nb;
  for (int i = 0; i < n; i += 4) {
    float va[4][kMR], vb[4][kMR];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const bool ia = i + u < na, ib = i + u < nb;
      const float* sa = A.row(ia ? A.c0 + i + u : A.c1, m0);
      const float* sb = B.row(ib ? B.c0 + i + u : B.c1, m0);
#pragma unroll
      for (int j = 0; j < kMR; ++j) {
        va[u][j] = (ia && m0 + j < M) ? sa[j * 256] : 0.f;
        vb[u][j] = (ib && m0 + j < M) ? sb[j * 256] : 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (i + u < na) {
#pragma unroll
        for (int j = 0; j < kMR; ++j) a[j] += va[u][j];
      }
      if (i + u < nb) {
#pragma unroll
        for (int j = 0; j < kMR; ++j) b[j] += vb[u][j];
      }
    }
  }
}

__device__ __forceinline__ bool next_item(int& item, int nx, int ny, int& x, int& y) {
  if (item >= nx * ny) return false;
  y = item / nx;
  x = item - y * nx;
  item += gridDim.x;
  return true;
}

// items (ceil(N / 256), ceil(M / kMR)), 256 threads: out[m][n] (+)= sum
__global__ void stream_reduce_f32_kernel(StreamSrc src, int M, int N, float* out, int ldo,
                                         int resid) {
  pdl_launch_dependents();
  pdl_wait();
  const int nx = (N + 255) / 256, ny = (M + kMR - 1) / kMR;
  int item = blockIdx.x, bx, by;
  while (next_item(item, nx, ny, bx, by)) {
    const int n = bx * 256 + threadIdx.x;
    if (n >= N) continue;
    const int m0 = by * kMR;
    float acc[kMR];
    TileSum(src, n).sum(m0, M, acc);
#pragma unroll
    for (int j = 0; j < kMR; ++j) {
      if (m0 + j >= M) break;
      float* o = out + static_cast<size_t>(m0 + j) * ldo + n;
      *o = resid ? *o + acc[j] : acc[j];
    }
  }
}

// items (ceil(F / 256), ceil(M / kMR)), 256 threads: gate column f, up column f + F
__global__ void stream_reduce_swiglu_kernel(StreamSrc src, int M, int F, bf16* out_hi,
                                            bf16* out_lo, int ldo, bool fp16, uint32_t* status) {
  pdl_launch_dependents();
  pdl_wait();
  uint32_t sat = 0;
  const int nx = (F + 255) / 256, ny = (M + kMR - 1) / kMR;
  int item = blockIdx.x, bx, by;
  while (next_item(item, nx, ny, bx, by)) {
    const int f = bx * 256 + threadIdx.x;
    if (f >= F) continue;
    const int m0 = by * kMR;
    float g[kMR], u[kMR];
    sum_pair(TileSum(src, f), TileSum(src, f + F), m0, M, g, u);
#pragma unroll
    for (int j = 0; j < kMR; ++j) {
      if (m0 + j >= M) break;
      store_split1(out_hi, out_lo, static_cast<size_t>(m0 + j) * ldo + f, silu_f(g[j]) * u[j], fp16, sat);
    }
  }
  report_saturation(status, sat);
}

// items (3d / 256, ceil(M / kMR)), 128 threads; 256 % hd == 0 and d % 256 == 0, so both
// halves of a rotary pair sit in one tile: thread p takes pair (i, i + hd/2) of local head
// p / (hd/2).
__global__ void stream_reduce_qkv_kernel(StreamSrc src, int M, EpiArgs e) {
  pdl_launch_dependents();
  pdl_wait();
  const int d = e.d, hd = e.hd, half = hd >> 1;
  const int p = threadIdx.x;
  const int i = p % half;
  const int nx = 3 * d / 256, ny = (M + kMR - 1) / kMR;
  int item = blockIdx.x, bx, by;
  while (next_item(item, nx, ny, bx, by)) {
    const int c = bx * 256 + (p / half) * hd + i;
    const int sec = c / d;
    const int head = (c - sec * d) / hd;
    const int m0 = by * kMR;
    float a[kMR], b[kMR];
    sum_pair(TileSum(src, c), TileSum(src, c + half), m0, M, a, b);
#pragma unroll
    for (int j = 0; j < kMR; ++j) {
      const int m = m0 + j;
      if (m >= M) break;
      const RowInfo ri = e.rows[m];
      float x = a[j], y = b[j];
      if (sec < 2) {
        const float2 cs = e.rope[static_cast<size_t>(ri.pos) * half + i];
        const float rx = x * cs.x - y * cs.y;
        const float ry = y * cs.x + x * cs.y;
        x = rx;
        y = ry;
      }
      if (sec == 0) {
        float* dst = e.out_q + static_cast<size_t>(m) * d + head * hd;
        dst[i] = x;
        dst[i + half] = y;
      } else {
        f16* dst = e.kv.base + static_cast<int64_t>(e.layer) * e.kv.layer_stride +
                   static_cast<int64_t>(ri.env) * e.kv.env_stride + (sec == 2 ? e.kv.kv_stride : 0) +
                   static_cast<int64_t>(head) * e.kv.head_stride + static_cast<int64_t>(ri.pos) * hd;
        uint8_t* res = e.kv.res ? e.kv.res + (dst - e.kv.base) / 2 : nullptr;
        store_kv_pairlanes(dst, res, i, x);
        store_kv_pairlanes(dst, res, i + half, y);
      }
    }
  }
}

// grid (M), 1024 threads (N % 4 == 0): h[m][n] += sum, then the RMSNorm of the updated row
// times w as the operand pair y_hi / y_lo (the next GEMM's A; bf16, or fp16 when fp16).  The row sums are in the same
// order as stream_reduce_f32_kernel's.  At most 48 registers: with one 1024-thread CTA on an
// SM, the next weight-streaming GEMM's CTA (192 threads x 40) still fits beside it.
__global__ void __maxnreg__(48) stream_reduce_resid_norm_kernel(StreamSrc src, int N, float* h,
                                                                         int ldh, const bf16* w, float eps,
                                                                         bf16* y_hi, bf16* y_lo, int ldy,
                                                                         bool fp16, uint32_t* status) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[32];
  const int m = blockIdx.x;
  float* hrow = h + static_cast<size_t>(m) * ldh;
  uint32_t sat = 0;
  float ss = 0.f;
  for (int n = threadIdx.x * 4; n < N; n += blockDim.x * 4) {
    const float4 acc = TileSum(src, n).sum4(m);
    float4 v = *reinterpret_cast<const float4*>(hrow + n);
    v.x += acc.x;
    v.y += acc.y;
    v.z += acc.z;
    v.w += acc.w;
    *reinterpret_cast<float4*>(hrow + n) = v;
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.f;
  for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) tot += red[i];
  const float r = rsqrtf(tot / static_cast<float>(N) + eps);
  for (int n = threadIdx.x * 4; n < N; n += blockDim.x * 4) {
    const float4 v = *reinterpret_cast<const float4*>(hrow + n);
    const uint2 ww = *reinterpret_cast<const uint2*>(w + n);
    const float2 w0 = unpack_bf16x2(ww.x), w1 = unpack_bf16x2(ww.y);
    uint2 hi, lo;
    split_pack2(v.x * r * w0.x, v.y * r * w0.y, hi.x, lo.x, fp16, sat);
    split_pack2(v.z * r * w1.x, v.w * r * w1.y, hi.y, lo.y, fp16, sat);
    *reinterpret_cast<uint2*>(y_hi + static_cast<size_t>(m) * ldy + n) = hi;
    *reinterpret_cast<uint2*>(y_lo + static_cast<size_t>(m) * ldy + n) = lo;
  }
  report_saturation(status, sat);
}

// ----------------------------------------------------------------------------- decode GEMM
// Weight-streaming GEMM for decode-sized batches (M <= 128 rows of activations), where the
// projections are bound by reading the weights from HBM once.
//  * swap-AB: the 128-row weight tile is the MMA's A operand and the batch (BNX rows, the
//    activation pair hi / lo) is its N, so no MMA row is wasted on padding and the
//    activation tiles cost smem fill BNX/128 of the weights';
//  * stream-K: the (n-tile, k-block) iteration space is cut into equal contiguous ranges,
//    one per CTA, so all SMs stream the same number of weight bytes; each run of one tile
//    inside a range accumulates in TMEM and is written as one fp32 partial (StreamSrc);
//  * weights are loaded evict-first, activations evict-last.
struct GemvParams {
  int N, K;
  int tiles, kbt;       // 256-row tiles of W, 64-wide k-blocks per tile
  int per_cta, max_seg; // stream-K range length and partial slots per CTA
  float* ws;
  uint32_t* status;
  bool fp16;            // operand format (weights and activation pair): fp16, else bf16
  uint64_t wait_limit;  // ns per bounded mbarrier wait
};

// TR = 256 weight rows per tile, as two M=128 MMAs sharing each activation tile, so the
// activation fill per weight byte is BNX/256 * 2 and 4 stages keep 128 KB of weights in flight.
template <int BNX, int STAGES>
__global__ void __launch_bounds__(kThreads, 1)
    gemv_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                   const __grid_constant__ CUtensorMap tmX2, const GemvParams p) {
  constexpr int TR = 256, NH = TR / 128;
  constexpr int W_HALF = 128 * BK * 2;
  constexpr int W_BYTES = NH * W_HALF;
  constexpr int X_BYTES = BNX * BK * 2;
  constexpr int STAGE_BYTES = W_BYTES + 2 * X_BYTES;
  constexpr uint32_t TMEM_COLS = 2 * NH * BNX;
  const uint32_t IDESC = idesc_for((1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(BNX >> 3) << 17) |
                                       (static_cast<uint32_t>(128 >> 4) << 24),
                                   p.fp16);
  static_assert(TMEM_COLS >= 32 && (TMEM_COLS & (TMEM_COLS - 1)) == 0, "TMEM allocation");

  pdl_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t tfull0 = empty0 + 8 * STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain_bar = tempty0 + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 4);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmW)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int total = p.tiles * p.kbt;
  const int g_begin = blockIdx.x * p.per_cta;
  const int g_end = min(g_begin + p.per_cta, total);
  const int t_first = g_begin / p.kbt;
  uint32_t* status = p.status;
  const uint64_t limit = p.wait_limit;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      // The weights do not depend on the previous kernel: the first STAGES weight tiles are
      // requested before waiting for it, the activations only after.
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_x = policy_evict_last();
      const int n = g_end - g_begin;
      const int pre = n < STAGES ? n : STAGES;
      uint32_t issued = 0, issued_phase = 0;
      for (int i = 0; i < pre; ++i) {
        const int g = g_begin + i, t = g / p.kbt, kb = g - t * p.kbt;
        const uint32_t sw = smem_u32(smem + i * STAGE_BYTES);
        mbar_arrive_expect_tx(full0 + 8 * i, STAGE_BYTES);
        tma_load_2d_hint(sw, &tmW, full0 + 8 * i, kb * BK, t * TR, pol_w);
        issued |= 1u << i;
      }
      pdl_wait_async();
      for (int i = 0; i < pre; ++i) {
        const int g = g_begin + i, t = g / p.kbt, kb = g - t * p.kbt;
        (void)t;
        const uint32_t sx = smem_u32(smem + i * STAGE_BYTES) + W_BYTES;
        tma_load_2d_hint(sx, &tmX, full0 + 8 * i, kb * BK, 0, pol_x);
        tma_load_2d_hint(sx + X_BYTES, &tmX2, full0 + 8 * i, kb * BK, 0, pol_x);
      }
      int stage = pre % STAGES;
      uint32_t phase = (pre == STAGES) ? 1u : 0u;
      for (int i = pre; i < n; ++i) {
        const int g = g_begin + i, t = g / p.kbt, kb = g - t * p.kbt;
        if (!wait_bounded(empty0 + 8 * stage, phase ^ 1u, abort_flag, status, limit)) break;
        const uint32_t fb = full0 + 8 * stage;
        const uint32_t sw = smem_u32(smem + stage * STAGE_BYTES);
        const uint32_t sx = sw + W_BYTES;
        mbar_arrive_expect_tx(fb, STAGE_BYTES);
        tma_load_2d_hint(sw, &tmW, fb, kb * BK, t * TR, pol_w);
        tma_load_2d_hint(sx, &tmX, fb, kb * BK, 0, pol_x);
        tma_load_2d_hint(sx + X_BYTES, &tmX2, fb, kb * BK, 0, pol_x);
        issued |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
      for (int s = 0; s < STAGES; ++s)
        if (issued & (1u << s)) wait_drain(full0 + 8 * s, (issued_phase >> s) & 1u, limit);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      bool ok = true;
      for (int g = g_begin; g < g_end && ok; ++it) {
        const int t = g / p.kbt;
        const int kb0 = g - t * p.kbt;
        const int kb1 = min(p.kbt, kb0 + (g_end - g));
        g += kb1 - kb0;
        const int acc = it & 1;
        const uint32_t acc_phase = (it >> 1) & 1;
        if (!wait_bounded(tempty0 + 8 * acc, acc_phase ^ 1u, abort_flag, status, limit)) break;
        tc_fence_after();
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!wait_bounded(full0 + 8 * stage, phase, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sw = smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sx = sw + W_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t xh = make_sdesc(sx + k * 32);
            const uint64_t xl = make_sdesc(sx + X_BYTES + k * 32);
#pragma unroll
            for (int h = 0; h < NH; ++h) {
              const uint32_t d_tmem = tmem_base + (acc * NH + h) * BNX;
              const uint64_t adesc = make_sdesc(sw + h * W_HALF + k * 32);
              tc_mma(d_tmem, adesc, xh, IDESC, (kb > kb0 || k > 0) ? 1u : 0u);
              tc_mma(d_tmem, adesc, xl, IDESC, 1u);
            }
          }
          tc_commit(empty0 + 8 * stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) tc_commit(tfull0 + 8 * acc);
      }
      tc_commit(drain_bar);
      wait_drain(drain_bar, 0, limit);
    }
  } else {
    // -------------------------------------------------------------- epilogue warps 2..5
    const int q = warp & 3;
    int it = 0;
    for (int g = g_begin; g < g_end; ++it) {
      const int t = g / p.kbt;
      const int kb0 = g - t * p.kbt;
      const int kb1 = min(p.kbt, kb0 + (g_end - g));
      g += kb1 - kb0;
      const int acc = it & 1;
      const uint32_t acc_phase = (it >> 1) & 1;
      int ok = 1;
      if (lane == 0) ok = wait_bounded(tfull0 + 8 * acc, acc_phase, abort_flag, status, limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int slot = blockIdx.x * p.max_seg + (t - t_first);
      // partial layout [slot][batch column][tile row]: for each batch column the 32 lanes of a
      // warp store 32 consecutive rows (coalesced), and the reduction reads rows contiguously
#pragma unroll
      for (int h = 0; h < NH; ++h) {
        const int r = h * 128 + q * 32 + lane;
        float* dst = p.ws + static_cast<size_t>(slot) * BNX * TR + r;
        const uint32_t trow = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + (acc * NH + h) * BNX;
#pragma unroll 1
        for (int c = 0; c < BNX; c += 16) {
          float v[16];
          ld16f(trow + c, v);
#pragma unroll
          for (int i = 0; i < 16; ++i) dst[static_cast<size_t>(c + i) * TR] = v[i];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
    }
  }

  // Lanes 1..31 of the producer and MMA warps got here long before their lane 0: reconverge
  // each warp first, since the CTA barrier counts whole converged warps.
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TMEM_COLS)
                 : "memory");
  }
}

// ----------------------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// 2-D map of 2-byte elements (bf16, or fp16 when fp16) over [rows, cols] (row stride ld
// elements), box {64, box_rows}, 128B swizzle.
bool make_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld,
              int box_rows, bool fp16 = false) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(ptr), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

struct Maps {
  CUtensorMap a, a2, b, b2;
};

template <int BN, int EPI, bool SPLIT>
int launch_kernel(const Maps& m, const Params& p, int grid, cudaStream_t stream) {
  // ~192 KB of stages: BN=256 -> 4 (3 split), BN=128 -> 6 (4 split)
  constexpr int STAGE = (SPLIT ? 2 : 1) * BM * BK * 2 + BN * BK * 2;
  constexpr int STAGES = (196608 / STAGE) < 8 ? (196608 / STAGE) : 8;
  constexpr int smem = STAGES * STAGE + 1024 + 256;
  static std::atomic<uint64_t> attr_done{0};
  auto kern = gemm_tc_kernel<BN, STAGES, EPI, SPLIT>;
  VLA_CUDA_TRY(set_smem_limit(kern, smem, attr_done));
  VLA_CUDA_TRY(launch_pdl(kern, dim3(grid), dim3(kThreads), smem, stream, m.a, m.a2, m.b, m.b2, p));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

template <int EPI, bool SPLIT>
int launch_pair_kernel(const Maps& m, const Params& p, int grid, cudaStream_t stream) {
  constexpr int STAGE = (SPLIT ? 2 : 1) * BM * BK * 2 + 128 * BK * 2;
  constexpr int STAGES = (196608 / STAGE) < 8 ? (196608 / STAGE) : 8;
  constexpr int smem = STAGES * STAGE + 1024 + 256;
  static std::atomic<uint64_t> attr_done{0};
  auto kern = gemm_tc2_kernel<STAGES, EPI, SPLIT>;
  VLA_CUDA_TRY(set_smem_limit(kern, smem, attr_done));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  VLA_CUDA_TRY(injected_launch_error());
  VLA_CUDA_TRY(cudaLaunchKernelEx(&cfg, kern, m.a, m.a2, m.b, m.b2, p));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

template <bool SPLIT>
int dispatch_pair(int epi, const Maps& m, const Params& p, int grid, cudaStream_t s) {
  switch (epi) {
    case EPI_F32: return launch_pair_kernel<EPI_F32, SPLIT>(m, p, grid, s);
    case EPI_RESID: return launch_pair_kernel<EPI_RESID, SPLIT>(m, p, grid, s);
    case EPI_SWIGLU: return launch_pair_kernel<EPI_SWIGLU, SPLIT>(m, p, grid, s);
    case EPI_QKV: return launch_pair_kernel<EPI_QKV, SPLIT>(m, p, grid, s);
  }
  return VLA_ERR_ARG;
}

template <int BN, bool SPLIT>
int dispatch_epi(int epi, const Maps& m, const Params& p, int grid, cudaStream_t s) {
  switch (epi) {
    case EPI_F32: return launch_kernel<BN, EPI_F32, SPLIT>(m, p, grid, s);
    case EPI_RESID: return launch_kernel<BN, EPI_RESID, SPLIT>(m, p, grid, s);
    case EPI_SWIGLU: return launch_kernel<BN, EPI_SWIGLU, SPLIT>(m, p, grid, s);
    case EPI_QKV: return launch_kernel<BN, EPI_QKV, SPLIT>(m, p, grid, s);
    case EPI_PARTIAL: return launch_kernel<BN, EPI_PARTIAL, SPLIT>(m, p, grid, s);
  }
  return VLA_ERR_ARG;
}

int blocks_for(int64_t n) {
  int64_t b = (n + 255) / 256;
  if (b > 4096) b = 4096;
  return static_cast<int>(b < 1 ? 1 : b);
}


// Applies the epilogue of `a` to summed partials.
template <class Src>
int launch_reduce(const Src& src, const GemmArgs& a, cudaStream_t stream) {
  const int epi = a.epi.kind;
  switch (epi) {
    case EPI_F32:
    case EPI_RESID: {
      float* out = (epi == EPI_F32) ? a.epi.out_f32 : a.epi.resid;
      const int ld = (epi == EPI_F32) ? a.epi.ldo : a.epi.ldr;
      VLA_CUDA_TRY(launch_pdl(reduce_f32_kernel<Src>, dim3(blocks_for(static_cast<int64_t>(a.M) * a.N)),
                              dim3(256), 0, stream, src, a.M, a.N, out, ld, epi == EPI_RESID ? 1 : 0));
      break;
    }
    case EPI_SWIGLU:
      VLA_CUDA_TRY(launch_pdl(reduce_swiglu_kernel<Src>, dim3(blocks_for(static_cast<int64_t>(a.M) * a.N / 2)),
                              dim3(256), 0, stream, src, a.M, a.N / 2, a.epi.out_hi, a.epi.out_lo, a.epi.ldo,
                              a.epi.fp16, a.epi.status));
      break;
    case EPI_QKV:
      VLA_CUDA_TRY(launch_pdl(reduce_qkv_kernel<Src>, dim3(blocks_for(static_cast<int64_t>(a.M) * a.N / 2)),
                              dim3(256), 0, stream, src, a.M, a.epi));
      break;
    default:
      return VLA_ERR_ARG;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

GemmCost gemm_cost(const GemmArgs& a) {
  // Algorithmic work of the model's product: 2MNK flops (the low-half MMAs of a split A are
  // not counted); bytes = A + B read once, output written once (+ read for the residual).
  GemmCost c;
  c.flops = 2.0 * a.M * static_cast<double>(a.N) * a.K;
  double out_bytes;
  switch (a.epi.kind) {
    case EPI_RESID: out_bytes = 8.0 * a.M * a.N; break;
    case EPI_SWIGLU: out_bytes = 2.0 * a.M * (a.N / 2) * (a.epi.out_lo ? 2 : 1); break;
    case EPI_QKV: out_bytes = 2.0 * a.M * a.N; break;
    default: out_bytes = 4.0 * a.M * a.N;
  }
  const double a_bytes = 2.0 * a.M * static_cast<double>(a.K) * (a.A_lo ? 2 : 1);
  c.bytes = a_bytes + 2.0 * static_cast<double>(a.N) * a.K + out_bytes;
  return c;
}

// Stream-K plan of the weight-streaming GEMM.
struct GemvPlan {
  int bnx, grid, tiles, kbt, per_cta, max_seg;
  size_t ws_bytes;
};
GemvPlan gemv_plan(int M, int N, int K, int num_sms) {
  GemvPlan g{};
  g.bnx = M <= 16 ? 16 : M <= 32 ? 32 : M <= 64 ? 64 : 128;
  g.tiles = (N + 255) / 256;
  g.kbt = (K + BK - 1) / BK;
  const int total = g.tiles * g.kbt;
  int grid = total < num_sms ? total : num_sms;
  g.per_cta = (total + grid - 1) / grid;
  g.grid = (total + g.per_cta - 1) / g.per_cta;
  g.max_seg = (g.per_cta - 1) / g.kbt + 2;
  g.ws_bytes = static_cast<size_t>(g.grid) * g.max_seg * 256 * g.bnx * sizeof(float);
  return g;
}

template <int BNX>
int launch_gemv(const CUtensorMap& w, const CUtensorMap& x, const CUtensorMap& x2,
                const GemvParams& p, int grid, cudaStream_t stream) {
  constexpr int STAGE = 256 * BK * 2 + 2 * BNX * BK * 2;
  constexpr int STAGES = (196608 / STAGE) < 8 ? (196608 / STAGE) : 8;
  constexpr int smem = STAGES * STAGE + 1024 + 256;
  static std::atomic<uint64_t> attr_done{0};
  auto kern = gemv_tc_kernel<BNX, STAGES>;
  VLA_CUDA_TRY(set_smem_limit(kern, smem, attr_done));
  VLA_CUDA_TRY(launch_pdl(kern, dim3(grid), dim3(kThreads), smem, stream, w, x, x2, p));
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace

// Exported for the attention kernels (tiles of the KV cache).
bool make_tensor_map_2d(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_rows,
                        bool fp16) {
  return make_map(m, ptr, rows, cols, ld, box_rows, fp16);
}

std::atomic<int> g_test_stall{0};

void gemm_stall_next_launch() { g_test_stall.store(1); }

int gemm_effective_splits(int K, int splits) {
  const int kbt = (K + BK - 1) / BK;
  if (splits < 1) splits = 1;
  if (splits > kbt) splits = kbt;
  const int kbps = (kbt + splits - 1) / splits;
  return (kbt + kbps - 1) / kbps;
}

size_t gemm_workspace_bytes(const GemmArgs& a) {
  const int s = gemm_effective_splits(a.K, a.splits);
  if (s <= 1) return 0;
  return static_cast<size_t>(s) * a.M * a.N * sizeof(float);
}

int gemm_launch(const GemmArgs& a, cudaStream_t stream, int num_sms, GemmCost* cost) {
  if (a.M < 1 || a.N < 1 || a.K < 1 || !a.A || !a.B) return VLA_ERR_ARG;
  if (a.block_n != 128 && a.block_n != 256) return VLA_ERR_ARG;
  // a following RMSNorm: only as the deferred form (ss_out), on an unsplit residual GEMM (its
  // low half is skipped when norm_lo is null)
  if (a.epi.norm_w && (!a.epi.ss_out || a.epi.kind != EPI_RESID || !a.epi.norm_hi))
    return VLA_ERR_ARG;
  if (a.epi.row_ss && a.epi.kind != EPI_QKV && a.epi.kind != EPI_SWIGLU) return VLA_ERR_ARG;
  if ((a.lda % 8) || (a.ldb % 8) || a.lda < a.K || a.ldb < a.K) return VLA_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(a.A) & 15) || (reinterpret_cast<uintptr_t>(a.B) & 15) ||
      (reinterpret_cast<uintptr_t>(a.A_lo) & 15))
    return VLA_ERR_ARG;
  const bool split = a.A_lo != nullptr;
  const int BN = a.block_n;
  const int epi = a.epi.kind;
  const bool swiglu = (epi == EPI_SWIGLU);
  if (swiglu && (a.N & 1)) return VLA_ERR_ARG;
  if (epi == EPI_QKV && (a.epi.d % BN || BN % a.epi.hd || a.N != 3 * a.epi.d)) return VLA_ERR_ARG;

  const int splits = gemm_effective_splits(a.K, a.splits);
  if (a.pair && (BN != 256 || splits != 1)) return VLA_ERR_ARG;
  if ((a.epi.ss_out || a.epi.row_ss) && splits != 1) return VLA_ERR_ARG;
  const int kbt = (a.K + BK - 1) / BK;
  Params p{};
  p.M = a.M;
  p.N = a.N;
  p.K = a.K;
  p.tiles_m = a.pair ? (a.M + 255) / 256 : (a.M + BM - 1) / BM;
  p.group_m = a.pair ? kGroupMPair : kGroupM;
  p.splits = splits;
  p.kb_total = kbt;
  p.kb_per_split = (kbt + splits - 1) / splits;
  p.epi = a.epi;
  p.wait_limit = g_wait_limit_ns.load(std::memory_order_relaxed);

  Maps maps;
  CUtensorMap &ma = maps.a, &mb = maps.b, &mb2 = maps.b2;
  const bool fp16 = a.epi.fp16;
  if (!make_map(&ma, a.A, a.M, a.K, a.lda, BM, fp16)) return cuda_fail(cudaErrorInvalidValue, "tensor map A");
  maps.a2 = ma;
  if (split && !make_map(&maps.a2, a.A_lo, a.M, a.K, a.lda, BM, fp16))
    return cuda_fail(cudaErrorInvalidValue, "tensor map A (low half)");
  int run_epi = epi;
  if (splits > 1) {
    // Split-K: plain tiles of B into the workspace, then a fixed-order reduction applying
    // the epilogue.
    if (!a.workspace || a.workspace_bytes < gemm_workspace_bytes(a)) return VLA_ERR_ARG;
    run_epi = EPI_PARTIAL;
    p.epi.out_f32 = a.workspace;
    p.tiles_n = (a.N + BN - 1) / BN;
    if (!make_map(&mb, a.B, a.N, a.K, a.ldb, BN, fp16)) return cuda_fail(cudaErrorInvalidValue, "tensor map B");
    mb2 = mb;
  } else if (swiglu) {
    const int F = a.N / 2;
    p.tiles_n = (F + BN / 2 - 1) / (BN / 2);
    const bf16* up = a.B + static_cast<size_t>(F) * a.ldb;
    if ((reinterpret_cast<uintptr_t>(up) & 15)) return VLA_ERR_ARG;
    if (!make_map(&mb, a.B, F, a.K, a.ldb, BN / 2, fp16) || !make_map(&mb2, up, F, a.K, a.ldb, BN / 2, fp16))
      return cuda_fail(cudaErrorInvalidValue, "tensor map B (gate/up)");
  } else {
    p.tiles_n = (a.N + BN - 1) / BN;
    // a pair's CTAs each load half of the 256-row B tile
    if (!make_map(&mb, a.B, a.N, a.K, a.ldb, a.pair ? BN / 2 : BN, fp16))
      return cuda_fail(cudaErrorInvalidValue, "tensor map B");
    mb2 = mb;
  }
  const int64_t units = static_cast<int64_t>(p.tiles_m) * p.tiles_n * p.splits;
  int rc;
  if (a.pair) {
    const int pairs = static_cast<int>(units < num_sms / 2 ? units : num_sms / 2);
    rc = split ? dispatch_pair<true>(epi, maps, p, 2 * pairs, stream)
               : dispatch_pair<false>(epi, maps, p, 2 * pairs, stream);
    if (rc != VLA_OK) return rc;
    if (cost) *cost = gemm_cost(a);
    return VLA_OK;
  }
  const int grid = static_cast<int>(units < num_sms ? units : num_sms);
  p.stall = g_test_stall.exchange(0);  // failure injection: consumed by one tile-GEMM launch
  if (split)
    rc = (BN == 256) ? dispatch_epi<256, true>(run_epi, maps, p, grid, stream)
                     : dispatch_epi<128, true>(run_epi, maps, p, grid, stream);
  else
    rc = (BN == 256) ? dispatch_epi<256, false>(run_epi, maps, p, grid, stream)
                     : dispatch_epi<128, false>(run_epi, maps, p, grid, stream);
  if (rc != VLA_OK) return rc;

  if (splits > 1) {
    const SplitSrc src{a.workspace, splits, a.M, a.N};
    if ((rc = launch_reduce(src, a, stream)) != VLA_OK) return rc;
  }
  if (cost) *cost = gemm_cost(a);
  return VLA_OK;
}


size_t gemv_workspace_bytes(int M, int N, int K, int num_sms) {
  if (M < 1 || M > 128) return 0;
  return gemv_plan(M, N, K, num_sms).ws_bytes;
}

int gemv_launch(const GemmArgs& a, cudaStream_t stream, int num_sms, GemmCost* cost) {
  if (a.M < 1 || a.M > 128 || a.N < 1 || a.K < 1 || !a.A || !a.A_lo || !a.B) return VLA_ERR_ARG;
  if ((a.lda % 8) || (a.ldb % 8) || a.lda < a.K || a.ldb < a.K) return VLA_ERR_ARG;
  if ((reinterpret_cast<uintptr_t>(a.A) & 15) || (reinterpret_cast<uintptr_t>(a.B) & 15) ||
      (reinterpret_cast<uintptr_t>(a.A_lo) & 15))
    return VLA_ERR_ARG;
  if (a.epi.kind == EPI_SWIGLU && (a.N & 1)) return VLA_ERR_ARG;
  if (a.epi.kind == EPI_QKV && a.N != 3 * a.epi.d) return VLA_ERR_ARG;
  if (a.epi.norm_w) {
    if (a.epi.kind != EPI_RESID || (a.N & 3) || (a.epi.ldr & 3) || (a.epi.ldn & 3) || !a.epi.norm_hi ||
        !a.epi.norm_lo || (reinterpret_cast<uintptr_t>(a.epi.resid) & 15) ||
        (reinterpret_cast<uintptr_t>(a.epi.norm_w) & 7) || (reinterpret_cast<uintptr_t>(a.epi.norm_hi) & 7) ||
        (reinterpret_cast<uintptr_t>(a.epi.norm_lo) & 7))
      return VLA_ERR_ARG;
  }
  const GemvPlan pl = gemv_plan(a.M, a.N, a.K, num_sms);
  if (!a.workspace || a.workspace_bytes < pl.ws_bytes || (reinterpret_cast<uintptr_t>(a.workspace) & 15))
    return VLA_ERR_ARG;
  CUtensorMap mw, mx, mx2;
  const bool fp16 = a.epi.fp16;
  if (!make_map(&mw, a.B, a.N, a.K, a.ldb, 256, fp16) || !make_map(&mx, a.A, a.M, a.K, a.lda, pl.bnx, fp16) ||
      !make_map(&mx2, a.A_lo, a.M, a.K, a.lda, pl.bnx, fp16))
    return cuda_fail(cudaErrorInvalidValue, "tensor maps (decode GEMM)");
  GemvParams p{};
  p.N = a.N;
  p.K = a.K;
  p.tiles = pl.tiles;
  p.kbt = pl.kbt;
  p.per_cta = pl.per_cta;
  p.max_seg = pl.max_seg;
  p.ws = a.workspace;
  p.status = a.epi.status;
  p.fp16 = fp16;
  p.wait_limit = g_wait_limit_ns.load(std::memory_order_relaxed);
  int rc;
  switch (pl.bnx) {
    case 16: rc = launch_gemv<16>(mw, mx, mx2, p, pl.grid, stream); break;
    case 32: rc = launch_gemv<32>(mw, mx, mx2, p, pl.grid, stream); break;
    case 64: rc = launch_gemv<64>(mw, mx, mx2, p, pl.grid, stream); break;
    default: rc = launch_gemv<128>(mw, mx, mx2, p, pl.grid, stream); break;
  }
  if (rc != VLA_OK) return rc;
  const StreamSrc src{a.workspace, pl.bnx, pl.kbt, pl.per_cta, pl.max_seg};
  const int ny = (a.M + kMR - 1) / kMR;
  auto grid_for = [&](int nx) { return dim3(nx * ny); };
  switch (a.epi.kind) {
    case EPI_F32:
    case EPI_RESID: {
      const bool resid = a.epi.kind == EPI_RESID;
      if (resid && a.epi.norm_w) {
        VLA_CUDA_TRY(launch_pdl(stream_reduce_resid_norm_kernel, dim3(a.M), dim3(1024), 0, stream, src, a.N,
                                a.epi.resid, a.epi.ldr, a.epi.norm_w, a.epi.norm_eps, a.epi.norm_hi,
                                a.epi.norm_lo, a.epi.ldn, fp16, a.epi.status));
        break;
      }
      VLA_CUDA_TRY(launch_pdl(stream_reduce_f32_kernel, grid_for((a.N + 255) / 256), dim3(256), 0, stream, src,
                              a.M, a.N, resid ? a.epi.resid : a.epi.out_f32, resid ? a.epi.ldr : a.epi.ldo,
                              resid ? 1 : 0));
      break;
    }
    case EPI_SWIGLU:
      VLA_CUDA_TRY(launch_pdl(stream_reduce_swiglu_kernel, grid_for((a.N / 2 + 255) / 256), dim3(256), 0,
                              stream, src, a.M, a.N / 2, a.epi.out_hi, a.epi.out_lo, a.epi.ldo, fp16,
                              a.epi.status));
      break;
    case EPI_QKV:
      if (256 % a.epi.hd == 0 && a.epi.d % 256 == 0) {
        VLA_CUDA_TRY(launch_pdl(stream_reduce_qkv_kernel, grid_for(a.N / 256), dim3(128), 0, stream, src, a.M,
                                a.epi));
      } else {
        // rotary pairs may straddle tiles: element-wise reduction
        if ((rc = launch_reduce(src, a, stream)) != VLA_OK) return rc;
        if (cost) *cost = gemm_cost(a);
        return VLA_OK;
      }
      break;
    default:
      return VLA_ERR_ARG;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  if (cost) *cost = gemm_cost(a);
  return VLA_OK;
}

}  // namespace vla

// ============================================================================= no-allocation
// Split-K GEMM whose partial sums live in a fixed, file-scope device array instead of a
// caller-provided workspace.  It serves callers that cannot allocate device memory, e.g.
// code running where every device byte belongs to another allocator (a host framework's
// memory pool, a plugin without access to it) or a control loop that must not pay the
// device-wide synchronisation of cudaMalloc / cudaFree.  The array is 8 MiB; every device
// that loads this library keeps it until the process exits.
namespace vla {
namespace {

constexpr size_t kNoAllocScratchFloats = static_cast<size_t>(2) << 20;  // 8 MiB of fp32
__device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
float* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  In host code the array's
// name is only a host-side stand-in, so the address is looked up once per device (with that
// device current) and cached.
int noalloc_scratch(float** out) {
  int dev = 0;
  VLA_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return record_error(VLA_ERR_UNSUPPORTED, "no-alloc GEMM: device index >= 64");
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    VLA_CUDA_TRY(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    g_noalloc_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return VLA_OK;
}

}  // namespace
}  // namespace vla

extern "C" int vla_op_gemm_bf16_noalloc(const void* A, const void* A_lo, int lda, const void* W,
                                        int ldw, float* C, int ldc, int M, int N, int K,
                                        int block_n, int splits, void* cuda_stream) {
  using namespace vla;
  if (!A || !W || !C || M < 1 || N < 1 || K < 1 || ldc < N)
    return record_error(VLA_ERR_ARG, "vla_op_gemm_bf16_noalloc: bad argument");
  GemmArgs g;
  g.A = static_cast<const bf16*>(A);
  g.A_lo = static_cast<const bf16*>(A_lo);
  g.lda = lda;
  g.B = static_cast<const bf16*>(W);
  g.ldb = ldw;
  g.M = M;
  g.N = N;
  g.K = K;
  g.block_n = block_n;
  g.splits = splits;
  g.epi.kind = EPI_F32;
  g.epi.out_f32 = C;
  g.epi.ldo = ldc;
  const size_t need = gemm_workspace_bytes(g);
  if (need > kNoAllocScratchFloats * sizeof(float))
    return record_error(VLA_ERR_CAPACITY,
                        "vla_op_gemm_bf16_noalloc: splits * M * N * 4 bytes exceeds the 8 MiB "
                        "static scratch; lower splits or use vla_op_gemm_bf16 with a workspace");
  if (need > 0) {
    // Every partial of every split is written before the reduction reads it, so the
    // previous call's contents never leak into this one and nothing needs clearing.
    int rc = noalloc_scratch(&g.workspace);
    if (rc != VLA_OK) return rc;
    g.workspace_bytes = kNoAllocScratchFloats * sizeof(float);
  }
  if (const int rs = op_status_word(&g.epi.status)) return rs;
  int dev = 0;
  VLA_CUDA_TRY(cudaGetDevice(&dev));
  int n_sms = 0;
  if (cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n_sms <= 0)
    n_sms = 148;
  const int rc = gemm_launch(g, static_cast<cudaStream_t>(cuda_stream), n_sms, nullptr);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA)
    return record_error(rc, "vla_op_gemm_bf16_noalloc: unsupported arguments");
  return rc;
}

