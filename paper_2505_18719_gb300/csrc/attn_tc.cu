// Chunk causal attention on the tcgen05 tensor cores (paper §3.1: the policy's Llama-2
// self-attention; §3.3: every chunk of a multi-turn trajectory attends to the whole context):
// query tiles of up to 128 rows of one env (a prefill chunk, or the teacher-forced action rows
// of the PPO ratio pass, Eq. 2) against keys 0..pos of that env, one CTA per (tile, head).
//
// Precision: the cached keys / values are fp16 plus a 4-bit residual (KVLayout), read here as
// the pair hi + lo; the queries (fp32) and the softmax weights are split into fp16 pairs too, and
// each product takes three MMAs into one fp32 accumulator:
//   S = Q_hi K_hi^T + Q_lo K_hi^T + Q_hi K_lo^T,    O += P_hi V_hi + P_lo V_hi + P_hi V_lo.
//
// Roles (448 threads):
//   warp 0      TMA producer: per 64-key block, K_hi and V_hi (tensor map over the whole cache,
//               128-byte swizzle) and the two residual byte ranges (bulk copies), three stages;
//   warp 1      TMEM owner (512 columns) and MMA issuer: S = Q K^T with Q read from TMEM (A
//               operand) and K from shared memory (K-major B); O += P V with P from TMEM and V
//               straight from the cache rows (keys x dims, the MN-major B operand); S is
//               double-buffered, and the issuer takes whichever of "S of the next block" and
//               "P V of the oldest pending block" is ready first;
//   warps 2-5   softmax, one query row per thread (= its TMEM lane): write Q into TMEM, read each
//               S block, online softmax in the exp2 domain with a lazily moved reference max (O
//               and the row sum are rescaled only when the block max exceeds it by more than 8,
//               so P <= 2^8), write P into TMEM, and finally O / l as the output pair;
//   warps 6-13  converters: K_lo and V_lo from the hi parts and their residual codes, in the hi
//               parts' own swizzled layout; values of keys past the last visible one are zeroed
//               (their P is 0, and a stale NaN would still poison the product).
// TMEM columns: S0 [0,64) S1 [64,128) O [128,128+HD) Q_hi [256,256+HD/2) Q_lo [256+HD/2,256+HD)
// P_hi [384,416) P_lo [416,448).  Every wait is bounded; on a timeout the CTA records
// VLA_STATUS_TIMEOUT, drains its copies and MMAs, frees TMEM and writes nothing.
#include <atomic>

#include "attention.h"
#include "gemm.h"
#include "ptx.cuh"

namespace vla {

namespace {

constexpr int kAtWarps = 14;
constexpr int kAtThreads = 32 * kAtWarps;
constexpr int kConvWarps = kAtWarps - 6;
constexpr int kStages = 3;
constexpr int kKeys = 64;  // keys per block
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0, kColO = 128, kColQ = 256, kColP = 384;

// Shared-memory matrix descriptor, 128-byte swizzle: atoms of 8 rows x 128 bytes, 1024 bytes
// apart along the rows (SBO); for an MN-major operand the 64-element column blocks lie `lbo`
// bytes apart (LBO; unused for K-major).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo = 16) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(lbo >> 4) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;          // descriptor version
  d |= static_cast<uint64_t>(2) << 61;          // 128-byte swizzle
  return d;
}
// kind::f16, fp16 A and B (format fields 0), fp32 D, M = 128, N; A K-major, B K-major or
// MN-major (bit 16).
__device__ __forceinline__ constexpr uint32_t idesc_f16(int N, bool b_mn_major = false) {
  return (1u << 4) | (b_mn_major ? (1u << 16) : 0u) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(128 >> 4) << 24);
}
// D (TMEM) (+)= A (TMEM) * B (shared memory)
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
      "%13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ __half2 u32_h2(uint32_t v) { return *reinterpret_cast<__half2*>(&v); }
__device__ __forceinline__ uint32_t h2_u32(__half2 v) { return *reinterpret_cast<uint32_t*>(&v); }
// (a, b) -> fp16 pairs hi = fp16(x), lo = fp16(x - hi), with packed conversions.
__device__ __forceinline__ void split_h2(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(a, b);
  const float2 f = __half22float2(h);
  hi = h2_u32(h);
  lo = h2_u32(__floats2half2_rn(a - f.x, b - f.y));
}
// Low parts of 8 cached fp16 values (one 16-byte chunk) from their 4-bit codes (4 bytes, element
// 2i in the low nibble of byte i): per element (2c - 15) * 2^(e - 30), e the value's fp16 exponent
// field, in fp16 arithmetic with no conversion instruction.  2c goes into the mantissa of 1024
// (fp16 bits 0x6400 | 2c), so 1024 + 2c - 1039 = 2c - 15 exactly; 2^(e - 30) is the value with
// mantissa and sign cleared (2^(e-15)) times 2^-15.  Exact for e >= 6; below that the term is
// under 2^-21 in magnitude and comes out as zero or a rounded subnormal.
__device__ __forceinline__ uint4 res_lo8(uint4 hi, uint32_t codes) {
  const uint32_t twice_lo = (codes << 1) & 0x1E1E1E1Eu;  // 2c of each byte's low nibble
  const uint32_t twice_hi = (codes >> 3) & 0x1E1E1E1Eu;  // 2c of each byte's high nibble
  auto pair = [&](uint32_t h2, uint32_t sel) {
    const uint32_t w = (__byte_perm(twice_lo, twice_hi, sel) & 0x00FF00FFu) | 0x64006400u;
    const __half2 k = __hsub2(u32_h2(w), u32_h2(0x640F640Fu));                      // 2c - 15
    const __half2 s = __hmul2(u32_h2(h2 & 0x7C007C00u), u32_h2(0x02000200u));       // 2^(e - 30)
    return h2_u32(__hmul2(k, s));
  };
  return make_uint4(pair(hi.x, 0x0400u), pair(hi.y, 0x0501u), pair(hi.z, 0x0602u), pair(hi.w, 0x0703u));
}

struct AtParams {
  const float* q;          // [rows, H*HD] f32, rotated
  bf16* out_hi;            // [rows, H*HD] operand pair (fp16 if fp16 else bf16)
  bf16* out_lo;
  const AttnTile* tiles;   // up to 128 rows each
  const uint8_t* res;      // residual plane of the cache
  int64_t layer_row0;      // first cache row (of HD elements) of this layer
  int64_t env_rows, kv_rows, head_rows;  // row strides: env, K->V, head (= cap)
  int cap, H;
  float scale_log2;
  bool fp16;
  uint32_t* status;
  uint64_t wait_limit;
};

template <int HD>
struct AtSmem {
  static constexpr int K_BYTES = kKeys * HD * 2;        // one 64-key tile of K (or V), fp16
  static constexpr int R_BYTES = kKeys * HD / 2;        // its residual codes
  // a stage: K_hi | V_hi | K_lo | V_lo | K codes | V codes (each tile 1024-byte aligned)
  static constexpr int STAGE = 4 * K_BYTES + 2 * R_BYTES;
  static constexpr int SMEM = 1024 + kStages * STAGE + 256;
  static_assert(STAGE % 1024 == 0, "stage alignment");
};

template <int HD>
__global__ void __launch_bounds__(kAtThreads, 1)
    attn_chunk_tc_kernel(const __grid_constant__ CUtensorMap tmKV, const AtParams p) {
  using Sm = AtSmem<HD>;
  constexpr int KB = HD / 64;  // 64-element column blocks of one K / V row
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * Sm::STAGE);
  // full[3] (loaded) conv[3] (low parts written) stfree[3] (the MMAs are done with the stage)
  // sfull[2] sfree[2] pfull pdone qready drain
  const uint32_t b0 = smem_u32(bars);
  auto BAR = [&](int i) { return b0 + 8u * static_cast<uint32_t>(i); };
  const uint32_t FULL = 0, CONV = 3, STFREE = 6, SFULL = 9, SFREE = 11, PFULL = 13, PDONE = 14, QREADY = 15,
                 DRAIN = 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 17);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();
  const AttnTile tile = p.tiles[blockIdx.x];
  const int head = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_keys = tile.pos0 + tile.nrows;
  const int nb = (n_keys + kKeys - 1) / kKeys;
  const int64_t krow0 = p.layer_row0 + tile.env * p.env_rows + head * p.head_rows;  // K rows of (env, head)
  const int64_t vrow0 = krow0 + p.kv_rows;
  uint32_t* status = p.status;
  const uint64_t limit = p.wait_limit;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(BAR(FULL + s), 1);
      mbar_init(BAR(CONV + s), kConvWarps);
      mbar_init(BAR(STFREE + s), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(BAR(SFULL + s), 1);
      mbar_init(BAR(SFREE + s), 4);
    }
    mbar_init(BAR(PFULL), 4);
    mbar_init(BAR(PDONE), 1);
    mbar_init(BAR(QREADY), 4);
    mbar_init(BAR(DRAIN), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmKV)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  auto stage_ptr = [&](int st) { return smem + st * Sm::STAGE; };

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------------ producer
      pdl_wait();  // the chunk's own keys / values were written by the q|k|v projection
      uint32_t issued = 0, issued_phase = 0;
      for (int b = 0; b < nb; ++b) {
        const int st = b % kStages, round = b / kStages;
        if (round >= 1 && !wait_bounded(BAR(STFREE + st), (round - 1) & 1, abort_flag, status, limit)) break;
        const uint32_t s_khi = smem_u32(stage_ptr(st)), s_vhi = s_khi + Sm::K_BYTES;
        const uint32_t s_kr = s_khi + 4 * Sm::K_BYTES, s_vr = s_kr + Sm::R_BYTES;
        const int key0 = b * kKeys;
        const int rows = min(kKeys, p.cap - key0);  // residual rows inside this (env, head)
        const uint32_t rbytes = static_cast<uint32_t>(rows) * (HD / 2);
        mbar_arrive_expect_tx(BAR(FULL + st), 2u * Sm::K_BYTES + 2u * rbytes);
#pragma unroll
        for (int kb = 0; kb < KB; ++kb) {
          tma_load_2d(s_khi + kb * (kKeys * 128), &tmKV, BAR(FULL + st), kb * 64, static_cast<int>(krow0 + key0));
          tma_load_2d(s_vhi + kb * (kKeys * 128), &tmKV, BAR(FULL + st), kb * 64, static_cast<int>(vrow0 + key0));
        }
        bulk_load(s_kr, p.res + (krow0 + key0) * (HD / 2), rbytes, BAR(FULL + st));
        bulk_load(s_vr, p.res + (vrow0 + key0) * (HD / 2), rbytes, BAR(FULL + st));
        issued |= 1u << st;
        issued_phase = (issued_phase & ~(1u << st)) | (static_cast<uint32_t>(round & 1) << st);
      }
      for (int st = 0; st < kStages; ++st)
        if (issued & (1u << st)) wait_drain(BAR(FULL + st), (issued_phase >> st) & 1u, limit);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------------ MMA issuer
      const uint32_t IS = idesc_f16(kKeys), IO = idesc_f16(HD, true);
      const uint32_t tS0 = tmem + kColS, tO = tmem + kColO;
      const uint32_t tQh = tmem + kColQ, tQl = tmem + kColQ + HD / 2;
      const uint32_t tPh = tmem + kColP, tPl = tmem + kColP + kKeys / 2;
      bool ok = wait_bounded(BAR(QREADY), 0, abort_flag, status, limit);
      int bs = 0, bo = 0;  // next block whose S, whose P V is to be issued
      uint64_t t_last = globaltimer();
      uint32_t spins = 0;
      while (ok && bo < nb) {
        if (bo < bs && mbar_test_wait(BAR(PFULL), bo & 1)) {
          // O += P V of block bo; the commit frees its stage and hands O / P back to the softmax
          tc_fence_after();
          const uint32_t s_vhi = smem_u32(stage_ptr(bo % kStages)) + Sm::K_BYTES;
          const uint32_t s_vlo = s_vhi + 2 * Sm::K_BYTES;
#pragma unroll
          for (int k = 0; k < kKeys / 16; ++k) {
            const uint64_t dh = sdesc_sw128(s_vhi + k * 2048, kKeys * 128);
            const uint64_t dl = sdesc_sw128(s_vlo + k * 2048, kKeys * 128);
            mma_ts(tO, tPh + k * 8, dh, IO, (bo > 0 || k > 0) ? 1u : 0u);
            mma_ts(tO, tPl + k * 8, dh, IO, 1u);
            mma_ts(tO, tPh + k * 8, dl, IO, 1u);
          }
          tc_commit(BAR(PDONE));
          tc_commit(BAR(STFREE + bo % kStages));
          ++bo;
          t_last = globaltimer();
        } else if (bs < nb && mbar_test_wait(BAR(CONV + bs % kStages), (bs / kStages) & 1) &&
                   (bs < 2 || mbar_test_wait(BAR(SFREE + (bs & 1)), ((bs >> 1) - 1) & 1))) {
          // S of block bs into buffer bs & 1
          tc_fence_after();
          const uint32_t s_khi = smem_u32(stage_ptr(bs % kStages)), s_klo = s_khi + 2 * Sm::K_BYTES;
          const uint32_t tS = tS0 + (bs & 1) * kKeys;
#pragma unroll
          for (int k = 0; k < HD / 16; ++k) {
            const uint32_t off = (k >> 2) * (kKeys * 128) + (k & 3) * 32;
            const uint64_t dh = sdesc_sw128(s_khi + off), dl = sdesc_sw128(s_klo + off);
            mma_ts(tS, tQh + k * 8, dh, IS, k > 0 ? 1u : 0u);
            mma_ts(tS, tQl + k * 8, dh, IS, 1u);
            mma_ts(tS, tQh + k * 8, dl, IS, 1u);
          }
          tc_commit(BAR(SFULL + (bs & 1)));
          ++bs;
          t_last = globaltimer();
        } else if (((++spins) & 63u) == 0) {
          if (*abort_flag) {
            ok = false;
          } else if (globaltimer() - t_last > limit) {
            *abort_flag = 1;
            if (status) atomicOr(status, VLA_STATUS_TIMEOUT);
            ok = false;
          }
        }
      }
      tc_commit(BAR(DRAIN));
      wait_drain(BAR(DRAIN), 0, limit);
    }
  } else if (warp < 6) {
    // ------------------------------------------------------------------ softmax (row per thread)
    const int q4 = warp & 3;                 // TMEM lane quarter of this warp
    const int r = q4 * 32 + lane;            // query row in the tile
    const bool valid = r < tile.nrows;
    const int qpos = tile.pos0 + min(r, tile.nrows - 1);
    const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
    const int dcols = p.H * HD;
    pdl_wait();
    // Q row -> fp16 pair in TMEM (A operand of S)
    {
      const float* qrow = p.q + static_cast<size_t>(tile.row0 + (valid ? r : 0)) * dcols + head * HD;
#pragma unroll 1
      for (int c = 0; c < HD; c += 64) {
        float4 x[16];  // 64 values in flight
#pragma unroll
        for (int i = 0; i < 16; ++i)
          x[i] = valid ? __ldg(reinterpret_cast<const float4*>(qrow + c) + i) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float4 v = x[half * 8 + i];
            split_h2(v.x, v.y, hi[2 * i], lo[2 * i]);
            split_h2(v.z, v.w, hi[2 * i + 1], lo[2 * i + 1]);
          }
          tmem_st16(tmem + lane_off + kColQ + (c + 32 * half) / 2, hi);
          tmem_st16(tmem + lane_off + kColQ + HD / 2 + (c + 32 * half) / 2, lo);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(QREADY));
    }
    float m_ref = -INFINITY, l = 0.f;
    bool ok = true;
    for (int b = 0; b < nb && ok; ++b) {
      const int st = b & 1;
      int w_ok = 1;
      if (lane == 0) w_ok = wait_bounded(BAR(SFULL + st), (b >> 1) & 1, abort_flag, status, limit) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w_ok, 0)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[kKeys];
#pragma unroll
      for (int c = 0; c < kKeys; c += 16) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_off + kColS + st * kKeys + c, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) s[c + i] = __uint_as_float(v[i]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(SFREE + st));
      const int key0 = b * kKeys;
      float mb = -INFINITY;
#pragma unroll
      for (int c = 0; c < kKeys; ++c) {
        s[c] = (key0 + c <= qpos) ? s[c] * p.scale_log2 : -INFINITY;
        mb = fmaxf(mb, s[c]);
      }
      // O and P are the MMA's until block b-1's products are done
      if (b >= 1) {
        if (lane == 0) w_ok = wait_bounded(BAR(PDONE), (b - 1) & 1, abort_flag, status, limit) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, w_ok, 0)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      float alpha = 1.f;
      if (mb > m_ref + 8.f) {
        // first block (m_ref = -inf) or a max well above the reference: move it
        alpha = exp2f(m_ref - mb);  // 0 on the first block
        m_ref = mb;
        l *= alpha;
      }
      if (b >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll 1
        for (int c = 0; c < HD; c += 16) {
          uint32_t v[16];
          tmem_ld16(tmem + lane_off + kColO + c, v);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
          tmem_st16(tmem + lane_off + kColO + c, v);
        }
      }
      float ps = 0.f;
#pragma unroll
      for (int c = 0; c < kKeys; c += 32) {
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float p0 = exp2f(s[c + 2 * i] - m_ref), p1 = exp2f(s[c + 2 * i + 1] - m_ref);
          ps += p0 + p1;
          split_h2(p0, p1, hi[i], lo[i]);
        }
        tmem_st16(tmem + lane_off + kColP + c / 2, hi);
        tmem_st16(tmem + lane_off + kColP + kKeys / 2 + c / 2, lo);
      }
      l += ps;
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(PFULL));
    }
    if (ok && nb > 0) {
      int w_ok = 1;
      if (lane == 0) w_ok = wait_bounded(BAR(PDONE), (nb - 1) & 1, abort_flag, status, limit) ? 1 : 0;
      if (__shfl_sync(0xffffffffu, w_ok, 0)) {
        tc_fence_after();
        const float inv = 1.f / l;
        const size_t off = static_cast<size_t>(tile.row0 + (valid ? r : 0)) * dcols + head * HD;
        uint32_t sat = 0;  // convex combinations of the cached values: the fp16 split never saturates
#pragma unroll 1
        for (int c = 0; c < HD; c += 16) {
          uint32_t v[16];
          tmem_ld16(tmem + lane_off + kColO + c, v);
          tmem_wait_ld();
          if (valid) {
            uint32_t h[8], lo[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
              split_pack2(__uint_as_float(v[2 * i]) * inv, __uint_as_float(v[2 * i + 1]) * inv, h[i], lo[i], p.fp16,
                          sat);
            uint4* dh = reinterpret_cast<uint4*>(p.out_hi + off + c);
            uint4* dl = reinterpret_cast<uint4*>(p.out_lo + off + c);
            dh[0] = make_uint4(h[0], h[1], h[2], h[3]);
            dh[1] = make_uint4(h[4], h[5], h[6], h[7]);
            dl[0] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            dl[1] = make_uint4(lo[4], lo[5], lo[6], lo[7]);
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------------ converters (warps 6-13)
    const int t = threadIdx.x - 6 * 32;
    constexpr int CH = HD / 8;  // 16-byte chunks of one row
    for (int b = 0; b < nb; ++b) {
      const int st = b % kStages;
      int w_ok = 1;
      if (lane == 0) w_ok = wait_bounded(BAR(FULL + st), (b / kStages) & 1, abort_flag, status, limit) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w_ok, 0)) break;
      uint8_t* sp = stage_ptr(st);
      const int live = n_keys - b * kKeys;  // keys of this block visible to some row
      // chunk index fastest over lanes: 8 lanes read one swizzled 128-byte row, a warp reads 128
      // consecutive code bytes
#pragma unroll 2
      for (int ch = t; ch < 2 * kKeys * CH; ch += 32 * kConvWarps) {
        const int w = ch / (kKeys * CH);  // 0: K, 1: V
        const int c = ch % CH, key = (ch / CH) % kKeys;
        const int off = (c >> 3) * (kKeys * 128) + key * 128 + (((c & 7) ^ (key & 7)) << 4);
        uint4* hi = reinterpret_cast<uint4*>(sp + w * Sm::K_BYTES + off);
        uint4* lo = reinterpret_cast<uint4*>(sp + (2 + w) * Sm::K_BYTES + off);
        if (w == 1 && key >= live) {
          *hi = make_uint4(0u, 0u, 0u, 0u);
          *lo = make_uint4(0u, 0u, 0u, 0u);
        } else {
          const uint32_t codes =
              *reinterpret_cast<const uint32_t*>(sp + 4 * Sm::K_BYTES + w * Sm::R_BYTES + key * (HD / 2) + c * 4);
          *lo = res_lo8(*hi, codes);
        }
      }
      fence_async_smem();  // the MMAs (async proxy) read what these generic stores wrote
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(CONV + st));
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

}  // namespace

int attn_chunk_tc_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles, int n_tiles,
                         KVLayout kv, int layer, int H, int hd, uint32_t* status, cudaStream_t stream, bool fp16) {
  if (n_tiles <= 0) return VLA_OK;
  if (!kv.res || (hd != 64 && hd != 128)) return VLA_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(kv.base) & 15) || (reinterpret_cast<uintptr_t>(kv.res) & 15))
    return VLA_ERR_ARG;
  AtParams p{};
  p.q = q;
  p.out_hi = out_hi;
  p.out_lo = out_lo;
  p.tiles = tiles;
  p.res = kv.res;
  // the cache as rows of hd elements: [layer][env][K,V][H][cap]
  p.head_rows = kv.cap;
  p.kv_rows = kv.kv_stride / hd;
  p.env_rows = kv.env_stride / hd;
  p.layer_row0 = static_cast<int64_t>(layer) * (kv.layer_stride / hd);
  p.cap = kv.cap;
  p.H = H;
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  p.fp16 = fp16;
  p.status = status;
  p.wait_limit = g_wait_limit_ns.load(std::memory_order_relaxed);
  // tensor map over every row of the cache (rows = layers * layer_stride / hd): row coordinates
  // must fit a signed 32-bit int
  const int64_t total_rows = static_cast<int64_t>(layer + 1) * (kv.layer_stride / hd);
  if (total_rows >= (static_cast<int64_t>(1) << 31)) return VLA_ERR_UNSUPPORTED;
  CUtensorMap map;
  if (!make_tensor_map_2d(&map, kv.base, total_rows, hd, hd, kKeys, true))
    return cuda_fail(cudaErrorInvalidValue, "tensor map (KV cache)");
  dim3 grid(n_tiles, H);
  if (hd == 128) {
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_chunk_tc_kernel<128>, AtSmem<128>::SMEM, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_chunk_tc_kernel<128>, grid, dim3(kAtThreads), AtSmem<128>::SMEM, stream, map, p));
  } else {
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_chunk_tc_kernel<64>, AtSmem<64>::SMEM, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_chunk_tc_kernel<64>, grid, dim3(kAtThreads), AtSmem<64>::SMEM, stream, map, p));
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
