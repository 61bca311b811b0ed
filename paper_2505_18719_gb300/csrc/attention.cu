// Causal attention over the per-environment KV cache (paper §3.1: the policy's Llama-2
// self-attention; §3.3: the whole trajectory is one context, so every chunk attends to all
// earlier turns).
//
//  * attn_chunk: query rows of one env at consecutive positions (a prefill chunk, or the
//    6 teacher-forced action rows of the score pass) against keys 0..pos of that env.
//    One CTA per (64-row tile, head); mma.sync tensor-core flash attention with fp32
//    accumulation on fp16 K/V, the fp32 queries and the softmax weights each taken as an
//    fp16 hi/lo pair; the output is written as the operand hi/lo pair the O-projection GEMM
//    reads (fp16 for the engine, bf16 for the op entry points).
//  * attn_decode: one query per env (the decode step) with the key range split across CTAs
//    (flash-decoding); each CTA writes its partial (max, sum, unnormalised output) and the
//    last CTA of the (env, head) to finish merges the splits in a fixed order.  16 lanes x
//    16 bytes read one 128-element key row, so each warp streams two rows per instruction.
//
// Keys visible to a query at position p are positions 0..p (all of them are in the cache:
// chunk rows write their K/V in the QKV epilogue before attention runs).
#include "attention.h"
#include "ptx.cuh"

namespace vla {

namespace {


// ------------------------------------------------------------------------ chunk (tensor core)
// Flash-attention over one 64-row query tile of one env and one head: S = Q K^T and O += P V
// on mma.sync m16n8k16 (fp16 inputs, fp32 accumulation), online softmax in the exp2 domain.
// 4 warps x 16 query rows; K/V blocks of 64 keys double-buffered in shared memory with
// cp.async (rows past the last visible key are zero-filled, never read from the cache).
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;  // 0 source bytes -> 16 zero bytes
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// (a, b) -> fp16 pairs hi = fp16(x), lo = fp16(x - hi): P V is taken as P_hi V + P_lo V so the
// softmax weights keep ~22 bits.
__device__ __forceinline__ void split_h2(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half ha = __float2half_rn(a), hb = __float2half_rn(b);
  __half2 h2 = __halves2half2(ha, hb);
  __half2 l2 = __floats2half2_rn(a - __half2float(ha), b - __half2float(hb));
  hi = *reinterpret_cast<uint32_t*>(&h2);
  lo = *reinterpret_cast<uint32_t*>(&l2);
}

template <int HD>
__global__ void __launch_bounds__(128) attn_chunk_mma_kernel(const float* q,
                                                             bf16* __restrict__ out_hi,
                                                             bf16* __restrict__ out_lo,
                                                             const AttnTile* __restrict__ tiles,
                                                             KVLayout kv, int layer, int H,
                                                             float scale_log2, bool fp16) {
  constexpr int KB = 64;       // keys per block
  constexpr int LD = HD + 8;   // padded row (halves): 16-byte rows land in distinct banks
  constexpr int CPR = HD / 8;  // 16-byte chunks per row
  constexpr int NT_D = HD / 8; // n-tiles over the head dim
  extern __shared__ __align__(16) f16 sm_h[];
  f16* Ks = sm_h;              // [2][KB][LD]
  f16* Vs = Ks + 2 * KB * LD;  // [2][KB][LD]

  pdl_launch_dependents();
  pdl_wait();
  const AttnTile t = tiles[blockIdx.x];
  const int head = blockIdx.y;
  const int d = H * HD;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tq = lane & 3;
  const f16* kbase = kv.base + static_cast<int64_t>(layer) * kv.layer_stride +
                     static_cast<int64_t>(t.env) * kv.env_stride +
                     static_cast<int64_t>(head) * kv.head_stride;
  const f16* vbase = kbase + kv.kv_stride;
  const int n_keys = t.pos0 + t.nrows;
  const int n_blocks = (n_keys + KB - 1) / KB;

  auto load_block = [&](int blk, int buf) {
    const int j0 = blk * KB;
    const uint32_t ks = static_cast<uint32_t>(__cvta_generic_to_shared(Ks + buf * KB * LD));
    const uint32_t vs = static_cast<uint32_t>(__cvta_generic_to_shared(Vs + buf * KB * LD));
    for (int i = tid; i < KB * CPR; i += 128) {
      const int r = i / CPR, c = (i - r * CPR) * 8;
      const bool ok = j0 + r < n_keys;
      const int64_t src = static_cast<int64_t>(ok ? j0 + r : 0) * HD + c;
      cp_async16(ks + (r * LD + c) * 2, kbase + src, ok);
      cp_async16(vs + (r * LD + c) * 2, vbase + src, ok);
    }
  };

  load_block(0, 0);
  cp_async_commit();

  // this thread's two rows and their positions (rows past nrows reuse the last position;
  // their results are never written)
  const int r0 = warp * 16 + g, r1 = r0 + 8;
  const int qpos0 = t.pos0 + min(r0, t.nrows - 1);
  const int qpos1 = t.pos0 + min(r1, t.nrows - 1);
  const int warp_last = t.pos0 + min(warp * 16 + 15, t.nrows - 1);
  const bool warp_active = warp * 16 < t.nrows;

  float o[NT_D][4];
#pragma unroll
  for (int i = 0; i < NT_D; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  // Q A-fragments straight from the fp32 rows, as fp16 hi/lo pairs (S = Q_hi K + Q_lo K).
  uint32_t qh[HD / 16][4], ql[HD / 16][4];
  {
    const int ra = min(r0, t.nrows - 1), rb = min(r1, t.nrows - 1);
    const float* qa = q + static_cast<size_t>(t.row0 + ra) * d + head * HD + 2 * tq;
    const float* qb = q + static_cast<size_t>(t.row0 + rb) * d + head * HD + 2 * tq;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
      const float2 x0 = *reinterpret_cast<const float2*>(qa + kk * 16);
      const float2 x1 = *reinterpret_cast<const float2*>(qb + kk * 16);
      const float2 x2 = *reinterpret_cast<const float2*>(qa + kk * 16 + 8);
      const float2 x3 = *reinterpret_cast<const float2*>(qb + kk * 16 + 8);
      split_h2(x0.x, x0.y, qh[kk][0], ql[kk][0]);
      split_h2(x1.x, x1.y, qh[kk][1], ql[kk][1]);
      split_h2(x2.x, x2.y, qh[kk][2], ql[kk][2]);
      split_h2(x3.x, x3.y, qh[kk][3], ql[kk][3]);
    }
  }

  for (int blk = 0; blk < n_blocks; ++blk) {
    if (blk + 1 < n_blocks) {
      load_block(blk + 1, (blk + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int j0 = blk * KB;
    if (warp_active && j0 <= warp_last) {
      const int buf = blk & 1;
      const uint32_t ks = static_cast<uint32_t>(__cvta_generic_to_shared(Ks + buf * KB * LD));
      const uint32_t vs = static_cast<uint32_t>(__cvta_generic_to_shared(Vs + buf * KB * LD));
      float s[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
        const int i = lane >> 3;
#pragma unroll
        for (int kk = 0; kk < HD / 16; kk += 2) {
          uint32_t b0, b1, b2, b3;
          const int key = nt * 8 + (lane & 7);
          const int dim = (kk + (i >> 1)) * 16 + (i & 1) * 8;
          ldsm_x4(ks + (key * LD + dim) * 2, b0, b1, b2, b3);
          mma16816(s[nt], qh[kk], b0, b1);
          mma16816(s[nt], ql[kk], b0, b1);
          mma16816(s[nt], qh[kk + 1], b2, b3);
          mma16816(s[nt], ql[kk + 1], b2, b3);
        }
      }
      // scale, causal mask, online softmax (rows r0: c 0,1; r1: c 2,3)
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int key = j0 + nt * 8 + 2 * tq + (c & 1);
          const int qp = (c < 2) ? qpos0 : qpos1;
          const float v = (key <= qp) ? s[nt][c] * scale_log2 : -INFINITY;
          s[nt][c] = v;
        }
        mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
        mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);  // finite: key j0 <= qpos
      const float a0 = exp2f(m0 - mn0), a1 = exp2f(m1 - mn1);
      m0 = mn0;
      m1 = mn1;
      float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        s[nt][0] = exp2f(s[nt][0] - mn0);
        s[nt][1] = exp2f(s[nt][1] - mn0);
        s[nt][2] = exp2f(s[nt][2] - mn1);
        s[nt][3] = exp2f(s[nt][3] - mn1);
        ps0 += s[nt][0] + s[nt][1];
        ps1 += s[nt][2] + s[nt][3];
      }
      l0 = l0 * a0 + ps0;  // per-thread partial row sums; reduced across the quad at the end
      l1 = l1 * a1 + ps1;
#pragma unroll
      for (int nt = 0; nt < NT_D; ++nt) {
        o[nt][0] *= a0;
        o[nt][1] *= a0;
        o[nt][2] *= a1;
        o[nt][3] *= a1;
      }
      // O += P V: P re-used from the S accumulators as the A operand, as an fp16 hi/lo pair
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t ph[4], pl[4];
        split_h2(s[2 * kk][0], s[2 * kk][1], ph[0], pl[0]);
        split_h2(s[2 * kk][2], s[2 * kk][3], ph[1], pl[1]);
        split_h2(s[2 * kk + 1][0], s[2 * kk + 1][1], ph[2], pl[2]);
        split_h2(s[2 * kk + 1][2], s[2 * kk + 1][3], ph[3], pl[3]);
        const int i = lane >> 3;
#pragma unroll
        for (int nt = 0; nt < NT_D; nt += 2) {
          uint32_t b0, b1, b2, b3;
          const int key = kk * 16 + (i & 1) * 8 + (lane & 7);
          const int dim = (nt + (i >> 1)) * 8;
          ldsm_x4_t(vs + (key * LD + dim) * 2, b0, b1, b2, b3);
          mma16816(o[nt], ph, b0, b1);
          mma16816(o[nt], pl, b0, b1);
          mma16816(o[nt + 1], ph, b2, b3);
          mma16816(o[nt + 1], pl, b2, b3);
        }
      }
    }
    __syncthreads();  // this buffer is refilled two blocks later
  }
  if (!warp_active) return;
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = 1.f / l0, inv1 = 1.f / l1;
  // outputs are convex combinations of fp16 values, so the fp16 split never saturates here
  uint32_t sat = 0;
#pragma unroll
  for (int nt = 0; nt < NT_D; ++nt) {
    const int col = head * HD + nt * 8 + 2 * tq;
    if (r0 < t.nrows) {
      const size_t off = static_cast<size_t>(t.row0 + r0) * d + col;
      uint32_t hi, lo;
      split_pack2(o[nt][0] * inv0, o[nt][1] * inv0, hi, lo, fp16, sat);
      *reinterpret_cast<uint32_t*>(out_hi + off) = hi;
      *reinterpret_cast<uint32_t*>(out_lo + off) = lo;
    }
    if (r1 < t.nrows) {
      const size_t off = static_cast<size_t>(t.row0 + r1) * d + col;
      uint32_t hi, lo;
      split_pack2(o[nt][2] * inv1, o[nt][3] * inv1, hi, lo, fp16, sat);
      *reinterpret_cast<uint32_t*>(out_hi + off) = hi;
      *reinterpret_cast<uint32_t*>(out_lo + off) = lo;
    }
  }
}

// ------------------------------------------------------------------ few-row chunk (residual cache)
// Query tiles of at most 16 rows (the teacher-forced action rows of the score pass, Eq. 2, or any
// chunk that short) against keys 0..pos of their env, the cache read as fp16 + 4-bit residual
// (hi + lo, KVLayout).  One CTA per (tile, head), 4 warps, 128 registers and one 45 KB stage so
// that four CTAs share an SM (the other CTAs' blocks are in flight while one computes): key
// blocks of 64 staged in shared memory by cp.async (fp16 parts and residual codes; keys past the
// tile's last position are zero-filled, never read), the tile's query rows as an fp16 pair in
// shared memory (ldmatrix A fragments); warp w takes keys 16w .. 16w+15 of every block with one
// m16n8k16 row tile (rows past the tile's last repeat its last row and are not written), the low
// parts decoded from the codes beside each B fragment:
//   S = Q_hi K_hi + Q_lo K_hi + Q_hi K_lo,   O += P_hi V_hi + P_lo V_hi + P_hi V_lo,
// online softmax per warp in the exp2 domain (Q pre-scaled by log2(e) / sqrt(hd)); the four warps'
// (max, sum, O) merge through shared memory at the end.  Each cached byte is read once per (tile,
// head), against a 128-row tensor-core tile that would spend 7/8 of its MMAs on padding rows.
template <int HD>
struct RowsSmem {
  static constexpr int KB = 64;                 // keys per staged block
  static constexpr int LD = HD + 8;             // padded fp16 row (halves): ldmatrix rows in distinct banks
  static constexpr int RB = HD / 2;             // residual bytes of one row
  static constexpr int RBP = RB + 16;           // padded code row: the fragment reads hit distinct banks
  static constexpr int PLANE = KB * LD * 2;     // bytes of one staged fp16 block
  static constexpr int CODES = KB * RBP;        // bytes of one staged code block
  static constexpr int STAGE = 2 * PLANE + 2 * CODES;  // K | V | K codes | V codes
  static constexpr int QPLANE = 16 * LD * 2;            // the tile's 16 query rows, fp16 (hi or lo)
  static constexpr int SMEM = STAGE + 2 * QPLANE;       // one stage: four CTAs share an SM
  static_assert(STAGE % 16 == 0 && 4 * 16 * HD * 4 + 4 * 16 * 2 * 4 <= STAGE, "staging / merge layout");
};

template <int HD>
__global__ void __launch_bounds__(128, 4) attn_rows_kernel(const float* q, bf16* out_hi, bf16* out_lo,
                                                           const AttnTile* tiles, KVLayout kv, int layer, int H,
                                                           float scale_log2, bool fp16, bool write_lo) {
  using Sm = RowsSmem<HD>;
  constexpr int KB = Sm::KB, LD = Sm::LD, RB = Sm::RB, RBP = Sm::RBP, PLANE = Sm::PLANE;
  constexpr int CPR = HD / 8;   // 16-byte chunks of an fp16 row
  constexpr int NT_D = HD / 8;  // n-tiles over the head dim
  constexpr int RWP = RBP / 4;  // 32-bit words of a padded code row
  extern __shared__ __align__(16) uint8_t sm_rows[];
  uint8_t* qs = sm_rows + Sm::STAGE;  // Q_hi [16][LD], then Q_lo [16][LD]

  pdl_launch_dependents();
  pdl_wait();
  const AttnTile t = tiles[blockIdx.x];
  const int head = blockIdx.y;
  const int d = H * HD;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tq = lane & 3;
  const int64_t e0 = static_cast<int64_t>(layer) * kv.layer_stride + static_cast<int64_t>(t.env) * kv.env_stride +
                     static_cast<int64_t>(head) * kv.head_stride;
  const f16* kbase = kv.base + e0;
  const f16* vbase = kbase + kv.kv_stride;
  const uint8_t* kres = kv.res + e0 / 2;
  const uint8_t* vres = kres + kv.kv_stride / 2;
  const int n_keys = t.pos0 + t.nrows;
  const int n_blocks = (n_keys + KB - 1) / KB;
  const int last_pos = n_keys - 1;

  auto load_block = [&](int blk) {
    const int j0 = blk * KB;
    const uint32_t s0 = smem_u32(sm_rows);
    for (int i = tid; i < KB * CPR; i += 128) {
      const int r = i / CPR, c = i - r * CPR;
      const bool ok = j0 + r < n_keys;
      const int64_t src = static_cast<int64_t>(ok ? j0 + r : 0) * HD + c * 8;
      cp_async16(s0 + (r * LD + c * 8) * 2, kbase + src, ok);
      cp_async16(s0 + PLANE + (r * LD + c * 8) * 2, vbase + src, ok);
    }
    for (int i = tid; i < KB * (RB / 16); i += 128) {
      const int r = i / (RB / 16), c = i - r * (RB / 16);
      const bool ok = j0 + r < n_keys;
      const int64_t src = static_cast<int64_t>(ok ? j0 + r : 0) * RB + c * 16;
      cp_async16(s0 + 2 * PLANE + r * RBP + c * 16, kres + src, ok);
      cp_async16(s0 + 2 * PLANE + Sm::CODES + r * RBP + c * 16, vres + src, ok);
    }
  };
  load_block(0);
  cp_async_commit();

  // the tile's 16 query rows (rows past the last repeat it) times log2(e) / sqrt(hd), as fp16
  // hi / lo planes: 8 threads per row, HD / 8 values each
  {
    constexpr int QPT = HD / 8;
    const int row = tid >> 3, c0 = (tid & 7) * QPT;
    const float* qr = q + static_cast<size_t>(t.row0 + min(row, t.nrows - 1)) * d + head * HD + c0;
    float4 x[QPT / 4];
#pragma unroll
    for (int i = 0; i < QPT / 4; ++i) x[i] = __ldcg(reinterpret_cast<const float4*>(qr) + i);
    uint32_t hi[QPT / 2], lo[QPT / 2];
#pragma unroll
    for (int i = 0; i < QPT / 4; ++i) {
      split_h2(x[i].x * scale_log2, x[i].y * scale_log2, hi[2 * i], lo[2 * i]);
      split_h2(x[i].z * scale_log2, x[i].w * scale_log2, hi[2 * i + 1], lo[2 * i + 1]);
    }
#pragma unroll
    for (int i = 0; i < QPT / 8; ++i) {
      reinterpret_cast<uint4*>(qs + (row * LD + c0) * 2)[i] = make_uint4(hi[4 * i], hi[4 * i + 1], hi[4 * i + 2], hi[4 * i + 3]);
      reinterpret_cast<uint4*>(qs + Sm::QPLANE + (row * LD + c0) * 2)[i] =
          make_uint4(lo[4 * i], lo[4 * i + 1], lo[4 * i + 2], lo[4 * i + 3]);
    }
  }
  // this thread's two rows (g and g + 8 of the tile) and their positions
  const int qpos0 = t.pos0 + min(g, t.nrows - 1), qpos1 = t.pos0 + min(g + 8, t.nrows - 1);
  const uint32_t qh_s = smem_u32(qs), ql_s = qh_s + Sm::QPLANE;
  // A-fragment address of this lane: row lane % 16, columns + 8 for lanes 16..31
  const uint32_t qa_off = ((lane & 15) * LD + (lane >> 4) * 8) * 2;

  float o[NT_D][4];
#pragma unroll
  for (int i = 0; i < NT_D; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const int im = lane >> 3;  // the ldmatrix sub-matrix this lane addresses

  for (int blk = 0; blk < n_blocks; ++blk) {
    cp_async_wait<0>();
    __syncthreads();
    const int k0 = blk * KB + warp * 16;  // this warp's first key
    if (k0 <= last_pos) {
      const uint32_t ks = smem_u32(sm_rows), vs = ks + PLANE;
      const uint32_t* kc = reinterpret_cast<const uint32_t*>(sm_rows + 2 * PLANE);
      const uint32_t* vc = reinterpret_cast<const uint32_t*>(sm_rows + 2 * PLANE + Sm::CODES);
      float s[2][4];
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; kk += 2) {
        uint32_t qh0[4], ql0[4], qh1[4], ql1[4];
        ldsm_x4(qh_s + qa_off + kk * 32, qh0[0], qh0[1], qh0[2], qh0[3]);
        ldsm_x4(ql_s + qa_off + kk * 32, ql0[0], ql0[1], ql0[2], ql0[3]);
        ldsm_x4(qh_s + qa_off + kk * 32 + 32, qh1[0], qh1[1], qh1[2], qh1[3]);
        ldsm_x4(ql_s + qa_off + kk * 32 + 32, ql1[0], ql1[1], ql1[2], ql1[3]);
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
          // this thread's B elements are in key row warp*16 + nt*8 + g; the codes of dims
          // 16kk + 2tq (+1) sit in byte tq of the row's word 2kk (+1 for dims + 8)
          uint32_t b0, b1, b2, b3;
          const int key = warp * 16 + nt * 8 + (lane & 7);
          const int dim = (kk + (im >> 1)) * 16 + (im & 1) * 8;
          ldsm_x4(ks + (key * LD + dim) * 2, b0, b1, b2, b3);
          const uint4 cw = *reinterpret_cast<const uint4*>(kc + (warp * 16 + nt * 8 + g) * RWP + 2 * kk);
          const int sh = 8 * tq;
          const uint32_t l0b = kv_res_lo2(b0, (cw.x >> sh) & 15u, (cw.x >> (sh + 4)) & 15u);
          const uint32_t l1b = kv_res_lo2(b1, (cw.y >> sh) & 15u, (cw.y >> (sh + 4)) & 15u);
          const uint32_t l2b = kv_res_lo2(b2, (cw.z >> sh) & 15u, (cw.z >> (sh + 4)) & 15u);
          const uint32_t l3b = kv_res_lo2(b3, (cw.w >> sh) & 15u, (cw.w >> (sh + 4)) & 15u);
          mma16816(s[nt], qh0, b0, b1);
          mma16816(s[nt], ql0, b0, b1);
          mma16816(s[nt], qh0, l0b, l1b);
          mma16816(s[nt], qh1, b2, b3);
          mma16816(s[nt], ql1, b2, b3);
          mma16816(s[nt], qh1, l2b, l3b);
        }
      }
      // causal mask, online softmax (row g: c 0, 1; row g + 8: c 2, 3)
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int kpos = k0 + nt * 8 + 2 * tq + (c & 1);
          if (kpos > ((c < 2) ? qpos0 : qpos1)) s[nt][c] = -INFINITY;
        }
        mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
        mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      // a row with no visible key yet (in this warp's share) keeps max -inf: reference 0, weights 0
      const float u0 = mn0 == -INFINITY ? 0.f : mn0, u1 = mn1 == -INFINITY ? 0.f : mn1;
      const float a0 = exp2f(m0 - u0), a1 = exp2f(m1 - u1);
      m0 = mn0;
      m1 = mn1;
      float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        s[nt][0] = exp2f(s[nt][0] - u0);
        s[nt][1] = exp2f(s[nt][1] - u0);
        s[nt][2] = exp2f(s[nt][2] - u1);
        s[nt][3] = exp2f(s[nt][3] - u1);
        ps0 += s[nt][0] + s[nt][1];
        ps1 += s[nt][2] + s[nt][3];
      }
      l0 = l0 * a0 + ps0;  // per-thread partial row sums, reduced across the quad at the end
      l1 = l1 * a1 + ps1;
#pragma unroll
      for (int nt = 0; nt < NT_D; ++nt) {
        o[nt][0] *= a0;
        o[nt][1] *= a0;
        o[nt][2] *= a1;
        o[nt][3] *= a1;
      }
      // O += P V: P from the S accumulators as the A operand (keys 0..7 of the warp's 16 in s[0],
      // 8..15 in s[1]), an fp16 hi / lo pair
      uint32_t ph[4], pl[4];
      split_h2(s[0][0], s[0][1], ph[0], pl[0]);
      split_h2(s[0][2], s[0][3], ph[1], pl[1]);
      split_h2(s[1][0], s[1][1], ph[2], pl[2]);
      split_h2(s[1][2], s[1][3], ph[3], pl[3]);
      // V^T fragments: this thread holds keys 2tq, 2tq + 1 (b0, b2) and 8 + 2tq, 9 + 2tq (b1, b3) of
      // the warp's 16 at dim 8n + g; that element's code is nibble g of the key row's word n
      const uint32_t* vrow = vc + (warp * 16 + 2 * tq) * RWP;
      const int key = warp * 16 + (im & 1) * 8 + (lane & 7);
      const int sh = 4 * g;
#pragma unroll
      for (int nt = 0; nt < NT_D; nt += 2) {
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vs + (key * LD + (nt + (im >> 1)) * 8) * 2, b0, b1, b2, b3);
        const uint2 c00 = *reinterpret_cast<const uint2*>(vrow + nt);            // key 2tq
        const uint2 c01 = *reinterpret_cast<const uint2*>(vrow + RWP + nt);      // key 2tq + 1
        const uint2 c10 = *reinterpret_cast<const uint2*>(vrow + 8 * RWP + nt);  // key 8 + 2tq
        const uint2 c11 = *reinterpret_cast<const uint2*>(vrow + 9 * RWP + nt);  // key 9 + 2tq
        const uint32_t l0b = kv_res_lo2(b0, (c00.x >> sh) & 15u, (c01.x >> sh) & 15u);
        const uint32_t l1b = kv_res_lo2(b1, (c10.x >> sh) & 15u, (c11.x >> sh) & 15u);
        const uint32_t l2b = kv_res_lo2(b2, (c00.y >> sh) & 15u, (c01.y >> sh) & 15u);
        const uint32_t l3b = kv_res_lo2(b3, (c10.y >> sh) & 15u, (c11.y >> sh) & 15u);
        mma16816(o[nt], ph, b0, b1);
        mma16816(o[nt], pl, b0, b1);
        mma16816(o[nt], ph, l0b, l1b);
        mma16816(o[nt + 1], ph, b2, b3);
        mma16816(o[nt + 1], pl, b2, b3);
        mma16816(o[nt + 1], ph, l2b, l3b);
      }
    }
    __syncthreads();  // every warp is done with the stage: the next block's copies may land
    if (blk + 1 < n_blocks) {
      load_block(blk + 1);
      cp_async_commit();
    }
  }

  // merge the four warps' partials: O [warp][16][HD] and (max, sum) [warp][16] over the stages
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  float* mo = reinterpret_cast<float*>(sm_rows);
  float* mml = mo + 4 * 16 * HD;
  {
    float* oa = mo + (warp * 16 + g) * HD + 2 * tq;
    float* ob = oa + 8 * HD;
#pragma unroll
    for (int nt = 0; nt < NT_D; ++nt) {
      *reinterpret_cast<float2*>(oa + nt * 8) = make_float2(o[nt][0], o[nt][1]);
      *reinterpret_cast<float2*>(ob + nt * 8) = make_float2(o[nt][2], o[nt][3]);
    }
    if (tq == 0) {
      *reinterpret_cast<float2*>(mml + (warp * 16 + g) * 2) = make_float2(m0, l0);
      *reinterpret_cast<float2*>(mml + (warp * 16 + g + 8) * 2) = make_float2(m1, l1);
    }
  }
  __syncthreads();
  constexpr int CPT = HD / 8;  // output columns per thread: 8 threads per row
  const int row = tid >> 3, c0 = (tid & 7) * CPT;
  if (row >= t.nrows) return;
  float mw[4], lw[4], mx = -INFINITY;
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const float2 ml = *reinterpret_cast<const float2*>(mml + (w * 16 + row) * 2);
    mw[w] = ml.x;
    lw[w] = ml.y;
    mx = fmaxf(mx, ml.x);  // finite: warp 0 holds key 0, visible to every row
  }
  float wt[4], lsum = 0.f;
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    wt[w] = exp2f(mw[w] - mx);  // 0 for a warp that saw no visible key of this row
    lsum += wt[w] * lw[w];
  }
  const float inv = 1.f / lsum;
  uint32_t sat = 0;  // convex combinations of cached values: the fp16 split never saturates
  uint32_t hi[CPT / 2], lo[CPT / 2];
#pragma unroll
  for (int c = 0; c < CPT; c += 2) {
    float v0 = 0.f, v1 = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float2 x = *reinterpret_cast<const float2*>(mo + (w * 16 + row) * HD + c0 + c);
      v0 += wt[w] * x.x;
      v1 += wt[w] * x.y;
    }
    split_pack2(v0 * inv, v1 * inv, hi[c / 2], lo[c / 2], fp16, sat);
  }
  const size_t off = static_cast<size_t>(t.row0 + row) * d + head * HD + c0;
#pragma unroll
  for (int i = 0; i < CPT / 8; ++i) {
    reinterpret_cast<uint4*>(out_hi + off)[i] = make_uint4(hi[4 * i], hi[4 * i + 1], hi[4 * i + 2], hi[4 * i + 3]);
    if (write_lo)
      reinterpret_cast<uint4*>(out_lo + off)[i] = make_uint4(lo[4 * i], lo[4 * i + 1], lo[4 * i + 2], lo[4 * i + 3]);
  }
}

// ---------------------------------------------------------------------------------- decode
// One query per (env, head, key range): 16 lanes x 16 bytes read one 128-element fp16 key row
// (with RES, also its 4-bit residual codes, 4 bytes per lane, and use hi + lo as the cached value),
// each lane group loads 4 key rows (K and V) before using any (memory-level parallelism), the
// dot products reduce with xor shuffles inside the group, online softmax per lane group; the
// groups of the CTA merge through shared memory into one partial (max, sum, unnormalised
// output) per range.  The last CTA of an (env, head) to finish (a ticket on counters[b * H +
// head], no waiting) merges the S partials in range order and writes the normalised output as
// the operand pair; with S == 1 the CTA writes it directly.
// NW = 2 warps per CTA; ptxas allocates 64 registers for both head dims with no spill, so 16
// CTAs fit on an SM and the 2048 (env, head) CTAs of a 64-env, 32-head step are all resident
// at once (one wave, no tail).  No minimum-blocks bound is given: capping at 64 forces a small
// spill in the 64-dim variant.
constexpr int kDecodeWarps = 2;
template <int HD, bool RES, int NW = kDecodeWarps>
__global__ void __launch_bounds__(NW * 32, RES ? 14 : 1) attn_decode_kernel(const float* q, const RowInfo* rows,
                                                          KVLayout kv, int layer, int H,
                                                          int chunk, int S, float scale_log2,
                                                          float* __restrict__ part_o,
                                                          float2* __restrict__ part_ml,
                                                          int* __restrict__ counters,
                                                          bf16* __restrict__ out_hi,
                                                          bf16* __restrict__ out_lo, bool fp16) {
  constexpr int LPK = HD / 8;     // lanes per key row (8 fp16 = 16 bytes per lane)
  constexpr int KPI = 32 / LPK;   // key rows per warp instruction
  constexpr int U = 4;            // key rows per lane group loaded ahead
  constexpr int NT = NW * 32;      // threads
  __shared__ float s_m[NW][KPI], s_l[NW][KPI];
  __shared__ float s_o[NW][KPI][HD];

  pdl_launch_dependents();
  pdl_wait();
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane / LPK, part = lane - sub * LPK;
  // the queries and row table come from the kernels just before (programmatic dependent
  // launch): read them at L2, never through the non-coherent read-only path
  RowInfo ri;
  ri.env = __ldcg(&rows[b].env);
  ri.pos = __ldcg(&rows[b].pos);
  const int d = H * HD;
  const int k_begin = split * chunk;
  const int k_end = min(k_begin + chunk, ri.pos + 1);

  float qv[8];
  {
    const float4* qp = reinterpret_cast<const float4*>(q + static_cast<size_t>(b) * d + head * HD + part * 8);
    const float4 q0 = __ldcg(qp), q1 = __ldcg(qp + 1);
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
  // RES: the residual codes of the same elements (half a byte each), read with the fp16 parts
  const uint8_t* kres = RES ? kv.res + (kbase - kv.base) / 2 : nullptr;
  const uint8_t* vres = RES ? kres + kv.kv_stride / 2 : nullptr;

  float m = -INFINITY, l = 0.f, o[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) o[e] = 0.f;

  for (int key0 = k_begin + warp * KPI * U; key0 < k_end; key0 += NW * KPI * U) {
    uint4 kk[U], vv[U];
    uint32_t kc[U], vc[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int key = key0 + u * KPI + sub;
      kk[u] = make_uint4(0, 0, 0, 0);
      vv[u] = make_uint4(0, 0, 0, 0);
      kc[u] = vc[u] = 0u;  // fp16 parts of 0: low parts 0 whatever the codes
      if (key < k_end) {
        kk[u] = *reinterpret_cast<const uint4*>(kbase + static_cast<int64_t>(key) * HD + part * 8);
        vv[u] = *reinterpret_cast<const uint4*>(vbase + static_cast<int64_t>(key) * HD + part * 8);
        if (RES) {
          kc[u] = *reinterpret_cast<const uint32_t*>(kres + static_cast<int64_t>(key) * (HD / 2) + part * 4);
          vc[u] = *reinterpret_cast<const uint32_t*>(vres + static_cast<int64_t>(key) * (HD / 2) + part * 4);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const bool valid = key0 + u * KPI + sub < k_end;
      const uint32_t w[4] = {kk[u].x, kk[u].y, kk[u].z, kk[u].w};
      float acc = 0.f;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_f16x2(w[e]);
        acc = fmaf(qv[2 * e], f.x, acc);
        acc = fmaf(qv[2 * e + 1], f.y, acc);
      }
      if (RES) {
        const uint4 kl = kv_res_lo8(kk[u], kc[u]);
        const uint32_t wl[4] = {kl.x, kl.y, kl.z, kl.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_f16x2(wl[e]);
          acc = fmaf(qv[2 * e], f.x, acc);
          acc = fmaf(qv[2 * e + 1], f.y, acc);
        }
      }
      // reduce across the LPK lanes of this key row (a row's lanes share `valid`; the xor
      // offsets stay inside the group)
#pragma unroll
      for (int off = LPK / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
      if (valid) {
        const float m_new = fmaxf(m, acc);
        const float alpha = exp2f(m - m_new);
        const float p = exp2f(acc - m_new);
        l = l * alpha + p;
        const uint32_t v4[4] = {vv[u].x, vv[u].y, vv[u].z, vv[u].w};
        uint32_t vl4[4] = {0u, 0u, 0u, 0u};
        if (RES) {
          const uint4 vl = kv_res_lo8(vv[u], vc[u]);
          vl4[0] = vl.x;
          vl4[1] = vl.y;
          vl4[2] = vl.z;
          vl4[3] = vl.w;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = unpack_f16x2(v4[e]);
          const float2 fl = unpack_f16x2(vl4[e]);
          o[2 * e] = fmaf(p, f.x + fl.x, o[2 * e] * alpha);
          o[2 * e + 1] = fmaf(p, f.y + fl.y, o[2 * e + 1] * alpha);
        }
        m = m_new;
      }
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
  for (int w = 0; w < NW; ++w)
    for (int k = 0; k < KPI; ++k) M = fmaxf(M, s_m[w][k]);
  float L = 0.f;
  for (int w = 0; w < NW; ++w)
    for (int k = 0; k < KPI; ++k)
      if (s_m[w][k] != -INFINITY) L += s_l[w][k] * exp2f(s_m[w][k] - M);
  const size_t bh = static_cast<size_t>(b) * H + head;
  const size_t out_off = static_cast<size_t>(b) * d + head * HD;
  uint32_t sat = 0;  // convex combinations of fp16 values: the fp16 split never saturates
  if (S == 1) {
    for (int c = threadIdx.x; c < HD; c += blockDim.x) {
      float acc = 0.f;
      for (int w = 0; w < NW; ++w)
        for (int k = 0; k < KPI; ++k)
          if (s_m[w][k] != -INFINITY) acc += s_o[w][k][c] * exp2f(s_m[w][k] - M);
      store_split1(out_hi, out_lo, out_off + c, acc / L, fp16, sat);
    }
    return;
  }
  const size_t slot = bh * S + split;
  for (int c = threadIdx.x; c < HD; c += blockDim.x) {
    float acc = 0.f;
    for (int w = 0; w < NW; ++w)
      for (int k = 0; k < KPI; ++k)
        if (s_m[w][k] != -INFINITY) acc += s_o[w][k][c] * exp2f(s_m[w][k] - M);
    part_o[slot * HD + c] = acc;
  }
  if (threadIdx.x == 0) part_ml[slot] = make_float2(M, L);

  // ticket: the partial is published (fence) before the counter moves
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(counters + bh, 1) == S - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  float Mx = -INFINITY;
  for (int s = 0; s < S; ++s) Mx = fmaxf(Mx, __ldcg(&part_ml[bh * S + s].x));
  float Lt = 0.f;
  float acc[(HD + NT - 1) / NT];
#pragma unroll
  for (int i = 0; i < (HD + NT - 1) / NT; ++i) acc[i] = 0.f;
  for (int s = 0; s < S; ++s) {
    const float2 ml = __ldcg(&part_ml[bh * S + s]);
    if (ml.x == -INFINITY) continue;
    const float w = exp2f(ml.x - Mx);
    Lt += ml.y * w;
#pragma unroll
    for (int i = 0; i < (HD + NT - 1) / NT; ++i) {
      const int c = threadIdx.x + i * NT;
      if (c < HD) acc[i] += __ldcg(&part_o[(bh * S + s) * HD + c]) * w;
    }
  }
#pragma unroll
  for (int i = 0; i < (HD + NT - 1) / NT; ++i) {
    const int c = threadIdx.x + i * NT;
    if (c < HD) {
      store_split1(out_hi, out_lo, out_off + c, acc[i] / Lt, fp16, sat);
    }
  }
  if (threadIdx.x == 0) counters[bh] = 0;  // ready for the next launch
}

}  // namespace

int attn_chunk_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles,
                      int n_tiles, KVLayout kv, int layer, int H, int hd, cudaStream_t stream, bool fp16) {
  if (n_tiles <= 0) return VLA_OK;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  dim3 grid(n_tiles, H);
  if (hd == 128) {
    const int smem = (4 * 64) * (128 + 8) * 2;
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_chunk_mma_kernel<128>, smem, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_chunk_mma_kernel<128>, grid, dim3(128), smem, stream, q, out_hi, out_lo,
                            tiles, kv, layer, H, scale_log2, fp16));
  } else if (hd == 64) {
    const int smem = (4 * 64) * (64 + 8) * 2;
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_chunk_mma_kernel<64>, smem, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_chunk_mma_kernel<64>, grid, dim3(128), smem, stream, q, out_hi, out_lo,
                            tiles, kv, layer, H, scale_log2, fp16));
  } else {
    return VLA_ERR_UNSUPPORTED;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int attn_rows_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles, int n_tiles, KVLayout kv,
                     int layer, int H, int hd, cudaStream_t stream, bool fp16, bool write_lo) {
  if (n_tiles <= 0) return VLA_OK;
  if (!kv.res || (hd != 64 && hd != 128)) return VLA_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(kv.base) & 15) || (reinterpret_cast<uintptr_t>(kv.res) & 15)) return VLA_ERR_ARG;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  const dim3 grid(n_tiles, H);
  if (hd == 128) {
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_rows_kernel<128>, RowsSmem<128>::SMEM, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_rows_kernel<128>, grid, dim3(128), RowsSmem<128>::SMEM, stream, q, out_hi, out_lo,
                            tiles, kv, layer, H, scale_log2, fp16, write_lo));
  } else {
    static std::atomic<uint64_t> attr_done{0};
    VLA_CUDA_TRY(set_smem_limit(attn_rows_kernel<64>, RowsSmem<64>::SMEM, attr_done));
    VLA_CUDA_TRY(launch_pdl(attn_rows_kernel<64>, grid, dim3(128), RowsSmem<64>::SMEM, stream, q, out_hi, out_lo,
                            tiles, kv, layer, H, scale_log2, fp16, write_lo));
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

int attn_decode_launch(const float* q, bf16* out_hi, bf16* out_lo, const RowInfo* rows, int B,
                       int max_ctx, KVLayout kv, int layer, int H, int hd, int chunk,
                       float* part_o, float2* part_ml, int* counters, cudaStream_t stream, bool fp16) {
  if (B <= 0) return VLA_OK;
  // equal key ranges (multiples of 16) no longer than `chunk`
  const int S = (max_ctx + chunk - 1) / chunk;
  const int c = ((max_ctx + S - 1) / S + 15) / 16 * 16;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  dim3 grid(S, H, B);
  auto go = [&](auto kern) {
    return launch_pdl(kern, grid, dim3(kDecodeWarps * 32), 0, stream, q, rows, kv, layer, H, c, S, scale_log2, part_o,
                      part_ml, counters, out_hi, out_lo, fp16);
  };
  const bool res = kv.res != nullptr;
  if (hd == 128) {
    VLA_CUDA_TRY(res ? go(attn_decode_kernel<128, true>) : go(attn_decode_kernel<128, false>));
  } else if (hd == 64) {
    VLA_CUDA_TRY(res ? go(attn_decode_kernel<64, true>) : go(attn_decode_kernel<64, false>));
  } else {
    return VLA_ERR_UNSUPPORTED;
  }
  note_launch();
  VLA_CUDA_TRY(cudaGetLastError());
  return VLA_OK;
}

}  // namespace vla
