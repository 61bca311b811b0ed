// Chunk causal attention on the tcgen05 tensor cores (paper §3.1: the policy's Llama-2
// self-attention; §3.3: every chunk of a multi-turn trajectory attends to the whole context):
// query tiles of up to 128 rows of one env (a prefill chunk, or the teacher-forced action rows
// of the PPO ratio pass, Eq. 2) against keys 0..pos of that env.  Persistent: one CTA per SM
// takes the (tile, head) items blockIdx.x, blockIdx.x + gridDim.x, ..., and every pipeline
// (copies, conversions, MMAs, softmax, output) runs on across item boundaries.
//
// Precision: the cached keys / values are fp16 plus a 4-bit residual (KVLayout), read here as
// the pair hi + lo; the queries (fp32) and the softmax weights are split into fp16 pairs too, and
// each product takes three MMAs into one fp32 accumulator:
//   S = Q_hi K_hi^T + Q_lo K_hi^T + Q_hi K_lo^T,    O += P_hi V_hi + P_lo V_hi + P_hi V_lo.
//
// Roles (448 threads):
//   warp 0       TMA producer: per 64-key block, K_hi and V_hi (tensor map over the whole cache,
//                128-byte swizzle) and their residual byte ranges (bulk copies), into two rings of
//                three slots: a K slot is free again once its block's S is done, a V slot once its
//                P V is done, so the keys of block g + 3 load while block g's softmax and P V run;
//   warp 1       TMEM owner (512 columns) and MMA issuer: S = Q K^T with Q read from TMEM (A
//                operand) and K from shared memory (K-major B); O += P V with P from TMEM and V
//                straight from the cache rows (keys x dims, the MN-major B operand); it takes
//                whichever of "S of the next block" and "P V of the oldest pending block" is
//                ready first;
//   warps 2-9    softmax, two warps per TMEM lane quarter (one query row per thread, each warp
//                of the pair half of the block's 64 keys and half of O's columns; the pair
//                exchanges row maxima and sums through shared memory): online softmax in the
//                exp2 domain with a lazily moved reference max (O and the row sum are rescaled
//                only when the block max exceeds it by more than 8, so P <= 2^8), P written over
//                the S columns it came from; after an item's first block they write the previous
//                item's O / l as the output operand pair;
//   warps 10-13  workers, per block: K_lo from K_hi and its residual codes (in K_hi's own swizzled
//                layout); at an item's first block its Q rows (times log2(e) / sqrt(hd)) as an fp16
//                pair into TMEM once the previous item's last S is done; then V_lo likewise, values
//                of keys past the last visible one zeroed (their P is 0, and a stale NaN would
//                still poison the product).
// TMEM columns: S/P [0,64) [64,128); O [128,128+HD) [128+HD,128+2HD) (items alternate);
// Q_hi [128+2HD,128+2.5HD) Q_lo [128+2.5HD,128+3HD).  Every wait is bounded; on a timeout the CTA
// records VLA_STATUS_TIMEOUT, drains its copies and MMAs, frees TMEM and stops.
#include <atomic>

#include "attention.h"
#include "gemm.h"
#include "ptx.cuh"

namespace vla {

namespace {

constexpr int kAtWarps = 14;
constexpr int kAtThreads = 32 * kAtWarps;
constexpr int kSoftWarps = 8;   // warps 2..9
constexpr int kWorkWarp0 = 10;  // warps 10..13
constexpr int kWorkWarps = 4;
constexpr int kStages = 3;
constexpr int kKeys = 64;  // keys per block
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0, kColO = 128;

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

__device__ __forceinline__ uint32_t h2_u32(__half2 v) { return *reinterpret_cast<uint32_t*>(&v); }
// (a, b) -> fp16 pairs hi = fp16(x), lo = fp16(x - hi), with packed conversions.
__device__ __forceinline__ void split_h2(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(a, b);
  const float2 f = __half22float2(h);
  hi = h2_u32(h);
  lo = h2_u32(__floats2half2_rn(a - f.x, b - f.y));
}
// 2^x (MUFU approximation, flush-to-zero; 2^-inf = 0)
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
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
  int n_items;             // tiles x heads
  float scale_log2;        // log2(e) / sqrt(HD), folded into the queries
  bool fp16;
  bool write_lo;           // write out_lo (else hi alone: the consumer reads the hi plane only)
  uint32_t* status;
  uint64_t wait_limit;
};

template <int HD>
struct AtSmem {
  static constexpr int K_BYTES = kKeys * HD * 2;        // one 64-key tile of K (or V), fp16
  static constexpr int R_BYTES = kKeys * HD / 2;        // its residual codes
  // a slot: hi | lo | codes of one 64-key tile (hi and lo 1024-byte aligned); the K ring's
  // kStages slots, then the V ring's
  static constexpr int SLOT = 2 * K_BYTES + R_BYTES;
  static constexpr int BARS = 512;                      // mbarriers, TMEM address, abort flag
  // + the softmax pairs' exchange: row maxima [2 blocks][2 halves][128] and partial row sums
  // [2 items][2 halves][128]
  static constexpr int SMEM = 1024 + 2 * kStages * SLOT + BARS + 2 * (2 * 2 * 128 * 4);
  static_assert(SLOT % 1024 == 0, "slot alignment");
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

// The j-th item of this CTA: (tile, head) number blockIdx.x + j * gridDim.x, tile-major.
struct Item {
  AttnTile tile;
  int head, n_keys, nb;
  int64_t krow0;  // first K row of (env, head) in the cache
};
__device__ __forceinline__ Item get_item(const AtParams& p, int j) {
  const int w = static_cast<int>(blockIdx.x) + j * static_cast<int>(gridDim.x);
  Item it;
  it.tile = p.tiles[w / p.H];
  it.head = w % p.H;
  it.n_keys = it.tile.pos0 + it.tile.nrows;
  it.nb = (it.n_keys + kKeys - 1) / kKeys;
  it.krow0 = p.layer_row0 + it.tile.env * p.env_rows + it.head * p.head_rows;
  return it;
}

// Bounded wait by lane 0, the verdict shared by the warp.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, uint32_t* status,
                                          uint64_t limit) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = wait_bounded(bar, parity, abort_flag, status, limit) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

template <int HD>
__global__ void __launch_bounds__(kAtThreads, 1)
    attn_chunk_tc_kernel(const __grid_constant__ CUtensorMap tmKV, const AtParams p) {
  using Sm = AtSmem<HD>;
  constexpr int KB = HD / 64;  // 64-element column blocks of one K / V row
  constexpr uint32_t kColQ = kColO + 2 * HD;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 2 * kStages * Sm::SLOT);
  float* xbuf = reinterpret_cast<float*>(smem + 2 * kStages * Sm::SLOT + Sm::BARS);  // [2][2][128] row maxima
  float* lbuf = xbuf + 2 * 2 * 128;                                                // [2][2][128] row sums
  const uint32_t b0 = smem_u32(bars);
  auto BAR = [&](int i) { return b0 + 8u * static_cast<uint32_t>(i); };
  // per K / V slot: full (loaded), conv (low part written), free (its MMAs done); per S/P
  // buffer: sfull (S written), sfree (P V done with it), pfull (P written); pdone (the latest
  // P V done); qready / qfree (Q written / the item's last S done); per item parity: odone (O
  // final); drain; per lane quarter and block parity: xch (the softmax pair's exchange written)
  const int FULLK = 0, FULLV = 3, CONVK = 6, CONVV = 9, KFREE = 12, VFREE = 15, SFULL = 18, SFREE = 20,
            PFULL = 22, PDONE = 24, QREADY = 25, QFREE = 26, ODONE = 27, DRAIN = 29, XCH = 30;
  static_assert(38 * 8 + 8 <= Sm::BARS, "barrier area");
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 38);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_my = (p.n_items - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                   static_cast<int>(gridDim.x);
  uint32_t* status = p.status;
  const uint64_t limit = p.wait_limit;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(BAR(FULLK + s), 1);
      mbar_init(BAR(FULLV + s), 1);
      mbar_init(BAR(CONVK + s), kWorkWarps);
      mbar_init(BAR(CONVV + s), kWorkWarps);
      mbar_init(BAR(KFREE + s), 1);
      mbar_init(BAR(VFREE + s), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(BAR(SFULL + s), 1);
      mbar_init(BAR(SFREE + s), 1);
      mbar_init(BAR(PFULL + s), kSoftWarps);
      mbar_init(BAR(ODONE + s), 1);
    }
    mbar_init(BAR(PDONE), 1);
    mbar_init(BAR(QREADY), kWorkWarps);
    mbar_init(BAR(QFREE), 1);
    mbar_init(BAR(DRAIN), 1);
    for (int s = 0; s < 8; ++s) mbar_init(BAR(XCH + s), 2);
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

  auto kslot = [&](int st) { return smem + st * Sm::SLOT; };
  auto vslot = [&](int st) { return smem + (kStages + st) * Sm::SLOT; };

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------------ producer
      pdl_wait_async();  // the chunks' own keys / values were written by the q|k|v projection
      // bit (ring * kStages + slot): a copy was issued there, with the phase it completes
      uint32_t issued = 0, issued_phase = 0;
      bool ok = true;
      int g = 0;  // block number over all of this CTA's items
      for (int j = 0; j < n_my && ok; ++j) {
        const Item it = get_item(p, j);
        for (int b = 0; b < it.nb && ok; ++b, ++g) {
          const int st = g % kStages, round = g / kStages;
          const int key0 = b * kKeys;
          const int rows = min(kKeys, p.cap - key0);  // residual rows inside this (env, head)
          const uint32_t rbytes = static_cast<uint32_t>(rows) * (HD / 2);
          // the K tile into its ring, then the V tile into its own
          for (int ring = 0; ring < 2; ++ring) {
            if (round >= 1 &&
                !wait_bounded(BAR((ring ? VFREE : KFREE) + st), (round - 1) & 1, abort_flag, status, limit)) {
              ok = false;
              break;
            }
            const uint32_t full = BAR((ring ? FULLV : FULLK) + st);
            const uint32_t s_hi = smem_u32(ring ? vslot(st) : kslot(st));
            const int64_t row0 = it.krow0 + (ring ? p.kv_rows : 0) + key0;
            mbar_arrive_expect_tx(full, Sm::K_BYTES + rbytes);
#pragma unroll
            for (int kb = 0; kb < KB; ++kb)
              tma_load_2d(s_hi + kb * (kKeys * 128), &tmKV, full, kb * 64, static_cast<int>(row0));
            bulk_load(s_hi + 2 * Sm::K_BYTES, p.res + row0 * (HD / 2), rbytes, full);
            const int bit = ring * kStages + st;
            issued |= 1u << bit;
            issued_phase = (issued_phase & ~(1u << bit)) | (static_cast<uint32_t>(round & 1) << bit);
          }
        }
      }
      for (int bit = 0; bit < 2 * kStages; ++bit)
        if (issued & (1u << bit))
          wait_drain(BAR((bit < kStages ? FULLK : FULLV) + bit % kStages), (issued_phase >> bit) & 1u, limit);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------------ MMA issuer
      const uint32_t IS = idesc_f16(kKeys), IO = idesc_f16(HD, true);
      const uint32_t tQh = tmem + kColQ, tQl = tmem + kColQ + HD / 2;
      // descriptors of slot 0's tiles; another slot (or k step) adds its byte offset / 16
      const uint64_t dK0 = sdesc_sw128(smem_u32(kslot(0)));
      const uint64_t dV0 = sdesc_sw128(smem_u32(vslot(0)), kKeys * 128);
      constexpr uint64_t kSlotStep = Sm::SLOT >> 4, kLoStep = Sm::K_BYTES >> 4;
      bool ok = true;
      // S cursor (item js, block bs, global block gs) and P V cursor (jo, bo, go)
      int js = 0, bs = 0, gs = 0, nbs = get_item(p, 0).nb;
      int jo = 0, bo = 0, go = 0, nbo = nbs;
      uint64_t t_last = globaltimer();
      uint32_t spins = 0;
      while (ok && jo < n_my) {
        bool did = false;
        if (go < gs && mbar_test_wait(BAR(PFULL + (go & 1)), (go >> 1) & 1) &&
            mbar_test_wait(BAR(CONVV + go % kStages), (go / kStages) & 1)) {
          // O(jo) (+)= P V of block go
          tc_fence_after();
          const uint64_t dvh = dV0 + (go % kStages) * kSlotStep;
          const uint32_t tO = tmem + kColO + (jo & 1) * HD;
          const uint32_t tPh = tmem + kColS + (go & 1) * kKeys, tPl = tPh + kKeys / 2;
#pragma unroll
          for (int k = 0; k < kKeys / 16; ++k) {
            const uint64_t dh = dvh + k * (2048 >> 4), dl = dh + kLoStep;
            mma_ts(tO, tPh + k * 8, dh, IO, (bo > 0 || k > 0) ? 1u : 0u);
            mma_ts(tO, tPl + k * 8, dh, IO, 1u);
            mma_ts(tO, tPh + k * 8, dl, IO, 1u);
          }
          tc_commit(BAR(PDONE));
          tc_commit(BAR(SFREE + (go & 1)));
          tc_commit(BAR(VFREE + go % kStages));
          if (bo == nbo - 1) tc_commit(BAR(ODONE + (jo & 1)));
          ++go;
          if (++bo == nbo) {
            bo = 0;
            if (++jo < n_my) nbo = get_item(p, jo).nb;
          }
          did = true;
        } else if (js < n_my && mbar_test_wait(BAR(CONVK + gs % kStages), (gs / kStages) & 1) &&
                   (gs < 2 || mbar_test_wait(BAR(SFREE + (gs & 1)), ((gs >> 1) - 1) & 1)) &&
                   (bs > 0 || mbar_test_wait(BAR(QREADY), js & 1))) {
          // S of block gs into buffer gs & 1
          tc_fence_after();
          const uint64_t dkh = dK0 + (gs % kStages) * kSlotStep;
          const uint32_t tS = tmem + kColS + (gs & 1) * kKeys;
#pragma unroll
          for (int k = 0; k < HD / 16; ++k) {
            const uint64_t dh = dkh + (((k >> 2) * (kKeys * 128) + (k & 3) * 32) >> 4), dl = dh + kLoStep;
            mma_ts(tS, tQh + k * 8, dh, IS, k > 0 ? 1u : 0u);
            mma_ts(tS, tQl + k * 8, dh, IS, 1u);
            mma_ts(tS, tQh + k * 8, dl, IS, 1u);
          }
          tc_commit(BAR(SFULL + (gs & 1)));
          tc_commit(BAR(KFREE + gs % kStages));
          if (bs == nbs - 1) tc_commit(BAR(QFREE));
          ++gs;
          if (++bs == nbs) {
            bs = 0;
            if (++js < n_my) nbs = get_item(p, js).nb;
          }
          did = true;
        }
        if (did) {
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
  } else if (warp < kWorkWarp0) {
    // ------------------------------------------------------------------ softmax (warps 2-9)
    const int q4 = warp & 3;                 // TMEM lane quarter of this warp
    const int hf = (warp - 2) >> 2;          // which 32 keys of a block, and which half of O's columns
    const int r = q4 * 32 + lane;            // query row in the tile
    const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
    const int dcols = p.H * HD;
    uint32_t sat = 0;  // convex combinations of the cached values: the fp16 split never saturates
    pdl_wait();        // the output may still be read by the previous kernel's predecessors
    // item jp's output, O / l as the operand pair: this warp's rows, its half of the columns
    auto epilogue = [&](int jp, float l_tot) -> bool {
      if (!warp_wait(BAR(ODONE + (jp & 1)), (jp >> 1) & 1, abort_flag, status, limit)) return false;
      tc_fence_after();
      const Item it = get_item(p, jp);
      const bool valid = r < it.tile.nrows;
      const float inv = 1.f / l_tot;
      const size_t off = static_cast<size_t>(it.tile.row0 + (valid ? r : 0)) * dcols + it.head * HD + hf * (HD / 2);
      const uint32_t tO = tmem + lane_off + kColO + (jp & 1) * HD + hf * (HD / 2);
#pragma unroll 1
      for (int c = 0; c < HD / 2; c += 16) {
        uint32_t v[16];
        tmem_ld16(tO + c, v);
        tmem_wait_ld();
        if (valid) {
          uint32_t h[8], lo[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            split_pack2(__uint_as_float(v[2 * i]) * inv, __uint_as_float(v[2 * i + 1]) * inv, h[i], lo[i], p.fp16,
                        sat);
          uint4* dh = reinterpret_cast<uint4*>(p.out_hi + off + c);
          dh[0] = make_uint4(h[0], h[1], h[2], h[3]);
          dh[1] = make_uint4(h[4], h[5], h[6], h[7]);
          if (p.write_lo) {
            uint4* dl = reinterpret_cast<uint4*>(p.out_lo + off + c);
            dl[0] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            dl[1] = make_uint4(lo[4], lo[5], lo[6], lo[7]);
          }
        }
      }
      return true;
    };
    // the pair's exchange at block g: this warp's value in, the partner's out
    auto exchange = [&](float* buf, int g, float v, float& other) -> bool {
      buf[hf * 128 + r] = v;
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(XCH + 2 * q4 + (g & 1)));
      if (!warp_wait(BAR(XCH + 2 * q4 + (g & 1)), (g >> 1) & 1, abort_flag, status, limit)) return false;
      other = buf[(hf ^ 1) * 128 + r];
      return true;
    };
    bool ok = true;
    int g = 0;
    float l_prev = 0.f;  // the previous item's partial row sum (this warp's keys)
    for (int j = 0; j < n_my && ok; ++j) {
      const Item it = get_item(p, j);
      const int qpos = it.tile.pos0 + min(r, it.tile.nrows - 1);
      const uint32_t tO = tmem + lane_off + kColO + (j & 1) * HD + hf * (HD / 2);
      float m_ref = -INFINITY, l = 0.f;
      for (int b = 0; b < it.nb; ++b, ++g) {
        if (!warp_wait(BAR(SFULL + (g & 1)), (g >> 1) & 1, abort_flag, status, limit)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tS = tmem + lane_off + kColS + (g & 1) * kKeys;
        float s[32];
        {
          uint32_t v0[16], v1[16];
          tmem_ld16(tS + hf * 32, v0);
          tmem_ld16(tS + hf * 32 + 16, v1);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            s[i] = __uint_as_float(v0[i]);
            s[16 + i] = __uint_as_float(v1[i]);
          }
        }
        const int key0 = b * kKeys + hf * 32;
        if (__any_sync(0xffffffffu, key0 + 31 > qpos)) {
#pragma unroll
          for (int c = 0; c < 32; ++c) s[c] = (key0 + c <= qpos) ? s[c] : -INFINITY;
        }
        float mb = s[0];
#pragma unroll
        for (int c = 1; c < 32; ++c) mb = fmaxf(mb, s[c]);
        // the pair's block maximum of row r (past the exchange both warps have read their S
        // columns, so P may overwrite them); an item's first block also carries the previous
        // item's partial row sums
        if (b == 0 && j > 0) lbuf[((j - 1) & 1) * 256 + hf * 128 + r] = l_prev;
        float mo;
        if (!exchange(xbuf + (g & 1) * 256, g, mb, mo)) {
          ok = false;
          break;
        }
        mb = fmaxf(mb, mo);
        float alpha = 1.f;
        if (mb > m_ref + 8.f) {
          // first block (m_ref = -inf) or a max well above the reference: move it
          alpha = ex2(m_ref - mb);  // 0 on the first block
          m_ref = mb;
          l *= alpha;
        }
        if (b >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {
          // O is the MMAs' until the previous block's P V is done
          if (!warp_wait(BAR(PDONE), (g - 1) & 1, abort_flag, status, limit)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < HD / 2; c += 16) {
            uint32_t v[16];
            tmem_ld16(tO + c, v);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
            tmem_st16(tO + c, v);
          }
        }
        // P over the S columns: hi of keys 2c, 2c + 1 in column c, lo 32 columns further
        {
          uint32_t hi[16], lo[16];
          float ps = 0.f;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float p0 = ex2(s[2 * i] - m_ref), p1 = ex2(s[2 * i + 1] - m_ref);
            ps += p0 + p1;
            split_h2(p0, p1, hi[i], lo[i]);
          }
          l += ps;
          tmem_st16(tS + hf * 16, hi);
          tmem_st16(tS + kKeys / 2 + hf * 16, lo);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(BAR(PFULL + (g & 1)));
        if (b == 0 && j > 0) {
          const float l_tot = l_prev + lbuf[((j - 1) & 1) * 256 + (hf ^ 1) * 128 + r];
          if (!epilogue(j - 1, l_tot)) {
            ok = false;
            break;
          }
        }
      }
      l_prev = l;
    }
    if (ok) {
      // the last item: its row sums through one more exchange, then its output
      const int j = n_my - 1;
      float lo_sum;
      if (exchange(lbuf + (j & 1) * 256, g, l_prev, lo_sum)) epilogue(j, l_prev + lo_sum);
    }
    report_saturation(status, sat);
  } else {
    // ------------------------------------------------------------------ workers (warps 10-13)
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;            // Q row written by this thread (its TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
    const int t = threadIdx.x - kWorkWarp0 * 32;
    const int dcols = p.H * HD;
    constexpr int CH = HD / 8;                             // 16-byte chunks of one row
    constexpr int ITER = kKeys * CH / (32 * kWorkWarps);   // chunks per thread and tile
    constexpr int KSTEP = 32 * kWorkWarps / CH;            // rows between a thread's chunks
    static_assert((32 * kWorkWarps) % CH == 0 && ITER >= 1, "converter tiling");
    pdl_wait();  // the queries were written by the q|k|v projection
    // Q rows of an item, times log2(e) / sqrt(HD), -> fp16 pair in TMEM (A operand of S)
    auto write_q = [&](const Item& it) {
      const bool valid = r < it.tile.nrows;
      const float* qrow = p.q + static_cast<size_t>(it.tile.row0 + (valid ? r : 0)) * dcols + it.head * HD;
#pragma unroll 1
      for (int c = 0; c < HD; c += 64) {
        float4 x[16];  // 64 values in flight
#pragma unroll
        for (int i = 0; i < 16; ++i)
          x[i] = valid ? __ldcg(reinterpret_cast<const float4*>(qrow + c) + i) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float4 v = x[half * 8 + i];
            split_h2(v.x * p.scale_log2, v.y * p.scale_log2, hi[2 * i], lo[2 * i]);
            split_h2(v.z * p.scale_log2, v.w * p.scale_log2, hi[2 * i + 1], lo[2 * i + 1]);
          }
          tmem_st16(tmem + lane_off + kColQ + (c + 32 * half) / 2, hi);
          tmem_st16(tmem + lane_off + kColQ + HD / 2 + (c + 32 * half) / 2, lo);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(BAR(QREADY));
    };
    auto prefetch_q = [&](const Item& it) {
      if (r < it.tile.nrows) {
        const float* qrow = p.q + static_cast<size_t>(it.tile.row0 + r) * dcols + it.head * HD;
#pragma unroll
        for (int c = 0; c < HD; c += 32) asm volatile("prefetch.global.L2 [%0];" ::"l"(qrow + c));
      }
    };
    // the low part of the tile in `slot` (hi | lo | codes): a thread's chunks all sit in one
    // column c (the stride over chunks is a multiple of CH), rows key0t, key0t + KSTEP, ...:
    // loads first, then decode and stores; keys >= live zeroed (hi and lo) when `zero_dead`
    auto convert = [&](uint8_t* slot, bool zero_dead, int live) {
      const int c = t % CH, key0t = t / CH;
      const int coff = (c >> 3) * (kKeys * 128) + key0t * 128 + (((c & 7) ^ (key0t & 7)) << 4);
      uint4 hv[ITER];
      uint32_t cv[ITER];
#pragma unroll
      for (int i = 0; i < ITER; ++i) {
        hv[i] = *reinterpret_cast<const uint4*>(slot + coff + i * KSTEP * 128);
        cv[i] = *reinterpret_cast<const uint32_t*>(slot + 2 * Sm::K_BYTES + (key0t + i * KSTEP) * (HD / 2) + c * 4);
      }
#pragma unroll
      for (int i = 0; i < ITER; ++i) {
        const int off = coff + i * KSTEP * 128;
        uint4* lo = reinterpret_cast<uint4*>(slot + Sm::K_BYTES + off);
        if (zero_dead && key0t + i * KSTEP >= live) {
          *reinterpret_cast<uint4*>(slot + off) = make_uint4(0u, 0u, 0u, 0u);
          *lo = make_uint4(0u, 0u, 0u, 0u);
        } else {
          *lo = kv_res_lo8(hv[i], cv[i]);
        }
      }
      fence_async_smem();  // the MMAs (async proxy) read what these generic stores wrote
      __syncwarp();
    };
    bool ok = true;
    int g = 0;
    for (int j = 0; j < n_my && ok; ++j) {
      const Item it = get_item(p, j);
      for (int b = 0; b < it.nb; ++b, ++g) {
        const int st = g % kStages, ph = (g / kStages) & 1;
        if (!warp_wait(BAR(FULLK + st), ph, abort_flag, status, limit)) {
          ok = false;
          break;
        }
        convert(kslot(st), false, 0);
        if (lane == 0) mbar_arrive(BAR(CONVK + st));
        if (b == 0) {
          // this item's queries, once the previous item's last S is done
          if (j > 0) {
            if (!warp_wait(BAR(QFREE), (j - 1) & 1, abort_flag, status, limit)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          write_q(it);
          if (j + 1 < n_my) prefetch_q(get_item(p, j + 1));
        }
        if (!warp_wait(BAR(FULLV + st), ph, abort_flag, status, limit)) {
          ok = false;
          break;
        }
        convert(vslot(st), true, it.n_keys - b * kKeys);  // keys of this block visible to some row
        if (lane == 0) mbar_arrive(BAR(CONVV + st));
      }
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
                         KVLayout kv, int layer, int H, int hd, uint32_t* status, cudaStream_t stream, bool fp16,
                         int num_sms, bool write_lo) {
  if (n_tiles <= 0) return VLA_OK;
  if (!kv.res || (hd != 64 && hd != 128) || num_sms <= 0) return VLA_ERR_UNSUPPORTED;
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
  p.n_items = n_tiles * H;
  p.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(hd));
  p.fp16 = fp16;
  p.write_lo = write_lo;
  p.status = status;
  p.wait_limit = g_wait_limit_ns.load(std::memory_order_relaxed);
  // tensor map over every row of the cache (rows = layers * layer_stride / hd): row coordinates
  // must fit a signed 32-bit int
  const int64_t total_rows = static_cast<int64_t>(layer + 1) * (kv.layer_stride / hd);
  if (total_rows >= (static_cast<int64_t>(1) << 31)) return VLA_ERR_UNSUPPORTED;
  CUtensorMap map;
  if (!make_tensor_map_2d(&map, kv.base, total_rows, hd, hd, kKeys, true))
    return cuda_fail(cudaErrorInvalidValue, "tensor map (KV cache)");
  // persistent: one CTA per SM (each holds ~220 KB of shared memory and all 512 TMEM columns)
  const dim3 grid(std::min(p.n_items, num_sms));
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
