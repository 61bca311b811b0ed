// Shared device/host helpers of libvla.so (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/vla.h"

namespace vla {

using bf16 = __nv_bfloat16;
using f16 = __half;  // KV-cache element type

// ----------------------------------------------------------------------------- launch log
// Every kernel launch goes through note_launch() so the handle can report how many of its
// kernels ran (the host counter is per process; handles keep their own copy too).
extern int64_t g_launch_count;
inline void note_launch() { ++g_launch_count; }

// ----------------------------------------------------------------------------- row info
// One entry per row of a packed chunk: env, absolute position, source kind, source index.
enum RowKind : int { ROW_VISUAL = 0, ROW_TEXT = 1, ROW_TOKEN = 2 };
struct RowInfo {
  int env, pos, kind, idx;
};

// KV cache geometry: [layer][env][2 (K,V)][H][cap][hd] fp16, plus a residual plane of the same
// geometry with one 4-bit code per element (two per byte: element 2i in the low nibble of byte
// i, 2i+1 in the high nibble), so element offset o has its code in byte o / 2 of `res`.
struct KVLayout {
  f16* base;          // whole cache
  uint8_t* res;       // residual codes (null: not written)
  int64_t layer_stride;
  int64_t env_stride;  // 2 * H * cap * hd
  int64_t kv_stride;   // H * cap * hd (V follows K)
  int64_t head_stride; // cap * hd
  int cap;
};

// 4-bit residual of a cached key / value x around hi = fp16(x): the code c in [0, 15] names the
// cell [(c - 8) / 16, (c - 7) / 16) of (x - hi) / ulp(hi) (clamped at both ends), and the value
// read back is hi + (2c - 15) ulp(hi) / 32, the cell's midpoint, within ulp(hi) / 32 of x: four
// bits past fp16's eleven.  ulp(hi) = 2^(e - 25) for the biased exponent e >= 1, 2^-24 for e = 0.
// x - hi is exact in fp32 and the scaling is by a power of two, so the code is exact.
__device__ __forceinline__ uint32_t kv_res_code(float x, f16 hi) {
  const uint32_t e = (__half_as_ushort(hi) >> 10) & 31u;
  const uint32_t ee = e ? e : 1u;
  const float scale = __uint_as_float((156u - ee) << 23);  // 16 / ulp(hi) = 2^(29 - ee)
  float j = floorf((x - __half2float(hi)) * scale);
  j = fminf(fmaxf(j, -8.f), 7.f);  // a NaN lands on -8: its value is NaN through hi anyway
  return static_cast<uint32_t>(static_cast<int>(j) + 8);
}
// Low parts of 8 cached fp16 values (one 16-byte chunk) from their 4-bit codes (4 bytes, element
// 2i in the low nibble of byte i): per element (2c - 15) * 2^(e - 30) = (2c - 15) ulp(hi) / 32, e
// the value's fp16 exponent field, in fp16 arithmetic with no conversion instruction.  2c goes
// into the mantissa of 1024 (fp16 bits 0x6400 | 2c), so 1024 + 2c - 1039 = 2c - 15 exactly;
// 2^(e - 30) is the value with mantissa and sign cleared (2^(e-15)) times 2^-15.  Exact for
// e >= 6; below that the term is under 2^-21 in magnitude and comes out as zero or a rounded
// subnormal.
// The pair form: h2 two fp16 values, w their 2c in the low bits of each half, or'ed with 0x6400.
__device__ __forceinline__ uint32_t kv_res_pair(uint32_t h2, uint32_t w) {
  const uint32_t e = h2 & 0x7C007C00u;
  const uint32_t c1039 = 0x640F640Fu, c2m15 = 0x02000200u;
  const __half2 k = __hsub2(*reinterpret_cast<const __half2*>(&w), *reinterpret_cast<const __half2*>(&c1039));
  const __half2 sc = __hmul2(*reinterpret_cast<const __half2*>(&e), *reinterpret_cast<const __half2*>(&c2m15));
  const __half2 r = __hmul2(k, sc);
  return *reinterpret_cast<const uint32_t*>(&r);
}
__device__ __forceinline__ uint4 kv_res_lo8(uint4 hi, uint32_t codes) {
  const uint32_t twice_lo = (codes << 1) & 0x1E1E1E1Eu;  // 2c of each byte's low nibble
  const uint32_t twice_hi = (codes >> 3) & 0x1E1E1E1Eu;  // 2c of each byte's high nibble
  auto pair = [&](uint32_t h2, uint32_t sel) {
    return kv_res_pair(h2, (__byte_perm(twice_lo, twice_hi, sel) & 0x00FF00FFu) | 0x64006400u);
  };
  return make_uint4(pair(hi.x, 0x0400u), pair(hi.y, 0x0501u), pair(hi.z, 0x0602u), pair(hi.w, 0x0703u));
}
// Low parts of two cached fp16 values h2 (element 0 in the low half) from their codes c0, c1.
__device__ __forceinline__ uint32_t kv_res_lo2(uint32_t h2, uint32_t c0, uint32_t c1) {
  return kv_res_pair(h2, (c0 << 1) | (c1 << 17) | 0x64006400u);
}

// ----------------------------------------------------------------------------- bf16 helpers
__device__ __forceinline__ float bf2f(bf16 x) { return __bfloat162float(x); }
__device__ __forceinline__ bf16 f2bf(float x) { return __float2bfloat16_rn(x); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t v) {
  __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&v);
  return __bfloat1622float2(b);
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_f16x2(uint32_t v) {
  __half2 b = *reinterpret_cast<__half2*>(&v);
  return __half22float2(b);
}

// A GEMM input activation x is stored as an unevaluated pair of bf16 values:
// hi = bf16(x), lo = bf16(x - hi), so hi + lo carries ~16 mantissa bits.  The GEMM multiplies
// both halves by the bf16 weights into one fp32 accumulator.
__device__ __forceinline__ void split_bf16(float x, bf16& hi, bf16& lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}
// Packs two consecutive values into (hi pair, lo pair) words.
__device__ __forceinline__ void split_pack2(float a, float b, uint32_t& hi, uint32_t& lo) {
  bf16 ha, la, hb, lb;
  split_bf16(a, ha, la);
  split_bf16(b, hb, lb);
  __nv_bfloat162 h2 = __halves2bfloat162(ha, hb), l2 = __halves2bfloat162(la, lb);
  hi = *reinterpret_cast<uint32_t*>(&h2);
  lo = *reinterpret_cast<uint32_t*>(&l2);
}

// The same pair in fp16: hi = fp16(x), lo = fp16(x - hi).  fp16 keeps 11 significant bits
// per half (bf16: 8), so the single hi alone is 8x closer to x than a bf16 hi; GEMMs fed the
// fp16 form run on fp16 weights.  A finite x beyond the fp16 range (|x| > 65504) saturates to
// +-65504 instead of turning into inf and sets `sat` (the kernel then raises
// VLA_STATUS_SATURATED); NaN and +-inf pass through unchanged, so a non-finite activation still
// reaches the action head's non-finite check.  The bf16 pair never saturates (fp32 range).
__device__ __forceinline__ void split_f16(float x, f16& hi, f16& lo, uint32_t& sat) {
  if (fabsf(x) > 65504.f && fabsf(x) != INFINITY) {
    x = copysignf(65504.f, x);
    sat = 1u;
  }
  hi = __float2half_rn(x);
  lo = __float2half_rn(x - __half2float(hi));
}
__device__ __forceinline__ void split_pack2_f16(float a, float b, uint32_t& hi, uint32_t& lo, uint32_t& sat) {
  f16 ha, la, hb, lb;
  split_f16(a, ha, la, sat);
  split_f16(b, hb, lb, sat);
  __half2 h2 = __halves2half2(ha, hb), l2 = __halves2half2(la, lb);
  hi = *reinterpret_cast<uint32_t*>(&h2);
  lo = *reinterpret_cast<uint32_t*>(&l2);
}
// Operand format chosen at run time (uniform across a launch): fp16 if `fp16`, else bf16.  Buffers of
// either format are 2-byte arrays; the pair halves come back as raw bits.
__device__ __forceinline__ void split_pack2(float a, float b, uint32_t& hi, uint32_t& lo, bool fp16,
                                            uint32_t& sat) {
  if (fp16)
    split_pack2_f16(a, b, hi, lo, sat);
  else
    split_pack2(a, b, hi, lo);
}
__device__ __forceinline__ void split_bits(float x, bool fp16, uint16_t& hi, uint16_t& lo, uint32_t& sat) {
  if (fp16) {
    f16 h, l;
    split_f16(x, h, l, sat);
    hi = __half_as_ushort(h);
    lo = __half_as_ushort(l);
  } else {
    bf16 h, l;
    split_bf16(x, h, l);
    hi = __bfloat16_as_ushort(h);
    lo = __bfloat16_as_ushort(l);
  }
}
// Stores x as the pair into hi[i] / lo[i] (2-byte elements of either format).
__device__ __forceinline__ void store_split1(void* hi, void* lo, size_t i, float x, bool fp16, uint32_t& sat) {
  uint16_t h, l;
  split_bits(x, fp16, h, l, sat);
  static_cast<uint16_t*>(hi)[i] = h;
  if (lo) static_cast<uint16_t*>(lo)[i] = l;
}
// Raises VLA_STATUS_SATURATED when this thread clamped a value (rare: one atomic per thread that did).
__device__ __forceinline__ void report_saturation(uint32_t* status, uint32_t sat) {
  if (sat && status) atomicOr(status, VLA_STATUS_SATURATED);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + expf(-x)); }

// ----------------------------------------------------------------------------- PDL
// Programmatic dependent launch: every kernel of the path is launched with programmatic
// stream serialization, lets its successor be scheduled early (launch_dependents) and waits
// for its predecessor's results (wait) before touching any memory the predecessor wrote or
// reads.  Data written by earlier kernels of the path is read with coherent loads (plain or
// ld.global.cg), never through the non-coherent read-only path (__ldg, const __restrict__):
// a kernel scheduled early can see stale read-only-cache lines there.  Without the launch
// attribute both instructions are no-ops.
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ----------------------------------------------------------------------------- test hooks
// Failure injection for the tests (set through vla_test_inject_launch_error): when armed with
// n >= 1, the n-th kernel launch from then on returns `g_inject_error` without launching, as a
// failed launch would; every launch site checks it first.  Nothing on the device is touched.
extern std::atomic<int64_t> g_inject_countdown;
extern std::atomic<int> g_inject_error;
inline cudaError_t injected_launch_error() {
  if (g_inject_countdown.load(std::memory_order_relaxed) <= 0) return cudaSuccess;
  if (g_inject_countdown.fetch_sub(1) == 1) return static_cast<cudaError_t>(g_inject_error.load());
  return cudaSuccess;
}
// Limit of every bounded mbarrier wait in the tcgen05 kernels, passed to each launch (1 s; a test
// hook lowers it so that a wait that nothing completes runs out quickly).
extern std::atomic<uint64_t> g_wait_limit_ns;
constexpr uint64_t kDefaultWaitLimitNs = 1000000000ull;

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args... args) {
  if (const cudaError_t inj = injected_launch_error()) return inj;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Raises a kernel's dynamic shared-memory limit on the current device.  Function attributes
// belong to each device's context, so the call is made once per (kernel, device): `done` holds
// one bit per device index < 64 (beyond that the call is repeated every time).  Host threads
// racing here at worst both make the call.
template <typename Kern>
inline cudaError_t set_smem_limit(Kern kern, int bytes, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0ull;
  if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
  return e;
}

// Makes `dev` current for the scope of one API call and gives the caller's device back on exit
// (the library must not change the current device of the calling thread).
struct DeviceGuard {
  int prev = -1;
  bool restore = false;
  cudaError_t err = cudaSuccess;
  explicit DeviceGuard(int dev) {
    err = cudaGetDevice(&prev);
    if (err == cudaSuccess && prev != dev) {
      err = cudaSetDevice(dev);
      restore = err == cudaSuccess;
    }
  }
  ~DeviceGuard() {
    if (restore) cudaSetDevice(prev);
  }
  DeviceGuard(const DeviceGuard&) = delete;
  DeviceGuard& operator=(const DeviceGuard&) = delete;
};

}  // namespace vla

// ----------------------------------------------------------------------------- host macros
#define VLA_CUDA_TRY(expr)                                   \
  do {                                                       \
    cudaError_t _e = (expr);                                 \
    if (_e != cudaSuccess) return ::vla::cuda_fail(_e, #expr); \
  } while (0)

namespace vla {
int cuda_fail(cudaError_t e, const char* what);  // records the message, returns VLA_ERR_CUDA
int record_error(int code, const char* msg);      // records the message, returns `code`
// Device address of the op entry points' status word on the current device (a file-scope
// device variable: looking it up allocates nothing).  VLA_OK or an error code.
int op_status_word(uint32_t** out);
}
