// Host engine behind the C ABI of include/vla.h: KV cache and workspace ownership, chunk
// bookkeeping for multi-turn trajectories, the 7-token decode loop and the teacher-forced
// score pass.
//
// Paper mapping: Algorithm 1 (rollout phase: π_θ generates v_out, f extracts a_t, Eq. 1
// sums token log-probs), §3.3 (a trajectory is one multi-turn context), Eq. 2 (the PPO
// ratio re-scores stored actions), §3.5 (large-batch decoding on one inference GPU).
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/vla.h"
#include "../../include/vla_ops.h"
#include "attention.h"
#include "gemm.h"
#include "misc.h"

namespace vla {

namespace {
thread_local std::string t_err;  // last error of this thread (for calls without a handle)
}

int cuda_fail(cudaError_t e, const char* what) {
  char buf[512];
  snprintf(buf, sizeof(buf), "CUDA error %d (%s) at %s", static_cast<int>(e),
           cudaGetErrorString(e), what);
  t_err = buf;
  return VLA_ERR_CUDA;
}

int record_error(int code, const char* msg) {
  t_err = msg;
  return code;
}

namespace {
// Status word of the op entry points (vla_ops.h): a file-scope device variable, one per device
// that loads the library, so that reporting a timeout or a saturation needs no allocation.
__device__ uint32_t g_op_status_word;
constexpr int kMaxOpDevices = 64;
std::mutex g_op_status_mu;
uint32_t* g_op_status_ptr[kMaxOpDevices] = {};
}  // namespace

int op_status_word(uint32_t** out) {
  int dev = 0;
  VLA_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxOpDevices) return record_error(VLA_ERR_UNSUPPORTED, "op status: device index >= 64");
  std::lock_guard<std::mutex> lock(g_op_status_mu);
  if (!g_op_status_ptr[dev]) {
    // the variable's name is only a host-side stand-in: ask for its address on this device
    void* p = nullptr;
    VLA_CUDA_TRY(cudaGetSymbolAddress(&p, g_op_status_word));
    g_op_status_ptr[dev] = static_cast<uint32_t*>(p);
  }
  *out = g_op_status_ptr[dev];
  return VLA_OK;
}

static int set_err(std::string* dst, int code, const std::string& msg) {
  t_err = msg;
  if (dst) *dst = msg;
  return code;
}

static int query_num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    return 148;
  return n;
}

// GEMM tiling / split-K plan for an M x N x K projection.
struct Plan {
  int block_n, splits;
};
static Plan plan_gemm(int M, int N, int K, int epi, int d, int num_sms) {
  const int tiles_m = (M + 127) / 128;
  int bn = 256;
  if (epi == EPI_QKV && (d % 256)) bn = 128;
  const int n_eff = (epi == EPI_SWIGLU) ? N / 2 : N;
  const int bn_eff = (epi == EPI_SWIGLU) ? bn / 2 : bn;
  int64_t units = static_cast<int64_t>(tiles_m) * ((n_eff + bn_eff - 1) / bn_eff);
  if (units >= num_sms) return {bn, 1};
  // Few tiles: narrower tiles, and split-K only when those still leave most SMs idle (at
  // 64 envs x 6 score rows, 96 full-K tiles on 152 SMs beat 192 half-K tiles plus the
  // reduction by ~20%).
  bn = 128;
  units = static_cast<int64_t>(tiles_m) * ((N + bn - 1) / bn);
  if (2 * units >= num_sms) return {bn, 1};
  const int kbt = (K + 63) / 64;
  int splits = static_cast<int>((num_sms + units / 2) / units);
  splits = std::max(1, std::min(splits, kbt / 2));
  if (splits == 1 && units < num_sms) {
    // keep the fused epilogue when split-K would not help
    bn = 128;
    if (epi == EPI_QKV && (d % 128)) bn = 256;
  }
  return {bn, splits};
}

struct EventPair {
  cudaEvent_t a, b;
  int cls;
};

}  // namespace vla

using namespace vla;

struct vla_handle {
  vla_config cfg{};
  int dev = 0;
  cudaStream_t stream = nullptr;
  int num_sms = 148;
  int max_tokens = 0;
  // borrowed weights (bf16); the projections are read through the fp16 copies below
  const bf16* embed = nullptr;
  std::vector<const bf16*> attn_norm, ffn_norm;
  std::vector<const bf16*> src_wqkv, src_wo, src_wgu, src_wdown;
  // owned fp16 copies of the projection matrices (one allocation, per layer q|k|v, o,
  // gate|up, down), written by vla_create and vla_sync_weights; wqkv .. wdown point into it
  f16* w16 = nullptr;
  std::vector<const bf16*> wqkv, wo, wgu, wdown;   // 2-byte fp16 elements (GemmArgs type)
  int* w16_range = nullptr;  // device flag: a converted weight was outside the fp16 range
  // operand format of every projection and of the activations that feed them
  bool fp16 = true;
  const bf16* final_norm = nullptr;
  const bf16* head_rows = nullptr;
  // owned device memory
  f16* kv = nullptr;      // KV cache [L][B][2][H][cap][hd] fp16
  uint8_t* kv_res = nullptr;  // its 4-bit residual codes, two per byte (KVLayout)
  KVLayout kvl{};
  float* h = nullptr;    // residual stream f32 [T, d]
  bf16* y = nullptr;     // RMSNorm output, operand pair: hi [T, d] then lo [T, d]
  float* q = nullptr;    // RoPE'd queries f32 [T, d]
  bf16* ao = nullptr;    // attention output, operand pair [2][T, d]
  bf16* u = nullptr;     // SwiGLU output, operand pair [2][T, F]
  float* ws = nullptr;
  size_t ws_bytes = 0;
  float* h_last = nullptr;
  float* head_in = nullptr;
  float* head_z = nullptr;  // action-bin logits [B * A, 256]
  float* head_entropy = nullptr;  // entropy of each action token's distribution [B, A]
  bool entropy_valid = false;     // set by decode / score, cleared by prefill / reset
  float* q_last = nullptr;  // last layer of a prefill: queries of each env's final row [B, d]
  // deferred RMSNorm between tile GEMMs: per-tile row sums of squares [d / 128 + 1][T], and
  // whether y currently holds an unnormalised row (h * w) whose scale the next GEMM applies
  float* ss_part = nullptr;
  bool y_deferred = false;
  int y_ss_tiles = 0;
  RowInfo* last_rows = nullptr;  // and those rows' RowInfo [B]
  float2* rope = nullptr;
  RowInfo* rows = nullptr;
  AttnTile* tiles = nullptr;
  int* sidx = nullptr;
  int* didx = nullptr;
  int* fed = nullptr;
  int* pending = nullptr;
  uint32_t* status = nullptr;
  float* part_o = nullptr;
  float2* part_ml = nullptr;
  int* attn_tickets = nullptr;  // [B * H], zero between decode-attention launches
  int attn_chunk = 320;  // max keys per decode-attention CTA
  int max_tiles = 0;
  // pinned host staging (ring of slots, each guarded by an event)
  static constexpr int kSlots = 4;
  void* stage_host[kSlots] = {};
  cudaEvent_t stage_ev[kSlots] = {};
  size_t stage_bytes = 0;
  int stage_next = 0;
  // host state per env
  std::vector<int> len, len_prefill;
  std::vector<uint8_t> has_pending, prefilled;
  int active_batch = 0;
  std::string err;
  // measurement
  uint32_t prof_mask = 0;
  std::vector<EventPair> ev_used, ev_free;
  int64_t prof_launches[VLA_KCLASS_COUNT] = {};
  double prof_ms[VLA_KCLASS_COUNT] = {};
  double prof_flops[VLA_KCLASS_COUNT] = {};
  double prof_bytes[VLA_KCLASS_COUNT] = {};
  int64_t launches_at_create = 0;
};

namespace vla {
namespace {

int fail(vla_handle* h, int code, const std::string& msg) { return set_err(h ? &h->err : nullptr, code, msg); }

// Returns a pinned staging slot whose previous upload has completed.
void* stage_slot(vla_handle* h, int* slot) {
  const int s = h->stage_next;
  h->stage_next = (s + 1) % vla_handle::kSlots;
  cudaEventSynchronize(h->stage_ev[s]);
  *slot = s;
  return h->stage_host[s];
}

int upload(vla_handle* h, void* dst, const void* src_host, size_t bytes) {
  if (!bytes) return VLA_OK;
  VLA_CUDA_TRY(cudaMemcpyAsync(dst, src_host, bytes, cudaMemcpyHostToDevice, h->stream));
  return VLA_OK;
}

// ---- measurement helpers
// Returns the index of the event pair bracketing the next launch, or -1 when class `cls`
// is not being timed.
int prof_begin(vla_handle* h, int cls) {
  if (!(h->prof_mask & (1u << cls))) return -1;
  if (h->ev_free.empty()) {
    EventPair e{};
    if (cudaEventCreate(&e.a) != cudaSuccess || cudaEventCreate(&e.b) != cudaSuccess) return -1;
    h->ev_free.push_back(e);
  }
  h->ev_used.push_back(h->ev_free.back());
  h->ev_free.pop_back();
  EventPair& p = h->ev_used.back();
  p.cls = cls;
  cudaEventRecord(p.a, h->stream);
  return static_cast<int>(h->ev_used.size()) - 1;
}
void prof_end(vla_handle* h, int ev, int cls, double flops, double bytes) {
  h->prof_launches[cls] += 1;
  h->prof_flops[cls] += flops;
  h->prof_bytes[cls] += bytes;
  if (ev >= 0) cudaEventRecord(h->ev_used[ev].b, h->stream);
}
void prof_harvest(vla_handle* h) {
  cudaStreamSynchronize(h->stream);
  for (auto& e : h->ev_used) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, e.a, e.b) == cudaSuccess) h->prof_ms[e.cls] += ms;
    h->ev_free.push_back(e);
  }
  h->ev_used.clear();
}

// Projections whose tile GEMMs (M > 128 rows: prefill, score, decode of more than 128 envs)
// also multiply the low half of the activation pair: q|k|v alone.  An fp16 activation alone is
// within 2^-11 relative of its value; with the KV cache carrying a 4-bit residual (read in full
// by the chunk attention), o, gate|up and down on hi alone keep the 7B action-bin logits closer
// to the exact model than all-but-gate|up pairs over a plain fp16 cache did.
// The weight-streaming GEMMs (M <= 128) always take both halves: they are bound by reading the
// weights, so the second MMA costs nothing there.
enum : unsigned { kProjQkv = 1, kProjO = 2, kProjGateUp = 4, kProjDown = 8 };
constexpr unsigned kTileLoMask = kProjQkv;
// Whether the projection `proj` of an M-row call reads the low half of its activation pair:
// the weight-streaming GEMM (M <= 128) always does, the tile GEMMs for kTileLoMask only.
constexpr bool gemm_reads_lo(int M, unsigned proj) { return M <= 128 || (kTileLoMask & proj) != 0; }

// A is the operand pair: hi at A, lo at A + a_plane (fp16 when h->fp16, else bf16).
// The GEMM that will consume h->y after a residual GEMM's RMSNorm (its N, K and epilogue).
struct NextGemm {
  int N, K, epi;
};

// epi.norm_w set (a residual GEMM followed by an RMSNorm into h->y): when this GEMM and `next`
// both run as unsplit tile GEMMs, y is written unnormalised with per-tile sums of squares and
// `next` applies the row scale in its epilogue; otherwise the norm is exact here (fused into
// the weight-streaming reduction, or its own kernel).
int run_gemm(vla_handle* h, int cls, const bf16* A, size_t a_plane, int lda, const bf16* W, int ldw,
             int M, int N, int K, EpiArgs epi, const NextGemm* next = nullptr) {
  const Plan pl = plan_gemm(M, N, K, epi.kind, h->cfg.d_model, h->num_sms);
  const bool stream_k = M <= 128;  // decode-sized: weight-streaming swap-AB GEMM
  const unsigned proj = epi.kind == EPI_QKV      ? kProjQkv
                        : epi.kind == EPI_SWIGLU ? kProjGateUp
                        : A == h->ao             ? kProjO
                                                 : kProjDown;
  GemmArgs g;
  g.A = A;
  g.A_lo = gemm_reads_lo(M, proj) ? A + a_plane : nullptr;
  g.lda = lda;
  g.B = W;
  g.ldb = ldw;
  g.M = M;
  g.N = N;
  g.K = K;
  g.block_n = pl.block_n;
  g.splits = pl.splits;
  g.workspace = h->ws;
  g.workspace_bytes = h->ws_bytes;
  epi.status = h->status;
  epi.fp16 = h->fp16;
  g.epi = epi;
  if (!stream_k && gemm_workspace_bytes(g) > h->ws_bytes) {
    g.splits = 1;
  }
  // Large tile GEMMs run on CTA pairs (256 x 256 tiles, 2-SM MMAs) when there are enough
  // pair tiles to cover half the SMs and M is large enough that 256-row tiles waste little
  // (at the score pass's 384 rows the pair's 512 padded rows made gate|up 117 us vs 92 us).
  if (!stream_k && g.splits == 1 && g.block_n == 256 && M >= 1024) {
    const int64_t pair_tiles = static_cast<int64_t>((M + 255) / 256) *
                               (epi.kind == EPI_SWIGLU ? (N / 2 + 127) / 128 : (N + 255) / 256);
    g.pair = pair_tiles >= h->num_sms / 2;
  }
  // A following RMSNorm is fused into the weight-streaming GEMM's reduction; after a tile GEMM
  // it is deferred to the consuming tile GEMM when both run unsplit, else its own kernel.
  const EpiArgs norm = epi;
  bool defer_norm = false;
  if (!stream_k && norm.norm_w && next && g.splits == 1 && M > 128 && N % 128 == 0) {
    const Plan pn = plan_gemm(M, next->N, next->K, next->epi, h->cfg.d_model, h->num_sms);
    defer_norm = pn.splits == 1;
  }
  if (!stream_k) {
    if (defer_norm)
      g.epi.ss_out = h->ss_part;
    else
      g.epi.norm_w = nullptr;
  }
  // the consumer of a deferred norm: y is unnormalised, scale its rows here
  const bool consume = (A == h->y) && h->y_deferred && (epi.kind == EPI_QKV || epi.kind == EPI_SWIGLU);
  if (consume) {
    if (stream_k || g.splits != 1) return fail(h, VLA_ERR_ARG, "deferred RMSNorm reached a split GEMM");
    g.epi.row_ss = h->ss_part;
    g.epi.row_ss_n = h->y_ss_tiles;
    g.epi.row_d = K;
    g.epi.row_eps = h->cfg.rms_eps;
  }
  if (h->ev_used.size() > 8192) prof_harvest(h);
  int ev = prof_begin(h, cls);
  GemmCost cost{0, 0};
  int rc = stream_k ? gemv_launch(g, h->stream, h->num_sms, &cost)
                    : gemm_launch(g, h->stream, h->num_sms, &cost);
  prof_end(h, ev, cls, cost.flops, cost.bytes);
  if (rc != VLA_OK) return fail(h, rc, t_err.empty() ? "gemm launch failed" : t_err);
  if (consume) h->y_deferred = false;
  if (defer_norm) {
    h->y_deferred = true;
    h->y_ss_tiles = (N + g.block_n - 1) / g.block_n;
  }
  if (!stream_k && norm.norm_w && !defer_norm) {
    ev = prof_begin(h, VLA_KCLASS_OTHER);
    rc = rmsnorm_launch(norm.resid, norm.ldr, norm.norm_w, M, N, norm.norm_eps, norm.norm_hi, norm.norm_lo,
                        h->stream, h->fp16, h->status);
    prof_end(h, ev, VLA_KCLASS_OTHER, 0, 6.0 * M * N);
    if (rc) return fail(h, rc, t_err);
  }
  return VLA_OK;
}

// Rows whose last-layer output is needed (a prefill only feeds the head with each env's
// final row): idx [n] into the chunk's rows, rows [n] their RowInfo, max_ctx = longest context.
struct LastRows {
  int n = 0;
  const int* idx = nullptr;
  const RowInfo* rows = nullptr;
  int max_ctx = 0;
};

// All decoder layers over M rows already assembled in h->h (Llama-2 layer, §3.1).
// decode == true: one query per env row (rows[b] gives env and position), split-K attention.
// Otherwise n_tiles attention tiles in h->tiles, the largest of tile_rows rows.
// last != nullptr: the last layer computes q|k|v (the KV cache) for all M rows but attention,
// O, SwiGLU FFN and the residual only for last->rows, whose output lands in h->h_last.
int forward_layers(vla_handle* h, int M, const RowInfo* rows_dev, bool decode, int n_tiles, int tile_rows,
                   int max_ctx, const LastRows* last = nullptr) {
  const vla_config& c = h->cfg;
  const int d = c.d_model, F = c.d_ffn, H = c.n_heads, hd = c.head_dim;
  const int gcls = decode ? VLA_KCLASS_GEMM_DECODE : VLA_KCLASS_GEMM_PREFILL;
  const size_t pd = static_cast<size_t>(h->max_tokens) * d;   // hi -> lo plane offsets
  const size_t pf = static_cast<size_t>(h->max_tokens) * F;
  int rc;
  // the first layer's attention RMSNorm; every later RMSNorm follows a residual add
  h->y_deferred = false;
  int ev = prof_begin(h, VLA_KCLASS_OTHER);
  if ((rc = rmsnorm_launch(h->h, d, h->attn_norm[0], M, d, c.rms_eps, h->y, h->y + pd, h->stream, h->fp16,
                           h->status)))
    return fail(h, rc, t_err);
  prof_end(h, ev, VLA_KCLASS_OTHER, 0, 6.0 * M * d);
  for (int l = 0; l < c.n_layers; ++l) {

    EpiArgs e;
    e.kind = EPI_QKV;
    e.out_q = h->q;
    e.rows = rows_dev;
    e.kv = h->kvl;
    e.layer = l;
    e.rope = h->rope;
    e.d = d;
    e.hd = hd;
    if ((rc = run_gemm(h, gcls, h->y, pd, d, h->wqkv[l], d, M, 3 * d, d, e))) return rc;

    const bool pruned = last && last->n > 0 && l + 1 == c.n_layers;
    int Mr = M;           // rows past the attention
    float* resid = h->h;  // their residual stream
    if (pruned) {
      ev = prof_begin(h, VLA_KCLASS_OTHER);
      if ((rc = gather_rows_launch(h->q, last->idx, last->n, d, h->q_last, h->stream)) ||
          (rc = gather_rows_launch(h->h, last->idx, last->n, d, h->h_last, h->stream)))
        return fail(h, rc, t_err);
      prof_end(h, ev, VLA_KCLASS_OTHER, 0, 16.0 * last->n * d);
      ev = prof_begin(h, VLA_KCLASS_ATTN_DECODE);
      rc = attn_decode_launch(h->q_last, h->ao, h->ao + pd, last->rows, last->n, last->max_ctx, h->kvl, l, H, hd,
                              h->attn_chunk, h->part_o, h->part_ml, h->attn_tickets, h->stream, h->fp16);
      prof_end(h, ev, VLA_KCLASS_ATTN_DECODE, 0, 0);
      Mr = last->n;
      resid = h->h_last;
    } else if (decode) {
      ev = prof_begin(h, VLA_KCLASS_ATTN_DECODE);
      rc = attn_decode_launch(h->q, h->ao, h->ao + pd, rows_dev, M, max_ctx, h->kvl, l, H, hd,
                              h->attn_chunk, h->part_o, h->part_ml, h->attn_tickets, h->stream, h->fp16);
      prof_end(h, ev, VLA_KCLASS_ATTN_DECODE, 0, 0);
    } else {
      ev = prof_begin(h, VLA_KCLASS_ATTN_PREFILL);
      // the low plane of the output only where the o projection reads it; tiles of at most 16
      // rows (the score pass) on the few-row kernel
      rc = tile_rows <= kAttnRowsMax
               ? attn_rows_launch(h->q, h->ao, h->ao + pd, h->tiles, n_tiles, h->kvl, l, H, hd, h->stream, h->fp16,
                                  gemm_reads_lo(M, kProjO))
               : attn_chunk_tc_launch(h->q, h->ao, h->ao + pd, h->tiles, n_tiles, h->kvl, l, H, hd, h->status,
                                      h->stream, h->fp16, h->num_sms, gemm_reads_lo(M, kProjO));
      prof_end(h, ev, VLA_KCLASS_ATTN_PREFILL, 0, 0);
    }
    if (rc) return fail(h, rc, t_err);

    EpiArgs eo;
    eo.kind = EPI_RESID;
    eo.resid = resid;
    eo.ldr = d;
    eo.norm_w = h->ffn_norm[l];
    eo.norm_eps = c.rms_eps;
    eo.norm_hi = h->y;
    // the low halves of y and u only where gate|up and down read them
    eo.norm_lo = gemm_reads_lo(Mr, kProjGateUp) ? h->y + pd : nullptr;
    eo.ldn = d;
    const NextGemm gate_up{2 * F, d, EPI_SWIGLU};
    if ((rc = run_gemm(h, gcls, h->ao, pd, d, h->wo[l], d, Mr, d, d, eo, &gate_up))) return rc;

    EpiArgs eg;
    eg.kind = EPI_SWIGLU;
    eg.out_hi = h->u;
    eg.out_lo = gemm_reads_lo(Mr, kProjDown) ? h->u + pf : nullptr;
    eg.ldo = F;
    if ((rc = run_gemm(h, gcls, h->y, pd, d, h->wgu[l], d, Mr, 2 * F, d, eg))) return rc;

    EpiArgs ed;
    ed.kind = EPI_RESID;
    ed.resid = resid;
    ed.ldr = d;
    if (l + 1 < c.n_layers) {
      ed.norm_w = h->attn_norm[l + 1];
      ed.norm_eps = c.rms_eps;
      ed.norm_hi = h->y;
      ed.norm_lo = h->y + pd;
      ed.ldn = d;
    }
    const NextGemm qkv_next{3 * d, d, EPI_QKV};
    if ((rc = run_gemm(h, gcls, h->u, pf, F, h->wdown[l], F, Mr, d, F, ed, &qkv_next))) return rc;
  }
  return VLA_OK;
}

bool finite_nonneg(float t) { return std::isfinite(t) && t >= 0.f; }

// fp16 elements of the projection copies: per layer 3d*d + d*d + 2F*d + d*F.
size_t w16_elems(const vla_config& c) {
  const size_t d = c.d_model, F = c.d_ffn;
  return static_cast<size_t>(c.n_layers) * (4 * d * d + 3 * F * d);
}

// Converts every borrowed bf16 projection matrix into the handle's fp16 copy on h->stream and
// waits; VLA_ERR_UNSUPPORTED when a weight was outside the fp16 range (clamped in the copy).
int convert_weights(vla_handle* h) {
  const vla_config& c = h->cfg;
  const size_t dd = static_cast<size_t>(c.d_model) * c.d_model, fd = static_cast<size_t>(c.d_ffn) * c.d_model;
  if (cudaMemsetAsync(h->w16_range, 0, sizeof(int), h->stream) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "weight conversion: flag reset");
  for (int l = 0; l < c.n_layers; ++l) {
    const struct {
      const bf16* src;
      const bf16* dst;
      size_t n;
    } m[4] = {{h->src_wqkv[l], h->wqkv[l], 3 * dd}, {h->src_wo[l], h->wo[l], dd},
              {h->src_wgu[l], h->wgu[l], 2 * fd}, {h->src_wdown[l], h->wdown[l], fd}};
    for (const auto& x : m) {
      const int rc = bf16_to_f16_launch(x.src, reinterpret_cast<f16*>(const_cast<bf16*>(x.dst)), x.n,
                                        h->w16_range, h->num_sms, h->stream);
      if (rc == VLA_ERR_ARG) return record_error(VLA_ERR_ARG, "weight conversion: a projection matrix is not 16-byte aligned");
      if (rc) return rc;
    }
  }
  int bad = 0;
  if (cudaMemcpyAsync(&bad, h->w16_range, sizeof(int), cudaMemcpyDeviceToHost, h->stream) != cudaSuccess ||
      cudaStreamSynchronize(h->stream) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "weight conversion");
  if (bad) return record_error(VLA_ERR_UNSUPPORTED, "a projection weight is outside the fp16 range (|w| > 65504)");
  return VLA_OK;
}

}  // namespace
}  // namespace vla

// =================================================================================== C ABI
extern "C" {

int vla_create(const vla_config* cfg, const vla_weights* w, void* cuda_stream, vla_handle** out) {
  if (out) *out = nullptr;
  if (!cfg || !w || !out) return set_err(nullptr, VLA_ERR_ARG, "vla_create: NULL argument");
  const vla_config& c = *cfg;
  if (c.n_layers < 1 || c.d_model < 1 || c.n_heads < 1 || c.head_dim < 1 || c.d_ffn < 1 ||
      c.vocab < 1 || c.max_batch < 1 || c.kv_capacity < 1 || c.max_tokens < 1 ||
      !(c.rms_eps >= 0.f) || !(c.rope_theta > 0.f))
    return set_err(nullptr, VLA_ERR_ARG, "vla_create: non-positive size in config");
  if (c.head_dim != 64 && c.head_dim != 128)
    return set_err(nullptr, VLA_ERR_UNSUPPORTED, "vla_create: head_dim must be 64 or 128");
  if (c.n_heads * c.head_dim != c.d_model || c.d_model % 128 || c.d_model > 6400 || c.d_ffn % 8)
    return set_err(nullptr, VLA_ERR_UNSUPPORTED,
                   "vla_create: need n_heads*head_dim == d_model, d_model % 128 == 0, d_model <= 6400, "
                   "d_ffn % 8 == 0");
  if (c.n_action_bins != 256 || c.vocab < 256 || c.action_dim < 1 || c.action_dim > 16)
    return set_err(nullptr, VLA_ERR_UNSUPPORTED,
                   "vla_create: need n_action_bins == 256, vocab >= 256, 1 <= action_dim <= 16");
  if (!w->embed || !w->attn_norm || !w->wqkv || !w->wo || !w->ffn_norm || !w->w_gate_up ||
      !w->w_down || !w->final_norm || !w->lm_head)
    return set_err(nullptr, VLA_ERR_ARG, "vla_create: NULL weight pointer");
  for (int l = 0; l < c.n_layers; ++l)
    if (!w->attn_norm[l] || !w->wqkv[l] || !w->wo[l] || !w->ffn_norm[l] || !w->w_gate_up[l] ||
        !w->w_down[l])
      return set_err(nullptr, VLA_ERR_ARG, "vla_create: NULL per-layer weight pointer");

  int dev = 0;
  if (const cudaError_t e = cudaGetDevice(&dev)) return cuda_fail(e, "vla_create: current device");
  vla_handle* h = new vla_handle();
  h->cfg = c;
  h->stream = static_cast<cudaStream_t>(cuda_stream);
  h->dev = dev;
  h->num_sms = query_num_sms();
  const int A = c.action_dim, B = c.max_batch, d = c.d_model, F = c.d_ffn, L = c.n_layers;
  h->max_tokens = std::max(c.max_tokens, std::max(B, (A - 1) * B));
  h->embed = static_cast<const bf16*>(w->embed);
  for (int l = 0; l < L; ++l) {
    h->attn_norm.push_back(static_cast<const bf16*>(w->attn_norm[l]));
    h->src_wqkv.push_back(static_cast<const bf16*>(w->wqkv[l]));
    h->src_wo.push_back(static_cast<const bf16*>(w->wo[l]));
    h->ffn_norm.push_back(static_cast<const bf16*>(w->ffn_norm[l]));
    h->src_wgu.push_back(static_cast<const bf16*>(w->w_gate_up[l]));
    h->src_wdown.push_back(static_cast<const bf16*>(w->w_down[l]));
  }
  h->final_norm = static_cast<const bf16*>(w->final_norm);
  h->head_rows = static_cast<const bf16*>(w->lm_head) + static_cast<size_t>(c.vocab - 256) * d;
  h->len.assign(B, 0);
  h->len_prefill.assign(B, 0);
  h->has_pending.assign(B, 0);
  h->prefilled.assign(B, 0);
  h->launches_at_create = g_launch_count;

  // KV cache geometry [layer][env][K,V][H][cap][hd]
  const int64_t cap = c.kv_capacity;
  h->kvl.cap = c.kv_capacity;
  h->kvl.head_stride = cap * c.head_dim;
  h->kvl.kv_stride = static_cast<int64_t>(c.n_heads) * h->kvl.head_stride;
  h->kvl.env_stride = 2 * h->kvl.kv_stride;
  h->kvl.layer_stride = static_cast<int64_t>(B) * h->kvl.env_stride;

  // split-K workspace: worst case over the decode / score projection shapes
  size_t ws = 0;
  std::vector<int> Ms = {B, (A - 1) * B};
  for (int M = 128; M <= h->max_tokens; M += 128) Ms.push_back(M);
  for (int M : Ms) {
    if (M < 1 || M > h->max_tokens) continue;
    const int shapes[4][4] = {{3 * d, d, EPI_QKV, 0}, {d, d, EPI_RESID, 0}, {2 * F, d, EPI_SWIGLU, 0}, {d, F, EPI_RESID, 0}};
    for (auto& s : shapes) {
      if (M <= 128) {
        ws = std::max(ws, gemv_workspace_bytes(M, s[0], s[1], h->num_sms));
        continue;
      }
      const Plan pl = plan_gemm(M, s[0], s[1], s[2], d, h->num_sms);
      const int sp = gemm_effective_splits(s[1], pl.splits);
      if (sp > 1) ws = std::max(ws, static_cast<size_t>(sp) * M * s[0] * sizeof(float));
    }
  }
  h->ws_bytes = ws;
  const int max_S = (c.kv_capacity + h->attn_chunk - 1) / h->attn_chunk;
  h->max_tiles = h->max_tokens / 64 + B + 1;
  const size_t T = h->max_tokens;

  auto alloc = [&](void** p, size_t bytes) -> bool {
    if (!bytes) return true;
    return cudaMalloc(p, bytes) == cudaSuccess;
  };
  bool ok = alloc(reinterpret_cast<void**>(&h->kv), static_cast<size_t>(L) * h->kvl.layer_stride * sizeof(f16)) &&
            alloc(reinterpret_cast<void**>(&h->kv_res), static_cast<size_t>(L) * h->kvl.layer_stride / 2) &&
            alloc(reinterpret_cast<void**>(&h->h), T * d * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->y), 2 * T * d * sizeof(bf16)) &&
            alloc(reinterpret_cast<void**>(&h->q), T * d * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->ao), 2 * T * d * sizeof(bf16)) &&
            alloc(reinterpret_cast<void**>(&h->u), 2 * T * F * sizeof(bf16)) &&
            alloc(reinterpret_cast<void**>(&h->ws), ws) &&
            alloc(reinterpret_cast<void**>(&h->h_last), static_cast<size_t>(B) * d * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->head_in), static_cast<size_t>(B) * A * d * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->head_z), static_cast<size_t>(B) * A * 256 * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->head_entropy), static_cast<size_t>(B) * A * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->q_last), static_cast<size_t>(B) * d * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->ss_part), static_cast<size_t>(d / 128 + 1) * T * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->last_rows), static_cast<size_t>(B) * sizeof(RowInfo)) &&
            alloc(reinterpret_cast<void**>(&h->rope), static_cast<size_t>(cap) * (c.head_dim / 2) * sizeof(float2)) &&
            alloc(reinterpret_cast<void**>(&h->rows), T * sizeof(RowInfo)) &&
            alloc(reinterpret_cast<void**>(&h->tiles), static_cast<size_t>(h->max_tiles) * sizeof(AttnTile)) &&
            alloc(reinterpret_cast<void**>(&h->sidx), std::max(T, static_cast<size_t>(B) * A) * sizeof(int)) &&
            alloc(reinterpret_cast<void**>(&h->didx), std::max(T, static_cast<size_t>(B) * A) * sizeof(int)) &&
            alloc(reinterpret_cast<void**>(&h->fed), static_cast<size_t>(B) * A * sizeof(int)) &&
            alloc(reinterpret_cast<void**>(&h->pending), static_cast<size_t>(B) * sizeof(int)) &&
            alloc(reinterpret_cast<void**>(&h->status), sizeof(uint32_t)) &&
            alloc(reinterpret_cast<void**>(&h->part_o), static_cast<size_t>(B) * c.n_heads * max_S * c.head_dim * sizeof(float)) &&
            alloc(reinterpret_cast<void**>(&h->part_ml), static_cast<size_t>(B) * c.n_heads * max_S * sizeof(float2)) &&
            alloc(reinterpret_cast<void**>(&h->attn_tickets), static_cast<size_t>(B) * c.n_heads * sizeof(int)) &&
            alloc(reinterpret_cast<void**>(&h->w16), w16_elems(c) * sizeof(f16)) &&
            alloc(reinterpret_cast<void**>(&h->w16_range), sizeof(int)) &&
            cudaMemset(h->attn_tickets, 0, static_cast<size_t>(B) * c.n_heads * sizeof(int)) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    vla_destroy(h);
    return set_err(nullptr, VLA_ERR_OOM, "vla_create: device allocation failed");
  }
  h->kvl.base = h->kv;
  h->kvl.res = h->kv_res;
  {
    const size_t dd = static_cast<size_t>(d) * d, fd = static_cast<size_t>(F) * d;
    f16* p = h->w16;
    for (int l = 0; l < L; ++l) {
      h->wqkv.push_back(reinterpret_cast<const bf16*>(p));
      p += 3 * dd;
      h->wo.push_back(reinterpret_cast<const bf16*>(p));
      p += dd;
      h->wgu.push_back(reinterpret_cast<const bf16*>(p));
      p += 2 * fd;
      h->wdown.push_back(reinterpret_cast<const bf16*>(p));
      p += fd;
    }
  }
  if (const int rc = convert_weights(h)) {
    const std::string msg = t_err;
    vla_destroy(h);
    return set_err(nullptr, rc, msg);
  }
  // pinned staging
  h->stage_bytes = T * sizeof(RowInfo) + static_cast<size_t>(h->max_tiles) * sizeof(AttnTile) +
                   2 * std::max(T, static_cast<size_t>(B) * A) * sizeof(int) + static_cast<size_t>(B) * sizeof(RowInfo) +
                   1024;
  for (int s = 0; s < vla_handle::kSlots; ++s) {
    if (cudaMallocHost(&h->stage_host[s], h->stage_bytes) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->stage_ev[s], cudaEventDisableTiming) != cudaSuccess) {
      cudaGetLastError();
      vla_destroy(h);
      return set_err(nullptr, VLA_ERR_OOM, "vla_create: pinned host allocation failed");
    }
  }
  // RoPE table in fp64 on the host: angle = pos * theta^(-2i/hd)
  {
    const int half = c.head_dim / 2;
    std::vector<float2> tab(static_cast<size_t>(cap) * half);
    for (int64_t p = 0; p < cap; ++p)
      for (int i = 0; i < half; ++i) {
        const double ang = static_cast<double>(p) *
                           std::pow(static_cast<double>(c.rope_theta), -2.0 * i / c.head_dim);
        tab[p * half + i] = make_float2(static_cast<float>(std::cos(ang)), static_cast<float>(std::sin(ang)));
      }
    if (cudaMemcpy(h->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemset(h->status, 0, sizeof(uint32_t)) != cudaSuccess ||
        cudaMemset(h->pending, 0, static_cast<size_t>(B) * sizeof(int)) != cudaSuccess) {
      const int rc = cuda_fail(cudaGetLastError(), "vla_create: initial copies");
      vla_destroy(h);
      return rc;
    }
  }
  *out = h;
  return VLA_OK;
}

int vla_prefill(vla_handle* h, int batch, const void* visual, int n_visual, const int32_t* token_ids,
                const int32_t* lengths, int max_len) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_prefill: NULL handle");
  const vla_config& c = h->cfg;
  if (batch < 1 || batch > c.max_batch) return fail(h, VLA_ERR_ARG, "vla_prefill: batch outside [1, max_batch]");
  if (n_visual < 0 || max_len < 0 || !lengths) return fail(h, VLA_ERR_ARG, "vla_prefill: bad n_visual / max_len / lengths");
  if (n_visual > 0 && !visual) return fail(h, VLA_ERR_ARG, "vla_prefill: NULL visual");
  int64_t total = 0;
  bool any_text = false;
  std::vector<int> chunk(batch);
  for (int b = 0; b < batch; ++b) {
    if (lengths[b] < 0 || lengths[b] > max_len) return fail(h, VLA_ERR_ARG, "vla_prefill: length outside [0, max_len]");
    any_text |= lengths[b] > 0;
    chunk[b] = (h->has_pending[b] ? 1 : 0) + n_visual + lengths[b];
    if (chunk[b] < 1) return fail(h, VLA_ERR_ARG, "vla_prefill: empty chunk");
    if (static_cast<int64_t>(h->len[b]) + chunk[b] + (c.action_dim - 1) > c.kv_capacity)
      return fail(h, VLA_ERR_CAPACITY, "vla_prefill: KV capacity of an env would be exceeded");
    total += chunk[b];
  }
  if (any_text && !token_ids) return fail(h, VLA_ERR_ARG, "vla_prefill: NULL token_ids");
  if (total > h->max_tokens) return fail(h, VLA_ERR_CAPACITY, "vla_prefill: more rows than max_tokens");
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_prefill: set device"), t_err);

  // host-side row table, attention tiles and last-row indices
  int slot;
  uint8_t* st = static_cast<uint8_t*>(stage_slot(h, &slot));
  RowInfo* rows = reinterpret_cast<RowInfo*>(st);
  AttnTile* tiles = reinterpret_cast<AttnTile*>(rows + total);
  int n_tiles = 0, tile_rows = 0;
  std::vector<int> last(batch);
  int r = 0;
  for (int b = 0; b < batch; ++b) {
    const int r0 = r;
    int pos = h->len[b];
    if (h->has_pending[b]) rows[r++] = RowInfo{b, pos++, ROW_TOKEN, b};
    for (int j = 0; j < n_visual; ++j) rows[r++] = RowInfo{b, pos++, ROW_VISUAL, b * n_visual + j};
    for (int j = 0; j < lengths[b]; ++j) rows[r++] = RowInfo{b, pos++, ROW_TEXT, b * max_len + j};
    for (int t0 = 0; t0 < chunk[b]; t0 += 128) {
      tiles[n_tiles++] = AttnTile{b, r0 + t0, std::min(128, chunk[b] - t0), h->len[b] + t0};
      tile_rows = std::max(tile_rows, std::min(128, chunk[b] - t0));
    }
    last[b] = r - 1;
  }
  int* sidx = reinterpret_cast<int*>(tiles + n_tiles);
  RowInfo* last_rows = reinterpret_cast<RowInfo*>(sidx + batch);
  LastRows lr;
  lr.n = batch;
  lr.idx = h->sidx;
  lr.rows = h->last_rows;
  for (int b = 0; b < batch; ++b) {
    sidx[b] = last[b];
    last_rows[b] = rows[last[b]];
    lr.max_ctx = std::max(lr.max_ctx, h->len[b] + chunk[b]);
  }
  int rc;
  if ((rc = upload(h, h->rows, rows, total * sizeof(RowInfo))) ||
      (rc = upload(h, h->tiles, tiles, n_tiles * sizeof(AttnTile))) ||
      (rc = upload(h, h->sidx, sidx, batch * sizeof(int))) ||
      (rc = upload(h, h->last_rows, last_rows, batch * sizeof(RowInfo))))
    return fail(h, rc, t_err);
  cudaEventRecord(h->stage_ev[slot], h->stream);

  int ev = prof_begin(h, VLA_KCLASS_OTHER);
  rc = assemble_launch(h->rows, static_cast<int>(total), static_cast<const bf16*>(visual), token_ids,
                       h->pending, h->embed, c.d_model, c.vocab, h->h, h->status, h->stream);
  prof_end(h, ev, VLA_KCLASS_OTHER, 0, 6.0 * total * c.d_model);
  if (rc) return fail(h, rc, t_err);
  // the last layer runs past q|k|v only for each env's final row, straight into h_last
  if ((rc = forward_layers(h, static_cast<int>(total), h->rows, false, n_tiles, tile_rows, 0, &lr))) return rc;

  for (int b = 0; b < batch; ++b) {
    h->len[b] += chunk[b];
    h->len_prefill[b] = h->len[b];
    h->has_pending[b] = 0;
    h->prefilled[b] = 1;
  }
  h->active_batch = batch;
  h->entropy_valid = false;
  return VLA_OK;
}

static int check_turn_state(vla_handle* h, const char* who) {
  if (h->active_batch < 1) return fail(h, VLA_ERR_STATE, std::string(who) + ": no prefill yet");
  for (int b = 0; b < h->active_batch; ++b)
    if (!h->prefilled[b]) return fail(h, VLA_ERR_STATE, std::string(who) + ": env reset since the last prefill");
  return VLA_OK;
}

int vla_decode_actions(vla_handle* h, const float* uniforms, float temperature, const int32_t* forced_tokens,
                       int32_t* tokens_out, float* logprobs_out, float* actions_out, float* logits_out) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_decode_actions: NULL handle");
  if (!finite_nonneg(temperature)) return fail(h, VLA_ERR_ARG, "vla_decode_actions: temperature must be finite and >= 0");
  if ((temperature > 0.f && !uniforms) || !tokens_out || !logprobs_out || !actions_out)
    return fail(h, VLA_ERR_ARG, "vla_decode_actions: NULL buffer");
  int rc;
  if ((rc = check_turn_state(h, "vla_decode_actions"))) return rc;
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_decode_actions: set device"), t_err);
  const vla_config& c = h->cfg;
  const int B = h->active_batch, A = c.action_dim, d = c.d_model;

  // decode rows of steps 1..A-1: env b at position len_prefill[b] + i - 1, fed token of step i-1
  int slot;
  RowInfo* rows = static_cast<RowInfo*>(stage_slot(h, &slot));
  for (int i = 1; i < A; ++i)
    for (int b = 0; b < B; ++b)
      rows[(i - 1) * B + b] = RowInfo{b, h->len_prefill[b] + i - 1, ROW_TOKEN, b * A + (i - 1)};
  if ((rc = upload(h, h->rows, rows, static_cast<size_t>(A - 1) * B * sizeof(RowInfo)))) return fail(h, rc, t_err);
  cudaEventRecord(h->stage_ev[slot], h->stream);
  int max_len_p = 0;
  for (int b = 0; b < B; ++b) max_len_p = std::max(max_len_p, h->len_prefill[b]);

  HeadArgs ha;
  ha.z = h->head_z;
  ha.entropy_out = h->head_entropy;
  ha.B = B;
  ha.n_pos = 1;
  ha.A = A;
  ha.final_norm = h->final_norm;
  ha.head_rows = h->head_rows;
  ha.d = d;
  ha.ldh = d;
  ha.eps = c.rms_eps;
  ha.temperature = temperature;
  ha.uniforms = temperature > 0.f ? uniforms : nullptr;
  ha.forced = forced_tokens;
  ha.forced_base = c.vocab - 256;
  ha.token_base = c.vocab - 256;
  ha.tokens_out = tokens_out;
  ha.lp_out = logprobs_out;
  ha.act_out = actions_out;
  ha.logits_out = logits_out;
  ha.fed_out = h->fed;
  ha.status = h->status;

  for (int i = 0; i < A; ++i) {
    if (i > 0) {
      const RowInfo* rows_i = h->rows + static_cast<size_t>(i - 1) * B;
      int ev = prof_begin(h, VLA_KCLASS_OTHER);
      rc = assemble_launch(rows_i, B, nullptr, nullptr, h->fed, h->embed, d, c.vocab, h->h, h->status, h->stream);
      prof_end(h, ev, VLA_KCLASS_OTHER, 0, 6.0 * B * d);
      if (rc) return fail(h, rc, t_err);
      if ((rc = forward_layers(h, B, rows_i, true, 0, 0, max_len_p + i))) return rc;
    }
    ha.h = (i == 0) ? h->h_last : h->h;
    ha.step = i;
    int ev = prof_begin(h, VLA_KCLASS_HEAD);
    rc = action_head_launch(ha, h->stream);
    prof_end(h, ev, VLA_KCLASS_HEAD, 2.0 * B * 256 * d, 2.0 * 256 * d + 4.0 * B * d);
    if (rc) return fail(h, rc, t_err);
  }
  // the last token stays pending
  if (cudaMemcpy2DAsync(h->pending, sizeof(int), h->fed + (A - 1), A * sizeof(int), sizeof(int), B,
                        cudaMemcpyDeviceToDevice, h->stream) != cudaSuccess)
    return fail(h, cuda_fail(cudaGetLastError(), "pending copy"), t_err);
  for (int b = 0; b < B; ++b) {
    h->len[b] = h->len_prefill[b] + (A - 1);
    h->has_pending[b] = 1;
  }
  h->entropy_valid = true;
  return VLA_OK;
}

int vla_score_actions(vla_handle* h, const int32_t* tokens, float temperature, float* logprobs_out,
                      float* logits_out) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_score_actions: NULL handle");
  if (!finite_nonneg(temperature)) return fail(h, VLA_ERR_ARG, "vla_score_actions: temperature must be finite and >= 0");
  if (!tokens || !logprobs_out) return fail(h, VLA_ERR_ARG, "vla_score_actions: NULL buffer");
  int rc;
  if ((rc = check_turn_state(h, "vla_score_actions"))) return rc;
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_score_actions: set device"), t_err);
  const vla_config& c = h->cfg;
  const int B = h->active_batch, A = c.action_dim, d = c.d_model;
  const int n = A - 1;  // teacher-forced rows per env
  const int M = n * B;

  int slot;
  uint8_t* st = static_cast<uint8_t*>(stage_slot(h, &slot));
  RowInfo* rows = reinterpret_cast<RowInfo*>(st);
  AttnTile* tiles = reinterpret_cast<AttnTile*>(rows + M);
  int* sidx = reinterpret_cast<int*>(tiles + B);
  int* didx = sidx + M;
  int n_tiles = 0;
  for (int b = 0; b < B; ++b) {
    for (int j = 0; j < n; ++j) {
      rows[b * n + j] = RowInfo{b, h->len_prefill[b] + j, ROW_TOKEN, b * A + j};
      sidx[b * n + j] = b * n + j;
      didx[b * n + j] = b * A + 1 + j;
    }
    if (n > 0) tiles[n_tiles++] = AttnTile{b, b * n, n, h->len_prefill[b]};
  }
  if ((rc = upload(h, h->rows, rows, M * sizeof(RowInfo))) ||
      (rc = upload(h, h->tiles, tiles, n_tiles * sizeof(AttnTile))) ||
      (rc = upload(h, h->sidx, sidx, M * sizeof(int))) ||
      (rc = upload(h, h->didx, didx, M * sizeof(int))))
    return fail(h, rc, t_err);
  cudaEventRecord(h->stage_ev[slot], h->stream);

  if (M > 0) {
    int ev = prof_begin(h, VLA_KCLASS_OTHER);
    rc = assemble_launch(h->rows, M, nullptr, nullptr, tokens, h->embed, d, c.vocab, h->h, h->status, h->stream);
    prof_end(h, ev, VLA_KCLASS_OTHER, 0, 6.0 * M * d);
    if (rc) return fail(h, rc, t_err);
    if ((rc = forward_layers(h, M, h->rows, false, n_tiles, n, 0))) return rc;
  }
  // head inputs: row b*A = prefill's last hidden, rows b*A+1+j = chunk rows
  if (cudaMemcpy2DAsync(h->head_in, static_cast<size_t>(A) * d * sizeof(float), h->h_last, d * sizeof(float),
                        d * sizeof(float), B, cudaMemcpyDeviceToDevice, h->stream) != cudaSuccess)
    return fail(h, cuda_fail(cudaGetLastError(), "head input copy"), t_err);
  if (M > 0 && (rc = scatter_rows_launch(h->h, h->sidx, h->didx, M, d, h->head_in, h->stream)))
    return fail(h, rc, t_err);

  HeadArgs ha;
  ha.z = h->head_z;
  ha.entropy_out = h->head_entropy;
  ha.h = h->head_in;
  ha.ldh = d;
  ha.B = B;
  ha.n_pos = A;
  ha.step = 0;
  ha.A = A;
  ha.final_norm = h->final_norm;
  ha.head_rows = h->head_rows;
  ha.d = d;
  ha.eps = c.rms_eps;
  ha.temperature = temperature;
  ha.uniforms = nullptr;
  ha.forced = tokens;
  ha.forced_base = c.vocab - 256;
  ha.token_base = c.vocab - 256;
  ha.lp_out = logprobs_out;
  ha.logits_out = logits_out;
  ha.status = h->status;
  int ev = prof_begin(h, VLA_KCLASS_HEAD);
  rc = action_head_launch(ha, h->stream);
  prof_end(h, ev, VLA_KCLASS_HEAD, 2.0 * B * A * 256 * d, 2.0 * 256 * d + 4.0 * B * A * d);
  if (rc) return fail(h, rc, t_err);
  if (cudaMemcpy2DAsync(h->pending, sizeof(int), tokens + (A - 1), A * sizeof(int), sizeof(int), B,
                        cudaMemcpyDeviceToDevice, h->stream) != cudaSuccess)
    return fail(h, cuda_fail(cudaGetLastError(), "pending copy"), t_err);
  for (int b = 0; b < B; ++b) {
    h->len[b] = h->len_prefill[b] + (A - 1);
    h->has_pending[b] = 1;
  }
  h->entropy_valid = true;
  return VLA_OK;
}

int vla_reset(vla_handle* h, const uint8_t* env_mask) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_reset: NULL handle");
  for (int b = 0; b < h->cfg.max_batch; ++b) {
    if (env_mask && !env_mask[b]) continue;
    h->len[b] = 0;
    h->len_prefill[b] = 0;
    h->has_pending[b] = 0;
    h->prefilled[b] = 0;
  }
  h->entropy_valid = false;
  return VLA_OK;
}

int vla_action_entropy(vla_handle* h, float* entropy_out) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_action_entropy: NULL handle");
  if (!entropy_out) return fail(h, VLA_ERR_ARG, "vla_action_entropy: NULL buffer");
  int rc;
  if ((rc = check_turn_state(h, "vla_action_entropy"))) return rc;
  if (!h->entropy_valid) return fail(h, VLA_ERR_STATE, "vla_action_entropy: no decode or score since the prefill");
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_action_entropy: set device"), t_err);
  const size_t n = static_cast<size_t>(h->active_batch) * h->cfg.action_dim;
  if (cudaMemcpyAsync(entropy_out, h->head_entropy, n * sizeof(float), cudaMemcpyDeviceToDevice, h->stream) !=
      cudaSuccess)
    return fail(h, cuda_fail(cudaGetLastError(), "entropy copy"), t_err);
  return VLA_OK;
}

int vla_value(vla_handle* h, const void* w_value, float bias, float* values_out) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_value: NULL handle");
  if (!w_value || !values_out || !std::isfinite(bias)) return fail(h, VLA_ERR_ARG, "vla_value: bad argument");
  int rc;
  if ((rc = check_turn_state(h, "vla_value"))) return rc;
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_value: set device"), t_err);
  const vla_config& c = h->cfg;
  rc = value_head_launch(h->h_last, c.d_model, h->active_batch, c.d_model, h->final_norm,
                         static_cast<const bf16*>(w_value), c.rms_eps, bias, values_out, h->stream);
  if (rc) return fail(h, rc, t_err);
  return VLA_OK;
}

int vla_gae(const float* rewards, const float* values, const float* dones, int M, int B, float gamma, float lam,
            float* adv_out, float* returns_out, void* cuda_stream) {
  if (!rewards || !values || !dones || !adv_out || M < 1 || B < 1 || !(gamma >= 0.f && gamma <= 1.f) ||
      !(lam >= 0.f && lam <= 1.f))
    return set_err(nullptr, VLA_ERR_ARG, "vla_gae: bad argument");
  const int rc = gae_launch(rewards, values, dones, M, B, gamma, lam, adv_out, returns_out,
                            static_cast<cudaStream_t>(cuda_stream));
  return rc;
}

int vla_ppo_clip(const float* lp_new, const float* lp_old, const float* adv, int N, int A, float eps,
                 float* objective_out, float* ratio_out, float* clip_frac_out, void* cuda_stream) {
  if (!lp_new || !lp_old || !adv || !objective_out || N < 1 || A < 1 || !(eps >= 0.f) || !std::isfinite(eps))
    return set_err(nullptr, VLA_ERR_ARG, "vla_ppo_clip: bad argument");
  return ppo_clip_launch(lp_new, lp_old, adv, N, A, eps, objective_out, ratio_out, clip_frac_out,
                         static_cast<cudaStream_t>(cuda_stream));
}

int vla_sync(vla_handle* h) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_sync: NULL handle");
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_sync: set device"), t_err);
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e != cudaSuccess) return fail(h, cuda_fail(e, "vla_sync: stream"), t_err);
  uint32_t st = 0;
  e = cudaMemcpy(&st, h->status, sizeof(uint32_t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail(h, cuda_fail(e, "vla_sync: status read"), t_err);
  if (st) {
    cudaMemset(h->status, 0, sizeof(uint32_t));
    std::string msg = "device status:";
    if (st & VLA_STATUS_BAD_TOKEN) msg += " token id out of range;";
    if (st & VLA_STATUS_NONFINITE) msg += " non-finite logit;";
    if (st & VLA_STATUS_TIMEOUT) msg += " GEMM pipeline wait timed out;";
    if (st & VLA_STATUS_BAD_FORCED) msg += " forced/scored token is not an action-bin id;";
    if (st & VLA_STATUS_SATURATED) msg += " an activation beyond the fp16 range was saturated;";
    char buf[32];
    snprintf(buf, sizeof(buf), " (0x%x)", st);
    return fail(h, VLA_ERR_DEVICE_STATUS, msg + buf);
  }
  return VLA_OK;
}

int vla_sync_weights(vla_handle* h) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_sync_weights: NULL handle");
  DeviceGuard dev_guard(h->dev);
  if (dev_guard.err != cudaSuccess) return fail(h, cuda_fail(dev_guard.err, "vla_sync_weights: set device"), t_err);
  const int rc = convert_weights(h);
  if (rc) return fail(h, rc, t_err);
  return VLA_OK;
}

int vla_context_length(const vla_handle* h, int env) {
  if (!h || env < 0 || env >= h->cfg.max_batch) return -1;
  return h->len[env];
}

const char* vla_last_error(const vla_handle* h) { return h ? h->err.c_str() : t_err.c_str(); }

void vla_destroy(vla_handle* h) {
  if (!h) return;
  DeviceGuard dev_guard(h->dev);  // best effort: the handle is freed whatever happens
  cudaStreamSynchronize(h->stream);
  void* bufs[] = {h->kv, h->kv_res, h->h, h->y, h->q, h->ao, h->u, h->ws, h->h_last, h->head_in, h->head_z, h->head_entropy, h->q_last, h->ss_part, h->last_rows, h->rope,
                  h->rows, h->tiles, h->sidx, h->didx, h->fed, h->pending, h->status, h->part_o,
                  h->part_ml, h->attn_tickets, h->w16, h->w16_range};
  for (void* p : bufs)
    if (p) cudaFree(p);
  for (int s = 0; s < vla_handle::kSlots; ++s) {
    if (h->stage_host[s]) cudaFreeHost(h->stage_host[s]);
    if (h->stage_ev[s]) cudaEventDestroy(h->stage_ev[s]);
  }
  for (auto& e : h->ev_used) {
    cudaEventDestroy(e.a);
    cudaEventDestroy(e.b);
  }
  for (auto& e : h->ev_free) {
    cudaEventDestroy(e.a);
    cudaEventDestroy(e.b);
  }
  delete h;
}

int vla_profile(vla_handle* h, uint32_t class_mask) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_profile: NULL handle");
  prof_harvest(h);
  h->prof_mask = class_mask;
  for (int i = 0; i < VLA_KCLASS_COUNT; ++i) {
    h->prof_launches[i] = 0;
    h->prof_ms[i] = h->prof_flops[i] = h->prof_bytes[i] = 0.0;
  }
  return VLA_OK;
}

int vla_profile_read(vla_handle* h, int64_t* launches, double* ms, double* flops, double* bytes) {
  if (!h) return set_err(nullptr, VLA_ERR_ARG, "vla_profile_read: NULL handle");
  prof_harvest(h);
  for (int i = 0; i < VLA_KCLASS_COUNT; ++i) {
    if (launches) launches[i] = h->prof_launches[i];
    if (ms) ms[i] = h->prof_ms[i];
    if (flops) flops[i] = h->prof_flops[i];
    if (bytes) bytes[i] = h->prof_bytes[i];
  }
  return VLA_OK;
}

int64_t vla_launch_count(const vla_handle* h) {
  return h ? g_launch_count - h->launches_at_create : g_launch_count;
}

// ---------------------------------------------------------------------------------- ops
}  // extern "C"

namespace {
// The GEMM op entry points, bf16 (fp16 == false) or fp16 operands.
int op_gemm(const std::string& name, bool fp16, const void* A, const void* A_lo, int lda, const void* W,
            int ldw, float* C, int ldc, int M, int N, int K, int block_n, int splits, float* workspace,
            void* cuda_stream) {
  if (!A || !W || !C || M < 1 || N < 1 || K < 1 || ldc < N)
    return set_err(nullptr, VLA_ERR_ARG, name + ": bad argument");
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
  g.workspace = workspace;
  g.workspace_bytes = workspace ? gemm_workspace_bytes(g) : 0;
  g.epi.kind = EPI_F32;
  g.epi.out_f32 = C;
  g.epi.ldo = ldc;
  g.epi.fp16 = fp16;
  if (splits > 1 && gemm_effective_splits(K, splits) > 1 && !workspace)
    return set_err(nullptr, VLA_ERR_ARG, name + ": splits > 1 needs a workspace");
  if (const int rs = op_status_word(&g.epi.status)) return rs;
  const int rc = gemm_launch(g, static_cast<cudaStream_t>(cuda_stream), query_num_sms(), nullptr);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA) return set_err(nullptr, rc, name + ": unsupported arguments");
  return rc;
}

int op_gemm_pair(const std::string& name, bool fp16, const void* A, const void* A_lo, int lda, const void* W,
                 int ldw, float* C, int ldc, int M, int N, int K, void* cuda_stream) {
  if (!A || !W || !C || M < 1 || N < 1 || K < 1 || ldc < N)
    return set_err(nullptr, VLA_ERR_ARG, name + ": bad argument");
  GemmArgs g;
  g.A = static_cast<const bf16*>(A);
  g.A_lo = static_cast<const bf16*>(A_lo);
  g.lda = lda;
  g.B = static_cast<const bf16*>(W);
  g.ldb = ldw;
  g.M = M;
  g.N = N;
  g.K = K;
  g.block_n = 256;
  g.splits = 1;
  g.pair = true;
  g.epi.kind = EPI_F32;
  g.epi.out_f32 = C;
  g.epi.ldo = ldc;
  g.epi.fp16 = fp16;
  if (const int rs = op_status_word(&g.epi.status)) return rs;
  const int rc = gemm_launch(g, static_cast<cudaStream_t>(cuda_stream), query_num_sms(), nullptr);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA) return set_err(nullptr, rc, name + ": unsupported arguments");
  return rc;
}

int op_gemm_decode(const std::string& name, bool fp16, const void* A, const void* A_lo, int lda, const void* W,
                   int ldw, float* C, int ldc, int M, int N, int K, float* workspace, size_t workspace_bytes,
                   void* cuda_stream) {
  if (!A || !A_lo || !W || !C || M < 1 || M > 128 || N < 1 || K < 1 || ldc < N || !workspace)
    return set_err(nullptr, VLA_ERR_ARG, name + ": bad argument");
  GemmArgs g;
  g.A = static_cast<const bf16*>(A);
  g.A_lo = static_cast<const bf16*>(A_lo);
  g.lda = lda;
  g.B = static_cast<const bf16*>(W);
  g.ldb = ldw;
  g.M = M;
  g.N = N;
  g.K = K;
  g.workspace = workspace;
  g.workspace_bytes = workspace_bytes;
  g.epi.kind = EPI_F32;
  g.epi.out_f32 = C;
  g.epi.ldo = ldc;
  g.epi.fp16 = fp16;
  if (const int rs = op_status_word(&g.epi.status)) return rs;
  const int rc = gemv_launch(g, static_cast<cudaStream_t>(cuda_stream), query_num_sms(), nullptr);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA)
    return set_err(nullptr, rc, name + ": unsupported arguments or workspace too small");
  return rc;
}
}  // namespace

extern "C" {

int vla_op_gemm_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C, int ldc,
                     int M, int N, int K, int block_n, int splits, float* workspace, void* cuda_stream) {
  return op_gemm("vla_op_gemm_bf16", false, A, A_lo, lda, W, ldw, C, ldc, M, N, K, block_n, splits, workspace,
                 cuda_stream);
}

int vla_op_gemm_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C, int ldc,
                    int M, int N, int K, int block_n, int splits, float* workspace, void* cuda_stream) {
  return op_gemm("vla_op_gemm_f16", true, A, A_lo, lda, W, ldw, C, ldc, M, N, K, block_n, splits, workspace,
                 cuda_stream);
}

int vla_op_gemm_pair_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C, int ldc,
                          int M, int N, int K, void* cuda_stream) {
  return op_gemm_pair("vla_op_gemm_pair_bf16", false, A, A_lo, lda, W, ldw, C, ldc, M, N, K, cuda_stream);
}

int vla_op_gemm_pair_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C, int ldc,
                         int M, int N, int K, void* cuda_stream) {
  return op_gemm_pair("vla_op_gemm_pair_f16", true, A, A_lo, lda, W, ldw, C, ldc, M, N, K, cuda_stream);
}

int vla_op_gemm_decode_bf16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C,
                            int ldc, int M, int N, int K, float* workspace, size_t workspace_bytes,
                            void* cuda_stream) {
  return op_gemm_decode("vla_op_gemm_decode_bf16", false, A, A_lo, lda, W, ldw, C, ldc, M, N, K, workspace,
                        workspace_bytes, cuda_stream);
}

int vla_op_gemm_decode_f16(const void* A, const void* A_lo, int lda, const void* W, int ldw, float* C,
                           int ldc, int M, int N, int K, float* workspace, size_t workspace_bytes,
                           void* cuda_stream) {
  return op_gemm_decode("vla_op_gemm_decode_f16", true, A, A_lo, lda, W, ldw, C, ldc, M, N, K, workspace,
                        workspace_bytes, cuda_stream);
}

size_t vla_op_gemm_decode_workspace_bytes(int M, int N, int K) {
  return gemv_workspace_bytes(M, N, K, query_num_sms());
}

int vla_op_action_head(const float* hs, int ldh, int B, int d, const void* final_norm, const void* head_rows,
                       float eps, const float* uniforms, float temperature, const int32_t* forced,
                       int32_t* bins_out, float* logprobs_out, float* actions_out, float* logits_out,
                       uint32_t* status, void* cuda_stream) {
  if (!hs || B < 1 || d < 8 || ldh < d || !final_norm || !head_rows || !logprobs_out || !logits_out || !status ||
      !finite_nonneg(temperature) || (temperature > 0.f && !uniforms))
    return set_err(nullptr, VLA_ERR_ARG, "vla_op_action_head: bad argument");
  HeadArgs ha;
  ha.z = logits_out;
  ha.h = hs;
  ha.ldh = ldh;
  ha.B = B;
  ha.n_pos = 1;
  ha.step = 0;
  ha.A = 1;
  ha.final_norm = static_cast<const bf16*>(final_norm);
  ha.head_rows = static_cast<const bf16*>(head_rows);
  ha.d = d;
  ha.eps = eps;
  ha.temperature = temperature;
  ha.uniforms = temperature > 0.f ? uniforms : nullptr;
  ha.forced = forced;
  ha.forced_base = 0;
  ha.token_base = 0;
  ha.bins_out = bins_out;
  ha.lp_out = logprobs_out;
  ha.act_out = actions_out;
  ha.logits_out = logits_out;
  ha.status = status;
  return action_head_launch(ha, static_cast<cudaStream_t>(cuda_stream));
}

static const int kOpAttnChunk = 320;

size_t vla_op_attn_decode_workspace_bytes(int B, int H, int hd, int max_ctx, int max_keys_per_cta) {
  if (B < 1 || H < 1 || hd < 1 || max_ctx < 1) return 0;
  const int chunk = max_keys_per_cta > 0 ? max_keys_per_cta : kOpAttnChunk;
  const size_t S = (static_cast<size_t>(max_ctx) + chunk - 1) / chunk;
  // RowInfo table, then partial outputs, (max, sum) pairs and the per-(env, head) tickets
  return static_cast<size_t>(B) * sizeof(RowInfo) + 256 + static_cast<size_t>(B) * H * S * hd * sizeof(float) +
         256 + static_cast<size_t>(B) * H * S * sizeof(float2) + 256 + static_cast<size_t>(B) * H * sizeof(int) +
         256 + 256;
}

static int op_attn_decode(const char* name, const float* q, const void* kv, const void* kv_res, int max_env, int H,
                          int hd, int cap, const int32_t* env, const int32_t* pos, int B, int max_ctx,
                          int max_keys_per_cta, void* out_hi, void* out_lo, float* workspace, size_t workspace_bytes,
                          void* cuda_stream) {
  const int chunk = max_keys_per_cta > 0 ? max_keys_per_cta : kOpAttnChunk;
  if ((reinterpret_cast<uintptr_t>(kv) & 15) || (reinterpret_cast<uintptr_t>(kv_res) & 15))
    return set_err(nullptr, VLA_ERR_ARG, std::string(name) + ": misaligned cache");
  if (!q || !kv || !env || !pos || !out_hi || !out_lo || !workspace || B < 1 || H < 1 || cap < 1 ||
      max_env < 1 || max_ctx < 1 || max_ctx > cap || (hd != 64 && hd != 128) || chunk < 16 ||
      workspace_bytes < vla_op_attn_decode_workspace_bytes(B, H, hd, max_ctx, chunk))
    return set_err(nullptr, VLA_ERR_ARG, std::string(name) + ": bad argument");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  // Row table from env / pos (a strided device copy each, no host round trip).
  RowInfo* rows = reinterpret_cast<RowInfo*>(workspace);
  if (cudaMemsetAsync(rows, 0, static_cast<size_t>(B) * sizeof(RowInfo), st) != cudaSuccess ||
      cudaMemcpy2DAsync(&rows[0].env, sizeof(RowInfo), env, sizeof(int32_t), sizeof(int32_t), B,
                        cudaMemcpyDeviceToDevice, st) != cudaSuccess ||
      cudaMemcpy2DAsync(&rows[0].pos, sizeof(RowInfo), pos, sizeof(int32_t), sizeof(int32_t), B,
                        cudaMemcpyDeviceToDevice, st) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), (std::string(name) + ": row table").c_str());
  char* base = reinterpret_cast<char*>(workspace) + ((static_cast<size_t>(B) * sizeof(RowInfo) + 255) / 256) * 256;
  const size_t S = (static_cast<size_t>(max_ctx) + chunk - 1) / chunk;
  float* part_o = reinterpret_cast<float*>(base);
  char* ml_base = base + ((static_cast<size_t>(B) * H * S * hd * sizeof(float) + 255) / 256) * 256;
  float2* part_ml = reinterpret_cast<float2*>(ml_base);
  int* counters = reinterpret_cast<int*>(ml_base + ((static_cast<size_t>(B) * H * S * sizeof(float2) + 255) / 256) * 256);
  if (cudaMemsetAsync(counters, 0, static_cast<size_t>(B) * H * sizeof(int), st) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), (std::string(name) + ": tickets").c_str());
  KVLayout L{};
  L.base = static_cast<f16*>(const_cast<void*>(kv));
  L.res = static_cast<uint8_t*>(const_cast<void*>(kv_res));
  L.cap = cap;
  L.head_stride = static_cast<int64_t>(cap) * hd;
  L.kv_stride = static_cast<int64_t>(H) * L.head_stride;
  L.env_stride = 2 * L.kv_stride;
  L.layer_stride = static_cast<int64_t>(max_env) * L.env_stride;
  const int rc = attn_decode_launch(q, static_cast<bf16*>(out_hi), static_cast<bf16*>(out_lo), rows, B, max_ctx, L,
                                    0, H, hd, chunk, part_o, part_ml, counters, st, false);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA) return set_err(nullptr, rc, std::string(name) + ": unsupported arguments");
  return rc;
}

int vla_op_attn_decode(const float* q, const void* kv, int max_env, int H, int hd, int cap, const int32_t* env,
                       const int32_t* pos, int B, int max_ctx, int max_keys_per_cta, void* out_hi, void* out_lo,
                       float* workspace, size_t workspace_bytes, void* cuda_stream) {
  return op_attn_decode("vla_op_attn_decode", q, kv, nullptr, max_env, H, hd, cap, env, pos, B, max_ctx,
                        max_keys_per_cta, out_hi, out_lo, workspace, workspace_bytes, cuda_stream);
}

int vla_op_attn_decode_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd, int cap,
                           const int32_t* env, const int32_t* pos, int B, int max_ctx, int max_keys_per_cta,
                           void* out_hi, void* out_lo, float* workspace, size_t workspace_bytes, void* cuda_stream) {
  if (!kv_res) return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_decode_res: bad argument");
  return op_attn_decode("vla_op_attn_decode_res", q, kv, kv_res, max_env, H, hd, cap, env, pos, B, max_ctx,
                        max_keys_per_cta, out_hi, out_lo, workspace, workspace_bytes, cuda_stream);
}

int vla_op_attn_chunk(const float* q, const void* kv, int max_env, int H, int hd, int cap,
                      const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev, void* out_hi,
                      void* out_lo, void* cuda_stream) {
  if (!q || !kv || !tiles_host || !tiles_dev || !out_hi || !out_lo || max_env < 1 || H < 1 || cap < 1 ||
      n_tiles < 1 || rows < 1 || (hd != 64 && hd != 128))
    return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_chunk: bad argument");
  for (int i = 0; i < n_tiles; ++i) {
    const int32_t* t = tiles_host + 4 * i;
    if (t[0] < 0 || t[0] >= max_env || t[2] < 1 || t[2] > 64 || t[3] < 0 || t[3] + t[2] > cap || t[1] < 0 ||
        t[1] + t[2] > rows)
      return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_chunk: tile outside the buffers");
  }
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemcpyAsync(tiles_dev, tiles_host, static_cast<size_t>(n_tiles) * 4 * sizeof(int32_t),
                      cudaMemcpyHostToDevice, st) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "vla_op_attn_chunk: tile copy");
  KVLayout L{};
  L.base = static_cast<f16*>(const_cast<void*>(kv));
  L.cap = cap;
  L.head_stride = static_cast<int64_t>(cap) * hd;
  L.kv_stride = static_cast<int64_t>(H) * L.head_stride;
  L.env_stride = 2 * L.kv_stride;
  L.layer_stride = static_cast<int64_t>(max_env) * L.env_stride;
  const int rc = attn_chunk_launch(q, static_cast<bf16*>(out_hi), static_cast<bf16*>(out_lo),
                                   reinterpret_cast<const AttnTile*>(tiles_dev), n_tiles, L, 0, H, hd, st, false);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA) return set_err(nullptr, rc, "vla_op_attn_chunk: unsupported arguments");
  return rc;
}

int vla_op_attn_chunk_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd, int cap,
                          const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev, void* out_hi,
                          void* out_lo, void* cuda_stream) {
  if (!q || !kv || !kv_res || !tiles_host || !tiles_dev || !out_hi || !out_lo || max_env < 1 || H < 1 || cap < 1 ||
      n_tiles < 1 || rows < 1 || (hd != 64 && hd != 128))
    return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_chunk_res: bad argument");
  for (int i = 0; i < n_tiles; ++i) {
    const int32_t* t = tiles_host + 4 * i;
    if (t[0] < 0 || t[0] >= max_env || t[2] < 1 || t[2] > 128 || t[3] < 0 || t[3] + t[2] > cap || t[1] < 0 ||
        t[1] + t[2] > rows)
      return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_chunk_res: tile outside the buffers");
  }
  uint32_t* status = nullptr;
  if (const int rs = op_status_word(&status)) return rs;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemcpyAsync(tiles_dev, tiles_host, static_cast<size_t>(n_tiles) * 4 * sizeof(int32_t),
                      cudaMemcpyHostToDevice, st) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "vla_op_attn_chunk_res: tile copy");
  KVLayout L{};
  L.base = static_cast<f16*>(const_cast<void*>(kv));
  L.res = static_cast<uint8_t*>(const_cast<void*>(kv_res));
  L.cap = cap;
  L.head_stride = static_cast<int64_t>(cap) * hd;
  L.kv_stride = static_cast<int64_t>(H) * L.head_stride;
  L.env_stride = 2 * L.kv_stride;
  L.layer_stride = static_cast<int64_t>(max_env) * L.env_stride;
  const int rc = attn_chunk_tc_launch(q, static_cast<bf16*>(out_hi), static_cast<bf16*>(out_lo),
                                      reinterpret_cast<const AttnTile*>(tiles_dev), n_tiles, L, 0, H, hd, status, st,
                                      false, query_num_sms(), true);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA)
    return set_err(nullptr, rc, "vla_op_attn_chunk_res: unsupported arguments or misaligned buffers");
  return rc;
}

int vla_op_attn_rows_res(const float* q, const void* kv, const void* kv_res, int max_env, int H, int hd, int cap,
                         const int32_t* tiles_host, int n_tiles, int rows, int32_t* tiles_dev, void* out_hi,
                         void* out_lo, void* cuda_stream) {
  if (!q || !kv || !kv_res || !tiles_host || !tiles_dev || !out_hi || !out_lo || max_env < 1 || H < 1 || cap < 1 ||
      n_tiles < 1 || rows < 1 || (hd != 64 && hd != 128))
    return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_rows_res: bad argument");
  for (int i = 0; i < n_tiles; ++i) {
    const int32_t* t = tiles_host + 4 * i;
    if (t[0] < 0 || t[0] >= max_env || t[2] < 1 || t[2] > kAttnRowsMax || t[3] < 0 || t[3] + t[2] > cap ||
        t[1] < 0 || t[1] + t[2] > rows)
      return set_err(nullptr, VLA_ERR_ARG, "vla_op_attn_rows_res: tile outside the buffers or over 16 rows");
  }
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  if (cudaMemcpyAsync(tiles_dev, tiles_host, static_cast<size_t>(n_tiles) * 4 * sizeof(int32_t),
                      cudaMemcpyHostToDevice, st) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "vla_op_attn_rows_res: tile copy");
  KVLayout L{};
  L.base = static_cast<f16*>(const_cast<void*>(kv));
  L.res = static_cast<uint8_t*>(const_cast<void*>(kv_res));
  L.cap = cap;
  L.head_stride = static_cast<int64_t>(cap) * hd;
  L.kv_stride = static_cast<int64_t>(H) * L.head_stride;
  L.env_stride = 2 * L.kv_stride;
  L.layer_stride = static_cast<int64_t>(max_env) * L.env_stride;
  const int rc = attn_rows_launch(q, static_cast<bf16*>(out_hi), static_cast<bf16*>(out_lo),
                                  reinterpret_cast<const AttnTile*>(tiles_dev), n_tiles, L, 0, H, hd, st, false, true);
  if (rc != VLA_OK && rc != VLA_ERR_CUDA)
    return set_err(nullptr, rc, "vla_op_attn_rows_res: unsupported arguments or misaligned buffers");
  return rc;
}

int vla_op_num_sms(void) { return query_num_sms(); }

int vla_op_rmsnorm(const float* hs, int ldh, int M, int d, const void* w, float eps, void* y_hi, void* y_lo,
                   int fp16, void* cuda_stream) {
  if (!hs || !w || !y_hi || !y_lo || M < 1 || d < 4 || (d & 3) || ldh < d || (ldh & 3) || !(eps >= 0.f) ||
      (reinterpret_cast<uintptr_t>(hs) & 15) || (reinterpret_cast<uintptr_t>(w) & 7) ||
      (reinterpret_cast<uintptr_t>(y_hi) & 7) || (reinterpret_cast<uintptr_t>(y_lo) & 7))
    return set_err(nullptr, VLA_ERR_ARG, "vla_op_rmsnorm: bad argument");
  uint32_t* status = nullptr;
  if (const int rs = op_status_word(&status)) return rs;
  return rmsnorm_launch(hs, ldh, static_cast<const bf16*>(w), M, d, eps, static_cast<bf16*>(y_hi),
                        static_cast<bf16*>(y_lo), static_cast<cudaStream_t>(cuda_stream), fp16 != 0, status);
}

int vla_op_read_status(void* cuda_stream, uint32_t* status_out) {
  if (!status_out) return set_err(nullptr, VLA_ERR_ARG, "vla_op_read_status: NULL status_out");
  uint32_t* word = nullptr;
  if (const int rs = op_status_word(&word)) return rs;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  VLA_CUDA_TRY(cudaMemcpyAsync(status_out, word, sizeof(uint32_t), cudaMemcpyDeviceToHost, st));
  VLA_CUDA_TRY(cudaMemsetAsync(word, 0, sizeof(uint32_t), st));
  VLA_CUDA_TRY(cudaStreamSynchronize(st));
  return VLA_OK;
}

// ------------------------------------------------------------------- failure injection (tests)
int vla_test_inject_launch_error(int64_t nth_launch, int cuda_error) {
  if (nth_launch < 0 || (nth_launch > 0 && cuda_error == 0))
    return set_err(nullptr, VLA_ERR_ARG, "vla_test_inject_launch_error: bad argument");
  g_inject_error.store(cuda_error);
  g_inject_countdown.store(nth_launch);
  return VLA_OK;
}

int vla_test_set_wait_limit_ns(uint64_t limit_ns) {
  g_wait_limit_ns.store(limit_ns ? limit_ns : kDefaultWaitLimitNs);
  return VLA_OK;
}

int vla_test_stall_next_gemm(void) {
  gemm_stall_next_launch();
  return VLA_OK;
}

}  // extern "C"
