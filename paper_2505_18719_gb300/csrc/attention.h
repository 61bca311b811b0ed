// Internal interface of the attention kernels (attention.cu).
#pragma once
#include "common.cuh"

namespace vla {

// A tile of up to 64 consecutive query rows of one env: packed rows row0 .. row0+nrows-1
// at positions pos0 .. pos0+nrows-1.
struct AttnTile {
  int env, row0, nrows, pos0;
};

// q: f32 [rows, H*hd]; out: hi/lo operand pair [rows, H*hd], fp16 if `fp16` else bf16; keys
// from the fp16 cache of `layer`.
int attn_chunk_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles,
                      int n_tiles, KVLayout kv, int layer, int H, int hd, cudaStream_t stream,
                      bool fp16);

// The same on the tcgen05 tensor cores with the cache read as fp16 + 4-bit residual (kv.res
// required): tiles of up to 128 rows; status gets VLA_STATUS_TIMEOUT if a pipeline wait runs out.
// write_lo = false leaves out_lo untouched (for a consumer that reads the hi plane alone).
int attn_chunk_tc_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles, int n_tiles,
                         KVLayout kv, int layer, int H, int hd, uint32_t* status, cudaStream_t stream, bool fp16,
                         int num_sms, bool write_lo);

// The same for tiles of at most 16 rows (kv.res required; not checked on the device: the caller
// guarantees nrows <= 16), on mma.sync with one CTA per (tile, head): each cached byte is read once
// per tile and head, with no padding rows beyond 16.  write_lo as attn_chunk_tc_launch.
constexpr int kAttnRowsMax = 16;
int attn_rows_launch(const float* q, bf16* out_hi, bf16* out_lo, const AttnTile* tiles, int n_tiles, KVLayout kv,
                     int layer, int H, int hd, cudaStream_t stream, bool fp16, bool write_lo);

// One query per env row b (rows[b] gives env and position); key range split into equal ranges
// of at most `chunk` keys (a multiple of 16 at least 16); partials in part_o [B*H*S*hd] f32 and part_ml [B*H*S]
// (S = ceil(max_ctx/chunk)); counters [B*H] int must be zero at launch and are zero again
// when the kernel completes.  The output pair is fp16 if `fp16`, else bf16.
int attn_decode_launch(const float* q, bf16* out_hi, bf16* out_lo, const RowInfo* rows, int B,
                       int max_ctx, KVLayout kv, int layer, int H, int hd, int chunk,
                       float* part_o, float2* part_ml, int* counters, cudaStream_t stream,
                       bool fp16);

}  // namespace vla
