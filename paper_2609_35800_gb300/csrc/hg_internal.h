// Launch parameter blocks and launcher entry points shared between the host
// runtime (hg_api.cu) and the kernel translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/headguard.h"
#include "hg_layout.cuh"

namespace hg {

// Per-layer placement: byte offset of the layer block in the arena and the
// layer's protection mask (bit h = KV head h protected).
struct LayerTable {
  uint64_t base[kMaxLayersPerLaunch];
  uint64_t mask[kMaxLayersPerLaunch];
};

struct QuantizeParams {
  Dims d;
  char* arena;
  int n_layers;
  int tile_origin;  // s mod 32: KIVI-style tile i covers [tile_origin - 32 + 64 i, +64) clipped to [0, T)
  LayerTable lt;
  const uint16_t* k[kMaxLayersPerLaunch];
  const uint16_t* v[kMaxLayersPerLaunch];
};

struct DequantParams {
  Dims d;
  const char* arena;
  int n_layers;
  LayerTable lt;
  int appended;  // appended tokens, the same in every layer of the launch
  int out_fp32;
  void* k_out;   // [n_layers][B][H][T + appended][128]
  void* v_out;
};

struct AppendParams {
  Dims d;
  char* arena;
  int n_layers;
  LayerTable lt;
  int appended[kMaxLayersPerLaunch];
  const uint16_t* k_new;  // [n_layers][B][H][128]
  const uint16_t* v_new;
};

// Decode work plan of one launch.  Each (layer, row, head) segment is cut into
// chunks of a fixed token count per segment kind; a CTA processes one chunk.
//   cbU  BF16 tokens of quantized / keys-only heads   (text, uncoded image, appended)
//   cqU  coded tokens of quantized heads               (codes for K and V)
//   cqK  coded tokens of keys-only heads               (BF16 K, coded V)
//   cbP  BF16 tokens of protected K+V heads
// Per layer, the host passes the resulting chunk counts of each kind.
struct DecodePlan {
  int cbU, cqU, cqK, cbP;
};

struct DecodeLayer {
  int appended;
  int nbU, nqU, nqK, nbP;  // chunks per head of each kind
  int items_per_row;       // chunks of all heads of one batch row
  int item_base;           // first work item of this layer in the launch
};

// Largest launch whose CTAs get a host-chosen item order.
constexpr int kMaxOrderedItems = 1024;
// Packed work item: layer in the launch (6 bits), KV head (6), chunk of the
// head (5), batch row (15).
HG_HD uint32_t order_record(int li, int b, int h, int r) {
  return (uint32_t)li | ((uint32_t)h << 6) | ((uint32_t)r << 12) | ((uint32_t)b << 17);
}
constexpr int kOrderMaxRow = 1 << 15, kOrderMaxChunk = 1 << 5;

struct DecodeParams {
  // The arena as a two-dimensional BF16 tensor [arena_bytes / 256][128]: every
  // BF16 token row of the cache is one row of it.  Boxes of kArenaBoxRows rows
  // x 64 channels, 128-byte swizzle.
  CUtensorMap arena_map;
  Dims d;
  const char* arena;
  int n_layers;
  DecodePlan plan;
  int max_items;       // split slots per (layer, row, head) in the workspace
  float scale_log2;    // softmax_scale * log2(e)
  const uint16_t* q;   // [n_layers][B][Hq][128]
  uint16_t* out;       // [n_layers][B][Hq][128]
  // Fused append (or null): the step's new K/V [n_layers][B][H][128], already
  // counted in `appended`; the chunk that holds the new position reads it from
  // here and writes it into the arena.
  const uint16_t* k_new;
  const uint16_t* v_new;
  int total_items;
  uint32_t* status;    // workspace status word (kStatus* bits; zero while healthy)
  uint32_t* counters;  // [n_layers][B][H]
  float* partials;     // [n_layers][B][H][max_items][G][132]
  LayerTable lt;
  DecodeLayer layer[kMaxLayersPerLaunch];
  // Work item of each CTA below n_order, as a packed record (order_record):
  // the kernel reads its item's coordinates instead of searching the layer
  // and head tables.  CTAs from n_order on take item blockIdx.x.
  int n_order;
  uint32_t order[kMaxOrderedItems];
};

// BF16 rows per TMA box of the arena tensor map.
constexpr int kArenaBoxRows = 16;

cudaError_t launch_quantize(const QuantizeParams& p, cudaStream_t s);
// Salient-token maps (AKVQ-style, Sec. 4) of every quantized head of the
// launch's layers, from the prefill keys; run before launch_quantize.
cudaError_t launch_salient(const QuantizeParams& p, cudaStream_t s);
// Shared memory of the salient selection: a score per image token plus a
// bit per image token.
inline size_t salient_smem_bytes(const Dims& d) { return (size_t)d.nq * 4 + (size_t)sal_blocks(d) * 4; }
constexpr size_t kMaxSalientSmem = 200 * 1024;
// Reconstruction of the launch's layers; sm_count sizes the tile spans.
cudaError_t launch_dequantize(const DequantParams& p, int sm_count, cudaStream_t s);
cudaError_t launch_append(const AppendParams& p, cudaStream_t s);
cudaError_t launch_decode(const DecodeParams& p, int grid_x, cudaStream_t s);
cudaError_t launch_wait_probe(uint32_t* result, uint32_t rounds, cudaStream_t s);
// The decode kernels for binary16 metadata pairs (called by launch_decode).
cudaError_t launch_decode_m16(const DecodeParams& p, int grid_x, cudaStream_t s);
// Most splits of one head the decode kernel's merge can take.
int decode_max_splits(int G);

// Decode attention with a scratch array as its workspace (the allocation-free
// entry point): the argument checks of hg_decode_attention and the arena's
// tensor map first, then a clear of the split counters only (the status word
// is left as the previous calls left it), then the launch.
hg_status decode_attention_on_scratch(const hg_cache* cache, int32_t layer_begin, int32_t layer_count,
                                      const void* q, void* out, float softmax_scale, void* scratch,
                                      size_t scratch_bytes, hg_stream_t stream);
// Device address of the allocation-free entry point's scratch array on the
// current device (its first 512 bytes are a workspace header with the status
// word at byte 0).
hg_status noalloc_scratch_address(void** out);

}  // namespace hg
