// Launch parameter blocks and launcher entry points shared between the host
// runtime (hg_api.cu) and the kernel translation units.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

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
  int n_tiles;      // 32-token tiles per (row, head)
  int tile_origin;  // tile i covers [tile_origin - 32 + 32 i, +32) clipped to [0, T)
  LayerTable lt;
  const uint16_t* k[kMaxLayersPerLaunch];
  const uint16_t* v[kMaxLayersPerLaunch];
};

struct DequantParams {
  Dims d;
  const char* arena;
  uint64_t layer_base;
  uint64_t mask;
  int appended;
  int out_fp32;
  void* k_out;
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

struct DecodeParams {
  Dims d;
  const char* arena;
  int n_layers;
  int cb, cq;          // chunk sizes (tokens) for BF16 and coded segments
  int max_items;       // split slots per (layer, row, head) in the workspace
  float scale_log2;    // softmax_scale * log2(e)
  const uint16_t* q;   // [n_layers][B][Hq][128]
  uint16_t* out;       // [n_layers][B][Hq][128]
  uint32_t* counters;  // [n_layers][B][H]
  float* partials;     // [n_layers][B][H][max_items][G][130]
  LayerTable lt;
  int appended[kMaxLayersPerLaunch];
  int items_per_row[kMaxLayersPerLaunch];
};

cudaError_t launch_quantize(const QuantizeParams& p, cudaStream_t s);
cudaError_t launch_dequantize(const DequantParams& p, cudaStream_t s);
cudaError_t launch_append(const AppendParams& p, cudaStream_t s);
cudaError_t launch_decode(const DecodeParams& p, int grid_x, cudaStream_t s);

}  // namespace hg
