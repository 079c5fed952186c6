// Decode attention for callers that cannot allocate device memory.
//
// Some callers are handed only their input and output buffers and may not
// allocate anything else on the device: operators plugged into an inference
// runtime whose plugin interface offers no workspace, code running while
// another framework owns the whole device memory pool, or decode loops that
// cannot afford the implicit device synchronisation of cudaMalloc.  For them
// hg_decode_attention_noalloc uses, as its split-K workspace, one file-scope
// device array of kScratchBytes (32 MiB) that every GPU loading this library
// keeps until the process exits.  Nothing here calls cudaMalloc, cudaFree or
// any other allocating routine.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/headguard.h"

namespace {

constexpr size_t kScratchBytes = size_t(32) << 20;
constexpr int kMaxDevices = 64;

// The shared scratch.  In host code this name is only a stand-in for the
// device array, never a usable address; the address comes from
// cudaGetSymbolAddress below.
__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device; looked up (and the
// library's module loaded) on the first call for that device.
hg_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return HG_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return HG_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr) return HG_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return HG_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" hg_status hg_decode_attention_noalloc(const hg_cache* cache, int32_t layer_begin,
                                                 int32_t layer_count, const void* q, void* out,
                                                 float softmax_scale, hg_stream_t stream) {
  // Same argument checks as hg_decode_attention, done before anything is enqueued.
  if (!cache || layer_begin < 0 || layer_count < 1 || !q || !out) return HG_ERR_INVALID_ARG;
  if (hg_cache_appended(cache, layer_begin) < 0 ||
      hg_cache_appended(cache, layer_begin + layer_count - 1) < 0)
    return HG_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out)) return HG_ERR_ALIGNMENT;
  if (!(softmax_scale == softmax_scale)) return HG_ERR_INVALID_ARG;
  size_t need = 0;
  hg_status st = hg_decode_workspace_size(cache, layer_count, &need);
  if (st != HG_OK) return st;
  if (need > kScratchBytes) return HG_ERR_WORKSPACE_TOO_SMALL;
  void* scratch = nullptr;
  st = scratch_address(&scratch);
  if (st != HG_OK) return st;
  // The array keeps whatever the previous call left; the status word and the
  // split counters must start at zero.
  if (cudaMemsetAsync(scratch, 0, need, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return HG_ERR_CUDA;
  return hg_decode_attention(cache, layer_begin, layer_count, q, out, softmax_scale, scratch,
                             kScratchBytes, stream);
}
