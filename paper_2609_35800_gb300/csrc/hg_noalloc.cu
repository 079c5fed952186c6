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
//
// The array is laid out as a decode workspace: a 512-byte header whose first
// word is the status word, the split counters, the split partials.  Every call
// clears the counters it uses; the status word is sticky (a wait that ran out
// in any call stays visible) until the caller clears it, and both are reached
// through hg_workspace_status / hg_workspace_clear with a null workspace.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/headguard.h"
#include "hg_internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(32) << 20;
constexpr int kMaxDevices = 64;

// The shared scratch (zero when the library's module is loaded).  In host code
// this name is only a stand-in for the device array, never a usable address;
// the address comes from cudaGetSymbolAddress below.
__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace hg {

// Device address of the scratch on the current device; looked up (and the
// library's module loaded) on the first call for that device.
hg_status noalloc_scratch_address(void** out) {
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

}  // namespace hg

extern "C" hg_status hg_decode_attention_noalloc(const hg_cache* cache, int32_t layer_begin,
                                                 int32_t layer_count, const void* q, void* out,
                                                 float softmax_scale, hg_stream_t stream) {
  // The host-side checks of hg_decode_attention that need no workspace, and
  // the size limit, before anything else.
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
  st = hg::noalloc_scratch_address(&scratch);
  if (st != HG_OK) return st;
  // The remaining checks, then a clear of the split counters (the array keeps
  // whatever the previous call left), then the launch.
  return hg::decode_attention_on_scratch(cache, layer_begin, layer_count, q, out, softmax_scale, scratch,
                                         kScratchBytes, stream);
}
