// Host runtime of the HeadGuard C ABI (include/headguard.h): argument
// validation, arena layout, decode work decomposition and kernel launches.
// Every check runs before anything is enqueued; no device memory is
// allocated here.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <climits>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/headguard.h"
#include "hg_internal.h"
#include "hg_layout.cuh"

using namespace hg;

struct hg_cache {
  hg_shape shape;
  hg_quant_config cfg;
  Dims d;
  std::vector<uint64_t> layer_mask;
  std::vector<uint64_t> layer_base;
  std::vector<int> appended;
  char* arena;
  size_t arena_bytes;
  size_t needed_bytes;
  // The arena as a BF16 tensor [arena_bytes / 256][128] for the decode
  // kernel's TMA loads; encoded by the first decode call.
  mutable CUtensorMap arena_map;
  mutable bool arena_map_ready;
};

namespace {


bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

hg_status validate(const hg_shape* sh, const hg_quant_config* c, const uint8_t* mask, Dims* d) {
  if (!sh || !c || !mask) return HG_ERR_INVALID_ARG;
  if (sh->batch < 1 || sh->num_layers < 1 || sh->num_kv_heads < 1 || sh->num_q_heads < 1 ||
      sh->seq_len < 1 || sh->img_start < 0 || sh->img_len < 0 || sh->max_new_tokens < 0)
    return HG_ERR_INVALID_ARG;
  if ((int64_t)sh->img_start + sh->img_len > sh->seq_len) return HG_ERR_INVALID_ARG;
  if (sh->num_q_heads % sh->num_kv_heads != 0) return HG_ERR_INVALID_ARG;
  if (sh->head_dim != kD) return HG_ERR_UNSUPPORTED;
  if (sh->num_kv_heads > kMaxHeads) return HG_ERR_UNSUPPORTED;
  if (sh->num_q_heads / sh->num_kv_heads > kMaxG) return HG_ERR_UNSUPPORTED;
  if (c->base != HG_BASE_MINMAX_TOKEN && c->base != HG_BASE_KIVI && c->base != HG_BASE_AKVQ_HADAMARD)
    return HG_ERR_INVALID_ARG;
  if (c->bits != 2 && c->bits != 3 && c->bits != 4) return HG_ERR_UNSUPPORTED;
  if (c->keys_only != 0 && c->keys_only != 1) return HG_ERR_INVALID_ARG;
  if (c->meta_bits != 0 && c->meta_bits != 32 && c->meta_bits != 64) return HG_ERR_INVALID_ARG;
  if (c->salient_permille < 0 || c->salient_permille > 1000) return HG_ERR_INVALID_ARG;
  // salient tokens (Sec. 4) belong to the AKVQ-style base (with K+V or K-only
  // protection)
  if (c->salient_permille > 0 && c->base != HG_BASE_AKVQ_HADAMARD) return HG_ERR_UNSUPPORTED;
  if (c->base == HG_BASE_KIVI) {
    if (c->kivi_group_tokens != kKiviGroup || c->kivi_group_channels != kKiviGroup)
      return HG_ERR_UNSUPPORTED;
    if (c->kivi_residual < 0) return HG_ERR_INVALID_ARG;
  }
  // every offset of a layer must stay far inside 64-bit and every token index in int
  const int64_t tok = (int64_t)sh->seq_len + sh->max_new_tokens;
  if (tok > (1 << 28)) return HG_ERR_UNSUPPORTED;
  if ((int64_t)sh->batch * sh->num_kv_heads > 65535) return HG_ERR_UNSUPPORTED;  // grid.y

  d->B = sh->batch;
  d->L = sh->num_layers;
  d->H = sh->num_kv_heads;
  d->Hq = sh->num_q_heads;
  d->G = sh->num_q_heads / sh->num_kv_heads;
  d->T = sh->seq_len;
  d->s = sh->img_start;
  d->n = sh->img_len;
  d->S_new = sh->max_new_tokens;
  d->base = c->base;
  d->bits = c->bits;
  d->keys_only = c->keys_only;
  d->residual = c->base == HG_BASE_KIVI ? c->kivi_residual : 0;
  d->meta16 = c->meta_bits == 32 ? 1 : 0;
  d->nq = quantized_count(d->T, d->s, d->n, d->base, d->residual);
  d->ns = c->salient_permille > 0 ? (int)(((int64_t)d->nq * c->salient_permille + 999) / 1000) : 0;
  // the salient selection keeps one score per image token in shared memory
  if (d->ns > 0 && salient_smem_bytes(*d) > kMaxSalientSmem) return HG_ERR_UNSUPPORTED;
  return HG_OK;
}

uint64_t layer_mask_bits(const uint8_t* mask, int layer, int H) {
  uint64_t m = 0;
  for (int h = 0; h < H; ++h)
    if (mask[(size_t)layer * H + h]) m |= (1ull << h);
  return m;
}

// Every region start and batch-row stride must be a multiple of 16 bytes (the
// kernels move data with 16-byte vector and asynchronous copies).
bool geometry_aligned(const Dims& d, const LayerGeom& g) {
  for (int h = 0; h < d.H; ++h) {
    const HeadGeom hd = head_geom(d, g, h);
    const uint64_t offs[] = {hd.kb, hd.vb, hd.kq, hd.kqm, hd.vq, hd.vqm, hd.kimg, hd.sal};
    for (uint64_t o : offs)
      if (o != kNone && (o & 15u)) return false;
    const uint64_t strides[] = {hd.kb_bs, hd.kq_bs, hd.kqm_bs, hd.vq_bs, hd.vqm_bs, hd.kimg_bs};
    for (uint64_t s : strides)
      if (s & 15u) return false;
  }
  return true;
}

// Arena layout: layer blocks back to back, each 256-byte aligned.
size_t compute_layout(const Dims& d, const uint8_t* mask, std::vector<uint64_t>* bases,
                      std::vector<uint64_t>* masks) {
  uint64_t off = 0;
  for (int l = 0; l < d.L; ++l) {
    const uint64_t m = layer_mask_bits(mask, l, d.H);
    const LayerGeom g = layer_geom(d, m);
    if (!geometry_aligned(d, g)) return 0;
    if (bases) bases->push_back(off);
    if (masks) masks->push_back(m);
    off += g.size;
  }
  return (size_t)off;
}

bool range_ok(const hg_cache* c, int32_t begin, int32_t count) {
  return c && count >= 1 && begin >= 0 && (int64_t)begin + count <= c->d.L;
}

// Decode work plan.  Chunk sizes are chosen so that a launch has at most one
// wave of work items (the CTAs that are resident at once: four per SM for up
// to 8 queries per KV head, two above) of similar cost.  Chunk sizes are
// multiples of 64 tokens and depend only on the layer range and the device,
// so the workspace bound holds for every appended count.
int sm_count() {
  // per device, filled on first use; concurrent first calls store the same value
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
  int n = cached[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    cached[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

int round_up_to(int x, int g) { return ((x + g - 1) / g) * g; }

// Split a segment of len tokens of bpt bytes each into pieces of about
// item_bytes; returns the chunk size in tokens (a multiple of granule).
int chunk_tokens(int len, double bpt, double item_bytes, int granule) {
  if (len <= 0) return granule;
  long long n = (long long)(len * bpt / item_bytes + 0.5);
  if (n < 1) n = 1;
  const int per = (int)((len + n - 1) / n);
  return round_up_to(per < 1 ? 1 : per, granule);
}

// Cost per token of each segment kind, in byte-equivalents: the bytes a chunk
// streams plus a compute term calibrated on measured per-CTA timelines of the
// decode kernel (a 2-bit coded token costs about 0.6 of a BF16 token's time
// although it moves 0.16 of its bytes).  Balancing cost rather than bytes
// keeps compute-heavy coded chunks short.
struct SegBytes {
  double bf16, coded_u, coded_k;
};

SegBytes seg_bytes(const Dims& d) {
  SegBytes b;
  const double codes = 16.0 * d.bits;  // 128 codes
  const double pair = (double)meta_pair_bytes(d);
  const double kmeta = d.base == kKivi ? 4.0 * pair : pair;
  const double vmeta = pair * vgroups(d);
  // compute term per coded token (3-bit: the 2-bit expansion plus its bit-2 plane)
  const double instr_u = d.base == kKivi ? (d.bits == 2 ? 66.0 : (d.bits == 3 ? 76.0 : 78.0))
                                         : (d.bits == 2 ? 30.0 : (d.bits == 3 ? 38.0 : 40.0));
  b.bf16 = 512.0 + 8.0 * 5.0;
  b.coded_u = 2.0 * codes + kmeta + vmeta + 8.0 * instr_u;
  b.coded_k = 256.0 + codes + vmeta + 8.0 * 16.0;
  return b;
}

int max_items_of(const Dims& d, const DecodePlan& p);
ChunkCounts counts_of(const Dims& d, int appended, const DecodePlan& p);

DecodePlan plan_decode(const hg_cache* c, int begin, int count) {
  const Dims& d = c->d;
  const SegBytes sb = seg_bytes(d);
  double total = 0.0;
  for (int l = begin; l < begin + count; ++l) {
    for (int h = 0; h < d.H; ++h) {
      const int cls = head_class(d, c->layer_mask[l], h);
      if (cls == kProtected) {
        total += d.T * sb.bf16;
      } else {
        const int nc = ncoded(d);
        total += (d.T - nc) * sb.bf16 + nc * (cls == kKeysOnly ? sb.coded_k : sb.coded_u);
      }
    }
  }
  total *= d.B;
  const int wave = (d.G <= 8 ? 4 : 2) * sm_count();
  double item = total / wave;
  if (item < 16384.0) item = 16384.0;
  // Grow the item size until the items (at the largest appended count) fit
  // one wave, or every segment is a single chunk.
  DecodePlan p;
  for (int iter = 0; iter < 64; ++iter, item *= 1.05) {
    p.cbU = chunk_tokens(d.T - ncoded(d) + d.S_new, sb.bf16, item, 64);
    p.cqU = chunk_tokens(ncoded(d), sb.coded_u, item, 64);
    p.cqK = chunk_tokens(ncoded(d), sb.coded_k, item, 64);
    p.cbP = chunk_tokens(d.T + d.S_new, sb.bf16, item, 64);
    long long items = 0;
    for (int l = begin; l < begin + count; ++l)
      items += (long long)d.B * row_chunks(d, c->layer_mask[l], counts_of(d, d.S_new, p));
    if (items <= wave) break;
    if (p.cbU >= d.T - ncoded(d) + d.S_new && p.cqU >= ncoded(d) && p.cqK >= ncoded(d) &&
        p.cbP >= d.T + d.S_new)
      break;
  }
  // The merging CTA stages every split's partial of a head in its stage buffer.
  while (max_items_of(d, p) > decode_max_splits(d.G)) {
    p.cbU *= 2;
    p.cqU *= 2;
    p.cqK *= 2;
    p.cbP *= 2;
  }
  return p;
}

ChunkCounts counts_of(const Dims& d, int appended, const DecodePlan& p) {
  return chunk_counts(d, appended, p.cbU, p.cqU, p.cqK, p.cbP);
}

// Split slots per (layer, row, head): the most chunks any head can have.
int max_items_of(const Dims& d, const DecodePlan& p) {
  const ChunkCounts c = counts_of(d, d.S_new, p);
  int nb, m = head_chunks(kQuantized, c, &nb);
  const int prot = head_chunks(d.keys_only ? kKeysOnly : kProtected, c, &nb);
  return m > prot ? m : prot;
}

size_t ws_size_for(const hg_cache* c, int begin, int count) {
  const DecodePlan p = plan_decode(c, begin, count);
  return (size_t)ws_bytes(c->d, count, max_items_of(c->d, p));
}

hg_status cuda_status(cudaError_t e) { return e == cudaSuccess ? HG_OK : HG_ERR_CUDA; }

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link
// against the driver library).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

// Every BF16 token row of the arena is a 256-byte row at a 256-byte offset:
// the arena is viewed as a BF16 tensor of arena_bytes / 256 rows of 128
// channels, read in boxes of kArenaBoxRows rows x 64 channels (128 bytes, the
// span of the 128-byte swizzle).
hg_status arena_tensor_map(const hg_cache* c) {
  if (c->arena_map_ready) return HG_OK;
  const uint64_t rows = c->arena_bytes / 256;
  if (rows == 0 || rows > (uint64_t)INT32_MAX) return HG_ERR_UNSUPPORTED;
  PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
  if (!encode) return HG_ERR_CUDA;
  const cuuint64_t dims[2] = {(cuuint64_t)kD, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {256};
  const cuuint32_t box[2] = {64, (cuuint32_t)kArenaBoxRows};
  const cuuint32_t estrides[2] = {1, 1};
  const CUresult r = encode(&c->arena_map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c->arena, dims, strides, box,
                            estrides, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return HG_ERR_CUDA;
  c->arena_map_ready = true;
  return HG_OK;
}

void fill_table(const hg_cache* c, int begin, int count, LayerTable* t) {
  for (int i = 0; i < count; ++i) {
    t->base[i] = c->layer_base[begin + i];
    t->mask[i] = c->layer_mask[begin + i];
  }
}

}  // namespace

extern "C" {

const char* hg_status_string(hg_status s) {
  switch (s) {
    case HG_OK: return "ok";
    case HG_ERR_INVALID_ARG: return "invalid argument";
    case HG_ERR_ALIGNMENT: return "device pointer not 16-byte aligned";
    case HG_ERR_UNSUPPORTED: return "unsupported configuration";
    case HG_ERR_WORKSPACE_TOO_SMALL: return "decode workspace too small";
    case HG_ERR_CAPACITY: return "appended tokens exceed max_new_tokens";
    case HG_ERR_CUDA: return "CUDA runtime error";
    case HG_ERR_ARENA_TOO_SMALL: return "cache arena too small";
  }
  return "unknown status";
}

hg_status hg_cache_layout(const hg_shape* shape, const hg_quant_config* config,
                          const uint8_t* head_mask, size_t* arena_bytes) {
  Dims d;
  const hg_status st = validate(shape, config, head_mask, &d);
  if (st != HG_OK) return st;
  if (!arena_bytes) return HG_ERR_INVALID_ARG;
  const size_t n = compute_layout(d, head_mask, nullptr, nullptr);
  if (n == 0) return HG_ERR_UNSUPPORTED;
  *arena_bytes = n;
  return HG_OK;
}

hg_status hg_cache_create(const hg_shape* shape, const hg_quant_config* config,
                          const uint8_t* head_mask, void* arena, size_t arena_bytes,
                          hg_cache** out) {
  Dims d;
  const hg_status st = validate(shape, config, head_mask, &d);
  if (st != HG_OK) return st;
  if (!out || !arena) return HG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(arena) & (kAlign - 1)) != 0) return HG_ERR_ALIGNMENT;
  hg_cache* c = new (std::nothrow) hg_cache();
  if (!c) return HG_ERR_INVALID_ARG;
  c->shape = *shape;
  c->cfg = *config;
  c->d = d;
  c->needed_bytes = compute_layout(d, head_mask, &c->layer_base, &c->layer_mask);
  if (c->needed_bytes == 0) {
    delete c;
    return HG_ERR_UNSUPPORTED;
  }
  if (arena_bytes < c->needed_bytes) {
    delete c;
    return HG_ERR_ARENA_TOO_SMALL;
  }
  c->appended.assign(d.L, 0);
  c->arena = static_cast<char*>(arena);
  c->arena_bytes = arena_bytes;
  *out = c;
  return HG_OK;
}

void hg_cache_destroy(hg_cache* cache) { delete cache; }

hg_status hg_cache_head_regions(const hg_cache* c, int32_t layer, int32_t head, hg_head_regions* out) {
  if (!c || !out || layer < 0 || layer >= c->d.L || head < 0 || head >= c->d.H) return HG_ERR_INVALID_ARG;
  const LayerGeom g = layer_geom(c->d, c->layer_mask[layer]);
  const HeadGeom hd = head_geom(c->d, g, head);
  const uint64_t base = c->layer_base[layer];
  auto abs = [&](uint64_t off) { return off == kNone ? kNone : base + off; };
  out->head_class = hd.cls;
  out->nq = c->d.nq;
  out->bf16_prefill = hd.bf16_prefill;
  out->bf16_capacity = hd.cap;
  out->kb = abs(hd.kb);
  out->vb = abs(hd.vb);
  out->kq = abs(hd.kq);
  out->kqm = abs(hd.kqm);
  out->vq = abs(hd.vq);
  out->vqm = abs(hd.vqm);
  out->kimg = abs(hd.kimg);
  out->kb_bstride = hd.kb_bs;
  out->kq_bstride = hd.kq_bs;
  out->kqm_bstride = hd.kqm_bs;
  out->vq_bstride = hd.vq_bs;
  out->vqm_bstride = hd.vqm_bs;
  out->kimg_bstride = hd.kimg_bs;
  out->sal = abs(hd.sal);
  out->sal_bstride = hd.sal_bs;
  out->n_coded = hd.cls == kProtected ? 0 : ncoded(c->d);
  out->n_salient = hd.cls == kProtected ? 0 : c->d.ns;
  return HG_OK;
}

int32_t hg_cache_appended(const hg_cache* c, int32_t layer) {
  if (!c || layer < 0 || layer >= c->d.L) return -1;
  return c->appended[layer];
}

hg_status hg_cache_reset_appended(hg_cache* c) {
  if (!c) return HG_ERR_INVALID_ARG;
  for (auto& a : c->appended) a = 0;
  return HG_OK;
}

hg_status hg_quantize_kv(hg_cache* c, int32_t layer_begin, int32_t layer_count,
                         const void* const* k, const void* const* v, hg_stream_t stream) {
  if (!range_ok(c, layer_begin, layer_count) || !k || !v) return HG_ERR_INVALID_ARG;
  for (int i = 0; i < layer_count; ++i) {
    if (!k[i] || !v[i]) return HG_ERR_INVALID_ARG;
    if (!aligned16(k[i]) || !aligned16(v[i])) return HG_ERR_ALIGNMENT;
  }
  const Dims& d = c->d;
  for (int done = 0; done < layer_count; done += kMaxLayersPerLaunch) {
    const int n = std::min(kMaxLayersPerLaunch, layer_count - done);
    QuantizeParams p;
    std::memset(&p, 0, sizeof p);
    p.d = d;
    p.arena = c->arena;
    p.n_layers = n;
    p.tile_origin = d.s % 32;
    fill_table(c, layer_begin + done, n, &p.lt);
    for (int i = 0; i < n; ++i) {
      p.k[i] = static_cast<const uint16_t*>(k[done + i]);
      p.v[i] = static_cast<const uint16_t*>(v[done + i]);
    }
    if (d.ns > 0) {  // the salient-token maps first: the quantizer reads them
      const hg_status st = cuda_status(launch_salient(p, reinterpret_cast<cudaStream_t>(stream)));
      if (st != HG_OK) return st;
    }
    const hg_status st = cuda_status(launch_quantize(p, reinterpret_cast<cudaStream_t>(stream)));
    if (st != HG_OK) return st;
  }
  for (int i = 0; i < layer_count; ++i) c->appended[layer_begin + i] = 0;
  return HG_OK;
}

hg_status hg_dequantize_kv(const hg_cache* c, int32_t layer_begin, int32_t layer_count, void* k_out,
                           void* v_out, int32_t out_fp32, hg_stream_t stream) {
  if (!range_ok(c, layer_begin, layer_count) || !k_out || !v_out) return HG_ERR_INVALID_ARG;
  if (!aligned16(k_out) || !aligned16(v_out)) return HG_ERR_ALIGNMENT;
  const int appended = c->appended[layer_begin];
  for (int i = 1; i < layer_count; ++i)
    if (c->appended[layer_begin + i] != appended) return HG_ERR_INVALID_ARG;
  const Dims& d = c->d;
  const size_t layer_bytes = (size_t)d.B * d.H * (size_t)(d.T + appended) * kD * (out_fp32 ? 4 : 2);
  for (int done = 0; done < layer_count; done += kMaxLayersPerLaunch) {
    const int n = std::min(kMaxLayersPerLaunch, layer_count - done);
    DequantParams p;
    std::memset(&p, 0, sizeof p);
    p.d = d;
    p.arena = c->arena;
    p.n_layers = n;
    fill_table(c, layer_begin + done, n, &p.lt);
    p.appended = appended;
    p.out_fp32 = out_fp32 ? 1 : 0;
    p.k_out = static_cast<char*>(k_out) + (size_t)done * layer_bytes;
    p.v_out = static_cast<char*>(v_out) + (size_t)done * layer_bytes;
    const hg_status st = cuda_status(launch_dequantize(p, sm_count(), reinterpret_cast<cudaStream_t>(stream)));
    if (st != HG_OK) return st;
  }
  return HG_OK;
}

hg_status hg_append_kv(hg_cache* c, int32_t layer_begin, int32_t layer_count, const void* k_new,
                       const void* v_new, hg_stream_t stream) {
  if (!range_ok(c, layer_begin, layer_count) || !k_new || !v_new) return HG_ERR_INVALID_ARG;
  if (!aligned16(k_new) || !aligned16(v_new)) return HG_ERR_ALIGNMENT;
  for (int i = 0; i < layer_count; ++i)
    if (c->appended[layer_begin + i] >= c->d.S_new) return HG_ERR_CAPACITY;
  const Dims& d = c->d;
  const size_t layer_elems = (size_t)d.B * d.H * kD;
  for (int done = 0; done < layer_count; done += kMaxLayersPerLaunch) {
    const int n = std::min(kMaxLayersPerLaunch, layer_count - done);
    AppendParams p;
    std::memset(&p, 0, sizeof p);
    p.d = d;
    p.arena = c->arena;
    p.n_layers = n;
    fill_table(c, layer_begin + done, n, &p.lt);
    for (int i = 0; i < n; ++i) p.appended[i] = c->appended[layer_begin + done + i];
    p.k_new = static_cast<const uint16_t*>(k_new) + (size_t)done * layer_elems;
    p.v_new = static_cast<const uint16_t*>(v_new) + (size_t)done * layer_elems;
    const hg_status st = cuda_status(launch_append(p, reinterpret_cast<cudaStream_t>(stream)));
    if (st != HG_OK) return st;
  }
  for (int i = 0; i < layer_count; ++i) c->appended[layer_begin + i] += 1;
  return HG_OK;
}

hg_status hg_decode_workspace_size(const hg_cache* c, int32_t layer_count, size_t* bytes) {
  if (!c || !bytes || layer_count < 1 || layer_count > c->d.L) return HG_ERR_INVALID_ARG;
  // A launch over more than kMaxLayersPerLaunch layers reuses the workspace for
  // each group of layers; the bound is the largest over every placement.
  size_t need = 0;
  for (int b = 0; b < c->d.L; ++b) {
    const int n = std::min<int>(std::min<int>(layer_count, kMaxLayersPerLaunch), c->d.L - b);
    need = std::max(need, ws_size_for(c, b, n));
  }
  *bytes = need;
  return HG_OK;
}

hg_status hg_workspace_clear(void* ws, size_t bytes, hg_stream_t stream) {
  if (!ws) {
    // the allocation-free entry point's scratch: its header (status word);
    // its split counters are cleared by every call
    void* scratch = nullptr;
    const hg_status st = noalloc_scratch_address(&scratch);
    if (st != HG_OK) return st;
    return cuda_status(cudaMemsetAsync(scratch, 0, kWsHeaderBytes, reinterpret_cast<cudaStream_t>(stream)));
  }
  return cuda_status(cudaMemsetAsync(ws, 0, bytes, reinterpret_cast<cudaStream_t>(stream)));
}

hg_status hg_check_bounded_wait(void* word, uint32_t rounds, hg_stream_t stream) {
  if (!word || rounds == 0 || rounds > 100000) return HG_ERR_INVALID_ARG;
  if (!aligned16(word)) return HG_ERR_ALIGNMENT;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(word, 0, sizeof(uint32_t), s);
  if (e == cudaSuccess) e = launch_wait_probe(static_cast<uint32_t*>(word), rounds, s);
  return cuda_status(e);
}

hg_status hg_workspace_status(const void* ws, uint32_t* status, hg_stream_t stream) {
  if (!status) return HG_ERR_INVALID_ARG;
  if (!ws) {  // the allocation-free entry point's scratch on the current device
    void* scratch = nullptr;
    const hg_status st = noalloc_scratch_address(&scratch);
    if (st != HG_OK) return st;
    ws = scratch;
  }
  if (!aligned16(ws)) return HG_ERR_ALIGNMENT;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint32_t v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, ws, sizeof v, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return HG_ERR_CUDA;
  *status = v;
  return HG_OK;
}

}  // extern "C"

namespace {

// CTA order of the work items.  Consecutive CTAs land on different SMs and
// CTA b and b + (number of SMs) mostly on the same one, so the items are
// sorted by estimated cost (largest first) and dealt out in rounds of one per
// SM, every other round reversed: each SM gets a mix of large and small items
// instead of whatever the (layer, row, head) enumeration puts together.
// Returns the number of ordered CTAs (0: natural order).
int order_items(const hg_cache* c, int begin, int count, const DecodeParams& p, int total,
                uint32_t* order) {
  if (total > kMaxOrderedItems || total < 2) return 0;
  const Dims& d = c->d;
  if (d.B > kOrderMaxRow || p.max_items > kOrderMaxChunk) return 0;
  const SegBytes sb = seg_bytes(d);
  std::vector<std::pair<double, int>> cost;
  std::vector<uint32_t> rec;
  cost.reserve(total);
  rec.reserve(total);
  int item = 0;
  for (int i = 0; i < count; ++i) {
    const DecodeLayer& L = p.layer[i];
    const ChunkCounts cc = {L.nbU, L.nqU, L.nqK, L.nbP};
    for (int b = 0; b < d.B; ++b) {
      for (int h = 0; h < d.H; ++h) {
        const int cls = head_class(d, c->layer_mask[begin + i], h);
        int nb;
        const int ni = head_chunks(cls, cc, &nb);
        const int blen = (cls == kProtected ? d.T : d.T - d.nq + d.ns) + L.appended;
        const int clen = ncoded(d);
        const int bc = (cls == kProtected) ? p.plan.cbP : p.plan.cbU;
        const int qc = (cls == kKeysOnly) ? p.plan.cqK : p.plan.cqU;
        const double qb = (cls == kKeysOnly) ? sb.coded_k : sb.coded_u;
        for (int r = 0; r < ni; ++r) {
          double w;
          if (r < nb) w = std::min(bc, blen - r * bc) * sb.bf16;
          else w = std::min(qc, clen - (r - nb) * qc) * qb;
          cost.emplace_back(w, item++);
          rec.push_back(order_record(i, b, h, r));
        }
      }
    }
  }
  if (item != total) return 0;
  std::stable_sort(cost.begin(), cost.end(),
                   [](const std::pair<double, int>& a, const std::pair<double, int>& b) { return a.first > b.first; });
  const int S = sm_count();
  for (int j = 0; j < total; ++j) {
    const int r = j / S, s = j % S;
    const bool full_round = (r + 1) * S <= total;
    const int blk = r * S + ((r & 1) && full_round ? S - 1 - s : s);
    order[blk] = rec[cost[j].second];
  }
  return total;
}

// Decode attention over layers [layer_begin, +layer_count); with k_new / v_new
// the step's new tokens (already counted in the cache's appended state) are
// read from the inputs and stored into the arena by the same launch.
hg_status decode_launch(const hg_cache* c, int32_t layer_begin, int32_t layer_count, const void* q,
                        const void* k_new, const void* v_new, void* out, float softmax_scale,
                        void* ws, size_t ws_bytes_given, hg_stream_t stream) {
  const Dims& d = c->d;
  const hg_status mst = arena_tensor_map(c);
  if (mst != HG_OK) return mst;
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt((float)kD);
  const size_t layer_elems = (size_t)d.B * d.Hq * kD;
  const size_t kv_elems = (size_t)d.B * d.H * kD;
  for (int done = 0; done < layer_count; done += kMaxLayersPerLaunch) {
    const int n = std::min(kMaxLayersPerLaunch, layer_count - done);
    DecodeParams p;
    std::memset(&p, 0, sizeof p);
    p.d = d;
    p.arena = c->arena;
    p.n_layers = n;
    p.plan = plan_decode(c, layer_begin + done, n);
    p.max_items = max_items_of(d, p.plan);
    p.scale_log2 = scale * 1.4426950408889634f;
    p.q = static_cast<const uint16_t*>(q) + (size_t)done * layer_elems;
    p.out = static_cast<uint16_t*>(out) + (size_t)done * layer_elems;
    if (k_new) {
      p.k_new = static_cast<const uint16_t*>(k_new) + (size_t)done * kv_elems;
      p.v_new = static_cast<const uint16_t*>(v_new) + (size_t)done * kv_elems;
    }
    char* wsb = static_cast<char*>(ws);
    p.arena_map = c->arena_map;
    p.status = reinterpret_cast<uint32_t*>(wsb);
    p.counters = reinterpret_cast<uint32_t*>(wsb + kWsHeaderBytes);
    p.partials = reinterpret_cast<float*>(wsb + kWsHeaderBytes + ws_counter_bytes(d, n));
    fill_table(c, layer_begin + done, n, &p.lt);
    int total = 0;
    for (int i = 0; i < n; ++i) {
      const int l = layer_begin + done + i;
      const ChunkCounts cc = counts_of(d, c->appended[l], p.plan);
      DecodeLayer& dl = p.layer[i];
      dl.appended = c->appended[l];
      dl.nbU = cc.nbU;
      dl.nqU = cc.nqU;
      dl.nqK = cc.nqK;
      dl.nbP = cc.nbP;
      dl.items_per_row = row_chunks(d, c->layer_mask[l], cc);
      dl.item_base = total;
      total += dl.items_per_row * d.B;
    }
    p.total_items = total;
    p.n_order = order_items(c, layer_begin + done, n, p, total, p.order);
    const hg_status st = cuda_status(launch_decode(p, total, reinterpret_cast<cudaStream_t>(stream)));
    if (st != HG_OK) return st;
  }
  return HG_OK;
}

hg_status decode_checks(const hg_cache* c, int32_t layer_begin, int32_t layer_count, const void* q,
                        void* out, float softmax_scale, void* ws, size_t ws_bytes_given) {
  if (!range_ok(c, layer_begin, layer_count) || !q || !out || !ws) return HG_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || !aligned16(ws)) return HG_ERR_ALIGNMENT;
  if (!(softmax_scale == softmax_scale)) return HG_ERR_INVALID_ARG;  // NaN
  for (int done = 0; done < layer_count; done += kMaxLayersPerLaunch) {
    const int n = std::min(kMaxLayersPerLaunch, layer_count - done);
    if (ws_bytes_given < ws_size_for(c, layer_begin + done, n)) return HG_ERR_WORKSPACE_TOO_SMALL;
  }
  return HG_OK;
}

}  // namespace

extern "C" {

hg_status hg_decode_attention(const hg_cache* c, int32_t layer_begin, int32_t layer_count,
                              const void* q, void* out, float softmax_scale, void* ws,
                              size_t ws_bytes_given, hg_stream_t stream) {
  const hg_status st = decode_checks(c, layer_begin, layer_count, q, out, softmax_scale, ws, ws_bytes_given);
  if (st != HG_OK) return st;
  return decode_launch(c, layer_begin, layer_count, q, nullptr, nullptr, out, softmax_scale, ws,
                       ws_bytes_given, stream);
}

hg_status hg_decode_step(hg_cache* c, int32_t layer_begin, int32_t layer_count, const void* q,
                         const void* k_new, const void* v_new, void* out, float softmax_scale,
                         void* ws, size_t ws_bytes_given, hg_stream_t stream) {
  hg_status st = decode_checks(c, layer_begin, layer_count, q, out, softmax_scale, ws, ws_bytes_given);
  if (st != HG_OK) return st;
  if (!k_new || !v_new) return HG_ERR_INVALID_ARG;
  if (!aligned16(k_new) || !aligned16(v_new)) return HG_ERR_ALIGNMENT;
  for (int i = 0; i < layer_count; ++i)
    if (c->appended[layer_begin + i] >= c->d.S_new) return HG_ERR_CAPACITY;
  for (int i = 0; i < layer_count; ++i) c->appended[layer_begin + i] += 1;
  st = decode_launch(c, layer_begin, layer_count, q, k_new, v_new, out, softmax_scale, ws,
                     ws_bytes_given, stream);
  if (st != HG_OK)
    for (int i = 0; i < layer_count; ++i) c->appended[layer_begin + i] -= 1;
  return st;
}

}  // extern "C"

namespace hg {

hg_status decode_attention_on_scratch(const hg_cache* c, int32_t layer_begin, int32_t layer_count,
                                      const void* q, void* out, float softmax_scale, void* scratch,
                                      size_t scratch_bytes, hg_stream_t stream) {
  hg_status st = decode_checks(c, layer_begin, layer_count, q, out, softmax_scale, scratch, scratch_bytes);
  if (st != HG_OK) return st;
  st = arena_tensor_map(c);
  if (st != HG_OK) return st;
  // launches over more than kMaxLayersPerLaunch layers reuse the counters of
  // the first group, and every launch leaves them at zero again
  const size_t counters = ws_counter_bytes(c->d, std::min<int>(layer_count, kMaxLayersPerLaunch));
  if (cudaMemsetAsync(static_cast<char*>(scratch) + kWsHeaderBytes, 0, counters,
                      reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return HG_ERR_CUDA;
  return decode_launch(c, layer_begin, layer_count, q, nullptr, nullptr, out, softmax_scale, scratch,
                       scratch_bytes, stream);
}

}  // namespace hg

extern "C" {

hg_status hg_select_heads(const float* g_scores, const float* o_scores, int32_t num_layers, int32_t num_q_heads,
                          int32_t num_kv_heads, int32_t k, uint8_t* mask_out) {
  if (!g_scores || !o_scores || !mask_out || num_layers <= 0 || num_q_heads <= 0 || num_kv_heads <= 0)
    return HG_ERR_INVALID_ARG;
  if (num_q_heads % num_kv_heads != 0) return HG_ERR_INVALID_ARG;
  const int G = num_q_heads / num_kv_heads;
  const int n = num_layers * num_kv_heads;
  for (int64_t i = 0; i < (int64_t)num_layers * num_q_heads; ++i)
    if (!std::isfinite(g_scores[i]) || !std::isfinite(o_scores[i])) return HG_ERR_INVALID_ARG;
  // per-KV-head group means, then standardisation over all KV heads
  std::vector<double> gb(n), ob(n), sc(n, 0.0);
  for (int l = 0; l < num_layers; ++l)
    for (int h = 0; h < num_kv_heads; ++h) {
      double sg = 0.0, so = 0.0;
      for (int j = 0; j < G; ++j) {
        sg += g_scores[(size_t)l * num_q_heads + h * G + j];
        so += o_scores[(size_t)l * num_q_heads + h * G + j];
      }
      gb[l * num_kv_heads + h] = sg / G;
      ob[l * num_kv_heads + h] = so / G;
    }
  for (const std::vector<double>* x : {&gb, &ob}) {
    double mean = 0.0, var = 0.0;
    for (double v : *x) mean += v;
    mean /= n;
    for (double v : *x) var += (v - mean) * (v - mean);
    const double sd = std::sqrt(var / n);
    if (sd > 0.0)
      for (int i = 0; i < n; ++i) sc[i] += ((*x)[i] - mean) / sd;
  }
  if (k < 0) k = (int)std::nearbyint(n / 8.0);
  if (k > n) k = n;
  std::vector<int> idx(n);
  for (int i = 0; i < n; ++i) idx[i] = i;
  std::stable_sort(idx.begin(), idx.end(), [&](int a, int b) { return sc[a] > sc[b]; });
  for (int i = 0; i < n; ++i) mask_out[i] = 0;
  for (int i = 0; i < k; ++i) mask_out[idx[i]] = 1;
  return HG_OK;
}

hg_status hg_cache_image_bits_per_elem(const hg_cache* c, double* bits) {
  if (!c || !bits) return HG_ERR_INVALID_ARG;
  const Dims& d = c->d;
  if (d.n == 0) return HG_ERR_INVALID_ARG;
  // stored bits over all image K/V elements of the cache
  double stored = 0.0;
  const double code_bits = (double)d.bits * kD;                 // per coded token vector
  const double pair = 8.0 * meta_pair_bytes(d);  // bits of one {scale, zero}
  const double kmeta_tok = d.base == kKivi ? pair * kD / kKiviGroup : pair;
  const double vmeta_tok = pair * vgroups(d);
  for (int l = 0; l < d.L; ++l) {
    for (int h = 0; h < d.H; ++h) {
      const int cls = head_class(d, c->layer_mask[l], h);
      // salient image tokens (heads with coded values) are BF16 like the
      // image tokens outside the eligible span
      const double coded = ncoded(d), bf16 = d.n - coded;
      double kb = 0, vb = 0;
      if (cls == kQuantized) {
        kb = coded * (code_bits + kmeta_tok) + bf16 * 16.0 * kD;
        vb = coded * (code_bits + vmeta_tok) + bf16 * 16.0 * kD;
      } else if (cls == kKeysOnly) {
        kb = (double)d.n * 16.0 * kD;
        vb = coded * (code_bits + vmeta_tok) + bf16 * 16.0 * kD;
      } else {
        kb = vb = (double)d.n * 16.0 * kD;
      }
      stored += (kb + vb) * d.B;
    }
  }
  *bits = stored / ((double)d.L * d.H * d.B * d.n * kD * 2.0);
  return HG_OK;
}

}  // extern "C"
