// Arena geometry of the mixed-precision KV cache, shared by the host runtime
// and the kernels.  Everything here is arithmetic on the cache dimensions and
// one layer's 64-bit protection mask (Sec. 3, "Applying protection"), so a
// kernel can locate any (layer, batch row, head) region from two words per
// layer held in its launch parameters.
#pragma once
#include <stdint.h>

#ifdef __CUDACC__
#define HG_HD __host__ __device__ __forceinline__
#else
#define HG_HD inline
#endif

namespace hg {

constexpr int kD = 128;            // head_dim (the paper's 128-d heads, Sec. 5.4)
constexpr int kMaxHeads = 64;      // one bit per KV head in a uint64 mask
constexpr int kMaxG = 16;          // query heads per KV head
constexpr int kMaxLayersPerLaunch = 64;
constexpr int kKiviGroup = 32;     // KIVI-style key group (tokens) and value group (channels)
constexpr uint64_t kAlign = 256;   // region alignment inside the arena
constexpr uint64_t kNone = ~0ull;

enum Base : int { kMinMax = 0, kKivi = 1, kAkvq = 2 };
enum HeadClass : int { kQuantized = 0, kKeysOnly = 1, kProtected = 2 };

struct Dims {
  int B, L, H, Hq, G, T, s, n, nq, S_new;
  int base, bits, keys_only, residual;
  int meta16;  // metadata pairs as binary16 {scale, zero} (4 bytes) instead of fp32 (8)
  int ns;      // salient image tokens kept BF16 per quantized head (AKVQ-style, Sec. 4)
};

HG_HD uint64_t align_up(uint64_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

HG_HD int popc64(uint64_t x) {
#ifdef __CUDA_ARCH__
  return __popcll(x);
#else
  return __builtin_popcountll(x);
#endif
}

// Image tokens eligible for low precision: [s, s + nq).  Whole span for the
// per-token bases; whole 32-token key groups before the BF16 residual window
// for KIVI-style.
HG_HD int quantized_count(int T, int s, int n, int base, int residual) {
  if (base != kKivi) return n;
  int end = s + n;
  if (T - residual < end) end = T - residual;
  int span = end - s;
  if (span <= 0) return 0;
  return (span / kKiviGroup) * kKiviGroup;
}

// Image tokens stored coded per head with coded values (quantized heads and
// keys-only heads): the eligible span less the salient tokens.  A keys-only
// head keeps the coded tokens' keys as BF16 rows, compacted the same way.
HG_HD int ncoded(const Dims& d) { return d.nq - d.ns; }
// Salient-token map of one (batch row, head with coded values): a bit per image token
// in 32-token blocks (uint32 [nblk]), then the number of salient tokens before
// each block (int32 [nblk]); rows padded to 16 bytes.
HG_HD int sal_blocks(const Dims& d) { return (d.nq + 31) / 32; }

// Bytes per token of one head's packed codes (128 codes).
HG_HD uint64_t code_bytes_per_token(const Dims& d) { return (uint64_t)kD * d.bits / 8; }
HG_HD uint64_t align16(uint64_t x) { return (x + 15) & ~15ull; }
// Bytes of one {scale, zero} metadata pair.
HG_HD uint64_t meta_pair_bytes(const Dims& d) { return d.meta16 ? 4 : 8; }
// Key metadata bytes for nq tokens of one batch row of one head (payload).
HG_HD uint64_t kmeta_bytes(const Dims& d) {
  return d.base == kKivi ? (uint64_t)(d.nq / kKiviGroup) * kD * meta_pair_bytes(d)
                         : (uint64_t)ncoded(d) * meta_pair_bytes(d);
}
// Value metadata groups per token.
HG_HD int vgroups(const Dims& d) { return d.base == kKivi ? kD / kKiviGroup : 1; }
HG_HD uint64_t vmeta_bytes(const Dims& d) { return (uint64_t)ncoded(d) * vgroups(d) * meta_pair_bytes(d); }
// Batch-row strides of the metadata arrays: padded to 16 bytes so that every
// row (and every head's block of rows) starts on a 16-byte boundary, as the
// 16-byte asynchronous copies of the decode kernel require.
HG_HD uint64_t kmeta_stride(const Dims& d) { return align16(kmeta_bytes(d)); }
HG_HD uint64_t vmeta_stride(const Dims& d) { return align16(vmeta_bytes(d)); }
HG_HD uint64_t sal_stride(const Dims& d) { return d.ns > 0 ? align16((uint64_t)sal_blocks(d) * 8) : 0; }

struct LayerGeom {
  uint64_t mask;
  int n_prot, n_U, n_PK, n_PKV, n_VQ;
  uint64_t kb, vb, kq, kqm, vq, vqm, kimg, sal, size;  // region offsets relative to the layer base
  uint64_t bf16_bytes;                             // size of the kb (and vb) region
};

HG_HD int cap_unprot(const Dims& d) { return d.T - d.nq + d.ns + d.S_new; }

HG_HD LayerGeom layer_geom(const Dims& d, uint64_t mask) {
  LayerGeom g;
  g.mask = mask;
  g.n_prot = popc64(mask);
  g.n_U = d.H - g.n_prot;
  g.n_PK = d.keys_only ? g.n_prot : 0;
  g.n_PKV = d.keys_only ? 0 : g.n_prot;
  g.n_VQ = g.n_U + g.n_PK;
  const uint64_t B = (uint64_t)d.B;
  const uint64_t nc = (uint64_t)ncoded(d);
  const uint64_t tok_bf16 = (uint64_t)d.H * cap_unprot(d) + (uint64_t)g.n_PKV * nc;
  g.bf16_bytes = align_up(B * tok_bf16 * kD * 2);
  uint64_t off = 0;
  g.kb = off; off += g.bf16_bytes;
  g.vb = off; off += g.bf16_bytes;
  g.kq = off; off += align_up((uint64_t)g.n_U * B * nc * code_bytes_per_token(d));
  g.kqm = off; off += align_up((uint64_t)g.n_U * B * kmeta_stride(d));
  g.vq = off; off += align_up((uint64_t)g.n_VQ * B * nc * code_bytes_per_token(d));
  g.vqm = off; off += align_up((uint64_t)g.n_VQ * B * vmeta_stride(d));
  g.kimg = off; off += align_up((uint64_t)g.n_PK * B * nc * kD * 2);
  g.sal = off; off += align_up((uint64_t)g.n_VQ * B * sal_stride(d));
  g.size = off;
  return g;
}

HG_HD int head_class(const Dims& d, uint64_t mask, int h) {
  if (!((mask >> h) & 1ull)) return kQuantized;
  return d.keys_only ? kKeysOnly : kProtected;
}

// One (layer, head): offsets of element [b=0][t=0] relative to the layer base,
// and byte strides between batch rows.
struct HeadGeom {
  int cls;
  int bf16_prefill;  // BF16 tokens that come from the prefill
  int cap;           // BF16 capacity (prefill + max_new_tokens)
  uint64_t kb, vb, kq, kqm, vq, vqm, kimg, sal;
  uint64_t kb_bs, kq_bs, kqm_bs, vq_bs, vqm_bs, kimg_bs, sal_bs;
};

HG_HD HeadGeom head_geom(const Dims& d, const LayerGeom& g, int h) {
  HeadGeom r;
  const uint64_t below = (h == 0) ? 0ull : (g.mask & ((h >= 64) ? ~0ull : ((1ull << h) - 1ull)));
  const int prot_below = popc64(below);
  const uint64_t B = (uint64_t)d.B;
  r.cls = head_class(d, g.mask, h);
  r.bf16_prefill = (r.cls == kProtected) ? d.T : d.T - d.nq + d.ns;
  r.cap = r.bf16_prefill + d.S_new;
  const uint64_t pkv_below = d.keys_only ? 0ull : (uint64_t)prot_below;
  // a protected K+V head holds ncoded(d) more BF16 tokens than the others
  const uint64_t tok_before = (uint64_t)h * cap_unprot(d) + pkv_below * (uint64_t)ncoded(d);
  r.kb_bs = (uint64_t)r.cap * kD * 2;
  r.kb = g.kb + B * tok_before * kD * 2;
  r.vb = g.vb + B * tok_before * kD * 2;
  const uint64_t nc = (uint64_t)ncoded(d);
  r.kq_bs = nc * code_bytes_per_token(d);
  r.kqm_bs = kmeta_stride(d);
  r.vq_bs = nc * code_bytes_per_token(d);
  r.vqm_bs = vmeta_stride(d);
  r.kimg_bs = nc * kD * 2;
  r.sal_bs = sal_stride(d);
  r.kq = r.kqm = r.vq = r.vqm = r.kimg = r.sal = kNone;
  if (r.cls == kQuantized) {
    const uint64_t u = (uint64_t)(h - prot_below);
    r.kq = g.kq + u * B * r.kq_bs;
    r.kqm = g.kqm + u * B * r.kqm_bs;
  }
  if (r.cls != kProtected) {
    const uint64_t vr = d.keys_only ? (uint64_t)h : (uint64_t)(h - prot_below);
    r.vq = g.vq + vr * B * r.vq_bs;
    r.vqm = g.vqm + vr * B * r.vqm_bs;
    if (d.ns > 0) r.sal = g.sal + vr * B * r.sal_bs;
  }
  if (r.cls == kKeysOnly) {
    r.kimg = g.kimg + (uint64_t)prot_below * B * r.kimg_bs;
  }
  return r;
}

// Position of prefill token t in a head's BF16 region, or -1 when the token is
// an image token of a head whose image tokens are coded (the salient ones of
// a quantized head sit at d.s + their rank among the salient tokens; the
// kernels place them).  Region order: leading text, salient image tokens,
// trailing text, appended tokens.
HG_HD int bf16_pos(const Dims& d, int cls, int t) {
  if (cls == kProtected) return t;
  if (t < d.s) return t;
  if (t < d.s + d.nq) return -1;
  return t - d.nq + d.ns;
}

// ---------------------------------------------------------------------------
// Decode work decomposition.  Each (layer, batch row, KV head) is cut into
// chunks: BF16 segments of quantized / keys-only heads into chunks of cbU
// tokens, coded segments into chunks of cqU (quantized heads) or cqK
// (keys-only heads) tokens, BF16 segments of protected K+V heads into chunks
// of cbP tokens.  A work item is one chunk.  Items of one (layer, row) are
// numbered head by head, BF16 chunks before coded chunks.
// ---------------------------------------------------------------------------
HG_HD int cdiv(int a, int b) { return (a + b - 1) / b; }

struct ChunkCounts {
  int nbU, nqU, nqK, nbP;
};

HG_HD ChunkCounts chunk_counts(const Dims& d, int appended, int cbU, int cqU, int cqK, int cbP) {
  ChunkCounts c;
  c.nbU = cdiv(d.T - d.nq + d.ns + appended, cbU);
  c.nqU = cdiv(ncoded(d), cqU);
  c.nqK = cdiv(ncoded(d), cqK);
  c.nbP = cdiv(d.T + appended, cbP);
  return c;
}

// Chunks of one head and how many of them are BF16 chunks.
HG_HD int head_chunks(int cls, const ChunkCounts& c, int* n_bf16) {
  if (cls == kProtected) {
    *n_bf16 = c.nbP;
    return c.nbP;
  }
  *n_bf16 = c.nbU;
  return c.nbU + (cls == kKeysOnly ? c.nqK : c.nqU);
}

HG_HD int row_chunks(const Dims& d, uint64_t mask, const ChunkCounts& c) {
  int tot = 0, nb;
  for (int h = 0; h < d.H; ++h) tot += head_chunks(head_class(d, mask, h), c, &nb);
  return tot;
}

// Decode workspace: a 512-byte header (status word at byte 0), a counter per
// (layer, row, head), then partial results
// [layer][row][head][split][G][kD + 4] floats (m, l, two pad, o[kD]).
constexpr uint64_t kWsHeaderBytes = 512;
constexpr uint32_t kStatusWaitTimeout = 1u;  // a wait for a tile's data ran out
HG_HD uint64_t ws_counter_bytes(const Dims& d, int n_layers) {
  return align_up((uint64_t)n_layers * d.B * d.H * 4);
}
HG_HD uint64_t ws_partial_floats_per_split(const Dims& d) { return (uint64_t)d.G * (kD + 4); }
HG_HD uint64_t ws_bytes(const Dims& d, int n_layers, int max_items) {
  return kWsHeaderBytes + ws_counter_bytes(d, n_layers) +
         align_up((uint64_t)n_layers * d.B * d.H * max_items * ws_partial_floats_per_split(d) * 4);
}

}  // namespace hg
