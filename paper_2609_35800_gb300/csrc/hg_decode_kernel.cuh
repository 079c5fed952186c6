// Split-K decode attention over the mixed-precision cache (tensor cores).
//
// One CTA per work item = one chunk of one (layer, batch row, KV head).  A
// chunk is uniform: a run of BF16 tokens (text, uncoded image tokens,
// protected heads, appended tokens), a run of coded image tokens (packed
// codes + fp32 scale/zero for K and V), or, for keys-only protected heads, BF16
// keys with coded values.  The only branch on the mask or the image span is
// therefore taken once per CTA.
//
// Tiles of the chunk stream through a TMA pipeline in a 64 KB shared buffer
// (two to four stages depending on the tile size, one mbarrier each): BF16
// rows arrive as tensor-map boxes with the 128-byte swizzle, packed codes and
// metadata as one bulk copy per array, all issued by one thread.  Each warp
// owns 16-token slices and computes, with mma.sync
// m16n8k16 (BF16 in, fp32 accumulate):
//   S^T[token][query] = K . q     A = keys (BF16 via ldmatrix, or codes
//                                 expanded exactly to BF16 in registers),
//                                 B = the G queries of the KV head (padded to 8)
//   O^T[chan][query] += V^T . P^T A = values (ldmatrix.trans, or codes),
//                                 B = P^T, transposed from the score fragment
//                                 with movmatrix.
// Coded keys are contracted in the code domain: with per-token groups
// k^_d = s c_d + z, so q.k^ = s (q.c) + z sum(q); the key codes enter the MMA
// as the exact BF16 values 128 + c (no subtraction), and the 128 sum(q) offset
// is removed in the fp32 epilogue; KIVI-style per-channel
// groups fold the channel scale into the query (q~_d = q_d s_d, split into a
// BF16 hi + lo pair) and add sum_d q_d z_d.  Values fold the token scale into
// P (p s) and add sum_t p_t z_t.  AKVQ-style keys are coded in the rotated
// domain; since the normalised Hadamard matrix is symmetric and orthonormal,
// <q, H k'> = <H q, k'>, so the query is rotated once per CTA (hi + lo split).
//
// The online softmax rescales its accumulators only when a running maximum
// grows by more than 2^8 (probabilities stay <= 256 before normalisation).
// Warps are combined in shared memory; a CTA that is not alone on its head
// writes an (m, l, o) partial to the workspace and the last CTA to arrive
// (atomic ticket, no waiting) merges them and writes the BF16 output.
//
// The kernel templates live in this header; hg_decode.cu instantiates them
// for fp32 metadata pairs and hg_decode_m16.cu for binary16 pairs, so the two
// sets compile in parallel.
#pragma once
#include <cuda_runtime.h>

#include <atomic>

#include "hg_common.cuh"
#include "hg_internal.h"
#include "hg_mma.cuh"

namespace hg {

namespace {

constexpr int kThreads = 128;
constexpr int kWarps = 4;
constexpr int kBufBytes = 49152;   // pipeline buffer (stages of one tile each)
constexpr int kBf16Tile = 48;      // tokens per tile of BF16 rows (K 12 KB + V 12 KB)
constexpr int kMixTile = 48;       // tokens per tile of BF16 keys + coded values
constexpr int kPartialStride = kD + 4;  // m, l, 2 pad, o[128]: rows of 528 bytes (16-byte multiple)
// Shared memory, from a 1024-byte aligned base (swizzled TMA boxes need it).
constexpr int kStageOff = 0;                    // pipeline buffer
// Four CTAs per SM for up to 8 queries per KV head (NT = 1), two above.
// Staged queries: row r (query r of the KV head), channel c at r * kQRow + c.
// The row stride of 36 16-byte units (4 mod 8) spreads the 16-byte reads of
// one warp in the KIVI-style key path (8 rows x 4 consecutive channel
// quads) over all banks.
constexpr int kQRow = 144;
__device__ __forceinline__ int qidx(int r, int c) { return r * kQRow + c; }

template <int NT>
struct SmemLayout {
  static constexpr int q = kStageOff + kBufBytes;  // float q[NT * 8][kQRow] (qidx)
  static constexpr int bar = q + NT * 8 * kQRow * 4;  // mbarrier per stage (4), abort flag
  static constexpr int bytes = bar + 64 + 1024;    // + alignment slack
};
constexpr int kMaxStages = 4;
constexpr unsigned kFull = 0xffffffffu;
// A wait for a tile is declared stuck after kWaitRounds suspensions of up to
// kWaitSleepNs each (about a second); a healthy wait ends within microseconds.
constexpr uint32_t kWaitRounds = 20000;
constexpr uint32_t kWaitSleepNs = 50000;

enum KMode { K_BF16 = 0, K_TOKEN = 1, K_KIVI = 2 };
enum VMode { V_BF16 = 0, V_TOKEN = 1, V_KIVI = 2 };

template <int VM>
struct NZOf {
  static constexpr int value = VM == V_TOKEN ? 1 : (VM == V_KIVI ? 4 : 1);
};

// Tokens per tile of coded K + coded V: per-token groups 256 (2-bit) / 128
// (4-bit); KIVI-style (32 bytes of key metadata per token) 128.
__host__ __device__ constexpr int coded_tile(int bits, int km) { return (bits == 2 && km != 2) ? 256 : 128; }

struct Seg {
  const char* k;   // BF16 key rows (K_BF16)
  const char* v;   // BF16 value rows (V_BF16)
  int k_row0;      // arena tensor-map row of key token 0 (K_BF16)
  int v_row0;      // arena tensor-map row of value token 0 (V_BF16)
  const char* kc;  // key codes
  const char* km;  // key metadata
  const char* vc;  // value codes
  const char* vm;  // value metadata
  // Fused append: BF16 row new_pos of this segment is stored from these
  // input rows into the arena before its tile is loaded (new_pos < 0: none).
  int new_pos;
  const char* k_new;
  const char* v_new;
};

// Mask of a code pair at bits [0, b) and [16, 16 + b).
template <int BITS>
__host__ __device__ constexpr uint32_t pair_mask() { return ((1u << BITS) - 1u) * 0x00010001u; }

template <int BITS>
__device__ __forceinline__ uint32_t pair2(uint32_t x) {  // codes at bits [0,b) and [16,16+b)
  return codes_bf16x2(x & pair_mask<BITS>());
}

// The same pair as the BF16 values (128 + code): exact, without the subtraction.
template <int BITS>
__device__ __forceinline__ uint32_t pair2_off(uint32_t x) {
  return (x & pair_mask<BITS>()) | 0x43004300u;
}

// FP16 forms for value codes: exact codes, and 1024 + code.
template <int BITS>
__device__ __forceinline__ uint32_t pair2_h(uint32_t x) {
  return codes_f16x2(x & pair_mask<BITS>());
}
template <int BITS>
__device__ __forceinline__ uint32_t pair2_off_h(uint32_t x) {
  return (x & pair_mask<BITS>()) | 0x64006400u;
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

template <int NT, int NZ>
struct WarpState {
  float o[NT][8][4];
  float corr[NT][4];  // 1024 * sum_t P'^T[t][q] for value codes carried as 1024 + c
  float vb;           // coded values: power-of-two bound of the value scales seen so far
  float m[NT][2];
  float l[NT][2];
  float z[NT][2][NZ];
};

// 2-bit codes of one word sit in pairs (j, j + 8) at bits (2j, 2j + 16).  Pair j
// is taken from (w >> 6 * (j / 3)) masked at bit 2 * (j % 3): that yields
// 4^(j % 3) * code, which stays inside the 7-bit BF16 mantissa of 128 + x, and
// costs one shift per three pairs.  The factor is removed where it is exact
// (a power of two on the other MMA operand or on the accumulator).
__device__ __forceinline__ int pos3(int j) { return 2 * (j % 3); }
__device__ __forceinline__ uint32_t pair2_scaled(uint32_t w, uint32_t w6, uint32_t w12, int j) {
  const uint32_t src = j < 3 ? w : (j < 6 ? w6 : w12);
  return (src & (0x00030003u << pos3(j))) | 0x43004300u;
}
// The same pair as the FP16 values 1024 + 4^(j % 3) * code (value codes).
__device__ __forceinline__ uint32_t pair2_scaled_h(uint32_t w, uint32_t w6, uint32_t w12, int j) {
  const uint32_t src = j < 3 ? w : (j < 6 ? w6 : w12);
  return (src & (0x00030003u << pos3(j))) | 0x64006400u;
}

// 1 / x for a power of two x in [2^-126, 2^126], exactly (exponent arithmetic).
__device__ __forceinline__ float pow2_inv(float x) { return __uint_as_float(0x7F000000u - __float_as_uint(x)); }

// 3-bit codes keep bits 0-1 in the 2-bit packing and bit 2 in a plane word
// per 32 codes (element e at bit e mod 32 with index bits 3 and 4 exchanged),
// so the bit-2 pair of two codes 8 apart in one 2-bit word sits 16 bits apart
// too.  plane_pair moves such a pair from bits (i, i + 16) of a plane-derived
// register to bits (p + 2, p + 18), on top of the 2-bit pair extracted at
// bits (p, p + 16); i and p are compile-time after unrolling.
__device__ __forceinline__ uint32_t plane_pair(uint32_t pl, int i, int p) {
  const int d = i - (p + 2);
  const uint32_t x = d >= 0 ? (pl >> d) : (pl << (-d));
  return x & (0x00010001u << (p + 2));
}
// prmt selector: byte bs of a into bytes 0-1 of the result, byte bs of b into
// bytes 2-3 (the plane bytes of two tokens or two channels, side by side).
__device__ __forceinline__ uint32_t plane_sel(int bs) {
  return (uint32_t)(bs | (bs << 4) | ((4 + bs) << 8) | ((4 + bs) << 12));
}

// Smallest power of two >= m (m > 0, finite).
__device__ __forceinline__ float pow2_ceil(float m) {
  return __uint_as_float((__float_as_uint(m) + 0x007FFFFFu) & 0xFF800000u);
}

// Metadata pairs {scale, zero} in a stage: MB = 8 for two fp32, MB = 4 for
// two binary16 (scale in the low half).  meta_quad reads pairs i..i+3 (i a
// multiple of 4: one 16-byte load at MB = 4, two at MB = 8).
template <int MB>
__device__ __forceinline__ float2 meta_pair(const char* base, int i) {
  if (MB == 4) return half2_bits_to_float2(reinterpret_cast<const uint32_t*>(base)[i]);
  return reinterpret_cast<const float2*>(base)[i];
}
template <int MB>
__device__ __forceinline__ void meta_quad(const char* base, int i, float2 (&m)[4]) {
  if (MB == 4) {
    const uint4 w = *reinterpret_cast<const uint4*>(base + i * 4);
    m[0] = half2_bits_to_float2(w.x);
    m[1] = half2_bits_to_float2(w.y);
    m[2] = half2_bits_to_float2(w.z);
    m[3] = half2_bits_to_float2(w.w);
  } else {
    const float4 a = *reinterpret_cast<const float4*>(base + i * 8);
    const float4 b = *reinterpret_cast<const float4*>(base + i * 8 + 16);
    m[0] = make_float2(a.x, a.y);
    m[1] = make_float2(a.z, a.w);
    m[2] = make_float2(b.x, b.y);
    m[3] = make_float2(b.z, b.w);
  }
}

template <int BITS, int KM, int VM, int MB>
struct Tile {
  static constexpr int tokens = (KM == K_BF16 && VM == V_BF16) ? kBf16Tile
                                : (KM == K_BF16 ? kMixTile : coded_tile(BITS, KM));
  static constexpr int kc_bytes = (KM == K_BF16) ? tokens * 256 : tokens * 16 * BITS;
  static constexpr int km_bytes = (KM == K_TOKEN) ? tokens * MB : (KM == K_KIVI ? tokens * 4 * MB : 0);
  static constexpr int vc_bytes = (VM == V_BF16) ? tokens * 256 : tokens * 16 * BITS;
  static constexpr int vm_bytes = (VM == V_TOKEN) ? tokens * MB : (VM == V_KIVI ? tokens * 4 * MB : 0);
  static constexpr int kc_off = 0;
  static constexpr int km_off = kc_off + kc_bytes;
  static constexpr int vc_off = km_off + km_bytes;
  static constexpr int vm_off = vc_off + vc_bytes;
  // stages start on 1024-byte boundaries (swizzled BF16 boxes)
  static constexpr int stage_bytes = ((vm_off + vm_bytes + 1023) / 1024) * 1024;
  static constexpr int stages = (kBufBytes / stage_bytes) > kMaxStages ? kMaxStages : (kBufBytes / stage_bytes);
  static_assert(stages >= 2, "a tile must fit twice in the pipeline buffer");
  static_assert(tokens % kArenaBoxRows == 0, "BF16 tiles are whole TMA boxes");
  static_assert(VM != V_BF16 || vc_off % 1024 == 0, "swizzled value boxes start on 1024-byte boundaries");
};

// One tile into a stage, issued by a single thread: the expected byte count
// on the stage's mbarrier, then the copies.  A BF16 operand of R rows lands
// as two column halves of R x 128 bytes (channels 0-63, 64-127), each written
// by TMA boxes of kArenaBoxRows rows with the 128-byte swizzle (16-byte chunk
// c of row r at chunk c ^ (r % 8)); rows past the chunk end are loaded too and
// ignored or zeroed by the consumers.  Packed codes and metadata arrive as one
// bulk copy per array (metadata rounded up to 16 bytes: the arena pads every
// metadata row to 16 bytes); bytes past nvalid tokens are left stale.
template <int BITS, int KM, int VM, int MB>
__device__ __forceinline__ void issue_tile(uint32_t st, uint32_t bar, const Seg& sg, int t0, int nvalid,
                                           const CUtensorMap* map) {
  using TL = Tile<BITS, KM, VM, MB>;
  constexpr int kmb = (KM == K_TOKEN) ? MB : 4 * MB;  // metadata bytes per token
  constexpr int vmb = (VM == V_TOKEN) ? MB : 4 * MB;
  constexpr int kBox = kArenaBoxRows * 128;  // bytes of one box
  const int boxes = (nvalid + kArenaBoxRows - 1) / kArenaBoxRows;
  const uint32_t kc_bytes = (KM == K_BF16) ? boxes * 2 * kBox : nvalid * 16 * BITS;
  const uint32_t km_bytes = (KM == K_BF16) ? 0u : (uint32_t)((nvalid * kmb + 15) & ~15);
  const uint32_t vc_bytes = (VM == V_BF16) ? boxes * 2 * kBox : nvalid * 16 * BITS;
  const uint32_t vm_bytes = (VM == V_BF16) ? 0u : (uint32_t)((nvalid * vmb + 15) & ~15);
  mbar_arrive_expect_tx(bar, kc_bytes + km_bytes + vc_bytes + vm_bytes);
  if (KM == K_BF16) {
    for (int bx = 0; bx < boxes; ++bx)
      for (int hf = 0; hf < 2; ++hf)
        tma_load_2d(st + TL::kc_off + hf * (TL::tokens * 128) + bx * kBox, map, hf * 64,
                    sg.k_row0 + t0 + bx * kArenaBoxRows, bar);
  } else {
    bulk_g2s(st + TL::kc_off, sg.kc + (size_t)t0 * 16 * BITS, kc_bytes, bar);
    bulk_g2s(st + TL::km_off, sg.km + (size_t)t0 * kmb, km_bytes, bar);
  }
  if (VM == V_BF16) {
    for (int bx = 0; bx < boxes; ++bx)
      for (int hf = 0; hf < 2; ++hf)
        tma_load_2d(st + TL::vc_off + hf * (TL::tokens * 128) + bx * kBox, map, hf * 64,
                    sg.v_row0 + t0 + bx * kArenaBoxRows, bar);
  } else {
    bulk_g2s(st + TL::vc_off, sg.vc + (size_t)t0 * 16 * BITS, vc_bytes, bar);
    bulk_g2s(st + TL::vm_off, sg.vm + (size_t)t0 * vmb, vm_bytes, bar);
  }
}

// Bounded wait for a phase of a stage's mbarrier.  On timeout, or once another
// warp gave up, marks the CTA aborted, records the failure in the workspace
// status word and returns false (the caller skips the tile's work).
__device__ __forceinline__ bool wait_tile(uint32_t bar, uint32_t parity, volatile int* abort, uint32_t* status,
                                          uint32_t rounds = kWaitRounds) {
  for (uint32_t i = 0; i < rounds; ++i) {
    if (mbar_try_wait_sleep(bar, parity, kWaitSleepNs)) return true;
    if (*abort) return false;
  }
  *abort = 1;
  atomicOr(status, kStatusWaitTimeout);
  return false;
}

// ---------------------------------------------------------------------------
// Query fragments
// ---------------------------------------------------------------------------
// hi + lo BF16 split of an fp32 pair (x = hi + lo to ~16 significant bits)
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  hi = pack_bf16x2(x0, x1);
  const float h0 = __uint_as_float(hi << 16), h1 = __uint_as_float(hi & 0xffff0000u);
  lo = pack_bf16x2(x0 - h0, x1 - h1);
}

// Natural channel order (BF16 keys): k-step j covers channels 16j..16j+15.
template <int NT>
__device__ __forceinline__ void qfrag_natural(uint32_t (&qb)[NT][8][2], const float* q_s, int g, int tq) {
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int r = nt * 8 + g;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = 16 * j + 2 * tq;
      qb[nt][j][0] = pack_bf16x2(q_s[qidx(r, c)], q_s[qidx(r, c + 1)]);
      qb[nt][j][1] = pack_bf16x2(q_s[qidx(r, c + 8)], q_s[qidx(r, c + 9)]);
    }
  }
}

// Channels matching the in-register expansion of a packed token row.
// 2-bit: thread tq reads words 2tq and 2tq+1; k-step j takes code pair
// (j, j+8) of each.  4-bit: thread tq reads words 4tq..4tq+3; k-step j takes
// pairs (i, i+4) and (i+1, i+5), i = 2 (j & 1), of word 4tq + j/2.
template <int BITS>
__device__ __forceinline__ void token_channels(int tq, int j, int (&c)[4]) {
  if (BITS != 4) {  // 2 bits, and the 2-bit part of 3-bit codes
    c[0] = 32 * tq + j;
    c[1] = 32 * tq + j + 8;
    c[2] = 32 * tq + 16 + j;
    c[3] = 32 * tq + 24 + j;
  } else {
    const int w = 4 * tq + (j >> 1), i = 2 * (j & 1);
    c[0] = 8 * w + i;
    c[1] = 8 * w + i + 4;
    c[2] = 8 * w + i + 1;
    c[3] = 8 * w + i + 5;
  }
}

// Query fragments for coded per-token keys.  2-bit: k-step j carries q / 4^(j % 3)
// to match the scaled key pairs.  Also returns, per query column of this
// thread, s1 = sum of the fragment values as the MMA sees them (for removing
// the 128 offset of the key codes) and s0 = sum of the unscaled queries.
template <int BITS, int NT, bool ROT>
__device__ __forceinline__ void qfrag_token(uint32_t (&qb)[NT][8][2], uint32_t (&ql)[NT][8][2],
                                            float (&s1)[NT][2], float (&s0)[NT][2],
                                            const float* q_s, int g, int tq) {
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int r = nt * 8 + g;
    float a1 = 0.f, a0 = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      int c[4];
      token_channels<BITS>(tq, j, c);
      const float f = (BITS != 4) ? 1.0f / (float)(1 << pos3(j)) : 1.0f;  // exact
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const float x0 = q_s[qidx(r, c[2 * hh])] * f, x1 = q_s[qidx(r, c[2 * hh + 1])] * f;
        uint32_t hi, lo = 0u;
        if (ROT) {
          split_pair(x0, x1, hi, lo);
        } else {
          hi = pack_bf16x2(x0, x1);  // exact: the queries are BF16
        }
        qb[nt][j][hh] = hi;
        ql[nt][j][hh] = lo;
        float h0, h1, l0, l1;
        bf16x2_to_f32(hi, h0, h1);
        bf16x2_to_f32(lo, l0, l1);
        const float part = (h0 + l0) + (h1 + l1);
        a1 += part;
        a0 += part * (1.0f / f);
      }
    }
    // totals for query g, then the values of this thread's columns 2tq, 2tq+1
    a1 += __shfl_xor_sync(kFull, a1, 1);
    a1 += __shfl_xor_sync(kFull, a1, 2);
    a0 += __shfl_xor_sync(kFull, a0, 1);
    a0 += __shfl_xor_sync(kFull, a0, 2);
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      s1[nt][e] = __shfl_sync(kFull, a1, (2 * tq + e) << 2);
      s0[nt][e] = __shfl_sync(kFull, a0, (2 * tq + e) << 2);
    }
  }
}

// ---------------------------------------------------------------------------
// Softmax update of one 16-token slice
// ---------------------------------------------------------------------------
template <int NT, int NZ>
__device__ __forceinline__ void softmax_update(WarpState<NT, NZ>& ws, float (&sc)[NT][4], float (&p)[NT][4]) {
  // The running maxima are only moved when a score exceeds them by 2^8, so the
  // exact column maxima are needed only when some lane sees such a score.
  bool need = false;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int e = 0; e < 2; ++e) need |= fmaxf(sc[nt][e], sc[nt][2 + e]) > ws.m[nt][e] + 8.0f;
  if (__any_sync(kFull, need)) {
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float v = fmaxf(sc[nt][e], sc[nt][2 + e]);
        v = fmaxf(v, __shfl_xor_sync(kFull, v, 4));
        v = fmaxf(v, __shfl_xor_sync(kFull, v, 8));
        v = fmaxf(v, __shfl_xor_sync(kFull, v, 16));
        const float mn = fmaxf(ws.m[nt][e], v);
        const float a = (ws.m[nt][e] == -INFINITY) ? 0.f : fast_exp2(ws.m[nt][e] - mn);
        ws.m[nt][e] = mn;
        ws.l[nt][e] *= a;
#pragma unroll
        for (int zz = 0; zz < NZ; ++zz) ws.z[nt][e][zz] *= a;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          ws.o[nt][mt][e] *= a;
          ws.o[nt][mt][2 + e] *= a;
        }
        ws.corr[nt][e] *= a;
        ws.corr[nt][2 + e] *= a;
      }
    }
  }
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int i = 0; i < 4; ++i) p[nt][i] = fast_exp2(sc[nt][i] - ws.m[nt][i & 1]);
#pragma unroll
    for (int e = 0; e < 2; ++e) ws.l[nt][e] += p[nt][e] + p[nt][2 + e];
  }
}

// B fragments of P^T (rows scaled by fg for token g, fg8 for token g+8), as a
// BF16 hi + lo pair: b[0..1] hi, b[2..3] lo, so that P is carried to ~16 bits.
__device__ __forceinline__ void pfrag(const float (&p)[4], float fg, float fg8, uint32_t (&b)[4]) {
  uint32_t h0, l0, h1, l1;
  split_pair(p[0] * fg, p[1] * fg, h0, l0);
  split_pair(p[2] * fg8, p[3] * fg8, h1, l1);
  b[0] = movtrans(h0);
  b[1] = movtrans(h1);
  b[2] = movtrans(l0);
  b[3] = movtrans(l1);
}

// O^T m-tile += A * P^T (hi and lo parts)
__device__ __forceinline__ void mma_pv(float (&o)[4], const uint32_t (&a)[4], const uint32_t (&b)[4]) {
  mma_bf16(o, a, b[0], b[1]);
  mma_bf16(o, a, b[2], b[3]);
}

// Coded values multiply exact FP16 codes by P' = p * s / vb in FP16 (one MMA;
// about 11 significant bits, so each product carries at most 2^-12 relative
// error, far inside the tolerance).  vb is a power of two bounding every value
// scale s seen so far, so P' <= p <= 256 never overflows, and only weights
// below ~1e-4 of the largest reach FP16's subnormal range; when a larger
// scale arrives, vb grows and the accumulators are rescaled exactly.  The
// accumulators are in units of vb.
__device__ __forceinline__ void pfrag16(const float (&p)[4], float fg, float fg8, uint32_t (&b)[2]) {
  b[0] = movtrans(pack_half2(p[0] * fg, p[1] * fg));
  b[1] = movtrans(pack_half2(p[2] * fg8, p[3] * fg8));
}

template <int NT, int NZ>
__device__ __forceinline__ void vscale_update(WarpState<NT, NZ>& ws, float smax) {
  if (__any_sync(kFull, smax > ws.vb)) {
    const float nb = pow2_ceil(warp_max(smax));
    const float a = ws.vb * pow2_inv(nb);  // a power of two: exact
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int mt = 0; mt < 8; ++mt)
#pragma unroll
        for (int i = 0; i < 4; ++i) ws.o[nt][mt][i] *= a;
#pragma unroll
      for (int i = 0; i < 4; ++i) ws.corr[nt][i] *= a;
    }
    ws.vb = nb;
  }
}

// ---------------------------------------------------------------------------
// One tile: every warp processes its 16-token slices
// ---------------------------------------------------------------------------
template <int BITS, int NT, int KM, int VM, bool ROT, int MB>
__device__ __forceinline__ void compute_tile(WarpState<NT, NZOf<VM>::value>& ws, const char* st,
                                             int nvalid, const uint32_t (&qb)[NT][8][2],
                                             const uint32_t (&ql)[NT][8][2], const float* q_s,
                                             const float (&s1)[NT][2], const float (&s0)[NT][2],
                                             float scale_log2, int warp, int lane) {
  using TL = Tile<BITS, KM, VM, MB>;
  constexpr int NZ = NZOf<VM>::value;
  const int g = lane >> 2, tq = lane & 3;
  const uint32_t st_u32 = smem_u32(st);
  const uint32_t* kc32 = reinterpret_cast<const uint32_t*>(st + TL::kc_off);
  const char* kmp = st + TL::km_off;
  const uint32_t* vc32 = reinterpret_cast<const uint32_t*>(st + TL::vc_off);
  const char* vmp = st + TL::vm_off;

  // KIVI-style keys: a warp takes whole 32-token groups (two slices) so the
  // group's scaled query fragments are built once.
  constexpr int SPU = (KM == K_KIVI) ? 2 : 1;  // slices per unit
  constexpr int UNITS = TL::tokens / (16 * SPU);
  for (int u = warp; u < UNITS; u += kWarps) {
    if (u * 16 * SPU >= nvalid) break;
    float acc[SPU][NT][4];
#pragma unroll
    for (int s = 0; s < SPU; ++s)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[s][nt][i] = 0.f;
    float zk[NT][2];  // KIVI-style: sum_c q_c z_c of the group, per query column
    uint32_t qh[NT][8][2], qlo[NT][8][2];  // KIVI-style: the group's scaled queries (hi + lo)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) zk[nt][0] = zk[nt][1] = 0.f;

    // ---------------- scores ----------------
    if (KM == K_BF16) {
      const int tok0 = u * 16;
      const int row = tok0 + (lane & 7) + 8 * ((lane >> 3) & 1);
      const uint32_t rbase = st_u32 + TL::kc_off + row * 128;
      const int rsw = lane & 7, ch = lane >> 4;  // row % 8; second 8 channels of the k-step
      float acc2[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc2[nt][i] = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        uint32_t a[4];
        ldsm_x4(a, rbase + (j >> 2) * (TL::tokens * 128) + (((2 * (j & 3) + ch) ^ rsw) << 4));
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          mma_bf16((j & 1) ? acc2[nt] : acc[0][nt], a, qb[nt][j][0], qb[nt][j][1]);
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[0][nt][i] += acc2[nt][i];
    } else if (KM == K_TOKEN) {
      const int tok0 = u * 16;
      float acc2[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc2[nt][i] = 0.f;
      if (BITS != 4) {
        constexpr int RW = 4 * BITS;  // words per token row
        const uint2 ka = *reinterpret_cast<const uint2*>(kc32 + (tok0 + g) * RW + 2 * tq);
        const uint2 kb = *reinterpret_cast<const uint2*>(kc32 + (tok0 + g + 8) * RW + 2 * tq);
        const uint32_t w[4] = {ka.x, kb.x, ka.y, kb.y};
        // 3 bits: plane word tq holds bit 2 of words 2tq (pairs at j, j + 16)
        // and 2tq + 1 (at j + 8, j + 24)
        uint32_t pl[4] = {0u, 0u, 0u, 0u};
        if (BITS == 3) {
          const uint32_t pa = kc32[(tok0 + g) * RW + 8 + tq], pb = kc32[(tok0 + g + 8) * RW + 8 + tq];
          pl[0] = pa;
          pl[1] = pb;
          pl[2] = pa >> 8;
          pl[3] = pb >> 8;
        }
        uint32_t w6[4], w12[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          w6[k] = w[k] >> 6;
          w12[k] = w[k] >> 12;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          uint32_t a[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            a[k] = pair2_scaled(w[k], w6[k], w12[k], j);
            if (BITS == 3) a[k] |= plane_pair(pl[k], j, pos3(j));
          }
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            float (&dst)[4] = (j & 1) ? acc2[nt] : acc[0][nt];
            mma_bf16(dst, a, qb[nt][j][0], qb[nt][j][1]);
            if (ROT) mma_bf16(dst, a, ql[nt][j][0], ql[nt][j][1]);
          }
        }
      } else {
        const uint4 ka = *reinterpret_cast<const uint4*>(kc32 + (tok0 + g) * 16 + 4 * tq);
        const uint4 kb = *reinterpret_cast<const uint4*>(kc32 + (tok0 + g + 8) * 16 + 4 * tq);
        const uint32_t wa[4] = {ka.x, ka.y, ka.z, ka.w};
        const uint32_t wb[4] = {kb.x, kb.y, kb.z, kb.w};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int wi = j >> 1, i = 2 * (j & 1);
          uint32_t a[4];
          a[0] = pair2_off<4>(wa[wi] >> (4 * i));
          a[1] = pair2_off<4>(wb[wi] >> (4 * i));
          a[2] = pair2_off<4>(wa[wi] >> (4 * i + 4));
          a[3] = pair2_off<4>(wb[wi] >> (4 * i + 4));
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            float (&dst)[4] = (j & 1) ? acc2[nt] : acc[0][nt];
            mma_bf16(dst, a, qb[nt][j][0], qb[nt][j][1]);
            if (ROT) mma_bf16(dst, a, ql[nt][j][0], ql[nt][j][1]);
          }
        }
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[0][nt][i] += acc2[nt][i];
    } else {  // K_KIVI: group u of the tile; channel c has (scale, zero) = meta[u][c]
      const int gm = u * kD;  // first metadata pair of the group
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const float* qr = q_s + (nt * 8 + g) * kQRow;
        float zpart = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          // k-slots 2tq, 2tq+1, 2tq+8, 2tq+9 of k-step j <-> channels 16j + 4tq + 0..3
          // (the four tq lanes read four different banks of codes and metadata)
          const int c0 = 16 * j + 4 * tq;
          float2 m[4];
          meta_quad<MB>(kmp, gm + c0, m);
          const float4 qv = *reinterpret_cast<const float4*>(qr + c0);
          split_pair(qv.x * m[0].x, qv.y * m[1].x, qh[nt][j][0], qlo[nt][j][0]);
          split_pair(qv.z * m[2].x, qv.w * m[3].x, qh[nt][j][1], qlo[nt][j][1]);
          zpart = fmaf(qv.x, m[0].y, zpart);
          zpart = fmaf(qv.y, m[1].y, zpart);
          zpart = fmaf(qv.z, m[2].y, zpart);
          zpart = fmaf(qv.w, m[3].y, zpart);
        }
        // sum over the four tq lanes of query g, then fetch the columns' values
        zpart += __shfl_xor_sync(kFull, zpart, 1);
        zpart += __shfl_xor_sync(kFull, zpart, 2);
        zk[nt][0] = __shfl_sync(kFull, zpart, (2 * tq) << 2);
        zk[nt][1] = __shfl_sync(kFull, zpart, (2 * tq + 1) << 2);
      }
    }

    // ---------------- per slice: (KIVI-style keys: scores), softmax, then P.V ----------------
    // The loop stays rolled: for KIVI-style keys (two slices per unit) an
    // unrolled copy doubles the longest code path of the kernel.
#pragma unroll 1
    for (int s = 0; s < SPU; ++s) {
      const int tok0 = (u * SPU + s) * 16;
      if (tok0 >= nvalid) break;
      float ks[NT][4];  // KIVI-style: this slice's scores against the scaled queries
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) ks[nt][i] = 0.f;
      if (KM == K_KIVI) {
        const uint32_t* gc = kc32 + u * kD * BITS;  // [128 channels][BITS words], token order
        // byte selector: byte (g/2) of a -> byte 0, byte (g/2) of b -> byte 2
        const uint32_t sel4 = (uint32_t)(g >> 1) | ((uint32_t)(4 + (g >> 1)) << 8);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int c0 = 16 * j + 4 * tq;
          // per channel: the word(s) of tokens 16s..16s+15 (3 bits: and the bit-2 plane)
          uint32_t w[4][2];
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) {
            if (BITS == 2) {
              w[cc][0] = gc[(c0 + cc) * 2 + s];
              w[cc][1] = 0u;
            } else if (BITS == 3) {
              w[cc][0] = gc[(c0 + cc) * 3 + s];
              w[cc][1] = gc[(c0 + cc) * 3 + 2];
            } else {
              const uint2 t2 = *reinterpret_cast<const uint2*>(gc + (c0 + cc) * 4 + 2 * s);
              w[cc][0] = t2.x;
              w[cc][1] = t2.y;
            }
          }
          uint32_t a[4];
          if (BITS == 2) {
            // the word's low half holds tokens 16s..16s+7, its high half the next 8
            a[0] = pair2<2>(prmt(w[0][0], w[1][0], 0x5410) >> (2 * g));
            a[1] = pair2<2>(prmt(w[0][0], w[1][0], 0x7632) >> (2 * g));
            a[2] = pair2<2>(prmt(w[2][0], w[3][0], 0x5410) >> (2 * g));
            a[3] = pair2<2>(prmt(w[2][0], w[3][0], 0x7632) >> (2 * g));
          } else if (BITS == 3) {
            // bit 2 of token 16s + i: plane byte s (i < 8) or 2 + s (i >= 8), bit i % 8
            const uint32_t lo0 = prmt(w[0][0], w[1][0], 0x5410) >> (2 * g);
            const uint32_t lo1 = prmt(w[0][0], w[1][0], 0x7632) >> (2 * g);
            const uint32_t lo2 = prmt(w[2][0], w[3][0], 0x5410) >> (2 * g);
            const uint32_t lo3 = prmt(w[2][0], w[3][0], 0x7632) >> (2 * g);
            const uint32_t h0 = prmt(w[0][1], w[1][1], plane_sel(s)) >> g;
            const uint32_t h1 = prmt(w[0][1], w[1][1], plane_sel(2 + s)) >> g;
            const uint32_t h2 = prmt(w[2][1], w[3][1], plane_sel(s)) >> g;
            const uint32_t h3 = prmt(w[2][1], w[3][1], plane_sel(2 + s)) >> g;
            a[0] = pair2<3>((lo0 & 0x00030003u) | ((h0 & 0x00010001u) << 2));
            a[1] = pair2<3>((lo1 & 0x00030003u) | ((h1 & 0x00010001u) << 2));
            a[2] = pair2<3>((lo2 & 0x00030003u) | ((h2 & 0x00010001u) << 2));
            a[3] = pair2<3>((lo3 & 0x00030003u) | ((h3 & 0x00010001u) << 2));
          } else {
            // words 2s, 2s+1 of a channel: tokens 16s..16s+7 and 16s+8..16s+15
            const int sh = 4 * (g & 1);
            a[0] = pair2<4>(prmt(w[0][0], w[1][0], sel4) >> sh);
            a[1] = pair2<4>(prmt(w[0][1], w[1][1], sel4) >> sh);
            a[2] = pair2<4>(prmt(w[2][0], w[3][0], sel4) >> sh);
            a[3] = pair2<4>(prmt(w[2][1], w[3][1], sel4) >> sh);
          }
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            mma_bf16(ks[nt], a, qh[nt][j][0], qh[nt][j][1]);
            mma_bf16(ks[nt], a, qlo[nt][j][0], qlo[nt][j][1]);
          }
        }
      }
      float sc[NT][4];
      if (KM == K_TOKEN) {
        // acc = sum_d (128 + f c_d) (q_d / f) = 128 s1 + q.c, so
        // score = s (acc - 128 s1) + z s0
        const float2 mg = meta_pair<MB>(kmp, tok0 + g), mg8 = meta_pair<MB>(kmp, tok0 + g + 8);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float off = -128.f * s1[nt][e];
            sc[nt][e] = fmaf(mg.x, acc[s][nt][e] + off, mg.y * s0[nt][e]) * scale_log2;
            sc[nt][2 + e] = fmaf(mg8.x, acc[s][nt][2 + e] + off, mg8.y * s0[nt][e]) * scale_log2;
          }
        }
      } else if (KM == K_KIVI) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) sc[nt][i] = (ks[nt][i] + zk[nt][i & 1]) * scale_log2;
      } else {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int i = 0; i < 4; ++i) sc[nt][i] = acc[s][nt][i] * scale_log2;
      }
      if (tok0 + 16 > nvalid) {
        const bool vg0 = tok0 + g < nvalid, vg8 = tok0 + g + 8 < nvalid;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          if (!vg0) sc[nt][0] = sc[nt][1] = -INFINITY;
          if (!vg8) sc[nt][2] = sc[nt][3] = -INFINITY;
        }
      }
      float p[NT][4];
      softmax_update<NT, NZ>(ws, sc, p);

      if (VM == V_BF16) {
        uint32_t b[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) pfrag(p[nt], 1.f, 1.f, b[nt]);
        if (tok0 + 16 > nvalid) {
          // rows past the end hold whatever follows in the arena: zero them so
          // that 0 * (non-finite) cannot reach the accumulators
          for (int i = lane; i < (tok0 + 16 - nvalid) * 16; i += 32) {
            const int rr = nvalid + (i >> 4), c = i & 15;
            *reinterpret_cast<uint4*>(const_cast<char*>(st) + TL::vc_off + (c >> 3) * (TL::tokens * 128) +
                                      rr * 128 + (c & 7) * 16) = make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_shared();  // the stage is refilled by TMA later
          __syncwarp();
        }
        const int row = tok0 + (lane & 7) + 8 * (lane >> 4);
        const uint32_t rbase = st_u32 + TL::vc_off + row * 128;
        const int rsw = lane & 7, ch = (lane >> 3) & 1;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          uint32_t a[4];
          ldsm_x4_trans(a, rbase + (mt >> 2) * (TL::tokens * 128) + (((2 * (mt & 3) + ch) ^ rsw) << 4));
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_pv(ws.o[nt][mt], a, b[nt]);
        }
      } else if (VM == V_TOKEN) {
        // metadata past the end of the tile is stale: its factors are zeroed
        const bool ok0 = tok0 + g < nvalid, ok8 = tok0 + g + 8 < nvalid;
        const float2 vg = ok0 ? meta_pair<MB>(vmp, tok0 + g) : make_float2(0.f, 0.f);
        const float2 vg8 = ok8 ? meta_pair<MB>(vmp, tok0 + g + 8) : make_float2(0.f, 0.f);
        vscale_update(ws, fmaxf(vg.x, vg8.x));
        const float inv = pow2_inv(ws.vb);
        uint32_t b[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          pfrag16(p[nt], vg.x * inv, vg8.x * inv, b[nt]);
#pragma unroll
          for (int e = 0; e < 2; ++e) ws.z[nt][e][0] += p[nt][e] * vg.y + p[nt][2 + e] * vg8.y;
        }
        // value codes enter as 1024 + f c; the 1024 part is collected in ws.corr
        // by one MMA on a constant tile and removed at the end (f: see pair2_scaled)
        {
          const uint32_t c1024[4] = {0x64006400u, 0x64006400u, 0x64006400u, 0x64006400u};
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_f16(ws.corr[nt], c1024, b[nt][0], b[nt][1]);
        }
        const int t0 = tok0 + 2 * tq;
        if (BITS != 4) {
          // word g of a token row holds channels 16g..16g+15
          constexpr int RW = 4 * BITS;  // words per token row
          const uint32_t w0 = vc32[t0 * RW + g], w1 = vc32[(t0 + 1) * RW + g];
          const uint32_t w8 = vc32[(t0 + 8) * RW + g], w9 = vc32[(t0 + 9) * RW + g];
          const uint32_t x[4] = {prmt(w0, w1, 0x5410), prmt(w0, w1, 0x7632), prmt(w8, w9, 0x5410),
                                 prmt(w8, w9, 0x7632)};
          // 3 bits: bit 2 of word g's codes 0-7 is byte g % 2 of plane word
          // 8 + g / 2, codes 8-15 byte 2 + g % 2; two tokens side by side
          uint32_t hp[4] = {0u, 0u, 0u, 0u};
          if (BITS == 3) {
            const int pw = 8 + (g >> 1), bs = g & 1;
            const uint32_t p0 = vc32[t0 * RW + pw], p1 = vc32[(t0 + 1) * RW + pw];
            const uint32_t p8 = vc32[(t0 + 8) * RW + pw], p9 = vc32[(t0 + 9) * RW + pw];
            hp[0] = prmt(p0, p1, plane_sel(bs));
            hp[1] = prmt(p0, p1, plane_sel(2 + bs));
            hp[2] = prmt(p8, p9, plane_sel(bs));
            hp[3] = prmt(p8, p9, plane_sel(2 + bs));
          }
          uint32_t x6[4], x12[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            x6[k] = x[k] >> 6;
            x12[k] = x[k] >> 12;
          }
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            uint32_t a[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              a[k] = pair2_scaled_h(x[k], x6[k], x12[k], mt);
              if (BITS == 3) a[k] |= plane_pair(hp[k], mt, pos3(mt));
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) mma_f16(ws.o[nt][mt], a, b[nt][0], b[nt][1]);
          }
        } else {
          // word 2g holds channels 16g..16g+7 (codes 0-3 low half, 4-7 high), 2g+1 the next 8
          const uint2 v0 = *reinterpret_cast<const uint2*>(vc32 + t0 * 16 + 2 * g);
          const uint2 v1 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 1) * 16 + 2 * g);
          const uint2 v8 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 8) * 16 + 2 * g);
          const uint2 v9 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 9) * 16 + 2 * g);
          const uint32_t xa = prmt(v0.x, v1.x, 0x5410), ya = prmt(v0.x, v1.x, 0x7632);
          const uint32_t xb = prmt(v0.y, v1.y, 0x5410), yb = prmt(v0.y, v1.y, 0x7632);
          const uint32_t xc = prmt(v8.x, v9.x, 0x5410), yc = prmt(v8.x, v9.x, 0x7632);
          const uint32_t xd = prmt(v8.y, v9.y, 0x5410), yd = prmt(v8.y, v9.y, 0x7632);
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            const int sh = 4 * (mt & 3);
            uint32_t a[4];
            a[0] = pair2_off_h<4>((mt < 4 ? xa : ya) >> sh);
            a[1] = pair2_off_h<4>((mt < 4 ? xb : yb) >> sh);
            a[2] = pair2_off_h<4>((mt < 4 ? xc : yc) >> sh);
            a[3] = pair2_off_h<4>((mt < 4 ? xd : yd) >> sh);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) mma_f16(ws.o[nt][mt], a, b[nt][0], b[nt][1]);
          }
        }
      } else {  // V_KIVI: 4 value groups of 32 channels; m-tile mt = channels 16mt..16mt+15
        float sv_g[4], zv_g[4], sv_g8[4], zv_g8[4];
        {
          // the four (scale, zero) pairs of a token; stale metadata past the end is zeroed
          const bool ok0 = tok0 + g < nvalid, ok8 = tok0 + g + 8 < nvalid;
          float2 a[4], c[4];
          meta_quad<MB>(vmp, (tok0 + g) * 4, a);
          meta_quad<MB>(vmp, (tok0 + g + 8) * 4, c);
#pragma unroll
          for (int jg = 0; jg < 4; ++jg) {
            sv_g[jg] = ok0 ? a[jg].x : 0.f;
            zv_g[jg] = ok0 ? a[jg].y : 0.f;
            sv_g8[jg] = ok8 ? c[jg].x : 0.f;
            zv_g8[jg] = ok8 ? c[jg].y : 0.f;
          }
        }
        vscale_update(ws, fmaxf(fmaxf(fmaxf(sv_g[0], sv_g[1]), fmaxf(sv_g[2], sv_g[3])),
                                fmaxf(fmaxf(sv_g8[0], sv_g8[1]), fmaxf(sv_g8[2], sv_g8[3]))));
        const float inv = pow2_inv(ws.vb);
        uint32_t b[NT][4][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
          for (int jg = 0; jg < 4; ++jg) {
            pfrag16(p[nt], sv_g[jg] * inv, sv_g8[jg] * inv, b[nt][jg]);
#pragma unroll
            for (int e = 0; e < 2; ++e)
              ws.z[nt][e][jg % NZ] += p[nt][e] * zv_g[jg] + p[nt][2 + e] * zv_g8[jg];
          }
        }
        const int t0 = tok0 + 2 * tq;
        constexpr int W = 4 * BITS;  // words per token
        const uint32_t sel4 = (uint32_t)(g >> 1) | ((uint32_t)(4 + (g >> 1)) << 8);
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          uint32_t a[4];
          if (BITS == 2) {
            const uint32_t w0 = vc32[t0 * W + mt], w1 = vc32[(t0 + 1) * W + mt];
            const uint32_t w8 = vc32[(t0 + 8) * W + mt], w9 = vc32[(t0 + 9) * W + mt];
            a[0] = pair2_h<2>(prmt(w0, w1, 0x5410) >> (2 * g));
            a[1] = pair2_h<2>(prmt(w0, w1, 0x7632) >> (2 * g));
            a[2] = pair2_h<2>(prmt(w8, w9, 0x5410) >> (2 * g));
            a[3] = pair2_h<2>(prmt(w8, w9, 0x7632) >> (2 * g));
          } else if (BITS == 3) {
            // channels 16mt + g and 16mt + 8 + g: bit 2 in byte mt % 2 and
            // 2 + mt % 2 of plane word 8 + mt / 2, bit g
            const uint32_t w0 = vc32[t0 * W + mt], w1 = vc32[(t0 + 1) * W + mt];
            const uint32_t w8 = vc32[(t0 + 8) * W + mt], w9 = vc32[(t0 + 9) * W + mt];
            const int pw = 8 + (mt >> 1), bs = mt & 1;
            const uint32_t p0 = vc32[t0 * W + pw], p1 = vc32[(t0 + 1) * W + pw];
            const uint32_t p8 = vc32[(t0 + 8) * W + pw], p9 = vc32[(t0 + 9) * W + pw];
            const uint32_t h0 = prmt(p0, p1, plane_sel(bs)) >> g, h1 = prmt(p0, p1, plane_sel(2 + bs)) >> g;
            const uint32_t h2 = prmt(p8, p9, plane_sel(bs)) >> g, h3 = prmt(p8, p9, plane_sel(2 + bs)) >> g;
            a[0] = pair2_h<3>(((prmt(w0, w1, 0x5410) >> (2 * g)) & 0x00030003u) | ((h0 & 0x00010001u) << 2));
            a[1] = pair2_h<3>(((prmt(w0, w1, 0x7632) >> (2 * g)) & 0x00030003u) | ((h1 & 0x00010001u) << 2));
            a[2] = pair2_h<3>(((prmt(w8, w9, 0x5410) >> (2 * g)) & 0x00030003u) | ((h2 & 0x00010001u) << 2));
            a[3] = pair2_h<3>(((prmt(w8, w9, 0x7632) >> (2 * g)) & 0x00030003u) | ((h3 & 0x00010001u) << 2));
          } else {
            const uint2 u0 = *reinterpret_cast<const uint2*>(vc32 + t0 * W + 2 * mt);
            const uint2 u1 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 1) * W + 2 * mt);
            const uint2 u8 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 8) * W + 2 * mt);
            const uint2 u9 = *reinterpret_cast<const uint2*>(vc32 + (t0 + 9) * W + 2 * mt);
            const int sh = 4 * (g & 1);
            a[0] = pair2_h<4>(prmt(u0.x, u1.x, sel4) >> sh);
            a[1] = pair2_h<4>(prmt(u0.y, u1.y, sel4) >> sh);
            a[2] = pair2_h<4>(prmt(u8.x, u9.x, sel4) >> sh);
            a[3] = pair2_h<4>(prmt(u8.y, u9.y, sel4) >> sh);
          }
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_f16(ws.o[nt][mt], a, b[nt][mt >> 1][0], b[nt][mt >> 1][1]);
        }
      }
    }
  }
  if (VM == V_TOKEN) {
    // Fold the tile's 1024 offsets into the accumulators.  Both grow with the
    // segment while their difference (the value sum) stays small; left to the
    // end of a long segment (thousands of tokens in one CTA), the fp32
    // accumulation error of the large common part would show in the result.
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int mt = 0; mt < 8; ++mt)
#pragma unroll
        for (int i = 0; i < 4; ++i) ws.o[nt][mt][i] -= ws.corr[nt][i];
#pragma unroll
      for (int i = 0; i < 4; ++i) ws.corr[nt][i] = 0.f;
    }
  }
}

// ---------------------------------------------------------------------------
// Combine of (m, l, o) partials of the same queries (the four warps of a CTA,
// or the splits of a head): part s, query j at parts + s * sstride + j * 132
// (m at +0, l at +1, o at +4).  With M = max_s m_s and f_s = 2^(m_s - M):
// o = sum_s f_s o_s / L, L = sum_s f_s l_s.  combine_weights leaves f_s in
// fw[s][j] (s < 16), L in fw[kFwL][j], M in fw[kFwM][j] and 1 / L in
// fw[kFwR][j] (rows of kMaxG).  Both steps are short dependency chains: eight
// threads per query reduce the weights with shuffles, and each thread then
// accumulates one channel of every query at once.
// ---------------------------------------------------------------------------
constexpr int kFwL = 16, kFwM = 17, kFwR = 18;
static_assert(kThreads == 8 * kMaxG, "eight combine threads per query");

__device__ __forceinline__ void combine_weights(const float* parts, int n, int sstride, int G, float* fw,
                                                int tid) {
  // thread t: query t / 8, parts t % 8 and t % 8 + 8
  const int j = tid >> 3, sl = tid & 7;
  const bool h0 = j < G && sl < n, h1 = j < G && sl + 8 < n;
  const float* pj = parts + j * kPartialStride;
  const float m0 = h0 ? pj[sl * sstride] : -INFINITY;
  const float l0 = h0 ? pj[sl * sstride + 1] : 0.f;
  const float m1 = h1 ? pj[(sl + 8) * sstride] : -INFINITY;
  const float l1 = h1 ? pj[(sl + 8) * sstride + 1] : 0.f;
  float M = fmaxf(m0, m1);
  M = fmaxf(M, __shfl_xor_sync(kFull, M, 1));
  M = fmaxf(M, __shfl_xor_sync(kFull, M, 2));
  M = fmaxf(M, __shfl_xor_sync(kFull, M, 4));
  const float f0 = (m0 == -INFINITY) ? 0.f : fast_exp2(m0 - M);
  const float f1 = (m1 == -INFINITY) ? 0.f : fast_exp2(m1 - M);
  float Ls = fmaf(f0, l0, f1 * l1);
  Ls += __shfl_xor_sync(kFull, Ls, 1);
  Ls += __shfl_xor_sync(kFull, Ls, 2);
  Ls += __shfl_xor_sync(kFull, Ls, 4);
  if (h0) fw[sl * kMaxG + j] = f0;
  if (h1) fw[(sl + 8) * kMaxG + j] = f1;
  if (j < G && sl == 0) {
    fw[kFwL * kMaxG + j] = Ls;
    fw[kFwM * kMaxG + j] = M;
    fw[kFwR * kMaxG + j] = 1.0f / Ls;
  }
  __syncthreads();
}

// Channel c of queries 0..JM-1 (those below G): acc[j] = sum_s f_s o_s[j][c].
template <int JM>
__device__ __forceinline__ void combine_out(const float* parts, int n, int sstride, const float* fw, int G, int c,
                                            float (&acc)[JM]) {
#pragma unroll
  for (int j = 0; j < JM; ++j) acc[j] = 0.f;
#pragma unroll 1
  for (int s = 0; s < n; ++s) {
    const float* ps = parts + s * sstride + 4 + c;
    const float* fs = fw + s * kMaxG;
#pragma unroll
    for (int j = 0; j < JM; ++j)
      if (j < G) acc[j] = fmaf(fs[j], ps[j * kPartialStride], acc[j]);
  }
}

// One combine pass: the weights, then channel `tid` of every query, written
// as the final BF16 output rows (out: row 0 of this head's queries) or as this
// split's partial (mine).  Not inlined: the warp combine and the split merge
// run the same instructions, so the merge -- once per head, at the end of the
// launch -- executes from cached code.
template <int JM>
__device__ __noinline__ void combine_pass(const float* src, int n, int sstride, float* fw, int G, int tid,
                                          bool final, uint16_t* out, float* mine) {
  combine_weights(src, n, sstride, G, fw, tid);
  float acc[JM];
  combine_out<JM>(src, n, sstride, fw, G, tid, acc);
#pragma unroll
  for (int j = 0; j < JM; ++j) {
    if (j >= G) break;
    if (final) {
      out[(size_t)j * kD + tid] = (uint16_t)f32_to_bf16_rn(acc[j] * fw[kFwR * kMaxG + j]);
    } else {
      mine[j * kPartialStride + 4 + tid] = acc[j];
      if (tid == 0) {
        mine[j * kPartialStride + 0] = fw[kFwM * kMaxG + j];
        mine[j * kPartialStride + 1] = fw[kFwL * kMaxG + j];
      }
    }
  }
}

// ---------------------------------------------------------------------------
// One work item with a given key / value mode: pipeline, then per-warp results
// into shared memory (m, l, o[q][channel]).
// ---------------------------------------------------------------------------
// 16-byte pieces of the staged queries per thread (piece i: query row i / 16,
// channels 8 (i % 16) .. + 7).
template <int NT>
struct QPieces {
  static constexpr int n = (NT * 8 * 16 + kThreads - 1) / kThreads;
};

template <int BITS, int NT, int KM, int VM, bool ROT, int MB>
__device__ __forceinline__ void run_item(char* smem, const Seg& sg, int tb, int te, const DecodeParams& p,
                                         const uint4 (&qv)[QPieces<NT>::n], int G, float* parts) {
  using TL = Tile<BITS, KM, VM, MB>;
  constexpr int NZ = NZOf<VM>::value;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tq = lane & 3;
  float* q_s = reinterpret_cast<float*>(smem + SmemLayout<NT>::q);
  char* stages = smem + kStageOff;

  // Every tile that fits the buffer goes in flight before anything else;
  // later tiles, if any, reuse stages as the ring advances.  Tile i uses stage
  // i % STAGES and phase i / STAGES of that stage's mbarrier.
  constexpr int STAGES = TL::stages;
  const float scale_log2 = p.scale_log2;
  const int n_tiles = (te - tb + TL::tokens - 1) / TL::tokens;
  const uint32_t st0 = smem_u32(stages);
  const uint32_t bars = smem_u32(smem + SmemLayout<NT>::bar);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + SmemLayout<NT>::bar + 8 * kMaxStages);
  constexpr int QV = QPieces<NT>::n;
  // Only the first tile goes in flight now: with every CTA of the launch
  // starting at once, first tiles alone make a burst the memory system serves
  // quickly, so compute starts early; the other stages are filled once the
  // first tile has landed.
  int issued = n_tiles > 0 ? 1 : 0;  // meaningful in thread 0
  if (tid == 0 && issued)
    issue_tile<BITS, KM, VM, MB>(st0, bars, sg, tb, min(TL::tokens, te - tb), &p.arena_map);

  // Queries of this KV head's group (fp32, rows >= G zero), rotated for
  // AKVQ-style coded keys.
#pragma unroll
  for (int k = 0; k < QV; ++k) {
    const int i = tid + k * kThreads;
    if (i < NT * 8 * 16) {
      // piece i: row i / 16, channels 8 (i % 16) .. + 7
      float4* dst = reinterpret_cast<float4*>(q_s + qidx(i >> 4, 8 * (i & 15)));
      float f[8];
      bf16x2_to_f32(qv[k].x, f[0], f[1]);
      bf16x2_to_f32(qv[k].y, f[2], f[3]);
      bf16x2_to_f32(qv[k].z, f[4], f[5]);
      bf16x2_to_f32(qv[k].w, f[6], f[7]);
      dst[0] = make_float4(f[0], f[1], f[2], f[3]);
      dst[1] = make_float4(f[4], f[5], f[6], f[7]);
    }
  }
  __syncthreads();
  if (ROT) {
    for (int j = warp; j < G; j += kWarps) {
      float x[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) x[i] = q_s[qidx(j, lane * 4 + i)];
      fwht128_warp(x, lane);
#pragma unroll
      for (int i = 0; i < 4; ++i) q_s[qidx(j, lane * 4 + i)] = x[i];
    }
    __syncthreads();
  }
  uint32_t qb[NT][8][2], ql[NT][8][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int j = 0; j < 8; ++j) qb[nt][j][0] = qb[nt][j][1] = ql[nt][j][0] = ql[nt][j][1] = 0u;
  float s1[NT][2], s0[NT][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) s1[nt][0] = s1[nt][1] = s0[nt][0] = s0[nt][1] = 0.f;
  if (KM == K_BF16) qfrag_natural<NT>(qb, q_s, g, tq);
  if (KM == K_TOKEN) qfrag_token<BITS, NT, ROT>(qb, ql, s1, s0, q_s, g, tq);

  WarpState<NT, NZ> ws;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      ws.m[nt][e] = -INFINITY;
      ws.l[nt][e] = 0.f;
#pragma unroll
      for (int zz = 0; zz < NZ; ++zz) ws.z[nt][e][zz] = 0.f;
    }
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
#pragma unroll
      for (int i = 0; i < 4; ++i) ws.o[nt][mt][i] = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) ws.corr[nt][i] = 0.f;
  }
  ws.vb = __uint_as_float(0x00800000u);  // 2^-126: no value scale seen yet

  for (int it = 0; it < n_tiles; ++it) {
    const int st = it % STAGES;
    const bool ok = __all_sync(kFull, !*abort && wait_tile(bars + 8 * st, (it / STAGES) & 1, abort, p.status));
    __syncthreads();
    if (tid == 0 && !*abort) {
      // tile 0 landed: fill the other stages; later, refill the stage of tile it - 1
      const int upto = (it == 0) ? min(n_tiles, STAGES) : min(n_tiles, it + STAGES);
      if (it > 0 && issued < upto) fence_proxy_async_shared();
      for (; issued < upto; ++issued)
        issue_tile<BITS, KM, VM, MB>(st0 + (issued % STAGES) * TL::stage_bytes, bars + 8 * (issued % STAGES), sg,
                                     tb + issued * TL::tokens, min(TL::tokens, te - tb - issued * TL::tokens),
                                     &p.arena_map);
    }
    if (ok)
      compute_tile<BITS, NT, KM, VM, ROT, MB>(ws, stages + st * TL::stage_bytes,
                                              min(TL::tokens, te - tb - it * TL::tokens), qb, ql, q_s, s1, s0,
                                              scale_log2, warp, lane);
  }
  if (tid == 0 && *abort) {
    // A stage is refilled only after its previous tile landed, so only the
    // last STAGES tiles can still be in flight: let them land (bounded)
    // before the buffer is reused or the CTA exits.
    for (int t = (issued > STAGES ? issued - STAGES : 0); t < issued; ++t)
      for (uint32_t i = 0; i < kWaitRounds && !mbar_try_wait_sleep(bars + 8 * (t % STAGES), (t / STAGES) & 1,
                                                                    kWaitSleepNs);
           ++i) {
      }
  }
  __syncthreads();  // stage buffers are reused for the reduction below

  // ---- per-warp results: reduce l and the value-zero terms over the 8 rows g ----
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float l = ws.l[nt][e];
      l += __shfl_xor_sync(kFull, l, 4);
      l += __shfl_xor_sync(kFull, l, 8);
      l += __shfl_xor_sync(kFull, l, 16);
#pragma unroll
      for (int zz = 0; zz < NZ; ++zz) {
        float z = ws.z[nt][e][zz];
        z += __shfl_xor_sync(kFull, z, 4);
        z += __shfl_xor_sync(kFull, z, 8);
        z += __shfl_xor_sync(kFull, z, 16);
        ws.z[nt][e][zz] = z;
      }
      const int q = nt * 8 + 2 * tq + e;
      float* prow = parts + (warp * kMaxG + q) * kPartialStride;  // (m, l, -, -, o[128])
      if (g == 0) {
        prow[0] = ws.m[nt][e];
        prow[1] = l;
      }
      float* orow = prow + 4;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        int c_lo, c_hi;  // channels of rows g and g+8 of m-tile mt
        if (VM == V_TOKEN) {
          // remove the 128 offset and the 4^(mt % 3) factor of 2-bit value pairs
          c_lo = 16 * g + mt;
          c_hi = 16 * g + 8 + mt;
          // and the units (vb) of the coded-value accumulators
          const float f = ((BITS != 4) ? 1.0f / (float)(1 << pos3(mt)) : 1.0f) * ws.vb;
          orow[c_lo] = (ws.o[nt][mt][e] - ws.corr[nt][e]) * f + ws.z[nt][e][0];
          orow[c_hi] = (ws.o[nt][mt][2 + e] - ws.corr[nt][2 + e]) * f + ws.z[nt][e][0];
        } else {
          c_lo = 16 * mt + g;
          c_hi = 16 * mt + 8 + g;
          const float z = (VM == V_KIVI) ? ws.z[nt][e][(mt >> 1) % NZ] : 0.f;
          const float f = (VM == V_KIVI) ? ws.vb : 1.0f;  // units of coded values
          orow[c_lo] = ws.o[nt][mt][e] * f + z;
          orow[c_hi] = ws.o[nt][mt][2 + e] * f + z;
        }
      }
    }
  }
}

template <int BITS, int NT, int BASE, int MB>
__global__ void __launch_bounds__(kThreads, NT == 1 ? 4 : 2)
decode_kernel(const __grid_constant__ DecodeParams p) {
  extern __shared__ __align__(1024) char smem_raw[];
  // swizzled TMA boxes need 1024-byte aligned shared addresses
  char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const Dims& d = p.d;
  // Programmatic dependent launch: the next launch on the stream (the next
  // layer's or step's decode) may be scheduled as soon as every CTA of this
  // one runs; it builds its prologue from its parameters and waits (below)
  // before it touches memory that earlier kernels write.
  grid_launch_dependents();
  if ((int)blockIdx.x >= p.total_items) return;
  if (threadIdx.x == 0) {
    const uint32_t bars = smem_u32(smem + SmemLayout<NT>::bar);
    for (int s = 0; s < kMaxStages; ++s) mbar_init(bars + 8 * s, 1);
    mbar_init_fence();
    *reinterpret_cast<volatile int*>(smem + SmemLayout<NT>::bar + 8 * kMaxStages) = 0;  // abort flag
    prefetch_tensormap(&p.arena_map);
  }
  // (layer, batch row, KV head, chunk) of this CTA's item: a packed record
  // for host-ordered CTAs, else a search of the layer and head tables
  int li = 0, b, h, r;
  if ((int)blockIdx.x < p.n_order) {
    const uint32_t e = p.order[blockIdx.x];
    li = (int)(e & 63u);
    h = (int)((e >> 6) & 63u);
    r = (int)((e >> 12) & 31u);
    b = (int)(e >> 17);
  } else {
    const int item = (int)blockIdx.x;
    while (li + 1 < p.n_layers && p.layer[li + 1].item_base <= item) ++li;
    const DecodeLayer& L0 = p.layer[li];
    const int in_layer = item - L0.item_base;
    b = in_layer / L0.items_per_row;
    r = in_layer - b * L0.items_per_row;
    const ChunkCounts c0 = {L0.nbU, L0.nqU, L0.nqK, L0.nbP};
    for (h = 0; h < d.H; ++h) {
      int nb0;
      const int n0 = head_chunks(head_class(d, p.lt.mask[li], h), c0, &nb0);
      if (r < n0) break;
      r -= n0;
    }
  }
  const int G = d.G;
  const DecodeLayer& L = p.layer[li];
  const uint64_t mask = p.lt.mask[li];
  const ChunkCounts cc = {L.nbU, L.nqU, L.nqK, L.nbP};
  const int cls = head_class(d, mask, h);
  int nb;
  const int ni = head_chunks(cls, cc, &nb);
  const LayerGeom lg = layer_geom(d, mask);
  const HeadGeom hd = head_geom(d, lg, h);
  const char* Lb = p.arena + p.lt.base[li];
  // Everything above comes from the launch parameters.  From here on the CTA
  // reads the queries, the new K/V, the arena and the workspace, which the
  // kernels before this one on the stream write.
  grid_dependency_wait();
  // The queries are requested first: they gate every warp's first tile, and
  // their latency overlaps the first tile's copy.
  const uint16_t* qg = p.q + (((size_t)li * d.B + b) * d.Hq + (size_t)h * G) * kD;
  uint4 qv[QPieces<NT>::n];
#pragma unroll
  for (int k = 0; k < QPieces<NT>::n; ++k) {
    const int i = threadIdx.x + k * kThreads;
    qv[k] = (i < G * 16) ? ldg16(qg + i * 8) : make_uint4(0u, 0u, 0u, 0u);
  }
  const bool coded = r >= nb;
  int tb, te;
  if (!coded) {
    const int c = (cls == kProtected) ? p.plan.cbP : p.plan.cbU;
    tb = r * c;
    te = min(tb + c, hd.bf16_prefill + L.appended);
  } else {
    const int c = (cls == kKeysOnly) ? p.plan.cqK : p.plan.cqU;
    tb = (r - nb) * c;
    te = min(tb + c, ncoded(d));
  }
  const int tid = threadIdx.x;

  // the warps' (m, l, o) partials [warp][16][132], in the stage buffer once the
  // tiles are consumed (the same row layout as the split partials)
  float* parts = reinterpret_cast<float*>(smem + kStageOff);
  Seg sg;
  sg.k = sg.v = sg.kc = sg.km = sg.vc = sg.vm = nullptr;
  sg.new_pos = -1;
  sg.k_new = sg.v_new = nullptr;
  sg.k_row0 = sg.v_row0 = 0;
  if (!coded) {
    sg.k = Lb + hd.kb + b * hd.kb_bs;
    sg.v = Lb + hd.vb + b * hd.kb_bs;
    sg.k_row0 = (int)((p.lt.base[li] + hd.kb + b * hd.kb_bs) >> 8);
    sg.v_row0 = (int)((p.lt.base[li] + hd.vb + b * hd.kb_bs) >> 8);
    const int pos = hd.bf16_prefill + L.appended - 1;  // the step's new token
    if (p.k_new && pos >= tb && pos < te) {
      const size_t row = (((size_t)li * d.B + b) * d.H + h) * kD;
      sg.new_pos = pos;
      sg.k_new = reinterpret_cast<const char*>(p.k_new + row);
      sg.v_new = reinterpret_cast<const char*>(p.v_new + row);
      // this CTA alone owns the position in this launch: store it in the
      // arena, ordered before the TMA reads of its tile
      if (threadIdx.x < 32) {
        const int c = threadIdx.x & 15;
        const char* src = (threadIdx.x < 16) ? sg.k_new : sg.v_new;
        char* dst = const_cast<char*>((threadIdx.x < 16) ? sg.k : sg.v) + (size_t)pos * 256;
        *reinterpret_cast<uint4*>(dst + c * 16) = ldg16(src + c * 16);
        fence_proxy_async_global();
      }
    }
    __syncthreads();  // barriers initialised, new row stored
    run_item<BITS, NT, K_BF16, V_BF16, false, MB>(smem, sg, tb, te, p, qv, G, parts);
  } else if (hd.cls == kKeysOnly) {
    __syncthreads();  // barriers initialised
    sg.k = Lb + hd.kimg + b * hd.kimg_bs;
    sg.k_row0 = (int)((p.lt.base[li] + hd.kimg + b * hd.kimg_bs) >> 8);
    sg.vc = Lb + hd.vq + b * hd.vq_bs;
    sg.vm = Lb + hd.vqm + b * hd.vqm_bs;
    if (BASE == kKivi)
      run_item<BITS, NT, K_BF16, V_KIVI, false, MB>(smem, sg, tb, te, p, qv, G, parts);
    else
      run_item<BITS, NT, K_BF16, V_TOKEN, false, MB>(smem, sg, tb, te, p, qv, G, parts);
  } else {
    __syncthreads();  // barriers initialised
    sg.kc = Lb + hd.kq + b * hd.kq_bs;
    sg.km = Lb + hd.kqm + b * hd.kqm_bs;
    sg.vc = Lb + hd.vq + b * hd.vq_bs;
    sg.vm = Lb + hd.vqm + b * hd.vqm_bs;
    if (BASE == kKivi)
      run_item<BITS, NT, K_KIVI, V_KIVI, false, MB>(smem, sg, tb, te, p, qv, G, parts);
    else if (BASE == kAkvq)
      run_item<BITS, NT, K_TOKEN, V_TOKEN, true, MB>(smem, sg, tb, te, p, qv, G, parts);
    else
      run_item<BITS, NT, K_TOKEN, V_TOKEN, false, MB>(smem, sg, tb, te, p, qv, G, parts);
  }
  __syncthreads();

  // ---- combine the warps, then write the output (a head in one chunk) or this
  // split's partial; the last split of a head to finish then runs the same
  // combine over all splits' partials ----
  float* fw = reinterpret_cast<float*>(smem + SmemLayout<NT>::q);  // weights; queries no longer needed
  const size_t out_row = ((size_t)li * d.B + b) * d.Hq + (size_t)h * G;
  const size_t head_lin = ((size_t)li * d.B + b) * d.H + h;
  float* part = p.partials + (head_lin * p.max_items) * (size_t)G * kPartialStride;
  float* mine = part + (size_t)r * G * kPartialStride;
  __shared__ int s_last;
  const float* src = parts;
  int n = kWarps, sstride = kMaxG * kPartialStride;
  bool final = ni == 1;
#pragma unroll 1
  for (;;) {
    combine_pass<NT * 8>(src, n, sstride, fw, G, tid, final, p.out + out_row * kD, mine);
    if (final) break;

    // Publish the partial and take a ticket with one acquire-release atomic:
    // the CTA barrier orders every thread's stores before thread 0's release
    // (release is cumulative); for the last CTA, the acquire side orders the
    // other CTAs' partials before its reads (extended to its threads by the
    // second barrier).  No full device fence is needed.
    __syncthreads();
    if (tid == 0) {
      unsigned prev;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;\n"
                   : "=r"(prev)
                   : "l"(p.counters + head_lin)
                   : "memory");
      s_last = (prev == (unsigned)(ni - 1));
    }
    __syncthreads();
    if (!s_last) return;

    // Last CTA of the head: all ni partials in one asynchronous sweep into the
    // stage buffer (the plan keeps them within it).
    const int bytes = ni * G * kPartialStride * 4;
    const uint32_t buf_u32 = smem_u32(smem + kStageOff);
    const char* psrc = reinterpret_cast<const char*>(part);
#pragma unroll 1
    for (int off = tid * 16; off < bytes; off += kThreads * 16) cp_async16(buf_u32 + off, psrc + off, 16);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    src = reinterpret_cast<const float*>(smem + kStageOff);  // [ni][G][132]
    n = ni;
    sstride = G * kPartialStride;
    final = true;
  }
  if (ni > 1 && tid == 0) atomicExch(p.counters + head_lin, 0u);
}

template <int BITS, int NT, int BASE, int MB>
cudaError_t launch_t(const DecodeParams& p, int grid_x, cudaStream_t s) {
  // set once per device; host threads that race here both set the same
  // attributes, and the flags themselves are atomic
  static std::atomic<bool> configured[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
    e = cudaFuncSetAttribute(decode_kernel<BITS, NT, BASE, MB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             SmemLayout<NT>::bytes);
    if (e != cudaSuccess) return e;
    // four CTAs of 54 KB share an SM: ask for the full shared-memory carve-out
    e = cudaFuncSetAttribute(decode_kernel<BITS, NT, BASE, MB>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) configured[dev].store(true, std::memory_order_release);
  }
  (void)grid_x;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.total_items, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = SmemLayout<NT>::bytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decode_kernel<BITS, NT, BASE, MB>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int BITS, int NT, int MB>
cudaError_t launch_base(const DecodeParams& p, int grid_x, cudaStream_t s) {
  switch (p.d.base) {
    case kKivi: return launch_t<BITS, NT, kKivi, MB>(p, grid_x, s);
    case kAkvq: return launch_t<BITS, NT, kAkvq, MB>(p, grid_x, s);
    default: return launch_t<BITS, NT, kMinMax, MB>(p, grid_x, s);
  }
}

// Every kernel shape for one metadata width (MB bytes per {scale, zero} pair).
template <int MB>
cudaError_t launch_decode_mb(const DecodeParams& p, int grid_x, cudaStream_t s) {
  if (p.d.bits == 2)
    return p.d.G <= 8 ? launch_base<2, 1, MB>(p, grid_x, s) : launch_base<2, 2, MB>(p, grid_x, s);
  if (p.d.bits == 3)
    return p.d.G <= 8 ? launch_base<3, 1, MB>(p, grid_x, s) : launch_base<3, 2, MB>(p, grid_x, s);
  return p.d.G <= 8 ? launch_base<4, 1, MB>(p, grid_x, s) : launch_base<4, 2, MB>(p, grid_x, s);
}

}  // namespace
}  // namespace hg
