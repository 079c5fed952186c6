// Quantize-pack, dequantize and append kernels of the HeadGuard KV cache.
//
// Quantize (Sec. 3 "Applying protection" over the Sec. 1 / Sec. 4 bases).
// A CTA is one warp: it stages the K rows or the V rows of a 32-token tile of
// one (layer, batch row, KV head) in shared memory with coalesced asynchronous
// copies and then works one lane per vector: per-token min-max rows (Sec. 1),
// AKVQ-style rows (Sec. 4: keys rotated by the Hadamard-128 in registers
// first, a row over a lane pair), KIVI-style value rows (four 32-channel
// groups) and KIVI-style key groups (one lane per channel pair over the 32
// image tokens of the tile).  The head's class and the image span are
// resolved once per CTA, so protected heads and text tokens take a uniform
// BF16 copy path.  Codes, scales and zeros follow the group quantizer exactly
// (round half to even of the IEEE quotient, no contraction).
#include <algorithm>
#include <climits>

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "hg_common.cuh"
#include "hg_internal.h"
#include "hg_mma.cuh"

namespace hg {

namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ void bf16x4_to_f32(uint2 w, float (&x)[4]) {
  bf16x2_to_f32(w.x, x[0], x[1]);
  bf16x2_to_f32(w.y, x[2], x[3]);
}

// ---------------------------------------------------------------------------
// Per-token min-max base: one thread per (token, K or V) vector.
//
// A CTA takes the K rows or the V rows of 32 tokens of one (layer, row, KV
// head), staged in shared memory with coalesced loads (272-byte row pitch, so
// that a lane's 16-byte reads of its own row are conflict free); lane i owns
// row i.  A coded vector is quantized by its lane alone -- min / max over
// bf16x2 pairs (exact), then per element
//   T = RN(d * r + 192), d = fl(x - min), r = RN(1 / scale):
// T lies in [128, 256), so its low 16 mantissa bits hold d * r to 2^-16 and
// bits 16.. hold floor(d * r + 0.5) once 0x8000 is added.  Within 2^-16 of
// a half-integer the exact rule (round-half-even of fl(d / scale)) may differ,
// so such an element takes one IEEE division (BF16 inputs make exact
// half-integer quotients common, so this is per element, not per vector).  The
// bound: |d r - d / scale| <= 16 * 2^-24 and the FMA and the reference
// quotient each round by at most 2^-17, so any element whose low bits are not
// within one unit of 0x8000 rounds the same way as the reference.
// Uncoded vectors (text, protected heads, keys of keys-only heads) are copied.
// ---------------------------------------------------------------------------
constexpr int kQTok = 32;
constexpr int kQPitch = 272;

// Round-half-even of fl(d / scale), clamped to the levels (IEEE division).
__device__ __noinline__ uint32_t exact_code(float d, float scale, float levels) {
  return (uint32_t)fminf(fmaxf(rintf(__fdiv_rn(d, scale)), 0.0f), levels);
}

// The packed bits of one 8-channel chunk: `lo` its 32 (4-bit) or 16 (2- and
// 3-bit) low code bits in channel order, `hb` its 8 bit-2 bits (3-bit).
template <int BITS>
__device__ __forceinline__ void chunk_bits(const uint32_t (&c)[8], uint32_t& lo, uint32_t& hb) {
  lo = 0u;
  hb = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    lo |= (BITS == 4) ? (c[i] << (4 * i)) : ((c[i] & 3u) << (2 * i));
    if (BITS == 3) hb |= ((c[i] >> 2) & 1u) << i;
  }
}

// The same from the eight T' words of the fast rule (code in bits 16..): each
// code is shifted straight into its packed position (one shift and one
// and-or per element instead of extracting it first).
template <int BITS>
__device__ __forceinline__ void chunk_bits_T(const uint32_t (&a)[8], uint32_t& lo, uint32_t& hb) {
  lo = 0u;
  hb = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (BITS == 4) {
      const uint32_t x = (4 * i >= 16) ? (a[i] << (4 * i - 16)) : (a[i] >> (16 - 4 * i));
      lo |= x & (15u << (4 * i));
    } else {
      lo |= (a[i] >> (16 - 2 * i)) & (3u << (2 * i));
      if (BITS == 3) hb |= (a[i] >> (18 - i)) & (1u << i);
    }
  }
}

// Chunks kg..kg+3 (kg a multiple of 4) into the packed row, one vector store
// per word run: 4 bits -> words kg..kg+3 (16 bytes); 2 and 3 bits -> words
// kg/2, kg/2 + 1 (8 bytes, chunk k in half k % 2 of word k / 2); 3 bits also
// plane word 8 + kg/4, chunk k's bit-2 byte at ((k >> 1) & 1) | ((k & 1) << 1)
// (channel index bits 3 and 4 exchanged).  A packed row is 16 x bits bytes on
// a 16-byte boundary.
template <int BITS>
__device__ __forceinline__ void store_group(int kg, const uint32_t (&lo)[4], const uint32_t (&hb)[4],
                                            uint32_t* codes) {
  if (BITS == 4) {
    *reinterpret_cast<uint4*>(codes + kg) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    return;
  }
  *reinterpret_cast<uint2*>(codes + (kg >> 1)) = make_uint2(lo[0] | (lo[1] << 16), lo[2] | (lo[3] << 16));
  if (BITS == 3) codes[8 + (kg >> 2)] = hb[0] | (hb[2] << 8) | (hb[1] << 16) | (hb[3] << 24);
}

// T' = RN(fl(x - min) r + C) for the four channel pairs of a chunk (the fast
// rule of chunk_codes), element 2i + j from half j of pair i.  Returns true
// when no element has T' low bits in [0, 7] (then every code is bits 16.. of
// T'); false when some element is near a tie and must take the exact rule.
__device__ __forceinline__ bool chunk_T(const uint64_t (&x2)[4], uint64_t mn2, uint64_t r2, uint64_t c2,
                                        uint32_t (&a)[8]) {
  uint32_t low = 0xffffffffu;  // per 16-bit half: the smallest low bits seen
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint64_t t2 = f32x2_fma(f32x2_sub(x2[i], mn2), r2, c2);
    a[2 * i] = (uint32_t)t2;
    a[2 * i + 1] = (uint32_t)(t2 >> 32);
    low = __vminu2(low, __byte_perm(a[2 * i], a[2 * i + 1], 0x5410));
  }
  return __vcmpleu2(low, 0x00070007u) == 0u;
}

// Code e (0..31, token order) of one KIVI-style key group row into its packed
// words: 2 / 4 bits at word e / (32 / bits), bit bits * (e mod 32 / bits); 3
// bits: bits 0-1 at word e / 16, bit 2 e mod 16, and bit 2 into plane word 2 at
// bit e with index bits 3 and 4 exchanged.  e is a compile-time constant after
// unrolling, so each is one shift and one or.
template <int BITS>
__device__ __forceinline__ void add_key_code(uint32_t (&wd)[BITS], int e, uint32_t c) {
  if (BITS == 3) {
    wd[e / 16] |= (c & 3u) << (2 * (e % 16));
    wd[2] |= ((c >> 2) & 1u) << ((e & 7) | (((e >> 4) & 1) << 3) | (((e >> 3) & 1) << 4));
  } else {
    constexpr int per = 32 / (BITS == 3 ? 2 : BITS);
    wd[e / per] |= c << (BITS * (e % per));
  }
}

// Two adjacent channels (2c, 2c + 1) of one KIVI-style key group: the 32
// bf16x2 words of the group's tokens at `col` (the group's first staged row,
// then a row pitch apart).  min / max of both channels at once over bf16x2
// pairs (exact); with fp32 metadata and both steps at least 2^-125, the codes
// of both channels come from the paired rule of the token rows (per-lane
// minimum and reciprocal), otherwise each channel takes the scalar group
// quantizer.  Codes and metadata as for one channel.
template <int BITS, bool M16>
__device__ __forceinline__ void quantize_key_pair(const char* col, uint32_t* dst0, uint32_t* dst1, char* meta,
                                                  size_t mi) {
  uint32_t w[kKiviGroup];
#pragma unroll
  for (int e = 0; e < kKiviGroup; ++e) w[e] = *reinterpret_cast<const uint32_t*>(col + (size_t)e * kQPitch);
  __nv_bfloat162 mn2 = *reinterpret_cast<const __nv_bfloat162*>(&w[0]), mx2 = mn2;
#pragma unroll
  for (int e = 1; e < kKiviGroup; ++e) {
    const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[e]);
    mn2 = __hmin2(mn2, h);
    mx2 = __hmax2(mx2, h);
  }
  constexpr uint32_t L = (1u << BITS) - 1u;
  const float levels = (float)L;
  float mn[2] = {__fadd_rn(__low2float(mn2), 0.0f), __fadd_rn(__high2float(mn2), 0.0f)};
  const float mx[2] = {__fadd_rn(__low2float(mx2), 0.0f), __fadd_rn(__high2float(mx2), 0.0f)};
  float sc[2];
  bool fast = true;  // both channels: the fast rule applies (see quantize_row_group)
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    sc[j] = __fdiv_rn(__fsub_rn(mx[j], mn[j]), levels);
    const float mn_x = mn[j];
    if (M16) {
      sc[j] = half_sat(sc[j]);
      mn[j] = half_sat(mn[j]);
      if (sc[j] > 0.0f) {
        const float rj = __frcp_rn(sc[j]);
        const float qlo = __fmul_rn(__fsub_rn(mn_x, mn[j]), rj), qhi = __fmul_rn(__fsub_rn(mx[j], mn[j]), rj);
        fast = fast && qlo > -0.25f && qhi < levels + 0.25f;
      } else {
        fast = false;
      }
    } else {
      fast = fast && sc[j] >= 2.3509887e-38f;
    }
    store_meta(meta, mi + j, sc[j], mn[j], M16);
  }
  uint32_t wd0[BITS], wd1[BITS];  // the two channels' packed words, filled code by code
#pragma unroll
  for (int i = 0; i < BITS; ++i) wd0[i] = wd1[i] = 0u;
  if (fast) {
    const float r0 = __frcp_rn(sc[0]), r1 = __frcp_rn(sc[1]);
    const uint64_t mn2p = f32x2(__float_as_uint(mn[0]), __float_as_uint(mn[1]));
    const uint64_t r2 = f32x2(__float_as_uint(r0), __float_as_uint(r1));
    const uint32_t cbits = __float_as_uint(192.50006103515625f);  // 192.5 + 4 * 2^-16 (see chunk_codes)
    const uint64_t c2 = f32x2(cbits, cbits);
#pragma unroll
    for (int e = 0; e < kKiviGroup; ++e) {
      const uint64_t t2 = f32x2_fma(f32x2_sub(f32x2(w[e] << 16, w[e] & 0xffff0000u), mn2p), r2, c2);
      const uint32_t a0 = (uint32_t)t2, a1 = (uint32_t)(t2 >> 32);
      uint32_t k0 = (a0 >> 16) & L, k1 = (a1 >> 16) & L;
      if (!(a0 & 0xfff8u)) k0 = exact_code(__fsub_rn(__uint_as_float(w[e] << 16), mn[0]), sc[0], levels);
      if (!(a1 & 0xfff8u)) k1 = exact_code(__fsub_rn(__uint_as_float(w[e] & 0xffff0000u), mn[1]), sc[1], levels);
      add_key_code<BITS>(wd0, e, k0);
      add_key_code<BITS>(wd1, e, k1);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const bool fast = sc[j] >= 2.3509887e-38f;  // 2^-125
      const float r = __frcp_rn(fast ? sc[j] : 1.0f);
#pragma unroll
      for (int e = 0; e < kKiviGroup; ++e) {
        const float x = __uint_as_float(j ? (w[e] & 0xffff0000u) : (w[e] << 16));
        const uint32_t c = (sc[j] == 0.0f) ? 0u : code_of(__fsub_rn(x, mn[j]), sc[j], r, levels, fast);
        if (j) add_key_code<BITS>(wd1, e, c);
        else add_key_code<BITS>(wd0, e, c);
      }
    }
  }
  // both channels' rows are contiguous (dst1 = dst0 + BITS) and start on a
  // 16-byte (2, 4 bits) or 8-byte (3 bits) boundary: vector stores
  if (BITS == 3) {
    uint2* d2 = reinterpret_cast<uint2*>(dst0);
    d2[0] = make_uint2(wd0[0], wd0[1]);
    d2[1] = make_uint2(wd0[2 % BITS], wd1[0]);
    d2[2] = make_uint2(wd1[1], wd1[2 % BITS]);
  } else {
    uint4* d4 = reinterpret_cast<uint4*>(dst0);
    if (BITS == 2) {
      d4[0] = make_uint4(wd0[0], wd0[1 % BITS], wd1[0], wd1[1 % BITS]);
    } else {
      d4[0] = make_uint4(wd0[0], wd0[1 % BITS], wd0[2 % BITS], wd0[3 % BITS]);
      d4[1] = make_uint4(wd1[0], wd1[1 % BITS], wd1[2 % BITS], wd1[3 % BITS]);
    }
  }
}

// Codes of the 8 channels of one chunk (four BF16 pairs w[0..3]) in a group
// with minimum mn and step scale > 0, r = RN(1 / scale):
//   M16 (binary16 metadata, always a normal r): a binary16 scale is at least
//     2^-24, so r is finite.  The rounded zero and scale can put a quotient
//     outside [0, levels]: q = d r is clamped to [-1, levels + 1] (which
//     decides no code differently), then T = RN(q + 192) lies in
//     [191, 193 + levels] and bits 16.. of T + 0x8001, less 0x4340, are the
//     unclamped code.  The two roundings (q, then T) keep T within 2^-16 of
//     fl(d / scale) + 192 for quotients that can decide a code, so an element
//     whose low bits are not within one unit of 0x8000 rounds as the exact
//     rule does; the others take it.
//   fast (scale >= 2^-125, 1 / scale finite): two channels per paired
//     operation, d = fl(x - min), then T' = RN(d r + C) with
//     C = 192.5 + 4 * 2^-16.  In [128, 256) the grid is 2^-16, so T' is
//     T = RN(d r + 192) moved by 0x8004 units (one unit more or less when
//     d r + 192 falls exactly between two grid points, where the shift by an
//     even count flips the tie-break).  Bits 16.. of T' are then
//     floor(d r + 0.5) away from ties, and the error of T' against the exact
//     quotient is below two units (0.5 FMA rounding, 1/16 for r, 1/16 for the
//     reference division, 1 for the tie-break), so every element within two
//     units of the half-integer boundary -- T' low bits in [2, 6] -- is among
//     those with low bits in [0, 7], which take the exact rule (chunk_T,
//     chunk_bits_T; a chunk with such an element goes through chunk_near_tie).
//   otherwise (tiny scale): the exact rule for every element.
template <int BITS, bool M16>
__device__ __forceinline__ void chunk_codes(const uint32_t (&w)[4], float mn, float scale, float r,
                                            uint32_t (&c8)[8]) {
  constexpr uint32_t L = (1u << BITS) - 1u;
  const float levels = (float)L;
  if constexpr (M16) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t hw = w[i >> 1];
      const float d = __fsub_rn(__uint_as_float((i & 1) ? (hw & 0xffff0000u) : (hw << 16)), mn);
      const float q = fminf(fmaxf(__fmul_rn(d, r), -1.0f), levels + 1.0f);
      const uint32_t a = __float_as_uint(__fadd_rn(q, 192.0f)) + 0x8001u;
      const int cu = min(max((int)(a >> 16) - 0x4340, 0), (int)L);
      c8[i] = ((a & 0xffffu) < 3u) ? exact_code(d, scale, levels) : (uint32_t)cu;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t hw = w[i >> 1];
      const float x = __uint_as_float((i & 1) ? (hw & 0xffff0000u) : (hw << 16));
      c8[i] = exact_code(__fsub_rn(x, mn), scale, levels);
    }
  }
}

// Codes of a chunk that has an element near a tie: bits 16.. of T' for the
// others, the exact rule for the elements with T' low bits in [0, 7].
// x(i) gives element i's value.
template <int BITS, class X>
__device__ __forceinline__ void chunk_near_tie(const uint32_t (&a)[8], X x, float mn, float scale,
                                               uint32_t (&c8)[8]) {
  constexpr uint32_t L = (1u << BITS) - 1u;
#pragma unroll
  for (int i = 0; i < 8; ++i)
    c8[i] = (a[i] & 0xfff8u) ? ((a[i] >> 16) & L) : exact_code(__fsub_rn(x(i), mn), scale, (float)L);
}

// Chunk k's codes written over its bits of a packed row that this thread has
// already stored: word k (4 bits), or half k % 2 of word k / 2 (2 and 3 bits)
// and, at 3 bits, byte ((k >> 1) & 1) | ((k & 1) << 1) of plane word 8 + k / 4
// (the layout of store_group).  The other chunks' bits are read back.
template <int BITS>
__device__ __forceinline__ void patch_chunk(int k, const uint32_t (&c)[8], uint32_t* codes) {
  uint32_t lo = 0u, hb = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    lo |= (BITS == 4) ? (c[i] << (4 * i)) : ((c[i] & 3u) << (2 * i));
    if (BITS == 3) hb |= ((c[i] >> 2) & 1u) << i;
  }
  if (BITS == 4) {
    codes[k] = lo;
    return;
  }
  const int sh = 16 * (k & 1);
  codes[k >> 1] = (codes[k >> 1] & ~(0xffffu << sh)) | (lo << sh);
  if (BITS == 3) {
    const int pb = 8 * (((k >> 1) & 1) | ((k & 1) << 1));
    codes[8 + (k >> 2)] = (codes[8 + (k >> 2)] & ~(0xffu << pb)) | (hb << pb);
  }
}

// One group of a BF16 row: chunks [k0, k0 + nk) (8 channels each) with their
// min / max over bf16x2 pairs (exact), signed zeros folded to +0,
// scale = fl((max - min) / levels), metadata stored at index mi (binary16
// pair with M16: codes against the rounded pair), codes 0 when scale == 0.
// The chunks go in groups of four (a KIVI-style value group whole), each
// group's packed words written by one vector store (store_group); the group
// loop stays rolled so that the code stays small in the instruction cache
// (eight chunks per step measured slower on the per-token rows).
// A chunk with an element near a tie (fast rule) is emitted with its fast
// codes and flagged; after the loop each thread codes its flagged chunks again,
// the flagged elements by the exact rule, and writes each chunk's bits over
// the stored ones (patch_chunk).  The threads of a warp do this side by side,
// so a warp pays for the largest number of flagged chunks of one thread
// instead of running every thread's near ties one after another inside the
// loop.
template <int BITS, bool M16>
__device__ __forceinline__ void quantize_row_group(const uint4* r4, int k0, int nk, uint32_t* codes, char* meta,
                                                   size_t mi) {
  __nv_bfloat162 mn2, mx2;
  {
    const uint4 v = r4[k0];
    mn2 = mx2 = *reinterpret_cast<const __nv_bfloat162*>(&v.x);
  }
#pragma unroll 4
  for (int k = k0; k < k0 + nk; ++k) {
    const uint4 v = r4[k];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
      mn2 = __hmin2(mn2, h);
      mx2 = __hmax2(mx2, h);
    }
  }
  float mn = fminf(__low2float(mn2), __high2float(mn2));
  float mx = fmaxf(__low2float(mx2), __high2float(mx2));
  mn = __fadd_rn(mn, 0.0f);  // -0 -> +0
  mx = __fadd_rn(mx, 0.0f);
  const float levels = (float)((1u << BITS) - 1u);
  float scale = __fdiv_rn(__fsub_rn(mx, mn), levels);
  const float mn_x = mn;  // the group's own minimum
  if (M16) {  // binary16 metadata: codes against the stored pair
    scale = half_sat(scale);
    mn = half_sat(mn);
  }
  store_meta(meta, mi, scale, mn, M16);
  bool fast = !M16 && scale >= 2.3509887e-38f;  // 2^-125: 1 / scale is finite
  const float r = (M16 || fast) ? __frcp_rn(scale) : 1.0f;
  if (M16 && scale > 0.0f) {
    // With the rounded pair the quotients fl(fl(x - min16) r) of the group run
    // monotonically from the group minimum's to the maximum's.  When both lie
    // well inside (-1/2, levels + 1/2), every code is in [0, levels] without a
    // clamp, and the fast rule of the fp32 pairs (exact against the IEEE
    // quotient, with the same near-tie window) applies to the stored pair.
    const float qlo = __fmul_rn(__fsub_rn(mn_x, mn), r), qhi = __fmul_rn(__fsub_rn(mx, mn), r);
    fast = qlo > -0.25f && qhi < levels + 0.25f;
  }
  const uint64_t mnp = f32x2(__float_as_uint(mn), __float_as_uint(mn));
  const uint64_t r2 = f32x2(__float_as_uint(r), __float_as_uint(r));
  const uint32_t cbits = __float_as_uint(192.50006103515625f);  // C = 192.5 + 4 * 2^-16
  const uint64_t c2 = f32x2(cbits, cbits);
  uint32_t ties = 0u;  // bit k - k0: chunk k has an element near a tie
#pragma unroll 1
  for (int kg = k0; kg < k0 + nk; kg += 4) {
    uint32_t lo[4], hb[4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k = kg + kk;
      const uint4 v = r4[k];
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
      if (fast) {
        uint64_t x2[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) x2[i] = f32x2(w[i] << 16, w[i] & 0xffff0000u);  // channels 2i, 2i + 1
        uint32_t a[8];
        if (!chunk_T(x2, mnp, r2, c2, a)) ties |= 1u << (k - k0);  // about one chunk in 100
        chunk_bits_T<BITS>(a, lo[kk], hb[kk]);
      } else {
        uint32_t c8[8];
        if (scale == 0.0f) {  // constant group (or a step below binary16 range): every code 0
#pragma unroll
          for (int i = 0; i < 8; ++i) c8[i] = 0u;
        } else {
          chunk_codes<BITS, M16>(w, mn, scale, r, c8);
        }
        chunk_bits<BITS>(c8, lo[kk], hb[kk]);
      }
    }
    store_group<BITS>(kg, lo, hb, codes);
  }
  while (ties) {
    const int k = k0 + (__ffs(ties) - 1);
    ties &= ties - 1;
    const uint4 v = r4[k];
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint64_t x2[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x2[i] = f32x2(w[i] << 16, w[i] & 0xffff0000u);
    uint32_t a[8], c8[8];
    chunk_T(x2, mnp, r2, c2, a);
    chunk_near_tie<BITS>(a, [&](int i) { return __uint_as_float((i & 1) ? (w[i >> 1] & 0xffff0000u) : (w[i >> 1] << 16)); },
                         mn, scale, c8);
    patch_chunk<BITS>(k, c8, codes);
  }
}

// Per-token min-max over the whole 128-channel row (Sec. 1), one group.
template <int BITS, bool M16>
__device__ __forceinline__ void quantize_row_token(const char* row_s, uint32_t* codes, char* meta, size_t mi) {
  quantize_row_group<BITS, M16>(reinterpret_cast<const uint4*>(row_s), 0, 16, codes, meta, mi);
}

// KIVI-style values (Sec. 4): four groups of 32 channels per token
// (metadata mi .. mi + 3); the packing is the per-token one (channel order).
template <int BITS, bool M16>
__device__ __forceinline__ void quantize_row_kivi_v(const char* row_s, uint32_t* codes, char* meta, size_t mi) {
#pragma unroll 1
  for (int j = 0; j < 4; ++j)
    quantize_row_group<BITS, M16>(reinterpret_cast<const uint4*>(row_s), 4 * j, 4, codes, meta, mi + j);
}

// ---------------------------------------------------------------------------
// AKVQ-style keys (Sec. 4): the BF16 row is widened into 64 packed fp32 pairs
// (channels 2m, 2m + 1), rotated by the normalised Hadamard-128 in registers
// -- stage h = 1 inside each pair, stages h = 2..64 on whole pairs (both
// halves of a pair meet the same partner offset), the 1/sqrt(128) factor once
// at the end, the same butterflies in the same order as the warp-wide
// transform -- and quantized per token like the min-max rows above, with the
// same exact code rule.  SPLIT = 2 spreads a row over the lanes hh = 0, 1 of
// a lane pair (pmask): lane hh holds pairs 32 hh .. 32 hh + 31 (channels
// 64 hh ..), runs stages 2..32 alone, meets its partner for stage 64 and for
// the row's min / max by shuffles, and codes chunks 8 hh .. 8 hh + 7 into its
// own words of the packed row (lane 0 stores the metadata).  Half the pairs
// per thread: twice the rows resident.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float pair_lo(uint64_t x) { return __uint_as_float((uint32_t)x); }
__device__ __forceinline__ float pair_hi(uint64_t x) { return __uint_as_float((uint32_t)(x >> 32)); }

__device__ __forceinline__ uint64_t shfl_xor_pair(unsigned mask, uint64_t x, int m) {
  const uint32_t lo = __shfl_xor_sync(mask, (uint32_t)x, m), hi = __shfl_xor_sync(mask, (uint32_t)(x >> 32), m);
  return ((uint64_t)hi << 32) | lo;
}

template <int BITS, bool M16, int SPLIT>
__device__ __forceinline__ void quantize_row_rotated(const char* row_s, int hh, unsigned pmask, uint32_t* codes,
                                                     char* meta, size_t mi) {
  constexpr int NP = 64 / SPLIT;  // pairs per thread
  constexpr int NK = 16 / SPLIT;  // chunks per thread
  const uint32_t* r32 = reinterpret_cast<const uint32_t*>(row_s) + NP * hh;
  const int k0 = NK * hh;
  uint64_t xp[NP];
#pragma unroll
  for (int m = 0; m < NP; ++m) {
    const uint32_t w = r32[m];
    const float a = __uint_as_float(w << 16), b = __uint_as_float(w & 0xffff0000u);
    xp[m] = f32x2(__float_as_uint(__fadd_rn(a, b)), __float_as_uint(__fsub_rn(a, b)));  // stage h = 1
  }
#pragma unroll
  for (int hp = 1; hp < NP; hp <<= 1) {  // stage h = 2 hp
#pragma unroll
    for (int m = 0; m < NP; ++m) {
      if (m & hp) continue;
      const uint64_t a = xp[m], b = xp[m + hp];
      xp[m] = f32x2_add(a, b);
      xp[m + hp] = f32x2_sub(a, b);
    }
  }
  if (SPLIT == 2) {  // stage h = 64: pair m of lane 0 with pair m of lane 1
#pragma unroll
    for (int m = 0; m < NP; ++m) {
      const uint64_t o = shfl_xor_pair(pmask, xp[m], 1);
      xp[m] = hh ? f32x2_sub(o, xp[m]) : f32x2_add(xp[m], o);
    }
  }
  {
    const uint32_t cb = __float_as_uint(hadamard_c());
    const uint64_t c2 = f32x2(cb, cb);
#pragma unroll
    for (int m = 0; m < NP; ++m) xp[m] = f32x2_mul(xp[m], c2);
  }
  // min / max of the rotated vector (exact; signed zeros folded to +0)
  float mn = fminf(pair_lo(xp[0]), pair_hi(xp[0])), mx = fmaxf(pair_lo(xp[0]), pair_hi(xp[0]));
  {
    float mn1 = fminf(pair_lo(xp[1]), pair_hi(xp[1])), mx1 = fmaxf(pair_lo(xp[1]), pair_hi(xp[1]));
#pragma unroll
    for (int m = 2; m < NP; m += 2) {
      mn = fminf(mn, fminf(pair_lo(xp[m]), pair_hi(xp[m])));
      mx = fmaxf(mx, fmaxf(pair_lo(xp[m]), pair_hi(xp[m])));
      mn1 = fminf(mn1, fminf(pair_lo(xp[m + 1]), pair_hi(xp[m + 1])));
      mx1 = fmaxf(mx1, fmaxf(pair_lo(xp[m + 1]), pair_hi(xp[m + 1])));
    }
    mn = fminf(mn, mn1);
    mx = fmaxf(mx, mx1);
  }
  if (SPLIT == 2) {
    mn = fminf(mn, __shfl_xor_sync(pmask, mn, 1));
    mx = fmaxf(mx, __shfl_xor_sync(pmask, mx, 1));
  }
  mn = __fadd_rn(mn, 0.0f);
  mx = __fadd_rn(mx, 0.0f);
  constexpr uint32_t L = (1u << BITS) - 1u;
  const float levels = (float)L;
  float scale = __fdiv_rn(__fsub_rn(mx, mn), levels);
  const float mn_x = mn;
  if (M16) {
    scale = half_sat(scale);
    mn = half_sat(mn);
  }
  if (hh == 0) store_meta(meta, mi, scale, mn, M16);
  uint32_t lo[NK], hb[NK];  // this thread's chunks k0..k0+NK-1, stored four at a time at the end
  auto store_all = [&]() {
#pragma unroll
    for (int g = 0; g < NK / 4; ++g) {
      const uint32_t l4[4] = {lo[4 * g], lo[4 * g + 1], lo[4 * g + 2], lo[4 * g + 3]};
      const uint32_t h4[4] = {hb[4 * g], hb[4 * g + 1], hb[4 * g + 2], hb[4 * g + 3]};
      store_group<BITS>(k0 + 4 * g, l4, h4, codes);
    }
  };
  if (scale == 0.0f) {
#pragma unroll
    for (int k = 0; k < NK; ++k) lo[k] = hb[k] = 0u;
    store_all();
    return;
  }
  bool fast = scale >= 2.3509887e-38f;  // the fast rule of the min-max rows (chunk_T)
  if (M16) {  // with the stored pair: when every quotient is well inside the levels (quantize_row_group)
    const float r = __frcp_rn(scale);
    const float qlo = __fmul_rn(__fsub_rn(mn_x, mn), r), qhi = __fmul_rn(__fsub_rn(mx, mn), r);
    fast = qlo > -0.25f && qhi < levels + 0.25f;
  }
  if (M16 && !fast) {  // as the min-max rows: the quotient clamped, then the same near-tie rule
    const float r = __frcp_rn(scale);
#pragma unroll
    for (int k = 0; k < NK; ++k) {
      uint32_t c8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const uint64_t x2 = xp[4 * k + (i >> 1)];
        const float d = __fsub_rn((i & 1) ? pair_hi(x2) : pair_lo(x2), mn);
        const float q = fminf(fmaxf(__fmul_rn(d, r), -1.0f), levels + 1.0f);
        const uint32_t a = __float_as_uint(__fadd_rn(q, 192.0f)) + 0x8001u;
        const int cu = min(max((int)(a >> 16) - 0x4340, 0), (int)L);
        c8[i] = ((a & 0xffffu) < 3u) ? exact_code(d, scale, levels) : (uint32_t)cu;
      }
      chunk_bits<BITS>(c8, lo[k], hb[k]);
    }
    store_all();
    return;
  }
  if (fast) {  // the fast rule of the min-max rows (chunk_T)
    const float r = __frcp_rn(scale);
    const uint64_t mn2 = f32x2(__float_as_uint(mn), __float_as_uint(mn));
    const uint64_t r2 = f32x2(__float_as_uint(r), __float_as_uint(r));
    const uint32_t cbits = __float_as_uint(192.50006103515625f);  // 192.5 + 4 * 2^-16
    const uint64_t c2 = f32x2(cbits, cbits);
#pragma unroll
    for (int k = 0; k < NK; ++k) {
      const uint64_t x2[4] = {xp[4 * k], xp[4 * k + 1], xp[4 * k + 2], xp[4 * k + 3]};
      uint32_t a[8];
      if (chunk_T(x2, mn2, r2, c2, a)) {
        chunk_bits_T<BITS>(a, lo[k], hb[k]);
      } else {
        uint32_t c8[8];
        chunk_near_tie<BITS>(a, [&](int i) { return (i & 1) ? pair_hi(x2[i >> 1]) : pair_lo(x2[i >> 1]); }, mn,
                             scale, c8);
        chunk_bits<BITS>(c8, lo[k], hb[k]);
      }
    }
    store_all();
    return;
  }
#pragma unroll
  for (int k = 0; k < NK; ++k) {  // tiny scale: the exact rule throughout
    uint32_t c8[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint64_t x2 = xp[4 * k + (i >> 1)];
      c8[i] = exact_code(__fsub_rn((i & 1) ? pair_hi(x2) : pair_lo(x2), mn), scale, levels);
    }
    chunk_bits<BITS>(c8, lo[k], hb[k]);
  }
  store_all();
}

// A BF16 row copied as it is (SPLIT = 2: lane hh of a pair copies its half).
template <int SPLIT = 1>
__device__ __forceinline__ void copy_row(char* dst, const char* row_s, int hh = 0) {
#pragma unroll
  for (int k = 0; k < 16 / SPLIT; ++k) {
    const int c = (16 / SPLIT) * hh + k;
    reinterpret_cast<uint4*>(dst)[c] = reinterpret_cast<const uint4*>(row_s)[c];
  }
}

// Staged rows of one warp tile: row r < n holds token t0 + r, 272-byte pitch.
using StagedRows = char[kQTok][kQPitch];

// Rows 0..n-1 of a tile to n consecutive BF16 rows at dst, by the whole warp:
// lane l stores chunk l % 16 of rows l / 16, l / 16 + 2, ... (512 contiguous
// bytes per store instruction).
__device__ __forceinline__ void copy_rows_warp(char* dst, const StagedRows& rows, int n) {
  const int col = threadIdx.x & 15;
#pragma unroll
  for (int i = 0; i < kQTok / 2; ++i) {
    const int r = (threadIdx.x >> 4) + 2 * i;
    if (r < n)
      *reinterpret_cast<uint4*>(dst + (size_t)r * 256 + col * 16) = *reinterpret_cast<const uint4*>(&rows[r][col * 16]);
  }
}

// Token span of a tile: rows r < n hold tokens t0 + r.
struct TileSpan {
  int t0, n, tlo;  // tlo: the unclipped tile start (KIVI-style tiles)
};

// Coalesced staging of one part (K or V rows) of a tile by the CTA's warp:
// lane l copies 16-byte chunks l, l + 32, ... of the tile's contiguous rows
// (every chunk in flight at once); the caller commits the group.
__device__ __forceinline__ void stage_rows(const QuantizeParams& p, int li, int b, int h, int kv, const TileSpan& sp,
                                           StagedRows& rows) {
  const Dims& d = p.d;
  const size_t row0 = ((size_t)b * d.H + h) * (size_t)d.T + sp.t0;
  const int col = threadIdx.x & 15;  // lane l: chunk l % 16 of rows l / 16, l / 16 + 2, ...
  const char* src = reinterpret_cast<const char*>((kv ? p.v[li] : p.k[li]) + row0 * kD) + col * 16;
#pragma unroll
  for (int i = 0; i < kQTok / 2; ++i) {
    const int r = (threadIdx.x >> 4) + 2 * i;
    if (r < sp.n) cp_async16(smem_u32(&rows[r][col * 16]), src + (size_t)r * 256, 16);
  }
}

// A tile whose rows all go, as they are, to consecutive BF16 rows -- a
// protected K+V head, a tile inside one text run, or the image keys of a
// keys-only head -- copied by the whole warp, two rows per store instruction,
// instead of each lane storing its own row in sixteen pieces.  Returns false
// for any other tile (the rows' own paths then run).  Salient tokens sit in
// coded image spans only, so a text run keeps consecutive positions.  (The
// per-token tiles use it; in the KIVI-style kernels, whose code is longer,
// the extra copy path measured 8% slower.)
__device__ __forceinline__ bool copy_tile_whole(const QuantizeParams& p, int li, int b, int kv, const TileSpan& sp,
                                                const StagedRows& rows, const HeadGeom& hd) {
  const Dims& d = p.d;
  const int qs = d.s, qe = d.s + d.nq, t0 = sp.t0, t1 = sp.t0 + sp.n;
  char* Lb = p.arena + p.lt.base[li];
  const char* dst;
  if (hd.cls == kProtected || t1 <= qs || t0 >= qe)
    dst = Lb + (kv ? hd.vb : hd.kb) + b * hd.kb_bs + (size_t)bf16_pos(d, hd.cls, t0) * 256;
  else if (kv == 0 && hd.cls == kKeysOnly && t0 >= qs && t1 <= qe && d.ns == 0)
    dst = Lb + hd.kimg + b * hd.kimg_bs + (size_t)(t0 - qs) * 256;
  else
    return false;
  copy_rows_warp(const_cast<char*>(dst), rows, sp.n);
  return true;
}

// The per-token bases, one thread per vector: min-max rows (Sec. 1) and
// AKVQ-style rows (Sec. 4: keys rotated first; values per token, unrotated).
// Tiles of 32 tokens from token 0; a CTA (one warp) takes the K rows or the V
// rows of a tile (PARTS 1: K only, 2: V only, 3: both, as two CTAs).  With
// salient tokens (AKVQ-style, Sec. 4) a thread finds its token in the head's
// map: a salient token's K and V rows go to the BF16 region at position
// s + (its rank), every other image token to coded slot ti - (the salient
// tokens before it).
template <int BITS, bool M16, int BASE, int PARTS>
struct TokenTiles {
  static constexpr int kNParts = PARTS == 3 ? 2 : 1;
  static __device__ __forceinline__ int part(int i) { return PARTS == 3 ? i : (PARTS == 1 ? 0 : 1); }
  static __device__ __forceinline__ TileSpan span(const QuantizeParams& p, int tx) {
    TileSpan sp;
    sp.t0 = sp.tlo = tx * kQTok;
    sp.n = min(kQTok, p.d.T - sp.t0);
    return sp;
  }
  // Row r of the tile; SPLIT = 2: lane hh of the row's lane pair (pmask).
  template <int SPLIT>
  static __device__ __forceinline__ void row(const QuantizeParams& p, int li, int b, int kv, const TileSpan& sp,
                                             const StagedRows& rows, const HeadGeom& hd, int r, int hh,
                                             unsigned pmask) {
    const Dims& d = p.d;
    char* Lb = p.arena + p.lt.base[li];
    const int t = sp.t0 + r;
    const bool coded = t >= d.s && t < d.s + d.nq;
    const int ti = t - d.s;
    int ci = ti, pos = bf16_pos(d, hd.cls, t);
    bool sal = false;
    if (BASE == kAkvq && coded && d.ns > 0 && hd.cls != kProtected) {
      const char* sm = Lb + hd.sal + b * hd.sal_bs;
      const int w = ti >> 5, e = ti & 31;
      const uint32_t sb = __ldg(reinterpret_cast<const uint32_t*>(sm) + w);
      const int rank = __ldg(reinterpret_cast<const int*>(sm + (size_t)sal_blocks(d) * 4) + w) +
                       __popc(sb & ((1u << e) - 1u));
      sal = (sb >> e) & 1u;
      ci = ti - rank;
      if (sal) pos = d.s + rank;
    }
    const char* row_s = rows[r];
    constexpr int W = 4 * BITS;
    if (kv == 0) {
      if (coded && hd.cls == kQuantized && !sal) {
        uint32_t* crow = reinterpret_cast<uint32_t*>(Lb + hd.kq + b * hd.kq_bs) + (size_t)ci * W;
        if (BASE == kAkvq)
          quantize_row_rotated<BITS, M16, SPLIT>(row_s, hh, pmask, crow, Lb + hd.kqm + b * hd.kqm_bs, ci);
        else if constexpr (SPLIT == 1)
          quantize_row_token<BITS, M16>(row_s, crow, Lb + hd.kqm + b * hd.kqm_bs, ci);
        return;
      }
      char* dst = (coded && hd.cls == kKeysOnly && !sal) ? Lb + hd.kimg + b * hd.kimg_bs + (size_t)ci * 256
                                                         : Lb + hd.kb + b * hd.kb_bs + (size_t)pos * 256;
      copy_row<SPLIT>(dst, row_s, hh);
    } else if constexpr (SPLIT == 1) {
      if (coded && hd.cls != kProtected && !sal) {
        quantize_row_token<BITS, M16>(row_s, reinterpret_cast<uint32_t*>(Lb + hd.vq + b * hd.vq_bs) + (size_t)ci * W,
                                      Lb + hd.vqm + b * hd.vqm_bs, ci);
        return;
      }
      copy_row<1>(Lb + hd.vb + b * hd.kb_bs + (size_t)pos * 256, row_s, 0);
    }
  }
  static __device__ __forceinline__ void process(const QuantizeParams& p, int li, int b, int kv, const TileSpan& sp,
                                                 const StagedRows& rows, const HeadGeom& hd) {
    if (copy_tile_whole(p, li, b, kv, sp, rows, hd)) return;
    if (BASE == kAkvq && PARTS == 1) {
      // rotated key rows: two lanes per row, rows lane / 2 and 16 + lane / 2
      // (both lanes of a pair take the same path, so the pair's shuffles meet)
      const int hh = threadIdx.x & 1;
      const unsigned pmask = 3u << (threadIdx.x & 30);
#pragma unroll 1
      for (int r = threadIdx.x >> 1; r < sp.n; r += 16) row<2>(p, li, b, kv, sp, rows, hd, r, hh, pmask);
      return;
    }
    if ((int)threadIdx.x < sp.n) row<1>(p, li, b, kv, sp, rows, hd, threadIdx.x, 0, 0u);
  }
};

// ---------------------------------------------------------------------------
// KIVI-style base (Sec. 4), on staged rows as above: one CTA (one warp) per
// (32-token tile, K or V rows, batch row, KV head, layer), tiles aligned so
// that each of the image's 32-token key groups (anchored at the image start)
// is one whole tile.  Values of every head whose image values are coded: one
// thread per token row, four 32-channel groups.  Keys of a quantized head:
// lane c quantizes channel pairs c and c + 32 over the tile's key group (32
// consecutive image tokens, packed in token order).  Every other row (text,
// the BF16 residual window and a trailing partial group, protected heads,
// keys of keys-only heads) is copied.
// ---------------------------------------------------------------------------
template <int BITS, bool M16, int PARTS>
struct KiviTiles {
  static constexpr int kNParts = PARTS == 3 ? 2 : 1;
  static __device__ __forceinline__ int part(int i) { return PARTS == 3 ? i : (PARTS == 1 ? 0 : 1); }
  // tile x: [origin - 32 + 32 x, + 32) clipped to [0, T), origin = s mod 32
  static __device__ __forceinline__ TileSpan span(const QuantizeParams& p, int tx) {
    TileSpan sp;
    sp.tlo = p.tile_origin - kKiviGroup + kQTok * tx;
    sp.t0 = max(sp.tlo, 0);
    sp.n = min(sp.tlo + kQTok, p.d.T) - sp.t0;
    return sp;
  }
  static __device__ __forceinline__ void process(const QuantizeParams& p, int li, int b, int kv, const TileSpan& sp,
                                                 const StagedRows& rows, const HeadGeom& hd) {
    const Dims& d = p.d;
    const int lane = threadIdx.x;
    char* Lb = p.arena + p.lt.base[li];
    const int qs = d.s, qe = d.s + d.nq;
    const int t0 = sp.t0, tlo = sp.tlo;
    constexpr int W = 4 * BITS;
    if (kv == 1) {
      if (lane >= sp.n) return;
      const int t = t0 + lane;
      const bool coded = t >= qs && t < qe;
      const int ti = t - qs;
      if (coded && hd.cls != kProtected)
        quantize_row_kivi_v<BITS, M16>(rows[lane], reinterpret_cast<uint32_t*>(Lb + hd.vq + b * hd.vq_bs) + (size_t)ti * W,
                                       Lb + hd.vqm + b * hd.vqm_bs, (size_t)ti * 4);
      else
        copy_row(Lb + hd.vb + b * hd.kb_bs + (size_t)bf16_pos(d, hd.cls, t) * 256, rows[lane]);
      return;
    }
    // keys: a whole image key group of a quantized head, by channel pairs
    // (uniform over the warp), else the rows are copied
    if (hd.cls == kQuantized && tlo >= qs && tlo + kKiviGroup <= qe && tlo == t0 && sp.n == kKiviGroup) {
      const int grp = (tlo - qs) / kKiviGroup;
#pragma unroll 1
      for (int c2 = lane; c2 < 64; c2 += 32) {
        uint32_t* dst = reinterpret_cast<uint32_t*>(Lb + hd.kq + b * hd.kq_bs) + ((size_t)grp * kD + 2 * c2) * BITS;
        quantize_key_pair<BITS, M16>(&rows[0][4 * c2], dst, dst + BITS, Lb + hd.kqm + b * hd.kqm_bs,
                                     (size_t)grp * kD + 2 * c2);
      }
      return;
    }
    if (lane >= sp.n) return;
    const int t = t0 + lane;
    const bool coded = t >= qs && t < qe;
    if (coded && hd.cls == kQuantized) return;  // unreachable: coded key groups are whole tiles
    copy_row((coded && hd.cls == kKeysOnly) ? Lb + hd.kimg + b * hd.kimg_bs + (size_t)(t - qs) * 256
                                            : Lb + hd.kb + b * hd.kb_bs + (size_t)bf16_pos(d, hd.cls, t) * 256,
             rows[lane]);
  }
};

// The quantizer kernel: one CTA of one warp per (tile, part); grid x = tile
// x part (part fastest), y = batch row x KV head, z = layer.  A warp
// stages its 32 rows, waits for its own copies and codes them; no CTA-wide
// barrier, so the warps of an SM (23 resident) run out of step and one
// warp's loads overlap another's coding.
template <class TP>
__global__ void __launch_bounds__(32) quantize_tiles_kernel(const __grid_constant__ QuantizeParams p) {
  __shared__ __align__(16) StagedRows rows;
  __shared__ HeadGeom s_hd;
  const int pi = blockIdx.x % TP::kNParts, tx = blockIdx.x / TP::kNParts;
  const int li = blockIdx.z, b = blockIdx.y / p.d.H, h = blockIdx.y % p.d.H;
  const int kv = TP::part(pi);
  const TileSpan sp = TP::span(p, tx);
  if (sp.n <= 0) return;
  stage_rows(p, li, b, h, kv, sp, rows);
  cp_async_commit();
  // the head's region map, once for the CTA while its copies are in flight
  // (64-bit arithmetic that would otherwise run in every thread)
  if (threadIdx.x == 0) s_hd = head_geom(p.d, layer_geom(p.d, p.lt.mask[li]), h);
  cp_async_wait<0>();
  __syncwarp();
  TP::process(p, li, b, kv, sp, rows, s_hd);
}

// ---------------------------------------------------------------------------
// AKVQ-style salient tokens (Sec. 4): one CTA per (batch row, KV head, layer);
// protected K+V heads (no coded image entries) return.  Squared key norms of the
// image tokens in the fixed binary32 order (a warp per token: lane l sums
// channels 4l..4l+3, then five butterfly rounds of pairwise sums), ns rounds
// of a CTA-wide arg-max (largest score, ties to the lower index), then the
// map: a bit per image token and the salient count before each 32-token block.
// ---------------------------------------------------------------------------
constexpr int kSalThreads = 256;

__global__ void __launch_bounds__(kSalThreads) salient_kernel(const __grid_constant__ QuantizeParams p) {
  const Dims& d = p.d;
  const int bh = blockIdx.x, li = blockIdx.y;
  const int b = bh / d.H, h = bh % d.H;
  const LayerGeom g = layer_geom(d, p.lt.mask[li]);
  const HeadGeom hd = head_geom(d, g, h);
  if (hd.cls == kProtected || d.ns <= 0) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nq = d.nq, nblk = sal_blocks(d);
  extern __shared__ __align__(16) float sal_smem[];
  float* score = sal_smem;                                     // [nq]
  uint32_t* bits = reinterpret_cast<uint32_t*>(sal_smem + nq);  // [nblk]

  const uint16_t* K = p.k[li] + (((size_t)b * d.H + h) * d.T + d.s) * kD;
  // four rows per warp in flight: their loads first, then each row's sum in
  // the same order as one row at a time
  constexpr int kRows = 4, kWarps = kSalThreads / 32;
  for (int i0 = warp; i0 < nq; i0 += kRows * kWarps) {
    uint2 w[kRows];
#pragma unroll
    for (int u = 0; u < kRows; ++u) {
      const int i = i0 + u * kWarps;
      w[u] = (i < nq) ? ldg8(K + (size_t)i * kD + lane * 4) : make_uint2(0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < kRows; ++u) {
      const int i = i0 + u * kWarps;
      float x[4];
      bf16x4_to_f32(w[u], x);
      float a = __fmul_rn(x[0], x[0]);
      a = __fadd_rn(a, __fmul_rn(x[1], x[1]));
      a = __fadd_rn(a, __fmul_rn(x[2], x[2]));
      a = __fadd_rn(a, __fmul_rn(x[3], x[3]));
#pragma unroll
      for (int m = 16; m >= 1; m >>= 1) a = __fadd_rn(a, __shfl_xor_sync(kFull, a, m));
      if (lane == 0 && i < nq) score[i] = a;
    }
  }
  __syncthreads();

  // The ns largest scores, ties to the lower index -- the set that ns rounds
  // of arg-max (taken tokens dropping out) would pick -- by a radix select on
  // the scores' bit patterns (non-negative floats order as their bits): four
  // 8-bit digits from the top, each pass a histogram of the candidates that
  // match the digits chosen so far and the digit where the count of larger
  // keys reaches ns.  Then every key above the final threshold T is taken,
  // and of the keys equal to T the first `need` by index.
  static_assert(kSalThreads == 256, "one histogram bin per thread");
  __shared__ uint32_t hist[256];
  __shared__ uint32_t s_prefix, s_need, s_eq;
  uint32_t prefix = 0u, pmask = 0u, need = (uint32_t)d.ns;
#pragma unroll 1
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    hist[tid] = 0u;  // kSalThreads == 256 bins
    __syncthreads();
    for (int i0 = warp * 32; i0 < nq; i0 += kSalThreads) {  // warp-uniform: lane i0 + lane
      const int i = i0 + lane;
      const uint32_t key = i < nq ? __float_as_uint(score[i]) : 0u;
      const bool cand = i < nq && (key & pmask) == prefix;
      const uint32_t dg = (key >> shift) & 255u;
      // one atomic per distinct digit of the warp's candidates
      const uint32_t act = __ballot_sync(kFull, cand);
      if (cand) {
        const uint32_t same = __match_any_sync(act, dg);
        if ((__ffs(same) - 1) == lane) atomicAdd(&hist[dg], (uint32_t)__popc(same));
      }
    }
    __syncthreads();
    if (warp == 0) {
      // lane l holds bins 255 - 8l .. 248 - 8l (largest digits first)
      uint32_t c[8], tot = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = hist[255 - 8 * lane - j];
        tot += c[j];
      }
      uint32_t incl = tot;  // keys in this lane's bins and all larger digits
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
      }
      const uint32_t excl = incl - tot;
      if (excl < need && need <= incl) {  // exactly one lane
        uint32_t above = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (above + c[j] >= need) {
            const uint32_t dg = 255u - 8u * lane - j;
            s_prefix = prefix | (dg << shift);
            s_need = need - above;
            s_eq = c[j];
            break;
          }
          above += c[j];
        }
      }
    }
    __syncthreads();
    prefix = s_prefix;
    need = s_need;
    pmask |= 255u << shift;
  }
  // T = prefix: `need` of the s_eq keys equal to T are taken, by index
  const uint32_t T = prefix;
  if (s_eq == need) {
    for (int w = warp; w < nblk; w += kSalThreads / 32) {
      const int i = w * 32 + lane;
      const bool take = i < nq && __float_as_uint(score[i]) >= T;
      const uint32_t word = __ballot_sync(kFull, take);
      if (lane == 0) bits[w] = word;
    }
  } else if (warp == 0) {
    uint32_t left = need;  // equal keys still to take, in index order
    for (int w = 0; w < nblk; ++w) {
      const int i = w * 32 + lane;
      const uint32_t key = i < nq ? __float_as_uint(score[i]) : 0u;
      const bool eq = i < nq && key == T;
      const uint32_t eqm = __ballot_sync(kFull, eq);
      const uint32_t before = __popc(eqm & ((1u << lane) - 1u));
      const bool take = i < nq && (key > T || (eq && before < left));
      const uint32_t word = __ballot_sync(kFull, take);
      const uint32_t ne = __popc(eqm);
      left = left > ne ? left - ne : 0u;
      if (lane == 0) bits[w] = word;
    }
  }
  __syncthreads();

  char* dst = p.arena + p.lt.base[li] + hd.sal + b * hd.sal_bs;
  uint32_t* out_bits = reinterpret_cast<uint32_t*>(dst);
  int* out_rank = reinterpret_cast<int*>(dst + (size_t)nblk * 4);
  for (int w = tid; w < nblk; w += kSalThreads) out_bits[w] = bits[w];
  if (tid == 0) {
    int acc = 0;
    for (int w = 0; w < nblk; ++w) {
      out_rank[w] = acc;
      acc += __popc(bits[w]);
    }
  }
}

// ---------------------------------------------------------------------------
// Reconstruction (Sec. 4: codes to floats, code * scale + zero; AKVQ-style keys
// rotated back; BF16 entries copied), every layer of the launch in original
// token order followed by the appended tokens.  One CTA per (32-token tile,
// batch row, KV head, layer); a half-warp owns one token row of K or of V,
// lane j of it channels 8j..8j+7, so every output row is one 256-byte (BF16)
// or 512-byte (fp32) store of 16 lanes and each lane issues its code,
// metadata and row loads independently (all four units of a thread at once).
// A BF16 entry written as BF16 is copied as it is.  The AKVQ-style inverse rotation runs
// its first three butterfly stages inside a lane and the last four across the
// half-warp, in the same order as the forward transform.
// ---------------------------------------------------------------------------
constexpr int kDqThreads = 256;
constexpr int kDqTile = 32;

// Two floats to BF16 bits (round to nearest even, low half first): one cvt.
__device__ __forceinline__ uint32_t pack_bf16x2_rn(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& w, float (&x)[8]) {
  bf16x2_to_f32(w.x, x[0], x[1]);
  bf16x2_to_f32(w.y, x[2], x[3]);
  bf16x2_to_f32(w.z, x[4], x[5]);
  bf16x2_to_f32(w.w, x[6], x[7]);
}

// Codes of channels 8c..8c+7 of a per-token packed row (channel order; 3 bits:
// the 2-bit half-word, then the plane byte of channels 8c..8c+7, which holds
// them in order at byte ((c >> 1) & 1) | ((c & 1) << 1) of plane word c / 4).
__device__ __forceinline__ void row_codes8(const uint32_t* row, int bits, int c, uint32_t (&code)[8]) {
  if (bits == 4) {
    const uint32_t w = __ldg(row + c);
#pragma unroll
    for (int i = 0; i < 8; ++i) code[i] = (w >> (4 * i)) & 15u;
    return;
  }
  const uint32_t half = (__ldg(row + (c >> 1)) >> (16 * (c & 1))) & 0xffffu;
#pragma unroll
  for (int i = 0; i < 8; ++i) code[i] = (half >> (2 * i)) & 3u;
  if (bits == 3) {
    const uint32_t pl = __ldg(row + 8 + (c >> 2)) >> (8 * (((c >> 1) & 1) | ((c & 1) << 1)));
#pragma unroll
    for (int i = 0; i < 8; ++i) code[i] |= ((pl >> i) & 1u) << 2;
  }
}

// Code of token e (0..31) of one KIVI-style key group row (one channel, token order).
__device__ __forceinline__ uint32_t kivi_code(const uint32_t* row, int bits, int e) {
  if (bits == 3) {
    const uint32_t lo = (__ldg(row + e / 16) >> (2 * (e % 16))) & 3u;
    const int pp = (e & 7) | (((e >> 4) & 1) << 3) | (((e >> 3) & 1) << 4);
    return lo | (((__ldg(row + 2) >> pp) & 1u) << 2);
  }
  const int per = 32 / bits;
  return (__ldg(row + e / per) >> (bits * (e % per))) & ((1u << bits) - 1u);
}

// Codes of token e of eight consecutive KIVI-style key rows (channels
// 8j..8j+7: BITS words each, contiguous): at 2 and 3 bits the 16 or 24 words
// arrive as 16-byte loads and each channel's word is selected in registers;
// at 4 bits the one word a channel needs is loaded alone.
template <int BITS>
__device__ __forceinline__ void kivi_codes8(const uint32_t* rows, int e, uint32_t (&code)[8]) {
  if constexpr (BITS == 4) {
#pragma unroll
    for (int i = 0; i < 8; ++i) code[i] = kivi_code(rows + i * BITS, BITS, e);
  } else {
    uint32_t w[8 * BITS];
#pragma unroll
    for (int v = 0; v < 2 * BITS; ++v) {
      const uint4 x = ldg16(rows + 4 * v);
      w[4 * v] = x.x;
      w[4 * v + 1] = x.y;
      w[4 * v + 2] = x.z;
      w[4 * v + 3] = x.w;
    }
    const bool hi = e >= 16;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t lo = ((hi ? w[i * BITS + 1] : w[i * BITS]) >> (2 * (e & 15))) & 3u;
      if (BITS == 3) {
        const int pp = (e & 7) | (((e >> 4) & 1) << 3) | (((e >> 3) & 1) << 4);
        code[i] = lo | (((w[i * BITS + 2] >> pp) & 1u) << 2);
      } else {
        code[i] = lo;
      }
    }
  }
}

// Metadata pairs of eight consecutive KIVI-style key rows from index i0 (a
// multiple of 8, so 64 or 32 contiguous bytes on a 16-byte boundary).
template <bool M16>
__device__ __forceinline__ void kivi_meta8(const char* base, size_t i0, float2 (&m)[8]) {
  if (M16) {
    const uint4* p = reinterpret_cast<const uint4*>(base + i0 * 4);
#pragma unroll
    for (int v = 0; v < 2; ++v) {
      const uint4 x = __ldg(p + v);
      m[4 * v] = half2_bits_to_float2(x.x);
      m[4 * v + 1] = half2_bits_to_float2(x.y);
      m[4 * v + 2] = half2_bits_to_float2(x.z);
      m[4 * v + 3] = half2_bits_to_float2(x.w);
    }
  } else {
    const float4* p = reinterpret_cast<const float4*>(base + i0 * 8);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const float4 x = __ldg(p + v);
      m[2 * v] = make_float2(x.x, x.y);
      m[2 * v + 1] = make_float2(x.z, x.w);
    }
  }
}

// Normalised Hadamard-128 of a vector spread over a half-warp, lane j holding
// channels 8j..8j+7: stages h = 1, 2, 4 in the lane, h = 8..64 with lane
// j ^ (h / 8); butterflies (a, b) -> (a + b, a - b), one multiply at the end.
__device__ __forceinline__ void fwht128_half(float (&x)[8], int j) {
#pragma unroll
  for (int h = 1; h < 8; h <<= 1) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (i & h) continue;
      const float a = x[i], b = x[i + h];
      x[i] = __fadd_rn(a, b);
      x[i + h] = __fsub_rn(a, b);
    }
  }
#pragma unroll
  for (int m = 1; m < 16; m <<= 1) {
    const bool upper = (j & m) != 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float p = __shfl_xor_sync(kFull, x[i], m);
      x[i] = upper ? __fsub_rn(p, x[i]) : __fadd_rn(x[i], p);
    }
  }
  const float c = hadamard_c();
#pragma unroll
  for (int i = 0; i < 8; ++i) x[i] = __fmul_rn(x[i], c);
}

// BITS, BASE and M16 are compile-time, so each (code width, base, metadata
// width) runs code of its own; a CTA takes a span of consecutive tiles of one
// (row, head, layer), so the head's region map and its barrier are paid once
// per span.
template <int BITS, int BASE, bool M16>
__global__ void __launch_bounds__(kDqThreads, 6) dequantize_kernel(const __grid_constant__ DequantParams p) {
  const Dims& d = p.d;
  const int li = blockIdx.z, bh = blockIdx.y;
  const int b = bh / d.H, h = bh % d.H;
  const int Tt = d.T + p.appended;
  // the head's region map, computed once for the CTA (64-bit arithmetic that
  // would otherwise cost every warp more instructions than its four units)
  __shared__ HeadGeom s_hd;
  if (threadIdx.x == 0) s_hd = head_geom(d, layer_geom(d, p.lt.mask[li]), h);
  __syncthreads();
  const HeadGeom& hd = s_hd;
  const char* Lb = p.arena + p.lt.base[li];
  const int qs = d.s, qe = d.s + d.nq;
  constexpr int W = kD * BITS / 32;
  const int j = threadIdx.x & 15;  // channels 8j..8j+7
  const size_t out_row0 = (((size_t)li * d.B + b) * d.H + h) * (size_t)Tt;
  const int ntiles = (Tt + kDqTile - 1) / kDqTile;
  const int span = (ntiles + (int)gridDim.x - 1) / (int)gridDim.x;
  const int x1 = min(((int)blockIdx.x + 1) * span, ntiles);

#pragma unroll 1
  for (int x = blockIdx.x * span; x < x1; ++x) {
    // a thread's two tokens (rows 16 apart), each with its K and V unit: the
    // token's coded slot and BF16 position found once for both
    int tk[2], ck[2], pk[2];
    bool codedk[2], salk[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int t = x * kDqTile + ((threadIdx.x >> 4) + 16 * r);
      const bool coded = (t >= qs) && (t < qe);
      const int ti = t - qs;
      int ci = ti, spos = 0;  // coded slot; BF16 position of a salient token (Sec. 4)
      bool sal = false;
      if (BASE == kAkvq && coded && d.ns > 0 && hd.cls != kProtected) {
        const char* sm = Lb + hd.sal + b * hd.sal_bs;
        const int w = ti >> 5, e = ti & 31;
        const uint32_t sb = __ldg(reinterpret_cast<const uint32_t*>(sm) + w);
        const int rank = __ldg(reinterpret_cast<const int*>(sm + (size_t)sal_blocks(d) * 4) + w) +
                         __popc(sb & ((1u << e) - 1u));
        sal = (sb >> e) & 1u;
        ci = ti - rank;
        spos = qs + rank;
      }
      tk[r] = t;
      ck[r] = ci;
      codedk[r] = coded;
      salk[r] = sal;
      pk[r] = (t >= d.T) ? hd.bf16_prefill + (t - d.T) : (sal ? spos : bf16_pos(d, hd.cls, t));
    }
    // unit u: K (u < 16 * kDqTile) or V, token (u >> 4) % kDqTile of the
    // tile; unrolled so that the loads of a thread's four units are in flight
    // together
#pragma unroll
    for (int u = threadIdx.x; u < 2 * kDqTile * 16; u += kDqThreads) {
      const bool is_k = u < kDqTile * 16;
      const int r = ((u - threadIdx.x) / kDqThreads) & 1;  // the thread's token of this unit
      const int t = tk[r];
      if (t >= Tt) continue;  // uniform over the half-warp
      const bool coded = codedk[r], sal = salk[r];
      const int ti = t - qs, ci = ck[r], pos = pk[r];
      const size_t o = (out_row0 + t) * kD + 8 * j;
      void* dst = is_k ? p.k_out : p.v_out;
      float x8[8];
      bool raw = false;  // a BF16 entry: `w` holds its 16 bytes
      uint4 w = make_uint4(0u, 0u, 0u, 0u);
      if (is_k) {
        if (coded && hd.cls == kQuantized && !sal) {
          uint32_t code[8];
          float2 m[8];
          if (BASE == kKivi) {
            const int grp = ti / kKiviGroup, e = ti % kKiviGroup;
            const uint32_t* codes = reinterpret_cast<const uint32_t*>(Lb + hd.kq + b * hd.kq_bs) +
                                    ((size_t)grp * kD + 8 * j) * BITS;
            kivi_codes8<BITS>(codes, e, code);
            kivi_meta8<M16>(Lb + hd.kqm + b * hd.kqm_bs, (size_t)grp * kD + 8 * j, m);
          } else {
            row_codes8(reinterpret_cast<const uint32_t*>(Lb + hd.kq + b * hd.kq_bs) + (size_t)ci * W, BITS, j,
                       code);
            const float2 m0 = load_meta(Lb + hd.kqm + b * hd.kqm_bs, ci, M16);
#pragma unroll
            for (int i = 0; i < 8; ++i) m[i] = m0;
          }
#pragma unroll
          for (int i = 0; i < 8; ++i) x8[i] = dequant1(code[i], m[i].x, m[i].y);
          if (BASE == kAkvq) fwht128_half(x8, j);  // inverse rotation (H is self-inverse)
        } else {
          const char* src = (coded && hd.cls == kKeysOnly && !sal)
                                ? Lb + hd.kimg + b * hd.kimg_bs + (size_t)ci * 256
                                : Lb + hd.kb + b * hd.kb_bs + (size_t)pos * 256;
          w = ldg16(src + j * 16);
          raw = true;
        }
      } else {
        if (coded && hd.cls != kProtected && !sal) {
          uint32_t code[8];
          row_codes8(reinterpret_cast<const uint32_t*>(Lb + hd.vq + b * hd.vq_bs) + (size_t)ci * W, BITS, j,
                     code);
          // KIVI-style: 32-channel groups, channels 8j.. in group j / 4
          const float2 m = load_meta(Lb + hd.vqm + b * hd.vqm_bs,
                                     (size_t)ci * vgroups(d) + (BASE == kKivi ? (j >> 2) : 0), M16);
#pragma unroll
          for (int i = 0; i < 8; ++i) x8[i] = dequant1(code[i], m.x, m.y);
        } else {
          w = ldg16(Lb + hd.vb + b * hd.kb_bs + (size_t)pos * 256 + j * 16);
          raw = true;
        }
      }
      if (p.out_fp32) {
        if (raw) bf16x8_to_f32(w, x8);
        float4* f = reinterpret_cast<float4*>(static_cast<float*>(dst) + o);
        f[0] = make_float4(x8[0], x8[1], x8[2], x8[3]);
        f[1] = make_float4(x8[4], x8[5], x8[6], x8[7]);
      } else {
        if (!raw)
          w = make_uint4(pack_bf16x2_rn(x8[0], x8[1]), pack_bf16x2_rn(x8[2], x8[3]),
                         pack_bf16x2_rn(x8[4], x8[5]), pack_bf16x2_rn(x8[6], x8[7]));
        *reinterpret_cast<uint4*>(static_cast<uint16_t*>(dst) + o) = w;
      }
    }
  }
}

// One decode token per (layer, row, head) into the head's BF16 region.
__global__ void __launch_bounds__(64) append_kernel(const __grid_constant__ AppendParams p) {
  const Dims& d = p.d;
  const int li = blockIdx.x, bh = blockIdx.y;
  const int b = bh / d.H, h = bh % d.H;
  const LayerGeom g = layer_geom(d, p.lt.mask[li]);
  const HeadGeom hd = head_geom(d, g, h);
  char* Lb = p.arena + p.lt.base[li];
  const int pos = hd.bf16_prefill + p.appended[li];
  const size_t src = (((size_t)li * d.B + b) * d.H + h) * kD;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32) {
    *reinterpret_cast<uint2*>(Lb + hd.kb + b * hd.kb_bs + ((size_t)pos * kD + lane * 4) * 2) =
        ldg8(p.k_new + src + lane * 4);
  } else {
    *reinterpret_cast<uint2*>(Lb + hd.vb + b * hd.kb_bs + ((size_t)pos * kD + lane * 4) * 2) =
        ldg8(p.v_new + src + lane * 4);
  }
}

}  // namespace

// Launch of the quantizer kernel over every tile of the launch's layers.
template <class TP>
cudaError_t launch_tiles(const QuantizeParams& p, int tiles_x, cudaStream_t s) {
  const dim3 grid((unsigned)(tiles_x * TP::kNParts), (unsigned)(p.d.B * p.d.H), (unsigned)p.n_layers);
  quantize_tiles_kernel<TP><<<grid, 32, 0, s>>>(p);
  return cudaGetLastError();
}

template <int BITS, bool M16>
cudaError_t launch_quantize_bits(const QuantizeParams& p, cudaStream_t s) {
  const Dims& d = p.d;
  if (d.base == kKivi) {
    const int tx = (d.T - p.tile_origin + kKiviGroup + kQTok - 1) / kQTok;
    // keys and values in launches of their own: each kernel holds one of the
    // two code paths, so the warps of an SM share less instruction cache
    const cudaError_t e = launch_tiles<KiviTiles<BITS, M16, 1>>(p, tx, s);
    if (e != cudaSuccess) return e;
    return launch_tiles<KiviTiles<BITS, M16, 2>>(p, tx, s);
  }
  const int tx = (d.T + kQTok - 1) / kQTok;
  if (d.base == kAkvq) {
    // keys and values in CTAs of their own: a rotated key row holds 64 fp32
    // pairs in registers, a value row far fewer, and a kernel's threads all
    // get the larger count -- split, twice as many key rows are resident
    const cudaError_t e = launch_tiles<TokenTiles<BITS, M16, kAkvq, 1>>(p, tx, s);
    if (e != cudaSuccess) return e;
    return launch_tiles<TokenTiles<BITS, M16, kAkvq, 2>>(p, tx, s);
  }
  return launch_tiles<TokenTiles<BITS, M16, kMinMax, 3>>(p, tx, s);
}

cudaError_t launch_quantize(const QuantizeParams& p, cudaStream_t s) {
  const bool m16 = p.d.meta16 != 0;
  if (p.d.bits == 2) return m16 ? launch_quantize_bits<2, true>(p, s) : launch_quantize_bits<2, false>(p, s);
  if (p.d.bits == 3) return m16 ? launch_quantize_bits<3, true>(p, s) : launch_quantize_bits<3, false>(p, s);
  return m16 ? launch_quantize_bits<4, true>(p, s) : launch_quantize_bits<4, false>(p, s);
}

cudaError_t launch_salient(const QuantizeParams& p, cudaStream_t s) {
  const size_t smem = salient_smem_bytes(p.d);
  if (smem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(salient_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid(p.d.B * p.d.H, p.n_layers, 1);
  salient_kernel<<<grid, kSalThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <int BITS, int BASE, bool M16>
cudaError_t launch_dequantize_t(const DequantParams& p, dim3 grid, cudaStream_t s) {
  dequantize_kernel<BITS, BASE, M16><<<grid, kDqThreads, 0, s>>>(p);
  return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_dequantize_bits(const DequantParams& p, dim3 grid, cudaStream_t s) {
  const bool m16 = p.d.meta16 != 0;
  if (p.d.base == kKivi)
    return m16 ? launch_dequantize_t<BITS, kKivi, true>(p, grid, s) : launch_dequantize_t<BITS, kKivi, false>(p, grid, s);
  if (p.d.base == kAkvq)
    return m16 ? launch_dequantize_t<BITS, kAkvq, true>(p, grid, s) : launch_dequantize_t<BITS, kAkvq, false>(p, grid, s);
  return m16 ? launch_dequantize_t<BITS, kMinMax, true>(p, grid, s)
             : launch_dequantize_t<BITS, kMinMax, false>(p, grid, s);
}

cudaError_t launch_dequantize(const DequantParams& p, int sm_count, cudaStream_t s) {
  const int Tt = p.d.T + p.appended;
  const int ntiles = (Tt + kDqTile - 1) / kDqTile;
  // spans of several tiles once the grid holds more than 16 waves of 6 CTAs
  // per SM (at most 8 tiles a CTA)
  const long long groups = (long long)p.d.B * p.d.H * p.n_layers;
  const long long waves16 = 16LL * 6 * (sm_count > 0 ? sm_count : 1);
  const int span = (int)std::max(1LL, std::min(8LL, groups * ntiles / waves16));
  dim3 grid((ntiles + span - 1) / span, p.d.B * p.d.H, p.n_layers);
  if (p.d.bits == 2) return launch_dequantize_bits<2>(p, grid, s);
  if (p.d.bits == 3) return launch_dequantize_bits<3>(p, grid, s);
  return launch_dequantize_bits<4>(p, grid, s);
}

cudaError_t launch_append(const AppendParams& p, cudaStream_t s) {
  dim3 grid(p.n_layers, p.d.B * p.d.H, 1);
  append_kernel<<<grid, 64, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace hg
