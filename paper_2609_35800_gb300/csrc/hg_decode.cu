// Split-K decode attention over the mixed-precision cache.
//
// One CTA per work item = one chunk of one (layer, batch row, KV head): either
// a run of BF16 tokens (text, image tokens not coded, protected heads,
// appended tokens) or a run of coded image tokens (codes + fp32 scale/zero for
// K and V, or BF16 K + coded V for keys-only protected heads).  The segment
// type is uniform inside a CTA, so the only branch on the mask or the image
// span is taken once per CTA.  Each warp streams 32-token tiles into shared
// memory, computes the G query heads' scores (lane = token), keeps an online
// softmax, and accumulates P.V (lane = 4 channels).  Warps are combined in
// shared memory; a CTA that is not alone on its head writes its (m, l, o)
// partial to the workspace and the last CTA to arrive (atomic ticket, no
// waiting) merges them and writes the BF16 output.
//
// AKVQ-style keys are coded in the rotated domain; since the normalised
// Hadamard matrix is symmetric and orthonormal, <q, H k'> = <H q, k'>, so the
// query is rotated once per CTA instead of inverse-rotating every key.
#include <cuda_runtime.h>

#include "hg_common.cuh"
#include "hg_internal.h"

namespace hg {

namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kTile = 32;
constexpr int kKRowHalves = kD + 8;                       // padded BF16 key row (272 bytes)
constexpr int kWarpTileBytes = kTile * kKRowHalves * 2 + kTile * kD * 2;  // K + V BF16 tiles
constexpr int kPartialStride = kD + 2;

template <int MAXG>
struct Smem {
  static constexpr int q_off = 0;                                   // float [MAXG][128]
  static constexpr int qr_off = q_off + MAXG * kD * 4;              // float [MAXG][128] rotated
  static constexpr int p_off = qr_off + MAXG * kD * 4;              // float [warps][32][MAXG]
  static constexpr int tile_off = p_off + kWarps * kTile * MAXG * 4;
  static constexpr int bytes = tile_off + kWarps * kWarpTileBytes;
};

__device__ __forceinline__ void warp_copy16(void* dst, const void* src, int nbytes, int lane) {
  for (int off = lane * 16; off < nbytes; off += 32 * 16)
    *reinterpret_cast<uint4*>(static_cast<char*>(dst) + off) =
        __ldg(reinterpret_cast<const uint4*>(static_cast<const char*>(src) + off));
}
__device__ __forceinline__ void warp_copy8(void* dst, const void* src, int nbytes, int lane) {
  for (int off = lane * 8; off < nbytes; off += 32 * 8)
    *reinterpret_cast<uint2*>(static_cast<char*>(dst) + off) =
        __ldg(reinterpret_cast<const uint2*>(static_cast<const char*>(src) + off));
}
// nt rows of 256 bytes into a tile with row pitch `pitch` bytes.
__device__ __forceinline__ void warp_copy_rows(char* dst, int pitch, const char* src, int nt, int lane) {
  for (int idx = lane; idx < nt * 16; idx += 32) {
    const int row = idx >> 4, col = idx & 15;
    *reinterpret_cast<uint4*>(dst + row * pitch + col * 16) =
        __ldg(reinterpret_cast<const uint4*>(src + row * 256 + col * 16));
  }
}

template <int BITS>
__device__ __forceinline__ void codes4(const uint32_t* row, int c4, uint32_t (&c)[4]) {
  // codes of channels 4*c4 .. 4*c4+3 from a packed 128-code row
  if (BITS == 2) {
    const uint32_t byte = (row[c4 >> 2] >> (8 * (c4 & 3))) & 0xffu;
#pragma unroll
    for (int i = 0; i < 4; ++i) c[i] = (byte >> (2 * i)) & 3u;
  } else {
    const uint32_t half = (row[c4 >> 1] >> (16 * (c4 & 1))) & 0xffffu;
#pragma unroll
    for (int i = 0; i < 4; ++i) c[i] = (half >> (4 * i)) & 15u;
  }
}

template <int MAXG, int BITS>
__global__ void __launch_bounds__(kThreads)
decode_kernel(const __grid_constant__ DecodeParams p) {
  extern __shared__ __align__(16) char smem[];
  using S = Smem<MAXG>;
  const Dims& d = p.d;
  const int li = blockIdx.y;
  const int ipr = p.items_per_row[li];
  const int item = blockIdx.x;
  if (item >= ipr * d.B) return;
  const int b = item / ipr;
  int r = item - b * ipr;
  const uint64_t mask = p.lt.mask[li];
  const int app = p.appended[li];
  int h = 0, nb = 0, ni = 0;
  for (; h < d.H; ++h) {
    ni = head_items(d, head_class(d, mask, h), app, p.cb, p.cq, &nb);
    if (r < ni) break;
    r -= ni;
  }
  const LayerGeom g = layer_geom(d, mask);
  const HeadGeom hd = head_geom(d, g, h);
  const char* Lb = p.arena + p.lt.base[li];
  const int G = d.G;
  const bool coded = r >= nb;
  int tb, te;
  if (!coded) {
    tb = r * p.cb;
    te = min(tb + p.cb, hd.bf16_prefill + app);
  } else {
    tb = (r - nb) * p.cq;
    te = min(tb + p.cq, d.nq);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int W = kD * BITS / 32;  // code words per token

  float* q_s = reinterpret_cast<float*>(smem + S::q_off);
  float* qr_s = reinterpret_cast<float*>(smem + S::qr_off);
  float* p_s = reinterpret_cast<float*>(smem + S::p_off) + warp * kTile * MAXG;
  char* tile = smem + S::tile_off + warp * kWarpTileBytes;

  // Queries of this KV head's group, as fp32.
  const uint16_t* qg = p.q + (((size_t)li * d.B + b) * d.Hq + (size_t)h * G) * kD;
  for (int i = threadIdx.x; i < G * kD; i += kThreads) q_s[i] = bf16_to_f32(qg[i]);
  const bool rot = coded && d.base == kAkvq && hd.cls == kQuantized;
  __syncthreads();
  if (rot) {
    for (int j = warp; j < G; j += kWarps) {
      float x[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) x[i] = q_s[j * kD + lane * 4 + i];
      fwht128_warp(x, lane);
#pragma unroll
      for (int i = 0; i < 4; ++i) qr_s[j * kD + lane * 4 + i] = x[i];
    }
    __syncthreads();
  }
  const float* qk_s = rot ? qr_s : q_s;  // queries used against this item's keys

  float m_run[MAXG], l_run[MAXG], o_acc[MAXG][4];
#pragma unroll
  for (int j = 0; j < MAXG; ++j) {
    m_run[j] = -INFINITY;
    l_run[j] = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) o_acc[j][e] = 0.f;
  }

  const bool k_bf16 = !coded || hd.cls == kKeysOnly;
  const bool kivi_k = coded && !k_bf16 && d.base == kKivi;
  const int vg = vgroups(d);
  // Tile buffer of a warp: [0, 8704) BF16 key rows (pitch 272 B) or key codes
  // (at 0, <= 2 KB) + key metadata (at 4096, <= 1 KB); [8704, 16896) BF16
  // value rows or value codes (at 8704) + value metadata (at 8704 + 4096).
  char* Ks = tile;
  char* Vs = tile + kTile * kKRowHalves * 2;
  uint32_t* Kcode = reinterpret_cast<uint32_t*>(tile);
  float2* Kmeta = reinterpret_cast<float2*>(tile + 4096);
  uint32_t* Vcode = reinterpret_cast<uint32_t*>(Vs);
  float2* Vmeta = reinterpret_cast<float2*>(Vs + 4096);

  const int n_tiles = (te - tb + kTile - 1) / kTile;
  for (int tt = warp; tt < n_tiles; tt += kWarps) {
    const int t0 = tb + tt * kTile;
    const int nt = min(kTile, te - t0);
    // ---- stage the tile ----
    if (!coded) {
      warp_copy_rows(Ks, kKRowHalves * 2, Lb + hd.kb + b * hd.kb_bs + (size_t)t0 * 256, nt, lane);
      warp_copy_rows(Vs, kD * 2, Lb + hd.vb + b * hd.kb_bs + (size_t)t0 * 256, nt, lane);
    } else {
      if (k_bf16) {
        warp_copy_rows(Ks, kKRowHalves * 2, Lb + hd.kimg + b * hd.kimg_bs + (size_t)t0 * 256, nt, lane);
      } else if (kivi_k) {
        const size_t grp = (size_t)t0 / kKiviGroup;
        warp_copy16(Kcode, Lb + hd.kq + b * hd.kq_bs + grp * kD * BITS * 4, kD * BITS * 4, lane);
        warp_copy16(Kmeta, Lb + hd.kqm + b * hd.kqm_bs + grp * kD * 8, kD * 8, lane);
      } else {
        warp_copy16(Kcode, Lb + hd.kq + b * hd.kq_bs + (size_t)t0 * W * 4, nt * W * 4, lane);
        warp_copy8(Kmeta, Lb + hd.kqm + b * hd.kqm_bs + (size_t)t0 * 8, nt * 8, lane);
      }
      warp_copy16(Vcode, Lb + hd.vq + b * hd.vq_bs + (size_t)t0 * W * 4, nt * W * 4, lane);
      warp_copy8(Vmeta, Lb + hd.vqm + b * hd.vqm_bs + (size_t)t0 * vg * 8, nt * vg * 8, lane);
    }
    __syncwarp();

    // ---- scores: lane = token ----
    float acc[MAXG];
#pragma unroll
    for (int j = 0; j < MAXG; ++j) acc[j] = 0.f;
    if (lane < nt) {
      if (k_bf16) {
        const char* krow = Ks + lane * kKRowHalves * 2;
#pragma unroll 2
        for (int c8 = 0; c8 < 16; ++c8) {
          const uint4 w = *reinterpret_cast<const uint4*>(krow + c8 * 16);
          float k[8];
          bf16x2_to_f32(w.x, k[0], k[1]);
          bf16x2_to_f32(w.y, k[2], k[3]);
          bf16x2_to_f32(w.z, k[4], k[5]);
          bf16x2_to_f32(w.w, k[6], k[7]);
#pragma unroll
          for (int j = 0; j < MAXG; ++j) {
            if (j < G) {
              const float4 qa = *reinterpret_cast<const float4*>(qk_s + j * kD + c8 * 8);
              const float4 qb = *reinterpret_cast<const float4*>(qk_s + j * kD + c8 * 8 + 4);
              float a = acc[j];
              a = fmaf(qa.x, k[0], a); a = fmaf(qa.y, k[1], a);
              a = fmaf(qa.z, k[2], a); a = fmaf(qa.w, k[3], a);
              a = fmaf(qb.x, k[4], a); a = fmaf(qb.y, k[5], a);
              a = fmaf(qb.z, k[6], a); a = fmaf(qb.w, k[7], a);
              acc[j] = a;
            }
          }
        }
      } else if (kivi_k) {
        // lane = token e of the 32-token group; channel c has its own (scale, zero)
        constexpr int per = 32 / BITS;
        const int e = lane;
#pragma unroll 4
        for (int c = 0; c < kD; ++c) {
          const uint32_t word = Kcode[c * BITS + e / per];
          const uint32_t code = (word >> (BITS * (e % per))) & ((1u << BITS) - 1u);
          const float2 m = Kmeta[c];
          const float x = dequant1(code, m.x, m.y);
#pragma unroll
          for (int j = 0; j < MAXG; ++j)
            if (j < G) acc[j] = fmaf(qk_s[j * kD + c], x, acc[j]);
        }
      } else {
        const uint32_t* crow = Kcode + lane * W;
        const float2 m = Kmeta[lane];
#pragma unroll 4
        for (int c4 = 0; c4 < kD / 4; ++c4) {
          uint32_t cc[4];
          codes4<BITS>(crow, c4, cc);
          float x[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) x[i] = dequant1(cc[i], m.x, m.y);
#pragma unroll
          for (int j = 0; j < MAXG; ++j) {
            if (j < G) {
              const float4 qa = *reinterpret_cast<const float4*>(qk_s + j * kD + c4 * 4);
              float a = acc[j];
              a = fmaf(qa.x, x[0], a); a = fmaf(qa.y, x[1], a);
              a = fmaf(qa.z, x[2], a); a = fmaf(qa.w, x[3], a);
              acc[j] = a;
            }
          }
        }
      }
    }

    // ---- online softmax (log2 domain) ----
#pragma unroll
    for (int j = 0; j < MAXG; ++j) {
      if (j < G) {
        const float s = (lane < nt) ? acc[j] * p.scale_log2 : -INFINITY;
        const float mt = warp_max(s);
        const float mnew = fmaxf(m_run[j], mt);
        const float alpha = exp2f(m_run[j] - mnew);
        const float pj = exp2f(s - mnew);
        l_run[j] = l_run[j] * alpha + pj;
#pragma unroll
        for (int e = 0; e < 4; ++e) o_acc[j][e] *= alpha;
        m_run[j] = mnew;
        p_s[lane * MAXG + j] = pj;
      }
    }
    __syncwarp();

    // ---- P.V: lane = channels 4*lane .. 4*lane+3 ----
    for (int i = 0; i < nt; ++i) {
      float v[4];
      if (!coded) {
        const uint2 w = *reinterpret_cast<const uint2*>(Vs + i * kD * 2 + lane * 8);
        bf16x2_to_f32(w.x, v[0], v[1]);
        bf16x2_to_f32(w.y, v[2], v[3]);
      } else {
        uint32_t cc[4];
        codes4<BITS>(Vcode + i * W, lane, cc);
        const float2 m = Vmeta[i * vg + (vg > 1 ? (lane >> 3) : 0)];
#pragma unroll
        for (int e = 0; e < 4; ++e) v[e] = dequant1(cc[e], m.x, m.y);
      }
#pragma unroll
      for (int j = 0; j < MAXG; ++j) {
        if (j < G) {
          const float pj = p_s[i * MAXG + j];
#pragma unroll
          for (int e = 0; e < 4; ++e) o_acc[j][e] = fmaf(pj, v[e], o_acc[j][e]);
        }
      }
    }
    __syncwarp();
  }

  // ---- combine the warps of this CTA ----
  __syncthreads();  // every warp is done with its tile buffers
  float* red_m = reinterpret_cast<float*>(smem + S::tile_off);  // [warps][MAXG]
  float* red_l = red_m + kWarps * MAXG;                          // [warps][MAXG]
  float* red_o = red_l + kWarps * MAXG;                          // [warps][MAXG][128]
#pragma unroll
  for (int j = 0; j < MAXG; ++j) {
    if (j < G) {
      const float lt = warp_sum(l_run[j]);
      if (lane == 0) {
        red_m[warp * MAXG + j] = m_run[j];
        red_l[warp * MAXG + j] = lt;
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) red_o[(warp * MAXG + j) * kD + lane * 4 + e] = o_acc[j][e];
    }
  }
  __syncthreads();

  const int c = threadIdx.x;  // channel
  const size_t out_row = ((size_t)li * d.B + b) * d.Hq + (size_t)h * G;
  if (ni == 1) {
    for (int j = 0; j < G; ++j) {
      float M = -INFINITY;
      for (int w = 0; w < kWarps; ++w) M = fmaxf(M, red_m[w * MAXG + j]);
      float O = 0.f, Ls = 0.f;
      for (int w = 0; w < kWarps; ++w) {
        const float f = exp2f(red_m[w * MAXG + j] - M);
        O += f * red_o[(w * MAXG + j) * kD + c];
        Ls += f * red_l[w * MAXG + j];
      }
      p.out[(out_row + j) * kD + c] = (uint16_t)f32_to_bf16_rn(O / Ls);
    }
    return;
  }

  const size_t head_lin = ((size_t)li * d.B + b) * d.H + h;
  float* part = p.partials + (head_lin * p.max_items) * (size_t)G * kPartialStride;
  {
    float* mine = part + (size_t)r * G * kPartialStride;
    for (int j = 0; j < G; ++j) {
      float M = -INFINITY;
      for (int w = 0; w < kWarps; ++w) M = fmaxf(M, red_m[w * MAXG + j]);
      float O = 0.f, Ls = 0.f;
      for (int w = 0; w < kWarps; ++w) {
        const float f = exp2f(red_m[w * MAXG + j] - M);
        O += f * red_o[(w * MAXG + j) * kD + c];
        Ls += f * red_l[w * MAXG + j];
      }
      mine[j * kPartialStride + 2 + c] = O;
      if (c == 0) {
        mine[j * kPartialStride + 0] = M;
        mine[j * kPartialStride + 1] = Ls;
      }
    }
  }
  __threadfence();
  __syncthreads();
  __shared__ int s_last;
  if (threadIdx.x == 0) {
    const unsigned prev = atomicAdd(p.counters + head_lin, 1u);
    s_last = (prev == (unsigned)(ni - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int j = 0; j < G; ++j) {
    float M = -INFINITY;
    for (int sidx = 0; sidx < ni; ++sidx)
      M = fmaxf(M, __ldcg(part + ((size_t)sidx * G + j) * kPartialStride));
    float O = 0.f, Ls = 0.f;
    for (int sidx = 0; sidx < ni; ++sidx) {
      const float* ps = part + ((size_t)sidx * G + j) * kPartialStride;
      const float f = exp2f(__ldcg(ps) - M);
      O += f * __ldcg(ps + 2 + c);
      Ls += f * __ldcg(ps + 1);
    }
    p.out[(out_row + j) * kD + c] = (uint16_t)f32_to_bf16_rn(O / Ls);
  }
  if (threadIdx.x == 0) atomicExch(p.counters + head_lin, 0u);
}

template <int MAXG, int BITS>
cudaError_t launch_decode_t(const DecodeParams& p, int grid_x, cudaStream_t s) {
  constexpr int smem = Smem<MAXG>::bytes;
  static bool configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 64 && !configured[dev]) {
    e = cudaFuncSetAttribute(decode_kernel<MAXG, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 grid(grid_x, p.n_layers, 1);
  decode_kernel<MAXG, BITS><<<grid, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_decode_bits(const DecodeParams& p, int grid_x, cudaStream_t s) {
  const int G = p.d.G;
  if (G <= 1) return launch_decode_t<1, BITS>(p, grid_x, s);
  if (G <= 2) return launch_decode_t<2, BITS>(p, grid_x, s);
  if (G <= 4) return launch_decode_t<4, BITS>(p, grid_x, s);
  if (G <= 8) return launch_decode_t<8, BITS>(p, grid_x, s);
  return launch_decode_t<16, BITS>(p, grid_x, s);
}

}  // namespace

cudaError_t launch_decode(const DecodeParams& p, int grid_x, cudaStream_t s) {
  return p.d.bits == 2 ? launch_decode_bits<2>(p, grid_x, s) : launch_decode_bits<4>(p, grid_x, s);
}

}  // namespace hg
