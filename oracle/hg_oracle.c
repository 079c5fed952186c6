/*
 * HeadGuard CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, deliberately unoptimised statement of what the mixed
 * precision KV-cache path computes.  Only the test-suite, the smoke check and
 * the benchmark's CPU-baseline leg may load this file's library; the product
 * library (paper_2609_35800_gb300) never links or calls it, and it shares no
 * code, header, table or helper with the CUDA path.
 *
 * Built with -O2 -ffp-contract=off -fno-fast-math so every float operation
 * below is one IEEE-754 binary32 operation rounded to nearest-even, exactly as
 * written (no fused multiply-add, no reassociation).
 *
 * Paper: "HeadGuard: Selective Head Protection for Low-Bit VLM KV-Cache
 * Quantization".  Sections referenced:
 *   Sec. 1        per-token min-max RTN (own min / max, nearest level)
 *   Sec. 3        applying protection (K+V, K-only; text stays BF16)
 *   Sec. 4        quantization setup (KIVI-style per-channel K / per-token V,
 *                 AKVQ-style query/key Hadamard rotation + per-token RTN,
 *                 simulated quantization: round to levels, reconstruct float)
 *   Sec. 5.4      storage model (32 bits metadata per 128-d vector)
 *
 * Readings of points the paper leaves open (each is listed in the design
 * notes of the repository):
 *   R1 rounding is round-half-to-even;
 *   R2 the zero point is the float group minimum (asymmetric, zero = min);
 *   R3 one IEEE division per element, d / scale;
 *   R4 a constant group stores scale 0 and codes 0 (reconstructs min exactly);
 *   R5 metadata is an fp32 (scale, zero) pair per group (64 bits);
 *   R6 "per token" means one (token, KV head) vector of 128 channels;
 *   R7 KIVI-style: 32-token key groups anchored at the image start, 32-channel
 *      value groups, the last R tokens of the prefill stay BF16, and image
 *      tokens of a trailing partial key group stay BF16;
 *   R9 the Hadamard scale 1/sqrt(128) is applied once, after the butterflies;
 *      values are not rotated;
 *   R11 softmax scale given by the caller, query head qh reads KV head
 *      qh / G, the decoded token attends to its own appended entry;
 *   R12 signed zeros: the group min and max are canonicalised with "+ 0.0f"
 *      so the stored metadata has one bit pattern.
 *   R13 32-bit metadata (the Sec. 5.4 storage model, optional): scale and
 *      zero are stored as binary16 (round to nearest even, magnitudes above
 *      65504 saturate to 65504), and the codes are computed against the
 *      stored values, so reconstruction uses exactly what is stored.
 *   R14 one contiguous image span [s, s + n), the same for every batch row.
 *   R15 AKVQ-style salient tokens (Sec. 4, optional): in each (batch row, KV
 *      head) that is not protected K+V, the keys and values of the ns image
 *      tokens with the largest squared key norm stay BF16, ties to the lower
 *      token index; ns = ceil(n * permille / 1000) ("a nominal 2%" is
 *      permille 20).  Sec. 4 keeps salient tokens whether or not a head is
 *      protected, so under K-only protection a protected head (whose image keys are BF16
 *      already) keeps its salient tokens' values BF16 and codes the rest of
 *      its image values.  The norm is taken on the unrotated BF16 key in
 *      binary32 in the fixed order of hgo_key_norm2, so that both
 *      implementations rank the same values.  The remaining image tokens are
 *      quantized in order and stored compacted.  Built for the per-token
 *      bases (the paper's salient tokens belong to the AKVQ-style base; the
 *      KIVI-style key groups of 32 consecutive tokens leave no room for
 *      them).
 *   R16 3-bit codes (the paper's 3-bit setting, Sec. 4 / Tab. 1): a group of
 *      n codes (n a multiple of 32) is stored as n/16 words holding bits 0-1
 *      of every code in the 2-bit packing, then n/32 words holding bit 2 of
 *      every code, one bit per code: element e at word e / 32, bit position
 *      (e mod 32) with its index bits 3 and 4 exchanged.  3 bits per code,
 *      and the bit-2 plane of two codes that share a 2-bit word at a 16-bit
 *      distance sits at a 16-bit distance too.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define HGO_D 128

enum { HGO_BASE_MINMAX = 0, HGO_BASE_KIVI = 1, HGO_BASE_AKVQ = 2 };

/* ------------------------------------------------------------------------ */
/* Element conversion                                                         */
/* ------------------------------------------------------------------------ */

/* BF16 is the upper half of a binary32: widening is an exact bit shift. */
float hgo_bf16_to_f32(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* ------------------------------------------------------------------------ */
/* Sec. 1 / Sec. 4: the group quantizer Q used by every base.                 */
/* ------------------------------------------------------------------------ */

/*
 * Quantize n values x[i*stride] to b-bit codes.  The range comes from the
 * group's own minimum and maximum (Sec. 1); every entry is rounded to the
 * nearest of the 2^b levels in that range (R1-R4, R12):
 *   mn, mx   = min, max of the group (signed zeros canonicalised to +0)
 *   scale    = fl32( fl32(mx - mn) / (2^b - 1) )
 *   code_i   = 0                                       if scale == 0
 *            = clamp(rint_even( fl32( fl32(x_i - mn) / scale ) ), 0, 2^b - 1)
 *   zero     = mn
 */
/* IEEE binary16 bits of a binary32 value: round to nearest even; magnitudes
 * of 65504 and above (and non-finite values) saturate to +-65504 (R13). */
uint16_t hgo_f32_to_f16(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    const uint32_t sign = (u >> 16) & 0x8000u;
    const uint32_t a = u & 0x7fffffffu;
    if (a >= 0x477fe000u) return (uint16_t)(sign | 0x7bffu);    /* >= 65504 */
    if (a <= 0x33000000u) return (uint16_t)sign;                 /* <= 2^-25: rounds to 0 */
    if (a < 0x38800000u) {                                       /* below 2^-14: subnormal */
        const uint32_t e = a >> 23, m = (a & 0x7fffffu) | 0x800000u;
        const uint32_t sh = 126u - e;                            /* value / 2^-24 = m / 2^sh */
        uint32_t q = m >> sh;
        const uint32_t rem = m & ((1u << sh) - 1u), half = 1u << (sh - 1u);
        if (rem > half || (rem == half && (q & 1u))) ++q;
        return (uint16_t)(sign | q);
    }
    uint32_t r = (a - 0x38000000u) >> 13;                        /* rebias 127 -> 15, 23 -> 10 bits */
    const uint32_t rem = a & 0x1fffu;
    if (rem > 0x1000u || (rem == 0x1000u && (r & 1u))) ++r;
    return (uint16_t)(sign | r);
}

float hgo_f16_to_f32(uint16_t h)
{
    const uint32_t sign = ((uint32_t)h & 0x8000u) << 16;
    const uint32_t e = ((uint32_t)h >> 10) & 0x1fu, m = (uint32_t)h & 0x3ffu;
    float f;
    if (e == 0) {
        f = (float)m * 5.9604644775390625e-8f; /* m * 2^-24, exact */
    } else {
        const uint32_t u = ((e + 112u) << 23) | (m << 13);
        memcpy(&f, &u, 4);
    }
    return sign ? -f : f;
}

/* The group quantizer with the metadata width as a parameter (meta16: R13). */
void hgo_quantize_group_m(const float *x, int n, int stride, int bits, int meta16,
                          uint8_t *codes, float *scale_out, float *zero_out)
{
    float mn = x[0], mx = x[0];
    for (int i = 1; i < n; ++i) {
        float xi = x[(long)i * stride];
        if (xi < mn) mn = xi;
        if (xi > mx) mx = xi;
    }
    mn = mn + 0.0f; /* R12 */
    mx = mx + 0.0f;
    const float levels = (float)((1 << bits) - 1);
    float scale = (mx - mn) / levels;
    float zero = mn;
    if (meta16) {
        scale = hgo_f16_to_f32(hgo_f32_to_f16(scale));
        zero = hgo_f16_to_f32(hgo_f32_to_f16(zero));
    }
    for (int i = 0; i < n; ++i) {
        if (scale == 0.0f) {
            codes[i] = 0;
            continue;
        }
        float d = x[(long)i * stride] - zero;
        float q = d / scale;
        float r = nearbyintf(q);
        if (r < 0.0f) r = 0.0f;
        if (r > levels) r = levels;
        codes[i] = (uint8_t)r;
    }
    *scale_out = scale;
    *zero_out = zero;
}

void hgo_quantize_group(const float *x, int n, int stride, int bits,
                        uint8_t *codes, float *scale_out, float *zero_out)
{
    hgo_quantize_group_m(x, n, stride, bits, 0, codes, scale_out, zero_out);
}

/* Sec. 4 "reconstructed as floating-point values": x^ = fl32(fl32(code*scale) + zero). */
float hgo_dequant(uint8_t code, float scale, float zero)
{
    float prod = (float)code * scale;
    return prod + zero;
}

/* R16: bit position of element e's bit 2 inside its 32-element plane word. */
int hgo_plane_pos(int e)
{
    const int r = e % 32;
    return (r & 7) | (((r >> 4) & 1) << 3) | (((r >> 3) & 1) << 4);
}

/*
 * Canonical bit packing: element e of a group goes to word e / (32/b), bit
 * offset b * (e mod 32/b), least significant bits first (b = 2, 4).  For
 * b = 3 (R16) the low two bits of every code are packed as for b = 2 into the
 * first n/16 words and bit 2 into n/32 plane words after them.
 */
void hgo_pack(const uint8_t *codes, int n, int bits, uint32_t *words)
{
    if (bits == 3) {
        const int nlo = n / 16, nhi = n / 32;
        for (int w = 0; w < nlo + nhi; ++w) words[w] = 0u;
        for (int e = 0; e < n; ++e) {
            words[e / 16] |= ((uint32_t)(codes[e] & 3u)) << (2 * (e % 16));
            words[nlo + e / 32] |= ((uint32_t)(codes[e] >> 2) & 1u) << hgo_plane_pos(e);
        }
        return;
    }
    const int per_word = 32 / bits;
    const int nwords = (n + per_word - 1) / per_word;
    for (int w = 0; w < nwords; ++w) words[w] = 0u;
    for (int e = 0; e < n; ++e)
        words[e / per_word] |= ((uint32_t)codes[e]) << (bits * (e % per_word));
}

/* Element e of a packed group of n codes. */
uint8_t hgo_unpack_group(const uint32_t *words, int n, int e, int bits)
{
    if (bits == 3) {
        const uint32_t lo = (words[e / 16] >> (2 * (e % 16))) & 3u;
        const uint32_t hi = (words[n / 16 + e / 32] >> hgo_plane_pos(e)) & 1u;
        return (uint8_t)(lo | (hi << 2));
    }
    const int per_word = 32 / bits;
    return (uint8_t)((words[e / per_word] >> (bits * (e % per_word))) & ((1u << bits) - 1u));
}

uint8_t hgo_unpack(const uint32_t *words, int e, int bits)
{
    return hgo_unpack_group(words, 0, e, bits == 3 ? 2 : bits);
}

/* ------------------------------------------------------------------------ */
/* Sec. 4, AKVQ-style base: orthonormal Hadamard-128 rotation.                */
/* ------------------------------------------------------------------------ */

/* fl32(1 / sqrt(128)), bit pattern 0x3DB504F3. */
static float hgo_hadamard_c(void)
{
    uint32_t u = 0x3DB504F3u;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/*
 * In-place normalised Walsh-Hadamard transform in Sylvester (natural) order.
 * Stages h = 1, 2, 4, ..., 64; within a stage every pair (a, b) =
 * (x[i+j], x[i+j+h]) becomes (a + b, a - b); the 1/sqrt(128) factor is one
 * multiply at the end (R9).  H is symmetric and orthonormal, so the same call
 * is its own inverse.
 */
void hgo_fwht128(float *x)
{
    for (int h = 1; h < HGO_D; h <<= 1) {
        for (int i = 0; i < HGO_D; i += 2 * h) {
            for (int j = i; j < i + h; ++j) {
                float a = x[j], b = x[j + h];
                x[j] = a + b;
                x[j + h] = a - b;
            }
        }
    }
    const float c = hgo_hadamard_c();
    for (int i = 0; i < HGO_D; ++i) x[i] = x[i] * c;
}

/* The same transform in binary64 with the exact scale 1/sqrt(128). */
void hgo_fwht128_f64(double *x)
{
    for (int h = 1; h < HGO_D; h <<= 1) {
        for (int i = 0; i < HGO_D; i += 2 * h) {
            for (int j = i; j < i + h; ++j) {
                double a = x[j], b = x[j + h];
                x[j] = a + b;
                x[j + h] = a - b;
            }
        }
    }
    const double c = 1.0 / sqrt((double)HGO_D);
    for (int i = 0; i < HGO_D; ++i) x[i] = x[i] * c;
}

/* ------------------------------------------------------------------------ */
/* Sec. 3 "Applying protection" + Sec. 4 bases: which entries are quantized.  */
/* ------------------------------------------------------------------------ */

/*
 * The image tokens eligible for low precision: [s, s + nq).  For per-token
 * min-max and AKVQ-style this is the whole image span.  For KIVI-style (R7)
 * only full 32-token key groups that lie inside [s, min(s + n, T - R)) are
 * eligible; the rest of the image stays BF16.  Returns nq.
 */
int hgo_quantized_count(int T, int s, int n, int base, int group_tokens, int residual)
{
    if (base != HGO_BASE_KIVI) return n;
    int end = s + n;
    if (T - residual < end) end = T - residual;
    int span = end - s;
    if (span <= 0) return 0;
    return (span / group_tokens) * group_tokens;
}

/*
 * Quantize one (batch row, KV head) of one layer.
 *
 *   k, v       [T][128] BF16 bit patterns, the prefill keys / values
 *   protect    the head's mask bit (Sec. 3): 1 keeps image K (and V unless
 *              keys_only) in BF16; text K/V are BF16 in every case
 *   outputs    kq, vq [T]          1 where that entry is quantized
 *              k_words             per-token bases: [nq][4*bits] (token order,
 *                                  128 channels packed); KIVI: [nq/32][128][bits]
 *                                  (one 32-token group of one channel per row)
 *              k_meta              per-token: [nq][2]; KIVI: [nq/32][128][2]
 *              v_words             [nq][4*bits] (channels packed, any base)
 *              v_meta              per-token: [nq][2]; KIVI: [nq][4][2]
 *              k_deq, v_deq        [T][128] fp32 reconstruction in the
 *                                  original domain (AKVQ keys: the inverse
 *                                  rotation done in fp32 as in hgo_fwht128)
 *              k_att               [T][128] fp64 keys for attention (AKVQ
 *                                  quantized keys: the inverse rotation of
 *                                  the fp32 reconstruction done in fp64), may
 *                                  be NULL
 *   Returns nq.  Metadata pairs are (scale, zero).
 */
float hgo_key_norm2(const uint16_t *krow);
void hgo_select_salient(const float *score, int n, int ns, int32_t *idx);

/*
 * n_salient > 0 (R15; per-token bases): for a head that is not protected K+V
 * (its image values are quantized), the n_salient image tokens of largest key
 * norm keep BF16 keys and values, their image-relative indices go to
 * `salient` (ascending), and the other image tokens are quantized in order
 * into the first nq - n_salient slots of the code and metadata arrays.  A
 * K-only protected head keeps every image key BF16, so only its values are
 * affected.
 */
int hgo_quantize_head_s(const uint16_t *k, const uint16_t *v, int T, int s, int n,
                        int base, int bits, int meta16, int protect, int keys_only,
                        int group_tokens, int group_channels, int residual, int n_salient,
                        uint8_t *kq, uint8_t *vq,
                        uint32_t *k_words, float *k_meta,
                        uint32_t *v_words, float *v_meta,
                        float *k_deq, float *v_deq, double *k_att, int32_t *salient)
{
    const int D = HGO_D;
    const int nq = hgo_quantized_count(T, s, n, base, group_tokens, residual);
    const int quant_k = !protect;
    const int quant_v = !protect || keys_only;
    const int wpt = D * bits / 32; /* words per 128-code vector */

    float xk[HGO_D], xv[HGO_D];
    uint8_t codes[HGO_D];

    /* R15: which image tokens stay BF16 (sal[i] for image token s + i) */
    uint8_t *sal = (uint8_t *)calloc((size_t)(nq > 0 ? nq : 1), 1);
    if (n_salient > 0 && quant_v && base != HGO_BASE_KIVI && nq > 0) {
        float *score = (float *)malloc(sizeof(float) * (size_t)nq);
        for (int i = 0; i < nq; ++i) score[i] = hgo_key_norm2(k + (long)(s + i) * D);
        hgo_select_salient(score, nq, n_salient, salient);
        for (int j = 0; j < n_salient; ++j) sal[salient[j]] = 1;
        free(score);
    }

    /* Start from the BF16 values everywhere; quantized entries are overwritten. */
    for (int t = 0; t < T; ++t) {
        kq[t] = 0;
        vq[t] = 0;
        for (int c = 0; c < D; ++c) {
            k_deq[(long)t * D + c] = hgo_bf16_to_f32(k[(long)t * D + c]);
            v_deq[(long)t * D + c] = hgo_bf16_to_f32(v[(long)t * D + c]);
            if (k_att) k_att[(long)t * D + c] = (double)k_deq[(long)t * D + c];
        }
    }

    /* ---- keys ---- */
    if (quant_k && nq > 0) {
        if (base == HGO_BASE_KIVI) {
            /* per channel, over each group of group_tokens consecutive tokens */
            const int ngroups = nq / group_tokens;
            float col[HGO_D > 64 ? HGO_D : 64];
            for (int g = 0; g < ngroups; ++g) {
                const int t0 = s + g * group_tokens;
                for (int c = 0; c < D; ++c) {
                    float scale, zero;
                    for (int e = 0; e < group_tokens; ++e)
                        col[e] = hgo_bf16_to_f32(k[(long)(t0 + e) * D + c]);
                    hgo_quantize_group_m(col, group_tokens, 1, bits, meta16, codes, &scale, &zero);
                    long row = (long)g * D + c;
                    hgo_pack(codes, group_tokens, bits, k_words + row * (group_tokens * bits / 32));
                    k_meta[row * 2 + 0] = scale;
                    k_meta[row * 2 + 1] = zero;
                    for (int e = 0; e < group_tokens; ++e) {
                        float r = hgo_dequant(codes[e], scale, zero);
                        k_deq[(long)(t0 + e) * D + c] = r;
                        if (k_att) k_att[(long)(t0 + e) * D + c] = (double)r;
                    }
                }
            }
        } else {
            for (int i = 0, ci = -1; i < nq; ++i) {
                const int t = s + i;
                if (sal[i]) continue; /* R15: stays BF16 */
                ++ci;
                float scale, zero;
                for (int c = 0; c < D; ++c) xk[c] = hgo_bf16_to_f32(k[(long)t * D + c]);
                if (base == HGO_BASE_AKVQ) hgo_fwht128(xk); /* rotate, then per-token RTN */
                hgo_quantize_group_m(xk, D, 1, bits, meta16, codes, &scale, &zero);
                hgo_pack(codes, D, bits, k_words + (long)ci * wpt);
                k_meta[(long)ci * 2 + 0] = scale;
                k_meta[(long)ci * 2 + 1] = zero;
                float r[HGO_D];
                for (int c = 0; c < D; ++c) r[c] = hgo_dequant(codes[c], scale, zero);
                if (base == HGO_BASE_AKVQ) {
                    if (k_att) {
                        double rd[HGO_D];
                        for (int c = 0; c < D; ++c) rd[c] = (double)r[c];
                        hgo_fwht128_f64(rd);
                        for (int c = 0; c < D; ++c) k_att[(long)t * D + c] = rd[c];
                    }
                    hgo_fwht128(r); /* inverse rotation back to the key domain */
                } else if (k_att) {
                    for (int c = 0; c < D; ++c) k_att[(long)t * D + c] = (double)r[c];
                }
                for (int c = 0; c < D; ++c) k_deq[(long)t * D + c] = r[c];
            }
        }
        for (int i = 0; i < nq; ++i) kq[s + i] = sal[i] ? 0 : 1;
    }

    /* ---- values (never rotated, R9) ---- */
    if (quant_v && nq > 0) {
        const int gsize = (base == HGO_BASE_KIVI) ? group_channels : D;
        const int ngr = D / gsize;
        for (int i = 0, ci = -1; i < nq; ++i) {
            const int t = s + i;
            if (sal[i]) continue; /* R15: stays BF16 */
            ++ci;
            for (int c = 0; c < D; ++c) xv[c] = hgo_bf16_to_f32(v[(long)t * D + c]);
            for (int j = 0; j < ngr; ++j) {
                float scale, zero;
                hgo_quantize_group_m(xv + j * gsize, gsize, 1, bits, meta16, codes + j * gsize, &scale, &zero);
                v_meta[((long)ci * ngr + j) * 2 + 0] = scale;
                v_meta[((long)ci * ngr + j) * 2 + 1] = zero;
                for (int e = 0; e < gsize; ++e)
                    v_deq[(long)t * D + j * gsize + e] = hgo_dequant(codes[j * gsize + e], scale, zero);
            }
            /* group j's element e is channel j*gsize + e: the channel-order packing */
            hgo_pack(codes, D, bits, v_words + (long)ci * wpt);
            vq[t] = 1;
        }
    }
    free(sal);
    return nq;
}

int hgo_quantize_head_m(const uint16_t *k, const uint16_t *v, int T, int s, int n,
                        int base, int bits, int meta16, int protect, int keys_only,
                        int group_tokens, int group_channels, int residual,
                        uint8_t *kq, uint8_t *vq,
                        uint32_t *k_words, float *k_meta,
                        uint32_t *v_words, float *v_meta,
                        float *k_deq, float *v_deq, double *k_att)
{
    return hgo_quantize_head_s(k, v, T, s, n, base, bits, meta16, protect, keys_only, group_tokens,
                               group_channels, residual, 0, kq, vq, k_words, k_meta, v_words, v_meta,
                               k_deq, v_deq, k_att, NULL);
}

/* ------------------------------------------------------------------------ */
/* Sec. 4 AKVQ-style salient tokens (R15).                                    */
/* ------------------------------------------------------------------------ */

/*
 * Squared norm of one BF16 key row in binary32, in a fixed order: 32 partial
 * sums of four consecutive channels each, ((x0^2 + x1^2) + x2^2) + x3^2, then
 * five pairwise rounds in which partial l becomes partial l + partial (l xor m)
 * for m = 16, 8, 4, 2, 1; the result is partial 0.
 */
float hgo_key_norm2(const uint16_t *krow)
{
    float part[32], next[32];
    for (int l = 0; l < 32; ++l) {
        float a = 0.0f;
        for (int j = 0; j < 4; ++j) {
            const float x = hgo_bf16_to_f32(krow[4 * l + j]);
            const float sq = x * x;
            a = (j == 0) ? sq : a + sq;
        }
        part[l] = a;
    }
    for (int m = 16; m >= 1; m >>= 1) {
        for (int l = 0; l < 32; ++l) next[l] = part[l] + part[l ^ m];
        memcpy(part, next, sizeof part);
    }
    return part[0];
}

/* Salient tokens per head for n image tokens at a per-mille rate, rounded up. */
int hgo_salient_count(int n, int permille)
{
    if (permille <= 0 || n <= 0) return 0;
    return (int)(((long)n * permille + 999) / 1000);
}

/*
 * The ns indices in [0, n) with the largest scores (ties: the lower index
 * first), written in ascending order.
 */
void hgo_select_salient(const float *score, int n, int ns, int32_t *idx)
{
    uint8_t *taken = (uint8_t *)calloc((size_t)(n > 0 ? n : 1), 1);
    for (int j = 0; j < ns; ++j) {
        int best = -1;
        for (int i = 0; i < n; ++i)
            if (!taken[i] && (best < 0 || score[i] > score[best])) best = i;
        if (best >= 0) taken[best] = 1;
    }
    int c = 0;
    for (int i = 0; i < n; ++i)
        if (taken[i]) idx[c++] = i;
    free(taken);
}

/*
 * One layer, every (batch row, KV head), with per-head output slots of fixed
 * size (heads that quantize nothing leave their slots untouched):
 *   k_words [B][H][nq*4*bits]   k_meta [B][H][km]   (km = nq*2, KIVI nq/32*128*2)
 *   v_words [B][H][nq*4*bits]   v_meta [B][H][vm]   (vm = nq*2, KIVI nq*4*2)
 *   kq, vq  [B][H][T]           k_deq, v_deq [B][H][T][128]   k_att likewise or NULL
 * head_mask[h] is the layer's protection mask.  Parallel over (b, h) when
 * built with OpenMP; every head is computed independently.
 */
int hgo_quantize_layer_s(const uint16_t *k, const uint16_t *v, int B, int H, int T,
                         int s, int n, int base, int bits, int meta16, const uint8_t *head_mask,
                         int keys_only, int group_tokens, int group_channels, int residual,
                         int n_salient,
                         uint8_t *kq, uint8_t *vq,
                         uint32_t *k_words, float *k_meta, uint32_t *v_words, float *v_meta,
                         float *k_deq, float *v_deq, double *k_att, int32_t *salient)
{
    const int D = HGO_D;
    const int nq = hgo_quantized_count(T, s, n, base, group_tokens, residual);
    if (n_salient < 0 || n_salient > nq) return -1;
    if (n_salient > 0 && base == HGO_BASE_KIVI) return -1; /* R15: per-token bases only */
    const long kw = (long)nq * D * bits / 32;
    const long km = (base == HGO_BASE_KIVI) ? (long)(nq / group_tokens) * D * 2 : (long)nq * 2;
    const long vm = (base == HGO_BASE_KIVI) ? (long)nq * (D / group_channels) * 2 : (long)nq * 2;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        const int h = bh % H;
        const long tok = (long)bh * T;
        hgo_quantize_head_s(k + tok * D, v + tok * D, T, s, n, base, bits, meta16, head_mask[h], keys_only,
                            group_tokens, group_channels, residual, n_salient, kq + tok, vq + tok,
                            k_words + bh * kw, k_meta + bh * km, v_words + bh * kw, v_meta + bh * vm,
                            k_deq + tok * D, v_deq + tok * D, k_att ? k_att + tok * D : NULL,
                            salient ? salient + (long)bh * n_salient : NULL);
    }
    return nq;
}

int hgo_quantize_layer_m(const uint16_t *k, const uint16_t *v, int B, int H, int T,
                         int s, int n, int base, int bits, int meta16, const uint8_t *head_mask,
                         int keys_only, int group_tokens, int group_channels, int residual,
                         uint8_t *kq, uint8_t *vq,
                         uint32_t *k_words, float *k_meta, uint32_t *v_words, float *v_meta,
                         float *k_deq, float *v_deq, double *k_att)
{
    return hgo_quantize_layer_s(k, v, B, H, T, s, n, base, bits, meta16, head_mask, keys_only,
                                group_tokens, group_channels, residual, 0, kq, vq, k_words, k_meta,
                                v_words, v_meta, k_deq, v_deq, k_att, NULL);
}

/* The 64-bit-metadata forms (R5). */
int hgo_quantize_head(const uint16_t *k, const uint16_t *v, int T, int s, int n,
                      int base, int bits, int protect, int keys_only,
                      int group_tokens, int group_channels, int residual,
                      uint8_t *kq, uint8_t *vq,
                      uint32_t *k_words, float *k_meta,
                      uint32_t *v_words, float *v_meta,
                      float *k_deq, float *v_deq, double *k_att)
{
    return hgo_quantize_head_m(k, v, T, s, n, base, bits, 0, protect, keys_only, group_tokens,
                               group_channels, residual, kq, vq, k_words, k_meta, v_words, v_meta,
                               k_deq, v_deq, k_att);
}

int hgo_quantize_layer(const uint16_t *k, const uint16_t *v, int B, int H, int T,
                       int s, int n, int base, int bits, const uint8_t *head_mask,
                       int keys_only, int group_tokens, int group_channels, int residual,
                       uint8_t *kq, uint8_t *vq,
                       uint32_t *k_words, float *k_meta, uint32_t *v_words, float *v_meta,
                       float *k_deq, float *v_deq, double *k_att)
{
    return hgo_quantize_layer_m(k, v, B, H, T, s, n, base, bits, 0, head_mask, keys_only,
                                group_tokens, group_channels, residual, kq, vq, k_words, k_meta,
                                v_words, v_meta, k_deq, v_deq, k_att);
}

/* ------------------------------------------------------------------------ */
/* Decode attention over the reconstructed cache, binary64.                   */
/* ------------------------------------------------------------------------ */

/*
 * One query vector q[128] against keys K[Tt][128] and values V[Tt][128]:
 *   score_t = sigma * sum_d q_d K_td,  p = softmax(score),  out_d = sum_t p_t V_td.
 * The softmax is taken after subtracting the maximum score, in binary64.
 */
void hgo_attention_one(const double *q, const double *K, const double *V, int Tt,
                       double sigma, double *out, double *scratch_scores)
{
    const int D = HGO_D;
    double m = -INFINITY;
    for (int t = 0; t < Tt; ++t) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d) acc += q[d] * K[(long)t * D + d];
        scratch_scores[t] = sigma * acc;
        if (scratch_scores[t] > m) m = scratch_scores[t];
    }
    double l = 0.0;
    for (int t = 0; t < Tt; ++t) {
        scratch_scores[t] = exp(scratch_scores[t] - m);
        l += scratch_scores[t];
    }
    for (int d = 0; d < D; ++d) out[d] = 0.0;
    for (int t = 0; t < Tt; ++t) {
        const double p = scratch_scores[t] / l;
        for (int d = 0; d < D; ++d) out[d] += p * V[(long)t * D + d];
    }
}

/*
 * Grouped-query decode for one layer (R11):
 *   q    [B][Hq][128] BF16 bit patterns (the step's queries)
 *   K, V [B][H][Tt][128] binary64 (dequantized prefill followed by the
 *        appended BF16 tokens, in any order: softmax attention is invariant
 *        under a permutation of the tokens)
 *   out  [B][Hq][128] binary64;  query head qh reads KV head qh / (Hq / H).
 */
int hgo_attention_layer(const uint16_t *q, const double *K, const double *V, int B, int Hq, int H,
                        int Tt, double sigma, double *out)
{
    const int D = HGO_D;
    if (H <= 0 || Hq % H != 0) return -1;
    const int G = Hq / H;
    int err = 0;
#pragma omp parallel
    {
        double *scores = (double *)malloc(sizeof(double) * (size_t)(Tt > 0 ? Tt : 1));
        if (!scores) {
#pragma omp atomic write
            err = -2;
        }
#pragma omp for schedule(dynamic, 1)
        for (int bq = 0; bq < B * Hq; ++bq) {
            if (!scores) continue;
            const int b = bq / Hq, qh = bq % Hq, h = qh / G;
            double qd[HGO_D];
            for (int d = 0; d < D; ++d) qd[d] = (double)hgo_bf16_to_f32(q[(long)bq * D + d]);
            const long kv = ((long)b * H + h) * Tt * D;
            hgo_attention_one(qd, K + kv, V + kv, Tt, sigma, out + (long)bq * D, scores);
        }
        free(scores);
    }
    return err;
}

/* ------------------------------------------------------------------------ */
/* Sec. 5.4 storage model.                                                    */
/* ------------------------------------------------------------------------ */

/*
 * Image-cache bits per element for 128-d K/V vectors: a quantized vector costs
 * bits + meta_bits/128 per element, a protected one 16.  With a fraction f of
 * heads protected, K+V protection gives (1-f)*q + f*16 for both K and V;
 * keys-only protection gives that for K and q for V, averaged over K and V.
 */
double hgo_image_bits_per_elem(int bits, int meta_bits, int head_dim, double frac_protected,
                               int keys_only)
{
    const double qbits = (double)bits + (double)meta_bits / (double)head_dim;
    const double kbits = (1.0 - frac_protected) * qbits + frac_protected * 16.0;
    const double vbits = keys_only ? qbits : kbits;
    return 0.5 * (kbits + vbits);
}
