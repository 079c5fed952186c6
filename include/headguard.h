/*
 * headguard.h -- C ABI of the HeadGuard mixed-precision KV-cache library
 * (GB300 / sm_103a).
 *
 * The library implements the data-parallel path of "HeadGuard: Selective Head
 * Protection for Low-Bit VLM KV-Cache Quantization":
 *   - quantize and bit-pack each layer's image-token keys / values with one of
 *     three base quantizers (Sec. 1 per-token min-max RTN; Sec. 4 KIVI-style
 *     per-channel keys / per-token values; Sec. 4 AKVQ-style Hadamard-128
 *     rotation + per-token RTN), keeping the protected KV heads' image keys
 *     (and values, unless keys-only) and every text token in BF16 (Sec. 3,
 *     "Applying protection");
 *   - reconstruct the cache as floating point (Sec. 4, simulated quantization:
 *     values rounded to the quantizer's levels and reconstructed as floats);
 *   - grouped-query decode attention that reads packed 2/3/4-bit codes and BF16
 *     entries in one pass.
 *
 * Conventions shared by every entry point
 *   Memory     The caller owns every byte.  The library never allocates device
 *              memory at run time; the cache lives in a caller-provided device
 *              "arena", and decode attention uses a caller-provided workspace
 *              (hg_decode_attention_noalloc instead uses a static 32 MiB array
 *              the library holds on every GPU that loads it).  The only host
 *              allocation is the hg_cache descriptor itself.
 *   Tensors    Device tensors are dense row-major BF16 (uint16 bit patterns)
 *              unless stated otherwise, head_dim = 128, and must be 16-byte
 *              aligned.  The per-step decode inputs and outputs (q, k_new,
 *              v_new, out) may instead be pinned host memory, which the
 *              kernels read and write directly over the host link (no copy
 *              engine round trip for a step's few hundred kilobytes).
 *   Streams    Every device operation is enqueued on the given stream
 *              (hg_stream_t is cudaStream_t; NULL means the legacy default
 *              stream) and returns before the GPU work completes.
 *   Errors     Arguments are validated on the host before anything is
 *              launched; a call that returns an error has enqueued nothing and
 *              changed no state.  HG_ERR_CUDA reports a launch error returned
 *              by the CUDA runtime (cudaGetLastError after the launch).
 *              The only polling waits in device code are decode CTAs waiting
 *              on mbarriers for their own tile copies, each bounded: one that runs out
 *              sets the workspace status word (hg_workspace_status) instead
 *              of hanging.
 *   Threads    A hg_cache may be used from one host thread at a time.
 */
#ifndef HEADGUARD_H
#define HEADGUARD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t, declared without the CUDA headers. */
typedef struct CUstream_st *hg_stream_t;

typedef enum hg_status {
    HG_OK = 0,
    HG_ERR_INVALID_ARG = 1,        /* null pointer, out-of-range index or size     */
    HG_ERR_ALIGNMENT = 2,          /* a device pointer is not 16-byte aligned       */
    HG_ERR_UNSUPPORTED = 3,        /* valid but not implemented (head_dim != 128 ..) */
    HG_ERR_WORKSPACE_TOO_SMALL = 4,/* decode workspace smaller than required         */
    HG_ERR_CAPACITY = 5,           /* append beyond max_new_tokens                   */
    HG_ERR_CUDA = 6,               /* the CUDA runtime reported an error             */
    HG_ERR_ARENA_TOO_SMALL = 7     /* cache arena smaller than hg_cache_layout says  */
} hg_status;

/* Base quantizers (Sec. 1 and Sec. 4). */
typedef enum hg_base {
    HG_BASE_MINMAX_TOKEN = 0,   /* per-token min-max, round to nearest level         */
    HG_BASE_KIVI = 1,           /* keys per channel over 32-token groups, values per
                                   token over 32-channel groups, BF16 residual window */
    HG_BASE_AKVQ_HADAMARD = 2   /* keys rotated by the orthonormal Hadamard-128, then
                                   per-token; values per-token, unrotated             */
} hg_base;

/* Cache geometry.  K/V of one layer are [batch][num_kv_heads][seq_len][head_dim].
 * The image tokens are the contiguous span [img_start, img_start + img_len), the
 * same for every batch row; every other prefill token is text (Sec. 3: text K/V
 * stay BF16).  max_new_tokens is the decode-time capacity for appended tokens. */
typedef struct hg_shape {
    int32_t batch;
    int32_t num_layers;
    int32_t num_kv_heads;     /* 1..64 */
    int32_t num_q_heads;      /* multiple of num_kv_heads, G = num_q_heads / num_kv_heads <= 16 */
    int32_t head_dim;         /* must be 128 (the paper's heads, Sec. 5.4) */
    int32_t seq_len;          /* prefill length T >= 1 */
    int32_t img_start;
    int32_t img_len;          /* img_start + img_len <= seq_len */
    int32_t max_new_tokens;
} hg_shape;

/* Quantizer configuration.  bits in {2, 3, 4} (3 bits: each group stores bits
 * 0-1 of its codes as in the 2-bit packing, then bit 2 as a plane of one bit
 * per code, element e at plane word e / 32, bit e mod 32 with index bits 3
 * and 4 exchanged).  keys_only selects K-only protection
 * (Sec. 3: protected heads keep image keys BF16, their image values follow the
 * base).  The KIVI-style group sizes must be 32; kivi_residual >= 0 is the number
 * of trailing prefill tokens kept BF16.  Unused fields are ignored for other bases.
 * meta_bits: metadata per group, 64 (or 0: the default) = an fp32 {scale, zero}
 * pair; 32 = a binary16 pair, the Sec. 5.4 storage model (2.25 bits per element
 * at 2 bits): scale and zero are rounded to nearest-even binary16 (magnitudes
 * >= 65504 saturate) and the codes are computed against the stored values.
 * salient_permille (0 = off; AKVQ-style base only, else HG_ERR_UNSUPPORTED):
 * Sec. 4's salient tokens, kept whether or not a head is protected.  In every
 * (batch row, KV head) that is not protected K+V, ceil(nq * salient_permille /
 * 1000) image tokens (20: the paper's nominal 2%) with the largest squared
 * norm of the unrotated BF16 key keep BF16 keys and values (a keys-only
 * protected head keeps every image key BF16 anyway, so there only its salient
 * values change); ties go to the lower token index.  The squared norm is summed in binary32 in a fixed order: 32 partial
 * sums of channels 4l..4l+3, ((x0^2 + x1^2) + x2^2) + x3^2, then five rounds
 * in which partial l adds partial (l xor m), m = 16, 8, 4, 2, 1.  The other
 * image tokens are coded in order, compacted. */
typedef struct hg_quant_config {
    int32_t base;
    int32_t bits;
    int32_t keys_only;
    int32_t kivi_group_tokens;
    int32_t kivi_group_channels;
    int32_t kivi_residual;
    int32_t meta_bits;
    int32_t salient_permille;
} hg_quant_config;

/* Opaque host-side descriptor of a cache arena (offsets, mask, appended counts). */
typedef struct hg_cache hg_cache;

/* Class of a (layer, KV head), from the protection mask (Sec. 3). */
typedef enum hg_head_class {
    HG_HEAD_QUANTIZED = 0,  /* image K and V follow the base quantizer          */
    HG_HEAD_KEYS_ONLY = 1,  /* protected, keys-only: image K BF16, image V coded */
    HG_HEAD_PROTECTED = 2   /* protected K+V: image K and V BF16                 */
} hg_head_class;

/* Where one (layer, KV head) lives in the arena.  Offsets are bytes from the
 * arena base of element [b = 0][t = 0]; each *_bstride is the byte stride
 * between batch rows; an absent region has offset UINT64_MAX.
 *   kb / vb   BF16 [batch][bf16_capacity][128]: the head's BF16 tokens in
 *             prefill order (text, image tokens not quantized), then appended
 *             tokens.  bf16_prefill of them come from the prefill.  With
 *             salient tokens: leading text, the salient image tokens in token
 *             order, trailing text, appended tokens.
 *   kq / kqm  key codes / metadata (quantized class only).  Per-token bases:
 *             codes uint32 [batch][nq][4*bits] (128 codes, channel order, packed
 *             LSB-first, 32/bits per word; 3 bits: 8 words + 4 plane words), metadata float2 {scale, zero}
 *             [batch][nq].  KIVI-style: codes [batch][nq/32][128][bits] (one
 *             32-token group of one channel, token order), metadata
 *             [batch][nq/32][128].
 *   vq / vqm  value codes [batch][nq][4*bits] (channel order), metadata
 *             [batch][nq][groups], groups = 1 (per token) or 4 (KIVI-style,
 *             channels 32j..32j+31).
 *   kimg      BF16 [batch][n_coded][128] image keys of a keys-only protected
 *             head (with salient tokens: those of the coded tokens, compacted;
 *             the salient tokens' keys sit in kb).
 *   sal       salient-token map of a head with coded values (salient tokens only):
 *             per batch row uint32 [ceil(nq/32)] (bit j of word w: image
 *             token 32w + j is salient), then int32 [ceil(nq/32)] (salient
 *             tokens before block w), row stride sal_bstride.
 * Quantized image tokens are [img_start, img_start + nq); nq equals img_len
 * except for KIVI-style, where only whole 32-token groups inside
 * [img_start, min(img_start + img_len, seq_len - kivi_residual)) are coded.
 * The code and metadata arrays hold n_coded tokens (nq less the n_salient
 * salient tokens of a head with coded values), in token order. */
typedef struct hg_head_regions {
    int32_t head_class;
    int32_t nq;
    int32_t bf16_prefill;
    int32_t bf16_capacity;
    uint64_t kb, vb, kq, kqm, vq, vqm, kimg;
    uint64_t kb_bstride, kq_bstride, kqm_bstride, vq_bstride, vqm_bstride, kimg_bstride;
    uint64_t sal, sal_bstride;
    int32_t n_coded, n_salient;
} hg_head_regions;

/* Bytes of device arena a cache of this shape / config / mask needs.
 * head_mask: host uint8 [num_layers][num_kv_heads], non-zero = protected
 * (Sec. 3, Eq. 2's selected set P).  Host only; no CUDA call. */
hg_status hg_cache_layout(const hg_shape *shape, const hg_quant_config *config,
                          const uint8_t *head_mask, size_t *arena_bytes);

/* Create the descriptor of a cache stored in `arena` (device, 256-byte aligned,
 * at least hg_cache_layout bytes; its contents need no initialisation).  The
 * descriptor copies shape, config and mask (the fixed head set chosen offline,
 * Sec. 3).  Host only; no CUDA call.
 * The arena must outlive the descriptor's use; hg_cache_destroy frees only the
 * descriptor. */
hg_status hg_cache_create(const hg_shape *shape, const hg_quant_config *config,
                          const uint8_t *head_mask, void *arena, size_t arena_bytes,
                          hg_cache **out);
void hg_cache_destroy(hg_cache *cache);

/* Region map of one (layer, head): where its BF16 rows, codes and metadata sit
 * in the arena.  The packed layout is this library's (the paper stores no
 * packed cache, Sec. 4).  Host only. */
hg_status hg_cache_head_regions(const hg_cache *cache, int32_t layer, int32_t head,
                                hg_head_regions *out);

/* Number of decode tokens appended so far to `layer` (host state; generated
 * tokens are text and stay BF16, Sec. 3). */
int32_t hg_cache_appended(const hg_cache *cache, int32_t layer);

/* Forget appended tokens (all layers); device memory is not touched.  (Cache
 * bookkeeping; the paper has no counterpart.) */
hg_status hg_cache_reset_appended(hg_cache *cache);

/* Quantize-pack layers [layer_begin, layer_begin + layer_count) from their BF16
 * prefill K/V (Sec. 3 protection over a Sec. 1 / Sec. 4 base).  k and v are HOST
 * arrays of layer_count DEVICE pointers, each [batch][num_kv_heads][seq_len][128]
 * BF16; they are only read and may be freed once the stream work completes.
 * Writes every region of those layers.  Packed codes and fp32 (scale, zero)
 * follow the group quantizer: scale = (max - min) / (2^bits - 1), code =
 * round-half-even((x - min) / scale), zero = min, codes 0 when scale == 0. */
hg_status hg_quantize_kv(hg_cache *cache, int32_t layer_begin, int32_t layer_count,
                         const void *const *k, const void *const *v, hg_stream_t stream);

/* Reconstruct layers [layer_begin, layer_begin + layer_count) as floating
 * point (Sec. 4: code * scale + zero, the AKVQ-style keys rotated back).
 * k_out / v_out: device [layer_count][batch][num_kv_heads][seq_len + appended][128],
 * fp32 when out_fp32 != 0, else BF16 (round to nearest even), tokens in
 * original order followed by the appended ones.  BF16 entries are copied
 * exactly.  Every layer of the range must hold the same number of appended
 * tokens (HG_ERR_INVALID_ARG otherwise); one launch per 64 layers. */
hg_status hg_dequantize_kv(const hg_cache *cache, int32_t layer_begin, int32_t layer_count,
                           void *k_out, void *v_out, int32_t out_fp32, hg_stream_t stream);

/* Append one decode token's K/V to layers [layer_begin, +layer_count) (text
 * tokens stay BF16, Sec. 3).  k_new / v_new: device BF16
 * [layer_count][batch][num_kv_heads][128].  Returns HG_ERR_CAPACITY if a layer
 * already holds max_new_tokens appended tokens.  Advances the host-side count. */
hg_status hg_append_kv(hg_cache *cache, int32_t layer_begin, int32_t layer_count,
                       const void *k_new, const void *v_new, hg_stream_t stream);

/* Workspace bytes hg_decode_attention needs for a launch over layer_count
 * layers (any appended count up to max_new_tokens).  The workspace holds the
 * split-K partials of the decode kernel (a GPU work decomposition; the paper
 * has no counterpart). */
hg_status hg_decode_workspace_size(const hg_cache *cache, int32_t layer_count, size_t *bytes);

/* Zero a workspace (cudaMemsetAsync; no counterpart in the paper).  Required
 * once before its first use; decode attention leaves it zeroed again on
 * completion.  Layout: a 512-byte header holding a status word at byte 0,
 * split counters, split partials.  workspace NULL: clear the status word of
 * the scratch array hg_decode_attention_noalloc uses on the current device
 * (`bytes` is ignored). */
hg_status hg_workspace_clear(void *workspace, size_t bytes, hg_stream_t stream);

/* Health of the decode launches that used a workspace: waits for `stream`,
 * then copies the workspace's status word to *status (host).  0 = healthy;
 * bit 0 (1) = a CTA's wait for a tile of its data ran out (after about a
 * second), after which that CTA skipped its remaining work and
 * let the copies it had issued land before exiting.  Decode CTAs wait with a
 * bound instead of hanging; after a non-zero status the outputs of the
 * launches since the last clear are undefined and the workspace must be
 * cleared (hg_workspace_clear) before it is used again.  workspace NULL: the
 * status word of the scratch array hg_decode_attention_noalloc uses on the
 * current device, which collects the failures of every allocation-free call
 * since it was last cleared with hg_workspace_clear(NULL, 0, stream).
 * (Failure detection of the kernels; the paper has no counterpart.) */
hg_status hg_workspace_status(const void *workspace, uint32_t *status, hg_stream_t stream);

/* Self-check of the bounded wait that guards every decode tile (failure
 * detection; the paper has no counterpart).  One CTA waits on an mbarrier
 * phase that has completed and on one that nothing will complete, each with
 * the decode kernel's wait routine bounded to `rounds` suspensions of up to
 * 50 us (1 <= rounds <= 100000).  `word`: device, 16-byte aligned, 4 bytes,
 * zeroed by this call; when the stream reaches the end it holds 3 if the
 * completed wait succeeded (bit 1) and the other one gave up and flagged the
 * timeout (bit 0).  Faults and hangs nothing: the wait that cannot succeed
 * returns after at most rounds * 50 us. */
hg_status hg_check_bounded_wait(void *word, uint32_t rounds, hg_stream_t stream);

/* Grouped-query decode attention of one step over layers
 * [layer_begin, +layer_count), reading packed codes and BF16 entries in one
 * pass: attention over the mixed-precision cache of Sec. 3 (protected and text
 * entries BF16, the other image entries the base quantizer's reconstruction,
 * which Sec. 4 feeds to attention as floating point; here the codes enter the
 * contraction directly).  q: device BF16 [layer_count][batch][num_q_heads][128]; out: device
 * BF16, same shape.  Query head qh attends with KV head qh / G over every
 * token of that head (prefill text, image, appended), with
 * score = softmax_scale * <q, k>; softmax_scale <= 0 selects 1/sqrt(128).
 * workspace: device, >= hg_decode_workspace_size(layer_count) bytes, zeroed
 * once by hg_workspace_clear; one launch at a time may use it. */
hg_status hg_decode_attention(const hg_cache *cache, int32_t layer_begin, int32_t layer_count,
                              const void *q, void *out, float softmax_scale,
                              void *workspace, size_t workspace_bytes, hg_stream_t stream);

/* One decode step in one launch: append the step's K/V (as hg_append_kv; text,
 * BF16, Sec. 3) and run grouped-query decode attention over every token
 * including the new one (as hg_decode_attention, Sec. 3 / Sec. 4).  k_new / v_new: device BF16
 * [layer_count][batch][num_kv_heads][128]; the other arguments as for
 * hg_decode_attention.  The work item that holds the new position reads it
 * from k_new / v_new and also stores it into the cache.  Returns
 * HG_ERR_CAPACITY if a layer already holds max_new_tokens appended tokens;
 * advances the host-side count on success. */
hg_status hg_decode_step(hg_cache *cache, int32_t layer_begin, int32_t layer_count, const void *q,
                         const void *k_new, const void *v_new, void *out, float softmax_scale,
                         void *workspace, size_t workspace_bytes, hg_stream_t stream);

/* Decode attention that allocates nothing: the same computation and arguments
 * as hg_decode_attention, minus the workspace.  For callers that may not
 * allocate device memory themselves -- an operator inside an inference
 * runtime whose plugin interface hands over only inputs and outputs, code
 * running while another framework owns the whole device memory pool, or a
 * decode loop that cannot afford cudaMalloc's implicit device
 * synchronisation.  (This entry point has no counterpart in the paper.)
 *   Scratch   the split-K workspace is one static device array of 32 MiB
 *             inside this library; every GPU that loads the library holds it
 *             until the process exits.  A launch whose workspace
 *             (hg_decode_workspace_size) exceeds 32 MiB is rejected with
 *             HG_ERR_WORKSPACE_TOO_SMALL before anything is enqueued.
 *   Set-up    the first call on a device (with that device current) looks up
 *             the array's device address with cudaGetSymbolAddress; make that
 *             first call before any stream capture.
 *   Sharing   every call uses the same array and clears its split counters
 *             (cudaMemsetAsync) before launching; calls that overlap on the
 *             GPU (different streams, or threads on the same device) race.
 *   Errors    the argument checks and the size limit run before anything is
 *             enqueued.  A bounded wait that runs out (see Errors above) sets
 *             the array's status word, which later calls leave set: read it
 *             with hg_workspace_status(NULL, &status, stream) and reset it
 *             with hg_workspace_clear(NULL, 0, stream); a non-zero word means
 *             the outputs of the calls since the last reset are undefined.
 * No cudaMalloc, cudaFree or other allocating routine is called. */
hg_status hg_decode_attention_noalloc(const hg_cache *cache, int32_t layer_begin,
                                      int32_t layer_count, const void *q, void *out,
                                      float softmax_scale, hg_stream_t stream);

/* Sec. 5.4 storage accounting of the arena's image-token regions: bits per
 * image K/V element actually stored (codes + 64-bit metadata + BF16 entries). */
hg_status hg_cache_image_bits_per_elem(const hg_cache *cache, double *bits);

/* Protected-head selection from per-query-head sensitivity scores (Sec. 3
 * "Selecting physical KV heads", Eq. 2): the query-head scores of each GQA
 * group (query head qh belongs to KV head qh / G, G = num_q_heads /
 * num_kv_heads) are averaged into per-KV-head scores g_i and o_i; each is
 * standardised over all num_layers * num_kv_heads KV heads, z(x) = (x - mean)
 * / std (population std; a constant score gives z = 0); s_i = z(g_i) + z(o_i);
 * the k heads with the largest s are protected, ties to the lower index i =
 * layer * num_kv_heads + head.  g_scores, o_scores: host float
 * [num_layers][num_q_heads], finite; k < 0 selects round(N_KV / 8); k is
 * clamped to [0, N_KV].  mask_out: host uint8 [num_layers][num_kv_heads], 1 =
 * protected (the head_mask of hg_cache_layout).  Arithmetic in binary64 on
 * the host; no device work.  HG_ERR_INVALID_ARG on a null pointer,
 * non-positive sizes, num_q_heads not a multiple of num_kv_heads, or a
 * non-finite score. */
hg_status hg_select_heads(const float *g_scores, const float *o_scores, int32_t num_layers,
                          int32_t num_q_heads, int32_t num_kv_heads, int32_t k, uint8_t *mask_out);

/* Static description of a status code (no counterpart in the paper). */
const char *hg_status_string(hg_status status);

#ifdef __cplusplus
}
#endif

#endif /* HEADGUARD_H */
