/*
 * witcert.h -- C ABI of the WitCert metered-KV-cache library for GB300
 * (sm_103a).  Paper: "WitCert: Sound Runtime Risk Observability and Gating
 * for KV-Cache Quantization", arxiv 2607.28699.
 *
 * The library implements the meter loop of §6 (box "The meter loop"): a
 * write path that quantizes post-RoPE keys/values and stores a per-token
 * band-norm residual witness, a fused decode-attention read path that also
 * computes the per-(layer, head, step) total-variation meter, and a gate.
 *
 * Conventions shared by every entry point
 *  - All tensor arguments are DEVICE pointers owned by the caller; the
 *    library allocates no memory and never synchronises the host with the
 *    device (kernels are enqueued on the caller's stream).  The only
 *    exception is wc_read_status, which synchronises the given stream.
 *  - Arguments are validated on the host before any launch.  On failure the
 *    call returns a non-zero wc_status, launches nothing and leaves a message
 *    for wc_last_error() (thread-local).
 *  - Faults that only the device can see (a page index outside the pool, a
 *    slot outside the pool, an asynchronous copy that did not complete within
 *    its bounded wait) are never trapped: the offending token or page is
 *    skipped and a bit is OR-ed into a caller-visible 32-bit status word.
 *  - All tensors are dense, row-major, 16-byte aligned (the decode kernel
 *    stages pages with bulk asynchronous copies).
 *  - head_dim = 128, page_size = 16, num_bands = 8 and 1 <= G <= 8 query heads
 *    per KV head are the supported shapes (the paper's 7B-class shapes).
 *
 * Paged cache layout for ONE layer (PagedAttention-style token slots; a
 * slot is page * 16 + offset; §6.2.3 "Storage side"):
 *   k_codes, v_codes [num_pages][Hkv][16][128]  int8 (WC_SCHEME_DITHER_INT8)
 *                                               or fp8 e4m3fn bytes (WC_SCHEME_FP8_E4M3)
 *   k_scale, v_scale [num_pages][Hkv][16]       fp16, dither scheme only (else NULL)
 *   k_witness        [num_pages][Hkv][16][8]    fp16, per-band residual norms
 *   v_witness        [num_pages][Hkv][16][2]    fp16 (||v^ - v||, ||v||) rounded up;
 *                                               optional, for the value side only
 * The grouped scheme (WC_SCHEME_DITHER_INT8_G32) instead holds
 *   k_scale, v_scale [num_pages][Hkv][16][4]    fp16, one per 32-channel group
 *   k_bypass         [num_pages][Hkv][16][2m]   fp16 exact values of the bypassed
 *                                               pairs, pair by pair (dims a, b)
 * and stores each row's 128 codes in a permuted channel order, with the
 * dither drawn by storage position (byte i of the Philox call for channel
 * group n serves storage position 16 n + i); storage position p holds channel
 *   K:  16 ((p >> 2) & 7) + 4 (p >> 5) + (p & 3)
 *   V:  16 ((p >> 1) & 7) + 8 (p & 1) + (p >> 4)
 * (a bypassed key channel holds code 0).  The bypass pairs of a layer,
 * bypass_pairs [Hkv][m] int32 in [0, 64), are RoPE pair indices: pair j is
 * dims (j, j + 64) for WC_ROPE_HALF and (2j, 2j + 1) for WC_ROPE_INTERLEAVED.
 */
#ifndef WITCERT_H
#define WITCERT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int wc_status;
enum {
    WC_OK = 0,
    WC_ERR_INVALID_ARG = 1,   /* null pointer, bad size or misaligned tensor      */
    WC_ERR_UNSUPPORTED = 2,   /* a shape or option this build does not implement  */
    WC_ERR_CUDA = 3,          /* a CUDA runtime call failed (message has details) */
    WC_ERR_WORKSPACE = 4,     /* workspace smaller than wc_workspace_size()       */
    WC_ERR_DEVICE_CHECK = 5   /* wc_read_status found device-side fault bits      */
};

/* Device status bits (wc_read_status, or the word a write call points to). */
enum {
    WC_DEV_BAD_SLOT = 1u,     /* write: slot >= num_pages * 16; token skipped    */
    WC_DEV_BAD_PAGE = 2u,     /* decode: block-table page outside [0, num_pages)  */
    WC_DEV_BAD_CTX = 4u,      /* decode: context length < 0 or > max_pages * 16   */
    WC_DEV_TIMEOUT = 8u,      /* decode: a bounded wait for staged data gave up   */
    WC_DEV_BAD_PAIR = 16u,    /* grouped scheme: a bypass pair outside [0, 64), or listed
                                 again, is ignored (its two stored values are 0) */
    WC_DEV_BAD_APPEND = 32u   /* append: slot_new[b] is not the slot of the context's last
                                 token; the token is not written */
};

typedef enum {
    /* Controlled quantizer of §4.2 ("Subtractive dither"): per token and KV
     * head, s = fp16_rn(fp32(amax) / 126.5f), code = round-half-even of the
     * exact x/s + xi clamped to [-127, 127], reconstruction s * (code - xi). */
    WC_SCHEME_DITHER_INT8 = 0,
    /* Black-box raw cast to fp8 e4m3fn (round to nearest even, saturating
     * finite overflow to +-448), no scale, no dither (§4.1, Fig. f5). */
    WC_SCHEME_FP8_E4M3 = 1,
    /* Subtractive-dither INT8 with one fp16 scale per token and 32-channel
     * group and a fixed per-(layer, KV head) set of m key RoPE pairs stored
     * exactly ("outlier bypass", left out of the group amax); §6.2.3, §6.2.5.  8-bit
     * dither only; written and read by the _g32 entry points. */
    WC_SCHEME_DITHER_INT8_G32 = 2
} wc_scheme;

typedef enum {
    /* RoPE frequency pair j occupies dims (j, j + 64) (half rotation). */
    WC_ROPE_HALF = 0,
    /* RoPE frequency pair j occupies dims (2j, 2j + 1) (interleaved). */
    WC_ROPE_INTERLEAVED = 1
} wc_rope_layout;

/* Static description of one model's paged cache. */
typedef struct {
    int32_t head_dim;       /* must be 128                                        */
    int32_t num_q_heads;    /* Hq; Hq % Hkv == 0 and Hq / Hkv <= 8                 */
    int32_t num_kv_heads;   /* Hkv, 1 .. 65535                                     */
    int32_t num_bands;      /* B, must be 8: 64 RoPE pairs in 8 contiguous bands   */
    int32_t page_size;      /* must be 16                                          */
    int32_t num_pages;      /* pages in each layer's pool                          */
    int32_t scheme;         /* wc_scheme                                           */
    int32_t rope_layout;    /* wc_rope_layout                                      */
    int32_t dither_bits;    /* 8 or 10 (dither scheme): resolution of xi           */
    int32_t reserved;       /* must be 0                                           */
    uint64_t seed;          /* Philox key (lo, hi 32 bits)                         */
} wc_cache_desc;

/*
 * Write path ("write kernel", §6.2.1; witness Eq. (witness), §4.1).
 *
 * For each token t < n_tok and KV head h, quantizes the post-RoPE fp16 rows
 * k[t][h][:] and v[t][h][:] with desc->scheme, writes the codes (and fp16
 * scales for the dither scheme) to slot slot_mapping[t] of this layer's
 * cache, and stores the K witness w_b = fp16_round_up(||k^_b - k_b||) for
 * the 8 RoPE bands.  The dither xi is Philox4x32-10 under key
 * (seed lo, seed hi) at counter (slot, layer * 65536 + h, group, tag), tag 0
 * for K and 1 for V; with dither_bits = 8 one counter covers 16 channels
 * (channel i of group g is byte i % 4 of word i / 4), with 10 it covers 8
 * (bits 16 * (i % 2) .. +9 of word i / 2); integer j maps to
 * xi = (j + 1/2) / 2^bits - 1/2.  The witness may exceed the exactly rounded
 * norm by one fp16 ulp (it is computed in fp32 and rounded up with margin),
 * never fall below it.
 *
 *   layer          0 .. 65535, keys the dither
 *   k, v           [n_tok][Hkv][128] fp16, device
 *   slot_mapping   [n_tok] int32, device; a negative slot skips the token,
 *                  a slot >= num_pages * 16 skips it and sets WC_DEV_BAD_SLOT
 *   k_scale,v_scale NULL for WC_SCHEME_FP8_E4M3
 *   dev_status     optional device uint32 that collects WC_DEV_* bits (OR)
 * Rows written by the same call must have distinct slots.
 */
wc_status wc_kv_quantize_witness(const wc_cache_desc* desc, int32_t layer,
                                 const void* k, const void* v,
                                 const int32_t* slot_mapping, int32_t n_tok,
                                 void* k_codes, void* v_codes,
                                 void* k_scale, void* v_scale, void* k_witness,
                                 uint32_t* dev_status, void* stream);

/*
 * wc_kv_quantize_witness that also stores the value witness of every written
 * V row (§3 output bound, §4.2 "Value side"): v_witness[slot] =
 * (||v^ - v||, ||v||), each rounded up to fp16 (never below the exact norm,
 * at most one fp16 step above).  v_witness 16-byte aligned, not NULL.
 */
wc_status wc_kv_quantize_witness_v(const wc_cache_desc* desc, int32_t layer,
                                   const void* k, const void* v,
                                   const int32_t* slot_mapping, int32_t n_tok,
                                   void* k_codes, void* v_codes,
                                   void* k_scale, void* v_scale, void* k_witness,
                                   void* v_witness, uint32_t* dev_status, void* stream);

/*
 * Bytes of workspace wc_metered_decode_attention needs for `batch`
 * sequences whose block tables hold `max_pages` pages, on the current
 * device (the split count depends on its SM count).  Returns 0 and sets
 * wc_last_error() on invalid arguments.  The workspace must be zero-filled
 * once after allocation; each call leaves it ready for the next one.
 */
size_t wc_workspace_size(const wc_cache_desc* desc, int32_t batch, int32_t max_pages);

/*
 * Metered decode attention (read path, §6.2.1-§6.2.2; Thm. "Sound black-box
 * logit bound"; Thm. "Sound replacement").
 *
 * For every sequence b and query head hq (KV head hq / G) over the
 * ctx_lens[b] cached tokens of this layer:
 *   out[b][hq][:]   = sum_t p~_t v^_t, p~ = softmax_t(q . k^_t / sqrt(128))
 *   c_t             = (1/sqrt(128)) sum_b ||q_b|| w_{t,b}
 *   meter_raw[b][hq] = 1/2 (A^2 - 1), A = sum_t p~_t e^{c_t}  (+inf on fp32 overflow)
 *   meter[b][hq]    = min(1, meter_raw)
 * meter_raw carries an upward margin sized to cover its fp32 evaluation
 * (checked on or above the fp64 value); a term or sum that overflows fp32
 * makes it +inf (never NaN), including a token whose softmax weight
 * underflows fp32 while its bound is huge.
 * The context is split across CTAs (one sequence: every KV head's pages in
 * equal splits; several sequences, whose lengths only the device sees: each
 * CTA serves one KV head and an equal share of the batch's pages laid end to
 * end, cut at sequence boundaries); partial softmax, output and A
 * accumulators are merged under log-sum-exp weights (A is a p~-weighted mean,
 * §6.2.2) by a second kernel, launched as a programmatic dependent of the
 * first (two launches per call).  A sequence with
 * ctx_len 0 gets out = 0 and meter = meter_raw = 0.
 *
 *   q            [batch][Hq][128] fp16 post-RoPE queries, device
 *   block_table  [batch][max_pages] int32 physical page of each logical page
 *   ctx_lens     [batch] int32, 0 .. max_pages * 16
 *   out          [batch][Hq][128] fp32; meter, meter_raw [batch][Hq] fp32
 *   workspace    >= wc_workspace_size(desc, batch, max_pages) bytes, zeroed
 *                once; holds the device status word (wc_read_status)
 * Calls sharing one workspace must be ordered on one stream.
 */
wc_status wc_metered_decode_attention(const wc_cache_desc* desc, int32_t layer,
                                      const void* q, const int32_t* block_table,
                                      int32_t max_pages, const int32_t* ctx_lens,
                                      int32_t batch,
                                      const void* k_codes, const void* v_codes,
                                      const void* k_scale, const void* v_scale,
                                      const void* k_witness,
                                      float* out, float* meter, float* meter_raw,
                                      void* workspace, size_t workspace_bytes,
                                      void* stream);

/*
 * Metered decode attention with the Tier-B sub-Gaussian certificate as well
 * (§4.2, Lemma "Uniform sub-Gaussian proxy"; dithered INT8 cache only).
 *
 * Same computation, arguments and outputs as wc_metered_decode_attention,
 * plus, for every sequence b and query head hq over its S = ctx_lens[b]
 * tokens:
 *   u_t             = sqrt(2 varsigma_t^2 log(2 S / delta_loc)),
 *   varsigma_t^2    = ||q||^2 s_t^2 / (12 * 128)   (s_t the stored fp16 K scale),
 *   meter_b_raw     = 1/2 (A_B^2 - 1), A_B = sum_t p~_t e^{u_t}  (+inf on overflow),
 *   meter_b         = min(1, meter_b_raw).
 * With probability at least 1 - delta_loc over the dither, |eps_t| <= u_t for
 * all S tokens and then TV <= meter_b_raw; the guarantee assumes queries that
 * do not depend on the stored dither (non-adaptive, §4.2 "Scope").  The
 * request-level budget delta_loc = delta_req / (L * H * T) is the caller's.
 *   delta_loc            in (0, 1), else WC_ERR_INVALID_ARG
 *   meter_b, meter_b_raw [batch][Hq] fp32, device
 * Returns WC_ERR_UNSUPPORTED for the fp8 scheme (no controlled quantizer).
 */
wc_status wc_metered_decode_attention_tier_b(const wc_cache_desc* desc, int32_t layer,
                                             const void* q, const int32_t* block_table,
                                             int32_t max_pages, const int32_t* ctx_lens,
                                             int32_t batch,
                                             const void* k_codes, const void* v_codes,
                                             const void* k_scale, const void* v_scale,
                                             const void* k_witness, double delta_loc,
                                             float* out, float* meter, float* meter_raw,
                                             float* meter_b, float* meter_b_raw,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream);

/*
 * Metered decode attention with the value-side terms and the output bound
 * (§3: ||y - y^|| <= 2 TV max_t ||v_t|| + sum_t p~_t rho^v_t; §4.2 "Value side
 * and the joint event").  Same computation, arguments and outputs as
 * wc_metered_decode_attention, plus for every sequence b and query head hq:
 *   value_term[b][hq] = sum_t p~_t rho^v_t          (rho^v from v_witness)
 *   v_max[b][hq]      = max_t ||v_t||                (over the KV head's tokens)
 *   out_bound[b][hq]  = 2 * meter[b][hq] * v_max + value_term   (bounds ||y - y^||)
 * The value term is deterministic given p~: it needs no probability budget.
 *   v_witness  as written by wc_kv_quantize_witness_v, 16-byte aligned
 *   value_term, v_max, out_bound [batch][Hq] fp32, device, not NULL
 */
wc_status wc_metered_decode_attention_v(const wc_cache_desc* desc, int32_t layer,
                                        const void* q, const int32_t* block_table,
                                        int32_t max_pages, const int32_t* ctx_lens,
                                        int32_t batch,
                                        const void* k_codes, const void* v_codes,
                                        const void* k_scale, const void* v_scale,
                                        const void* k_witness, const void* v_witness,
                                        float* out, float* meter, float* meter_raw,
                                        float* value_term, float* v_max, float* out_bound,
                                        void* workspace, size_t workspace_bytes,
                                        void* stream);

/*
 * Allocation-free metered decode.  The paper has no counterpart: this is a
 * deployment convenience for callers that cannot allocate device memory at
 * decode time (a runtime that pre-plans every buffer, code running inside an
 * allocator's own hooks, a process under a fixed memory budget) and so cannot
 * provide the workspace wc_metered_decode_attention needs.
 *
 * Same computation, arguments and outputs as wc_metered_decode_attention,
 * without the workspace.  Its scratch is one fixed 16 MiB device array built
 * into the library; every GPU that loads the library keeps it until the
 * process exits.  The call never allocates or frees memory.
 *   dev_status  device uint32 that collects the WC_DEV_* bits (OR), required
 *               (not NULL: the built-in scratch has no word a caller can read);
 *               read and clear it with wc_read_status(dev_status, 1, ...).
 * Returns WC_ERR_UNSUPPORTED, launching nothing, when the decode would need
 * more scratch than 16 MiB (about 3700 partial results: one per (KV head,
 * split) for one sequence; for several sequences the SM count (8 per SM's two
 * CTAs for fp8 and the 10-bit dither) plus batch x Hkv; the count follows
 * wc_workspace_size's plan).
 * The first call on each device, and the first after its context has been
 * recreated (cudaDeviceReset), looks up the scratch address
 * (cudaGetSymbolAddress); make that first call before any stream capture.
 * All calls share the one scratch array and it keeps the last call's
 * contents: calls that can overlap on the GPU (different streams, or several
 * host threads) race and must be ordered by the caller.
 */
wc_status wc_metered_decode_attention_noalloc(const wc_cache_desc* desc, int32_t layer,
                                              const void* q, const int32_t* block_table,
                                              int32_t max_pages, const int32_t* ctx_lens,
                                              int32_t batch,
                                              const void* k_codes, const void* v_codes,
                                              const void* k_scale, const void* v_scale,
                                              const void* k_witness,
                                              float* out, float* meter, float* meter_raw,
                                              uint32_t* dev_status, void* stream);

/*
 * One decode step with the write of its new token fused in: the effect of
 * wc_kv_quantize_witness for the tokens k_new[b], v_new[b] at slots
 * slot_new[b] (codes, scales, K witness; no value witness), followed by
 * wc_metered_decode_attention, in one pair of launches.  The new token of
 * sequence b is the last of its context: slot_new[b] must be the slot of
 * logical position ctx_lens[b] - 1 (block_table[b][(ctx - 1) / 16] * 16 +
 * (ctx - 1) % 16); otherwise it is not written and WC_DEV_BAD_APPEND is set.
 * slot_new[b] < 0: no new token for sequence b.  The token is quantized by
 * the CTA that reads the sequence's last page, before it reads it; that page
 * must belong to sequence b alone (no other sequence of the call may map it,
 * as with prefix sharing), since only that CTA is ordered after the write.
 *   k_new, v_new  [batch][Hkv][128] fp16 post-RoPE, device, 16-byte aligned
 *   slot_new      [batch] int32, device
 * The cache arrays are written, hence not const.  WC_ERR_UNSUPPORTED for any
 * scheme but WC_SCHEME_DITHER_INT8 with dither_bits 8 (write, then decode).
 */
wc_status wc_metered_decode_attention_append(const wc_cache_desc* desc, int32_t layer,
                                             const void* q, const int32_t* block_table,
                                             int32_t max_pages, const int32_t* ctx_lens,
                                             int32_t batch,
                                             void* k_codes, void* v_codes,
                                             void* k_scale, void* v_scale, void* k_witness,
                                             const void* k_new, const void* v_new,
                                             const int32_t* slot_new,
                                             float* out, float* meter, float* meter_raw,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream);

/*
 * Metered decode attention with the per-page terms of block-level repair
 * selection (§6.3.5 "Block-level paging").  Same computation, arguments and
 * outputs as wc_metered_decode_attention, plus for every sequence b, query
 * head hq and logical page j < ceil(ctx_lens[b] / 16):
 *   page_terms[b][hq][j]  = (m_j, d_j) fp32: page j's share of D = A - 1,
 *                           d_j = sum_{t in j} 2^(y_t - m_j) (e^{c_t} - 1), summed
 *                           against a reference m_j (y_t the logit in log2 units)
 *   softmax_norm[b][hq]   = (M, L) fp32 with p~_t = 2^(y_t - M) / L
 * so that page j contributes C_j = d_j 2^(m_j - M) / L to D.  Entries of
 * pages at or past the context are not written; a page outside the pool (see
 * WC_DEV_BAD_PAGE) gets (-inf, 0).  The outputs feed wc_repair_select.
 *   page_terms    [batch][Hq][max_pages][2] fp32, device, 8-byte aligned
 *   softmax_norm  [batch][Hq][2] fp32, device, 8-byte aligned
 */
wc_status wc_metered_decode_attention_repair(const wc_cache_desc* desc, int32_t layer,
                                             const void* q, const int32_t* block_table,
                                             int32_t max_pages, const int32_t* ctx_lens,
                                             int32_t batch,
                                             const void* k_codes, const void* v_codes,
                                             const void* k_scale, const void* v_scale,
                                             const void* k_witness,
                                             float* out, float* meter, float* meter_raw,
                                             float* page_terms, float* softmax_norm,
                                             void* workspace, size_t workspace_bytes,
                                             void* stream);

/*
 * Block-level repair selection (§6.3.5 "Block-level paging").  With p~ held
 * fixed, paging in the exact keys of logical page j (witness 0) lowers D by
 * exactly C_j, so the fewest pages that bring the meter to tau are the
 * largest contributions.  For every cell (b, hq), with n = ceil(ctx_lens[b]/16):
 *   contrib[b][hq][j]    = C_j, j < n (fp32; optional, NULL: not stored)
 *   repair_pages[b][hq][0 .. k-1] = logical pages by decreasing C_j (ties to the
 *                          lower page; a NaN contribution ranks first), where k
 *                          is the least count with 1/2 R_k (R_k + 2) <= tau in fp32,
 *                          R_k = the sum of the contributions not in the list;
 *                          k = n when no count is enough (tau < 0 or NaN)
 *   n_repair[b][hq]      = k;  d_after[b][hq] = R_k
 * Cells of several layers can be selected in one call by stacking them along
 * batch (the layouts are contiguous over [layer][batch]; ctx_lens then holds
 * one entry per stacked row).  Cells with keep_q[cell] != 0 (the gate kept
 * them) get k = 0 and d_after = D.  keep_q may be NULL: every cell is selected.  Entries of
 * repair_pages past k are not written.  One CTA per cell; the sort holds
 * max_pages 8-byte keys in shared memory, so max_pages <= 16384
 * (WC_ERR_UNSUPPORTED above).
 *   page_terms, softmax_norm  as written by wc_metered_decode_attention_repair
 *   ctx_lens     [batch] int32 (as for the decode); keep_q [batch][Hq] uint8 or NULL
 *   contrib      [batch][Hq][max_pages] fp32 or NULL; repair_pages [batch][Hq][max_pages]
 *                int32; n_repair [batch][Hq] int32; d_after [batch][Hq] fp32 -- device
 *   dev_status   optional device uint32 that collects WC_DEV_BAD_CTX (OR)
 */
wc_status wc_repair_select(const float* page_terms, const float* softmax_norm,
                           const int32_t* ctx_lens, int32_t batch, int32_t num_q_heads,
                           int32_t max_pages, const uint8_t* keep_q, float tau,
                           float* contrib, int32_t* repair_pages, int32_t* n_repair,
                           float* d_after, uint32_t* dev_status, void* stream);

/*
 * Write path of the grouped scheme (§6.2.3 "Storage side", §6.2.5 "Fixed-channel
 * outlier bypass"): as wc_kv_quantize_witness, with for each row and group g
 * of 32 channels s_g = fp16_rn(fp32(amax_g) / 126.5f), amax_g over the
 * group's channels that are not bypassed (a key row's bypassed channels, the
 * 2m dims of bypass_pairs[h], are stored exactly in k_bypass with code 0;
 * value rows have no bypass).  The K witness covers the residual of every
 * channel (0 on the bypassed ones).
 *   desc->scheme    WC_SCHEME_DITHER_INT8_G32 with dither_bits 8
 *   k_scale, v_scale, k_bypass, bypass_pairs  as in the layout above
 *   num_bypass_pairs  m in [0, 16]; k_bypass and bypass_pairs may be NULL if 0.
 *                   The pairs of a head should be distinct: an index outside [0, 64)
 *                   or repeated is ignored (its entries store 0, WC_DEV_BAD_PAIR).
 *   dev_status      optional device uint32: WC_DEV_BAD_SLOT, WC_DEV_BAD_PAIR
 */
wc_status wc_kv_quantize_witness_g32(const wc_cache_desc* desc, int32_t layer, const void* k,
                                     const void* v, const int32_t* slot_mapping, int32_t n_tok,
                                     void* k_codes, void* v_codes, void* k_scale, void* v_scale,
                                     void* k_witness, void* k_bypass, const int32_t* bypass_pairs,
                                     int32_t num_bypass_pairs, uint32_t* dev_status, void* stream);

/*
 * Metered decode attention over a grouped-scheme cache: the same outputs as
 * wc_metered_decode_attention, from k^_c = s_{g(c)} (code_c - xi_c) (exact
 * fp16 values on the bypassed key channels) and v^ likewise.  With meter_b
 * and meter_b_raw not NULL also the Tier-B meter (§4.2) with the grouped proxy
 *   varsigma_t^2 = (1 / (12 * 128)) sum_{c not bypassed} q_c^2 s_{g(c),t}^2
 * (delta_loc in (0, 1)); both NULL: not computed.
 */
wc_status wc_metered_decode_attention_g32(const wc_cache_desc* desc, int32_t layer,
                                          const void* q, const int32_t* block_table,
                                          int32_t max_pages, const int32_t* ctx_lens,
                                          int32_t batch,
                                          const void* k_codes, const void* v_codes,
                                          const void* k_scale, const void* v_scale,
                                          const void* k_witness, const void* k_bypass,
                                          const int32_t* bypass_pairs, int32_t num_bypass_pairs,
                                          double delta_loc,
                                          float* out, float* meter, float* meter_raw,
                                          float* meter_b, float* meter_b_raw,
                                          void* workspace, size_t workspace_bytes, void* stream);

/*
 * Bypass-pair calibration (§6.2.5 "Fixed-channel outlier bypass": the
 * massive-activation RoPE pairs are stable across tokens, so a fixed set per
 * (layer, KV head) chosen from a prefix suffices).  For each KV head h,
 * pairs[h][0 .. m-1] = the m RoPE pairs of largest energy
 * sum_t (k[t][h][a]^2 + k[t][h][b]^2) over the n_tok rows (fp32 sums; ties to
 * the lower pair), in increasing pair order.
 *   k      [n_tok][Hkv][128] fp16 post-RoPE keys, device, 16-byte aligned
 *   m      in [0, 16]; pairs [Hkv][m] int32, device
 */
wc_status wc_select_bypass_pairs(const void* k, int32_t n_tok, int32_t num_kv_heads,
                                 int32_t rope_layout, int32_t m, int32_t* pairs, void* stream);

/*
 * Gate (§6 meter-loop box; certified tau < 1 vs risk-ranked tau >= 1, §4.3).
 *
 * keep_q[i] = (meter_raw[i] <= tau) in fp32 (equality keeps the compressed
 * path; +inf and NaN fall back).  Cells come in groups of `group`
 * consecutive query heads sharing one KV head; keep_kv[i / group] = AND of
 * its group (any-of-G fallback).  n_kept[0] = kept query-head cells,
 * n_kept[1] = kept KV-head cells.  One CTA; no atomics; n_kept need not be
 * zeroed.
 *   meter_raw [n_cells] fp32; keep_q [n_cells] uint8; keep_kv [n_cells/group]
 *   uint8; n_kept [2] int32 -- all device.
 */
wc_status wc_gate(const float* meter_raw, int32_t n_cells, int32_t group, float tau,
                  uint8_t* keep_q, uint8_t* keep_kv, int32_t* n_kept, void* stream);

/*
 * Joint gate (§4.2 "Value side and the joint event"): pass_K and pass_V.
 * keep_q[i] = (meter_raw[i] <= tau_k) && (value_term[i] <= tau_v * v_max[i]),
 * all in fp32 (the product rounded once); otherwise as wc_gate.  Reading:
 * the paper names pass_V without a formula; here it bounds the value term
 * relative to the largest value norm.
 *   value_term, v_max [n_cells] fp32, device (from wc_metered_decode_attention_v)
 */
wc_status wc_gate_joint(const float* meter_raw, const float* value_term, const float* v_max,
                        int32_t n_cells, int32_t group, float tau_k, float tau_v,
                        uint8_t* keep_q, uint8_t* keep_kv, int32_t* n_kept, void* stream);

/*
 * Synchronises `stream`, copies the device status word held in `workspace`
 * (or pointed to by a write call's dev_status, when `is_status_word` != 0)
 * to *bits, clears it on the device, and returns WC_ERR_DEVICE_CHECK if
 * any bit was set.  Diagnostic only: the other calls never synchronise.
 */
wc_status wc_read_status(void* workspace_or_word, int32_t is_status_word,
                         uint32_t* bits, void* stream);

/*
 * Failure-detection test support (no counterpart in the paper; the library's
 * own test of its bounded waits).  Runs wc_metered_decode_attention for one
 * sequence (batch 1, dithered INT8 cache with the 8-bit dither) except that
 * the copies of logical page `stall_page` are never issued: the consumer that
 * waits for that page, and then its producer, give up after a short bounded
 * wait (64 tries of mbarrier.try_wait), set WC_DEV_TIMEOUT in the workspace's
 * status word and finish; copies already issued are waited for before the
 * kernel exits.  Nothing faults or hangs, and the context stays usable: read
 * the bits with wc_read_status.  The outputs of the call are not meaningful.
 *   stall_page  in [0, max_pages), else WC_ERR_INVALID_ARG
 * Other arguments as wc_metered_decode_attention (ctx_lens holds one length).
 */
wc_status wc_testing_decode_stalled_page(const wc_cache_desc* desc, int32_t layer,
                                         const void* q, const int32_t* block_table,
                                         int32_t max_pages, const int32_t* ctx_lens,
                                         const void* k_codes, const void* v_codes,
                                         const void* k_scale, const void* v_scale,
                                         const void* k_witness,
                                         float* out, float* meter, float* meter_raw,
                                         void* workspace, size_t workspace_bytes,
                                         int32_t stall_page, void* stream);

/* Thread-local description of the last non-OK status on this thread. */
const char* wc_last_error(void);

/* Library version, (major << 16) | minor. */
int32_t wc_version(void);

#ifdef __cplusplus
}
#endif

#endif /* WITCERT_H */
