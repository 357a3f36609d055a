// extern "C" boundary: host-side argument checks and kernel launches.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include "wc_kernels.cuh"

namespace {

thread_local std::string g_last_error;

wc_status fail(wc_status st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
wc_status fail(wc_status st, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

wc_status cuda_fail(cudaError_t e, const char* what) {
    return fail(WC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// allow_grouped: the grouped scheme is accepted only by its own (_g32) entry
// points and the workspace query; every other entry point rejects it.
wc_status check_desc(const wc_cache_desc* d, bool allow_grouped = false) {
    if (!d) return fail(WC_ERR_INVALID_ARG, "desc is NULL");
    if (d->head_dim != wc::kHeadDim) return fail(WC_ERR_UNSUPPORTED, "head_dim must be 128 (got %d)", d->head_dim);
    if (d->page_size != wc::kPage) return fail(WC_ERR_UNSUPPORTED, "page_size must be 16 (got %d)", d->page_size);
    if (d->num_bands != wc::kBands) return fail(WC_ERR_UNSUPPORTED, "num_bands must be 8 (got %d)", d->num_bands);
    if (d->num_kv_heads < 1 || d->num_kv_heads > 65535)
        return fail(WC_ERR_INVALID_ARG, "num_kv_heads must be in [1, 65535] (got %d)", d->num_kv_heads);
    if (d->num_q_heads < 1 || d->num_q_heads % d->num_kv_heads != 0)
        return fail(WC_ERR_INVALID_ARG, "num_q_heads (%d) must be a positive multiple of num_kv_heads (%d)",
                    d->num_q_heads, d->num_kv_heads);
    if (d->num_q_heads / d->num_kv_heads > wc::kMaxGroup)
        return fail(WC_ERR_UNSUPPORTED, "at most %d query heads per KV head (got %d)", wc::kMaxGroup,
                    d->num_q_heads / d->num_kv_heads);
    if (d->num_pages < 1) return fail(WC_ERR_INVALID_ARG, "num_pages must be positive (got %d)", d->num_pages);
    if ((long long)d->num_pages * wc::kPage > 0x7FFFFFFFLL)
        return fail(WC_ERR_UNSUPPORTED, "num_pages * 16 must fit in int32");
    if (d->scheme == WC_SCHEME_DITHER_INT8_G32) {
        if (!allow_grouped)
            return fail(WC_ERR_UNSUPPORTED, "the grouped scheme is written and read by the _g32 entry points");
        if (d->dither_bits != 8) return fail(WC_ERR_UNSUPPORTED, "the grouped scheme uses the 8-bit dither");
    } else if (d->scheme != WC_SCHEME_DITHER_INT8 && d->scheme != WC_SCHEME_FP8_E4M3) {
        return fail(WC_ERR_UNSUPPORTED, "unknown scheme %d", d->scheme);
    }
    if (d->rope_layout != WC_ROPE_HALF && d->rope_layout != WC_ROPE_INTERLEAVED)
        return fail(WC_ERR_UNSUPPORTED, "unknown rope_layout %d", d->rope_layout);
    if (d->scheme == WC_SCHEME_DITHER_INT8 && d->dither_bits != 8 && d->dither_bits != 10)
        return fail(WC_ERR_UNSUPPORTED, "dither_bits must be 8 or 10 (got %d)", d->dither_bits);
    if (d->reserved != 0) return fail(WC_ERR_INVALID_ARG, "reserved must be 0");
    return WC_OK;
}

wc_status check_cache(const wc_cache_desc* d, const void* kc, const void* vc, const void* ks, const void* vs,
                      const void* kw) {
    if (!kc || !vc || !kw) return fail(WC_ERR_INVALID_ARG, "cache pointers must not be NULL");
    if (!aligned16(kc) || !aligned16(vc) || !aligned16(kw))
        return fail(WC_ERR_INVALID_ARG, "cache arrays must be 16-byte aligned");
    if (d->scheme == WC_SCHEME_DITHER_INT8 || d->scheme == WC_SCHEME_DITHER_INT8_G32) {
        if (!ks || !vs) return fail(WC_ERR_INVALID_ARG, "k_scale/v_scale are required by the dither scheme");
        if (!aligned16(ks) || !aligned16(vs)) return fail(WC_ERR_INVALID_ARG, "scale arrays must be 16-byte aligned");
    } else if (ks || vs) {
        return fail(WC_ERR_INVALID_ARG, "k_scale/v_scale must be NULL for the fp8 scheme");
    }
    return WC_OK;
}

int current_sm_count(int* out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -1;
    if (cudaDeviceGetAttribute(out, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
    return 0;
}

}  // namespace

extern "C" {

int32_t wc_version(void) { return (1 << 16) | 0; }

const char* wc_last_error(void) { return g_last_error.c_str(); }

// Bypass arguments of the grouped scheme: m in [0, 16]; the pair list and the
// exact-value array are required when m > 0.
static wc_status check_bypass(const void* k_bypass, const int32_t* bypass_pairs, int32_t m) {
    if (m < 0 || m > 16) return fail(WC_ERR_INVALID_ARG, "num_bypass_pairs must be in [0, 16] (got %d)", m);
    if (m > 0 && (!k_bypass || !bypass_pairs))
        return fail(WC_ERR_INVALID_ARG, "k_bypass and bypass_pairs must not be NULL when num_bypass_pairs > 0");
    if (m > 0 && !aligned16(k_bypass)) return fail(WC_ERR_INVALID_ARG, "k_bypass must be 16-byte aligned");
    return WC_OK;
}

static wc_status write_tokens(const wc_cache_desc* desc, int32_t layer, const void* k, const void* v,
                              const int32_t* slot_mapping, int32_t n_tok, void* k_codes, void* v_codes,
                              void* k_scale, void* v_scale, void* k_witness, void* v_witness,
                              uint32_t* dev_status, void* stream, bool grouped = false, void* k_bypass = nullptr,
                              const int32_t* bypass_pairs = nullptr, int32_t num_bypass = 0) {
    if (wc_status st = check_desc(desc, grouped)) return st;
    if (grouped) {
        if (desc->scheme != WC_SCHEME_DITHER_INT8_G32)
            return fail(WC_ERR_INVALID_ARG, "the _g32 entry points need desc->scheme = WC_SCHEME_DITHER_INT8_G32");
        if (wc_status st = check_bypass(k_bypass, bypass_pairs, num_bypass)) return st;
    }
    if (layer < 0 || layer > 65535) return fail(WC_ERR_INVALID_ARG, "layer must be in [0, 65535] (got %d)", layer);
    if (n_tok < 0) return fail(WC_ERR_INVALID_ARG, "n_tok must be >= 0 (got %d)", n_tok);
    if ((long long)n_tok * desc->num_kv_heads > 0x7FFFFFFFLL - 8)
        return fail(WC_ERR_UNSUPPORTED, "n_tok * num_kv_heads must fit in int32");
    if (n_tok > 0 && (!k || !v || !slot_mapping)) return fail(WC_ERR_INVALID_ARG, "k, v, slot_mapping must not be NULL");
    if (!aligned16(k) || !aligned16(v)) return fail(WC_ERR_INVALID_ARG, "k and v must be 16-byte aligned");
    if (wc_status st = check_cache(desc, k_codes, v_codes, k_scale, v_scale, k_witness)) return st;
    if (v_witness && !aligned16(v_witness)) return fail(WC_ERR_INVALID_ARG, "v_witness must be 16-byte aligned");
    if (n_tok == 0) return WC_OK;
    wc::WriteParams p;
    p.k = static_cast<const __half*>(k);
    p.v = static_cast<const __half*>(v);
    p.slot_mapping = slot_mapping;
    p.k_codes = k_codes;
    p.v_codes = v_codes;
    p.k_scale = static_cast<__half*>(k_scale);
    p.v_scale = static_cast<__half*>(v_scale);
    p.k_witness = static_cast<__half*>(k_witness);
    p.v_witness = static_cast<__half*>(v_witness);
    p.k_bypass = static_cast<__half*>(k_bypass);
    p.bypass_pairs = bypass_pairs;
    p.num_bypass = num_bypass;
    p.dev_status = dev_status;
    p.n_tok = n_tok;
    p.num_kv_heads = desc->num_kv_heads;
    p.num_pages = desc->num_pages;
    p.layer = layer;
    p.rope_layout = desc->rope_layout;
    p.keys = wc::make_philox_keys(desc->seed);
    cudaError_t e = wc::launch_write(p, desc->scheme, desc->dither_bits, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "write kernel launch");
}

wc_status wc_kv_quantize_witness(const wc_cache_desc* desc, int32_t layer, const void* k, const void* v,
                                 const int32_t* slot_mapping, int32_t n_tok, void* k_codes, void* v_codes,
                                 void* k_scale, void* v_scale, void* k_witness, uint32_t* dev_status,
                                 void* stream) {
    return write_tokens(desc, layer, k, v, slot_mapping, n_tok, k_codes, v_codes, k_scale, v_scale, k_witness,
                        nullptr, dev_status, stream);
}

wc_status wc_kv_quantize_witness_v(const wc_cache_desc* desc, int32_t layer, const void* k, const void* v,
                                   const int32_t* slot_mapping, int32_t n_tok, void* k_codes, void* v_codes,
                                   void* k_scale, void* v_scale, void* k_witness, void* v_witness,
                                   uint32_t* dev_status, void* stream) {
    if (!v_witness) return fail(WC_ERR_INVALID_ARG, "v_witness must not be NULL");
    return write_tokens(desc, layer, k, v, slot_mapping, n_tok, k_codes, v_codes, k_scale, v_scale, k_witness,
                        v_witness, dev_status, stream);
}

wc_status wc_kv_quantize_witness_g32(const wc_cache_desc* desc, int32_t layer, const void* k, const void* v,
                                     const int32_t* slot_mapping, int32_t n_tok, void* k_codes, void* v_codes,
                                     void* k_scale, void* v_scale, void* k_witness, void* k_bypass,
                                     const int32_t* bypass_pairs, int32_t num_bypass_pairs, uint32_t* dev_status,
                                     void* stream) {
    return write_tokens(desc, layer, k, v, slot_mapping, n_tok, k_codes, v_codes, k_scale, v_scale, k_witness,
                        nullptr, dev_status, stream, true, k_bypass, bypass_pairs, num_bypass_pairs);
}

wc_status wc_select_bypass_pairs(const void* k, int32_t n_tok, int32_t num_kv_heads, int32_t rope_layout, int32_t m,
                                 int32_t* pairs, void* stream) {
    if (n_tok < 0) return fail(WC_ERR_INVALID_ARG, "n_tok must be >= 0 (got %d)", n_tok);
    if (num_kv_heads < 1 || num_kv_heads > 65535)
        return fail(WC_ERR_INVALID_ARG, "num_kv_heads must be in [1, 65535] (got %d)", num_kv_heads);
    if (rope_layout != WC_ROPE_HALF && rope_layout != WC_ROPE_INTERLEAVED)
        return fail(WC_ERR_UNSUPPORTED, "unknown rope_layout %d", rope_layout);
    if (m < 0 || m > 16) return fail(WC_ERR_INVALID_ARG, "m must be in [0, 16] (got %d)", m);
    if (m == 0) return WC_OK;
    if (!pairs || (n_tok > 0 && !k)) return fail(WC_ERR_INVALID_ARG, "k and pairs must not be NULL");
    cudaError_t e = wc::launch_select_pairs(static_cast<const __half*>(k), n_tok, num_kv_heads, rope_layout, m, pairs,
                                            static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "pair selection kernel launch");
}

size_t wc_workspace_size(const wc_cache_desc* desc, int32_t batch, int32_t max_pages) {
    if (check_desc(desc, true) != WC_OK) return 0;
    if (batch < 1 || max_pages < 1) {
        fail(WC_ERR_INVALID_ARG, "batch and max_pages must be positive");
        return 0;
    }
    int sms = 0;
    if (current_sm_count(&sms) != 0) {
        fail(WC_ERR_CUDA, "no current CUDA device to size the workspace for");
        return 0;
    }
    return wc::plan_decode(batch, desc->num_kv_heads, max_pages, sms, desc->scheme, desc->dither_bits).total;
}

// Metered decode with a caller workspace; meter_b != NULL also asks for the
// Tier-B meters (dithered INT8 only).
static wc_status decode_with_workspace(const wc_cache_desc* desc, int32_t layer, const void* q,
                                       const int32_t* block_table, int32_t max_pages, const int32_t* ctx_lens,
                                       int32_t batch, const void* k_codes, const void* v_codes,
                                       const void* k_scale, const void* v_scale, const void* k_witness,
                                       float* out, float* meter, float* meter_raw, float* meter_b,
                                       float* meter_b_raw, double delta_loc, const void* v_witness,
                                       float* value_term, float* v_max, float* out_bound, float* page_terms,
                                       float* softmax_norm, void* workspace, size_t workspace_bytes,
                                       void* stream, bool grouped = false, const void* k_bypass = nullptr,
                                       const int32_t* bypass_pairs = nullptr, int32_t num_bypass = 0,
                                       const void* k_new = nullptr, const void* v_new = nullptr,
                                       const int32_t* slot_new = nullptr, int32_t stall_page = -1) {
    if (wc_status st = check_desc(desc, grouped)) return st;
    if (k_new || v_new || slot_new) {
        if (!k_new || !v_new || !slot_new)
            return fail(WC_ERR_INVALID_ARG, "k_new, v_new and slot_new must not be NULL");
        if (!aligned16(k_new) || !aligned16(v_new))
            return fail(WC_ERR_INVALID_ARG, "k_new and v_new must be 16-byte aligned");
        if (desc->scheme != WC_SCHEME_DITHER_INT8 || desc->dither_bits != 8)
            return fail(WC_ERR_UNSUPPORTED,
                        "the fused append is implemented for the dithered INT8 cache with the 8-bit dither");
        if (meter_b || value_term || page_terms)
            return fail(WC_ERR_UNSUPPORTED, "the append, Tier B, the value side and the repair terms are separate calls");
    }
    if (grouped) {
        if (desc->scheme != WC_SCHEME_DITHER_INT8_G32)
            return fail(WC_ERR_INVALID_ARG, "the _g32 entry points need desc->scheme = WC_SCHEME_DITHER_INT8_G32");
        if (wc_status st = check_bypass(k_bypass, bypass_pairs, num_bypass)) return st;
    }
    if (page_terms || softmax_norm) {
        if (!page_terms || !softmax_norm)
            return fail(WC_ERR_INVALID_ARG, "page_terms and softmax_norm must not be NULL");
        if ((reinterpret_cast<uintptr_t>(page_terms) & 7u) || (reinterpret_cast<uintptr_t>(softmax_norm) & 7u))
            return fail(WC_ERR_INVALID_ARG, "page_terms and softmax_norm must be 8-byte aligned");
        if (meter_b || value_term)
            return fail(WC_ERR_UNSUPPORTED, "the repair terms, Tier B and the value side are separate calls");
    }
    if (value_term || v_max || out_bound || v_witness) {
        if (!value_term || !v_max || !out_bound || !v_witness)
            return fail(WC_ERR_INVALID_ARG, "v_witness, value_term, v_max and out_bound must not be NULL");
        if (!aligned16(v_witness)) return fail(WC_ERR_INVALID_ARG, "v_witness must be 16-byte aligned");
        if (meter_b) return fail(WC_ERR_UNSUPPORTED, "Tier B and the value side are separate calls");
    }
    if (meter_b || meter_b_raw) {
        if (desc->scheme == WC_SCHEME_FP8_E4M3)
            return fail(WC_ERR_UNSUPPORTED, "Tier B needs the dithered INT8 cache (a controlled quantizer)");
        if (!meter_b || !meter_b_raw) return fail(WC_ERR_INVALID_ARG, "meter_b and meter_b_raw must not be NULL");
        if (!(delta_loc > 0.0 && delta_loc < 1.0))
            return fail(WC_ERR_INVALID_ARG, "delta_loc must be in (0, 1) (got %g)", delta_loc);
    }
    if (layer < 0 || layer > 65535) return fail(WC_ERR_INVALID_ARG, "layer must be in [0, 65535] (got %d)", layer);
    if (batch < 0 || batch > 65535) return fail(WC_ERR_INVALID_ARG, "batch must be in [0, 65535] (got %d)", batch);
    if (max_pages < 1) return fail(WC_ERR_INVALID_ARG, "max_pages must be positive (got %d)", max_pages);
    if ((long long)max_pages * wc::kPage > 0x7FFFFFFFLL) return fail(WC_ERR_UNSUPPORTED, "max_pages too large");
    if (batch == 0) return WC_OK;
    if (!q || !block_table || !ctx_lens || !out || !meter || !meter_raw || !workspace)
        return fail(WC_ERR_INVALID_ARG, "q, block_table, ctx_lens, out, meter, meter_raw, workspace must not be NULL");
    if (!aligned16(q)) return fail(WC_ERR_INVALID_ARG, "q must be 16-byte aligned");
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(WC_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    if (wc_status st = check_cache(desc, k_codes, v_codes, k_scale, v_scale, k_witness)) return st;
    int sms = 0;
    if (current_sm_count(&sms) != 0) return fail(WC_ERR_CUDA, "cannot query the current device");
    const wc::DecodePlan pl = wc::plan_decode(batch, desc->num_kv_heads, max_pages, sms, desc->scheme, desc->dither_bits);
    if (workspace_bytes < pl.total)
        return fail(WC_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, pl.total);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    wc::DecodeParams p;
    p.q = static_cast<const __half*>(q);
    p.block_table = block_table;
    p.ctx_lens = ctx_lens;
    p.k_codes = static_cast<const uint8_t*>(k_codes);
    p.v_codes = static_cast<const uint8_t*>(v_codes);
    p.k_scale = static_cast<const __half*>(k_scale);
    p.v_scale = static_cast<const __half*>(v_scale);
    p.k_witness = static_cast<const __half*>(k_witness);
    p.out = out;
    p.meter = meter;
    p.meter_raw = meter_raw;
    p.meter_b = meter_b;
    p.meter_b_raw = meter_b_raw;
    p.tb_log_2_over_delta = meter_b ? (float)std::log(2.0 / delta_loc) : 0.0f;
    p.v_witness = static_cast<const __half*>(v_witness);
    p.value_term = value_term;
    p.v_max = v_max;
    p.out_bound = out_bound;
    p.page_terms = reinterpret_cast<float2*>(page_terms);
    p.softmax_norm = reinterpret_cast<float2*>(softmax_norm);
    p.k_bypass = static_cast<const __half*>(k_bypass);
    p.bypass_pairs = bypass_pairs;
    p.num_bypass = num_bypass;
    p.k_new = static_cast<const __half*>(k_new);
    p.v_new = static_cast<const __half*>(v_new);
    p.slot_new = slot_new;
    p.stall_page = stall_page;
    p.status = reinterpret_cast<uint32_t*>(ws);
    p.partials = reinterpret_cast<float*>(ws + pl.partials_off);
    p.batch = batch;
    p.max_pages = max_pages;
    p.num_q_heads = desc->num_q_heads;
    p.num_kv_heads = desc->num_kv_heads;
    p.group = desc->num_q_heads / desc->num_kv_heads;
    p.num_pages = desc->num_pages;
    p.layer = layer;
    p.rope_layout = desc->rope_layout;
    p.splits = pl.splits;
    p.pages_per_split = pl.pages_per_split;
    p.keys = wc::make_philox_keys(desc->seed);
    cudaError_t e = wc::launch_decode(p, desc->scheme, desc->dither_bits, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "decode kernel launch");
}

wc_status wc_metered_decode_attention(const wc_cache_desc* desc, int32_t layer, const void* q,
                                      const int32_t* block_table, int32_t max_pages, const int32_t* ctx_lens,
                                      int32_t batch, const void* k_codes, const void* v_codes,
                                      const void* k_scale, const void* v_scale, const void* k_witness,
                                      float* out, float* meter, float* meter_raw, void* workspace,
                                      size_t workspace_bytes, void* stream) {
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, nullptr, nullptr, 0.0, nullptr, nullptr,
                                 nullptr, nullptr, nullptr, nullptr, workspace, workspace_bytes, stream);
}

wc_status wc_testing_decode_stalled_page(const wc_cache_desc* desc, int32_t layer, const void* q,
                                        const int32_t* block_table, int32_t max_pages, const int32_t* ctx_lens,
                                        const void* k_codes, const void* v_codes, const void* k_scale,
                                        const void* v_scale, const void* k_witness, float* out, float* meter,
                                        float* meter_raw, void* workspace, size_t workspace_bytes,
                                        int32_t stall_page, void* stream) {
    if (wc_status st = check_desc(desc)) return st;
    if (desc->scheme != WC_SCHEME_DITHER_INT8 || desc->dither_bits != 8)
        return fail(WC_ERR_UNSUPPORTED, "the stalled-page test runs the dithered INT8 cache with the 8-bit dither");
    if (stall_page < 0 || stall_page >= max_pages)
        return fail(WC_ERR_INVALID_ARG, "stall_page must be in [0, max_pages) (got %d)", stall_page);
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, 1, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, nullptr, nullptr, 0.0, nullptr, nullptr,
                                 nullptr, nullptr, nullptr, nullptr, workspace, workspace_bytes, stream, false, nullptr,
                                 nullptr, 0, nullptr, nullptr, nullptr, stall_page);
}

wc_status wc_metered_decode_attention_tier_b(const wc_cache_desc* desc, int32_t layer, const void* q,
                                             const int32_t* block_table, int32_t max_pages,
                                             const int32_t* ctx_lens, int32_t batch, const void* k_codes,
                                             const void* v_codes, const void* k_scale, const void* v_scale,
                                             const void* k_witness, double delta_loc, float* out, float* meter,
                                             float* meter_raw, float* meter_b, float* meter_b_raw,
                                             void* workspace, size_t workspace_bytes, void* stream) {
    if (!meter_b || !meter_b_raw) return fail(WC_ERR_INVALID_ARG, "meter_b and meter_b_raw must not be NULL");
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, meter_b, meter_b_raw, delta_loc,
                                 nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, workspace, workspace_bytes,
                                 stream);
}

wc_status wc_metered_decode_attention_v(const wc_cache_desc* desc, int32_t layer, const void* q,
                                        const int32_t* block_table, int32_t max_pages, const int32_t* ctx_lens,
                                        int32_t batch, const void* k_codes, const void* v_codes,
                                        const void* k_scale, const void* v_scale, const void* k_witness,
                                        const void* v_witness, float* out, float* meter, float* meter_raw,
                                        float* value_term, float* v_max, float* out_bound, void* workspace,
                                        size_t workspace_bytes, void* stream) {
    if (!v_witness || !value_term || !v_max || !out_bound)
        return fail(WC_ERR_INVALID_ARG, "v_witness, value_term, v_max and out_bound must not be NULL");
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, nullptr, nullptr, 0.0, v_witness,
                                 value_term, v_max, out_bound, nullptr, nullptr, workspace, workspace_bytes, stream);
}

wc_status wc_metered_decode_attention_repair(const wc_cache_desc* desc, int32_t layer, const void* q,
                                             const int32_t* block_table, int32_t max_pages,
                                             const int32_t* ctx_lens, int32_t batch, const void* k_codes,
                                             const void* v_codes, const void* k_scale, const void* v_scale,
                                             const void* k_witness, float* out, float* meter, float* meter_raw,
                                             float* page_terms, float* softmax_norm, void* workspace,
                                             size_t workspace_bytes, void* stream) {
    if (!page_terms || !softmax_norm)
        return fail(WC_ERR_INVALID_ARG, "page_terms and softmax_norm must not be NULL");
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, nullptr, nullptr, 0.0, nullptr, nullptr,
                                 nullptr, nullptr, page_terms, softmax_norm, workspace, workspace_bytes, stream);
}

wc_status wc_metered_decode_attention_append(const wc_cache_desc* desc, int32_t layer, const void* q,
                                             const int32_t* block_table, int32_t max_pages,
                                             const int32_t* ctx_lens, int32_t batch, void* k_codes, void* v_codes,
                                             void* k_scale, void* v_scale, void* k_witness, const void* k_new,
                                             const void* v_new, const int32_t* slot_new, float* out, float* meter,
                                             float* meter_raw, void* workspace, size_t workspace_bytes,
                                             void* stream) {
    if (!k_new || !v_new || !slot_new) return fail(WC_ERR_INVALID_ARG, "k_new, v_new and slot_new must not be NULL");
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, nullptr, nullptr, 0.0, nullptr, nullptr,
                                 nullptr, nullptr, nullptr, nullptr, workspace, workspace_bytes, stream, false,
                                 nullptr, nullptr, 0, k_new, v_new, slot_new);
}

wc_status wc_metered_decode_attention_g32(const wc_cache_desc* desc, int32_t layer, const void* q,
                                          const int32_t* block_table, int32_t max_pages, const int32_t* ctx_lens,
                                          int32_t batch, const void* k_codes, const void* v_codes,
                                          const void* k_scale, const void* v_scale, const void* k_witness,
                                          const void* k_bypass, const int32_t* bypass_pairs,
                                          int32_t num_bypass_pairs, double delta_loc, float* out, float* meter,
                                          float* meter_raw, float* meter_b, float* meter_b_raw, void* workspace,
                                          size_t workspace_bytes, void* stream) {
    return decode_with_workspace(desc, layer, q, block_table, max_pages, ctx_lens, batch, k_codes, v_codes, k_scale,
                                 v_scale, k_witness, out, meter, meter_raw, meter_b, meter_b_raw, delta_loc, nullptr,
                                 nullptr, nullptr, nullptr, nullptr, nullptr, workspace, workspace_bytes, stream, true,
                                 k_bypass, bypass_pairs, num_bypass_pairs);
}

wc_status wc_repair_select(const float* page_terms, const float* softmax_norm, const int32_t* ctx_lens,
                           int32_t batch, int32_t num_q_heads, int32_t max_pages, const uint8_t* keep_q, float tau,
                           float* contrib, int32_t* repair_pages, int32_t* n_repair, float* d_after,
                           uint32_t* dev_status, void* stream) {
    if (batch < 0 || batch > 65535) return fail(WC_ERR_INVALID_ARG, "batch must be in [0, 65535] (got %d)", batch);
    if (num_q_heads < 1 || num_q_heads > 65535)
        return fail(WC_ERR_INVALID_ARG, "num_q_heads must be in [1, 65535] (got %d)", num_q_heads);
    if (max_pages < 1) return fail(WC_ERR_INVALID_ARG, "max_pages must be positive (got %d)", max_pages);
    if (max_pages > wc::kRepairMaxPages)
        return fail(WC_ERR_UNSUPPORTED, "max_pages must be at most %d (got %d)", wc::kRepairMaxPages, max_pages);
    if (batch == 0) return WC_OK;
    if (!page_terms || !softmax_norm || !ctx_lens || !repair_pages || !n_repair || !d_after)
        return fail(WC_ERR_INVALID_ARG,
                    "page_terms, softmax_norm, ctx_lens, repair_pages, n_repair, d_after must not be NULL");
    if ((reinterpret_cast<uintptr_t>(page_terms) & 7u) || (reinterpret_cast<uintptr_t>(softmax_norm) & 7u))
        return fail(WC_ERR_INVALID_ARG, "page_terms and softmax_norm must be 8-byte aligned");
    wc::RepairParams p;
    p.page_terms = reinterpret_cast<const float2*>(page_terms);
    p.softmax_norm = reinterpret_cast<const float2*>(softmax_norm);
    p.ctx_lens = ctx_lens;
    p.keep_q = keep_q;
    p.contrib = contrib;
    p.repair_pages = repair_pages;
    p.n_repair = n_repair;
    p.d_after = d_after;
    p.status = dev_status;
    p.batch = batch;
    p.num_q_heads = num_q_heads;
    p.max_pages = max_pages;
    p.tau = tau;
    cudaError_t e = wc::launch_repair_select(p, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "repair selection kernel launch");
}

static wc_status gate_impl(const float* meter_raw, const float* value_term, const float* v_max, int32_t n_cells,
                          int32_t group, float tau, float tau_v, uint8_t* keep_q, uint8_t* keep_kv,
                          int32_t* n_kept, void* stream) {
    if (n_cells < 0 || group < 1 || n_cells % group != 0)
        return fail(WC_ERR_INVALID_ARG, "n_cells (%d) must be a non-negative multiple of group (%d)", n_cells, group);
    if (!n_kept) return fail(WC_ERR_INVALID_ARG, "n_kept must not be NULL");
    if (n_cells > 0 && (!meter_raw || !keep_q || !keep_kv))
        return fail(WC_ERR_INVALID_ARG, "meter_raw, keep_q, keep_kv must not be NULL");
    cudaError_t e = wc::launch_gate(meter_raw, value_term, v_max, n_cells, group, tau, tau_v, keep_q, keep_kv, n_kept,
                                    static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "gate kernel launch");
}

wc_status wc_gate(const float* meter_raw, int32_t n_cells, int32_t group, float tau, uint8_t* keep_q,
                  uint8_t* keep_kv, int32_t* n_kept, void* stream) {
    return gate_impl(meter_raw, nullptr, nullptr, n_cells, group, tau, 0.0f, keep_q, keep_kv, n_kept, stream);
}

wc_status wc_gate_joint(const float* meter_raw, const float* value_term, const float* v_max, int32_t n_cells,
                        int32_t group, float tau_k, float tau_v, uint8_t* keep_q, uint8_t* keep_kv, int32_t* n_kept,
                        void* stream) {
    if (n_cells > 0 && (!value_term || !v_max))
        return fail(WC_ERR_INVALID_ARG, "value_term and v_max must not be NULL");
    return gate_impl(meter_raw, value_term, v_max, n_cells, group, tau_k, tau_v, keep_q, keep_kv, n_kept, stream);
}

wc_status wc_read_status(void* workspace_or_word, int32_t is_status_word, uint32_t* bits, void* stream) {
    (void)is_status_word;   // the status word sits at offset 0 of a workspace
    if (!workspace_or_word || !bits) return fail(WC_ERR_INVALID_ARG, "pointers must not be NULL");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint32_t host = 0;
    cudaError_t e = cudaMemcpyAsync(&host, workspace_or_word, sizeof host, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(workspace_or_word, 0, sizeof host, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device status word");
    *bits = host;
    if (host) return fail(WC_ERR_DEVICE_CHECK, "device status bits 0x%x", host);
    return WC_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of the metered decode call.
//
// Some callers cannot allocate device memory when they call the decode: code
// running where cudaMalloc is forbidden or unsafe (inside a custom allocator's
// hooks, under a memory budget that must not move, or from a runtime that
// pre-plans every buffer and hands the library only its inputs and outputs).
// For them the scratch the decode needs (per-split partial results) lives in
// one fixed device array compiled into this library.  Every GPU that loads the
// library holds this array until the process exits.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB per device
constexpr int kNoAllocMaxDevices = 64;

// File-scope device scratch.  In host code this name is only a stand-in for
// the device array, never a device address: the address is looked up with
// cudaGetSymbolAddress (below) and passed to the kernels.
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

// The address belongs to the module as loaded into one device context; a
// context that is torn down and recreated (cudaDeviceReset) loads the module
// again.  So the address is cached per device together with the context it
// was looked up in, and looked up again when the current context differs.
using CtxGetCurrentFn = int (*)(void**);   // cuCtxGetCurrent through the runtime's driver entry point

CtxGetCurrentFn ctx_get_current() {
    static std::once_flag once;
    static CtxGetCurrentFn fn = nullptr;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<CtxGetCurrentFn>(f);
    });
    return fn;
}

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kNoAllocMaxDevices] = {};
void* g_noalloc_ctx[kNoAllocMaxDevices] = {};

// Address of the scratch in the current device's current context.
wc_status noalloc_scratch(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(WC_ERR_UNSUPPORTED, "device index %d too large", dev);
    CtxGetCurrentFn get = ctx_get_current();
    if (!get) return fail(WC_ERR_CUDA, "cannot query the current device context");
    void* ctx = nullptr;   // null until the runtime has made a context current on this thread
    if (get(&ctx) != 0) return fail(WC_ERR_CUDA, "cannot query the current device context");
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!ctx || !g_noalloc_ptr[dev] || g_noalloc_ctx[dev] != ctx) {
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);   // also makes the device's context current
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress of the decode scratch");
        if (get(&ctx) != 0 || !ctx) return fail(WC_ERR_CUDA, "cannot query the current device context");
        g_noalloc_ptr[dev] = ptr;
        g_noalloc_ctx[dev] = ctx;
    }
    *out = g_noalloc_ptr[dev];
    return WC_OK;
}

}  // namespace

extern "C" wc_status wc_metered_decode_attention_noalloc(
    const wc_cache_desc* desc, int32_t layer, const void* q, const int32_t* block_table, int32_t max_pages,
    const int32_t* ctx_lens, int32_t batch, const void* k_codes, const void* v_codes, const void* k_scale,
    const void* v_scale, const void* k_witness, float* out, float* meter, float* meter_raw, uint32_t* dev_status,
    void* stream) {
    if (wc_status st = check_desc(desc)) return st;
    if (layer < 0 || layer > 65535) return fail(WC_ERR_INVALID_ARG, "layer must be in [0, 65535] (got %d)", layer);
    if (batch < 0 || batch > 65535) return fail(WC_ERR_INVALID_ARG, "batch must be in [0, 65535] (got %d)", batch);
    if (max_pages < 1) return fail(WC_ERR_INVALID_ARG, "max_pages must be positive (got %d)", max_pages);
    if ((long long)max_pages * wc::kPage > 0x7FFFFFFFLL) return fail(WC_ERR_UNSUPPORTED, "max_pages too large");
    if (batch == 0) return WC_OK;
    if (!q || !block_table || !ctx_lens || !out || !meter || !meter_raw || !dev_status)
        return fail(WC_ERR_INVALID_ARG, "q, block_table, ctx_lens, out, meter, meter_raw, dev_status must not be NULL");
    if (!aligned16(q)) return fail(WC_ERR_INVALID_ARG, "q must be 16-byte aligned");
    if (wc_status st = check_cache(desc, k_codes, v_codes, k_scale, v_scale, k_witness)) return st;
    int sms = 0;
    if (current_sm_count(&sms) != 0) return fail(WC_ERR_CUDA, "cannot query the current device");
    const wc::DecodePlan pl = wc::plan_decode(batch, desc->num_kv_heads, max_pages, sms, desc->scheme, desc->dither_bits);
    if (pl.total > kNoAllocScratchBytes)
        return fail(WC_ERR_UNSUPPORTED,
                    "this decode needs %zu bytes of scratch but the built-in scratch holds %zu; "
                    "use wc_metered_decode_attention with a caller workspace",
                    pl.total, kNoAllocScratchBytes);
    void* scratch = nullptr;
    if (wc_status st = noalloc_scratch(&scratch)) return st;
    uint8_t* ws = static_cast<uint8_t*>(scratch);
    wc::DecodeParams p;
    p.q = static_cast<const __half*>(q);
    p.block_table = block_table;
    p.ctx_lens = ctx_lens;
    p.k_codes = static_cast<const uint8_t*>(k_codes);
    p.v_codes = static_cast<const uint8_t*>(v_codes);
    p.k_scale = static_cast<const __half*>(k_scale);
    p.v_scale = static_cast<const __half*>(v_scale);
    p.k_witness = static_cast<const __half*>(k_witness);
    p.out = out;
    p.meter = meter;
    p.meter_raw = meter_raw;
    p.meter_b = nullptr;
    p.meter_b_raw = nullptr;
    p.tb_log_2_over_delta = 0.0f;
    p.v_witness = nullptr;
    p.value_term = nullptr;
    p.v_max = nullptr;
    p.out_bound = nullptr;
    p.status = dev_status;
    p.partials = reinterpret_cast<float*>(ws + pl.partials_off);
    p.batch = batch;
    p.max_pages = max_pages;
    p.num_q_heads = desc->num_q_heads;
    p.num_kv_heads = desc->num_kv_heads;
    p.group = desc->num_q_heads / desc->num_kv_heads;
    p.num_pages = desc->num_pages;
    p.layer = layer;
    p.rope_layout = desc->rope_layout;
    p.splits = pl.splits;
    p.pages_per_split = pl.pages_per_split;
    p.keys = wc::make_philox_keys(desc->seed);
    cudaError_t e = wc::launch_decode(p, desc->scheme, desc->dither_bits, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? WC_OK : cuda_fail(e, "decode kernel launch");
}
