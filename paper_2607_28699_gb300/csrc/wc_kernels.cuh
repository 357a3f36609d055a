// Launch parameters and launchers of the WitCert kernels (host + device).
#pragma once

#include <cuda_runtime.h>

#include "wc_common.cuh"

namespace wc {

struct WriteParams {
    const __half* k;
    const __half* v;
    const int32_t* slot_mapping;
    void* k_codes;
    void* v_codes;
    __half* k_scale;
    __half* v_scale;
    __half* k_witness;
    __half* v_witness;    // [slot][2] (rho^v, ||v||) rounded up, nullptr: not stored
    __half* k_bypass = nullptr;              // grouped scheme: [slot][2m] exact bypassed values
    const int32_t* bypass_pairs = nullptr;   // grouped scheme: [Hkv][m] RoPE pair indices
    int32_t num_bypass = 0;                  // m
    uint32_t* dev_status;
    int32_t n_tok, num_kv_heads, num_pages, layer, rope_layout;
    PhiloxKeys keys;
};

struct DecodeParams {
    const __half* q;
    const int32_t* block_table;
    const int32_t* ctx_lens;
    const uint8_t* k_codes;
    const uint8_t* v_codes;
    const __half* k_scale;
    const __half* v_scale;
    const __half* k_witness;
    float* out;
    float* meter;
    float* meter_raw;
    float* meter_b;       // Tier-B meters (§4.2), nullptr: not computed
    float* meter_b_raw;
    float tb_log_2_over_delta;   // log(2 / delta_loc) for Tier B
    const __half* v_witness;     // [slot][2] (rho^v, ||v||) for the value side
    float* value_term;           // value side outputs, nullptr: not computed
    float* v_max;
    float* out_bound;
    // Block-level repair selection (§6.3.5), nullptr: not emitted.  Per page j of
    // each (sequence, query head): (m_j, d_j), the page's share of D summed
    // against the running maximum m_j, so that it contributes d_j 2^(m_j - M) / L;
    // per (sequence, query head): (M, L), the final log2-domain maximum and sum.
    float2* page_terms = nullptr;     // [batch][Hq][max_pages]
    float2* softmax_norm = nullptr;   // [batch][Hq]
    // append: the step's new token of each sequence, quantized and stored by the
    // decode itself before it reads it (nullptr: none)
    const __half* k_new = nullptr;     // [batch][Hkv][128] fp16
    const __half* v_new = nullptr;
    const int32_t* slot_new = nullptr;   // [batch], < 0: no new token
    // grouped scheme: exact bypassed key values [slot][2m] and the pair set [Hkv][m]
    const __half* k_bypass = nullptr;
    const int32_t* bypass_pairs = nullptr;
    int32_t num_bypass = 0;
    // failure-detection test only (wc_testing_decode_stalled_page): the logical
    // page whose copies are never issued, so that the bounded waits run out; -1: none
    int32_t stall_page = -1;
    uint32_t* status;     // workspace word
    float* partials;      // [batch * Hkv * splits] (flattened: [splits + batch * Hkv]) x [kMaxGroup][kPartialStride]
    int32_t batch, max_pages, num_q_heads, num_kv_heads, group, num_pages, layer, rope_layout;
    // pages_per_split == 0 marks the flattened plan (warp-specialized kernel,
    // batch > 1): the grid is `splits` CTAs, a multiple of Hkv; CTA c serves KV
    // head c mod Hkv with the (c / Hkv)-th equal share of the batch's pages laid
    // end to end, cut at sequence boundaries into segments.  Share j's segment of
    // sequence b writes partial h (shares + batch) + j + b (unique: along the
    // pages each next segment increments j, b or both), so splits + batch Hkv
    // partials suffice.
    int32_t splits, pages_per_split;
    PhiloxKeys keys;
};

// Per (query head, split) partial: acc[128] | m | l | D | Tier-B D | value
// term | max ||v|| | pad.  140 floats: in the CTA merge's shared buffer the
// rows of the heads one warp instruction touches then start in distinct bank
// groups (12 words apart modulo 32; 136 would put two heads on each group).
constexpr int kPartialStride = kHeadDim + 12;

// Workspace layout (bytes): [0, 256) status word, then the partials
// (256-byte aligned).
struct DecodePlan {
    int splits;            // flattened plan: the grid's CTAs
    int pages_per_split;   // 0: the flattened plan
    size_t partials_off, total;
};

DecodePlan plan_decode(int batch, int num_kv_heads, int max_pages, int num_sms, int scheme, int bits);

// Launch `kernel` on `stream` as a programmatic dependent of the preceding work.
template <typename Kernel, typename Params>
inline cudaError_t launch_pdl(Kernel kernel, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              const Params& p) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, p);
}

struct RepairParams {
    const float2* page_terms;     // [batch][Hq][max_pages] (m_j, d_j)
    const float2* softmax_norm;   // [batch][Hq] (M, L)
    const int32_t* ctx_lens;
    const uint8_t* keep_q;        // [batch][Hq], nullptr: every cell is repaired
    float* contrib;               // [batch][Hq][max_pages] C_j, nullptr: not stored
    int32_t* repair_pages;        // [batch][Hq][max_pages] logical pages in paging order
    int32_t* n_repair;            // [batch][Hq]
    float* d_after;               // [batch][Hq] D left after the listed pages
    uint32_t* status;             // optional device word, WC_DEV_BAD_CTX
    int32_t batch, num_q_heads, max_pages;
    float tau;
};

// Largest block-table width the selection handles (its sort holds one cell's
// pages in shared memory).
constexpr int kRepairMaxPages = 16384;
// Page streams (producer / consumer warp pairs) per CTA of the grouped-scheme
// decode; the split planner sizes splits by it.
constexpr int kG32PageStreams = 6;

cudaError_t launch_write(const WriteParams& p, int scheme, int bits, cudaStream_t stream);
cudaError_t launch_decode(const DecodeParams& p, int scheme, int bits, cudaStream_t stream);
cudaError_t launch_decode_g32(const DecodeParams& p, cudaStream_t stream);
cudaError_t launch_repair_select(const RepairParams& p, cudaStream_t stream);
cudaError_t launch_select_pairs(const __half* k, int n_tok, int num_kv_heads, int rope_layout, int m, int32_t* pairs,
                                cudaStream_t stream);
cudaError_t launch_gate(const float* meter_raw, const float* value_term, const float* v_max, int n_cells, int group,
                        float tau, float tau_v, uint8_t* keep_q, uint8_t* keep_kv, int32_t* n_kept,
                        cudaStream_t stream);

}  // namespace wc
