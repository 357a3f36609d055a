// Metered decode attention (§6 meter loop, read path; §6.2.1-§6.2.2):
// dequantize the paged cache, compute the compressed attention output, and in
// the same pass accumulate the Tier-A e-form meter
//   c_t = (1/sqrt d) sum_b ||q_b|| w_{t,b}        (Thm. "Sound black-box logit bound")
//   A   = sum_t p~_t e^{c_t},  meter = min(1, (A^2 - 1)/2)   (Thm. "Sound replacement")
// merged across context splits under log-sum-exp weights (A is a p~-weighted
// mean, so it merges exactly like the output; §6.2.2).
//
// Grid (splits, Hkv, batch), or under the flattened plan (kXFlat: the 10-bit
// dither on a batch that leaves SMs idle) one CTA per 8 warp shares of the
// batch's pages; 8 warps per CTA, two CTAs per SM.  Each warp owns
// a 3-stage ring of page buffers in shared memory that its lane 0 fills ahead
// of use: the K and V code tiles (2 KiB each) by tensor-map TMA with the
// 128-byte swizzle (so the 16-byte reads of a warp phase hit distinct banks),
// scales and witness by bulk copies, all completing on the stage's mbarrier;
// a page is 16 tokens of one KV head.  Warps run independently until the
// CTA's closing merge.
//
// Per page a warp computes, on mma.sync (fp16 in, fp32 accumulate):
//   QK:    S[token][head]  = code . q - h' . q                m16n8k16, A = codes / dither
//   bound: C[token][head]  = W[token][band] . a[band][head]    m16n8k8, a = ||q_b||/sqrt(d) (hi + lo)
//   PV:    acc[dim][head] += V^T P^T - H^T P^T                 m16n8k16, B = P^T (hi + lo, movmatrix)
// Integer codes and the dither enter the tensor cores as exact fp16 values
// (h' = 4 + j/256 for 8-bit, 1 + j/1024 for 10-bit dither; xi = h' - kappa),
// so code - xi = code - h' + kappa is carried exactly to the fp32 accumulators.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <mutex>

#include "decode_common.cuh"
#include "write_row.cuh"

namespace wc {

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kStages = 3;
constexpr int kMinBlocks = 2;            // two CTAs (16 warps) per SM
constexpr int kStageBytes = 4416;        // copy bytes: K codes | V codes | K scale | V scale | witness
// Shared memory: the K and V code tiles of every (warp, stage), [16][128] bytes
// each, written by tensor-map TMA with the 128-byte swizzle (1024-byte aligned
// regions), then each stage's scales and witness, then the barriers.
constexpr int kTileRegion = kWarps * kStages * 2048;
constexpr int kOffKs = 0, kOffVs = 32, kOffW = 64;   // within a stage's small part
constexpr int kOffVw = 320;              // value witness [16][2] fp16 (value side)
constexpr int kSmallStride = 384;
constexpr int kSmemBytes = 2 * kTileRegion + kWarps * kStages * kSmallStride + kWarps * kStages * 8 + 1024;

// The per-token kernel's parameters: the code tiles' tensor maps and the call.
struct DkParams {
    CUtensorMap k_map;   // k_codes as [num_pages * Hkv][16][128] bytes, box = one page of one head
    CUtensorMap v_map;
    DecodeParams p;
};

// §6.3.5 "Block-level paging": the share of D of logical page lp for this
// thread's softmax heads 2c, 2c+1, kept against the running maximum it was
// summed under; with the final (M, L) the page contributes d 2^(m - M) / L.
// dpg holds the thread's tokens g, g+8 on entry; the sum runs over the rows g.
__device__ __forceinline__ void emit_page_terms(const DecodeParams& p, int b, int h, int G, int lp, int g, int c,
                                                float (&dpg)[2], const float (&m_run)[2]) {
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
        dpg[0] += __shfl_xor_sync(0xffffffffu, dpg[0], o);
        dpg[1] += __shfl_xor_sync(0xffffffffu, dpg[1], o);
    }
    if (g == 0) {
        float2* dst = p.page_terms + ((size_t)b * p.num_q_heads + (size_t)h * G) * p.max_pages + lp;
        if (2 * c < G) dst[(size_t)(2 * c) * p.max_pages] = make_float2(m_run[0], dpg[0]);
        if (2 * c + 1 < G) dst[(size_t)(2 * c + 1) * p.max_pages] = make_float2(m_run[1], dpg[1]);
    }
}

// A page the kernel could not read (outside the pool) contributes nothing.
__device__ __forceinline__ void emit_skipped_page(const DecodeParams& p, int b, int h, int G, int lp, int lane) {
    if (lane < G)
        p.page_terms[((size_t)b * p.num_q_heads + (size_t)h * G + lane) * p.max_pages + lp] =
            make_float2(-INFINITY, 0.f);
}

// q fragment of the B operand (head g, channels 32c + 2i, +1 in word i).
__device__ __forceinline__ void load_q_frag(const DecodeParams& p, int b, int h, int G, int g, int c,
                                            uint32_t (&qw)[16]) {
    const bool row_valid = g < G;
    const uint4* qsrc = reinterpret_cast<const uint4*>(
        p.q + ((size_t)b * p.num_q_heads + (size_t)h * G + (row_valid ? g : 0)) * kHeadDim + 32 * c);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 v = row_valid ? __ldg(qsrc + i) : make_uint4(0, 0, 0, 0);
        qw[4 * i] = v.x; qw[4 * i + 1] = v.y; qw[4 * i + 2] = v.z; qw[4 * i + 3] = v.w;
    }
}

// A warp's pages in order.  Split plan: pages warp, warp + 8, ... of one
// sequence's split.  Flattened plan: a contiguous range of the batch's pages
// laid end to end, sequence after sequence (sequences without pages hold
// none of it).  dk_next is called only while the range has another page.
struct DkWalk {
    int b, lp, np;   // sequence, logical page, the sequence's page count
};
template <bool kFlat>
__device__ __forceinline__ void dk_next(const DecodeParams& p, DkWalk& w) {
    if constexpr (!kFlat) {
        w.lp += kWarps;
    } else if (++w.lp >= w.np) {
        do {
            ++w.b;
            w.np = (clamped_ctx(p, w.b) + kPage - 1) / kPage;
        } while (w.np == 0 && w.b + 1 < p.batch);
        w.lp = 0;
    }
}

template <int kScheme, int kBits, int kX>
__global__ void __launch_bounds__(kThreads, kMinBlocks) decode_kernel(const __grid_constant__ DkParams dp) {
    constexpr bool kTierB = (kX & kXTierB) != 0, kValue = (kX & kXValue) != 0, kRepair = (kX & kXRepair) != 0;
    const DecodeParams& p = dp.p;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, c = lane & 3;
    // split plan: grid (splits, Hkv, batch); flattened plan (kXFlat): grid (CTAs),
    // CTA c serving KV head c mod Hkv, each warp its own share of the batch's pages
    constexpr bool kFlat = (kX & kXFlat) != 0;
    const int split = kFlat ? 0 : (int)blockIdx.x;
    const int h = kFlat ? (int)blockIdx.x % p.num_kv_heads : (int)blockIdx.y;
    int b = kFlat ? 0 : (int)blockIdx.z;   // the sequence whose pages are being consumed
    const int G = p.group;
    constexpr bool kInt8 = (kScheme == WC_SCHEME_DITHER_INT8);

    uint8_t* my_k = smem + warp * kStages * 2048;   // this warp's K code tiles; its V tiles kTileRegion on
    uint8_t* my_small = smem + 2 * kTileRegion + warp * kStages * kSmallStride;
    uint64_t* bars =
        reinterpret_cast<uint64_t*>(smem + 2 * kTileRegion + kWarps * kStages * kSmallStride) + warp * kStages;
    if (lane == 0)
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
    fence_barrier_init();
    // the dependent merge may be scheduled now: it waits for this whole grid
    // (griddepcontrol.wait) and launches only once every CTA here has started
    grid_dep_launch();
    grid_dep_wait();   // q, page tables and the cache may come from the preceding kernel

    const bool row_valid = g < G;
    const int p0 = split * p.pages_per_split;                          // split plan
    const int32_t* bt_row = p.block_table + (size_t)b * p.max_pages;   // split plan
    int ring[kStages];   // physical pages of this warp's next kStages pages
    uint32_t qw[16];     // head g, channels 32c + 2i, +1 in word i
    int ctx, n_my;
    DkWalk cw, iw;       // flattened plan: the page being consumed, the next page to issue
    if constexpr (!kFlat) {
        // Independent loads first: context length, this warp's first page-table
        // entries and the query fragments do not depend on one another.
        const int lim = min(p0 + p.pages_per_split, p.max_pages);
#pragma unroll
        for (int k = 0; k < kStages; ++k) {
            const int lp = p0 + warp + kWarps * k;
            ring[k] = lp < lim ? __ldg(bt_row + lp) : -1;
        }
        ctx = __ldg(p.ctx_lens + b);
        load_q_frag(p, b, h, G, g, c, qw);
        if (ctx < 0 || ctx > p.max_pages * kPage) {
            if (threadIdx.x == 0 && split == 0 && h == 0) atomicOr(p.status, WC_DEV_BAD_CTX);
            ctx = max(0, min(ctx, p.max_pages * kPage));
        }
        const int npages = (ctx + kPage - 1) / kPage;
        const int p1 = min(p0 + p.pages_per_split, npages);
        n_my = (p1 - p0 - warp > 0) ? (p1 - p0 - warp + kWarps - 1) / kWarps : 0;
        cw = iw = DkWalk{b, 0, 0};
    } else {
        // Warp share J = (c / Hkv) * 8 + warp takes pages [J R, (J + 1) R) of the
        // batch's pages laid end to end, R = ceil(total / shares), shares =
        // splits / Hkv; a scan of the page counts finds where each range starts.
        __shared__ int s_wtot[kWarps];
        __shared__ long long s_start[kWarps];
        const int t = threadIdx.x, per = (p.batch + kThreads - 1) / kThreads;
        int loc = 0;
        bool bad = false;
        for (int i = 0; i < per; ++i) {
            const int bb = t * per + i;
            if (bb < p.batch) {
                const int cx = __ldg(p.ctx_lens + bb);
                bad |= cx < 0 || cx > p.max_pages * kPage;
                loc += (max(0, min(cx, p.max_pages * kPage)) + kPage - 1) / kPage;
            }
        }
        if (bad && blockIdx.x == 0) atomicOr(p.status, WC_DEV_BAD_CTX);
        int inc = loc;   // inclusive scan over the warp
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += v;
        }
        if (lane == 31) s_wtot[warp] = inc;
        __syncthreads();
        int before = 0, total = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const int v = s_wtot[w];
            total += v;
            if (w < warp) before += v;
        }
        const int excl = before + inc - loc;   // pages of the sequences before this thread's
        const int shares = max(1, p.splits / p.num_kv_heads);
        const long long R = max(1LL, ((long long)total + shares - 1) / shares);
        const long long j0 = (long long)((int)blockIdx.x / p.num_kv_heads) * kWarps;
        for (int w = 0; w < kWarps; ++w) {
            const long long lo = (j0 + w) * R;
            if (lo < total && excl <= lo && lo < (long long)excl + loc) {
                long long acc = excl;   // exactly one thread: the one whose sequences hold lo
                for (int i = 0; i < per; ++i) {
                    const int bb = t * per + i;
                    if (bb >= p.batch) break;
                    const int np = (clamped_ctx(p, bb) + kPage - 1) / kPage;
                    if (lo < acc + np) {
                        s_start[w] = ((long long)bb << 32) | (long long)(lo - acc);
                        break;
                    }
                    acc += np;
                }
            }
        }
        __syncthreads();
        const long long lo = (j0 + warp) * R;
        n_my = (int)max(0LL, min((long long)total, lo + R) - lo);
        if (n_my > 0) {
            const long long st = s_start[warp];
            cw.b = (int)(st >> 32);
            cw.lp = (int)(st & 0xffffffffLL);
            cw.np = (clamped_ctx(p, cw.b) + kPage - 1) / kPage;
        } else {
            cw = DkWalk{0, 0, 0};
        }
        iw = cw;
#pragma unroll
        for (int k = 0; k < kStages; ++k) {
            ring[k] = k < n_my ? __ldg(p.block_table + (size_t)iw.b * p.max_pages + iw.lp) : -1;
            if (k + 1 < n_my) dk_next<true>(p, iw);
        }
        ctx = 0;
    }
    const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;

    // ---- per-warp stage ring --------------------------------------------------
    auto issue = [&](int k, int phys) {
        if (k >= n_my || lane != 0) return;
        uint64_t* bar = &bars[k % kStages];
        if (phys < 0 || phys >= p.num_pages) {
            atomicOr(p.status, WC_DEV_BAD_PAGE);
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
            return;
        }
        const int s = k % kStages;
        uint8_t* st = my_small + s * kSmallStride;
        const int z = phys * p.num_kv_heads + h;
        const size_t ph = (size_t)z;
        constexpr uint32_t bytes = (kInt8 ? kStageBytes : (2048 + 2048 + 256)) + (kValue ? 64 : 0);
        mbar_arrive_expect_tx(bar, bytes);
        tma_page(my_k + s * 2048, &dp.k_map, z, bar);
        tma_page(my_k + kTileRegion + s * 2048, &dp.v_map, z, bar);
        if constexpr (kInt8) {
            bulk_g2s(st + kOffKs, p.k_scale + ph * kPage, 32, bar);
            bulk_g2s(st + kOffVs, p.v_scale + ph * kPage, 32, bar);
        }
        bulk_g2s(st + kOffW, p.k_witness + ph * (kPage * kBands), 256, bar);
        if constexpr (kValue) bulk_g2s(st + kOffVw, p.v_witness + ph * (kPage * 2), 64, bar);
    };
    __syncwarp();
#pragma unroll
    for (int k = 0; k < kStages; ++k) issue(k, ring[k]);

    // ---- per sequence: band norms and the bound operand ----------------------------
    // (once under the split plan; at each sequence's first page under the flattened plan)
    float alpha0, alpha1, zoff0, zoff1;
    uint32_t a_hi, a_lo;   // B operand of the bound: a[head g][bands 2c, 2c+1]
    auto query_setup = [&]() {
    float qsum = 0.f, part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&qw[i]));
        qsum += f.x + f.y;
        part[i >> 2] = fmaf(f.x, f.x, fmaf(f.y, f.y, part[i >> 2]));   // channels 32c + 8(i>>2) .. +7
    }
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 1);
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 2);
    // Tier B (§4.2): u_t = alpha s_t with alpha = sqrt(2 log(2S/delta) ||q||^2 / (12 d)),
    // for this thread's softmax heads 2c and 2c+1
    alpha0 = alpha1 = 0.f;
    if constexpr (kTierB) {
        float qn2 = part[0] + part[1] + part[2] + part[3];   // ||q_g||^2 over channels 32c .. 32c+31
        qn2 += __shfl_xor_sync(0xffffffffu, qn2, 1);
        qn2 += __shfl_xor_sync(0xffffffffu, qn2, 2);
        const float lg = p.tb_log_2_over_delta + logf((float)max(ctx, 1));   // log(2S / delta)
        const float al = sqrtf(2.0f * lg * qn2 * (1.0f / (12.0f * kHeadDim)));
        alpha0 = __shfl_sync(0xffffffffu, al, 8 * c);
        alpha1 = __shfl_sync(0xffffffffu, al, 8 * c + 4);
    }
    float band_a, band_b;   // squared norms of bands 2c and 2c+1 of head g
    if (p.rope_layout == WC_ROPE_HALF) {
        // lane c holds the first (c < 2) or second (c >= 2) halves of bands 4(c&1) + i
#pragma unroll
        for (int i = 0; i < 4; ++i) part[i] += __shfl_xor_sync(0xffffffffu, part[i], 2);
        const int src = (lane & ~3) | (c >> 1);
        float v[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) v[i] = __shfl_sync(0xffffffffu, part[i], src);
        band_a = (c & 1) ? v[2] : v[0];
        band_b = (c & 1) ? v[3] : v[1];
    } else {
        band_a = part[0] + part[1];   // dims 32c .. 32c+15 = band 2c
        band_b = part[2] + part[3];
    }
    a_hi = a_lo = 0;
    if (row_valid) {
        const float x0 = sqrtf(band_a) * kRsd, x1 = sqrtf(band_b) * kRsd;
        const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
        a_hi = pack_h2(__half2float(h0), __half2float(h1));
        a_lo = pack_h2(x0 - __half2float(h0), x1 - __half2float(h1));
    }
    // this thread's softmax heads are 2c and 2c+1: kappa * sum(q) for each
    constexpr float kKappa = kInt8 ? DitherConst<kBits == 10 ? 10 : 8>::kappa : 0.f;
    zoff0 = kKappa * __shfl_sync(0xffffffffu, qsum, 8 * c);
    zoff1 = kKappa * __shfl_sync(0xffffffffu, qsum, 8 * c + 4);
    };
    if constexpr (!kFlat) query_setup();

    // ---- running state (heads 2c, 2c+1) ----------------------------------------------
    // Log2-domain softmax reference, moved lazily: only when a page's max
    // exceeds it by more than 8 (P may reach 2^8 in between).
    float m_run[2], l_part[2], d_part[2], spv_part[2];
    float db_part[2];   // Tier-B meter accumulator (kTierB)
    float vt_part[2];   // value side: sum p~ rho^v (kValue)
    float vmax;         // value side: max ||v|| over this thread's tokens
    float acc[8][4];
    int lam_exp;        // P * s_v * 2^lam_exp stays below 2^14 (fp16): s_v * 2^lam_exp < 2^6
    auto reset_state = [&]() {
        m_run[0] = m_run[1] = -INFINITY;
        l_part[0] = l_part[1] = d_part[0] = d_part[1] = spv_part[0] = spv_part[1] = 0.f;
        db_part[0] = db_part[1] = vt_part[0] = vt_part[1] = 0.f;
        vmax = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
        lam_exp = kInt8 ? INT_MIN : 6;
    };
    reset_state();
    bool failed = false;
    int consumed = 0;
    // ---- a warp's rows: totals for heads 2c, 2c+1 (reduced over the token rows g),
    // then its partial [head][kPartialStride] at wb (shared memory for the CTA merge
    // of the split plan, the workspace under the flattened plan)
    auto warp_rows = [&](float* wb) {
#pragma unroll
        for (int o = 4; o < 32; o <<= 1)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                l_part[e] += __shfl_xor_sync(0xffffffffu, l_part[e], o);
                d_part[e] += __shfl_xor_sync(0xffffffffu, d_part[e], o);
                if constexpr (kTierB) db_part[e] += __shfl_xor_sync(0xffffffffu, db_part[e], o);
                if constexpr (kValue) vt_part[e] += __shfl_xor_sync(0xffffffffu, vt_part[e], o);
                spv_part[e] += __shfl_xor_sync(0xffffffffu, spv_part[e], o);
            }
        if constexpr (kValue)
            for (int o = 1; o < 32; o <<= 1) vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
        const float inv_lam = kInt8 ? pow2(lam_exp == INT_MIN ? 0 : -lam_exp) : pow2(-lam_exp);
        const float kap = kInt8 ? DitherConst<kBits == 10 ? 10 : 8>::kappa : 0.f;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            float* row = wb + (2 * c + e) * kPartialStride + 16 * g;   // dims 16g .. 16g+15
            const float add = kap * spv_part[e];
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                float4 v;
                v.x = fmaf(acc[2 * q4][e], inv_lam, add);
                v.y = fmaf(acc[2 * q4][e + 2], inv_lam, add);
                v.z = fmaf(acc[2 * q4 + 1][e], inv_lam, add);
                v.w = fmaf(acc[2 * q4 + 1][e + 2], inv_lam, add);
                *reinterpret_cast<float4*>(row + 4 * q4) = v;
            }
            if (g == 0) {
                wb[(2 * c + e) * kPartialStride + kHeadDim + 0] = m_run[e];
                wb[(2 * c + e) * kPartialStride + kHeadDim + 1] = l_part[e];
                wb[(2 * c + e) * kPartialStride + kHeadDim + 2] = d_part[e];
                if constexpr (kTierB) wb[(2 * c + e) * kPartialStride + kHeadDim + 3] = db_part[e];
                if constexpr (kValue) {
                    wb[(2 * c + e) * kPartialStride + kHeadDim + 4] = vt_part[e];
                    wb[(2 * c + e) * kPartialStride + kHeadDim + 5] = vmax;
                }
            }
        }
    };
    // flattened plan: warp share J's part of sequence b is partial h (shares + batch) + J + b
    // (unique; a unit's partials consecutive, as the merge reads them)
    auto flat_partial = [&]() {
        const int shares = max(1, p.splits / p.num_kv_heads);
        const int J = ((int)blockIdx.x / p.num_kv_heads) * kWarps + warp;
        return p.partials + ((size_t)h * (shares + p.batch) + J + b) * (kMaxGroup * kPartialStride);
    };

    for (int k = 0; k < n_my; ++k) {
        int lp, phys_issue;   // this page; the page-table entry of the page issued at the end of the iteration
        if constexpr (kFlat) {
            if (k == 0 || cw.b != b) {   // a sequence's first page of this warp (warp-uniform)
                if (k > 0) warp_rows(flat_partial());
                b = cw.b;
                ctx = clamped_ctx(p, b);
                load_q_frag(p, b, h, G, g, c, qw);
                query_setup();
                reset_state();
            }
            lp = cw.lp;
            phys_issue = (k + kStages < n_my) ? __ldg(p.block_table + (size_t)iw.b * p.max_pages + iw.lp) : -1;
        } else {
            lp = p0 + warp + kWarps * k;
            phys_issue = (k + kStages < n_my) ? __ldg(bt_row + lp + kWarps * kStages) : -1;
        }
        const int phys = ring[0];
        const bool page_ok = phys >= 0 && phys < p.num_pages;
        const bool landed = mbar_wait_bounded(&bars[k % kStages], (uint32_t)((k / kStages) & 1));
        if (!__all_sync(0xffffffffu, landed)) {   // warp-uniform decision
            if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
            failed = true;
            break;
        }
        consumed = k + 1;
        if (page_ok) {
            const uint8_t* st = my_small + (k % kStages) * kSmallStride;
            const uint8_t* kt = my_k + (k % kStages) * 2048;   // V tile at kt + kTileRegion
            const uint32_t slot0 = (uint32_t)phys * kPage;
            const int nvalid = min(kPage, ctx - lp * kPage);

            // ---------------- QK: S[token][head] --------------------------------
            // rows g and g+8 are tokens g and g+8; d*[0..3] =
            // (tok g, head 2c), (tok g, 2c+1), (tok g+8, 2c), (tok g+8, 2c+1)
            float dc[4] = {0.f, 0.f, 0.f, 0.f}, dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int gp = 0; gp < 2; ++gp) {                 // channels 32c + 16gp .. +15
                const uint4 ka = *reinterpret_cast<const uint4*>(kt + swz(g, 2 * c + gp));
                const uint4 kb = *reinterpret_cast<const uint4*>(kt + swz(g + 8, 2 * c + gp));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const int ks = 4 * gp + kk;              // channels 32c + 4ks .. +3
                    const uint32_t wa = word_of(ka, kk), wb = word_of(kb, kk);
                    uint32_t A[4];
                    if constexpr (kInt8) {
                        const uint32_t xa = wa ^ 0x80808080u, xb = wb ^ 0x80808080u;
                        A[0] = s8x2_to_h2(xa, kSel01);
                        A[1] = s8x2_to_h2(xb, kSel01);
                        A[2] = s8x2_to_h2(xa, kSel23);
                        A[3] = s8x2_to_h2(xb, kSel23);
                    } else {
                        A[0] = e4m3x2_to_h2(wa);
                        A[1] = e4m3x2_to_h2(wb);
                        A[2] = e4m3x2_to_h2(wa >> 16);
                        A[3] = e4m3x2_to_h2(wb >> 16);
                    }
                    mma16816(dc, A, qw[2 * ks], qw[2 * ks + 1]);
                }
            }
            if constexpr (kInt8) {
                constexpr int kCalls = (kBits == 10) ? 4 : 2;     // Philox calls per token
                constexpr int kSteps = 8 / kCalls;                // k-steps covered by one call
#pragma unroll
                for (int gi = 0; gi < kCalls; ++gi) {
                    const uint4 da = philox(slot0 + g, c1, (uint32_t)(kCalls * c + gi), 0u, p.keys);
                    const uint4 db = philox(slot0 + g + 8, c1, (uint32_t)(kCalls * c + gi), 0u, p.keys);
#pragma unroll
                    for (int kk = 0; kk < kSteps; ++kk) {
                        const int ks = kSteps * gi + kk;
                        uint32_t A[4];
                        if constexpr (kBits == 8) {
                            const uint32_t xa = word_of(da, kk), xb = word_of(db, kk);
                            A[0] = h8(xa, kSel01);
                            A[1] = h8(xb, kSel01);
                            A[2] = h8(xa, kSel23);
                            A[3] = h8(xb, kSel23);
                        } else {
                            A[0] = h10(word_of(da, 2 * kk));
                            A[1] = h10(word_of(db, 2 * kk));
                            A[2] = h10(word_of(da, 2 * kk + 1));
                            A[3] = h10(word_of(db, 2 * kk + 1));
                        }
                        mma16816(dd, A, qw[2 * ks], qw[2 * ks + 1]);
                    }
                }
            }

            // ---------------- logits, bound, softmax ------------------------------
            float cb[4] = {0.f, 0.f, 0.f, 0.f};
            {
                const uint32_t wa = *reinterpret_cast<const uint32_t*>(st + kOffW + (g * kBands + 2 * c) * 2);
                const uint32_t wb = *reinterpret_cast<const uint32_t*>(st + kOffW + ((g + 8) * kBands + 2 * c) * 2);
                mma1688(cb, wa, wb, a_hi);
                mma1688(cb, wa, wb, a_lo);
            }
            float sk[2] = {1.f, 1.f}, sv[2] = {1.f, 1.f};   // tokens g, g+8
            if constexpr (kInt8) {
                const __half* ks = reinterpret_cast<const __half*>(st + kOffKs);
                const __half* vs = reinterpret_cast<const __half*>(st + kOffVs);
                sk[0] = __half2float(ks[g]); sk[1] = __half2float(ks[g + 8]);
                sv[0] = __half2float(vs[g]); sv[1] = __half2float(vs[g + 8]);
            }
            float y[4], P[4];
            const bool ok0 = g < nvalid, ok1 = g + 8 < nvalid;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = i >> 1, e = i & 1;
                const bool ok = r ? ok1 : ok0;
                const float raw = kInt8 ? (dc[i] - dd[i] + (e ? zoff1 : zoff0)) : dc[i];
                y[i] = ok ? raw * (sk[r] * kRsdLog2e) : -INFINITY;
                if (!ok) cb[i] = 0.f;                 // tail slots may hold any bits
            }
            if (!ok0) sv[0] = 0.f;
            if (!ok1) sv[1] = 0.f;
            if constexpr (kTierB) {
                if (!ok0) sk[0] = 0.f;
                if (!ok1) sk[1] = 0.f;
            }
            float rho[2] = {0.f, 0.f};   // value witness of tokens g, g+8 (0 past the context)
            if constexpr (kValue) {
                const float2 w0 = __half22float2(*reinterpret_cast<const __half2*>(st + kOffVw + 4 * g));
                const float2 w1 = __half22float2(*reinterpret_cast<const __half2*>(st + kOffVw + 4 * (g + 8)));
                if (ok0) { rho[0] = w0.x; vmax = fmaxf(vmax, w0.y); }
                if (ok1) { rho[1] = w1.x; vmax = fmaxf(vmax, w1.y); }
            }
            float mx0 = fmaxf(y[0], y[2]), mx1 = fmaxf(y[1], y[3]);
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
            }
            const bool mv0 = mx0 > m_run[0] + 8.0f, mv1 = mx1 > m_run[1] + 8.0f;
            if (__any_sync(0xffffffffu, mv0 || mv1)) {
                const float a0 = mv0 ? (m_run[0] == -INFINITY ? 0.f : fast_exp2(m_run[0] - mx0)) : 1.f;
                const float a1 = mv1 ? (m_run[1] == -INFINITY ? 0.f : fast_exp2(m_run[1] - mx1)) : 1.f;
                if (mv0) m_run[0] = mx0;
                if (mv1) m_run[1] = mx1;
                l_part[0] *= a0; d_part[0] *= a0; spv_part[0] *= a0;
                l_part[1] *= a1; d_part[1] *= a1; spv_part[1] *= a1;
                if constexpr (kTierB) { db_part[0] *= a0; db_part[1] *= a1; }
                if constexpr (kValue) { vt_part[0] *= a0; vt_part[1] *= a1; }
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    acc[mt][0] *= a0; acc[mt][2] *= a0;
                    acc[mt][1] *= a1; acc[mt][3] *= a1;
                }
            }
            float dpg[2] = {0.f, 0.f};   // this page's share of D (kRepair)
            float cl[4], ub[4];          // the bounds in log2 units (ub: Tier B)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                cl[i] = cb[i] * kLog2e;
                ub[i] = kTierB ? ((i & 1) ? alpha1 : alpha0) * sk[i >> 1] * kLog2e : 0.f;
            }
            bool huge;                   // warp-uniform: a bound of kHugeLog2 or more (meter_term)
            {
                float big = fmaxf(fmaxf(cl[0], cl[1]), fmaxf(cl[2], cl[3]));
                if constexpr (kTierB) big = fmaxf(big, fmaxf(fmaxf(ub[0], ub[1]), fmaxf(ub[2], ub[3])));
                huge = __any_sync(0xffffffffu, big >= kHugeLog2);
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = i >> 1, e = i & 1;
                const float pe = fast_exp2(y[i] - m_run[e]);     // 0 for masked tokens
                l_part[e] += pe;
                if (!huge) {
                    const float em1 = fast_exp2(cl[i]) - 1.f;
                    d_part[e] = fmaf(pe, em1, d_part[e]);
                    if constexpr (kRepair) dpg[e] = fmaf(pe, em1, dpg[e]);
                    if constexpr (kTierB) db_part[e] = fmaf(pe, fast_exp2(ub[i]) - 1.f, db_part[e]);
                }
                if constexpr (kValue) vt_part[e] = fmaf(pe, rho[r], vt_part[e]);
                P[i] = pe * sv[r];
                spv_part[e] += P[i];
            }
            if (huge) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = i & 1;
                    const float t = y[i] - m_run[e];
                    const float dt = meter_term(t, cl[i]);
                    d_part[e] += dt;
                    if constexpr (kRepair) dpg[e] += dt;
                    if constexpr (kTierB) db_part[e] += meter_term(t, ub[i]);
                }
            }
            if constexpr (kRepair) emit_page_terms(p, b, h, G, lp, g, c, dpg, m_run);
            if constexpr (kInt8) {
                const float smax = fmaxf(sv[0], sv[1]);
                const float wmax = __int_as_float(__reduce_max_sync(0xffffffffu, __float_as_int(smax)));
                if (wmax > 0.f) {
                    const int e = ((__float_as_int(wmax) >> 23) & 0xFF) - 126;   // wmax < 2^e
                    const int want = 6 - e;
                    if (lam_exp == INT_MIN) {
                        lam_exp = want;
                    } else if (want < lam_exp) {
                        const float f = pow2(want - lam_exp);
#pragma unroll
                        for (int mt = 0; mt < 8; ++mt)
#pragma unroll
                            for (int e2 = 0; e2 < 4; ++e2) acc[mt][e2] *= f;
                        lam_exp = want;
                    }
                }
            }
            // B = P^T for PV as two fp16 terms (hi + lo): the output is a sum with
            // heavy cancellation, one fp16 rounding of P is not accurate enough.
            // Packed as 8x8 blocks [token][head] (tokens 0-7 and 8-15) and
            // transposed with movmatrix into (P[tok 2c][head g], P[tok 2c+1][head g]).
            uint32_t bp0, bp1, bl0, bl1;
            {
                const float lam = pow2(lam_exp == INT_MIN ? 0 : lam_exp);
                const float x0 = P[0] * lam, x1 = P[1] * lam, x2 = P[2] * lam, x3 = P[3] * lam;
                const uint32_t h01 = pack_h2(x0, x1), h23 = pack_h2(x2, x3);
                const float2 r01 = __half22float2(*reinterpret_cast<const __half2*>(&h01));
                const float2 r23 = __half22float2(*reinterpret_cast<const __half2*>(&h23));
                const uint32_t l01 = pack_h2(x0 - r01.x, x1 - r01.y), l23 = pack_h2(x2 - r23.x, x3 - r23.y);
                bp0 = movmatrix_t(h01);
                bp1 = movmatrix_t(h23);
                bl0 = movmatrix_t(l01);
                bl1 = movmatrix_t(l23);
            }

            // ---------------- PV: acc[dim][head] ------------------------------------
            const int tv[4] = {2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9};
            uint4 vq[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                vq[j] = *reinterpret_cast<const uint4*>(kt + kTileRegion + swz(tv[j], g));
                // an fp8 NaN byte in an unused tail slot would poison P = 0 columns
                if (!kInt8 && tv[j] >= nvalid) vq[j] = make_uint4(0, 0, 0, 0);
            }
            if constexpr (kInt8) {
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    const int wi = mt >> 1, pos = 2 * (mt & 1);
                    uint32_t A[4];
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr) {
                        const uint32_t X = prmt(word_of(vq[2 * pr], wi) ^ 0x80808080u,
                                                word_of(vq[2 * pr + 1], wi) ^ 0x80808080u, sel_interleave(pos));
                        A[2 * pr] = s8x2_to_h2(X, kSel01);
                        A[2 * pr + 1] = s8x2_to_h2(X, kSel23);
                    }
                    mma16816(acc[mt], A, bp0, bp1);
                    mma16816(acc[mt], A, bl0, bl1);
                }
                const uint32_t bn0 = bp0 ^ 0x80008000u, bn1 = bp1 ^ 0x80008000u;
                const uint32_t bm0 = bl0 ^ 0x80008000u, bm1 = bl1 ^ 0x80008000u;
                constexpr int kHalves = (kBits == 10) ? 2 : 1;
#pragma unroll
                for (int hf = 0; hf < kHalves; ++hf) {
                    uint4 dv[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        dv[j] = philox(slot0 + tv[j], c1, (uint32_t)((kBits == 10) ? 2 * g + hf : g), 1u, p.keys);
#pragma unroll
                    for (int mm = 0; mm < 8 / kHalves; ++mm) {
                        const int mt = hf * (8 / kHalves) + mm;
                        const int wi = mt >> 1, pos = 2 * (mt & 1);
                        uint32_t H[4];
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            if constexpr (kBits == 8) {
                                const uint32_t Y = prmt(word_of(dv[2 * pr], wi), word_of(dv[2 * pr + 1], wi),
                                                        sel_interleave(pos));
                                H[2 * pr] = h8(Y, kSel01);
                                H[2 * pr + 1] = h8(Y, kSel23);
                            } else {
                                const uint32_t wa = word_of(dv[2 * pr], mt & 3), wb = word_of(dv[2 * pr + 1], mt & 3);
                                H[2 * pr] = h10(prmt(wa, wb, 0x5410u));
                                H[2 * pr + 1] = h10(prmt(wa, wb, 0x7632u));
                            }
                        }
                        mma16816(acc[mt], H, bn0, bn1);
                        mma16816(acc[mt], H, bm0, bm1);
                    }
                }
            } else {
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    const int wi = mt >> 1, pos = 2 * (mt & 1);
                    uint32_t A[4];
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr) {
                        const uint32_t X = prmt(word_of(vq[2 * pr], wi), word_of(vq[2 * pr + 1], wi),
                                                sel_interleave(pos));
                        A[2 * pr] = e4m3x2_to_h2(X);
                        A[2 * pr + 1] = e4m3x2_to_h2(X >> 16);
                    }
                    mma16816(acc[mt], A, bp0, bp1);
                    mma16816(acc[mt], A, bl0, bl1);
                }
            }
        } else if constexpr (kRepair) {
            emit_skipped_page(p, b, h, G, lp, lane);
        }
        __syncwarp();
        issue(k + kStages, phys_issue);
        if constexpr (kFlat) {
            if (k + kStages + 1 < n_my) dk_next<true>(p, iw);
            if (k + 1 < n_my) dk_next<true>(p, cw);
        }
#pragma unroll
        for (int i = 0; i + 1 < kStages; ++i) ring[i] = ring[i + 1];
        ring[kStages - 1] = phys_issue;
    }
    if (failed) {
        // let copies still in flight land before the CTA's smem is released
        for (int k = consumed; k < min(n_my, consumed + kStages); ++k)
            (void)mbar_wait_bounded(&bars[k % kStages], (uint32_t)((k / kStages) & 1));
    }

    if constexpr (kFlat) {
        if (n_my > 0) warp_rows(flat_partial());
        return;
    }

    // ---- CTA merge: warps -> shared, one partial per CTA -----------------------------
    __syncthreads();   // stage buffers are reused below
    float* mbuf = reinterpret_cast<float*>(smem);   // [warp][head][kPartialStride]
    warp_rows(mbuf + warp * kMaxGroup * kPartialStride);
    __syncthreads();
    const size_t unit = (size_t)b * p.num_kv_heads + h;
    float* part_out = p.partials + (unit * p.splits + split) * (kMaxGroup * kPartialStride);
    // thread -> (head, 4-dim chunk); chunk 32 carries (M, l, D)
    for (int idx = threadIdx.x; idx < G * 33; idx += kThreads) {
        const int hh = idx / 33, ch = idx % 33;
        float mw[kWarps];
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            mw[w] = mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim];
            M = fmaxf(M, mw[w]);
        }
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        const int col = (ch < 32) ? 4 * ch : kHeadDim + 1;   // chunk 32: l, D
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            if (mw[w] == -INFINITY) continue;   // a warp without pages: its values are not read
            const float wt = fast_exp2(mw[w] - M);
            const float* src = mbuf + (w * kMaxGroup + hh) * kPartialStride + col;
            if (ch < 32) {
                const float4 v = *reinterpret_cast<const float4*>(src);
                s.x = fmaf(wt, v.x, s.x); s.y = fmaf(wt, v.y, s.y);
                s.z = fmaf(wt, v.z, s.z); s.w = fmaf(wt, v.w, s.w);
            } else {
                s.x = fmaf(wt, src[0], s.x);   // l
                s.y = fmaf(wt, src[1], s.y);   // D
                if constexpr (kTierB) s.z = fmaf(wt, src[2], s.z);   // Tier-B D
                if constexpr (kValue) s.w = fmaf(wt, src[3], s.w);   // value term
            }
        }
        float* dst = part_out + hh * kPartialStride;
        if (ch < 32) {
            *reinterpret_cast<float4*>(dst + 4 * ch) = s;
        } else {
            dst[kHeadDim] = M;
            dst[kHeadDim + 1] = s.x;
            dst[kHeadDim + 2] = s.y;
            if constexpr (kTierB) dst[kHeadDim + 3] = s.z;
            if constexpr (kValue) {
                float vm = 0.f;
                for (int w = 0; w < kWarps; ++w)
                    vm = fmaxf(vm, mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim + 5]);
                dst[kHeadDim + 4] = s.w;
                dst[kHeadDim + 5] = vm;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Warp-specialized variant for the dithered INT8 cache with 8-bit dither.
//
// One CTA per SM with 8 consumer / 8 producer warp pairs.  Producer warp w
// serves consumer warp w through a 2-stage ring: it issues the page's copies
// (K and V code tiles by tensor-map TMA with the 128-byte swizzle, scales and
// witness by bulk copy) and regenerates the page's dither (Philox4x32-10) in
// registers, storing it as byte tiles j[token][channel] under the same
// swizzle, so the consumer reads dither words with the same conflict-free
// 16-byte shared loads as codes.  The consumer runs the attention, bound and
// meter math with no Philox on its path.  Per stage:
// `full` completes when the copies have landed and the dither tiles are
// written (two arrivals + the copy bytes); `empty` when the consumer has
// released it.  All waits are bounded.
// ---------------------------------------------------------------------------
constexpr int kWsPairs = 8;
// Built with -DWC_METER_OFF (a second library the benchmark loads to measure the
// certificate's cost, §8(d)): the warp-specialized decode then skips the
// witness copy, the bound MMAs and the meter accumulator; the meter it
// reports is not a bound.  The shipped library is built without it.
#ifdef WC_METER_OFF
constexpr bool kMeterOff = true;
#else
constexpr bool kMeterOff = false;
#endif
constexpr int kWsThreads = 64 * kWsPairs;
constexpr int kWsStages = 2;
constexpr int kWsOffK = 0;          // K codes [16][128], swizzled (1024-aligned)
constexpr int kWsOffV = 2048;       // V codes [16][128], swizzled
constexpr int kWsOffKd = 4096;      // K dither bytes [16][128], swizzled
constexpr int kWsOffVd = 6144;      // V dither bytes [16][128], swizzled
constexpr int kWsOffKs = 8192;      // K scales [16] fp16
constexpr int kWsOffVs = 8224;      // V scales [16] fp16
constexpr int kWsOffW = 8256;       // witness [16][8] fp16
constexpr int kWsOffHdr = 8512;     // physical page (or -1)
constexpr int kWsOffVw = 8528;      // value witness [16][2] fp16 (value side)
constexpr int kWsStageBytes = 9216;
static_assert(kWsOffVw + 64 <= kWsStageBytes && kWsStageBytes % 1024 == 0, "stage layout");
constexpr int kWsBarBytes = kWsPairs * kWsStages * 2 * 8;
constexpr int kWsSmemBytes = kWsPairs * kWsStages * kWsStageBytes + kWsBarBytes + 1024;   // + alignment slack
// flattened plan: the CTA merge's own buffer after the barriers
constexpr int kWsMergeOff = kWsPairs * kWsStages * kWsStageBytes + kWsBarBytes;
constexpr int kWsSmemFlat = kWsSmemBytes + kWsPairs * kMaxGroup * kPartialStride * 4;
static_assert(kWsMergeOff % 16 == 0 && kWsSmemFlat <= 232448, "flattened plan's shared memory");
static_assert(kWsSmemBytes <= 232448, "exceeds the per-CTA shared memory limit");
static_assert(kWsPairs * kMaxGroup * kPartialStride * 4 <= kWsPairs * kWsStages * kWsStageBytes, "merge buffer");

struct WsParams {
    CUtensorMap k_map;   // k_codes as [num_pages * Hkv][16][128] bytes, box = one page of one head
    CUtensorMap v_map;
    DecodeParams p;
    WriteParams w;       // the cache as the write path sees it (append variant)
};

// Append (kXAppend): the step's new token of sequence b, the last of its
// context, is quantized and stored by the producer warp that stages the
// sequence's last page, before it issues the copies of the segment that holds
// that page.  Its slot must
// be that of the context's last token (else WC_DEV_BAD_APPEND, not written),
// so no other CTA reads it.  Lanes 0-7 hold the row (write path layout); the
// generic-proxy stores are fenced against the async-proxy copies that follow.
__device__ __forceinline__ void append_new_token(const WsParams& wp, int b, int h, int phys, int ctx, int lane) {
    const DecodeParams& p = wp.p;
    const int slot = __ldg(p.slot_new + b);
    if (slot < 0) return;   // warp-uniform: no new token for this sequence
    if (slot != phys * kPage + (ctx - 1) % kPage) {
        if (lane == 0) atomicOr(p.status, WC_DEV_BAD_APPEND);
        return;
    }
    const bool live = lane < 8;
    const int sub = lane & 7;
    const size_t off = ((size_t)b * p.num_kv_heads + h) * kHeadDim + sub * 16;
    uint4 rk[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)}, rv[2] = {rk[0], rk[1]};
    if (live) {
        rk[0] = __ldg(reinterpret_cast<const uint4*>(p.k_new + off));
        rk[1] = __ldg(reinterpret_cast<const uint4*>(p.k_new + off) + 1);
        rv[0] = __ldg(reinterpret_cast<const uint4*>(p.v_new + off));
        rv[1] = __ldg(reinterpret_cast<const uint4*>(p.v_new + off) + 1);
    }
    write_row<WC_SCHEME_DITHER_INT8, 8>(wp.w, rk, slot, live, h, 0, sub, nullptr, nullptr);
    write_row<WC_SCHEME_DITHER_INT8, 8>(wp.w, rv, slot, live, h, 1, sub, nullptr, nullptr);
    asm volatile("fence.proxy.async.global;" ::: "memory");
    __syncwarp();
}

__device__ __forceinline__ void consumer_sync() {   // the 8 consumer warps only
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kWsPairs) : "memory");
}



template <int kX>
__global__ void __launch_bounds__(kWsThreads, 1) decode_ws_kernel(const __grid_constant__ WsParams wp) {
    constexpr bool kTierB = (kX & kXTierB) != 0, kValue = (kX & kXValue) != 0, kRepair = (kX & kXRepair) != 0;
    constexpr bool kAppend = (kX & kXAppend) != 0;
    constexpr bool kFlat = (kX & kXFlat) != 0;   // flattened split plan (pages_per_split == 0)
    constexpr bool kStall = (kX & kXStall) != 0;
    constexpr int kTries = kStall ? kStallTries : kMaxWaitTries;
    const DecodeParams& p = wp.p;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool producer = warp >= kWsPairs;
    const int pw = producer ? warp - kWsPairs : warp;     // pair index
    const int g = lane >> 2, c = lane & 3;
    const int G = p.group;
    constexpr float kKappa = DitherConst<8>::kappa;

    uint8_t* stages = smem + pw * kWsStages * kWsStageBytes;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kWsPairs * kWsStages * kWsStageBytes) + pw * 2 * kWsStages;
    uint64_t* empty = full + kWsStages;
    if (producer && lane == 0)
        for (int s = 0; s < kWsStages; ++s) {
            mbar_init(&full[s], 2);
            mbar_init(&empty[s], 1);
        }
    fence_barrier_init();
    __syncthreads();   // every barrier is initialised before any warp waits on it
    // the dependent merge may be scheduled now: it waits for this whole grid
    // (griddepcontrol.wait), and it launches only once every CTA of this grid
    // has started, so its CTAs never hold resources this grid still needs
    grid_dep_launch();
    if (!kFlat && lane == 0 && p.max_pages > 0) {
        // Split plan.  While the preceding kernel drains: warm L2 with this pair's
        // first page and the CTA's query rows.  The context length and page-table
        // entry read here may still be changing, so they serve only as prefetch
        // addresses (clamped into the cache); the loads bypass L1, which therefore
        // holds no copy that the reads after the wait could hit.
        const int b = blockIdx.z, h = blockIdx.y, p0 = blockIdx.x * p.pages_per_split;
        const int32_t* bt_row = p.block_table + (size_t)b * p.max_pages;
        if (producer) {
            const int ctx_hint = __ldcg(p.ctx_lens + b);
            if (p0 + pw < p.max_pages && (p0 + pw) * kPage < ctx_hint) {
                const int ph_hint = min(max(__ldcg(bt_row + p0 + pw), 0), p.num_pages - 1);
                const size_t z = (size_t)ph_hint * p.num_kv_heads + h;
                bulk_prefetch_l2(p.k_codes + z * (kPage * kHeadDim), kPage * kHeadDim);
                bulk_prefetch_l2(p.v_codes + z * (kPage * kHeadDim), kPage * kHeadDim);
                bulk_prefetch_l2(p.k_scale + z * kPage, 32);
                bulk_prefetch_l2(p.v_scale + z * kPage, 32);
                bulk_prefetch_l2(p.k_witness + z * (kPage * kBands), 256);
            }
        } else if (pw == 0) {
            bulk_prefetch_l2(p.q + ((size_t)b * p.num_q_heads + (size_t)h * G) * kHeadDim, G * kHeadDim * 2);
        }
    }
    grid_dep_wait();   // q, page tables and the cache may come from the preceding kernel

    // Split plan: this pair's first page-table entry and the consumer's query
    // fragment are loaded alongside the context length (both in bounds
    // whatever the length; used only if the pair has pages).
    int phys_first = -1;
    uint32_t qw[16];
    if constexpr (!kFlat) {
        if (producer && p.max_pages > 0)
            phys_first = __ldg(p.block_table + (size_t)blockIdx.z * p.max_pages +
                               min((int)blockIdx.x * p.pages_per_split + pw, p.max_pages - 1));
        if (!producer) load_q_frag(p, blockIdx.z, blockIdx.y, G, g, c, qw);
    }
    WsSeg sg;
    bool have;
    WsSeg* my_seg = nullptr;   // flattened plan: this warp's walker, in shared memory
    if constexpr (kFlat) {
        __shared__ int s_wtot[kWsThreads / 32];
        __shared__ long long s_start;
        __shared__ WsSeg s_seg[kWsThreads / 32];
        have = ws_first_segment<true>(p, sg, s_wtot, &s_start);
        my_seg = &s_seg[warp];
        if (lane == 0) *my_seg = sg;
        __syncwarp();
    } else {
        have = ws_first_segment<false>(p, sg, nullptr, nullptr);
    }

    if (producer) {
        int k = 0, issued = 0;   // stage ring position, continued across segments
        bool stop = false;
        // one segment's pages (the split plan has one segment: no loop around it)
        auto produce = [&](const WsSeg& cs) {
            const int b = cs.b, h = cs.h, ctx = cs.ctx, npages = cs.np;
            const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;
            const int32_t* bt_row = p.block_table + (size_t)b * p.max_pages;
            int first;
            const int n_seg = ws_seg_pages<kWsPairs>(cs, pw, first);
            int phys_next = kFlat ? (n_seg > 0 ? __ldg(bt_row + first) : -1) : phys_first;
            if constexpr (kAppend) {
                // The stream that stages the sequence's last page in this segment stores
                // the new token before the segment's first page (not inside the page
                // loop), so its write overlaps the other streams' pages and the loop
                // carries no write code.  Its copies are issued after the token's stores.
                const int lpl = npages - 1;
                if (n_seg > 0 && lpl >= first && (lpl - first) % kWsPairs == 0 && lpl < cs.e) {
                    const int phl = __ldg(bt_row + lpl);
                    if (phl >= 0 && phl < p.num_pages) append_new_token(wp, b, h, phl, ctx, lane);
                }
            }
            for (int i = 0; i < n_seg; ++i, ++k) {
                const int lp = first + kWsPairs * i;
                const int s = k % kWsStages;
                if (k >= kWsStages) {
                    const bool freed = mbar_wait_bounded<kTries>(&empty[s], (uint32_t)(((k / kWsStages) - 1) & 1));
                    if (!__all_sync(0xffffffffu, freed)) {
                        if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
                        stop = true;
                        break;
                    }
                }
                const int phys = phys_next;
                if (i + 1 < n_seg) phys_next = __ldg(bt_row + lp + kWsPairs);
                const bool ok = phys >= 0 && phys < p.num_pages;
                uint8_t* st = stages + s * kWsStageBytes;
                if constexpr (kStall) {   // failure-detection test: this page is never staged
                    if (lp == p.stall_page) {
                        issued = k + 1;
                        continue;
                    }
                }
                if (lane == 0) {
                    *reinterpret_cast<int*>(st + kWsOffHdr) = ok ? phys : -1;
                    if (ok) {
                        const int z = phys * p.num_kv_heads + h;
                        const size_t ph = (size_t)z;
                        mbar_arrive_expect_tx(&full[s],
                                              (uint32_t)(kStageBytes - (kMeterOff ? 256 : 0) + (kValue ? 64 : 0)));
                        tma_page(st + kWsOffK, &wp.k_map, z, &full[s]);
                        tma_page(st + kWsOffV, &wp.v_map, z, &full[s]);
                        bulk_g2s(st + kWsOffKs, p.k_scale + ph * kPage, 32, &full[s]);
                        bulk_g2s(st + kWsOffVs, p.v_scale + ph * kPage, 32, &full[s]);
                        if constexpr (!kMeterOff)
                            bulk_g2s(st + kWsOffW, p.k_witness + ph * (kPage * kBands), 256, &full[s]);
                        if constexpr (kValue) bulk_g2s(st + kWsOffVw, p.v_witness + ph * (kPage * 2), 64, &full[s]);
                    } else {
                        atomicOr(p.status, WC_DEV_BAD_PAGE);
                        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&full[s])) : "memory");
                    }
                }
                issued = k + 1;
                if (ok) {
                    // dither bytes j[token][channel]: one Philox call covers 16
                    // channels of one token (channel i = byte i%4 of word i/4).
                    // Each lane draws K and V for the same (token, channel group)
                    // (tokens g, g+8 x groups 2c, 2c+1), so the two calls share
                    // their first round's product.
                    const uint32_t slot0 = (uint32_t)phys * kPage;
                    uint4 dk[4], dv[4];
                    {   // call 2i: K, 2i+1: V of token g + 8 (i >> 1), group 2c + (i & 1)
                        uint32_t x0[8], x1[8], x2[8], x3[8];
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const int i = j >> 1;
                            x0[j] = slot0 + g + 8 * (i >> 1);
                            x1[j] = c1;
                            x2[j] = (uint32_t)(2 * c + (i & 1));
                            x3[j] = (uint32_t)(j & 1);
                        }
                        philox_n<8>(x0, x1, x2, x3, p.keys);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            dk[i] = make_uint4(x0[2 * i], x1[2 * i], x2[2 * i], x3[2 * i]);
                            dv[i] = make_uint4(x0[2 * i + 1], x1[2 * i + 1], x2[2 * i + 1], x3[2 * i + 1]);
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int off = swz(g + 8 * (i >> 1), 2 * c + (i & 1));
                        *reinterpret_cast<uint4*>(st + kWsOffKd + off) = dk[i];
                        *reinterpret_cast<uint4*>(st + kWsOffVd + off) = dv[i];
                    }
                }
                __syncwarp();
                if (lane == 0)   // second arrival: dither tiles and header are written
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&full[s])) : "memory");
            }
        };
        if constexpr (kFlat) {
            for (bool more = have; more && !stop; more = ws_step<kWsPairs, true>(p, my_seg, lane)) produce(*my_seg);
        } else {
            produce(sg);
        }
        // copies still in flight must land before the CTA's smem is released
        for (int j = max(0, issued - kWsStages); j < issued; ++j)
            (void)mbar_wait_bounded<kTries>(&full[j % kWsStages], (uint32_t)((j / kWsStages) & 1));
        return;
    }

    // ---------------------------- consumer warps ------------------------------------
    // The CTA merge's buffer [warp][head][kPartialStride]: the stage area in the
    // split plan (one segment, the producers are done with it), a buffer of its
    // own in the flattened plan (the producers stage the next segment meanwhile).
    float* mbuf = reinterpret_cast<float*>(kFlat ? smem + kWsMergeOff : smem);
    // Token rows: row g of the QK and softmax tiles holds token t0, row g + 8
    // token t1 (tok_row), so that the P fragment transposed by movmatrix pairs
    // tokens (4c, 4c+1) and (4c+2, 4c+3), as ldmatrix.trans delivers V.
    const int t0 = tok_row(g), t1 = tok_row(g + 8);
    int k = 0;   // stage ring position, continued across segments
    bool failed = false;
    // one segment: query setup, pages, CTA merge (the split plan has one segment)
    auto consume = [&](const WsSeg& cs) {
        const int b = cs.b, h = cs.h, ctx = cs.ctx;
        const bool row_valid = g < G;
        if constexpr (kFlat) load_q_frag(p, b, h, G, g, c, qw);
        float qsum = 0.f, part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&qw[i]));
            qsum += f.x + f.y;
            part[i >> 2] = fmaf(f.x, f.x, fmaf(f.y, f.y, part[i >> 2]));
        }
        qsum += __shfl_xor_sync(0xffffffffu, qsum, 1);
        qsum += __shfl_xor_sync(0xffffffffu, qsum, 2);
        // Tier B (§4.2): u_t = alpha s_t with alpha = sqrt(2 log(2S/delta) ||q||^2 / (12 d)),
        // for this thread's softmax heads 2c and 2c+1
        float alpha0 = 0.f, alpha1 = 0.f;
        if constexpr (kTierB) {
            float qn2 = part[0] + part[1] + part[2] + part[3];   // ||q_g||^2 over channels 32c .. 32c+31
            qn2 += __shfl_xor_sync(0xffffffffu, qn2, 1);
            qn2 += __shfl_xor_sync(0xffffffffu, qn2, 2);
            const float lg = p.tb_log_2_over_delta + logf((float)max(ctx, 1));   // log(2S / delta)
            const float al = sqrtf(2.0f * lg * qn2 * (1.0f / (12.0f * kHeadDim)));
            alpha0 = __shfl_sync(0xffffffffu, al, 8 * c);
            alpha1 = __shfl_sync(0xffffffffu, al, 8 * c + 4);
        }
        float band_a, band_b;
        if (p.rope_layout == WC_ROPE_HALF) {
#pragma unroll
            for (int i = 0; i < 4; ++i) part[i] += __shfl_xor_sync(0xffffffffu, part[i], 2);
            const int src = (lane & ~3) | (c >> 1);
            float v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) v[i] = __shfl_sync(0xffffffffu, part[i], src);
            band_a = (c & 1) ? v[2] : v[0];
            band_b = (c & 1) ? v[3] : v[1];
        } else {
            band_a = part[0] + part[1];
            band_b = part[2] + part[3];
        }
        uint32_t a_hi = 0, a_lo = 0;   // ||q_b|| log2(e) / sqrt(d), hi + lo: the bound in log2 units
        if (row_valid) {
            const float x0 = sqrtf(band_a) * kRsdLog2e, x1 = sqrtf(band_b) * kRsdLog2e;
            const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
            a_hi = pack_h2(__half2float(h0), __half2float(h1));
            a_lo = pack_h2(x0 - __half2float(h0), x1 - __half2float(h1));
        }
        const float zoff0 = kKappa * __shfl_sync(0xffffffffu, qsum, 8 * c);
        const float zoff1 = kKappa * __shfl_sync(0xffffffffu, qsum, 8 * c + 4);

        float m_run[2] = {-INFINITY, -INFINITY};
        float l_part[2] = {0.f, 0.f}, d_part[2] = {0.f, 0.f}, spv_part[2] = {0.f, 0.f};
        float db_part[2] = {0.f, 0.f};   // Tier-B meter accumulator (kTierB)
        float vt_part[2] = {0.f, 0.f};   // value side: sum p~ rho^v (kValue)
        float vmax = 0.f;                // value side: max ||v|| over this thread's tokens
        float acc[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
        int lam_exp = INT_MIN;
        float sv_lim = 1.17549435e-38f;   // 2^(6 - lam_exp); until the first positive scale, FLT_MIN

        int first;
        const int n_seg = ws_seg_pages<kWsPairs>(cs, pw, first);
        for (int i = 0; i < n_seg && !failed; ++i, ++k) {
            const int s = k % kWsStages;
            const bool landed = mbar_wait_bounded<kTries>(&full[s], (uint32_t)((k / kWsStages) & 1));
            if (!__all_sync(0xffffffffu, landed)) {
                if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
                failed = true;   // later pages are not waited for; the merges still run
                break;
            }
            const uint8_t* st = stages + s * kWsStageBytes;
            const int lp = first + kWsPairs * i;
            if (*reinterpret_cast<const int*>(st + kWsOffHdr) >= 0) {
                const int nvalid = min(kPage, ctx - lp * kPage);

                // ---------------- QK: S[token][head] = code.q - h'.q -------------------
                // Row g of the QK tile holds token t0, row g + 8 token t1 (see tok_row).
                float dc[4] = {0.f, 0.f, 0.f, 0.f}, dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int gp = 0; gp < 2; ++gp) {
                    const int q16 = 2 * c + gp;   // 16-byte chunk: channels 32c + 16gp .. +15
                    const uint4 ka = *reinterpret_cast<const uint4*>(st + kWsOffK + swz(t0, q16));
                    const uint4 kb = *reinterpret_cast<const uint4*>(st + kWsOffK + swz(t1, q16));
                    const uint4 ja = *reinterpret_cast<const uint4*>(st + kWsOffKd + swz(t0, q16));
                    const uint4 jb = *reinterpret_cast<const uint4*>(st + kWsOffKd + swz(t1, q16));
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const int ks = 4 * gp + kk;
                        const uint32_t xa = word_of(ka, kk) ^ 0x80808080u, xb = word_of(kb, kk) ^ 0x80808080u;
                        const uint32_t A[4] = {s8x2_to_h2(xa, kSel01), s8x2_to_h2(xb, kSel01), s8x2_to_h2(xa, kSel23),
                                               s8x2_to_h2(xb, kSel23)};
                        mma16816(dc, A, qw[2 * ks], qw[2 * ks + 1]);
                        const uint32_t ya = word_of(ja, kk), yb = word_of(jb, kk);
                        const uint32_t H[4] = {h8(ya, kSel01), h8(yb, kSel01), h8(ya, kSel23), h8(yb, kSel23)};
                        mma16816(dd, H, qw[2 * ks], qw[2 * ks + 1]);
                    }
                }

                // ---------------- logits, bound, softmax ------------------------------
                float cb[4] = {0.f, 0.f, 0.f, 0.f};   // log2-domain bound (a carries log2 e)
                if constexpr (!kMeterOff) {
                    const uint32_t wa = *reinterpret_cast<const uint32_t*>(st + kWsOffW + (t0 * kBands + 2 * c) * 2);
                    const uint32_t wb = *reinterpret_cast<const uint32_t*>(st + kWsOffW + (t1 * kBands + 2 * c) * 2);
                    mma1688(cb, wa, wb, a_hi);
                    mma1688(cb, wa, wb, a_lo);
                }
                const __half* ksc = reinterpret_cast<const __half*>(st + kWsOffKs);
                const __half* vsc = reinterpret_cast<const __half*>(st + kWsOffVs);
                float sk[2] = {__half2float(ksc[t0]), __half2float(ksc[t1])};
                float sv[2] = {__half2float(vsc[t0]), __half2float(vsc[t1])};
                float y[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = i >> 1, e = i & 1;
                    y[i] = (dc[i] - dd[i] + (e ? zoff1 : zoff0)) * (sk[r] * kRsdLog2e);
                }
                float rho[2] = {0.f, 0.f};   // value witness of tokens t0, t1 (0 past the context)
                if constexpr (kValue) {
                    const float2 w0 = __half22float2(*reinterpret_cast<const __half2*>(st + kWsOffVw + 4 * t0));
                    const float2 w1 = __half22float2(*reinterpret_cast<const __half2*>(st + kWsOffVw + 4 * t1));
                    rho[0] = w0.x;
                    rho[1] = w1.x;
                    if (nvalid == kPage) vmax = fmaxf(vmax, fmaxf(w0.y, w1.y));
                    else {
                        if (t0 < nvalid) vmax = fmaxf(vmax, w0.y);
                        if (t1 < nvalid) vmax = fmaxf(vmax, w1.y);
                    }
                }
                if (nvalid < kPage) {   // the context's last page (warp-uniform): slots past it hold any bits
                    const bool ok0 = t0 < nvalid, ok1 = t1 < nvalid;
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (!((i >> 1) ? ok1 : ok0)) {
                            y[i] = -INFINITY;
                            cb[i] = 0.f;
                        }
                    if (!ok0) sv[0] = sk[0] = rho[0] = 0.f;
                    if (!ok1) sv[1] = sk[1] = rho[1] = 0.f;
                }
                // running maximum, moved lazily: only when a logit exceeds it by more
                // than 8 (the column maximum over the token rows is reduced only then)
                {
                    float mx0 = fmaxf(y[0], y[2]), mx1 = fmaxf(y[1], y[3]);
                    if (__any_sync(0xffffffffu, mx0 > m_run[0] + 8.0f || mx1 > m_run[1] + 8.0f)) {
#pragma unroll
                        for (int o = 4; o < 32; o <<= 1) {
                            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
                            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
                        }
                        const bool mv0 = mx0 > m_run[0] + 8.0f, mv1 = mx1 > m_run[1] + 8.0f;
                        const float a0 = mv0 ? (m_run[0] == -INFINITY ? 0.f : fast_exp2(m_run[0] - mx0)) : 1.f;
                        const float a1 = mv1 ? (m_run[1] == -INFINITY ? 0.f : fast_exp2(m_run[1] - mx1)) : 1.f;
                        if (mv0) m_run[0] = mx0;
                        if (mv1) m_run[1] = mx1;
                        l_part[0] *= a0; d_part[0] *= a0; spv_part[0] *= a0;
                        l_part[1] *= a1; d_part[1] *= a1; spv_part[1] *= a1;
                        if constexpr (kTierB) { db_part[0] *= a0; db_part[1] *= a1; }
                        if constexpr (kValue) { vt_part[0] *= a0; vt_part[1] *= a1; }
#pragma unroll
                        for (int mt = 0; mt < 8; ++mt) {
                            acc[mt][0] *= a0; acc[mt][2] *= a0;
                            acc[mt][1] *= a1; acc[mt][3] *= a1;
                        }
                    }
                }
                // P * s_v * 2^lam_exp stays below 2^14 (fp16): s_v * 2^lam_exp < 2^6.
                // lam_exp only decreases; sv_lim = 2^(6 - lam_exp) is the scale at which it must.
                if (__any_sync(0xffffffffu, fmaxf(sv[0], sv[1]) >= sv_lim)) {
                    const float smax = fmaxf(sv[0], sv[1]);
                    const float wmax = __int_as_float(__reduce_max_sync(0xffffffffu, __float_as_int(smax)));
                    const int e = ((__float_as_int(wmax) >> 23) & 0xFF) - 126;   // wmax < 2^e
                    const int want = 6 - e;
                    if (lam_exp != INT_MIN) {   // want < lam_exp here
                        const float f = pow2(want - lam_exp);
#pragma unroll
                        for (int mt = 0; mt < 8; ++mt)
#pragma unroll
                            for (int e2 = 0; e2 < 4; ++e2) acc[mt][e2] *= f;
                        spv_part[0] *= f;
                        spv_part[1] *= f;
                    }
                    lam_exp = want;
                    sv_lim = pow2(6 - lam_exp);
                }
                const float lam = pow2(lam_exp == INT_MIN ? 0 : lam_exp);
                const float svl[2] = {sv[0] * lam, sv[1] * lam};   // exact: lam is a power of two
                float dpg[2] = {0.f, 0.f};   // this page's share of D (kRepair)
                float x[4];                  // P * s_v * lam, the PV operand
                float ub[4];                 // Tier-B bound in log2 units (kTierB)
#pragma unroll
                for (int i = 0; i < 4; ++i) ub[i] = kTierB ? ((i & 1) ? alpha1 : alpha0) * sk[i >> 1] * kLog2e : 0.f;
                bool huge = false;           // warp-uniform: a bound of kHugeLog2 or more (meter_term)
                if constexpr (!kMeterOff || kTierB) {
                    float big = kMeterOff ? 0.f : fmaxf(fmaxf(cb[0], cb[1]), fmaxf(cb[2], cb[3]));
                    if constexpr (kTierB) big = fmaxf(big, fmaxf(fmaxf(ub[0], ub[1]), fmaxf(ub[2], ub[3])));
                    huge = __any_sync(0xffffffffu, big >= kHugeLog2);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = i >> 1, e = i & 1;
                    const float pe = fast_exp2(y[i] - m_run[e]);
                    l_part[e] += pe;
                    if (!huge) {
                        if constexpr (!kMeterOff) {
                            const float em1 = fast_exp2(cb[i]) - 1.f;
                            d_part[e] = fmaf(pe, em1, d_part[e]);
                            if constexpr (kRepair) dpg[e] = fmaf(pe, em1, dpg[e]);
                        }
                        if constexpr (kTierB) db_part[e] = fmaf(pe, fast_exp2(ub[i]) - 1.f, db_part[e]);
                    }
                    if constexpr (kValue) vt_part[e] = fmaf(pe, rho[r], vt_part[e]);
                    x[i] = pe * svl[r];
                    spv_part[e] += x[i];     // sum P s_v, in the lam frame
                }
                if (huge) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int e = i & 1;
                        const float t = y[i] - m_run[e];
                        if constexpr (!kMeterOff) {
                            const float dt = meter_term(t, cb[i]);
                            d_part[e] += dt;
                            if constexpr (kRepair) dpg[e] += dt;
                        }
                        if constexpr (kTierB) db_part[e] += meter_term(t, ub[i]);
                    }
                }
                if constexpr (kRepair) emit_page_terms(p, b, h, G, lp, g, c, dpg, m_run);
                uint32_t bp0, bp1, bl0, bl1;
                {
                    const uint32_t h01 = pack_h2(x[0], x[1]), h23 = pack_h2(x[2], x[3]);
                    const float2 r01 = __half22float2(*reinterpret_cast<const __half2*>(&h01));
                    const float2 r23 = __half22float2(*reinterpret_cast<const __half2*>(&h23));
                    const uint32_t l01 = pack_h2(x[0] - r01.x, x[1] - r01.y), l23 = pack_h2(x[2] - r23.x, x[3] - r23.y);
                    // B operand: P[tokens 4c, 4c+1][head g] and P[tokens 4c+2, 4c+3][head g]
                    bp0 = movmatrix_t(h01);
                    bp1 = movmatrix_t(h23);
                    bl0 = movmatrix_t(l01);
                    bl1 = movmatrix_t(l23);
                }

                // ---------------- PV: acc[dim][head] += (code - h') P -----------------
                // ldmatrix.trans of a 16x16 byte block (tokens x dims 16mt..16mt+15)
                // gives lane (g, c) dims 16mt + g (first word) and 16mt + g + 8 (second)
                // at tokens 4c .. 4c+3: the A operand with k slots 2c, 2c+1, 2c+8,
                // 2c+9 holding tokens 4c .. 4c+3, the order B was built in.
#pragma unroll
                for (int mp = 0; mp < 4; ++mp) {   // m-tiles 2mp, 2mp+1
                    uint32_t v[4], j[4];
                    ldsm_t_b8_x2(v, st + kWsOffV + swz(lane & 15, 2 * mp + (lane >> 4)));
                    ldsm_t_b8_x2(j, st + kWsOffVd + swz(lane & 15, 2 * mp + (lane >> 4)));
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        const int mt = 2 * mp + u;
                        const uint32_t x0 = v[2 * u] ^ 0x80808080u, x1 = v[2 * u + 1] ^ 0x80808080u;
                        const uint32_t A[4] = {s8x2_to_h2(x0, kSel01), s8x2_to_h2(x1, kSel01), s8x2_to_h2(x0, kSel23),
                                               s8x2_to_h2(x1, kSel23)};
                        mma16816(acc[mt], A, bp0, bp1);
                        mma16816(acc[mt], A, bl0, bl1);
                        const uint32_t H[4] = {nh8(j[2 * u], kSel01), nh8(j[2 * u + 1], kSel01),
                                               nh8(j[2 * u], kSel23), nh8(j[2 * u + 1], kSel23)};
                        mma16816(acc[mt], H, bp0, bp1);
                        mma16816(acc[mt], H, bl0, bl1);
                    }
                }
            } else if constexpr (kRepair) {
                emit_skipped_page(p, b, h, G, lp, lane);
            }
            __syncwarp();
            if (lane == 0)   // release the stage to the producer
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&empty[s])) : "memory");
        }

        // ---- warp totals for heads 2c, 2c+1 (reduce over the token rows g) ----------------
#pragma unroll
        for (int o = 4; o < 32; o <<= 1)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                l_part[e] += __shfl_xor_sync(0xffffffffu, l_part[e], o);
                d_part[e] += __shfl_xor_sync(0xffffffffu, d_part[e], o);
                if constexpr (kTierB) db_part[e] += __shfl_xor_sync(0xffffffffu, db_part[e], o);
                if constexpr (kValue) vt_part[e] += __shfl_xor_sync(0xffffffffu, vt_part[e], o);
                spv_part[e] += __shfl_xor_sync(0xffffffffu, spv_part[e], o);
            }
        if constexpr (kValue)
            for (int o = 1; o < 32; o <<= 1) vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
        const float inv_lam = pow2(lam_exp == INT_MIN ? 0 : -lam_exp);

        // ---- CTA merge over the consumer warps: one partial per segment --------------------
        consumer_sync();   // all consumers are done with their stages and with mbuf's last use
        {
            float* wb = mbuf + pw * kMaxGroup * kPartialStride;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                float* row = wb + (2 * c + e) * kPartialStride;
                const float add = kKappa * spv_part[e] * inv_lam;   // spv is in the lam frame
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {   // m-tile rows g, g + 8: dims 16 mt + g, 16 mt + g + 8
                    row[16 * mt + g] = fmaf(acc[mt][e], inv_lam, add);
                    row[16 * mt + g + 8] = fmaf(acc[mt][e + 2], inv_lam, add);
                }
                if (g == 0) {
                    wb[(2 * c + e) * kPartialStride + kHeadDim + 0] = m_run[e];
                    wb[(2 * c + e) * kPartialStride + kHeadDim + 1] = l_part[e];
                    wb[(2 * c + e) * kPartialStride + kHeadDim + 2] = d_part[e];
                    if constexpr (kTierB) wb[(2 * c + e) * kPartialStride + kHeadDim + 3] = db_part[e];
                    if constexpr (kValue) {
                        wb[(2 * c + e) * kPartialStride + kHeadDim + 4] = vt_part[e];
                        wb[(2 * c + e) * kPartialStride + kHeadDim + 5] = vmax;
                    }
                }
            }
        }
        consumer_sync();
        const size_t unit = (size_t)b * p.num_kv_heads + h;
        // flattened plan: share j's segment of sequence b goes to partial h (shares + batch) + j + b
        const int shares = p.splits / p.num_kv_heads;
        const size_t pid = kFlat ? (size_t)h * (shares + p.batch) + blockIdx.x / p.num_kv_heads + b
                                 : unit * p.splits + blockIdx.x;
        float* part_out = p.partials + pid * (kMaxGroup * kPartialStride);
        for (int idx = threadIdx.x; idx < G * 33; idx += 32 * kWsPairs) {
            const int hh = idx / 33, ch = idx % 33;
            float mw[kWsPairs];
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kWsPairs; ++w) {
                mw[w] = mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim];
                M = fmaxf(M, mw[w]);
            }
            float4 s4 = make_float4(0.f, 0.f, 0.f, 0.f);
            const int col = (ch < 32) ? 4 * ch : kHeadDim + 1;
#pragma unroll
            for (int w = 0; w < kWsPairs; ++w) {
                if (mw[w] == -INFINITY) continue;   // a warp without pages: its values are not read
                const float wt = fast_exp2(mw[w] - M);
                const float* src = mbuf + (w * kMaxGroup + hh) * kPartialStride + col;
                if (ch < 32) {
                    const float4 v = *reinterpret_cast<const float4*>(src);
                    s4.x = fmaf(wt, v.x, s4.x); s4.y = fmaf(wt, v.y, s4.y);
                    s4.z = fmaf(wt, v.z, s4.z); s4.w = fmaf(wt, v.w, s4.w);
                } else {
                    s4.x = fmaf(wt, src[0], s4.x);
                    s4.y = fmaf(wt, src[1], s4.y);
                    if constexpr (kTierB) s4.z = fmaf(wt, src[2], s4.z);
                    if constexpr (kValue) s4.w = fmaf(wt, src[3], s4.w);
                }
            }
            float* dst = part_out + hh * kPartialStride;
            if (ch < 32) {
                *reinterpret_cast<float4*>(dst + 4 * ch) = s4;
            } else {
                dst[kHeadDim] = M;
                dst[kHeadDim + 1] = s4.x;
                dst[kHeadDim + 2] = s4.y;
                if constexpr (kTierB) dst[kHeadDim + 3] = s4.z;
                if constexpr (kValue) {
                    float vm = 0.f;
                    for (int w = 0; w < kWsPairs; ++w)
                        vm = fmaxf(vm, mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim + 5]);
                    dst[kHeadDim + 4] = s4.w;
                    dst[kHeadDim + 5] = vm;
                }
            }
        }
    };
    if constexpr (kFlat) {
        for (bool more = have; more; more = ws_step<kWsPairs, true>(p, my_seg, lane)) consume(*my_seg);
    } else {
        if (have) consume(sg);
    }
}

// Merge of the per-split partials of one (sequence, query head), 32 output
// dims per CTA: out = sum_s w_s acc_s / sum_s w_s l_s with w_s = 2^(m_s - M),
// D = sum_s w_s D_s / sum_s w_s l_s, meter_raw = D (D + 2) / 2 (§6.2.2: the
// meter accumulator merges under the same LSE weights as the output).  Each
// warp folds its splits with a running maximum in one pass.
constexpr int kMergeWarps = 8;

template <int kX>
__global__ void __launch_bounds__(32 * kMergeWarps) merge_kernel(const __grid_constant__ DecodeParams p) {
    grid_dep_launch();   // the next kernel waits for this grid before reading its outputs
    grid_dep_wait();
    const int chunk = blockIdx.x, hq = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int h = hq / p.group, hh = hq % p.group;
    const size_t unit = (size_t)b * p.num_kv_heads + h;
    const int count = p.splits;   // split plan with many splits (otherwise merge_warp_kernel)
    const float* base = p.partials + unit * p.splits * (kMaxGroup * kPartialStride) + hh * kPartialStride;
    const size_t split_stride = kMaxGroup * kPartialStride;
    __shared__ float red[kMergeWarps][38];

    // all of this warp's split rows of a round are loaded before any is
    // combined, so the loads overlap (one memory latency per round, not per split)
    constexpr int kMaxRows = 16;   // rows per warp and round
    constexpr bool tier_b = (kX & kXTierB) != 0, vside = (kX & kXValue) != 0, repair = (kX & kXRepair) != 0;
    float M = -INFINITY, acc = 0.f, L = 0.f, Dn = 0.f, Db = 0.f, Vt = 0.f, Vm = 0.f;
    for (int s0 = warp; s0 < count; s0 += kMergeWarps * kMaxRows) {
        float ms[kMaxRows], v[kMaxRows], ls[kMaxRows], ds[kMaxRows], dbs[kMaxRows], vts[kMaxRows];
#pragma unroll
        for (int i = 0; i < kMaxRows; ++i) {
            const int s = s0 + i * kMergeWarps;
            ms[i] = -INFINITY;
            v[i] = ls[i] = ds[i] = dbs[i] = vts[i] = 0.f;
            if (s < count) {
                const float* ps = base + s * split_stride;
                ms[i] = __ldcg(ps + kHeadDim);
                v[i] = __ldcg(ps + 32 * chunk + lane);
                ls[i] = __ldcg(ps + kHeadDim + 1);
                ds[i] = __ldcg(ps + kHeadDim + 2);
                if (tier_b) dbs[i] = __ldcg(ps + kHeadDim + 3);
                if (vside) {
                    vts[i] = __ldcg(ps + kHeadDim + 4);
                    Vm = fmaxf(Vm, __ldcg(ps + kHeadDim + 5));
                }
            }
        }
        float Mr = M;
#pragma unroll
        for (int i = 0; i < kMaxRows; ++i) Mr = fmaxf(Mr, ms[i]);
        if (Mr == -INFINITY) continue;
        if (Mr > M) {   // move the running sums to the new reference
            const float f = (M == -INFINITY) ? 0.f : fast_exp2(M - Mr);
            acc *= f; L *= f; Dn *= f; Db *= f; Vt *= f;
            M = Mr;
        }
#pragma unroll
        for (int i = 0; i < kMaxRows; ++i) {
            if (ms[i] == -INFINITY) continue;          // empty split: values not read
            const float w = fast_exp2(ms[i] - M);
            acc = fmaf(w, v[i], acc);
            L = fmaf(w, ls[i], L);
            Dn = fmaf(w, ds[i], Dn);
            Db = fmaf(w, dbs[i], Db);
            Vt = fmaf(w, vts[i], Vt);
        }
    }
    red[warp][lane] = acc;
    if (lane == 0) {
        red[warp][32] = M;
        red[warp][33] = L;
        red[warp][34] = Dn;
        red[warp][35] = Db;
        red[warp][36] = Vt;
        red[warp][37] = Vm;
    }
    __syncthreads();
    if (warp == 0) {
        float Mt = -INFINITY;
#pragma unroll
        for (int w = 0; w < kMergeWarps; ++w) Mt = fmaxf(Mt, red[w][32]);
        float a = 0.f, l = 0.f, dn = 0.f, db = 0.f, vt = 0.f, vm = 0.f;
        if (vside)
            for (int w = 0; w < kMergeWarps; ++w) vm = fmaxf(vm, red[w][37]);
        if (Mt != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kMergeWarps; ++w) {
                if (red[w][32] == -INFINITY) continue;
                const float f = fast_exp2(red[w][32] - Mt);
                a = fmaf(f, red[w][lane], a);
                l = fmaf(f, red[w][33], l);
                dn = fmaf(f, red[w][34], dn);
                db = fmaf(f, red[w][35], db);
                vt = fmaf(f, red[w][36], vt);
            }
        }
        const size_t cell = (size_t)b * p.num_q_heads + hq;
        p.out[cell * kHeadDim + 32 * chunk + lane] = l > 0.f ? a / l : 0.f;
        if (chunk == 0 && lane == 0) {
            float raw = 0.f;
            if (l > 0.f) {
                const float D = d_upper(dn / l);        // A - 1, rounded up
                raw = raw_or_inf(0.5f * D * (D + 2.0f));   // (A^2 - 1) / 2, +inf on overflow
            }
            p.meter_raw[cell] = raw;
            p.meter[cell] = fminf(1.0f, raw);
            if (repair) p.softmax_norm[cell] = make_float2(Mt, l);
            if (tier_b) {
                float rb = 0.f;
                if (l > 0.f) {
                    const float D = d_upper(db / l);
                    rb = raw_or_inf(0.5f * D * (D + 2.0f));
                }
                p.meter_b_raw[cell] = rb;
                p.meter_b[cell] = fminf(1.0f, rb);
            }
            if (vside) {   // ||y - y^|| <= 2 TV max ||v|| + sum p~ rho^v, TV <= meter
                const float vterm = l > 0.f ? vt / l * kDRel : 0.f;   // rounded up like D
                p.value_term[cell] = vterm;
                p.v_max[cell] = vm;
                p.out_bound[cell] = 2.0f * fminf(1.0f, raw) * vm + vterm;
            }
        }
    }
}

}  // namespace

static bool use_ws(int scheme, int bits) { return scheme == WC_SCHEME_DITHER_INT8 && bits == 8; }

// Resident decode CTAs per SM: the warp-specialized kernel and the grouped
// kernel take a whole SM, the per-token kernel two CTAs.
static int ctas_per_sm(int scheme, int bits) {
    return (use_ws(scheme, bits) || scheme == WC_SCHEME_DITHER_INT8_G32) ? 1 : kMinBlocks;
}

// Page streams per CTA: warps, or warp pairs.
static long streams_per_cta(int scheme) { return scheme == WC_SCHEME_DITHER_INT8_G32 ? kG32PageStreams : 8; }

// Split plan.  A CTA's n page streams each take every n-th page of its split,
// so a split of P pages costs ceil(P / n) page steps, and a wave of resident
// CTAs adds a fixed prologue / epilogue of about one and a half page steps.
// The split count minimises
//     waves * (ceil(pages_per_split / n) + 1.5),   waves = ceil(CTAs / resident CTAs),
// so a grid never spills a small remainder into an extra wave; splits keep at
// least n pages (one per stream).  Ties go to fewer splits (less to merge).
DecodePlan plan_decode(int batch, int num_kv_heads, int max_pages, int num_sms, int scheme, int bits) {
    DecodePlan pl;
    const long units = (long)batch * num_kv_heads;
    const long slots = std::max<long>(1, (long)num_sms * ctas_per_sm(scheme, bits));
    const long kStreams = streams_per_cta(scheme);
    constexpr long kWaveCost2 = 3;    // per-wave fixed cost, in half page steps
    const long max_splits = std::max<long>(1, std::min<long>(max_pages / kStreams, 4 * slots));
    long best_pps = std::max(max_pages, 1), best_cost = -1;
    for (long sp = 1; sp <= max_splits; ++sp) {
        const long pps = (max_pages + sp - 1) / sp;
        const long splits = (max_pages + pps - 1) / pps;
        if (splits != sp) continue;   // same plan as a smaller split count
        const long waves = (splits * units + slots - 1) / slots;
        const long cost = waves * (2 * ((pps + kStreams - 1) / kStreams) + kWaveCost2);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best_pps = pps;
        }
    }
    pl.pages_per_split = (int)best_pps;
    pl.splits = (int)std::max<long>(1, (max_pages + best_pps - 1) / best_pps);
    long partials = units * pl.splits;
    // A batch of several sequences (lengths unknown to the host, often ragged)
    // takes the flattened plan: Hkv x floor(resident CTAs / Hkv) CTAs, all
    // resident, each taking equal shares of one KV head's pages; a share per CTA
    // for the warp-specialized kernels (one CTA per SM), a share per warp for
    // the per-token kernel (two CTAs of 8 warps per SM).  The per-token kernel
    // takes it only for the 10-bit dither and only when the split plan would
    // leave resident CTA slots empty: a warp's share ends in a partial of its
    // own (4.5 KB), which costs less than the idle SMs only where pages are
    // expensive (the dither regenerated in the warp); split-plan CTAs are
    // scheduled as SMs free up, which already evens out a ragged batch that
    // fills a wave, and fp8 pages are cheap.
    const bool per_warp = ctas_per_sm(scheme, bits) > 1;
    const bool flat_ok = !per_warp || (scheme == WC_SCHEME_DITHER_INT8 && pl.splits * units < slots);
    if (batch > 1 && (long long)batch * max_pages < (1LL << 31) && flat_ok) {
        const int ctas = num_kv_heads * std::max(1, (int)(slots / num_kv_heads));
        pl.splits = per_warp ? ctas * kWarps : ctas;   // shares: the merge reads splits / Hkv per head
        pl.pages_per_split = 0;
        partials = pl.splits + units;
    }
    auto align = [](size_t x) { return (x + 255) & ~(size_t)255; };
    pl.partials_off = 256;
    pl.total = align(pl.partials_off + sizeof(float) * (size_t)partials * kMaxGroup * kPartialStride);
    return pl;
}

// The merge is launched early (programmatic dependent) and its CTAs become
// resident on the SMs the decode grid frees first.  When the merge grid fits
// in one wave, each CTA also reserves more than half of an SM's shared memory
// (unused), so no two share an SM and the merge runs spread over the GPU
// instead of packed onto the first few SMs to free up.
constexpr int kMergeSpreadSmem = 118784;

// Merge where a unit has only a few partials: the flattened plan (its
// sequence's cuts) and a split plan of at most kWarpMergeSplits splits (a
// batch of sequences on the per-token kernel).  One warp per (sequence, query
// head, 32 output dims) folds all of them in order with the same
// running-maximum update as merge_kernel, so a CTA of 8 warps serves 8 outputs
// and needs no block barrier, and a batch's merge is one wave of short warps
// rather than several waves of CTAs with a block reduction each.
constexpr int kWarpMergeSplits = 8;

template <int kX>
__global__ void __launch_bounds__(32 * kMergeWarps) merge_warp_kernel(const __grid_constant__ DecodeParams p) {
    grid_dep_launch();   // the next kernel waits for this grid before reading its outputs
    grid_dep_wait();
    const int lane = threadIdx.x & 31;
    const long long item = (long long)blockIdx.x * kMergeWarps + (threadIdx.x >> 5);
    if (item >= (long long)p.batch * p.num_q_heads * (kHeadDim / 32)) return;   // warp-uniform
    const int chunk = (int)(item % (kHeadDim / 32));
    const int hq = (int)((item / (kHeadDim / 32)) % p.num_q_heads);
    const int b = (int)(item / ((kHeadDim / 32) * p.num_q_heads));
    const int h = hq / p.group, hh = hq % p.group;
    constexpr bool tier_b = (kX & kXTierB) != 0, vside = (kX & kXValue) != 0, repair = (kX & kXRepair) != 0;

    const int nb = (max(0, min(__ldg(p.ctx_lens + b), p.max_pages * kPage)) + kPage - 1) / kPage;
    int count;
    const float* base;
    if (p.pages_per_split > 0) {
        // Split plan: the unit's splits are consecutive; those past the
        // sequence's last page hold no pages (their maximum is -inf) and are
        // not read.
        count = min(p.splits, (nb + p.pages_per_split - 1) / p.pages_per_split);
        base = p.partials + ((size_t)b * p.num_kv_heads + h) * p.splits * (kMaxGroup * kPartialStride) +
               hh * kPartialStride;
    } else {
        // Flattened plan.  The batch's pages lie end to end (sequence b from
        // P_b = sum_{b' < b} n_b', page counts of the clamped context lengths, as
        // in the decode); share j of the splits / Hkv shares took positions
        // [j R, (j + 1) R), R = ceil(total / shares), in each head, so the unit's
        // segments are those of shares P_b / R .. (P_b + n_b - 1) / R, stored at
        // partials h (shares + batch) + j + b, consecutive.
        int before = 0, total = 0;
        for (int i = lane; i < p.batch; i += 32) {
            const int np = (max(0, min(__ldg(p.ctx_lens + i), p.max_pages * kPage)) + kPage - 1) / kPage;
            total += np;
            if (i < b) before += np;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            before += __shfl_xor_sync(0xffffffffu, before, o);
            total += __shfl_xor_sync(0xffffffffu, total, o);
        }
        const int shares = max(1, p.splits / p.num_kv_heads);
        const long long R = max(1LL, ((long long)total + shares - 1) / shares);
        const long long j0 = before / R;
        count = nb > 0 ? (int)(((long long)before + nb - 1) / R - j0 + 1) : 0;
        base = p.partials + ((size_t)h * (shares + p.batch) + (size_t)(j0 + b)) * (kMaxGroup * kPartialStride) +
               hh * kPartialStride;
    }

    constexpr int kRows = 8;   // rows loaded per round before any is combined
    float M = -INFINITY, acc = 0.f, L = 0.f, Dn = 0.f, Db = 0.f, Vt = 0.f, Vm = 0.f;
    for (int s0 = 0; s0 < count; s0 += kRows) {
        float ms[kRows], v[kRows], ls[kRows], ds[kRows], dbs[kRows], vts[kRows];
#pragma unroll
        for (int i = 0; i < kRows; ++i) {
            ms[i] = -INFINITY;
            v[i] = ls[i] = ds[i] = dbs[i] = vts[i] = 0.f;
            if (s0 + i < count) {
                const float* ps = base + (size_t)(s0 + i) * (kMaxGroup * kPartialStride);
                ms[i] = __ldcg(ps + kHeadDim);
                v[i] = __ldcg(ps + 32 * chunk + lane);
                ls[i] = __ldcg(ps + kHeadDim + 1);
                ds[i] = __ldcg(ps + kHeadDim + 2);
                if (tier_b) dbs[i] = __ldcg(ps + kHeadDim + 3);
                if (vside) {
                    vts[i] = __ldcg(ps + kHeadDim + 4);
                    Vm = fmaxf(Vm, __ldcg(ps + kHeadDim + 5));
                }
            }
        }
        float Mr = M;
#pragma unroll
        for (int i = 0; i < kRows; ++i) Mr = fmaxf(Mr, ms[i]);
        if (Mr == -INFINITY) continue;
        if (Mr > M) {
            const float f = (M == -INFINITY) ? 0.f : fast_exp2(M - Mr);
            acc *= f; L *= f; Dn *= f; Db *= f; Vt *= f;
            M = Mr;
        }
#pragma unroll
        for (int i = 0; i < kRows; ++i) {
            if (ms[i] == -INFINITY) continue;
            const float w = fast_exp2(ms[i] - M);
            acc = fmaf(w, v[i], acc);
            L = fmaf(w, ls[i], L);
            Dn = fmaf(w, ds[i], Dn);
            Db = fmaf(w, dbs[i], Db);
            Vt = fmaf(w, vts[i], Vt);
        }
    }
    const size_t cell = (size_t)b * p.num_q_heads + hq;
    p.out[cell * kHeadDim + 32 * chunk + lane] = L > 0.f ? acc / L : 0.f;
    if (chunk == 0 && lane == 0) {
        float raw = 0.f;
        if (L > 0.f) {
            const float D = d_upper(Dn / L);
            raw = raw_or_inf(0.5f * D * (D + 2.0f));
        }
        p.meter_raw[cell] = raw;
        p.meter[cell] = fminf(1.0f, raw);
        if (repair) p.softmax_norm[cell] = make_float2(M, L);
        if (tier_b) {
            float rb = 0.f;
            if (L > 0.f) {
                const float D = d_upper(Db / L);
                rb = raw_or_inf(0.5f * D * (D + 2.0f));
            }
            p.meter_b_raw[cell] = rb;
            p.meter_b[cell] = fminf(1.0f, rb);
        }
        if (vside) {
            const float vterm = L > 0.f ? Vt / L * kDRel : 0.f;
            p.value_term[cell] = vterm;
            p.v_max[cell] = Vm;
            p.out_bound[cell] = 2.0f * fminf(1.0f, raw) * Vm + vterm;
        }
    }
}

template <int kX>
static cudaError_t launch_merge(const DecodeParams& p, cudaStream_t stream) {
    static std::once_flag once;
    static int num_sms = 0;   // 0: the spread request is not used
    std::call_once(once, [] {
        int dev = 0, n = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
            cudaFuncSetAttribute(merge_kernel<kX>, cudaFuncAttributeMaxDynamicSharedMemorySize, kMergeSpreadSmem) ==
                cudaSuccess)
            num_sms = n;
        (void)cudaFuncSetAttribute(merge_kernel<kX>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                   (int)cudaSharedmemCarveoutMaxShared);
        (void)cudaGetLastError();   // a refused hint leaves no sticky error behind
    });
    if (p.pages_per_split == 0 || p.splits <= kWarpMergeSplits) {   // a few partials per unit
        const long warps = (long)p.batch * p.num_q_heads * (kHeadDim / 32);
        return launch_pdl(merge_warp_kernel<kX>, dim3((unsigned)((warps + kMergeWarps - 1) / kMergeWarps)),
                          dim3(32 * kMergeWarps), 0, stream, p);
    }
    const dim3 grid(kHeadDim / 32, p.num_q_heads, p.batch);
    const long ctas = (long)grid.x * grid.y * grid.z;
    const size_t smem = (num_sms > 0 && ctas <= num_sms) ? kMergeSpreadSmem : 0;
    return launch_pdl(merge_kernel<kX>, grid, dim3(32 * kMergeWarps), smem, stream, p);
}

cudaError_t launch_merge_x(const DecodeParams& p, int x, cudaStream_t stream) {
    return x == kXTierB ? launch_merge<kXTierB>(p, stream)
         : x == kXValue ? launch_merge<kXValue>(p, stream)
         : x == kXRepair ? launch_merge<kXRepair>(p, stream) : launch_merge<0>(p, stream);
}

template <int kScheme, int kBits, int kX>
static cudaError_t launch_one(const DecodeParams& p, cudaStream_t stream) {
    static bool configured = false;   // per process; the attributes are per function
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_kernel<kScheme, kBits, kX>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return e;
        // the library's kernels all prefer the largest shared-memory carveout,
        // so consecutive launches do not reconfigure the L1 / shared split
        e = cudaFuncSetAttribute(decode_kernel<kScheme, kBits, kX>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    DkParams dp;
    dp.p = p;
    if (!encode_page_map(&dp.k_map, p.k_codes, p.num_pages, p.num_kv_heads) ||
        !encode_page_map(&dp.v_map, p.v_codes, p.num_pages, p.num_kv_heads))
        return cudaErrorInvalidValue;
    // split plan: (splits, Hkv, batch); flattened plan: one CTA per 8 warp shares
    const dim3 grid = (kX & kXFlat) ? dim3(p.splits / kWarps) : dim3(p.splits, p.num_kv_heads, p.batch);
    cudaError_t e = launch_pdl(decode_kernel<kScheme, kBits, kX>, grid, dim3(kThreads), kSmemBytes, stream, dp);
    if (e != cudaSuccess) return e;
    // the merge is a programmatic dependent too: its CTAs are scheduled while
    // the decode grid drains and wait (griddepcontrol.wait) for all of it
    return launch_merge<kX & ~kXFlat>(p, stream);
}

// The per-token kernel for the extras in x (Tier B only with the dither).
template <int kScheme, int kBits, int kF>
static cudaError_t launch_one_x(const DecodeParams& p, int x, cudaStream_t stream) {
    if constexpr (kScheme == WC_SCHEME_FP8_E4M3) {
        return x == kXValue  ? launch_one<kScheme, kBits, kXValue | kF>(p, stream)
             : x == kXRepair ? launch_one<kScheme, kBits, kXRepair | kF>(p, stream)
                             : launch_one<kScheme, kBits, kF>(p, stream);
    } else {
        return x == kXTierB  ? launch_one<kScheme, kBits, kXTierB | kF>(p, stream)
             : x == kXValue  ? launch_one<kScheme, kBits, kXValue | kF>(p, stream)
             : x == kXRepair ? launch_one<kScheme, kBits, kXRepair | kF>(p, stream)
                             : launch_one<kScheme, kBits, kF>(p, stream);
    }
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (the
// library does not link the driver library itself).
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}

// One layer's code array [num_pages][Hkv][16][128] bytes as a 3-D tensor
// (channel, slot, page * Hkv + head); a box is one page of one head, written
// to shared memory with the 128-byte swizzle.
bool encode_page_map(CUtensorMap* map, const void* codes, int num_pages, int num_kv_heads) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return false;
    const cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)kPage, (cuuint64_t)num_pages * num_kv_heads};
    const cuuint64_t strides[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)kHeadDim * kPage};
    const cuuint32_t box[3] = {(cuuint32_t)kHeadDim, (cuuint32_t)kPage, 1};
    const cuuint32_t elem[3] = {1, 1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void*>(codes), dims, strides, box, elem,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int kX>
static cudaError_t launch_ws(const DecodeParams& p, cudaStream_t stream) {
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_ws_kernel<kX>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kWsSmemFlat);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(decode_ws_kernel<kX>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    WsParams wp;
    wp.p = p;
    if constexpr ((kX & kXAppend) != 0) {   // the cache as the write path sees it
        WriteParams& w = wp.w;
        w.k = w.v = nullptr;
        w.slot_mapping = p.slot_new;
        w.k_codes = const_cast<uint8_t*>(p.k_codes);
        w.v_codes = const_cast<uint8_t*>(p.v_codes);
        w.k_scale = const_cast<__half*>(p.k_scale);
        w.v_scale = const_cast<__half*>(p.v_scale);
        w.k_witness = const_cast<__half*>(p.k_witness);
        w.v_witness = nullptr;
        w.dev_status = p.status;
        w.n_tok = p.batch;
        w.num_kv_heads = p.num_kv_heads;
        w.num_pages = p.num_pages;
        w.layer = p.layer;
        w.rope_layout = p.rope_layout;
        w.keys = p.keys;
    }
    if (!encode_page_map(&wp.k_map, p.k_codes, p.num_pages, p.num_kv_heads) ||
        !encode_page_map(&wp.v_map, p.v_codes, p.num_pages, p.num_kv_heads))
        return cudaErrorInvalidValue;
    const bool flat = p.pages_per_split == 0;
    const dim3 grid = flat ? dim3(p.splits, 1, 1) : dim3(p.splits, p.num_kv_heads, p.batch);
    cudaError_t e = launch_pdl(decode_ws_kernel<kX>, grid, dim3(kWsThreads), flat ? kWsSmemFlat : kWsSmemBytes, stream, wp);
    if (e != cudaSuccess) return e;
    return launch_merge<kX & ~(kXAppend | kXFlat | kXStall)>(p, stream);
}

template <int kF>
static cudaError_t launch_ws_x(const DecodeParams& p, int x, cudaStream_t stream) {
    return x == kXTierB  ? launch_ws<kXTierB | kF>(p, stream)
         : x == kXValue  ? launch_ws<kXValue | kF>(p, stream)
         : x == kXRepair ? launch_ws<kXRepair | kF>(p, stream)
         : x == kXAppend ? launch_ws<kXAppend | kF>(p, stream) : launch_ws<kF>(p, stream);
}

cudaError_t launch_decode(const DecodeParams& p, int scheme, int bits, cudaStream_t stream) {
    if (p.batch == 0) return cudaSuccess;
    if (scheme == WC_SCHEME_DITHER_INT8_G32) return launch_decode_g32(p, stream);
    // Tier B (dithered INT8 only), the value side and the repair terms are
    // requested by separate entry points, never together (checked by the caller)
    const int x = (p.meter_b ? kXTierB : 0) | (p.value_term ? kXValue : 0) | (p.page_terms ? kXRepair : 0) |
                  (p.k_new ? kXAppend : 0);
    if (scheme == WC_SCHEME_FP8_E4M3)   // always the split plan (plan_decode)
        return p.pages_per_split == 0 ? cudaErrorNotSupported : launch_one_x<WC_SCHEME_FP8_E4M3, 8, 0>(p, x, stream);
    if (p.stall_page >= 0)   // failure-detection test (checked by the caller: 8-bit dither, no extras)
        return use_ws(scheme, bits) && p.pages_per_split > 0 && x == 0 ? launch_ws<kXStall>(p, stream)
                                                                        : cudaErrorNotSupported;
    if (use_ws(scheme, bits))   // pages_per_split == 0: the flattened plan
        return p.pages_per_split == 0 ? launch_ws_x<kXFlat>(p, x, stream) : launch_ws_x<0>(p, x, stream);
    return p.pages_per_split == 0 ? launch_one_x<WC_SCHEME_DITHER_INT8, 10, kXFlat>(p, x, stream)
                                  : launch_one_x<WC_SCHEME_DITHER_INT8, 10, 0>(p, x, stream);
}

}  // namespace wc
