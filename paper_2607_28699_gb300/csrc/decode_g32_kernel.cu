// Metered decode attention over the grouped-scale cache (§6.2.3 "Storage
// side" and §6.2.5 "Fixed-channel outlier bypass"): one fp16 scale per token and
// 32-channel group, and the m key RoPE pairs of a (layer, KV head) stored
// exactly.  Warp-specialized like the per-token kernel: 6 producer / 6 consumer
// warp pairs per CTA, one CTA per SM (at 384 threads the consumer keeps its ~165
// registers without spilling; 8 pairs with a producer -> consumer register
// split measured slower).  A producer stages a page (code tiles by TMA with the
// 128-byte swizzle; scales, witness and bypass values by bulk copy) and
// regenerates its dither into swizzled byte tiles; its consumer runs the math
// below with no Philox on its path.  The split plans (one sequence: equal
// splits; a batch: the flattened plan's per-head shares, walked as segments),
// the split-K partials and the merges are the per-token kernel's.  What differs
// from the per-token math:
//
//  - A row is stored in the order the mma fragments consume it (storage
//    position p of K holds channel 16 ((p >> 2) & 7) + 4 (p >> 5) + (p & 3),
//    of V channel 16 ((p >> 1) & 7) + 8 (p & 1) + (p >> 4)), with the dither
//    drawn by storage position.  So the code and dither tiles are the
//    per-token kernel's, while every QK k-step and every PV m-tile meets a
//    single channel group.
//  - QK: the q operand is gathered in that order, with the bypassed channels
//    zeroed; after the two k-steps of a group the accumulators are folded,
//    raw += s_g (code.q - h'.q + kappa sum_g q), and the exact bypassed
//    values enter through one m16n8k8 mma per 8 bypassed dims.
//  - PV: one P operand per group (P s_g, hi + lo), and the kappa term per
//    group; the output rows of m-tile mt are channels 16 mt .. 16 mt + 15.
//  - Tier B (§4.2) with the grouped proxy
//    varsigma_t^2 = (1/(12 d)) sum_g ||q_g'||^2 s_{g,t}^2 (bypassed channels left out).
#include "decode_common.cuh"

namespace wc {

namespace {

constexpr int kGMaxBypass = 16;

struct G32Params {
    CUtensorMap k_map;   // k_codes as [num_pages * Hkv][16][128] bytes, box = one page of one head
    CUtensorMap v_map;
    DecodeParams p;
};

constexpr int kGwPairs = kG32PageStreams;
constexpr int kGwThreads = 64 * kGwPairs;
constexpr int kGwStages = 2;
// stage: K codes | V codes | K dither | V dither (16 x 128 bytes each, swizzled) |
// K scales [16][4] | V scales [16][4] | witness [16][8] | bypass [16][2m] | header
constexpr int kGwOffK = 0, kGwOffV = 2048, kGwOffKd = 4096, kGwOffVd = 6144;
constexpr int kGwOffKs = 8192, kGwOffVs = 8320, kGwOffW = 8448, kGwOffB = 8704, kGwOffHdr = 9728;
constexpr int kGwStageBytes = 10240;
static_assert(kGwOffB + 16 * 2 * kGMaxBypass * 2 <= kGwOffHdr && kGwOffHdr + 16 <= kGwStageBytes, "stage layout");
constexpr int kGwSmemBytes = kGwPairs * kGwStages * kGwStageBytes + kGwPairs * kGwStages * 2 * 8 + 1024;
// flattened plan: the CTA merge's own buffer after the barriers
constexpr int kGwMergeOff = kGwPairs * kGwStages * kGwStageBytes + kGwPairs * kGwStages * 2 * 8;
constexpr int kGwSmemFlat = kGwSmemBytes + kGwPairs * kMaxGroup * kPartialStride * 4;
static_assert(kGwMergeOff % 16 == 0 && kGwSmemFlat <= 232448, "flattened plan's shared memory");
static_assert(kGwPairs * kMaxGroup * kPartialStride * 4 <= kGwPairs * kGwStages * kGwStageBytes, "merge buffer");
static_assert(kGwSmemBytes <= 232448, "exceeds the per-CTA shared memory limit");

__device__ __forceinline__ void gw_consumer_sync() {   // the consumer warps only
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kGwPairs) : "memory");
}

template <int kX>
__global__ void __launch_bounds__(kGwThreads, 1) decode_g32_ws_kernel(const __grid_constant__ G32Params gparams) {
    constexpr bool kTierB = (kX & kXTierB) != 0;
    constexpr bool kFlat = (kX & kXFlat) != 0;   // flattened split plan (pages_per_split == 0)
    constexpr float kKappa = DitherConst<8>::kappa;
    const DecodeParams& p = gparams.p;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const bool producer = warp >= kGwPairs;
    const int pw = producer ? warp - kGwPairs : warp;
    const int g = lane >> 2, c = lane & 3;
    const int G = p.group;
    const int m = p.num_bypass, nb = 2 * m;

    uint8_t* stages = smem + pw * kGwStages * kGwStageBytes;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + kGwPairs * kGwStages * kGwStageBytes) + pw * 2 * kGwStages;
    uint64_t* empty = full + kGwStages;
    if (producer && lane == 0)
        for (int s = 0; s < kGwStages; ++s) {
            mbar_init(&full[s], 2);
            mbar_init(&empty[s], 1);
        }
    fence_barrier_init();
    __syncthreads();   // every barrier is initialised before any warp waits on it
    grid_dep_launch();
    grid_dep_wait();   // q, page tables and the cache may come from the preceding kernel

    // split plan: this pair's first page-table entry, loaded alongside the context
    // length (in bounds whatever the length; used only if the pair has pages)
    int phys_first = -1;
    if constexpr (!kFlat) {
        if (producer && p.max_pages > 0)
            phys_first = __ldg(p.block_table + (size_t)blockIdx.z * p.max_pages +
                               min((int)blockIdx.x * p.pages_per_split + pw, p.max_pages - 1));
    }
    WsSeg sg;
    bool have;
    WsSeg* my_seg = nullptr;   // flattened plan: this warp's walker, in shared memory
    if constexpr (kFlat) {
        __shared__ int s_wtot[kGwThreads / 32];
        __shared__ long long s_start;
        __shared__ WsSeg s_seg[kGwThreads / 32];
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
            const int b = cs.b, h = cs.h;
            const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;
            const int32_t* bt_row = p.block_table + (size_t)b * p.max_pages;
            int first;
            const int n_seg = ws_seg_pages<kGwPairs>(cs, pw, first);
            int phys_next = kFlat ? (n_seg > 0 ? __ldg(bt_row + first) : -1) : phys_first;
            for (int i = 0; i < n_seg; ++i, ++k) {
                const int lp = first + kGwPairs * i;
                const int s = k % kGwStages;
                if (k >= kGwStages) {
                    const bool freed = mbar_wait_bounded(&empty[s], (uint32_t)(((k / kGwStages) - 1) & 1));
                    if (!__all_sync(0xffffffffu, freed)) {
                        if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
                        stop = true;
                        break;
                    }
                }
                const int phys = phys_next;
                if (i + 1 < n_seg) phys_next = __ldg(bt_row + lp + kGwPairs);
                const bool ok = phys >= 0 && phys < p.num_pages;
                uint8_t* st = stages + s * kGwStageBytes;
                if (lane == 0) {
                    *reinterpret_cast<int*>(st + kGwOffHdr) = ok ? phys : -1;
                    if (ok) {
                        const int z = phys * p.num_kv_heads + h;
                        const size_t ph = (size_t)z;
                        mbar_arrive_expect_tx(&full[s], (uint32_t)(4096 + 128 + 128 + 256 + 64 * m));
                        tma_page(st + kGwOffK, &gparams.k_map, z, &full[s]);
                        tma_page(st + kGwOffV, &gparams.v_map, z, &full[s]);
                        bulk_g2s(st + kGwOffKs, p.k_scale + ph * (kPage * 4), 128, &full[s]);
                        bulk_g2s(st + kGwOffVs, p.v_scale + ph * (kPage * 4), 128, &full[s]);
                        bulk_g2s(st + kGwOffW, p.k_witness + ph * (kPage * kBands), 256, &full[s]);
                        if (m > 0) bulk_g2s(st + kGwOffB, p.k_bypass + ph * (kPage * nb), (uint32_t)(64 * m), &full[s]);
                    } else {
                        atomicOr(p.status, WC_DEV_BAD_PAGE);
                        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&full[s])) : "memory");
                    }
                }
                issued = k + 1;
                if (ok) {   // dither bytes j[token][storage position], swizzled like the code tiles
                    // K and V of tokens g, g+8 x position chunks 2c, 2c+1 (call 2i: K, 2i+1:
                    // V), advanced round by round
                    const uint32_t slot0 = (uint32_t)phys * kPage;
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
                        const int off = swz(g + 8 * (i >> 1), 2 * c + (i & 1));
                        *reinterpret_cast<uint4*>(st + kGwOffKd + off) =
                            make_uint4(x0[2 * i], x1[2 * i], x2[2 * i], x3[2 * i]);
                        *reinterpret_cast<uint4*>(st + kGwOffVd + off) =
                            make_uint4(x0[2 * i + 1], x1[2 * i + 1], x2[2 * i + 1], x3[2 * i + 1]);
                    }
                }
                __syncwarp();
                if (lane == 0)   // second arrival: dither tiles and header are written
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&full[s])) : "memory");
            }
        };
        if constexpr (kFlat) {
            for (bool more = have; more && !stop; more = ws_step<kGwPairs, true>(p, my_seg, lane)) produce(*my_seg);
        } else {
            produce(sg);
        }
        // copies still in flight must land before the CTA's smem is released
        for (int j = max(0, issued - kGwStages); j < issued; ++j)
            (void)mbar_wait_bounded(&full[j % kGwStages], (uint32_t)((j / kGwStages) & 1));
        return;
    }

    // ---- consumer: dither read from the stage ------------------------------------------
    // The CTA merge's buffer [warp][head][kPartialStride]: the stage area in the
    // split plan (one segment, the producers are done with it), a buffer of its
    // own in the flattened plan (the producers stage the next segment meanwhile).
    float* mbuf = reinterpret_cast<float*>(kFlat ? smem + kGwMergeOff : smem);
    int k = 0;   // stage ring position, continued across segments
    bool failed = false;
    // one segment: query setup, pages, CTA merge (the split plan has one segment)
    auto consume = [&](const WsSeg& cs) {
        const int b = cs.b, h = cs.h;
        const int ctx = cs.ctx;
        const bool row_valid = g < G;
        const __half* qrow = p.q + ((size_t)b * p.num_q_heads + (size_t)h * G + (row_valid ? g : 0)) * kHeadDim;
        uint32_t qn[16];   // head g, channels 32c + 2i, +1 in word i (channel order: group c)
        uint32_t qw[16];   // head g, channels 16ks + 4c + 2hh, +1 in word 2ks + hh (storage order)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint4 v = row_valid ? __ldg(reinterpret_cast<const uint4*>(qrow + 32 * c) + i) : make_uint4(0, 0, 0, 0);
            qn[4 * i] = v.x; qn[4 * i + 1] = v.y; qn[4 * i + 2] = v.z; qn[4 * i + 3] = v.w;
        }
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            const uint2 v = row_valid ? __ldg(reinterpret_cast<const uint2*>(qrow + 16 * ks + 4 * c)) : make_uint2(0, 0);
            qw[2 * ks] = v.x;
            qw[2 * ks + 1] = v.y;
        }

        // ---- the bypassed key channels --------------------------------------------
        // nmask: bypassed channels of group c (bit d - 32c); pmask: bypassed slots of
        // qw (bit 4 ks + j for channel 16 ks + 4c + j); qb[t]: B operand of bypass
        // tile t, q at the dims of entries 8t + 2c, +1 (pair 4t + c) for head g.
        const int32_t* prs = p.bypass_pairs + (size_t)h * m;
        uint32_t nmask = 0, pmask = 0, pvalid = 0;   // pvalid: bit t for a pair index in range
        uint32_t qb[4] = {0u, 0u, 0u, 0u};
        uint32_t seen_lo = 0u, seen_hi = 0u;   // pair indices met so far: a repeated pair is ignored
        for (int t = 0; t < m; ++t) {
            const int j = __ldg(prs + t);
            const bool again = j >= 0 && j < kHeadDim / 2 && (((j < 32 ? seen_lo : seen_hi) >> (j & 31)) & 1u);
            if (j < 0 || j >= kHeadDim / 2 || again) {
                if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(p.status, WC_DEV_BAD_PAIR);
                continue;
            }
            if (j < 32) seen_lo |= 1u << j;
            else seen_hi |= 1u << (j - 32);
            pvalid |= 1u << t;
            const int da = p.rope_layout == WC_ROPE_HALF ? j : 2 * j;
            const int db = p.rope_layout == WC_ROPE_HALF ? j + kHeadDim / 2 : 2 * j + 1;
            if ((da >> 5) == c) nmask |= 1u << (da & 31);
            if ((db >> 5) == c) nmask |= 1u << (db & 31);
            if (((da >> 2) & 3) == c) pmask |= 1u << (4 * (da >> 4) + (da & 3));
            if (((db >> 2) & 3) == c) pmask |= 1u << (4 * (db >> 4) + (db & 3));
            if ((t & 3) == c && row_valid) {   // pair t = 4 (t >> 2) + c: entries 2t, 2t + 1 of tile t >> 2
                const unsigned short qa = __ldg(reinterpret_cast<const unsigned short*>(qrow) + da);
                const unsigned short qbv = __ldg(reinterpret_cast<const unsigned short*>(qrow) + db);
                const uint32_t w = (uint32_t)qa | ((uint32_t)qbv << 16);
                const int tile = t >> 2;
                qb[0] = tile == 0 ? w : qb[0];
                qb[1] = tile == 1 ? w : qb[1];
                qb[2] = tile == 2 ? w : qb[2];
                qb[3] = tile == 3 ? w : qb[3];
            }
        }
#pragma unroll
        for (int w = 0; w < 16; ++w) {   // word w holds slots 2w (low half) and 2w + 1
            const uint32_t mk = (pmask >> (2 * w)) & 3u;
            qw[w] &= ((mk & 1u) ? 0xFFFF0000u : 0xFFFFFFFFu) & ((mk & 2u) ? 0x0000FFFFu : 0xFFFFFFFFu);
        }
        const int nbt = (nb + 7) >> 3;   // bypass tiles of 8 dims

        // ---- per-group sums of q (bypassed channels left out), band norms ---------
        float qs = 0.f, qq = 0.f, part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&qn[i]));
            const bool b0 = (nmask >> (2 * i)) & 1u, b1 = (nmask >> (2 * i + 1)) & 1u;
            qs += (b0 ? 0.f : f.x) + (b1 ? 0.f : f.y);
            qq = fmaf(b0 ? 0.f : f.x, f.x, fmaf(b1 ? 0.f : f.y, f.y, qq));
            part[i >> 2] = fmaf(f.x, f.x, fmaf(f.y, f.y, part[i >> 2]));   // channels 32c + 8(i>>2) .. +7
        }
        // kappa sum_g q and ||q_g'||^2 of group G for this thread's softmax heads 2c, 2c+1
        float zo[4][2], qn2[4][2];
#pragma unroll
        for (int gi = 0; gi < 4; ++gi)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                zo[gi][e] = kKappa * __shfl_sync(0xffffffffu, qs, 4 * (2 * c + e) + gi);
                qn2[gi][e] = __shfl_sync(0xffffffffu, qq, 4 * (2 * c + e) + gi);
            }
        float tbk = 0.f;   // 2 log(2S/delta) / (12 d)
        if constexpr (kTierB)
            tbk = 2.0f * (p.tb_log_2_over_delta + logf((float)max(ctx, 1))) * (1.0f / (12.0f * kHeadDim));
        float band_a, band_b;   // squared norms of bands 2c and 2c+1 of head g (all channels)
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
        uint32_t a_hi = 0, a_lo = 0;   // B operand of the bound: a[head g][bands 2c, 2c+1], log2 units
        if (row_valid) {
            const float x0 = sqrtf(band_a) * kRsdLog2e, x1 = sqrtf(band_b) * kRsdLog2e;
            const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
            a_hi = pack_h2(__half2float(h0), __half2float(h1));
            a_lo = pack_h2(x0 - __half2float(h0), x1 - __half2float(h1));
        }

        // ---- running state (heads 2c, 2c+1) ----------------------------------------------
        float m_run[2] = {-INFINITY, -INFINITY};
        float l_part[2] = {0.f, 0.f}, d_part[2] = {0.f, 0.f}, db_part[2] = {0.f, 0.f};
        float spv[4][2] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};   // sum P s_g per group
        float acc[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
        int lam_exp = INT_MIN;   // P s_g 2^lam_exp stays below 2^14 (fp16)
        float sv_lim = 1.17549435e-38f;   // 2^(6 - lam_exp): the scale at which lam_exp must drop
        const int tv[4] = {2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9};

        int first;
        const int n_seg = ws_seg_pages<kGwPairs>(cs, pw, first);
        for (int i = 0; i < n_seg && !failed; ++i, ++k) {
            const int s = k % kGwStages;
            const bool landed = mbar_wait_bounded(&full[s], (uint32_t)((k / kGwStages) & 1));
            if (!__all_sync(0xffffffffu, landed)) {   // warp-uniform decision
                if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
                failed = true;   // later pages are not waited for; the merges still run
                break;
            }
            const uint8_t* st = stages + s * kGwStageBytes;
            const int lp = first + kGwPairs * i;
            if (*reinterpret_cast<const int*>(st + kGwOffHdr) >= 0) {
                const int nvalid = min(kPage, ctx - lp * kPage);
                const bool ok0 = g < nvalid, ok1 = g + 8 < nvalid;
                // group scales of tokens g, g + 8
                float sk[2][4], sv[2][4];
                {
                    const uint2 ka = *reinterpret_cast<const uint2*>(st + kGwOffKs + 8 * g);
                    const uint2 kb = *reinterpret_cast<const uint2*>(st + kGwOffKs + 8 * (g + 8));
                    const uint2 va = *reinterpret_cast<const uint2*>(st + kGwOffVs + 8 * g);
                    const uint2 vb = *reinterpret_cast<const uint2*>(st + kGwOffVs + 8 * (g + 8));
                    const uint32_t w[4][2] = {{ka.x, ka.y}, {kb.x, kb.y}, {va.x, va.y}, {vb.x, vb.y}};
#pragma unroll
                    for (int r = 0; r < 2; ++r)
#pragma unroll
                        for (int q2 = 0; q2 < 2; ++q2) {
                            const float2 fk = __half22float2(*reinterpret_cast<const __half2*>(&w[r][q2]));
                            const float2 fv = __half22float2(*reinterpret_cast<const __half2*>(&w[2 + r][q2]));
                            sk[r][2 * q2] = fk.x; sk[r][2 * q2 + 1] = fk.y;
                            sv[r][2 * q2] = fv.x; sv[r][2 * q2 + 1] = fv.y;
                        }
                }
                if (nvalid < kPage) {   // the context's last page (warp-uniform): tail slots hold any bits
#pragma unroll
                    for (int gi = 0; gi < 4; ++gi) {
                        if (!ok0) { sk[0][gi] = 0.f; sv[0][gi] = 0.f; }
                        if (!ok1) { sk[1][gi] = 0.f; sv[1][gi] = 0.f; }
                    }
                }

                // ---------------- QK, folded per group ------------------------------------
                // rows g, g+8 are tokens g, g+8; raw[i] = (tok g, head 2c), (g, 2c+1), (g+8, 2c), (g+8, 2c+1)
                float raw[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int gp = 0; gp < 2; ++gp) {   // storage positions 32c + 16gp .. +15: k-steps 4gp .. 4gp+3
                    const uint4 ka = *reinterpret_cast<const uint4*>(st + kGwOffK + swz(g, 2 * c + gp));
                    const uint4 kb = *reinterpret_cast<const uint4*>(st + kGwOffK + swz(g + 8, 2 * c + gp));
                    const uint4 da = *reinterpret_cast<const uint4*>(st + kGwOffKd + swz(g, 2 * c + gp));
                    const uint4 db = *reinterpret_cast<const uint4*>(st + kGwOffKd + swz(g + 8, 2 * c + gp));
                    float dc[4] = {0.f, 0.f, 0.f, 0.f}, dd[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const int ks = 4 * gp + kk;
                        const uint32_t xa = word_of(ka, kk) ^ 0x80808080u, xb = word_of(kb, kk) ^ 0x80808080u;
                        const uint32_t A[4] = {s8x2_to_h2(xa, kSel01), s8x2_to_h2(xb, kSel01), s8x2_to_h2(xa, kSel23),
                                               s8x2_to_h2(xb, kSel23)};
                        mma16816(dc, A, qw[2 * ks], qw[2 * ks + 1]);
                        const uint32_t ya = word_of(da, kk), yb = word_of(db, kk);
                        const uint32_t H[4] = {h8(ya, kSel01), h8(yb, kSel01), h8(ya, kSel23), h8(yb, kSel23)};
                        mma16816(dd, H, qw[2 * ks], qw[2 * ks + 1]);
                        if (kk & 1) {   // group 2gp + kk/2 complete: raw += s_g (code.q - h'.q + kappa sum_g q)
                            const int gi = 2 * gp + (kk >> 1);
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                raw[i] = fmaf(sk[i >> 1][gi], dc[i] - dd[i] + zo[gi][i & 1], raw[i]);
                                dc[i] = dd[i] = 0.f;
                            }
                        }
                    }
                }
                // exact bypassed values: raw += K_bypass . q_bypass, tiles of 8 entries
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    if (t < nbt) {
                        const int e0 = 8 * t + 2 * c;   // entries e0, e0 + 1 = pair 4t + c
                        const bool use = e0 < nb && ((pvalid >> (4 * t + c)) & 1u);
                        const uint32_t a0 = use ? *reinterpret_cast<const uint32_t*>(st + kGwOffB + (g * nb + e0) * 2) : 0u;
                        const uint32_t a1 =
                            use ? *reinterpret_cast<const uint32_t*>(st + kGwOffB + ((g + 8) * nb + e0) * 2) : 0u;
                        mma1688(raw, a0, a1, qb[t]);
                    }
                }

                // ---------------- logits, bound, softmax ------------------------------
                float cb[4] = {0.f, 0.f, 0.f, 0.f};
                {
                    const uint32_t wa = *reinterpret_cast<const uint32_t*>(st + kGwOffW + (g * kBands + 2 * c) * 2);
                    const uint32_t wb = *reinterpret_cast<const uint32_t*>(st + kGwOffW + ((g + 8) * kBands + 2 * c) * 2);
                    mma1688(cb, wa, wb, a_hi);
                    mma1688(cb, wa, wb, a_lo);
                }
                float y[4], u[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = i >> 1, e = i & 1;
                    y[i] = raw[i] * kRsdLog2e;
                    if constexpr (kTierB) {   // u = sqrt(2 log(2S/delta) varsigma^2), grouped proxy
                        float ss = 0.f;
#pragma unroll
                        for (int gi = 0; gi < 4; ++gi) ss = fmaf(qn2[gi][e] * sk[r][gi], sk[r][gi], ss);
                        u[i] = sqrtf(tbk * ss);
                    }
                }
                if (nvalid < kPage) {
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (!((i >> 1) ? ok1 : ok0)) {
                            y[i] = -INFINITY;
                            cb[i] = 0.f;
                        }
                }
                float mx0 = fmaxf(y[0], y[2]), mx1 = fmaxf(y[1], y[3]);
                // the reference moves lazily (a logit above it by more than 8); the
                // column maximum over the token rows is reduced only then
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
                    l_part[0] *= a0; d_part[0] *= a0; db_part[0] *= a0;
                    l_part[1] *= a1; d_part[1] *= a1; db_part[1] *= a1;
#pragma unroll
                    for (int gi = 0; gi < 4; ++gi) { spv[gi][0] *= a0; spv[gi][1] *= a1; }
#pragma unroll
                    for (int mt = 0; mt < 8; ++mt) {
                        acc[mt][0] *= a0; acc[mt][2] *= a0;
                        acc[mt][1] *= a1; acc[mt][3] *= a1;
                    }
                }
                float pe[4], ub[4];           // ub: the Tier-B bound in log2 units
#pragma unroll
                for (int i = 0; i < 4; ++i) ub[i] = kTierB ? u[i] * kLog2e : 0.f;
                bool huge;                    // warp-uniform: a bound of kHugeLog2 or more (meter_term)
                {
                    float big = fmaxf(fmaxf(cb[0], cb[1]), fmaxf(cb[2], cb[3]));
                    if constexpr (kTierB) big = fmaxf(big, fmaxf(fmaxf(ub[0], ub[1]), fmaxf(ub[2], ub[3])));
                    huge = __any_sync(0xffffffffu, big >= kHugeLog2);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = i & 1;
                    pe[i] = fast_exp2(y[i] - m_run[e]);     // 0 for masked tokens
                    l_part[e] += pe[i];
                    if (!huge) {
                        d_part[e] = fmaf(pe[i], fast_exp2(cb[i]) - 1.f, d_part[e]);
                        if constexpr (kTierB) db_part[e] = fmaf(pe[i], fast_exp2(ub[i]) - 1.f, db_part[e]);
                    }
#pragma unroll
                    for (int gi = 0; gi < 4; ++gi) spv[gi][e] = fmaf(pe[i], sv[i >> 1][gi], spv[gi][e]);
                }
                if (huge) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int e = i & 1;
                        const float t = y[i] - m_run[e];
                        d_part[e] += meter_term(t, cb[i]);
                        if constexpr (kTierB) db_part[e] += meter_term(t, ub[i]);
                    }
                }
                {   // P s_g 2^lam_exp < 2^14: s_g 2^lam_exp < 2^6 for every group of the page;
                    // lam_exp only decreases, checked per lane against sv_lim, reduced only then
                    float smax = 0.f;
#pragma unroll
                    for (int gi = 0; gi < 4; ++gi) smax = fmaxf(smax, fmaxf(sv[0][gi], sv[1][gi]));
                    if (__any_sync(0xffffffffu, smax >= sv_lim)) {
                        const float wmax = __int_as_float(__reduce_max_sync(0xffffffffu, __float_as_int(smax)));
                        const int ex = ((__float_as_int(wmax) >> 23) & 0xFF) - 126;   // wmax < 2^ex
                        const int want = 6 - ex;
                        if (lam_exp != INT_MIN) {   // want < lam_exp here
                            const float f = pow2(want - lam_exp);
#pragma unroll
                            for (int mt = 0; mt < 8; ++mt)
#pragma unroll
                                for (int e2 = 0; e2 < 4; ++e2) acc[mt][e2] *= f;
                        }
                        lam_exp = want;
                        sv_lim = pow2(6 - lam_exp);
                    }
                }
                const float lam = pow2(lam_exp == INT_MIN ? 0 : lam_exp);

                // ---------------- PV: acc[dim][head], one P operand per group -----------
                // m-tile mt covers channels 16 mt .. 16 mt + 15 (group mt / 2); row g is
                // channel 16 mt + g, row g + 8 channel 16 mt + g + 8
                uint4 vq[4], dv[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    vq[j] = *reinterpret_cast<const uint4*>(st + kGwOffV + swz(tv[j], g));
                    dv[j] = *reinterpret_cast<const uint4*>(st + kGwOffVd + swz(tv[j], g));
                }
#pragma unroll
                for (int gi = 0; gi < 4; ++gi) {
                    uint32_t bp0, bp1, bl0, bl1;   // B = (P s_g)^T 2^lam, hi + lo
                    {
                        const float x0 = pe[0] * sv[0][gi] * lam, x1 = pe[1] * sv[0][gi] * lam;
                        const float x2 = pe[2] * sv[1][gi] * lam, x3 = pe[3] * sv[1][gi] * lam;
                        const uint32_t h01 = pack_h2(x0, x1), h23 = pack_h2(x2, x3);
                        const float2 r01 = __half22float2(*reinterpret_cast<const __half2*>(&h01));
                        const float2 r23 = __half22float2(*reinterpret_cast<const __half2*>(&h23));
                        const uint32_t l01 = pack_h2(x0 - r01.x, x1 - r01.y), l23 = pack_h2(x2 - r23.x, x3 - r23.y);
                        bp0 = movmatrix_t(h01);
                        bp1 = movmatrix_t(h23);
                        bl0 = movmatrix_t(l01);
                        bl1 = movmatrix_t(l23);
                    }
#pragma unroll
                    for (int mm = 0; mm < 2; ++mm) {
                        const int mt = 2 * gi + mm, wi = mt >> 1, pos = 2 * (mt & 1);
                        uint32_t A[4], H[4];
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            const uint32_t X = prmt(word_of(vq[2 * pr], wi) ^ 0x80808080u,
                                                    word_of(vq[2 * pr + 1], wi) ^ 0x80808080u, sel_interleave(pos));
                            A[2 * pr] = s8x2_to_h2(X, kSel01);
                            A[2 * pr + 1] = s8x2_to_h2(X, kSel23);
                            const uint32_t Y = prmt(word_of(dv[2 * pr], wi), word_of(dv[2 * pr + 1], wi),
                                                    sel_interleave(pos));
                            H[2 * pr] = nh8(Y, kSel01);       // -h'
                            H[2 * pr + 1] = nh8(Y, kSel23);
                        }
                        mma16816(acc[mt], A, bp0, bp1);
                        mma16816(acc[mt], A, bl0, bl1);
                        mma16816(acc[mt], H, bp0, bp1);
                        mma16816(acc[mt], H, bl0, bl1);
                    }
                }
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
#pragma unroll
                for (int gi = 0; gi < 4; ++gi) spv[gi][e] += __shfl_xor_sync(0xffffffffu, spv[gi][e], o);
            }
        const float inv_lam = pow2(lam_exp == INT_MIN ? 0 : -lam_exp);

        // ---- CTA merge over the consumer warps: one partial per segment --------------------
        gw_consumer_sync();   // all consumers are done with their stages and with mbuf's last use
        {
            float* wb = mbuf + pw * kMaxGroup * kPartialStride;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                float* row = wb + (2 * c + e) * kPartialStride;
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {   // channels 16 mt + g and 16 mt + g + 8
                    const float add = kKappa * spv[mt >> 1][e];
                    row[16 * mt + g] = fmaf(acc[mt][e], inv_lam, add);
                    row[16 * mt + g + 8] = fmaf(acc[mt][e + 2], inv_lam, add);
                }
                if (g == 0) {
                    row[kHeadDim + 0] = m_run[e];
                    row[kHeadDim + 1] = l_part[e];
                    row[kHeadDim + 2] = d_part[e];
                    if constexpr (kTierB) row[kHeadDim + 3] = db_part[e];
                }
            }
        }
        gw_consumer_sync();
        const size_t unit = (size_t)b * p.num_kv_heads + h;
        // flattened plan: share j's segment of sequence b goes to partial h (shares + batch) + j + b
        const int shares = p.splits / p.num_kv_heads;
        const size_t pid = kFlat ? (size_t)h * (shares + p.batch) + blockIdx.x / p.num_kv_heads + b
                                 : unit * p.splits + blockIdx.x;
        float* part_out = p.partials + pid * (kMaxGroup * kPartialStride);
        // thread -> (head, 4-dim chunk); chunk 32 carries (M, l, D, D_B)
        for (int idx = threadIdx.x; idx < G * 33; idx += 32 * kGwPairs) {
            const int hh = idx / 33, ch = idx % 33;
            float mw[kGwPairs];
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kGwPairs; ++w) {
                mw[w] = mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim];
                M = fmaxf(M, mw[w]);
            }
            float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
            const int col = (ch < 32) ? 4 * ch : kHeadDim + 1;
#pragma unroll
            for (int w = 0; w < kGwPairs; ++w) {
                if (mw[w] == -INFINITY) continue;   // a warp without pages: its values are not read
                const float wt = fast_exp2(mw[w] - M);
                const float* src = mbuf + (w * kMaxGroup + hh) * kPartialStride + col;
                if (ch < 32) {
                    const float4 v = *reinterpret_cast<const float4*>(src);
                    s.x = fmaf(wt, v.x, s.x); s.y = fmaf(wt, v.y, s.y);
                    s.z = fmaf(wt, v.z, s.z); s.w = fmaf(wt, v.w, s.w);
                } else {
                    s.x = fmaf(wt, src[0], s.x);                          // l
                    s.y = fmaf(wt, src[1], s.y);                          // D
                    if constexpr (kTierB) s.z = fmaf(wt, src[2], s.z);   // Tier-B D
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
            }
        }
    };
    if constexpr (kFlat) {
        for (bool more = have; more; more = ws_step<kGwPairs, true>(p, my_seg, lane)) consume(*my_seg);
    } else {
        if (have) consume(sg);
    }
}

template <int kX>
cudaError_t launch_g32_ws(const DecodeParams& p, cudaStream_t stream) {
    static bool configured = false;   // per process; the attributes are per function
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_g32_ws_kernel<kX>, cudaFuncAttributeMaxDynamicSharedMemorySize, kGwSmemFlat);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(decode_g32_ws_kernel<kX>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    G32Params gp;
    gp.p = p;
    if (!encode_page_map(&gp.k_map, p.k_codes, p.num_pages, p.num_kv_heads) ||
        !encode_page_map(&gp.v_map, p.v_codes, p.num_pages, p.num_kv_heads))
        return cudaErrorInvalidValue;
    const bool flat = p.pages_per_split == 0;
    const dim3 grid = flat ? dim3(p.splits, 1, 1) : dim3(p.splits, p.num_kv_heads, p.batch);
    cudaError_t e = launch_pdl(decode_g32_ws_kernel<kX>, grid, dim3(kGwThreads), flat ? kGwSmemFlat : kGwSmemBytes,
                               stream, gp);
    if (e != cudaSuccess) return e;
    return launch_merge_x(p, kX & ~kXFlat, stream);
}

}  // namespace

cudaError_t launch_decode_g32(const DecodeParams& p, cudaStream_t stream) {
    if (p.pages_per_split == 0)   // the flattened plan
        return p.meter_b ? launch_g32_ws<kXTierB | kXFlat>(p, stream) : launch_g32_ws<kXFlat>(p, stream);
    return p.meter_b ? launch_g32_ws<kXTierB>(p, stream) : launch_g32_ws<0>(p, stream);
}

}  // namespace wc
