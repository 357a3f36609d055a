// Metered decode attention (§6 meter loop, read path; §6.2.1-§6.2.2):
// dequantize the paged cache, compute the compressed attention output, and in
// the same pass accumulate the Tier-A e-form meter
//   c_t = (1/sqrt d) sum_b ||q_b|| w_{t,b}        (Thm. "Sound black-box logit bound")
//   A   = sum_t p~_t e^{c_t},  meter = min(1, (A^2 - 1)/2)   (Thm. "Sound replacement")
// merged across context splits under log-sum-exp weights (A is a p~-weighted
// mean, so it merges exactly like the output; §6.2.2).
//
// Grid (splits, Hkv, batch); 4 warps per CTA.  Each warp owns a 4-stage ring
// of page buffers in shared memory filled by bulk asynchronous copies
// (cp.async.bulk + mbarrier) that its lane 0 issues ahead of use; a page is
// 16 tokens of one KV head (2 KiB K codes, 2 KiB V codes, scales, witness).
//
// Per page a warp computes, with mma.m16n8k16 (fp16 in, fp32 accumulate):
//   QK:  D[head][token] = q . code - q . h'   (A = q, B = codes / dither),
//   PV:  acc[dim][head] += code^T P - h'^T P (A = V codes / dither, B = P),
// and the bound C[head][token] = a[head][band] . W[token][band] with
// mma.m16n8k8 (a split into two fp16 terms).  Integer codes and the dither
// (h' = 4 + j/256 for 8-bit, 1 + j/1024 for 10-bit; xi = h' - kappa) are
// exact fp16 operands, so code - xi = code - h' + kappa is carried exactly
// until the fp32 accumulators.
#include <algorithm>
#include <climits>

#include "wc_kernels.cuh"

namespace wc {

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kStages = 3;
constexpr int kMinBlocks = 2;            // two CTAs (16 warps) per SM
constexpr int kStageBytes = 4416;   // K codes | V codes | K scale | V scale | witness
constexpr int kOffV = 2048, kOffKs = 4096, kOffVs = 4128, kOffW = 4160;
constexpr int kSmemBytes = kWarps * kStages * kStageBytes + kWarps * kStages * 8 + kMaxGroup * kHeadDim * 2;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRsdLog2e = 0.08838834764831845f * 1.4426950408889634f;  // log2(e)/sqrt(128)

constexpr uint32_t kSel01 = 0x4140u, kSel23 = 0x4342u;   // [x0,K,x1,K], [x2,K,x3,K]

__device__ __forceinline__ uint32_t sel_interleave(int p) {  // [a_p, b_p, a_p+1, b_p+1]
    return p == 0 ? 0x5140u : 0x7362u;
}

template <int kBits>
struct DitherConst;
template <>
struct DitherConst<8> {  // xi = (j + 1/2)/256 - 1/2 = h' - kappa, h' = 4 + j/256
    static constexpr float kappa = 4.498046875f;
};
template <>
struct DitherConst<10> {  // xi = (j + 1/2)/1024 - 1/2 = h' - kappa, h' = 1 + j/1024
    static constexpr float kappa = 1.49951171875f;
};

// Two int8 codes as the fp16 pair 1152 + code (exact): (code ^ 0x80) in the
// low mantissa byte of 1024.0.  The constant 1152 is removed once per logit.
__device__ __forceinline__ uint32_t s8x2_biased(uint32_t w_xor80, uint32_t sel) {
    return prmt(w_xor80, 0x64646464u, sel);
}

// h' pair (fp16) for two 8-bit dithers: bytes of x at the selector.
__device__ __forceinline__ uint32_t h8(uint32_t x, uint32_t sel) { return prmt(x, 0x44444444u, sel); }
// h' pair (fp16) for two 10-bit dithers in the low bits of each 16-bit lane.
__device__ __forceinline__ uint32_t h10(uint32_t x) { return (x & 0x03FF03FFu) | 0x3C003C00u; }

// 2^n for -126 <= n <= 127.
__device__ __forceinline__ float pow2(int n) { return __int_as_float((127 + n) << 23); }

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
    return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
}

template <int kScheme, int kBits>
__global__ void __launch_bounds__(kThreads, kMinBlocks) decode_kernel(const __grid_constant__ DecodeParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, c = lane & 3;
    const int split = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
    const int G = p.group;
    constexpr bool kInt8 = (kScheme == WC_SCHEME_DITHER_INT8);

    uint8_t* my_stages = smem + warp * kStages * kStageBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kWarps * kStages * kStageBytes) + warp * kStages;
    if (lane == 0)
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
    fence_barrier_init();
    grid_dep_wait();   // q, page tables and the cache may come from the preceding kernel

    int ctx = __ldg(p.ctx_lens + b);
    if (ctx < 0 || ctx > p.max_pages * kPage) {
        if (threadIdx.x == 0 && split == 0 && h == 0) atomicOr(p.status, WC_DEV_BAD_CTX);
        ctx = max(0, min(ctx, p.max_pages * kPage));
    }
    const int npages = (ctx + kPage - 1) / kPage;
    const int p0 = split * p.pages_per_split;
    const int p1 = min(p0 + p.pages_per_split, npages);
    const int n_my = (p1 - p0 - warp > 0) ? (p1 - p0 - warp + kWarps - 1) / kWarps : 0;
    const int32_t* bt_row = p.block_table + (size_t)b * p.max_pages;
    const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;

    // ---- per-warp stage ring -------------------------------------------------
    __syncwarp();

    auto issue = [&](int k) {
        if (k >= n_my || lane != 0) return;
        const int phys = __ldg(bt_row + p0 + warp + kWarps * k);
        uint64_t* bar = &bars[k % kStages];
        if (phys < 0 || phys >= p.num_pages) {
            atomicOr(p.status, WC_DEV_BAD_PAGE);
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
            return;
        }
        uint8_t* st = my_stages + (k % kStages) * kStageBytes;
        const size_t ph = (size_t)phys * p.num_kv_heads + h;
        constexpr uint32_t bytes = kInt8 ? kStageBytes : (2048 + 2048 + 256);
        mbar_arrive_expect_tx(bar, bytes);
        bulk_g2s(st, p.k_codes + ph * (kPage * kHeadDim), 2048, bar);
        bulk_g2s(st + kOffV, p.v_codes + ph * (kPage * kHeadDim), 2048, bar);
        if constexpr (kInt8) {
            bulk_g2s(st + kOffKs, p.k_scale + ph * kPage, 32, bar);
            bulk_g2s(st + kOffVs, p.v_scale + ph * kPage, 32, bar);
        }
        bulk_g2s(st + kOffW, p.k_witness + ph * (kPage * kBands), 256, bar);
    };
    for (int k = 0; k < kStages; ++k) issue(k);

    // ---- query fragments, band norms ------------------------------------------
    const bool row_valid = g < G;
    // q of the CTA's G heads, fp16 [kMaxGroup][128], after the stage rings
    uint32_t* q_sm = reinterpret_cast<uint32_t*>(smem + kWarps * kStages * kStageBytes + kWarps * kStages * 8);
    for (int i = threadIdx.x; i < kMaxGroup * kHeadDim / 8; i += kThreads) {
        const int hh = i / (kHeadDim / 8), col = i % (kHeadDim / 8);
        uint4 v = make_uint4(0, 0, 0, 0);
        if (hh < G) v = __ldg(reinterpret_cast<const uint4*>(p.q + ((size_t)b * p.num_q_heads + (size_t)h * G + hh) * kHeadDim) + col);
        reinterpret_cast<uint4*>(q_sm)[i] = v;
    }
    __syncthreads();
    const uint4* my_q = reinterpret_cast<const uint4*>(q_sm + g * (kHeadDim / 2) + 16 * c);   // head g, ch 32c..
    uint32_t qw[16];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 v = my_q[i];
        qw[4 * i] = v.x; qw[4 * i + 1] = v.y; qw[4 * i + 2] = v.z; qw[4 * i + 3] = v.w;
    }
    float qsum = 0.f, part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&qw[i]));
        qsum += f.x + f.y;
        part[i >> 2] = fmaf(f.x, f.x, fmaf(f.y, f.y, part[i >> 2]));   // channels 32c + 8(i>>2) .. +7
    }
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 1);
    qsum += __shfl_xor_sync(0xffffffffu, qsum, 2);
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
    uint32_t a_hi = 0, a_lo = 0;   // bound A fragment, rows g (rows g+8 are zero)
    if (row_valid) {
        const float x0 = sqrtf(band_a) * 0.08838834764831845f, x1 = sqrtf(band_b) * 0.08838834764831845f;
        const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
        a_hi = pack_h2(__half2float(h0), __half2float(h1));
        a_lo = pack_h2(x0 - __half2float(h0), x1 - __half2float(h1));
    }
    // q . (code - xi) = q . code - q . h' + kappa sum(q)
    const float zoff = kInt8 ? DitherConst<kBits == 10 ? 10 : 8>::kappa * qsum : 0.f;

    // ---- running state -----------------------------------------------------------
    // Log2-domain softmax reference m_run, moved lazily: only when a page's max
    // exceeds it by more than 8 (P may reach 2^8 in between).
    float m_run = -INFINITY;
    float l_part = 0.f, d_part = 0.f, spv_part = 0.f;
    float acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
    // P * s_v * 2^lam_exp stays below 2^14 (fp16): s_v * 2^lam_exp < 2^6.
    int lam_exp = kInt8 ? INT_MIN : 6;
    bool failed = false;
    int consumed = 0;
    int phys_next = n_my > 0 ? __ldg(bt_row + p0 + warp) : 0;

    for (int k = 0; k < n_my; ++k) {
        const int lp = p0 + warp + kWarps * k;
        const int phys = phys_next;
        if (k + 1 < n_my) phys_next = __ldg(bt_row + lp + kWarps);
        const bool page_ok = phys >= 0 && phys < p.num_pages;
        const bool landed = mbar_wait_bounded(&bars[k % kStages], (uint32_t)((k / kStages) & 1));
        if (!__all_sync(0xffffffffu, landed)) {   // warp-uniform decision
            if (lane == 0) atomicOr(p.status, WC_DEV_TIMEOUT);
            failed = true;
            break;
        }
        consumed = k + 1;
        if (page_ok) {
            const uint8_t* st = my_stages + (k % kStages) * kStageBytes;
            const uint32_t slot0 = (uint32_t)phys * kPage;
            const int nvalid = min(kPage, ctx - lp * kPage);

            // ---------------- QK: D[head][token] ------------------------------
            float dc[2][4], dd[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) dc[nt][e] = dd[nt][e] = 0.f;
            uint32_t qf[16];   // reloaded per page: keeps 16 registers free across the loop
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint4 v = my_q[i];
                qf[4 * i] = v.x; qf[4 * i + 1] = v.y; qf[4 * i + 2] = v.z; qf[4 * i + 3] = v.w;
            }
            // codes first, then the dither: their operands are never live together
#pragma unroll
            for (int gp = 0; gp < 2; ++gp) {                 // channels 32c + 16gp .. +15
                uint4 kq[2];
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
                    kq[nt] = *reinterpret_cast<const uint4*>(st + (8 * nt + g) * kHeadDim + 32 * c + 16 * gp);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const int ks = 4 * gp + kk;              // channels 32c + 4ks .. +3
                    const uint32_t A[4] = {qf[2 * ks], 0u, qf[2 * ks + 1], 0u};
#pragma unroll
                    for (int nt = 0; nt < 2; ++nt) {
                        const uint32_t w = word_of(kq[nt], kk);
                        if constexpr (kInt8) {
                            const uint32_t wx = w ^ 0x80808080u;
                            mma16816(dc[nt], A, s8x2_to_h2(wx, kSel01), s8x2_to_h2(wx, kSel23));
                        } else {
                            mma16816(dc[nt], A, e4m3x2_to_h2(w), e4m3x2_to_h2(w >> 16));
                        }
                    }
                }
            }
            if constexpr (kInt8) {
                constexpr int kCalls = (kBits == 10) ? 4 : 2;     // Philox calls per token
                constexpr int kBatch = (kBits == 10) ? 2 : 2;     // calls per token in flight
#pragma unroll
                for (int g0 = 0; g0 < kCalls; g0 += kBatch) {
                  uint4 dkb[kBatch][2];
#pragma unroll
                  for (int bi = 0; bi < kBatch; ++bi)
#pragma unroll
                    for (int nt = 0; nt < 2; ++nt)
                        dkb[bi][nt] = philox(slot0 + 8 * nt + g, c1, (uint32_t)(kCalls * c + g0 + bi), 0u, p.keys);
#pragma unroll
                  for (int bi = 0; bi < kBatch; ++bi) {
                    const int gi = g0 + bi;
                    const uint4* dk = dkb[bi];
                    constexpr int kSteps = 8 / kCalls;            // k-steps covered by one call
#pragma unroll
                    for (int kk = 0; kk < kSteps; ++kk) {
                        const int ks = kSteps * gi + kk;
                        const uint32_t A[4] = {qf[2 * ks], 0u, qf[2 * ks + 1], 0u};
#pragma unroll
                        for (int nt = 0; nt < 2; ++nt) {
                            uint32_t h0, h1;
                            if constexpr (kBits == 8) {
                                const uint32_t dw = word_of(dk[nt], kk);
                                h0 = h8(dw, kSel01);
                                h1 = h8(dw, kSel23);
                            } else {
                                h0 = h10(word_of(dk[nt], 2 * kk));
                                h1 = h10(word_of(dk[nt], 2 * kk + 1));
                            }
                            mma16816(dd[nt], A, h0, h1);
                        }
                    }
                  }
                }
            }

            // ---------------- logits, bound, softmax --------------------------
            float y[2][2], cb[2][2], sv[2][2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                float db[4] = {0.f, 0.f, 0.f, 0.f};
                const uint32_t wreg = *reinterpret_cast<const uint32_t*>(
                    st + kOffW + ((8 * nt + g) * kBands + 2 * c) * 2);
                mma1688(db, a_hi, 0u, wreg);
                mma1688(db, a_lo, 0u, wreg);
                float sk0 = 1.f, sk1 = 1.f;
                if constexpr (kInt8) {
                    const float2 sk = __half22float2(
                        *reinterpret_cast<const __half2*>(st + kOffKs + (8 * nt + 2 * c) * 2));
                    const float2 vv = __half22float2(
                        *reinterpret_cast<const __half2*>(st + kOffVs + (8 * nt + 2 * c) * 2));
                    sk0 = sk.x; sk1 = sk.y;
                    sv[nt][0] = vv.x; sv[nt][1] = vv.y;
                } else {
                    sv[nt][0] = sv[nt][1] = 1.f;
                }
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int t = 8 * nt + 2 * c + e;
                    const float raw = kInt8 ? (dc[nt][e] - dd[nt][e] + zoff) : dc[nt][e];
                    const bool ok = t < nvalid;
                    y[nt][e] = ok ? raw * ((e ? sk1 : sk0) * kRsdLog2e) : -INFINITY;
                    cb[nt][e] = ok ? db[e] : 0.f;   // tail slots may hold any bits
                    if (!ok) sv[nt][e] = 0.f;
                }
            }
            float mx = fmaxf(fmaxf(y[0][0], y[0][1]), fmaxf(y[1][0], y[1][1]));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const bool move = mx > m_run + 8.0f;
            if (__any_sync(0xffffffffu, move)) {
                const float alpha = move ? (m_run == -INFINITY ? 0.f : fast_exp2(m_run - mx)) : 1.f;
                if (move) m_run = mx;
                l_part *= alpha;
                d_part *= alpha;
                spv_part *= alpha;
                const float a0 = __shfl_sync(0xffffffffu, alpha, 8 * c);      // head 2c
                const float a1 = __shfl_sync(0xffffffffu, alpha, 8 * c + 4);  // head 2c+1
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    acc[mt][0] *= a0; acc[mt][2] *= a0;
                    acc[mt][1] *= a1; acc[mt][3] *= a1;
                }
            }
            float P[2][2];
            float smax = 0.f;
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float pe = fast_exp2(y[nt][e] - m_run);    // 0 for masked tokens
                    l_part += pe;
                    d_part = fmaf(pe, fast_exp2(cb[nt][e] * kLog2e) - 1.f, d_part);
                    const float pv = pe * sv[nt][e];
                    spv_part += pv;
                    P[nt][e] = pv;
                    smax = fmaxf(smax, sv[nt][e]);
                }
            if constexpr (kInt8) {
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
            const float lam = pow2(lam_exp == INT_MIN ? 0 : lam_exp);
            // B = P^T as a sum of two fp16 terms (hi + lo): the output is a
            // sum with heavy cancellation, so one fp16 rounding of P is not
            // accurate enough.  Tokens 2c, 2c+1 (b*0) and 8+2c, 9+2c (b*1).
            uint32_t bp0, bp1, bl0, bl1;
            {
                const float x00 = P[0][0] * lam, x01 = P[0][1] * lam, x10 = P[1][0] * lam, x11 = P[1][1] * lam;
                bp0 = pack_h2(x00, x01);
                bp1 = pack_h2(x10, x11);
                const float2 r0 = __half22float2(*reinterpret_cast<const __half2*>(&bp0));
                const float2 r1 = __half22float2(*reinterpret_cast<const __half2*>(&bp1));
                bl0 = pack_h2(x00 - r0.x, x01 - r0.y);
                bl1 = pack_h2(x10 - r1.x, x11 - r1.y);
            }

            // ---------------- PV: acc[dim][head] ------------------------------
            const int tv[4] = {2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9};
            uint4 vq[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                vq[j] = *reinterpret_cast<const uint4*>(st + kOffV + tv[j] * kHeadDim + 16 * g);
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
        }
        __syncwarp();
        issue(k + kStages);
    }
    if (failed) {
        // let copies still in flight land before the CTA's smem is released
        for (int k = consumed; k < min(n_my, consumed + kStages); ++k)
            (void)mbar_wait_bounded(&bars[k % kStages], (uint32_t)((k / kStages) & 1));
    }

    // ---- warp partials -> shared, merge the warps of this CTA ----------------------
#pragma unroll
    for (int o = 1; o < 4; o <<= 1) {
        l_part += __shfl_xor_sync(0xffffffffu, l_part, o);
        d_part += __shfl_xor_sync(0xffffffffu, d_part, o);
        spv_part += __shfl_xor_sync(0xffffffffu, spv_part, o);
    }
    const float inv_lam = kInt8 ? pow2(lam_exp == INT_MIN ? 0 : -lam_exp) : pow2(-lam_exp);
    const float kap = kInt8 ? DitherConst<kBits == 10 ? 10 : 8>::kappa : 0.f;
    const float spv0 = __shfl_sync(0xffffffffu, spv_part, 8 * c);
    const float spv1 = __shfl_sync(0xffffffffu, spv_part, 8 * c + 4);
    __syncthreads();   // stage buffers are reused below
    float* mbuf = reinterpret_cast<float*>(smem);   // [warp][head][kPartialStride]
    {
        float* wb = mbuf + warp * kMaxGroup * kPartialStride;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
            const int d0 = 16 * g + 2 * mt;
            wb[(2 * c) * kPartialStride + d0] = fmaf(acc[mt][0], inv_lam, kap * spv0);
            wb[(2 * c + 1) * kPartialStride + d0] = fmaf(acc[mt][1], inv_lam, kap * spv1);
            wb[(2 * c) * kPartialStride + d0 + 1] = fmaf(acc[mt][2], inv_lam, kap * spv0);
            wb[(2 * c + 1) * kPartialStride + d0 + 1] = fmaf(acc[mt][3], inv_lam, kap * spv1);
        }
        if (c == 0) {
            wb[g * kPartialStride + kHeadDim + 0] = m_run;
            wb[g * kPartialStride + kHeadDim + 1] = l_part;
            wb[g * kPartialStride + kHeadDim + 2] = d_part;
        }
    }
    __syncthreads();
    const size_t unit = (size_t)b * p.num_kv_heads + h;
    float* part_out = p.partials + (unit * p.splits + split) * (kMaxGroup * kPartialStride);
    float* wts = reinterpret_cast<float*>(smem) + kWarps * kMaxGroup * kPartialStride;   // [head][warp]
    if (threadIdx.x < kMaxGroup) {
        const int hh = threadIdx.x;
        float M = -INFINITY;
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim]);
        for (int w = 0; w < kWarps; ++w) {
            const float mw = mbuf[(w * kMaxGroup + hh) * kPartialStride + kHeadDim];
            wts[hh * (kWarps + 1) + w] = (mw == -INFINITY) ? 0.f : fast_exp2(mw - M);
        }
        wts[hh * (kWarps + 1) + kWarps] = M;
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < G * (kHeadDim + 3); idx += kThreads) {
        const int hh = idx / (kHeadDim + 3), col = idx % (kHeadDim + 3);
        const float* wh = wts + hh * (kWarps + 1);
        float v = wh[kWarps];   // M
        if (col != kHeadDim) {
            v = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) v = fmaf(wh[w], mbuf[(w * kMaxGroup + hh) * kPartialStride + col], v);
        }
        part_out[hh * kPartialStride + col] = v;
    }
    // the merge kernel (launched as a programmatic dependent) may start now;
    // it waits for this whole grid before reading the partials
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Merge of the per-split partials of one (sequence, query head), 32 output
// dims per CTA: out = sum_s w_s acc_s / sum_s w_s l_s with w_s = 2^(m_s - M),
// D = sum_s w_s D_s / sum_s w_s l_s, meter_raw = D (D + 2) / 2 (§6.2.2: the
// meter accumulator merges under the same LSE weights as the output).
constexpr int kMergeWarps = 8;

__global__ void __launch_bounds__(32 * kMergeWarps) merge_kernel(const __grid_constant__ DecodeParams p) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int chunk = blockIdx.x, hq = blockIdx.y, b = blockIdx.z;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int h = hq / p.group, hh = hq % p.group;
    const size_t unit = (size_t)b * p.num_kv_heads + h;
    const float* base = p.partials + unit * p.splits * (kMaxGroup * kPartialStride) + hh * kPartialStride;
    const size_t split_stride = kMaxGroup * kPartialStride;
    __shared__ float red[kMergeWarps][36];
    __shared__ float sM;

    float M = -INFINITY;
#pragma unroll 4
    for (int s = warp; s < p.splits; s += kMergeWarps) M = fmaxf(M, __ldcg(base + s * split_stride + kHeadDim));
    if (lane == 0) red[warp][0] = M;
    __syncthreads();
    if (threadIdx.x == 0) {
        float m = -INFINITY;
        for (int w = 0; w < kMergeWarps; ++w) m = fmaxf(m, red[w][0]);
        sM = m;
    }
    __syncthreads();
    M = sM;
    float acc = 0.f, L = 0.f, Dn = 0.f;
    if (M != -INFINITY) {
#pragma unroll 4
        for (int s = warp; s < p.splits; s += kMergeWarps) {
            const float* ps = base + s * split_stride;
            const float ms = __ldcg(ps + kHeadDim);
            const float w = (ms == -INFINITY) ? 0.f : fast_exp2(ms - M);
            acc = fmaf(w, __ldcg(ps + 32 * chunk + lane), acc);
            L = fmaf(w, __ldcg(ps + kHeadDim + 1), L);
            Dn = fmaf(w, __ldcg(ps + kHeadDim + 2), Dn);
        }
    }
    __syncthreads();
    red[warp][lane] = acc;
    if (lane == 0) {
        red[warp][32] = L;
        red[warp][33] = Dn;
    }
    __syncthreads();
    if (warp == 0) {
        float a = 0.f, l = 0.f, dn = 0.f;
#pragma unroll
        for (int w = 0; w < kMergeWarps; ++w) {
            a += red[w][lane];
            l += red[w][32];
            dn += red[w][33];
        }
        const size_t cell = (size_t)b * p.num_q_heads + hq;
        p.out[cell * kHeadDim + 32 * chunk + lane] = l > 0.f ? a / l : 0.f;
        if (chunk == 0 && lane == 0) {
            float raw = 0.f;
            if (l > 0.f) {
                const float D = dn / l;                 // A - 1
                raw = 0.5f * D * (D + 2.0f);            // (A^2 - 1) / 2, +inf on overflow
            }
            p.meter_raw[cell] = raw;
            p.meter[cell] = fminf(1.0f, raw);
        }
    }
}

}  // namespace

DecodePlan plan_decode(int batch, int num_kv_heads, int max_pages, int num_sms) {
    DecodePlan pl;
    const long units = (long)batch * num_kv_heads;
    const long target = (long)num_sms * kMinBlocks;   // resident CTAs
    long pps = (max_pages * units + target - 1) / target;
    pps = std::max<long>(pps, 16);
    pps = std::min<long>(pps, std::max(max_pages, 1));
    pl.pages_per_split = (int)pps;
    pl.splits = (int)std::max<long>(1, (max_pages + pps - 1) / pps);
    auto align = [](size_t x) { return (x + 255) & ~(size_t)255; };
    pl.counters_off = 256;
    pl.partials_off = 256;
    pl.total = align(pl.partials_off + sizeof(float) * (size_t)units * pl.splits * kMaxGroup * kPartialStride);
    return pl;
}

template <int kScheme, int kBits>
static cudaError_t launch_one(const DecodeParams& p, cudaStream_t stream) {
    static bool configured = false;   // per process; the attribute is per function
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(decode_kernel<kScheme, kBits>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    dim3 grid(p.splits, p.num_kv_heads, p.batch);
    cudaError_t e = launch_pdl(decode_kernel<kScheme, kBits>, grid, dim3(kThreads), kSmemBytes, stream, p);
    if (e != cudaSuccess) return e;
    // the merge is a programmatic dependent too: its CTAs are scheduled while
    // the decode grid drains and wait (griddepcontrol.wait) for all of it
    return launch_pdl(merge_kernel, dim3(kHeadDim / 32, p.num_q_heads, p.batch), dim3(32 * kMergeWarps), 0,
                      stream, p);
}

cudaError_t launch_decode(const DecodeParams& p, int scheme, int bits, cudaStream_t stream) {
    if (p.batch == 0) return cudaSuccess;
    if (scheme == WC_SCHEME_FP8_E4M3) return launch_one<WC_SCHEME_FP8_E4M3, 8>(p, stream);
    if (bits == 8) return launch_one<WC_SCHEME_DITHER_INT8, 8>(p, stream);
    return launch_one<WC_SCHEME_DITHER_INT8, 10>(p, stream);
}

}  // namespace wc
