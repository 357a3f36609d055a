// One row of the write path (quantize, witness, store), shared by the write
// kernel and by the decode variant that appends the step's new token
// (§6.2.1 write kernel; §4.1 Eq. witness; §4.2 subtractive dither; §6.2.3
// grouped scales and bypass).  8 lanes per row, 16 channels per lane; the
// whole warp calls it (full-warp shuffles), lanes of other rows not live.
#pragma once

#include <type_traits>

#include "wc_kernels.cuh"

namespace wc {

namespace {

// Quantizer: code = round-half-even of the exact real v = x/s + xi, clamped to
// [-127, 127].  With s a normal fp16, s >= (amax / 126.5)(1 - 2^-24)(1 - 2^-11),
// so |x/s| <= 126.57 and |v| < 127.07: the clamp cannot bind.  The fp32
// estimate est = fma(x, 1/s, xi), 1/s as recip_scale gives it, then differs from v by at most
// |x/s| (2^-24 + 2^-46) (the reciprocal) + ulp(est)/2 < 7.6e-6 + 3.9e-6 < 1.2e-5, so
// rounding est gives round(v) unless est lies within 1.2e-5 of a half-integer.
// The fast pass flags estimates within 2e-5 of a tie (4 elements in 10^5).
// Flagged rows, and rows whose scale is an fp16 subnormal (where the clamp
// matters), are re-decided exactly: the FMA residual x - s*(k +- 1/2 - xi)
// has exactly the sign of s*(v - (k +- 1/2)), because k +- 1/2 - xi is exact
// in fp32.
__device__ __forceinline__ float exact_round(float x, float s, float xi, float k) {
    const float up = fmaf(-s, k + 0.5f - xi, x);   // sign of x/s + xi - (k + 1/2)
    const float dn = fmaf(-s, k - 0.5f - xi, x);   // sign of x/s + xi - (k - 1/2)
    const bool k_odd = (__float_as_uint(k + 12582912.0f) & 1u) != 0u;
    if (up > 0.0f || (up == 0.0f && k_odd)) k += 1.0f;
    else if (dn < 0.0f || (dn == 0.0f && k_odd)) k -= 1.0f;
    return fminf(127.0f, fmaxf(-127.0f, k));
}

// fp32(amax) / 126.5 rounded to nearest even, for amax a non-negative fp16 value
// or +inf: q0 = amax * RN(1/126.5), then one correction with the exact remainder
// amax - q0 * 126.5 (Markstein, IBM J. Res. Dev. 34(1), 1990).  For every finite
// fp16 amax the result equals the IEEE quotient (checked exhaustively with exact
// rational arithmetic in tests/test_write_scale.py).
__device__ __forceinline__ float div_126_5(float amax) {
    constexpr float kInv = 0x1.03091cp-7f;   // RN(1 / 126.5)
    const float q0 = amax * kInv;
    const float r = fmaf(-q0, 126.5f, amax);
    return amax == INFINITY ? amax : fmaf(r, kInv, q0);
}

// 1/s for a positive fp16 scale s (0 for +inf): rcp.approx (documented within
// one ulp) refined by one Newton-Raphson step y (2 - s y).  The step squares the
// approximation's relative error e (to e^2 < 2^-46 for |e| <= 2^-23; below 2^-24
// still for any |e| <= 2^-12) and its final fma rounds once, so the result lies
// within 2^-24 + 2^-46 of 1/s relative: the reciprocal error the estimate bound
// above allows.
__device__ __forceinline__ float recip_scale(float s) {
    if (!(s < INFINITY)) return 0.0f;
    float y;
    asm("rcp.approx.f32 %0, %1;" : "=f"(y) : "f"(s));
    return fmaf(y, fmaf(-s, y, 1.0f), y);
}

// Norm for a witness, rounded up to fp16: the smallest fp16 h with
// h * h >= S, S = sum inflated by 2^-18 (rounded up), which covers the fp32
// accumulation error of the sum (a band: 16 squares, < 2^-20 relative; a
// whole row: 128 squares in 16 FMAs and 3 shuffle adds per lane, < 2^-19.7).  So h is never below the
// exact norm rounded up and at most one fp16 step above it.  h * h is exact in
// fp32 (11 significant bits), so one check on each side of the rounded-up
// approximate root fixes it.
__device__ __forceinline__ __half norm_up_fp16(float sum) {
    const float S = __fmul_ru(sum, 1.0f + 1.0f / (1 << 18));
    float y;
    asm("sqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(S));
    unsigned short hb = __half_as_ushort(__float2half_ru(y));
    const float hf = __half2float(__ushort_as_half(hb));
    if (hf * hf < S) {
        ++hb;
    } else if (hb != 0) {
        const float pf = __half2float(__ushort_as_half((unsigned short)(hb - 1)));
        if (pf * pf >= S) --hb;
    }
    return __ushort_as_half(hb);
}

// Rounding bias 1.5 * 2^23: for |k| < 2^22, t = k + kBias holds k exactly and
// the low byte of its bits is k's two's-complement byte.
constexpr float kBias = 12582912.0f;

// Dither word byte (i % 4) placed as the float 1 + j/2^15 (bits 0x3F80jj00).
__device__ __forceinline__ uint32_t xi_sel(int i) { return 0x7604u | ((uint32_t)(i & 3) << 4); }

// x[i] for a lane-uniform runtime index i in [0, 16), without local memory.
__device__ __forceinline__ float pick16(const float (&x)[16], int i) {
    float v = x[0];
#pragma unroll
    for (int k = 1; k < 16; ++k) v = (i == k) ? x[k] : v;
    return v;
}

// Bypass set of one KV head in shared memory (grouped scheme, per-head grid):
// the bypassed channels as a 128-bit mask, the k_bypass entry of each channel
// (-1: not bypassed), and the pairs whose index is out of range.
struct BypassTable {
    uint32_t mask[4];
    uint32_t bad;
    int8_t entry[kHeadDim];
};

// Row stride of the grouped scheme's shared rows: 160 bytes puts the four
// units of a warp on distinct bank groups.
constexpr int kXRowStride = 160;

// One row (K or V) of one (token, KV head): 8 lanes, 16 channels each.
// xrow: the unit's shared row (grouped scheme only); tab: the head's bypass
// table, or nullptr (then each K row reads the pair list itself).
// pre_w: this lane's dither word of the row when the caller drew it already
// (8-bit dither; several rows' calls advanced together), else nullptr.
template <int kScheme, int kBits>
__device__ __forceinline__ void write_row(const WriteParams& p, uint4 (&raw)[2], int slot, bool live_unit, int h,
                                          int row, int sub, uint8_t* xrow, const BypassTable* tab,
                                          const uint4* pre_w = nullptr) {
    constexpr bool kGrouped = kScheme == WC_SCHEME_DITHER_INT8_G32;
    constexpr bool kDither = kScheme != WC_SCHEME_FP8_E4M3;
    const bool bad = slot >= p.num_pages * kPage;
    const bool active = live_unit && slot >= 0 && !bad;
    if (live_unit && bad && sub == 0 && row == 0 && p.dev_status) atomicOr(p.dev_status, WC_DEV_BAD_SLOT);
    if (!active) raw[0] = raw[1] = make_uint4(0, 0, 0, 0);
    float x[16];
    {
        const __half2* hv = reinterpret_cast<const __half2*>(raw);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const float2 f = __half22float2(hv[i]);
            x[2 * i] = f.x;
            x[2 * i + 1] = f.y;
        }
    }

    uint32_t codes[4];
    // K rows, and V rows when the value witness is stored: squared residual
    // sums over dims 16*sub + [0,8), + [8,16)
    float lo = 0.0f, hi = 0.0f;
    const bool resid = row == 0 || p.v_witness != nullptr;   // warp-uniform
    float s = 0.0f;
    uint32_t bmask = 0;   // grouped K rows: bypassed channels among 16 sub .. 16 sub + 15
    if constexpr (kGrouped) {
        if (row == 0 && tab != nullptr) {
            bmask = (tab->mask[sub >> 1] >> (16 * (sub & 1))) & 0xFFFFu;
        } else if (row == 0) {
            const int32_t* pr = p.bypass_pairs + (size_t)h * p.num_bypass;
            for (int t = 0; t < p.num_bypass; ++t) {
                const int j = __ldg(pr + t);
                if (j < 0 || j >= kHeadDim / 2) {
                    if (live_unit && sub == 0 && p.dev_status) atomicOr(p.dev_status, WC_DEV_BAD_PAIR);
                    continue;
                }
                const int a = p.rope_layout == WC_ROPE_HALF ? j : 2 * j;
                const int b = p.rope_layout == WC_ROPE_HALF ? j + kHeadDim / 2 : 2 * j + 1;
                if ((a >> 4) == sub) bmask |= 1u << (a & 15);
                if ((b >> 4) == sub) bmask |= 1u << (b & 15);
            }
        }
    }
    if constexpr (kDither) {
        float amax = 0.0f;
#pragma unroll
        for (int i = 0; i < 16; ++i) amax = fmaxf(amax, ((bmask >> i) & 1u) ? 0.0f : fabsf(x[i]));
        // the row (8 lanes) or the 32-channel group (a lane pair)
#pragma unroll
        for (int o = 1; o < (kGrouped ? 2 : 8); o <<= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        __half sh = __float2half_rn(div_126_5(amax));
        if (__half_as_ushort(sh) == 0 && amax > 0.0f) sh = __ushort_as_half((unsigned short)1);
        s = __half2float(sh);
        const float inv_s = s > 0.0f ? recip_scale(s) : 0.0f;

        // dither words for channels 16*sub .. 16*sub + 15
        const uint32_t slot_u = (uint32_t)max(slot, 0);
        const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;
        uint32_t dw[8];
        if constexpr (kBits == 8) {
            const uint4 w = pre_w ? *pre_w : philox(slot_u, c1, (uint32_t)sub, (uint32_t)row, p.keys);
            dw[0] = w.x; dw[1] = w.y; dw[2] = w.z; dw[3] = w.w;
            if constexpr (kGrouped) {
                // storage-position bytes -> this lane's channels 16 sub + i
                __syncwarp();
                *reinterpret_cast<uint4*>(xrow + 16 * sub) = w;
                __syncwarp();
                if (row == 0) {   // channel 16 sub + 4q + j is at position 32q + 4 sub + j
#pragma unroll
                    for (int q = 0; q < 4; ++q) dw[q] = *reinterpret_cast<const uint32_t*>(xrow + 32 * q + 4 * sub);
                } else {          // channel 16 sub + 8e + g is at position 16g + 2 sub + e
                    uint32_t u[8];
#pragma unroll
                    for (int g = 0; g < 8; ++g) u[g] = *reinterpret_cast<const uint16_t*>(xrow + 16 * g + 2 * sub);
                    const uint32_t t01 = u[0] | (u[1] << 16), t23 = u[2] | (u[3] << 16);
                    const uint32_t t45 = u[4] | (u[5] << 16), t67 = u[6] | (u[7] << 16);
                    dw[0] = prmt(t01, t23, 0x6420u);   // e = 0, g = 0..3
                    dw[1] = prmt(t45, t67, 0x6420u);   // e = 0, g = 4..7
                    dw[2] = prmt(t01, t23, 0x7531u);   // e = 1, g = 0..3
                    dw[3] = prmt(t45, t67, 0x7531u);   // e = 1, g = 4..7
                }
            }
        } else {
#pragma unroll
            for (int gi = 0; gi < 2; ++gi) {
                const uint4 w = philox(slot_u, c1, (uint32_t)(2 * sub + gi), (uint32_t)row, p.keys);
                dw[4 * gi + 0] = w.x; dw[4 * gi + 1] = w.y; dw[4 * gi + 2] = w.z; dw[4 * gi + 3] = w.w;
            }
        }
        // With s a normal fp16 (or 0), |x| <= amax <= 126.5 s (1 + 2^-11), so
        // |x/s + xi| < 127.06 and the clamp to [-127, 127] cannot bind; only rows
        // whose scale fell into the fp16 subnormals need it.
        const bool need_clamp = !__all_sync(0xffffffffu, s == 0.0f || s >= 6.103515625e-05f);
        // xi = (j + 1/2)/N - 1/2 built exactly from the bits of j (recomputed
        // where needed rather than held in registers)
        auto xi_of = [&](int i) -> float {
            if constexpr (kBits == 8) {
                // 1 + j/2^15 from one byte permute; 128 (1 + j/2^15) - (128 + 255/512)
                // = (j + 1/2)/256 - 1/2 is exact in one fma
                const float f = __uint_as_float(prmt(dw[i >> 2], 0x3F800000u, xi_sel(i)));
                return fmaf(f, 128.0f, -128.498046875f);
            } else {
                const int sh = 16 * (i & 1);             // field i%2 of word i/2
                const uint32_t mant = ((dw[i >> 1] >> sh) & 0x3FFu) << 13;
                constexpr float kOff = 1.0f + 1023.0f / 2048.0f;
                return __uint_as_float(0x3F800000u | mant) - kOff;
            }
        };
        uint32_t tb[16];   // bits of t = k + kBias: the low byte is the code
        // Fast pass (no clamp): round the fp32 estimate, track its largest
        // distance from the rounded value and, in K warps, accumulate the
        // squared residual on the way.  A warp in which some estimate lies
        // within 2e-5 of a tie, or whose rows need the clamp, redoes its rows
        // exactly below (about one warp in fifty, and rows with tiny amax).
        auto fast_pass = [&](auto with_residual) -> float {
            float dev = 0.0f;
            if constexpr (!kGrouped && kBits == 8) {
                // Channel pairs on the packed fp32x2 path: each lane of __ffma2_rn /
                // __fadd2_rn rounds like the scalar fmaf / add, so est, t, k and r are
                // the scalar pass's bits.  est - k and k - xi are taken as fma(-1, k,
                // est) and fma(-1, xi, k) (exact products, the same roundings), and
                // r = fma(-s, k - xi, x) is the residual with its sign flipped.  The
                // squared residuals sum in two chains per half; the 2^-18 margin of
                // norm_up_fp16 covers the fp32 error of any summation order.
                const float2 inv2 = make_float2(inv_s, inv_s), ns2 = make_float2(-s, -s);
                const float2 m1 = make_float2(-1.0f, -1.0f), c128 = make_float2(128.0f, 128.0f);
                const float2 off = make_float2(-128.498046875f, -128.498046875f);
                const float2 pb = make_float2(kBias, kBias), nb = make_float2(-kBias, -kBias);
                float2 alo = make_float2(0.0f, 0.0f), ahi = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int i = 0; i < 16; i += 2) {
                    const float2 f = make_float2(__uint_as_float(prmt(dw[i >> 2], 0x3F800000u, xi_sel(i))),
                                                 __uint_as_float(prmt(dw[(i + 1) >> 2], 0x3F800000u, xi_sel(i + 1))));
                    const float2 xi = __ffma2_rn(f, c128, off);   // (j + 1/2)/256 - 1/2, as xi_of
                    const float2 x2 = make_float2(x[i], x[i + 1]);
                    const float2 est = __ffma2_rn(x2, inv2, xi);
                    const float2 t = __fadd2_rn(est, pb);
                    const float2 k = __fadd2_rn(t, nb);
                    const float2 d = __ffma2_rn(k, m1, est);
                    dev = fmaxf(dev, fmaxf(fabsf(d.x), fabsf(d.y)));
                    tb[i] = __float_as_uint(t.x);
                    tb[i + 1] = __float_as_uint(t.y);
                    if constexpr (decltype(with_residual)::value) {
                        const float2 r = __ffma2_rn(ns2, __ffma2_rn(xi, m1, k), x2);
                        if (i < 8) alo = __ffma2_rn(r, r, alo);
                        else ahi = __ffma2_rn(r, r, ahi);
                    }
                }
                if constexpr (decltype(with_residual)::value) {
                    lo = alo.x + alo.y;
                    hi = ahi.x + ahi.y;
                }
                return dev;
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const bool byp = kGrouped && ((bmask >> i) & 1u);   // exact channel: code 0, no residual
                    const float xi = xi_of(i);
                    const float est = byp ? 0.0f : fmaf(x[i], inv_s, xi);   // s = 0: x = 0, est = xi, k = 0
                    const float t = est + kBias;
                    const float k = t - kBias;
                    dev = fmaxf(dev, fabsf(est - k));
                    tb[i] = __float_as_uint(t);
                    if constexpr (decltype(with_residual)::value) {
                        const float r = byp ? 0.0f : fmaf(s, k - xi, -x[i]);   // x^ - x, one rounding
                        if (i < 8) lo = fmaf(r, r, lo);
                        else hi = fmaf(r, r, hi);
                    }
                }
                return dev;
            }
        };
        bool exact = need_clamp;
        if (!exact) {
            const float dev = resid ? fast_pass(std::true_type{}) : fast_pass(std::false_type{});
            exact = __any_sync(0xffffffffu, dev > 0.49998f);
        }
        if (exact) {
            lo = hi = 0.0f;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const bool byp = kGrouped && ((bmask >> i) & 1u);
                const float xi = xi_of(i);
                const float est = fminf(127.0f, fmaxf(-127.0f, fmaf(x[i], inv_s, xi)));
                const float k = byp ? 0.0f : exact_round(x[i], s, xi, (est + kBias) - kBias);
                tb[i] = __float_as_uint(k + kBias);
                if (resid) {
                    const float r = byp ? 0.0f : fmaf(s, k - xi, -x[i]);
                    if (i < 8) lo = fmaf(r, r, lo);
                    else hi = fmaf(r, r, hi);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
            codes[i] = prmt(prmt(tb[4 * i], tb[4 * i + 1], 0x0040u), prmt(tb[4 * i + 2], tb[4 * i + 3], 0x0040u),
                            0x5410u);
        if constexpr (kGrouped) {   // channel order -> storage order
            __syncwarp();
            if (row == 0) {
#pragma unroll
                for (int q = 0; q < 4; ++q) *reinterpret_cast<uint32_t*>(xrow + 32 * q + 4 * sub) = codes[q];
            } else {
#pragma unroll
                for (int g = 0; g < 8; ++g)   // bytes of channels 16 sub + g and 16 sub + 8 + g
                    *reinterpret_cast<uint16_t*>(xrow + 16 * g + 2 * sub) =
                        (uint16_t)((tb[g] & 0xFFu) | ((tb[8 + g] & 0xFFu) << 8));
            }
            __syncwarp();
            const uint4 st = *reinterpret_cast<const uint4*>(xrow + 16 * sub);
            codes[0] = st.x; codes[1] = st.y; codes[2] = st.z; codes[3] = st.w;
        }
    } else {
        const uint32_t* hw = reinterpret_cast<const uint32_t*>(raw);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            uint16_t c2;
            asm("cvt.rn.satfinite.e4m3x2.f16x2 %0, %1;" : "=h"(c2) : "r"(hw[i]));
            const uint32_t cc = (uint32_t)c2;   // low half -> low byte
            if ((i & 1) == 0) codes[i >> 1] = cc;
            else codes[i >> 1] |= cc << 16;
            if (resid) {
                const uint32_t back = e4m3x2_to_h2(cc);
                const float2 xr = __half22float2(*reinterpret_cast<const __half2*>(&back));
                const float r0 = xr.x - x[2 * i], r1 = xr.y - x[2 * i + 1];
                if (i < 4) lo = fmaf(r1, r1, fmaf(r0, r0, lo));
                else hi = fmaf(r1, r1, fmaf(r0, r0, hi));
            }
        }
    }

    // ---- stores ------------------------------------------------------------
    const int page = active ? slot / kPage : 0, off = slot & (kPage - 1);
    const size_t rowidx = ((size_t)page * p.num_kv_heads + h) * kPage + off;
    if (active) {
        uint8_t* dst = static_cast<uint8_t*>(row == 0 ? p.k_codes : p.v_codes) + rowidx * kHeadDim + sub * 16;
        *reinterpret_cast<uint4*>(dst) = make_uint4(codes[0], codes[1], codes[2], codes[3]);
        if constexpr (kScheme == WC_SCHEME_DITHER_INT8) {
            if (sub == 0) (row == 0 ? p.k_scale : p.v_scale)[rowidx] = __float2half_rn(s);
        }
        if constexpr (kGrouped) {
            if ((sub & 1) == 0) (row == 0 ? p.k_scale : p.v_scale)[rowidx * 4 + (sub >> 1)] = __float2half_rn(s);
            if (row == 0 && p.num_bypass > 0 && tab != nullptr) {
                __half* bdst = p.k_bypass + rowidx * (2 * p.num_bypass);
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    if ((bmask >> i) & 1u) bdst[tab->entry[16 * sub + i]] = __float2half_rn(x[i]);
                if (sub == 0)   // an ignored pair stores zeros
                    for (uint32_t bad = tab->bad; bad != 0u; bad &= bad - 1u) {
                        const int t = __ffs(bad) - 1;
                        bdst[2 * t] = bdst[2 * t + 1] = __float2half_rn(0.0f);
                    }
            } else if (row == 0 && p.num_bypass > 0) {   // the exact values of the bypassed pairs, pair by pair
                const int32_t* pr = p.bypass_pairs + (size_t)h * p.num_bypass;
                __half* bdst = p.k_bypass + rowidx * (2 * p.num_bypass);
                uint32_t seen = 0;   // this lane's channels stored already: a repeated pair stores zeros
                for (int t = 0; t < p.num_bypass; ++t) {
                    const int j = __ldg(pr + t);
                    if (j < 0 || j >= kHeadDim / 2) {   // an ignored pair stores zeros
                        if (sub == 0) bdst[2 * t] = bdst[2 * t + 1] = __float2half_rn(0.0f);
                        continue;
                    }
                    const int a = p.rope_layout == WC_ROPE_HALF ? j : 2 * j;
                    const int b = p.rope_layout == WC_ROPE_HALF ? j + kHeadDim / 2 : 2 * j + 1;
                    if ((a >> 4) == sub) {
                        const bool again = (seen >> (a & 15)) & 1u;
                        bdst[2 * t] = __float2half_rn(again ? 0.0f : pick16(x, a & 15));
                        if (again && live_unit && p.dev_status) atomicOr(p.dev_status, WC_DEV_BAD_PAIR);
                        seen |= 1u << (a & 15);
                    }
                    if ((b >> 4) == sub) {
                        const bool again = (seen >> (b & 15)) & 1u;
                        bdst[2 * t + 1] = __float2half_rn(again ? 0.0f : pick16(x, b & 15));
                        seen |= 1u << (b & 15);
                    }
                }
            }
        }
    }
    if (row != 0) {   // warp-uniform
        if (p.v_witness != nullptr) {
            // value witness (§3 output bound): ||v^ - v|| and ||v|| of the row, rounded up
            float rr = lo + hi, vv = 0.0f;
#pragma unroll
            for (int i = 0; i < 16; ++i) vv = fmaf(x[i], x[i], vv);
#pragma unroll
            for (int o = 1; o < 8; o <<= 1) {
                rr += __shfl_xor_sync(0xffffffffu, rr, o);
                vv += __shfl_xor_sync(0xffffffffu, vv, o);
            }
            if (active && sub == 0)
                *reinterpret_cast<__half2*>(p.v_witness + rowidx * 2) =
                    __halves2half2(norm_up_fp16(rr), norm_up_fp16(vv));
        }
        return;
    }

    // ---- witness (K warps) --------------------------------------------------
    const float lo_p = __shfl_xor_sync(0xffffffffu, lo, 4);
    const float hi_p = __shfl_xor_sync(0xffffffffu, hi, 4);
    if (active) {
        __half* wdst = p.k_witness + rowidx * kBands;
        if (p.rope_layout == WC_ROPE_HALF) {
            // dims 16*sub..+7 and +8..+15 are the first (sub < 4) or second
            // (sub >= 4) halves of bands 2*(sub&3) and 2*(sub&3)+1.
            if (sub < 4)
                *reinterpret_cast<__half2*>(wdst + 2 * sub) =
                    __halves2half2(norm_up_fp16(lo + lo_p), norm_up_fp16(hi + hi_p));
        } else {
            wdst[sub] = norm_up_fp16(lo + hi);
        }
    }
}


}  // namespace

}  // namespace wc
