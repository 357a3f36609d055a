// Write path: quantize post-RoPE K/V rows into the paged cache and store the
// K band-norm residual witness (§6.2.1 write kernel; §4.1 Eq. witness;
// §4.2 subtractive dither).
//
// One warp handles two (token, KV head) units.  Lanes 8r .. 8r+7 own row r of
// {K unit0, V unit0, K unit1, V unit1}; each lane owns 16 consecutive
// channels, so it loads 32 B of fp16, stores 16 B of codes, and (for the
// dither scheme) consumes exactly one Philox4x32-10 call per 16 channels.
#include "wc_kernels.cuh"

namespace wc {

namespace {

// Quantizer: code = round-half-even of the exact real x/s + xi, clamped to
// [-127, 127].  The fp32 estimate est = fma(x, 1/s, xi) is within 3e-5 of the
// exact value whenever |est| <= 127.5 (1/s and the product each carry at most
// 2^-24 relative error), so its rounding is exact unless est lies within 1e-4
// of a half-integer (about 2 elements in 10^4); beyond +-127 the clamp
// decides.  Near-ties are re-decided exactly in a separate pass: the FMA
// residual x - s*(k +- 1/2 - xi) has exactly the sign of the exact value,
// because k +- 1/2 - xi is exact in fp32.
__device__ __forceinline__ float exact_round(float x, float s, float xi, float k) {
    const float up = fmaf(-s, k + 0.5f - xi, x);   // sign of x/s + xi - (k + 1/2)
    const float dn = fmaf(-s, k - 0.5f - xi, x);   // sign of x/s + xi - (k - 1/2)
    const bool k_odd = (__float_as_uint(k + 12582912.0f) & 1u) != 0u;
    if (up > 0.0f || (up == 0.0f && k_odd)) k += 1.0f;
    else if (dn < 0.0f || (dn == 0.0f && k_odd)) k -= 1.0f;
    return fminf(127.0f, fmaxf(-127.0f, k));
}

// Low byte of the integer held (exactly) in float k, |k| < 2^22: two's complement.
__device__ __forceinline__ uint32_t code_byte(float k) {
    return __float_as_uint(k + 12582912.0f) & 0xFFu;    // 1.5 * 2^23 bias
}

template <int kScheme, int kBits>
__global__ void __launch_bounds__(128) write_kernel(const __grid_constant__ WriteParams p) {
    grid_dep_wait();      // inputs may come from the preceding kernel
    grid_dep_launch();    // a dependent decode waits for this whole grid anyway
    const int lane = threadIdx.x & 31;
    const int unit = (blockIdx.x * 4 + (threadIdx.x >> 5)) * 2 + (lane >> 4);  // token*Hkv + h
    const int row = (lane >> 3) & 1;                                             // 0 = K, 1 = V
    const int sub = lane & 7;                                                    // 16-channel chunk
    const bool live_unit = unit < p.n_tok * p.num_kv_heads;
    const int tok = live_unit ? unit / p.num_kv_heads : 0;
    const int h = live_unit ? unit % p.num_kv_heads : 0;
    const int slot = live_unit ? __ldg(p.slot_mapping + tok) : -1;
    // the row loads do not depend on the slot: issue them alongside its load
    const __half* src = (row == 0 ? p.k : p.v) + ((size_t)tok * p.num_kv_heads + h) * kHeadDim + sub * 16;
    uint4 raw[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
    if (live_unit) {
        raw[0] = __ldg(reinterpret_cast<const uint4*>(src));
        raw[1] = __ldg(reinterpret_cast<const uint4*>(src) + 1);
    }
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
    float r[16];
    float s = 0.0f;
    if constexpr (kScheme == WC_SCHEME_DITHER_INT8) {
        float amax = 0.0f;
#pragma unroll
        for (int i = 0; i < 16; ++i) amax = fmaxf(amax, fabsf(x[i]));
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        __half sh = __float2half_rn(__fdiv_rn(amax, 126.5f));
        if (__half_as_ushort(sh) == 0 && amax > 0.0f) sh = __ushort_as_half((unsigned short)1);
        s = __half2float(sh);
        const float inv_s = s > 0.0f ? __frcp_rn(s) : 0.0f;

        // dither words for channels 16*sub .. 16*sub + 15
        const uint32_t slot_u = (uint32_t)max(slot, 0);
        const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;
        uint32_t dw[8];
        if constexpr (kBits == 8) {
            const uint4 w = philox(slot_u, c1, (uint32_t)sub, (uint32_t)row, p.keys);
            dw[0] = w.x; dw[1] = w.y; dw[2] = w.z; dw[3] = w.w;
        } else {
#pragma unroll
            for (int gi = 0; gi < 2; ++gi) {
                const uint4 w = philox(slot_u, c1, (uint32_t)(2 * sub + gi), (uint32_t)row, p.keys);
                dw[4 * gi + 0] = w.x; dw[4 * gi + 1] = w.y; dw[4 * gi + 2] = w.z; dw[4 * gi + 3] = w.w;
            }
        }
        uint32_t cb[16];
        float xis[16], ks[16];
        uint32_t near_tie = 0u;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            // xi = (j + 1/2)/N - 1/2 built exactly from the bits of j:
            // (1 + j/N) - (1 + (N-1)/(2N))
            uint32_t mant;
            if constexpr (kBits == 8) {
                const int sh = 8 * (i & 3);              // byte i%4 of word i/4
                mant = ((dw[i >> 2] >> sh) & 0xFFu) << 15;
            } else {
                const int sh = 16 * (i & 1);             // field i%2 of word i/2
                mant = ((dw[i >> 1] >> sh) & 0x3FFu) << 13;
            }
            constexpr float kOff = 1.0f + (float)((1 << kBits) - 1) / (float)(2 << kBits);
            const float xi = __uint_as_float(0x3F800000u | mant) - kOff;   // exact
            // clamp first (values beyond +-127 saturate), then round to nearest
            // even with the 1.5 * 2^23 bias; s = 0 gives x = 0, est = xi, k = 0
            const float est = fminf(127.0f, fmaxf(-127.0f, fmaf(x[i], inv_s, xi)));
            const float kr = (est + 12582912.0f) - 12582912.0f;
            if (fabsf(est - kr) > 0.4999f) near_tie |= 1u << i;
            xis[i] = xi;
            ks[i] = kr;
        }
        if (__any_sync(0xffffffffu, near_tie != 0u)) {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (near_tie & (1u << i)) ks[i] = exact_round(x[i], s, xis[i], ks[i]);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            r[i] = fmaf(s, ks[i] - xis[i], -x[i]);        // x^ - x, one rounding
            cb[i] = code_byte(ks[i]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
            codes[i] = prmt(prmt(cb[4 * i], cb[4 * i + 1], 0x0040u), prmt(cb[4 * i + 2], cb[4 * i + 3], 0x0040u),
                            0x5410u);
    } else {
        const uint32_t* hw = reinterpret_cast<const uint32_t*>(raw);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            uint16_t c2;
            asm("cvt.rn.satfinite.e4m3x2.f16x2 %0, %1;" : "=h"(c2) : "r"(hw[i]));
            const uint32_t cc = (uint32_t)c2;   // low half -> low byte
            if ((i & 1) == 0) codes[i >> 1] = cc;
            else codes[i >> 1] |= cc << 16;
            const uint32_t back = e4m3x2_to_h2(cc);
            const float2 xr = __half22float2(*reinterpret_cast<const __half2*>(&back));
            r[2 * i] = xr.x - x[2 * i];
            r[2 * i + 1] = xr.y - x[2 * i + 1];
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
    }

    // ---- witness (K rows only) --------------------------------------------
    float lo = 0.0f, hi = 0.0f;   // sums over dims 16*sub + [0,8) and + [8,16)
#pragma unroll
    for (int i = 0; i < 8; ++i) lo = fmaf(r[i], r[i], lo);
#pragma unroll
    for (int i = 8; i < 16; ++i) hi = fmaf(r[i], r[i], hi);
    const float lo_p = __shfl_xor_sync(0xffffffffu, lo, 4);
    const float hi_p = __shfl_xor_sync(0xffffffffu, hi, 4);
    if (active && row == 0) {
        // fp32 sums carry < 2^-20 relative error; inflate by that margin
        // before rounding up so the stored witness never under-states.
        constexpr float kMargin = 1.0f + 1.0f / (1 << 19);
        __half* wdst = p.k_witness + rowidx * kBands;
        if (p.rope_layout == WC_ROPE_HALF) {
            // dims 16*sub..+7 and +8..+15 are the first (sub < 4) or second
            // (sub >= 4) halves of bands 2*(sub&3) and 2*(sub&3)+1.
            if (sub < 4) {
                const float b0 = __fmul_ru(__fsqrt_ru(lo + lo_p), kMargin);
                const float b1 = __fmul_ru(__fsqrt_ru(hi + hi_p), kMargin);
                const __half2 w2 = __halves2half2(__float2half_ru(b0), __float2half_ru(b1));
                *reinterpret_cast<__half2*>(wdst + 2 * sub) = w2;
            }
        } else {
            wdst[sub] = __float2half_ru(__fmul_ru(__fsqrt_ru(lo + hi), kMargin));
        }
    }
}

}  // namespace

cudaError_t launch_write(const WriteParams& p, int scheme, int bits, cudaStream_t stream) {
    const int units = p.n_tok * p.num_kv_heads;
    const int blocks = (units + 7) / 8;
    if (blocks == 0) return cudaSuccess;
    static bool configured = false;   // same carveout as the decode kernels: no L1/shared reconfiguration
    if (!configured) {
        const void* fns[3] = {(const void*)write_kernel<WC_SCHEME_FP8_E4M3, 8>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 8>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 10>};
        for (const void* f : fns) {
            cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout,
                                                 (int)cudaSharedmemCarveoutMaxShared);
            if (e != cudaSuccess) return e;
        }
        configured = true;
    }
    if (scheme == WC_SCHEME_FP8_E4M3)
        return launch_pdl(write_kernel<WC_SCHEME_FP8_E4M3, 8>, dim3(blocks), dim3(128), 0, stream, p);
    if (bits == 8) return launch_pdl(write_kernel<WC_SCHEME_DITHER_INT8, 8>, dim3(blocks), dim3(128), 0, stream, p);
    return launch_pdl(write_kernel<WC_SCHEME_DITHER_INT8, 10>, dim3(blocks), dim3(128), 0, stream, p);
}

}  // namespace wc
