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

// round-half-even of the exact real x/s + xi, clamped to [-127, 127].
// k0 from an fp32 estimate is within 1 of the answer whenever |x/s| < 2^21;
// the FMA residuals x - s*(k0 +- 1/2 - xi) have exactly the sign of the
// exact value (k0 +- 1/2 - xi is exact in fp32), which settles the rounding.
__device__ __forceinline__ int dither_code(float x, float s, float inv_s, float xi) {
    const float est = fmaf(x, inv_s, xi);
    if (!(fabsf(est) < 200.0f)) return est > 0.0f ? 127 : -127;
    float k = rintf(est);
    const float up = fmaf(-s, k + 0.5f - xi, x);   // sign of x/s + xi - (k + 1/2)
    const float dn = fmaf(-s, k - 0.5f - xi, x);   // sign of x/s + xi - (k - 1/2)
    const bool k_odd = (((int)k) & 1) != 0;
    if (up > 0.0f || (up == 0.0f && k_odd)) k += 1.0f;
    else if (dn < 0.0f || (dn == 0.0f && k_odd)) k -= 1.0f;
    return max(-127, min(127, (int)k));
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

        // dither integers j for channels 16*sub .. 16*sub + 15
        uint32_t jw[8];  // 16-bit lanes: j of channel (2i, 2i+1) in (lo, hi)
        const uint32_t slot_u = (uint32_t)max(slot, 0);
        const uint32_t c1 = (uint32_t)p.layer * 65536u + (uint32_t)h;
        if constexpr (kBits == 8) {
            const uint4 w = philox(slot_u, c1, (uint32_t)sub, (uint32_t)row, p.keys);
            const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                jw[2 * i] = prmt(ww[i], 0u, 0x4140u);      // bytes 0,1 -> 16-bit lanes
                jw[2 * i + 1] = prmt(ww[i], 0u, 0x4342u);  // bytes 2,3
            }
        } else {
#pragma unroll
            for (int g = 0; g < 2; ++g) {
                const uint4 w = philox(slot_u, c1, (uint32_t)(2 * sub + g), (uint32_t)row, p.keys);
                jw[4 * g + 0] = w.x & 0x03FF03FFu;
                jw[4 * g + 1] = w.y & 0x03FF03FFu;
                jw[4 * g + 2] = w.z & 0x03FF03FFu;
                jw[4 * g + 3] = w.w & 0x03FF03FFu;
            }
        }
        constexpr float kInvN = 1.0f / (float)(1 << kBits);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const uint32_t j = (jw[i >> 1] >> (16 * (i & 1))) & 0xFFFFu;
            const float xi = ((float)j + 0.5f) * kInvN - 0.5f;   // exact
            int k = 0;
            if (s > 0.0f) k = dither_code(x[i], s, inv_s, xi);
            r[i] = fmaf(s, (float)k - xi, -x[i]);                // x^ - x, one rounding
            const uint32_t b = (uint32_t)(k & 0xFF);
            if ((i & 3) == 0) codes[i >> 2] = b;
            else codes[i >> 2] |= b << (8 * (i & 3));
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
