// Constants and helpers shared by the decode kernels (fragment layouts of
// mma.sync m16n8k16 / m16n8k8 and the exact int8 / dither -> fp16 operands).
#pragma once

#include <cuda.h>

#include <climits>

#include "wc_kernels.cuh"

namespace wc {

namespace {

// Extra outputs compiled into a decode kernel (template bit mask).
constexpr int kXTierB = 1;   // Tier-B meter (§4.2)
constexpr int kXValue = 2;   // value-side witness terms and output bound (§3, §4.2)
constexpr int kXRepair = 4;  // per-page meter terms for block-level repair selection (§6.3.5)
constexpr int kXAppend = 8;  // the decode writes the step's new token before reading it
constexpr int kXFlat = 16;   // warp-specialized kernel under the flattened split plan
// failure-detection test (warp-specialized kernel, split plan): one page's
// copies are never issued and every wait gives up after kStallTries tries
constexpr int kXStall = 32;
constexpr int kStallTries = 64;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRsd = 0.08838834764831845f;                      // 1/sqrt(128)
constexpr float kRsdLog2e = 0.08838834764831845f * 1.4426950408889634f;

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

// h' pair (fp16) for two 8-bit dithers: bytes of x at the selector.
__device__ __forceinline__ uint32_t h8(uint32_t x, uint32_t sel) { return prmt(x, 0x44444444u, sel); }
// -h' pair (fp16) for two 8-bit dithers: the same bytes under a negative high byte.
__device__ __forceinline__ uint32_t nh8(uint32_t x, uint32_t sel) { return prmt(x, 0xC4C4C4C4u, sel); }
// h' pair (fp16) for two 10-bit dithers in the low bits of each 16-bit lane.
__device__ __forceinline__ uint32_t h10(uint32_t x) { return (x & 0x03FF03FFu) | 0x3C003C00u; }

// Upward margin on the merged e-form accumulator D = E_p~[e^c - 1] (and the
// Tier-B one) before the meter (A^2 - 1)/2 = D (D + 2)/2 is formed, so the
// fp32 meter lands on or above the exact value of §3 Thm. "Sound replacement"
// instead of within rounding either side of it.  It covers:
//  - ex2.approx near 1 (relative error below 2^-22 of 2^c, i.e. an absolute
//    error below 2^-22 in each e^c - 1 and so in their p~-weighted mean): kDAbs;
//  - the fp32 sums of p~ and p~ (e^c - 1) (per lane about a thousand terms
//    at 32k tokens, then the warp, CTA and split merges: n u < 2^-13), the
//    hi + lo fp16 bound operand (2^-22) and the rounding of the logits that
//    move p~ (their effect on D, measured against the fp64 oracle, stays near
//    10^-5 relative): kDRel, at about 4x the larger of these.
// At 1 + 2^-12 it stays well inside the 1e-3 relative parity tolerance.
constexpr float kDRel = 1.0f + 0x1p-12f;
constexpr float kDAbs = 0x1p-21f;
__device__ __forceinline__ float d_upper(float d) { return fmaf(d, kDRel, kDAbs); }

// One token's meter term p~ (e^c - 1) in the log2 frame of the running maximum:
// t = y - m (p~ = 2^t, flushed to 0 below 2^-126) and cl = c log2(e).  The
// kernels use the product 2^t (2^cl - 1) as long as every cl of the page is below
// kHugeLog2: an underflowed 2^t then drops less than 2^(64 - 126) per token,
// far inside kDAbs.  A page with a larger bound (a key row of huge magnitude;
// never with ordinary inputs) takes its terms from meter_term, which uses
// 2^(t + cl) from kHugeLog2 on, its exponent raised by a bound on the two fp32
// roundings of t + cl + margin: at least the term, and finite wherever the term
// is, so a token whose weight underflows but whose bound does not still counts
// (the product gives 0, or 0 * inf = NaN).
constexpr float kHugeLog2 = 64.0f;
__device__ __forceinline__ float meter_term(float t, float cl) {
    if (cl < kHugeLog2) return fast_exp2(t) * (fast_exp2(cl) - 1.f);
    if (t == -INFINITY) return 0.f;   // a token past the context
    return fast_exp2(t + cl + (fabsf(t) + cl) * 0x1p-22f);
}

// NaN only arises in the meter from 0 * inf or inf - inf, i.e. from a term or a
// sum that overflowed: report it as +inf, the bound's overflow value.
__device__ __forceinline__ float raw_or_inf(float raw) { return raw == raw ? raw : INFINITY; }

// 2^n for -126 <= n <= 127.
__device__ __forceinline__ float pow2(int n) { return __int_as_float((127 + n) << 23); }

__device__ __forceinline__ uint32_t word_of(const uint4& v, int i) {
    return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
}

// Transpose of an 8x8 b16 matrix held in the mma fragment layout.
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

// Token held by row r of a 16-row QK / softmax tile in the warp-specialized
// decode: rows 2i, 2i+1 hold tokens 4i, 4i+1 and rows 8+2i, 9+2i tokens
// 4i+2, 4i+3, so the P fragment transposed by movmatrix gives lane (g, c) the
// tokens 4c .. 4c+3 that ldmatrix.trans delivers for V.
__device__ __forceinline__ int tok_row(int r) { return 4 * ((r & 7) >> 1) + 2 * (r >> 3) + (r & 1); }

// ldmatrix.trans of two 16x16 byte blocks: lanes 0-15 address the 16 rows of
// the first, lanes 16-31 those of the second; lane (g, c) receives, per block,
// column g (first word) and column g + 8 (second word) at rows 4c .. 4c+3.
__device__ __forceinline__ void ldsm_t_b8_x2(uint32_t (&d)[4], const void* row) {
    asm volatile("ldmatrix.sync.aligned.m16n16.x2.trans.shared.b8 {%0, %1, %2, %3}, [%4];"
                 : "=r"(d[0]), "=r"(d[1]), "=r"(d[2]), "=r"(d[3])
                 : "r"(smem_addr(row)));
}

// Byte offset of 16-byte chunk q of token row t in a tile written with the
// 128-byte swizzle (tile 1024-byte aligned): chunk q of row t sits at chunk
// q ^ (t & 7), so the 8 rows a warp touches per instruction hit distinct banks.
__device__ __forceinline__ int swz(int t, int q) { return t * kHeadDim + 16 * (q ^ (t & 7)); }

__device__ __forceinline__ void tma_page(void* dst, const CUtensorMap* map, int z, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(z), "r"(smem_addr(bar))
        : "memory");
}


// A CTA's work as segments: pages [a, e) of unit (b, h); page stream (warp
// pair) w of the CTA's n takes pages a + ((w - ph) mod n) + n i.  Split plan: one segment, the
// CTA's split (possibly empty).  Flattened plan: CTA c serves KV head
// h = c mod Hkv and takes share j = c / Hkv of the batch's pages laid end to
// end (sequence after sequence), cut at sequence boundaries; the Hkv CTAs of a
// share read the same pages together (the heads of a page are adjacent in the
// cache).  ph keeps the streams' round robin running across the cuts, so
// every stream gets ceil or floor of (hi - lo) / n pages.
struct WsSeg {
    int b, h, a, e, ph, ctx, np;
    long long pos;      // flattened position of page a
    long long lo, hi;   // the CTA's share
};

__device__ __forceinline__ int clamped_ctx(const DecodeParams& p, int b) {
    return max(0, min(__ldg(p.ctx_lens + b), p.max_pages * kPage));
}

// First segment; called by every thread of the CTA (the flattened plan scans
// the batch's page counts with two block barriers).  False: no pages.
template <bool kFlat>
__device__ __forceinline__ bool ws_first_segment(const DecodeParams& p, WsSeg& sg, int* s_wtot, long long* s_start) {
    if constexpr (!kFlat) {
        sg.b = blockIdx.z;
        sg.h = blockIdx.y;
        int ctx = __ldg(p.ctx_lens + sg.b);
        if (ctx < 0 || ctx > p.max_pages * kPage) {
            if (threadIdx.x == 0 && blockIdx.x == 0 && sg.h == 0) atomicOr(p.status, WC_DEV_BAD_CTX);
            ctx = max(0, min(ctx, p.max_pages * kPage));
        }
        sg.ctx = ctx;
        sg.np = (ctx + kPage - 1) / kPage;
        sg.a = blockIdx.x * p.pages_per_split;
        sg.e = min(sg.a + p.pages_per_split, sg.np);
        sg.ph = 0;
        sg.pos = sg.lo = sg.hi = 0;
        return true;
    } else {
        const int nt = blockDim.x, t = threadIdx.x, per = (p.batch + nt - 1) / nt;
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
            if ((t & 31) >= o) inc += v;
        }
        if ((t & 31) == 31) s_wtot[t >> 5] = inc;
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < nt / 32; ++w) {
            const int v = s_wtot[w];
            total += v;
            if (w < (t >> 5)) before += v;
        }
        const int excl = before + inc - loc;   // pages of the sequences before this thread's
        const int hk = p.num_kv_heads, shares = max(1, p.splits / hk);
        const long long R = max(1LL, ((long long)total + shares - 1) / shares);
        const long long lo = (long long)(blockIdx.x / hk) * R, hi = min((long long)total, lo + R);
        if (lo < hi && excl <= lo && lo < (long long)excl + loc) {
            long long acc = excl;   // exactly one thread: the one whose sequences hold lo
            for (int i = 0; i < per; ++i) {
                const int bb = t * per + i;
                if (bb >= p.batch) break;
                const int np = (clamped_ctx(p, bb) + kPage - 1) / kPage;
                if (lo < acc + np) {
                    *s_start = ((long long)bb << 32) | (long long)(lo - acc);
                    break;
                }
                acc += np;
            }
        }
        __syncthreads();
        if (lo >= hi) return false;
        const long long st = *s_start;
        sg.b = (int)(st >> 32);
        sg.a = (int)(st & 0xffffffffLL);
        sg.h = blockIdx.x % hk;
        sg.ctx = clamped_ctx(p, sg.b);
        sg.np = (sg.ctx + kPage - 1) / kPage;
        sg.e = (int)min((long long)sg.np, sg.a + (hi - lo));
        sg.ph = 0;
        sg.pos = sg.lo = lo;
        sg.hi = hi;
        return true;
    }
}

// Next segment of the flattened plan (the next sequence with pages); false
// at the end of the CTA's share, and always in the split plan.
template <int kStreams, bool kFlat>
__device__ __forceinline__ bool ws_next_segment(const DecodeParams& p, WsSeg& sg) {
    if constexpr (!kFlat) return false;
    sg.pos += sg.e - sg.a;
    if (sg.pos >= sg.hi) return false;
    do {   // sequences without pages hold no part of the share
        if (sg.b + 1 >= p.batch) return false;
        ++sg.b;
        sg.ctx = clamped_ctx(p, sg.b);
        sg.np = (sg.ctx + kPage - 1) / kPage;
    } while (sg.np == 0);
    sg.a = 0;
    sg.e = (int)min((long long)sg.np, sg.hi - sg.pos);
    sg.ph = (int)((sg.pos - sg.lo) % kStreams);
    return true;
}


// Flattened plan: each warp's walker lives in a shared slot, so that only the
// current segment's indices take registers in the page loop; lane 0 advances it.
template <int kStreams, bool kFlat>
__device__ __forceinline__ bool ws_step(const DecodeParams& p, WsSeg* slot, int lane) {
    if constexpr (!kFlat) {
        return false;
    } else {
        __syncwarp();
        int more = 0;
        if (lane == 0) more = ws_next_segment<kStreams, true>(p, *slot);
        __syncwarp();
        return __shfl_sync(0xffffffffu, more, 0) != 0;
    }
}
template <int kStreams>
__device__ __forceinline__ int ws_seg_pages(const WsSeg& sg, int w, int& first) {
    first = sg.a + (int)((unsigned)(w - sg.ph + kStreams) % kStreams);
    return first < sg.e ? (sg.e - first + kStreams - 1) / kStreams : 0;
}

}  // namespace

// One layer's code array [num_pages][Hkv][16][128] bytes as a 3-D tensor map
// (channel, slot, page * Hkv + head) whose box is one page of one head,
// written to shared memory with the 128-byte swizzle (swz above).
bool encode_page_map(CUtensorMap* map, const void* codes, int num_pages, int num_kv_heads);

// The split-K merge for the extra outputs in the bit mask x (0, kXTierB,
// kXValue or kXRepair), launched as a programmatic dependent of the decode.
cudaError_t launch_merge_x(const DecodeParams& p, int x, cudaStream_t stream);

}  // namespace wc
