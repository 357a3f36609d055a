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
constexpr int kXRepair = 4;  // per-page meter terms for block-level repair selection (§6.4)
constexpr int kXAppend = 8;  // the decode writes the step's new token before reading it
constexpr int kXFlat = 16;   // warp-specialized kernel under the flattened split plan
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
// h' pair (fp16) for two 10-bit dithers in the low bits of each 16-bit lane.
__device__ __forceinline__ uint32_t h10(uint32_t x) { return (x & 0x03FF03FFu) | 0x3C003C00u; }

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

}  // namespace

// One layer's code array [num_pages][Hkv][16][128] bytes as a 3-D tensor map
// (channel, slot, page * Hkv + head) whose box is one page of one head,
// written to shared memory with the 128-byte swizzle (swz above).
bool encode_page_map(CUtensorMap* map, const void* codes, int num_pages, int num_kv_heads);

// The split-K merge for the extra outputs in the bit mask x (0, kXTierB,
// kXValue or kXRepair), launched as a programmatic dependent of the decode.
cudaError_t launch_merge_x(const DecodeParams& p, int x, cudaStream_t stream);

}  // namespace wc
