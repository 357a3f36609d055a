// Write path: quantize post-RoPE K/V rows into the paged cache and store the
// K band-norm residual witness (§6.2.1 write kernel; §4.1 Eq. witness;
// §4.2 subtractive dither).
//
// A CTA of 4 warps handles eight (token, KV head) units: warps 0 and 2 the K
// rows, warps 1 and 3 the V rows, 8 lanes per row.  Each lane owns 16
// consecutive channels, so it loads 32 B of fp16, stores 16 B of codes, and
// (for the dither schemes) consumes exactly one Philox4x32-10 call per 16
// channels.
//
// Grouped scheme (§6.2.3 "Storage side" and §6.2.5 "Fixed-channel outlier bypass"):
// one fp16 scale per 32-channel group (a lane pair), the group amax leaving
// out the bypassed channels of the KV head's fixed RoPE pairs, which are
// stored exactly (fp16, code 0).  A row is stored in a permuted channel order
// with the dither drawn by storage position; storage position p holds channel
//   K:  16 ((p >> 2) & 7) + 4 (p >> 5) + (p & 3)
//   V:  16 ((p >> 1) & 7) + 8 (p & 1) + (p >> 4)
// (the decode's fragment order: each QK k-step and each PV m-tile then meets
// one group).  The lane's Philox call covers storage positions 16 sub .. +15;
// dither bytes and codes move between storage and channel order through a
// 128-byte shared row per unit, so quantization runs in channel order.
#include <cooperative_groups.h>

#include "write_row.cuh"

namespace cg = cooperative_groups;

namespace wc {

namespace {

// Tasks of 4 tokens per warp whose loads are all issued before any is used:
// more bytes in flight per SM (the kernel is otherwise bound by load latency).
constexpr int kWriteTasks = 2;
// The grouped scheme's row routine is much larger: one task per warp keeps the
// kernel's code small enough for the instruction cache.
__host__ __device__ constexpr int write_tasks(int scheme) {
    return scheme == WC_SCHEME_DITHER_INT8_G32 ? 1 : kWriteTasks;
}
__host__ __device__ constexpr int write_units_per_cta(int scheme) { return 2 * 4 * write_tasks(scheme); }
constexpr int kPerHeadMinTokens = 16;                     // per-head grid from this many tokens on

// Two ways of cutting the units (token, KV head) into 4-unit tasks:
//  kPerHead: grid (token groups, Hkv), a task = 4 consecutive tokens of one
//            head, so a warp's code, scale and witness stores are contiguous
//            runs of consecutive slots (prefill);
//  else:     one index over units u = token * Hkv + h, a task = 4 consecutive
//            units, so a one-token write of up to 8 KV heads is a single CTA
//            (decode steps, where every SM the next decode needs counts).
// Resident CTAs per SM the register budget is sized for: seven (72 registers)
// for the dithered schemes, ten for fp8.  The 8-bit dither's packed fast pass
// then spills 4 bytes; the extra warps per SM still take 4-5% off a prefill
// write against six CTAs at 80 registers, and eight (64 registers, 48 bytes of
// spill) are slower again.
__host__ __device__ constexpr int write_min_blocks(int scheme) {
    return scheme == WC_SCHEME_FP8_E4M3 ? 10 : 7;
}
template <int kScheme, int kBits, bool kPerHead>
__global__ void __launch_bounds__(128, write_min_blocks(kScheme)) write_kernel(const __grid_constant__ WriteParams p) {
    constexpr bool kGrouped = kScheme == WC_SCHEME_DITHER_INT8_G32;
    __shared__ __align__(16) uint8_t xrows[kGrouped ? 4 * 4 * kXRowStride : 16];   // [warp][unit][row]
    __shared__ BypassTable btab;
    grid_dep_launch();    // a dependent decode may be scheduled now: it waits for this whole grid
    grid_dep_wait();      // inputs may come from the preceding kernel
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const BypassTable* tab = nullptr;
    if constexpr (kGrouped && kPerHead) {   // one KV head per CTA: its bypass set, once
        if (threadIdx.x < kHeadDim) btab.entry[threadIdx.x] = -1;
        if (threadIdx.x < 4) btab.mask[threadIdx.x] = 0u;
        if (threadIdx.x == 0) btab.bad = 0u;
        __syncthreads();
        if (threadIdx.x < p.num_bypass) {
            const int t = threadIdx.x;
            const int32_t* pr = p.bypass_pairs + (size_t)blockIdx.y * p.num_bypass;
            const int j = __ldg(pr + t);
            bool dup = false;   // a pair listed again is ignored after its first occurrence
            for (int u = 0; u < t; ++u) dup = dup || __ldg(pr + u) == j;
            if (j < 0 || j >= kHeadDim / 2 || dup) {
                atomicOr(&btab.bad, 1u << t);
                if (p.dev_status) atomicOr(p.dev_status, WC_DEV_BAD_PAIR);
            } else {
                const int a = p.rope_layout == WC_ROPE_HALF ? j : 2 * j;
                const int b = p.rope_layout == WC_ROPE_HALF ? j + kHeadDim / 2 : 2 * j + 1;
                btab.entry[a] = (int8_t)(2 * t);
                btab.entry[b] = (int8_t)(2 * t + 1);
                atomicOr(&btab.mask[a >> 5], 1u << (a & 31));
                atomicOr(&btab.mask[b >> 5], 1u << (b & 31));
            }
        }
        __syncthreads();
        tab = &btab;
    }
    // Warps 0, 2 take the K rows and warps 1, 3 the V rows of the same units,
    // so the residual and witness work stays in whole warps; lanes 8i .. 8i+7
    // own unit i of a 4-unit task.
    const int row = warp & 1;                                                  // 0 = K, 1 = V
    const int sub = lane & 7;                                                  // 16-channel chunk
    constexpr int kTasks = write_tasks(kScheme);
    const int first = (blockIdx.x * 2 + (warp >> 1)) * (4 * kTasks) + (lane >> 3);
    const int n_first = kPerHead ? p.n_tok : p.n_tok * p.num_kv_heads;
    bool live[kTasks];
    int slot[kTasks], hs[kTasks];
    uint4 raw[kTasks][2];
#pragma unroll
    for (int t = 0; t < kTasks; ++t) {
        const int idx = first + 4 * t;   // a token (kPerHead) or a unit
        live[t] = idx < n_first;
        int tok = 0, h = 0;
        if (live[t]) {
            if (kPerHead) {
                tok = idx;
                h = blockIdx.y;
            } else {
                tok = idx / p.num_kv_heads;
                h = idx - tok * p.num_kv_heads;
            }
        }
        hs[t] = h;
        slot[t] = live[t] ? __ldg(p.slot_mapping + tok) : -1;
        raw[t][0] = raw[t][1] = make_uint4(0, 0, 0, 0);
        if (live[t]) {
            const uint4* src = reinterpret_cast<const uint4*>(
                (row == 0 ? p.k : p.v) + ((size_t)tok * p.num_kv_heads + h) * kHeadDim + sub * 16);
            raw[t][0] = __ldg(src);
            raw[t][1] = __ldg(src + 1);
        }
    }
    // 8-bit dither: the tasks' Philox calls (one per lane each) advanced together
    uint4 w[kTasks];
    constexpr bool kPre = kScheme != WC_SCHEME_FP8_E4M3 && kBits == 8;
    if constexpr (kPre) {
        uint32_t x0[kTasks], x1[kTasks], x2[kTasks], x3[kTasks];
#pragma unroll
        for (int t = 0; t < kTasks; ++t) {
            x0[t] = (uint32_t)max(slot[t], 0);
            x1[t] = (uint32_t)p.layer * 65536u + (uint32_t)hs[t];
            x2[t] = (uint32_t)sub;
            x3[t] = (uint32_t)row;
        }
        philox_n<kTasks>(x0, x1, x2, x3, p.keys);
#pragma unroll
        for (int t = 0; t < kTasks; ++t) w[t] = make_uint4(x0[t], x1[t], x2[t], x3[t]);
    }
#pragma unroll
    for (int t = 0; t < kTasks; ++t)
        if (__any_sync(0xffffffffu, live[t]))   // warp-uniform: a task past the end is skipped whole
            write_row<kScheme, kBits>(p, raw[t], slot[t], live[t], hs[t], row, sub,
                                      kGrouped ? xrows + (warp * 4 + (lane >> 3)) * kXRowStride : xrows, tab,
                                      kPre ? &w[t] : nullptr);
}

// Bypass-pair calibration: a cluster of 8 CTAs of 32 warps per KV head.  Warp
// w of cluster rank r sums rows 32 r + w + 256 i: one 256-byte row per warp load,
// lane l squaring channels 4l .. 4l + 3.  Each CTA adds its warps' sums in a
// fixed order; rank 0 adds the 8 CTAs' sums (distributed shared memory, rank
// order), adds channels into pairs, and selects a pair iff fewer than m pairs
// rank above it (larger energy, or equal energy and a lower index).
constexpr int kSelPairThreads = 1024;
constexpr int kSelPairCluster = 8;

__global__ void __cluster_dims__(kSelPairCluster, 1, 1) __launch_bounds__(kSelPairThreads)
    select_pairs_kernel(const __half* __restrict__ k, int n_tok, int num_kv_heads, int rope_layout, int m,
                        int32_t* __restrict__ pairs) {
    __shared__ float part[kSelPairThreads / 32][kHeadDim];
    __shared__ float energy[kHeadDim / 2];
    __shared__ int chosen[kHeadDim / 2];
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int h = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int kWarpsPerHead = kSelPairCluster * kSelPairThreads / 32;
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll 4
    for (int t = rank * (kSelPairThreads / 32) + warp; t < n_tok; t += kWarpsPerHead) {
        const uint2 w = __ldg(reinterpret_cast<const uint2*>(k + ((size_t)t * num_kv_heads + h) * kHeadDim) + lane);
        const float2 f01 = __half22float2(*reinterpret_cast<const __half2*>(&w.x));
        const float2 f23 = __half22float2(*reinterpret_cast<const __half2*>(&w.y));
        a0 = fmaf(f01.x, f01.x, a0);
        a1 = fmaf(f01.y, f01.y, a1);
        a2 = fmaf(f23.x, f23.x, a2);
        a3 = fmaf(f23.y, f23.y, a3);
    }
    part[warp][4 * lane] = a0;
    part[warp][4 * lane + 1] = a1;
    part[warp][4 * lane + 2] = a2;
    part[warp][4 * lane + 3] = a3;
    __syncthreads();
    if (tid < kHeadDim) {   // this CTA's channel sums in a fixed order (each thread its own column)
        float e = 0.f;
        for (int w = 0; w < kSelPairThreads / 32; ++w) e += part[w][tid];
        part[0][tid] = e;
    }
    cluster.sync();   // every CTA's sums are in its row 0
    if (rank == 0) {
        if (tid < kHeadDim) {
            float e = 0.f;
            for (int r = 0; r < kSelPairCluster; ++r) e += cluster.map_shared_rank(&part[0][0], r)[tid];
            part[1][tid] = e;
        }
        __syncthreads();
        const int j = tid;
        if (j < kHeadDim / 2) {
            const int a = rope_layout == WC_ROPE_HALF ? j : 2 * j;
            const int b = rope_layout == WC_ROPE_HALF ? j + kHeadDim / 2 : 2 * j + 1;
            energy[j] = part[1][a] + part[1][b];
        }
        __syncthreads();
        if (j < kHeadDim / 2) {
            const float e = energy[j];
            int rnk = 0;
            for (int i = 0; i < kHeadDim / 2; ++i) rnk += (energy[i] > e || (energy[i] == e && i < j)) ? 1 : 0;
            chosen[j] = rnk < m;
        }
        __syncthreads();
        if (j < kHeadDim / 2 && chosen[j]) {
            int pos = 0;
            for (int i = 0; i < j; ++i) pos += chosen[i];
            if (pos < m) pairs[(size_t)h * m + pos] = j;   // NaN energies can make more than m ranks fall below m
        }
    }
    cluster.sync();   // the other CTAs' shared memory stays alive until rank 0 has read it
}

}  // namespace

cudaError_t launch_select_pairs(const __half* k, int n_tok, int num_kv_heads, int rope_layout, int m, int32_t* pairs,
                                cudaStream_t stream) {
    select_pairs_kernel<<<dim3(kSelPairCluster, num_kv_heads), kSelPairThreads, 0, stream>>>(k, n_tok, num_kv_heads,
                                                                                            rope_layout, m, pairs);
    return cudaGetLastError();
}

cudaError_t launch_write(const WriteParams& p, int scheme, int bits, cudaStream_t stream) {
    if (p.n_tok == 0) return cudaSuccess;
    static bool configured = false;   // same carveout as the decode kernels: no L1/shared reconfiguration
    if (!configured) {
        const void* fns[8] = {(const void*)write_kernel<WC_SCHEME_FP8_E4M3, 8, false>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 8, false>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 10, false>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8_G32, 8, false>,
                              (const void*)write_kernel<WC_SCHEME_FP8_E4M3, 8, true>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 8, true>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8, 10, true>,
                              (const void*)write_kernel<WC_SCHEME_DITHER_INT8_G32, 8, true>};
        for (const void* f : fns) {
            cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout,
                                                 (int)cudaSharedmemCarveoutMaxShared);
            if (e != cudaSuccess) return e;
        }
        configured = true;
    }
    const bool per_head = p.n_tok >= kPerHeadMinTokens;
    const int upc = write_units_per_cta(scheme);
    const dim3 grid = per_head ? dim3((p.n_tok + upc - 1) / upc, p.num_kv_heads)
                               : dim3((p.n_tok * p.num_kv_heads + upc - 1) / upc);
    auto go = [&](auto kernel) { return launch_pdl(kernel, grid, dim3(128), 0, stream, p); };
    if (scheme == WC_SCHEME_FP8_E4M3)
        return per_head ? go(write_kernel<WC_SCHEME_FP8_E4M3, 8, true>) : go(write_kernel<WC_SCHEME_FP8_E4M3, 8, false>);
    if (scheme == WC_SCHEME_DITHER_INT8_G32)
        return per_head ? go(write_kernel<WC_SCHEME_DITHER_INT8_G32, 8, true>)
                        : go(write_kernel<WC_SCHEME_DITHER_INT8_G32, 8, false>);
    if (bits == 8)
        return per_head ? go(write_kernel<WC_SCHEME_DITHER_INT8, 8, true>)
                        : go(write_kernel<WC_SCHEME_DITHER_INT8, 8, false>);
    return per_head ? go(write_kernel<WC_SCHEME_DITHER_INT8, 10, true>)
                    : go(write_kernel<WC_SCHEME_DITHER_INT8, 10, false>);
}

}  // namespace wc
