// Block-level repair selection (§6.4 "Block-level paging").  The e-form
// certificate is block decomposable: with p~ held fixed, replacing the keys of
// logical page j by their exact values (witness 0, so c_t = 0) lowers D = A - 1
// by exactly C_j = sum_{t in j} p~_t (e^{c_t} - 1).  For each cell the gate sent
// to fallback, pages rank by decreasing C_j (ties to the lower page), and the
// page-in list is the shortest prefix after which the meter of the rest,
// 1/2 R (R + 2) with R the sum of the contributions not yet paged in, is at
// most tau.
//
// One CTA per (sequence, query head).  The decode's per-page terms (m_j, d_j)
// are normalised with the cell's final (M, L), sorted in shared memory (bitonic,
// 64-bit keys: the contribution's bits above the complemented page index, so
// that a descending sort ranks by contribution, then by lower page; NaN above
// +inf), and summed from the tail for the remaining excess R.
#include <climits>

#include "wc_kernels.cuh"

namespace wc {

namespace {

constexpr int kSelThreads = 512;

__device__ __forceinline__ float key_value(unsigned long long key) { return __uint_as_float((uint32_t)(key >> 32)); }

__global__ void __launch_bounds__(kSelThreads) repair_select_kernel(const __grid_constant__ RepairParams p) {
    extern __shared__ unsigned long long keys[];   // [n2]
    __shared__ float warp_tot[kSelThreads / 32];
    __shared__ int warp_min[kSelThreads / 32];
    __shared__ float r_at_k;
    const int hq = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const size_t cell = (size_t)b * p.num_q_heads + hq;
    int ctx = p.ctx_lens[b];
    if (ctx < 0 || ctx > p.max_pages * kPage) {
        if (tid == 0 && hq == 0 && p.status) atomicOr(p.status, WC_DEV_BAD_CTX);
        ctx = max(0, min(ctx, p.max_pages * kPage));
    }
    const int n = (ctx + kPage - 1) / kPage;
    int n2 = 1;
    while (n2 < n) n2 <<= 1;

    // ---- C_j = d_j 2^(m_j - M) / L in logical page order ---------------------------
    const float2 nm = p.softmax_norm[cell];
    const float2* terms = p.page_terms + cell * p.max_pages;
    for (int j = tid; j < n2; j += kSelThreads) {
        unsigned long long key = 0ull;   // padding: below every page (C = +0, index bits 0)
        if (j < n) {
            const float2 t = terms[j];
            float cj = (nm.y > 0.f && t.y != 0.f) ? __fdiv_rn(t.y * exp2f(t.x - nm.x), nm.y) : 0.f;
            if (cj <= 0.f) cj = 0.f;   // -0 ranks as +0; NaN stays and ranks first
            if (p.contrib) p.contrib[cell * p.max_pages + j] = cj;
            key = ((unsigned long long)__float_as_uint(cj) << 32) | (0xFFFFFFFFu - (uint32_t)j);
        }
        keys[j] = key;
    }
    const bool kept = p.keep_q != nullptr && p.keep_q[cell] != 0;

    // ---- descending bitonic sort (skipped for kept cells: nothing is paged in) ----
    if (!kept) {
        for (int k = 2; k <= n2; k <<= 1)
            for (int j = k >> 1; j > 0; j >>= 1) {
                __syncthreads();
                for (int i = tid; i < n2 / 2; i += kSelThreads) {
                    const int lo = ((i & ~(j - 1)) << 1) | (i & (j - 1)), hi = lo + j;
                    const bool desc = (lo & k) == 0;
                    const unsigned long long a = keys[lo], c = keys[hi];
                    if ((a < c) == desc) {
                        keys[lo] = c;
                        keys[hi] = a;
                    }
                }
            }
    }
    __syncthreads();

    // ---- remaining sums R_i = sum of the ranked contributions from i on ---------
    // thread t owns positions [t E, t E + E) and sums them from the tail; the
    // sums of the later threads enter as an offset
    const int E = n2 > kSelThreads ? n2 / kSelThreads : 1;
    const int i0 = tid * E;
    const bool active = i0 < n2;
    float tot = 0.f;
    if (active)
        for (int i = i0 + E - 1; i >= i0; --i) tot += key_value(keys[i]);
    float suf = tot;   // inclusive suffix over the warp's lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float v = __shfl_down_sync(0xffffffffu, suf, o);
        if (lane + o < 32) suf += v;
    }
    if (lane == 0) warp_tot[warp] = suf;
    float offset = __shfl_down_sync(0xffffffffu, suf, 1);   // later lanes of this warp
    if (lane == 31) offset = 0.f;
    __syncthreads();
    for (int w = kSelThreads / 32 - 1; w > warp; --w) offset += warp_tot[w];

    int cand = INT_MAX;
    if (!kept && active) {
        float s = offset;
        for (int i = i0 + E - 1; i >= i0; --i) {
            s += key_value(keys[i]);
            if (0.5f * s * (s + 2.0f) <= p.tau) cand = i;   // NaN -> false
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cand = min(cand, __shfl_xor_sync(0xffffffffu, cand, o));
    if (lane == 0) warp_min[warp] = cand;
    __syncthreads();
    int kmin = INT_MAX;
    for (int w = 0; w < kSelThreads / 32; ++w) kmin = min(kmin, warp_min[w]);
    const int kstar = kept ? 0 : min(kmin, n);   // every page when no prefix is enough
    if (kstar >= n) {
        if (tid == 0) r_at_k = 0.f;
    } else if (active && kstar >= i0 && kstar < i0 + E) {
        float s = offset;
        for (int i = i0 + E - 1; i >= kstar; --i) s += key_value(keys[i]);
        r_at_k = s;
    }
    __syncthreads();
    for (int i = tid; i < kstar; i += kSelThreads)
        p.repair_pages[cell * p.max_pages + i] = (int32_t)(0xFFFFFFFFu - (uint32_t)(keys[i] & 0xFFFFFFFFull));
    if (tid == 0) {
        p.n_repair[cell] = kstar;
        p.d_after[cell] = r_at_k;
    }
}

}  // namespace

cudaError_t launch_repair_select(const RepairParams& p, cudaStream_t stream) {
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(repair_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)(kRepairMaxPages * sizeof(unsigned long long)));
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(repair_select_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    if (p.batch == 0) return cudaSuccess;
    int n2 = 1;
    while (n2 < p.max_pages) n2 <<= 1;
    const size_t smem = (size_t)n2 * sizeof(unsigned long long);
    repair_select_kernel<<<dim3(p.num_q_heads, p.batch), kSelThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace wc
