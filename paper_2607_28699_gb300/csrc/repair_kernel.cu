// Block-level repair selection (§6.3.5 "Block-level paging").  The e-form
// certificate is block decomposable: with p~ held fixed, replacing the keys of
// logical page j by their exact values (witness 0, so c_t = 0) lowers D = A - 1
// by exactly C_j = sum_{t in j} p~_t (e^{c_t} - 1).  For each cell the gate sent
// to fallback, pages rank by decreasing C_j (ties to the lower page), and the
// page-in list is the shortest prefix after which the meter of the rest,
// 1/2 R (R + 2) with R the sum of the contributions not yet paged in, is at
// most tau.
//
// One CTA per (sequence, query head).  The decode's per-page terms (m_j, d_j)
// are normalised with the cell's final (M, L) and sorted by a bitonic network
// over 64-bit keys (the contribution's bits above the complemented page index,
// so that a descending sort ranks by contribution, then by lower page; NaN
// above +inf).  The keys stay in registers: the network's exchanges within a
// thread and within a warp need no shared memory, only those across warps go
// through it.  The remaining excess R is then summed from the tail.
#include <climits>

#include "wc_kernels.cuh"

namespace wc {

namespace {

constexpr int kSelThreads = 512;

__device__ __forceinline__ float key_value(unsigned long long key) { return __uint_as_float((uint32_t)(key >> 32)); }

// Bitonic compare-exchange seen from element i, whose partner is i ^ j, in the
// merge of size k: blocks with (i & k) == 0 sort descending (the lower index
// keeps the larger key), the others ascending.  For j >= KPT and k > j every
// position a thread holds has the same bits j and k, so one flag serves all.
__device__ __forceinline__ bool bitonic_takes_max(int i, int j, int k) { return ((i & k) == 0) == ((i & j) == 0); }

__device__ __forceinline__ unsigned long long pick(bool take_max, unsigned long long mine, unsigned long long other) {
    return take_max ? (mine > other ? mine : other) : (mine < other ? mine : other);
}

// KPT keys per thread: thread t holds sorted positions [t KPT, t KPT + KPT).
template <int KPT>
__global__ void __launch_bounds__(kSelThreads) repair_select_kernel(const __grid_constant__ RepairParams p) {
    constexpr int N = kSelThreads * KPT;   // sorted length: the block table, padded to a power of two
    constexpr int W = 32 * KPT;            // positions held by one warp
    extern __shared__ unsigned long long xs[];   // [N] exchange buffer of the cross-warp stages
    __shared__ float warp_tot[kSelThreads / 32];
    __shared__ int warp_min[kSelThreads / 32];
    __shared__ float r_at_k;
    const int hq = blockIdx.x, b = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int base = tid * KPT;
    const size_t cell = (size_t)b * p.num_q_heads + hq;

    // the page terms are read whatever the context length (every block-table
    // column is in bounds), so that no load waits for another
    const float2* terms = p.page_terms + cell * p.max_pages;
    const float2 nm = p.softmax_norm[cell];
    const bool kept = p.keep_q != nullptr && p.keep_q[cell] != 0;
    int ctx = p.ctx_lens[b];
    if (ctx < 0 || ctx > p.max_pages * kPage) {
        if (tid == 0 && hq == 0 && p.status) atomicOr(p.status, WC_DEV_BAD_CTX);
        ctx = max(0, min(ctx, p.max_pages * kPage));
    }
    const int n = (ctx + kPage - 1) / kPage;

    // ---- C_j = d_j 2^(m_j - M) / L in logical page order ---------------------------
    unsigned long long key[KPT];
#pragma unroll
    for (int r = 0; r < KPT; ++r) {
        const int j = base + r;
        const float2 t = j < p.max_pages ? terms[j] : make_float2(-INFINITY, 0.f);
        key[r] = 0ull;   // padding: below every page (C = +0, index bits 0)
        if (j < n) {
            float cj = (nm.y > 0.f && t.y != 0.f) ? __fdiv_rn(t.y * exp2f(t.x - nm.x), nm.y) : 0.f;
            if (cj <= 0.f) cj = 0.f;   // -0 ranks as +0; NaN stays and ranks first
            if (p.contrib) p.contrib[cell * p.max_pages + j] = cj;
            key[r] = ((unsigned long long)__float_as_uint(cj) << 32) | (0xFFFFFFFFu - (uint32_t)j);
        }
    }

    // ---- descending bitonic sort (skipped for kept cells: nothing is paged in) ----
    if (!kept) {
        // exchange layout: position i lives at word i ^ sw(i / KPT), sw(t) a permutation of
        // the thread's KPT words that gives the 16 lanes of a half-warp 16 distinct bank
        // pairs; a partner i ^ j (j >= 32 KPT) flips only bits >= 5 of the thread index,
        // which sw does not read, so loads use the same sw
        const int sw = KPT >= 16 ? (tid & 15) : (((tid * KPT) >> 4) & (KPT - 1));
        for (int k = 2; k <= N; k <<= 1) {
            for (int j = k >> 1; j >= W; j >>= 1) {   // partner in another warp
                const bool tm = bitonic_takes_max(base, j, k);
#pragma unroll
                for (int r = 0; r < KPT; ++r) xs[(base + r) ^ sw] = key[r];
                __syncthreads();
#pragma unroll
                for (int r = 0; r < KPT; ++r) key[r] = pick(tm, key[r], xs[((base + r) ^ j) ^ sw]);
                __syncthreads();
            }
            for (int j = min(k >> 1, W >> 1); j >= KPT; j >>= 1) {   // partner in this warp
                const bool tm = bitonic_takes_max(base, j, k);
                const int lm = j / KPT;
#pragma unroll
                for (int r = 0; r < KPT; ++r) key[r] = pick(tm, key[r], __shfl_xor_sync(0xffffffffu, key[r], lm));
            }
#pragma unroll
            for (int j = KPT >> 1; j > 0; j >>= 1) {   // partner in this thread
                if (j <= (k >> 1)) {
#pragma unroll
                    for (int r = 0; r < KPT; ++r)
                        if ((r & j) == 0) {
                            const bool desc = ((base + r) & k) == 0;
                            const unsigned long long a = key[r], c = key[r | j];
                            if ((a < c) == desc) {
                                key[r] = c;
                                key[r | j] = a;
                            }
                        }
                }
            }
        }
    }

    // ---- remaining sums R_i = sum of the ranked contributions from i on ---------
    // each thread sums its KPT positions from the tail; the later threads'
    // sums enter as an offset
    float tot = 0.f;
#pragma unroll
    for (int r = KPT - 1; r >= 0; --r) tot += key_value(key[r]);
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
    if (!kept) {
        float s = offset;
#pragma unroll
        for (int r = KPT - 1; r >= 0; --r) {
            s += key_value(key[r]);
            if (0.5f * s * (s + 2.0f) <= p.tau) cand = base + r;   // NaN -> false
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
    } else if (kstar >= base && kstar < base + KPT) {
        float s = offset;
#pragma unroll
        for (int r = KPT - 1; r >= 0; --r)
            if (base + r >= kstar) s += key_value(key[r]);
        r_at_k = s;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < KPT; ++r)
        if (base + r < kstar)
            p.repair_pages[cell * p.max_pages + base + r] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key[r] & 0xFFFFFFFFull));
    if (tid == 0) {
        p.n_repair[cell] = kstar;
        p.d_after[cell] = r_at_k;
    }
}

template <int KPT>
cudaError_t launch_kpt(const RepairParams& p, cudaStream_t stream) {
    static bool configured = false;
    constexpr size_t smem = (size_t)kSelThreads * KPT * sizeof(unsigned long long);
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(repair_select_kernel<KPT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(repair_select_kernel<KPT>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    repair_select_kernel<KPT><<<dim3(p.num_q_heads, p.batch), kSelThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_repair_select(const RepairParams& p, cudaStream_t stream) {
    static_assert(kRepairMaxPages == 32 * kSelThreads, "the largest instance holds 32 keys per thread");
    if (p.batch == 0) return cudaSuccess;
    const int need = (p.max_pages + kSelThreads - 1) / kSelThreads;   // keys per thread, rounded up to 2^m
    if (need <= 1) return launch_kpt<1>(p, stream);
    if (need <= 2) return launch_kpt<2>(p, stream);
    if (need <= 4) return launch_kpt<4>(p, stream);
    if (need <= 8) return launch_kpt<8>(p, stream);
    if (need <= 16) return launch_kpt<16>(p, stream);
    return launch_kpt<32>(p, stream);
}

}  // namespace wc
