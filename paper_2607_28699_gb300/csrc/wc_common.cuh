// Device helpers shared by the WitCert kernels (sm_103a).
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/witcert.h"

namespace wc {

constexpr int kHeadDim = 128;
constexpr int kPage = 16;
constexpr int kBands = 8;
constexpr int kMaxGroup = 8;

// Philox4x32-10 (Salmon et al., SC'11): round constants of the published
// algorithm.
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;
constexpr int kPhiloxRounds = 10;

// Round keys (key bumped by the Weyl constants before rounds 1..9),
// computed once on the host so each round XORs a kernel-parameter word.
struct PhiloxKeys {
    uint32_t k0[kPhiloxRounds];
    uint32_t k1[kPhiloxRounds];
};

inline PhiloxKeys make_philox_keys(uint64_t seed) {
    PhiloxKeys k;
    uint32_t a = (uint32_t)(seed & 0xFFFFFFFFull), b = (uint32_t)(seed >> 32);
    for (int r = 0; r < kPhiloxRounds; ++r) {
        k.k0[r] = a;
        k.k1[r] = b;
        a += kPhiloxW0;
        b += kPhiloxW1;
    }
    return k;
}

__device__ __forceinline__ uint4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                        const PhiloxKeys& key) {
#pragma unroll
    for (int r = 0; r < kPhiloxRounds; ++r) {
        const uint64_t p0 = (uint64_t)kPhiloxM0 * c0;
        const uint64_t p1 = (uint64_t)kPhiloxM1 * c2;
        const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        c0 = hi1 ^ c1 ^ key.k0[r];
        c1 = lo1;
        c2 = hi0 ^ c3 ^ key.k1[r];
        c3 = lo0;
    }
    return make_uint4(c0, c1, c2, c3);
}

// N independent Philox4x32-10 calls advanced round by round: counters in
// (x0, x1, x2, x3)[j], results in place.  The calls' multiplies issue back to
// back, so their latencies overlap (one call's rounds are a dependent chain).
template <int N>
__device__ __forceinline__ void philox_n(uint32_t (&x0)[N], uint32_t (&x1)[N], uint32_t (&x2)[N], uint32_t (&x3)[N],
                                         const PhiloxKeys& key) {
#pragma unroll
    for (int r = 0; r < kPhiloxRounds; ++r) {
#pragma unroll
        for (int j = 0; j < N; ++j) {
            const uint64_t p0 = (uint64_t)kPhiloxM0 * x0[j];
            const uint64_t p1 = (uint64_t)kPhiloxM1 * x2[j];
            const uint32_t n0 = (uint32_t)(p1 >> 32) ^ x1[j] ^ key.k0[r];
            const uint32_t n2 = (uint32_t)(p0 >> 32) ^ x3[j] ^ key.k1[r];
            x1[j] = (uint32_t)p1;
            x3[j] = (uint32_t)p0;
            x0[j] = n0;
            x2[j] = n2;
        }
    }
}

// ---- byte / half packing -------------------------------------------------

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// Two signed int8 codes (bytes i0, i1 of w, each 0..3) as an exact half2.
// (code ^ 0x80) placed in the low mantissa byte of 1024.0 gives
// 1024 + 128 + code exactly; subtracting 1152 leaves code.
__device__ __forceinline__ uint32_t s8x2_to_h2(uint32_t w_xor80, uint32_t sel) {
    const uint32_t h = prmt(w_xor80, 0x64646464u, sel);
    __half2 v = *reinterpret_cast<const __half2*>(&h);
    v = __hsub2(v, __half2half2(__ushort_as_half((unsigned short)0x6480)));  // 1152.0
    return *reinterpret_cast<const uint32_t*>(&v);
}

// Two fp8 e4m3fn bytes (low 16 bits of w) as half2 (exact).
__device__ __forceinline__ uint32_t e4m3x2_to_h2(uint32_t w16) {
    uint32_t d;
    asm("{\n\t.reg .b16 lo;\n\tmov.b32 {lo, _}, %1;\n\tcvt.rn.f16x2.e4m3x2 %0, lo;\n\t}"
        : "=r"(d) : "r"(w16));
    return d;
}

__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
    __half2 v = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

// ---- legacy warp MMA (fp16 in, fp32 accumulate) --------------------------

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void mma1688(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t b0) {
    asm volatile(
        "mma.sync.aligned.m16n8k8.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(b0));
}

// ---- mbarrier + bulk asynchronous copy (TMA, non-tensor form) ------------

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;\n\tfence.proxy.async.shared::cta;" ::
                     : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

// Bulk copy global -> this CTA's shared memory, completion counted in bytes
// on `bar`.  dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// L2 prefetch of a contiguous range (a hint: no data is returned).  src
// 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity), "r"(1000000u)
        : "memory");
    return ok != 0;
}

// Bounded wait: each try_wait suspends for at most ~1 ms (hint above), so
// kMaxWaitTries bounds the wait to a few seconds before giving up.
constexpr int kMaxWaitTries = 4000;

template <int kTries = kMaxWaitTries>
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
    for (int i = 0; i < kTries; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

// Programmatic dependent launch: a kernel launched with the attribute may start
// while its predecessor drains; grid_dep_wait() blocks until the predecessor grid
// has completed and its memory is visible (a no-op for ordinary launches).
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

}  // namespace wc
