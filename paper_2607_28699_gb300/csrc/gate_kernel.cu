// Gate (§6 meter-loop box; certified vs risk-ranked thresholds, §4.3):
// keep the compressed path of a query-head cell iff meter_raw <= tau, and of
// a KV head iff all of its G query heads keep (any-of-G fallback).  The joint
// gate (§4.2 "Value side and the joint event") also requires the value term
// to be at most tau_v * max ||v|| (pass_V), decided in float32.
#include "wc_kernels.cuh"

namespace wc {

namespace {

constexpr int kGateThreads = 1024;

// One CTA (counts reduced in a fixed order, no atomics).  A thread takes whole
// KV heads: the first 8 meters of a head are loaded before any is compared, so a
// head costs one memory latency, not one per query head.
__global__ void __launch_bounds__(kGateThreads) gate_kernel(const float* __restrict__ meter_raw,
                                                            const float* __restrict__ value_term,
                                                            const float* __restrict__ v_max, int n_cells,
                                                            int group, float tau, float tau_v, uint8_t* keep_q,
                                                            uint8_t* keep_kv, int32_t* n_kept) {
    grid_dep_launch();   // a dependent launch may be queued now: it waits for this grid
    grid_dep_wait();     // the meters may come from the preceding kernel
    int kept_q = 0, kept_kv = 0;
    const int n_kv = n_cells / group;
    for (int i = threadIdx.x; i < n_kv; i += kGateThreads) {
        const size_t base = (size_t)i * group;
        float m[kMaxGroup], vt[kMaxGroup], vm[kMaxGroup];
#pragma unroll
        for (int j = 0; j < kMaxGroup; ++j) {
            m[j] = vt[j] = vm[j] = 0.f;
            if (j < group) {
                m[j] = meter_raw[base + j];
                if (value_term) {
                    vt[j] = value_term[base + j];
                    vm[j] = v_max[base + j];
                }
            }
        }
        bool all = true;
#pragma unroll
        for (int j = 0; j < kMaxGroup; ++j) {
            if (j < group) {
                bool k = m[j] <= tau;                                          // NaN -> false
                if (value_term) k = k && vt[j] <= __fmul_rn(tau_v, vm[j]);
                keep_q[base + j] = k ? 1 : 0;
                kept_q += k;
                all = all && k;
            }
        }
        for (int j = kMaxGroup; j < group; ++j) {   // groups wider than 8 query heads
            bool k = meter_raw[base + j] <= tau;
            if (value_term) k = k && value_term[base + j] <= __fmul_rn(tau_v, v_max[base + j]);
            keep_q[base + j] = k ? 1 : 0;
            kept_q += k;
            all = all && k;
        }
        keep_kv[i] = all ? 1 : 0;
        kept_kv += all;
    }
    __shared__ int red[2][kGateThreads / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        kept_q += __shfl_xor_sync(0xffffffffu, kept_q, o);
        kept_kv += __shfl_xor_sync(0xffffffffu, kept_kv, o);
    }
    if ((threadIdx.x & 31) == 0) {
        red[0][threadIdx.x >> 5] = kept_q;
        red[1][threadIdx.x >> 5] = kept_kv;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int a = 0, b = 0;
        for (int w = 0; w < kGateThreads / 32; ++w) {
            a += red[0][w];
            b += red[1][w];
        }
        n_kept[0] = a;
        n_kept[1] = b;
    }
}

}  // namespace

cudaError_t launch_gate(const float* meter_raw, const float* value_term, const float* v_max, int n_cells, int group,
                        float tau, float tau_v, uint8_t* keep_q, uint8_t* keep_kv, int32_t* n_kept,
                        cudaStream_t stream) {
    static bool configured = false;   // same carveout as the decode kernels
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(gate_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                             (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    // a programmatic dependent of the preceding kernel (the decode's merge): its CTA
    // becomes resident while that grid drains and waits for it (griddepcontrol.wait)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(kGateThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gate_kernel, meter_raw, value_term, v_max, n_cells, group, tau, tau_v, keep_q,
                              keep_kv, n_kept);
}

}  // namespace wc
