// Gate (§6 meter-loop box; certified vs risk-ranked thresholds, §4.3):
// keep the compressed path of a query-head cell iff meter_raw <= tau, and of
// a KV head iff all of its G query heads keep (any-of-G fallback).  The joint
// gate (§4.2 "Value side and the joint event") also requires the value term
// to be at most tau_v * max ||v|| (pass_V), decided in float32.
#include "wc_kernels.cuh"

namespace wc {

namespace {

constexpr int kGateThreads = 256;

__global__ void __launch_bounds__(kGateThreads) gate_kernel(const float* __restrict__ meter_raw,
                                                            const float* __restrict__ value_term,
                                                            const float* __restrict__ v_max, int n_cells,
                                                            int group, float tau, float tau_v, uint8_t* keep_q,
                                                            uint8_t* keep_kv, int32_t* n_kept) {
    int kept_q = 0, kept_kv = 0;
    const int n_kv = n_cells / group;
    for (int i = threadIdx.x; i < n_kv; i += kGateThreads) {
        bool all = true;
        for (int j = 0; j < group; ++j) {
            const size_t cell = (size_t)i * group + j;
            bool k = meter_raw[cell] <= tau;                                    // NaN -> false
            if (value_term) k = k && value_term[cell] <= __fmul_rn(tau_v, v_max[cell]);
            keep_q[cell] = k ? 1 : 0;
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
    gate_kernel<<<1, kGateThreads, 0, stream>>>(meter_raw, value_term, v_max, n_cells, group, tau, tau_v, keep_q,
                                                keep_kv, n_kept);
    return cudaGetLastError();
}

}  // namespace wc
