// k_probe.cu -- a measurement aid, not part of the path: the fp32 FMA
// throughput of the device, against which the exact search's ALU roofline is
// stated (SMs x 128 lanes x 2 flops x the SM clock is the nominal figure).
#include "fw_internal.h"

namespace fw {
namespace {

constexpr int PR_T = 256;    // threads per block
constexpr int PR_CHAINS = 16;  // independent FMA chains per thread (covers the FMA latency)

__global__ void __launch_bounds__(PR_T) k_fma_probe(int iters, float *out)
{
    const float b = 0.999999f, c = 1e-7f * (float)(threadIdx.x + 1);
    float x[PR_CHAINS];
#pragma unroll
    for (int i = 0; i < PR_CHAINS; ++i) x[i] = (float)(i + 1) * 1e-3f;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < PR_CHAINS; ++i) x[i] = fmaf(x[i], b, c);
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < PR_CHAINS; ++i) s += x[i];
    out[(int64_t)blockIdx.x * PR_T + threadIdx.x] = s;
}

}  // namespace

fw_status fp32_fma_probe(int blocks, int iters, float *out, cudaStream_t s)
{
    FW_LAUNCH(k_fma_probe, (unsigned)blocks, PR_T, 0, s, iters, out);
    return FW_OK;
}

}  // namespace fw
