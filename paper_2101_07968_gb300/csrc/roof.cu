// Integer-ALU roof probe (measurement support, not part of the method).
//
// Runs exactly the per-transition operations of the DP fill -- max, subtract,
// min -- on register-resident values, 8 independent transitions per iteration
// and no memory traffic, so that the time of a launch gives the peak rate of DP
// transitions one GB300 can sustain for that operation mix and width.
#include "common.cuh"

namespace dc {
namespace {

template <typename T>
__global__ void __launch_bounds__(1024) roof_kernel(int64_t iters, uint32_t *__restrict__ sink)
{
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    T v[8], R[8], S[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        v[j] = T(tid * 2654435761u + 977u * j);
        R[j] = T(tid ^ (0x9e37u * (j + 1)));
        S[j] = T(j + 1);
    }
    for (int64_t it = 0; it < iters; it += 4) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = dmin(v[j], T(dmax(v[(j + 1) & 7], R[j]) - S[j]));
        }
    }
    uint64_t acc = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) acc ^= uint64_t(v[j]);
    sink[tid] = uint32_t(acc ^ (acc >> 32));
}

}  // namespace

cudaError_t launch_roof(int variant, int blocks, int threads, int64_t iters, uint32_t *sink,
                        cudaStream_t stream)
{
    if (variant == 0)
        roof_kernel<uint32_t><<<blocks, threads, 0, stream>>>(iters, sink);
    else
        roof_kernel<uint64_t><<<blocks, threads, 0, stream>>>(iters, sink);
    return cudaGetLastError();
}

}  // namespace dc
