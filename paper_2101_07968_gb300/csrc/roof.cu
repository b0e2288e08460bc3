// Integer-ALU roof probe (measurement support, not part of the method).
//
// Runs exactly the per-transition operations of a DP fill on register-resident
// values, with no memory traffic, so that the time of a launch gives the peak
// rate of DP transitions one GB300 can sustain for that operation mix:
//  * 32-bit (the shifted form of the 32-bit passes): one add-then-max per
//    candidate and one 3-input min per two candidates;
//  * 64-bit (the work-list passes): max, subtract, min.
// Every thread performs 8 transitions per unit of `iters`.
#include "common.cuh"

namespace dc {
namespace {

__global__ void __launch_bounds__(1024) roof_kernel_s32(int64_t iters, uint32_t *__restrict__ sink)
{
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    int32_t v[8], Q[8], G[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        v[j] = int32_t((tid * 2654435761u + 977u * j) >> 3);
        Q[j] = -int32_t((tid ^ (0x9e37u * (j + 1))) & 0xfffffu);
        G[j] = j + 1;
    }
    for (int64_t it = 0; it < iters; it += 4) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            // 4 accumulators fold 2 candidates each: 8 transitions
#pragma unroll
            for (int j = u & 1; j < 8; j += 2) {
                const int32_t a = __viaddmax_s32(v[(j + 1) & 7], Q[j], G[j]);
                const int32_t b = __viaddmax_s32(v[(j + 3) & 7], Q[(j + 1) & 7], G[(j + 1) & 7]);
                v[j] = __vimin3_s32(v[j], a, b);
            }
        }
    }
    uint32_t acc = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) acc ^= uint32_t(v[j]);
    sink[tid] = acc;
}

__global__ void __launch_bounds__(1024) roof_kernel_u64(int64_t iters, uint32_t *__restrict__ sink)
{
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    uint64_t v[8], R[8], S[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        v[j] = uint64_t(tid * 2654435761u + 977u * j);
        R[j] = uint64_t(tid ^ (0x9e37u * (j + 1)));
        S[j] = uint64_t(j + 1);
    }
    for (int64_t it = 0; it < iters; it += 4) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = dmin(v[j], uint64_t(dmax(v[(j + 1) & 7], R[j]) - S[j]));
        }
    }
    uint64_t acc = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) acc ^= v[j];
    sink[tid] = uint32_t(acc ^ (acc >> 32));
}

}  // namespace

cudaError_t launch_roof(int variant, int blocks, int threads, int64_t iters, uint32_t *sink,
                        cudaStream_t stream)
{
    if (variant == 0)
        roof_kernel_s32<<<blocks, threads, 0, stream>>>(iters, sink);
    else
        roof_kernel_u64<<<blocks, threads, 0, stream>>>(iters, sink);
    return cudaGetLastError();
}

}  // namespace dc
