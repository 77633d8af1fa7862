// Measured ceilings of the two on-chip resources that bound the simulation kernel (sm_103a):
//
//   k_int_peak   - integer issue: every thread runs 8 independent chains of x = (x + a) ^ b (one
//                  add and one xor per link; the two cannot be fused into one instruction), at
//                  full occupancy, so the count of integer operations per second is the rate at
//                  which the SMs issue integer ALU instructions.
//   k_smem_peak  - shared-memory bandwidth: every warp reads 16-byte words of a 16 KB shared
//                  buffer, lane i the word after lane i-1 (a conflict-free 512-byte access, four
//                  wavefronts), at full occupancy; bytes per second of shared-memory reads.
//
// The paper has no counterpart: these are the denominators of the roofline fractions that the
// benchmark reports for the simulation kernel, measured on the GPU that runs it instead of taken
// from a nominal lane count and clock.
#include <cuda_runtime.h>

#include <algorithm>

#include "sim_peaks.h"

namespace {

constexpr int kThreads = 256;
constexpr int kChains = 8;
constexpr int kSmemWords = 1024;  // int4 words: 16 KB

__global__ void __launch_bounds__(kThreads) k_int_peak(int iters, unsigned a, unsigned b, unsigned *sink) {
    unsigned x[kChains];
#pragma unroll
    for (int j = 0; j < kChains; ++j) x[j] = threadIdx.x * 2654435761u + blockIdx.x * 40503u + unsigned(j);
    #pragma unroll 1
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
#pragma unroll
            for (int j = 0; j < kChains; ++j) x[j] = (x[j] + a) ^ b;
        }
    }
    unsigned r = 0;
#pragma unroll
    for (int j = 0; j < kChains; ++j) r ^= x[j];
    if (r == 0x9e3779b9u) sink[blockIdx.x] = r;  // keeps the chains live; practically never stored
}

__global__ void __launch_bounds__(kThreads) k_smem_peak(int iters, unsigned *sink) {
    __shared__ int4 buf[kSmemWords];
    for (int i = threadIdx.x; i < kSmemWords; i += blockDim.x)
        buf[i] = make_int4(i, i * 3, i * 5, i * 7);
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    int4 acc = make_int4(0, 0, 0, 0);
    #pragma unroll 1
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int4 v = buf[((it * 8 + j + warp) * 32 + lane) & (kSmemWords - 1)];
            acc.x += v.x;
            acc.y ^= v.y;
            acc.z += v.z;
            acc.w ^= v.w;
        }
    }
    if ((acc.x ^ acc.y ^ acc.z ^ acc.w) == 0x7f4a7c15) sink[blockIdx.x] = unsigned(acc.x);
}

}  // namespace

extern "C" int sim_measure_peaks(double *out) {
    if (!out) return -1;
    int dev = 0, n_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -4;
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    int per_sm_int = 0, per_sm_smem = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_int, k_int_peak, kThreads, 0);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_smem, k_smem_peak, kThreads, 0);
    const int blocks_int = n_sm * std::max(per_sm_int, 1);
    const int blocks_smem = n_sm * std::max(per_sm_smem, 1);
    unsigned *sink = nullptr;
    if (cudaMalloc(&sink, sizeof(unsigned) * size_t(std::max(blocks_int, blocks_smem))) != cudaSuccess) return -6;
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    const int it_int = 20000, it_smem = 20000;
    float best_int = 1e30f, best_smem = 1e30f;
    for (int rep = 0; rep < 4; ++rep) {  // the first of each is a warm-up
        float ms = 0.f;
        cudaEventRecord(e0);
        k_int_peak<<<blocks_int, kThreads>>>(it_int, 0x9e3779b9u, 0x7f4a7c15u, sink);
        cudaEventRecord(e1);
        cudaEventSynchronize(e1);
        cudaEventElapsedTime(&ms, e0, e1);
        if (rep > 0) best_int = std::min(best_int, ms);
        cudaEventRecord(e0);
        k_smem_peak<<<blocks_smem, kThreads>>>(it_smem, sink);
        cudaEventRecord(e1);
        cudaEventSynchronize(e1);
        cudaEventElapsedTime(&ms, e0, e1);
        if (rep > 0) best_smem = std::min(best_smem, ms);
    }
    const cudaError_t err = cudaGetLastError();
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    cudaFree(sink);
    if (err != cudaSuccess) return -4;
    const double int_ops = double(blocks_int) * kThreads * double(it_int) * 4.0 * kChains * 2.0;
    const double smem_bytes = double(blocks_smem) * kThreads * double(it_smem) * 8.0 * 16.0;
    out[0] = int_ops / (double(best_int) * 1e-3);
    out[1] = smem_bytes / (double(best_smem) * 1e-3);
    out[2] = best_int;
    out[3] = best_smem;
    return 0;
}
