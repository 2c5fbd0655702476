// Measurement probes: the peaks that the kernels of this library are
// reported against where no vendor figure applies.
//  - probe_fma: long independent chains of fp32 fused multiply-adds (FFMA),
//    or of packed pairs (FFMA2, two fp32 FMAs per instruction), per thread:
//    the FP32 ALU peak the posterior / acquisition kernels are bound by;
//  - probe_gather: dependent walks through an array of 8-byte nodes in
//    shared memory, one walk per thread, each step one node load whose index
//    depends on the previous node and the walker's feature vector, the
//    access pattern of the forest kernel's tree walks: its node-visit peak.
// Results land in `sink` so that no chain is dead code.
#include "device_common.cuh"
#include "internal.h"

namespace {

constexpr int kChains = 8;

template <bool PACKED>
__global__ void __launch_bounds__(256) probe_fma(int iters, float seed, float* sink) {
    if (PACKED) {
        float2 acc[kChains];
#pragma unroll
        for (int k = 0; k < kChains; ++k) acc[k] = make_float2(seed + k, seed - k + threadIdx.x * 1e-7f);
        const float2 mul = make_float2(0.999999f, 0.9999999f), add = make_float2(1e-7f, -1e-7f);
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int k = 0; k < kChains; ++k) acc[k] = __ffma2_rn(acc[k], mul, add);
        }
        float s = 0.0f;
#pragma unroll
        for (int k = 0; k < kChains; ++k) s += acc[k].x + acc[k].y;
        if (s == 1234.5f) sink[blockIdx.x] = s;  // practically never true; keeps the chains live
    } else {
        float acc[2 * kChains];
#pragma unroll
        for (int k = 0; k < 2 * kChains; ++k) acc[k] = seed + k + threadIdx.x * 1e-7f;
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int k = 0; k < 2 * kChains; ++k) acc[k] = fmaf(acc[k], 0.999999f, 1e-7f);
        }
        float s = 0.0f;
#pragma unroll
        for (int k = 0; k < 2 * kChains; ++k) s += acc[k];
        if (s == 1234.5f) sink[blockIdx.x] = s;
    }
}

// Node: {float threshold, u16 left, u8 feature, u8 flags}, as scoot_node.
__global__ void __launch_bounds__(256) probe_gather(int n_nodes, int steps, uint32_t seed, float* sink) {
    extern __shared__ __align__(16) uint2 nodes[];
    // A complete binary tree of n_nodes nodes with random thresholds.
    for (int k = threadIdx.x; k < n_nodes; k += blockDim.x) {
        uint32_t h = (uint32_t)k * 2654435761u ^ seed;
        h ^= h >> 15;
        const float thr = (float)(h & 0xFFFF) * (1.0f / 65536.0f);
        // node k splits (children 2k + 1 and 2k + 2) when both exist, else is a leaf
        const uint32_t left = 2u * (uint32_t)k + 2u < (uint32_t)n_nodes ? 2u * (uint32_t)k + 1u : 0u;
        nodes[k] = make_uint2(__float_as_uint(thr), left | ((h >> 16) & 7u) << 16);
    }
    __syncthreads();
    float x[8];
    uint32_t h = (blockIdx.x * blockDim.x + threadIdx.x) * 747796405u + seed;
#pragma unroll
    for (int f = 0; f < 8; ++f) {
        h = h * 1664525u + 1013904223u;
        x[f] = (float)(h >> 8) * (1.0f / 16777216.0f);
    }
    uint32_t node = 0, visits = 0;
    for (int s = 0; s < steps; ++s) {
        const uint2 nd = nodes[node];
        const uint32_t left = nd.y & 0xFFFFu;
        const int feat = (int)((nd.y >> 16) & 7u);
        // a leaf (left == 0) restarts the walk at the root, as the next tree would
        node = left == 0u ? 0u : left + (x[feat] > __uint_as_float(nd.x) ? 1u : 0u);
        ++visits;
    }
    // seed is a run-time value, so the walk cannot be proven dead; a node
    // index never equals it in practice
    if (node == seed) sink[blockIdx.x] = (float)visits;
}

}  // namespace

extern "C" {

scoot_status scoot_probe_fma(scoot_ctx* ctx, int32_t packed, int32_t blocks, int32_t iters, float* sink,
                             void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (blocks < 1 || iters < 1 || !sink) return scoot_fail(ctx, SCOOT_EINVAL, "bad probe arguments");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (packed)
        probe_fma<true><<<blocks, 256, 0, st>>>(iters, 1.0f, sink);
    else
        probe_fma<false><<<blocks, 256, 0, st>>>(iters, 1.0f, sink);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_probe_gather(scoot_ctx* ctx, int32_t n_nodes, int32_t blocks, int32_t steps, float* sink,
                                void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n_nodes < 1 || n_nodes > 12288 || blocks < 1 || steps < 1 || !sink)
        return scoot_fail(ctx, SCOOT_EINVAL, "bad probe arguments");
    const size_t smem = (size_t)n_nodes * 8;
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(probe_gather, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    probe_gather<<<blocks, 256, smem, static_cast<cudaStream_t>(stream)>>>(n_nodes, steps, 0x9E3779B9u, sink);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // extern "C"
