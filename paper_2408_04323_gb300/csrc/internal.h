// Internal definitions shared by the host and CUDA translation units of libscoot.
#pragma once

#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <string>

#include "../../include/scoot.h"

#ifdef __CUDACC__
#include <cuda_runtime.h>
#endif

// Bits of the device error word.
#define SCOOT_DEVERR_INDEX   1u   // a node, feature or box index out of range
#define SCOOT_DEVERR_TIMEOUT 2u   // a bounded wait gave up

struct scoot_ctx {
    int32_t device = 0;
    std::string err;
    void* ws = nullptr;          // device workspace (grown on demand)
    size_t ws_bytes = 0;
    uint32_t* d_err = nullptr;   // device error word
};

scoot_status scoot_fail(scoot_ctx* ctx, scoot_status s, const char* fmt, ...);
// Make ctx->device current; sets an error on failure.
scoot_status scoot_enter(scoot_ctx* ctx);
// Ensure at least `bytes` of workspace (synchronising the device if it grows).
scoot_status scoot_workspace(scoot_ctx* ctx, size_t bytes);

static inline bool scoot_aligned16(const void* p) {
    return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// Checks shared by the device entry points.
scoot_status scoot_check_pool(scoot_ctx* ctx, const uint32_t* cand, int64_t n, int64_t ld, int32_t d);

#ifdef __CUDACC__
// Index list of live candidates built by scoot_compact in the context workspace.
struct ScootList {
    int32_t* list;
    unsigned int* count;
};
// Compacts the indices i < n with mask[i] != 0 into out->list (count on the
// device); where mask[i] == 0, fill[i] = fill_bits if fill is not NULL.
scoot_status scoot_compact(scoot_ctx* ctx, const uint8_t* mask, int64_t n, uint32_t* fill, uint32_t fill_bits,
                           cudaStream_t st, ScootList* out);

#define SCOOT_CUDA(ctx, call)                                                          \
    do {                                                                               \
        cudaError_t e_ = (call);                                                       \
        if (e_ != cudaSuccess)                                                         \
            return scoot_fail((ctx), SCOOT_ECUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
    } while (0)
#define SCOOT_LAUNCHED(ctx)                                                            \
    do {                                                                               \
        cudaError_t e_ = cudaGetLastError();                                           \
        if (e_ != cudaSuccess)                                                         \
            return scoot_fail((ctx), SCOOT_ECUDA, "kernel launch: %s", cudaGetErrorString(e_)); \
    } while (0)
#endif
