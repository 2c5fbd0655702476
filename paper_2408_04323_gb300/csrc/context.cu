// Context: the device it is bound to, its workspace and its device error word.
#include <cstdarg>
#include <cstdio>
#include <new>

#include "internal.h"

scoot_status scoot_fail(scoot_ctx* ctx, scoot_status s, const char* fmt, ...) {
    if (ctx) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        std::vsnprintf(buf, sizeof(buf), fmt, ap);
        va_end(ap);
        ctx->err = buf;
    }
    return s;
}

scoot_status scoot_enter(scoot_ctx* ctx) {
    if (!ctx) return SCOOT_EINVAL;
    ctx->err.clear();
    cudaError_t e = cudaSetDevice(ctx->device);
    if (e != cudaSuccess) return scoot_fail(ctx, SCOOT_ECUDA, "cudaSetDevice(%d): %s", ctx->device, cudaGetErrorString(e));
    return SCOOT_OK;
}

scoot_status scoot_workspace(scoot_ctx* ctx, size_t bytes) {
    if (bytes <= ctx->ws_bytes) return SCOOT_OK;
    size_t want = bytes < (size_t(1) << 20) ? (size_t(1) << 20) : bytes;
    if (ctx->ws) {
        // The old buffer may still be read by queued kernels.
        SCOOT_CUDA(ctx, cudaDeviceSynchronize());
        SCOOT_CUDA(ctx, cudaFree(ctx->ws));
        ctx->ws = nullptr;
        ctx->ws_bytes = 0;
    }
    cudaError_t e = cudaMalloc(&ctx->ws, want);
    if (e != cudaSuccess) {
        ctx->ws = nullptr;
        return scoot_fail(ctx, SCOOT_ENOMEM, "workspace of %zu bytes: %s", want, cudaGetErrorString(e));
    }
    ctx->ws_bytes = want;
    return SCOOT_OK;
}

static scoot_status record_event(scoot_ctx* ctx, void* st) {
    const size_t k = ctx->mark_kind.size();
    if (k >= (size_t)SCOOT_MAX_MARKS + 1) return SCOOT_OK;  // later launches are not timed
    if (ctx->events.size() <= k) {
        cudaEvent_t e;
        SCOOT_CUDA(ctx, cudaEventCreate(&e));
        ctx->events.push_back(e);
    }
    SCOOT_CUDA(ctx, cudaEventRecord(static_cast<cudaEvent_t>(ctx->events[k]), static_cast<cudaStream_t>(st)));
    return SCOOT_OK;
}

scoot_status scoot_marks_begin(scoot_ctx* ctx, void* st) {
    if (!ctx->timing) return SCOOT_OK;
    ctx->mark_kind.clear();
    scoot_status s = record_event(ctx, st);
    if (s == SCOOT_OK) ctx->mark_kind.push_back(-1);
    return s;
}

scoot_status scoot_mark(scoot_ctx* ctx, void* st, int32_t kind) {
    if (!ctx->timing || ctx->mark_kind.empty()) return SCOOT_OK;
    scoot_status s = record_event(ctx, st);
    if (s == SCOOT_OK && ctx->mark_kind.size() < (size_t)SCOOT_MAX_MARKS + 1) ctx->mark_kind.push_back(kind);
    return s;
}

scoot_status scoot_check_pool(scoot_ctx* ctx, const uint32_t* cand, int64_t n, int64_t ld, int32_t d) {
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n = %lld < 0", (long long)n);
    if (d < 1 || d > SCOOT_MAX_DIM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "d = %d outside 1..%d", d, SCOOT_MAX_DIM);
    if (n == 0) return SCOOT_OK;
    if (!cand) return scoot_fail(ctx, SCOOT_EINVAL, "cand is NULL");
    if (!scoot_aligned16(cand)) return scoot_fail(ctx, SCOOT_EINVAL, "cand is not 16-byte aligned");
    if (ld < n || (ld & 3)) return scoot_fail(ctx, SCOOT_EINVAL, "ld = %lld must be >= n and a multiple of 4", (long long)ld);
    return SCOOT_OK;
}

extern "C" {

scoot_status scoot_ctx_create(int32_t device, scoot_ctx** out) {
    if (!out) return SCOOT_EINVAL;
    *out = nullptr;
    int count = 0;
    if (cudaGetDeviceCount(&count) != cudaSuccess || device < 0 || device >= count) {
        cudaGetLastError();
        return SCOOT_ECUDA;
    }
    scoot_ctx* ctx = new (std::nothrow) scoot_ctx();
    if (!ctx) return SCOOT_ENOMEM;
    ctx->device = device;
    if (cudaSetDevice(device) != cudaSuccess || cudaMalloc(&ctx->d_err, sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        delete ctx;
        return SCOOT_ECUDA;
    }
    if (cudaMemset(ctx->d_err, 0, sizeof(uint32_t)) != cudaSuccess) {
        cudaFree(ctx->d_err);
        delete ctx;
        return SCOOT_ECUDA;
    }
    *out = ctx;
    return SCOOT_OK;
}

scoot_status scoot_ctx_destroy(scoot_ctx* ctx) {
    if (!ctx) return SCOOT_OK;
    cudaSetDevice(ctx->device);
    cudaDeviceSynchronize();
    for (void* e : ctx->events) cudaEventDestroy(static_cast<cudaEvent_t>(e));
    if (ctx->ws) cudaFree(ctx->ws);
    if (ctx->d_err) cudaFree(ctx->d_err);
    delete ctx;
    return SCOOT_OK;
}

const char* scoot_last_error(const scoot_ctx* ctx) {
    return ctx ? ctx->err.c_str() : "null context";
}

scoot_status scoot_ctx_check(scoot_ctx* ctx, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    uint32_t word = 0;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SCOOT_CUDA(ctx, cudaMemcpyAsync(&word, ctx->d_err, sizeof(word), cudaMemcpyDeviceToHost, st));
    SCOOT_CUDA(ctx, cudaStreamSynchronize(st));
    if (word) SCOOT_CUDA(ctx, cudaMemsetAsync(ctx->d_err, 0, sizeof(uint32_t), st));
    if (word & SCOOT_DEVERR_TIMEOUT) return scoot_fail(ctx, SCOOT_ETIMEOUT, "a bounded device wait gave up");
    if (word & SCOOT_DEVERR_INDEX) return scoot_fail(ctx, SCOOT_EDEVICE, "a kernel met an index out of range");
    if (word & SCOOT_DEVERR_VALUE)
        return scoot_fail(ctx, SCOOT_EINVAL,
                          "a kernel met a non-finite feature, a label other than 0/1, or a fantasy state that does "
                          "not match its call");
    if (word & SCOOT_DEVERR_CAPACITY)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED,
                          "a kernel ran out of capacity (more than %d candidates survived the pivots of a Pareto "
                          "filter, or the fantasised front needed more boxes than box_cap)", SCOOT_PARETO_CAP);
    return SCOOT_OK;
}

scoot_status scoot_ctx_set_timing(scoot_ctx* ctx, int32_t enable) {
    if (!ctx) return SCOOT_EINVAL;
    ctx->timing = enable != 0;
    ctx->mark_kind.clear();
    return SCOOT_OK;
}

scoot_status scoot_ctx_set_tensor_cores(scoot_ctx* ctx, int32_t enable) {
    if (!ctx) return SCOOT_EINVAL;
    ctx->tensor_cores = enable != 0;
    return SCOOT_OK;
}

scoot_status scoot_ctx_phase_times(scoot_ctx* ctx, int32_t cap, int32_t* h_kind, float* h_ms, int32_t* count) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!count || cap < 0 || (cap > 0 && (!h_kind || !h_ms))) return scoot_fail(ctx, SCOOT_EINVAL, "bad output");
    const int n = ctx->mark_kind.empty() ? 0 : (int)ctx->mark_kind.size() - 1;
    *count = n;
    if (n == 0) return SCOOT_OK;
    SCOOT_CUDA(ctx, cudaEventSynchronize(static_cast<cudaEvent_t>(ctx->events[n])));
    for (int k = 0; k < n && k < cap; ++k) {
        h_kind[k] = ctx->mark_kind[k + 1];
        SCOOT_CUDA(ctx, cudaEventElapsedTime(&h_ms[k], static_cast<cudaEvent_t>(ctx->events[k]),
                                             static_cast<cudaEvent_t>(ctx->events[k + 1])));
    }
    return SCOOT_OK;
}

scoot_status scoot_ctx_workspace_bytes(const scoot_ctx* ctx, int64_t* bytes) {
    if (!ctx || !bytes) return SCOOT_EINVAL;
    *bytes = (int64_t)ctx->ws_bytes;
    return SCOOT_OK;
}

}  // extern "C"
