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
        return scoot_fail(ctx, SCOOT_EINVAL, "a kernel met a non-finite feature or a label other than 0/1");
    if (word & SCOOT_DEVERR_CAPACITY)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "more than %d candidates survived the pivots of a Pareto filter",
                          SCOOT_PARETO_CAP);
    return SCOOT_OK;
}

scoot_status scoot_ctx_workspace_bytes(const scoot_ctx* ctx, int64_t* bytes) {
    if (!ctx || !bytes) return SCOOT_EINVAL;
    *bytes = (int64_t)ctx->ws_bytes;
    return SCOOT_OK;
}

}  // extern "C"
