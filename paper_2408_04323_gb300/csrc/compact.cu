// Stream compaction of the live candidates (mask[i] != 0) into an index list
// held in the context's workspace, so that the forest walk and the scoring
// kernels spend their lanes on candidates that are still in play.  Entries of
// an optional output array that belong to masked-out candidates receive a
// fill value in the same pass (0 votes, -inf acquisition).
#include "internal.h"

namespace {

constexpr int kCompactThreads = 256;

__global__ void __launch_bounds__(kCompactThreads)
compact_kernel(const uint8_t* __restrict__ mask, int64_t n, int32_t* __restrict__ list,
               unsigned int* __restrict__ count, uint32_t* __restrict__ fill, uint32_t fill_bits, int fill_rows,
               int64_t fill_ld) {
    __shared__ unsigned int warp_count[kCompactThreads / 32];
    __shared__ unsigned int block_base;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t stride = (int64_t)gridDim.x * kCompactThreads;
    for (int64_t i0 = (int64_t)blockIdx.x * kCompactThreads; i0 < n; i0 += stride) {
        const int64_t i = i0 + threadIdx.x;
        const bool in = i < n;
        const bool live = in && mask[i] != 0;
        if (in && !live && fill)
            for (int r = 0; r < fill_rows; ++r) fill[r * fill_ld + i] = fill_bits;
        const unsigned int ballot = __ballot_sync(0xffffffffu, live);
        if (lane == 0) warp_count[warp] = __popc(ballot);
        __syncthreads();
        if (threadIdx.x == 0) {
            unsigned int total = 0;
            for (int w = 0; w < kCompactThreads / 32; ++w) {
                const unsigned int c = warp_count[w];
                warp_count[w] = total;  // exclusive prefix
                total += c;
            }
            block_base = total ? atomicAdd(count, total) : 0u;
        }
        __syncthreads();
        if (live) {
            const unsigned int below = __popc(ballot & ((1u << lane) - 1u));
            list[block_base + warp_count[warp] + below] = (int32_t)i;
        }
        __syncthreads();  // warp_count / block_base are rewritten next iteration
    }
}

}  // namespace

scoot_status scoot_compact(scoot_ctx* ctx, const uint8_t* mask, int64_t n, uint32_t* fill, uint32_t fill_bits,
                           cudaStream_t st, ScootList* out, int fill_rows, int64_t fill_ld) {
    if (n > 0x7FFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "compaction of %lld > 2^31 candidates", (long long)n);
    const size_t bytes = 256 + (size_t)n * sizeof(int32_t);
    scoot_status s = scoot_workspace(ctx, bytes);
    if (s != SCOOT_OK) return s;
    out->count = static_cast<unsigned int*>(ctx->ws);
    out->list = reinterpret_cast<int32_t*>(static_cast<char*>(ctx->ws) + 256);
    SCOOT_CUDA(ctx, cudaMemsetAsync(out->count, 0, sizeof(unsigned int), st));
    if (n == 0) return SCOOT_OK;
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, ctx->device);
    int64_t blocks = (n + kCompactThreads - 1) / kCompactThreads;
    const int64_t cap = (int64_t)(sms > 0 ? sms : 1) * 8;
    if (blocks > cap) blocks = cap;
    compact_kernel<<<(unsigned)blocks, kCompactThreads, 0, st>>>(mask, n, out->list, out->count, fill, fill_bits,
                                                                 fill_rows, fill_ld);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}
