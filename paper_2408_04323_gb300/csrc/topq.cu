// Top-q selection for parallel suggestion (Section 4.7): the q largest
// acquisition values among eligible candidates, ties broken by the lowest
// index, in two passes.
//
// Every eligible candidate i becomes one 64-bit key whose order is the
// selection order: the high word is the acquisition value mapped to an
// order-preserving unsigned integer, the low word is 0xFFFFFFFF - i, so a
// larger key means a larger value or, on equal values, a lower index.
// Keys are unique, so "the q largest keys" is a single well-defined set.
//  pass 1: each block keeps, per thread, a sorted register list of its QT
//          best keys over a contiguous slice of the pool, then extracts the
//          block's q best by q rounds of a block-wide maximum;
//  pass 2: one block merges the per-block lists the same way.
// The per-block lists live in the context's workspace.
#include <mutex>

#include "device_common.cuh"
#include "internal.h"

namespace {

using namespace scoot_dev;

constexpr int kTopqThreads = 128;
constexpr int kMergeThreads = 256;

template <int QT>
__device__ __forceinline__ void insert(uint64_t (&lst)[QT], uint64_t x) {
    if (x <= lst[QT - 1]) return;
#pragma unroll
    for (int p = QT - 1; p > 0; --p) {
        const uint64_t prev = lst[p - 1];
        lst[p] = x > prev ? prev : (x > lst[p] ? x : lst[p]);
    }
    if (x > lst[0]) lst[0] = x;
}

__device__ __forceinline__ uint64_t warp_max(uint64_t v) {
    for (int o = 16; o > 0; o >>= 1) {
        const uint64_t w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

// q rounds of a block-wide maximum over the heads of the per-thread sorted
// lists; the winner pops its head.  Writes at most q keys to out (0 = none).
template <int QT>
__device__ void block_extract(uint64_t (&lst)[QT], int q, uint64_t* out) {
    __shared__ uint64_t wmax[32];
    __shared__ uint64_t best;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    for (int r = 0; r < q; ++r) {
        const uint64_t m = warp_max(lst[0]);
        if (lane == 0) wmax[warp] = m;
        __syncthreads();
        if (warp == 0) {
            uint64_t v = lane < nw ? wmax[lane] : 0ull;
            v = warp_max(v);
            if (lane == 0) best = v;
        }
        __syncthreads();
        const uint64_t b = best;
        if (threadIdx.x == 0) out[r] = b;
        if (b != 0ull && lst[0] == b) {
#pragma unroll
            for (int p = 0; p < QT - 1; ++p) lst[p] = lst[p + 1];
            lst[QT - 1] = 0ull;
        }
        __syncthreads();  // wmax / best are rewritten next round
    }
}

template <int QT>
__global__ void __launch_bounds__(kTopqThreads)
topq_pass1(const float* __restrict__ acq, const uint8_t* __restrict__ mask, int64_t n, int64_t slice,
           int q, uint64_t* __restrict__ partial) {
    uint64_t lst[QT];
#pragma unroll
    for (int p = 0; p < QT; ++p) lst[p] = 0ull;
    const int64_t b0 = (int64_t)blockIdx.x * slice;
    const int64_t b1 = b0 + slice < n ? b0 + slice : n;
    for (int64_t i = b0 + threadIdx.x; i < b1; i += blockDim.x) {
        const float v = acq[i];
        if ((mask == nullptr || mask[i] != 0) && !(v != v) && v != -INFINITY)
            insert<QT>(lst, make_key(v, (uint32_t)i));
    }
    block_extract<QT>(lst, q, partial + (int64_t)blockIdx.x * q);
}

template <int QT>
__global__ void __launch_bounds__(kMergeThreads)
topq_pass2(const uint64_t* __restrict__ partial, int64_t total, int q, int64_t* __restrict__ idx,
           float* __restrict__ val, int32_t* __restrict__ count) {
    __shared__ uint64_t result[SCOOT_MAX_Q];
    uint64_t lst[QT];
#pragma unroll
    for (int p = 0; p < QT; ++p) lst[p] = 0ull;
    for (int64_t k = threadIdx.x; k < total; k += blockDim.x) {
        const uint64_t x = partial[k];
        if (x) insert<QT>(lst, x);
    }
    block_extract<QT>(lst, q, result);
    __syncthreads();
    if (threadIdx.x == 0) {
        int c = 0;
        for (int r = 0; r < q; ++r) {
            const uint64_t k = result[r];
            if (k) {
                idx[r] = key_index(k);
                val[r] = key_value(k);
                ++c;
            } else {
                idx[r] = -1;
                val[r] = -INFINITY;
            }
        }
        *count = c;
    }
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

template <int QT>
scoot_status run(scoot_ctx* ctx, const float* acq, const uint8_t* mask, int64_t n, int q, int64_t* idx,
                 float* val, int32_t* count, cudaStream_t st) {
    // One slice per block; at least 8 keys per thread, at most 4 blocks per SM.
    int64_t blocks = (n + kTopqThreads * 8 - 1) / (kTopqThreads * 8);
    const int64_t cap = (int64_t)sm_count(ctx->device) * 4;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    const int64_t slice = (n + blocks - 1) / blocks;
    scoot_status s = scoot_workspace(ctx, (size_t)blocks * q * sizeof(uint64_t));
    if (s != SCOOT_OK) return s;
    uint64_t* partial = static_cast<uint64_t*>(ctx->ws);
    topq_pass1<QT><<<(unsigned)blocks, kTopqThreads, 0, st>>>(acq, mask, n, slice, q, partial);
    SCOOT_LAUNCHED(ctx);
    topq_pass2<QT><<<1, kMergeThreads, 0, st>>>(partial, blocks * q, q, idx, val, count);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // namespace

extern "C" scoot_status scoot_select_topq(scoot_ctx* ctx, const float* acq, const uint8_t* mask, int64_t n,
                                          int32_t q, int64_t* idx, float* val, int32_t* count,
                                          void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (q < 1 || q > SCOOT_MAX_Q) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "q = %d outside 1..%d", q, SCOOT_MAX_Q);
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n < 0");
    if (n > 0xFFFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n = %lld >= 2^32", (long long)n);
    if (!idx || !val || !count || (n > 0 && !acq)) return scoot_fail(ctx, SCOOT_EINVAL, "NULL output or input");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (q <= 1) return run<1>(ctx, acq, mask, n, q, idx, val, count, st);
    if (q <= 4) return run<4>(ctx, acq, mask, n, q, idx, val, count, st);
    if (q <= 16) return run<16>(ctx, acq, mask, n, q, idx, val, count, st);
    return run<64>(ctx, acq, mask, n, q, idx, val, count, st);
}

// ---------------------------------------------------------------------------
// Allocation-free variant.
//
// Some callers cannot allocate device memory when they select: code running
// under an allocator that forbids new allocations while it is active (for
// example a caching allocator in the middle of a stream capture, or an
// embedding process whose memory pool is sized up front), or callers that
// hold no scoot_ctx because creating one allocates.  For them the per-block
// partial lists live in this fixed device array instead of a workspace.  The
// array exists once per device for as long as the library is loaded.

namespace {

constexpr int kStaticKeys = 32768;  // 256 KiB of 64-bit keys
static __device__ __align__(256) uint64_t g_topq_scratch[kStaticKeys];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
uint64_t* g_scratch_ptr[kMaxDevices];  // guarded by g_scratch_mutex; NULL until a lookup succeeds

// Device address of the scratch array on `device` (current), looked up on
// the first call that needs it.  A failed lookup is not remembered: the next
// call tries again, so one call made at a bad moment (inside a stream
// capture, say) does not disable the entry point for the process.
uint64_t* scratch_on(int device) {
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_ptr[device]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_topq_scratch) != cudaSuccess) {
            cudaGetLastError();  // this call reports the failure; leave no error pending
            return nullptr;
        }
        g_scratch_ptr[device] = static_cast<uint64_t*>(p);
    }
    return g_scratch_ptr[device];
}

}  // namespace

extern "C" scoot_status scoot_select_topq_static(const float* acq, const uint8_t* mask, int64_t n, int32_t q,
                                                 int64_t* idx, float* val, int32_t* count, void* stream) {
    if (q < 1 || q > SCOOT_MAX_Q) return SCOOT_EUNSUPPORTED;
    if (n < 0) return SCOOT_EINVAL;
    if (n > 0xFFFFFFFFll) return SCOOT_EUNSUPPORTED;
    if (!idx || !val || !count || (n > 0 && !acq)) return SCOOT_EINVAL;
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kMaxDevices) {
        cudaGetLastError();
        return SCOOT_ECUDA;
    }
    // Host code cannot use the array's name as a device pointer: its address
    // on this device is looked up with the device current.
    uint64_t* partial = scratch_on(device);
    if (!partial) return SCOOT_ECUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) {
        cudaGetLastError();
        return SCOOT_ECUDA;
    }
    // Blocks are capped so that blocks * q keys fit the array; every key pass
    // 2 reads is written by pass 1 of the same call, so nothing needs clearing.
    int64_t blocks = (n + kTopqThreads * 8 - 1) / (kTopqThreads * 8);
    int64_t cap = (int64_t)(sms > 0 ? sms : 1) * 4;
    if (cap > kStaticKeys / q) cap = kStaticKeys / q;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    const int64_t slice = (n + blocks - 1) / blocks;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // An error left pending by the caller's earlier work is not this call's:
    // clear it so that the status below reports only these two launches.
    cudaGetLastError();
    auto go = [&](auto p1, auto p2) {
        p1<<<(unsigned)blocks, kTopqThreads, 0, st>>>(acq, mask, n, slice, q, partial);
        p2<<<1, kMergeThreads, 0, st>>>(partial, blocks * q, q, idx, val, count);
    };
    if (q <= 1) go(topq_pass1<1>, topq_pass2<1>);
    else if (q <= 4) go(topq_pass1<4>, topq_pass2<4>);
    else if (q <= 16) go(topq_pass1<16>, topq_pass2<16>);
    else go(topq_pass1<64>, topq_pass2<64>);
    return cudaGetLastError() == cudaSuccess ? SCOOT_OK : SCOOT_ECUDA;
}
