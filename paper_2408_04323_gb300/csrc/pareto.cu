// Pareto front of three maximised acquisition rows and a random k-subset of
// it: the parallel suggestion of MACE for one objective (Section 4.7, with
// the UCB, PI and EI rows of Section 4.5).
//
// The filter is exact and works in four steps:
//  1. pivots: the front of a strided sample of at most kSample candidates,
//     found by a chunk-local filter (pareto_local) and an all-pairs filter
//     of its survivors (pareto_global);
//  2. pivot_filter: every eligible candidate is compared with the pivots
//     (at most kPivCap, held in shared memory) and dropped at the first
//     pivot that dominates it; the others (at most SCOOT_PARETO_CAP) are
//     kept;
//  3. pareto_global: the kept candidates are compared with each other; those
//     none of them dominates form the front;
//  4. pareto_pick (one block): k rounds, each taking the front member with
//     the smallest (SplitMix64 key, index) pair above the previous pick.
// Why it is exact: any eligible candidate can serve as a pivot, so a
// dropped candidate is dominated and not on the front; a front member is
// never dropped; and a kept candidate x that some y dominates is dominated by
// a kept candidate too, since y is either kept or dropped for a pivot p that
// dominates y and hence x (p is kept: pivots are mutually non-dominating).
// The same argument covers the chunk-local filter of step 1 (a chunk's
// maximal elements play the pivots' part).
#include "internal.h"

namespace {

constexpr int kPThreads = 256;
constexpr int kChunk = kPThreads;            // candidates per chunk of the sample filter (one per thread)
constexpr int kGTile = 2048;                 // entries per shared-memory tile of the all-pairs filter
constexpr int kSample = 16384;               // candidates in the pivot sample
constexpr int kPivCap = 1024;                // pivots kept (any subset of the sample front serves)
constexpr int kCap = SCOOT_PARETO_CAP;
constexpr int kPickThreads = 1024;

struct ParetoHead {
    unsigned int n_samp;    // sample candidates kept by the chunk-local filter
    unsigned int n_piv;     // pivots found (only the first kPivCap are stored)
    unsigned int n_surv;    // candidates kept by the pivot filter (may exceed kCap)
    unsigned int n_front;   // front members
    unsigned int overflow;  // the pivot filter kept more than kCap candidates
    unsigned int pad[59];   // 256 bytes
};

constexpr size_t kSampOffset = sizeof(ParetoHead);
constexpr size_t kPivOffset = kSampOffset + (size_t)kSample * sizeof(float4);
constexpr size_t kSurvOffset = kPivOffset + (size_t)kPivCap * sizeof(float4);
constexpr size_t kFrontOffset = kSurvOffset + (size_t)kCap * sizeof(float4);
constexpr size_t kWorkBytes = kFrontOffset + (size_t)kCap * sizeof(float4);

// y dominates x: >= in every row and > in one.  NaN never dominates.
__device__ __forceinline__ bool dominates(float4 y, float4 x) {
    return y.x >= x.x && y.y >= x.y && y.z >= x.z && (y.x > x.x || y.y > x.y || y.z > x.z);
}

// Candidate i as (UCB, PI, EI, index bits); false (and -inf rows, which
// dominate no eligible candidate) when it is not eligible.
__device__ __forceinline__ bool load_triple(const float* __restrict__ acq, int64_t lda,
                                            const uint8_t* __restrict__ mask, int64_t i, float4& x) {
    // The four loads are independent (acq is readable for every i < n).
    const bool live = mask == nullptr || __ldg(mask + i) != 0;
    float u = __ldg(acq + i), p = __ldg(acq + lda + i), e = __ldg(acq + 2 * lda + i);
    const bool ok = live && !(isnan(u) || isnan(p) || isnan(e)) && u != -INFINITY && p != -INFINITY &&
                    e != -INFINITY;
    if (!ok) u = p = e = -INFINITY;
    x = make_float4(u, p, e, __uint_as_float((uint32_t)i));
    return ok;
}

// Step 1a: candidates i = s * stride (s < n_pos) in chunks of kChunk; the
// eligible ones no candidate of their chunk dominates go to out (capacity
// kSample >= n_pos, so it cannot fill).  One warp tests one candidate at a
// time, 64 comparisons per step, and stops at the first dominator.
__global__ void __launch_bounds__(kPThreads)
pareto_local(const float* __restrict__ acq, int64_t lda, const uint8_t* __restrict__ mask, int64_t n_pos,
             int64_t stride, float4* __restrict__ out, unsigned int* __restrict__ n_out) {
    __shared__ float4 tri[kChunk];
    __shared__ unsigned int elig[kChunk / 32];  // bit b of word w: chunk entry 32 w + b is eligible
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t n_chunks = (n_pos + kChunk - 1) / kChunk;
    for (int64_t c = blockIdx.x; c < n_chunks; c += gridDim.x) {
        {
            const int t = threadIdx.x;
            const int64_t s = c * kChunk + t;
            float4 x = make_float4(-INFINITY, -INFINITY, -INFINITY, 0.f);
            const bool ok = s < n_pos && load_triple(acq, lda, mask, s * stride, x);
            tri[t] = x;
            const unsigned int b = __ballot_sync(0xffffffffu, ok);
            if (lane == 0) elig[warp] = b;
        }
        __syncthreads();
        for (int w = warp; w < kChunk / 32; w += kPThreads / 32) {
            unsigned int bits = elig[w];  // the same in every lane
            while (bits) {
                const int j = w * 32 + __ffs(bits) - 1;
                bits &= bits - 1u;
                const float4 x = tri[j];
                bool dominated = false;
                for (int t = 0; t < kChunk; t += 64) {
                    const bool d = dominates(tri[t + lane], x) || dominates(tri[t + 32 + lane], x);
                    if (__any_sync(0xffffffffu, d)) {
                        dominated = true;
                        break;
                    }
                }
                if (!dominated && lane == 0) {
                    const unsigned int pos = atomicAdd(n_out, 1u);
                    if (pos < (unsigned int)kSample) out[pos] = x;
                }
            }
        }
        __syncthreads();  // tri and elig are rewritten for the next chunk
    }
}

// All-pairs filter of a short list: entries of in[0 .. min(*n_in, in_cap))
// that no entry dominates go to out; *n_out counts them all, only the first
// out_cap are stored.  A block takes eight entries at a time (one per warp)
// and streams the list through shared memory in tiles; a warp compares its
// entry with 64 tile entries per step and stops at the first dominator, the
// block at the first tile after which all eight are settled.  Does nothing
// once the pivot filter has overflowed.
__global__ void __launch_bounds__(kPThreads)
pareto_global(const float4* __restrict__ in, const unsigned int* __restrict__ n_in, unsigned int in_cap,
              float4* __restrict__ out, unsigned int* __restrict__ n_out, unsigned int out_cap,
              const unsigned int* __restrict__ overflow) {
    __shared__ float4 tile[kGTile];
    if (*overflow) return;  // the same value in every thread
    const unsigned int ns = min(*n_in, in_cap);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int kWarps = kPThreads / 32;
    for (unsigned int s0 = blockIdx.x * kWarps; s0 < ns; s0 += gridDim.x * kWarps) {
        const unsigned int s = s0 + warp;
        const bool alive = s < ns;
        const float4 x = alive ? in[s] : make_float4(0.f, 0.f, 0.f, 0.f);
        bool dominated = false;
        for (unsigned int t0 = 0; t0 < ns; t0 += kGTile) {
            const int cnt = (int)min((unsigned int)kGTile, ns - t0);
            __syncthreads();  // the previous tile is no longer read
            for (int t = threadIdx.x; t < cnt; t += kPThreads) tile[t] = in[t0 + t];
            for (int t = cnt + threadIdx.x; t < ((cnt + 63) & ~63); t += kPThreads)
                tile[t] = make_float4(-INFINITY, -INFINITY, -INFINITY, 0.f);
            __syncthreads();
            if (alive && !dominated)
                for (int t = 0; t < cnt; t += 64) {
                    const bool d = dominates(tile[t + lane], x) || dominates(tile[t + 32 + lane], x);
                    if (__any_sync(0xffffffffu, d)) {
                        dominated = true;
                        break;
                    }
                }
            if (__syncthreads_and(!alive || dominated)) break;
        }
        if (alive && !dominated && lane == 0) {
            const unsigned int pos = atomicAdd(n_out, 1u);
            if (pos < out_cap) out[pos] = x;
        }
    }
}

// Step 2: every candidate against the pivots in shared memory; a thread
// takes kFilterPer candidates at a time (their loads issued together).
constexpr int kFilterPer = 4;

__global__ void __launch_bounds__(kPThreads)
pivot_filter(const float* __restrict__ acq, int64_t lda, const uint8_t* __restrict__ mask, int64_t n,
             ParetoHead* __restrict__ head, const float4* __restrict__ piv, float4* __restrict__ surv,
             uint32_t* __restrict__ err) {
    __shared__ float4 sp[kPivCap];
    const int lane = threadIdx.x & 31;
    const int np = (int)min(head->n_piv, (unsigned int)kPivCap);
    for (int t = threadIdx.x; t < np; t += kPThreads) sp[t] = piv[t];
    __syncthreads();
    const int64_t step = (int64_t)gridDim.x * kPThreads * kFilterPer;
    for (int64_t base = (int64_t)blockIdx.x * kPThreads * kFilterPer; base < n; base += step) {
        float4 x[kFilterPer];
        bool keep[kFilterPer];
#pragma unroll
        for (int r = 0; r < kFilterPer; ++r) {
            const int64_t i = base + r * kPThreads + threadIdx.x;
            keep[r] = i < n && load_triple(acq, lda, mask, i, x[r]);
        }
#pragma unroll
        for (int r = 0; r < kFilterPer; ++r) {
            if (keep[r])
                for (int p = 0; p < np; ++p)
                    if (dominates(sp[p], x[r])) {
                        keep[r] = false;
                        break;
                    }
            const unsigned int ballot = __ballot_sync(0xffffffffu, keep[r]);
            if (ballot) {
                const int leader = __ffs(ballot) - 1;
                unsigned int pos0 = 0;
                if (lane == leader) pos0 = atomicAdd(&head->n_surv, (unsigned int)__popc(ballot));
                pos0 = __shfl_sync(0xffffffffu, pos0, leader);
                if (keep[r]) {
                    const unsigned int pos = pos0 + __popc(ballot & ((1u << lane) - 1u));
                    if (pos < (unsigned int)kCap) {
                        surv[pos] = x[r];
                    } else {
                        head->overflow = 1u;
                        atomicOr(err, SCOOT_DEVERR_CAPACITY);
                    }
                }
            }
        }
    }
}

// Output i (0-based) of the SplitMix64 generator seeded with `seed`
// (Steele, Lea and Flood, OOPSLA 2014): the state after i + 1 steps of the
// golden-ratio increment, passed through the generator's finaliser.
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t i) {
    uint64_t z = seed + (i + 1ull) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ bool pair_less(uint64_t ka, uint32_t ia, uint64_t kb, uint32_t ib) {
    return ka < kb || (ka == kb && ia < ib);
}

__global__ void __launch_bounds__(kPickThreads)
pareto_pick(const ParetoHead* __restrict__ head, const float4* __restrict__ front, int k, uint64_t seed,
            int64_t* __restrict__ idx, int32_t* __restrict__ count, int64_t* __restrict__ front_out,
            int64_t front_cap) {
    __shared__ uint64_t wk[kPickThreads / 32];
    __shared__ uint32_t wi[kPickThreads / 32];
    __shared__ uint64_t best_k;
    __shared__ uint32_t best_i;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool over = head->overflow != 0u;
    const unsigned int F = over ? 0u : head->n_front;
    if (front_out)
        for (int64_t t = tid; t < (int64_t)F && t < front_cap; t += kPickThreads) front_out[t] = (int64_t)__float_as_uint(front[t].w);
    // Index sentinel: real indices are below 2^31, so (max, max) is no pair.
    const uint32_t kNone = 0xFFFFFFFFu;
    uint64_t pk = 0;
    uint32_t pi = kNone;  // previous pick; kNone: none yet
    int picked = 0;
    for (int r = 0; r < k; ++r) {
        uint64_t bk = ~0ull;
        uint32_t bi = kNone;
        for (unsigned int t = tid; t < F; t += kPickThreads) {
            const uint32_t i = __float_as_uint(front[t].w);
            const uint64_t key = splitmix64_at(seed, i);
            const bool above = pi == kNone || pair_less(pk, pi, key, i);
            if (above && pair_less(key, i, bk, bi)) {
                bk = key;
                bi = i;
            }
        }
        for (int o = 16; o > 0; o >>= 1) {
            const uint64_t ok = __shfl_xor_sync(0xffffffffu, bk, o);
            const uint32_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (pair_less(ok, oi, bk, bi)) {
                bk = ok;
                bi = oi;
            }
        }
        if (lane == 0) {
            wk[warp] = bk;
            wi[warp] = bi;
        }
        __syncthreads();
        if (warp == 0) {
            bk = wk[lane];
            bi = wi[lane];
            for (int o = 16; o > 0; o >>= 1) {
                const uint64_t ok = __shfl_xor_sync(0xffffffffu, bk, o);
                const uint32_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
                if (pair_less(ok, oi, bk, bi)) {
                    bk = ok;
                    bi = oi;
                }
            }
            if (lane == 0) {
                best_k = bk;
                best_i = bi;
            }
        }
        __syncthreads();
        pk = best_k;
        pi = best_i;
        __syncthreads();  // best_k / best_i are rewritten next round
        if (pi == kNone) break;  // the front is exhausted (same in every thread)
        if (tid == 0) idx[r] = (int64_t)pi;
        ++picked;
    }
    if (tid == 0) {
        for (int r = picked; r < k; ++r) idx[r] = -1;
        count[0] = over ? -1 : picked;
        count[1] = over ? -1 : (int32_t)F;
    }
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

}  // namespace

extern "C" {

scoot_status scoot_select_pareto(scoot_ctx* ctx, const float* acq, int64_t lda, const uint8_t* mask, int64_t n,
                                 int32_t k, uint64_t seed, int64_t* idx, int32_t* count, int64_t* front,
                                 int64_t front_cap, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n = %lld < 0", (long long)n);
    if (n > 0x7FFFFFFFll) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n = %lld >= 2^31", (long long)n);
    if (k < 1 || k > SCOOT_MAX_Q) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "k = %d outside 1..%d", k, SCOOT_MAX_Q);
    if (!idx || !count) return scoot_fail(ctx, SCOOT_EINVAL, "idx or count is NULL");
    if (n > 0 && !acq) return scoot_fail(ctx, SCOOT_EINVAL, "acq is NULL");
    if (n > 0 && lda < n) return scoot_fail(ctx, SCOOT_EINVAL, "lda = %lld < n", (long long)lda);
    if (front && front_cap < 0) return scoot_fail(ctx, SCOOT_EINVAL, "front_cap < 0");
    if ((s = scoot_workspace(ctx, kWorkBytes)) != SCOOT_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    ParetoHead* head = reinterpret_cast<ParetoHead*>(ws);
    float4* samp = reinterpret_cast<float4*>(ws + kSampOffset);
    float4* piv = reinterpret_cast<float4*>(ws + kPivOffset);
    float4* surv = reinterpret_cast<float4*>(ws + kSurvOffset);
    float4* fr = reinterpret_cast<float4*>(ws + kFrontOffset);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SCOOT_CUDA(ctx, cudaMemsetAsync(head, 0, sizeof(ParetoHead), st));
    if (n > 0) {
        const int sms = sm_count(ctx->device);
        const int64_t stride = (n + kSample - 1) / kSample;
        const int64_t n_pos = (n + stride - 1) / stride;
        const int64_t chunks = (n_pos + kChunk - 1) / kChunk;
        pareto_local<<<(unsigned)chunks, kPThreads, 0, st>>>(acq, lda, mask, n_pos, stride, samp, &head->n_samp);
        SCOOT_LAUNCHED(ctx);
        pareto_global<<<(unsigned)sms, kPThreads, 0, st>>>(samp, &head->n_samp, kSample, piv, &head->n_piv,
                                                            kPivCap, &head->overflow);
        SCOOT_LAUNCHED(ctx);
        int64_t blocks = (n + kPThreads * kFilterPer - 1) / (kPThreads * kFilterPer);
        if (blocks > (int64_t)sms * 8) blocks = (int64_t)sms * 8;
        pivot_filter<<<(unsigned)blocks, kPThreads, 0, st>>>(acq, lda, mask, n, head, piv, surv, ctx->d_err);
        SCOOT_LAUNCHED(ctx);
        pareto_global<<<(unsigned)(sms * 8), kPThreads, 0, st>>>(surv, &head->n_surv, kCap, fr, &head->n_front,
                                                                  kCap, &head->overflow);
        SCOOT_LAUNCHED(ctx);
    }
    pareto_pick<<<1, kPickThreads, 0, st>>>(head, fr, k, seed, idx, count, front, front ? front_cap : 0);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // extern "C"
