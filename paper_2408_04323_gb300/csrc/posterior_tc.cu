// GP posterior (Section 4.3) with the whitened rows V = L^{-1} k(X, x) on
// the fifth-generation tensor cores (tcgen05), for n_pad <= 256 rows.
//
// V^T = K*^T L^{-T} is a dense contraction: for a tile of 128 candidates,
// A = K*^T [128 x n] (the candidates' covariance rows) and B = L^{-1} [n x n]
// (row i of B is row i of L^{-1}, so D[x][i] = sum_c K*[c][x] L^{-1}[i][c]).
// Both operands are fp32 values split into three bf16 parts,
//   x = x_h + x_m + x_l  (x_h = bf16(x), x_m = bf16(x - x_h), x_l = bf16(x - x_h - x_m)),
// which hold all 24 bits of an fp32 significand (each part to within 2^-8
// of the remainder it takes).  The product keeps the six part products down
// to order 2^-16 and drops m l, l m and l l (order 2^-24, one fp32
// rounding).  The tensor core's fp32 accumulation truncates once per MMA
// relative to the accumulator's magnitude, so the full-size products h h go
// to a main accumulator (one truncation per 16 columns of L^{-1}) and the
// five smaller ones (h m, m h, h l, l h, m m) to a correction accumulator,
// where their truncations weigh 2^-8 less; V = main + corr.
//
// One CTA per SM, 16 SIMT warps and a control warp: SIMT thread t serves
// candidate row t mod 128 (the TMEM lane its warp can read) and column
// quarter t / 128.  Per objective the
// rows of L^{-1} go in k-blocks of 32 columns; k-block kb only reaches output
// rows i >= 32 kb (L^{-1} is lower triangular), so its products are MMAs of
// N = n_pad - 32 kb columns starting at column 32 kb of each accumulator
// (main at TMEM columns [0, n_pad), corrections at [n_pad, 2 n_pad)).  Pipeline per
// k-block g (counted over the CTA's whole sequence):
//   - wait until the MMAs of g - 2 are done (mbarrier), freeing A slot g mod 2
//     and B slot (g + 1) mod 3;
//   - cp.async the three B parts of k-block g + 1 (from the split copy of
//     L^{-1} prepared once per call by bsplit_kernel) into B slot (g + 1) mod 3;
//   - every SIMT thread evaluates its 8 covariances of k-block g, splits them,
//     stores the parts into A slot g mod 2 and arrives on its full barrier
//     (the MMAs of g - 1 run meanwhile);
//   - the control thread waits for A and B of g, issues the 12 MMAs of k-block
//     g (2 K-steps x 6 part products) and commits them to mbarrier g mod 2.
// After the last k-block the threads read D back (tcgen05.ld), write V in the
// tiled float4-group layout of the fantasy pass (vtile_index), and finish mu
// and sigma^2, or in their place the acquisition (EI, or MACE's UCB, PI and
// EI) when V is not wanted.
//
// Operand layout in shared memory: the canonical no-swizzle K-major form of
// a 32-wide k-block: 8-row x 16-byte core matrices, 128 bytes apart along K
// (leading byte offset) and 512 bytes apart along the rows (stride byte
// offset).
#include <cuda_bf16.h>

#include "device_common.cuh"
#include "internal.h"

namespace {

using namespace scoot_dev;

constexpr int kTM = 128;          // candidates per tile: the MMA's M and the TMEM lanes
constexpr int kKB = 32;           // columns of L^{-1} per k-block
constexpr int kQt = 4;            // threads per candidate row (column quarters of a k-block)
constexpr int kThr = kTM * kQt;   // SIMT threads (16 warps); one more warp issues copies and MMAs
constexpr int kParts = 3;         // bf16 parts of an fp32 operand
constexpr uint32_t kLBO = 128;    // bytes between core matrices along K
constexpr uint32_t kSBO = 512;    // bytes between 8-row groups of a k-block
constexpr uint32_t kAPart = kTM * kKB * 2;  // bytes of one part of an A k-block (8 KiB)
constexpr int kMaxD = SCOOT_MAX_DIM;
constexpr unsigned long long kWaitNs = 2000000000ull;  // bounded waits give up after 2 s

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// Byte offset of element (row, kk) of a k-block in the canonical layout.
__host__ __device__ __forceinline__ uint32_t canon_off(int row, int kk) {
    return (uint32_t)((row & 7) * 16 + (row >> 3) * (int)kSBO + (kk >> 3) * (int)kLBO + (kk & 7) * 2);
}

// Shared-memory matrix descriptor (tcgen05): start address, leading and
// stride byte offsets (each >> 4), descriptor version 1, no swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
    return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)((kLBO >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((kSBO >> 4) & 0x3FFFu) << 32) | (1ull << 46);
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, M = 128, N columns.
__device__ __forceinline__ uint32_t instr_desc(uint32_t N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((N >> 3) << 17) | ((uint32_t)(kTM >> 4) << 24);
}

// The three bf16 parts of x.
__device__ __forceinline__ void split3(float x, __nv_bfloat16& h, __nv_bfloat16& m, __nv_bfloat16& l) {
    h = __float2bfloat16_rn(x);
    const float r1 = x - __bfloat162float(h);  // exact
    m = __float2bfloat16_rn(r1);
    const float r2 = r1 - __bfloat162float(m);  // exact
    l = __float2bfloat16_rn(r2);
}

__device__ __forceinline__ uint32_t pack2(__nv_bfloat16 lo, __nv_bfloat16 hi) {
    return (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
}

// split3 of a pair (x0 in the low halves), with paired conversions: the parts
// as packed bf16 pairs h, m, l.
__device__ __forceinline__ void split3x2(float x0, float x1, uint32_t& h, uint32_t& m, uint32_t& l) {
    const __nv_bfloat162 hb = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(hb);
    const float2 r1 = __fadd2_rn(make_float2(x0, x1), make_float2(-hf.x, -hf.y));  // exact
    const __nv_bfloat162 mb = __floats2bfloat162_rn(r1.x, r1.y);
    const float2 mf = __bfloat1622float2(mb);
    const float2 r2 = __fadd2_rn(r1, make_float2(-mf.x, -mf.y));                    // exact
    const __nv_bfloat162 lb = __floats2bfloat162_rn(r2.x, r2.y);
    h = *reinterpret_cast<const uint32_t*>(&hb);
    m = *reinterpret_cast<const uint32_t*>(&mb);
    l = *reinterpret_cast<const uint32_t*>(&lb);
}

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Waits (bounded) until the phase of the given parity of an mbarrier has
// completed; false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t addr, uint32_t parity) {
    const unsigned long long t0 = global_ns();
    while (true) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(addr), "r"(parity)
            : "memory");
        if (done) return true;
        if (global_ns() - t0 > kWaitNs) return false;
    }
}

// The covariance's square root and exponential on the MUFU unit: sqrt.approx
// and ex2.approx (relative error of order 2^-22 each; exp(-a) = 2^(-a log2 e),
// the product's rounding adding a relative 2^-24 a), a few instructions fewer
// per covariance than the IEEE-rounded sqrtf and expf.  At a > 20, where the
// product's rounding weighs most, k < 4e-7 s_f^2.
constexpr float kLog2e = 1.4426950408889634f;
__device__ __forceinline__ float sqrt_hw(float x) {
    float y;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float ex2_hw(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// The Matérn polynomial factor at a = sqrt(2 nu) r: 1 + a (nu = 3/2) or
// 1 + a + a^2 / 3 (nu = 5/2).
__device__ __forceinline__ float matern_poly(float a, bool m32) {
    return m32 ? 1.0f + a : fmaf(a, fmaf(a, 0.33333333333333333f, 1.0f), 1.0f);
}

// B = L^{-1} of every objective, split into bf16 parts, per k-block of 32
// columns in the canonical layout: [M][n_pad / 32][3][n_pad rows x 64 bytes].
// One thread per (objective, k-block, row, group of 8 columns).
__device__ __forceinline__ float linv_at(const float* tiles, int n, int row, int c) {
    // tiles: row block rb, column chunk cj; tile[jj][ii] = L^{-1}[64 rb + ii][32 cj + jj]
    const int rb = row >> 6, ii = row & 63, cj = c >> 5, jj = c & 31;
    return (row < n && c <= row) ? tiles[((size_t)(rb * (rb + 1) + cj) * 32 + jj) * 64 + ii] : 0.0f;
}

__global__ void __launch_bounds__(256) bsplit_kernel(const float* tiles_all, int n_tiles, int n, int n_pad, int M,
                                                     uint8_t* out) {
    const int KB = n_pad / kKB;
    const size_t chunk = (size_t)n_pad * 64;
    const int64_t total = (int64_t)M * KB * n_pad * (kKB / 8);
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int kg = (int)(e % (kKB / 8));
        int64_t rest = e / (kKB / 8);
        const int row = (int)(rest % n_pad);
        rest /= n_pad;
        const int kb = (int)(rest % KB), m = (int)(rest / KB);
        const float* tiles = tiles_all + (size_t)m * n_tiles * 32 * 64;
        uint32_t w[kParts][4];
#pragma unroll
        for (int u = 0; u < 8; u += 2) {
            const int c = kb * kKB + kg * 8 + u;
            __nv_bfloat16 h0, m0, l0, h1, m1, l1;
            split3(linv_at(tiles, n, row, c), h0, m0, l0);
            split3(linv_at(tiles, n, row, c + 1), h1, m1, l1);
            w[0][u / 2] = pack2(h0, h1);
            w[1][u / 2] = pack2(m0, m1);
            w[2][u / 2] = pack2(l0, l1);
        }
        uint8_t* base = out + ((size_t)(m * KB + kb) * kParts) * chunk + canon_off(row, kg * 8);
#pragma unroll
        for (int p = 0; p < kParts; ++p)
            *reinterpret_cast<uint4*>(base + p * chunk) = make_uint4(w[p][0], w[p][1], w[p][2], w[p][3]);
    }
}

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count));
}

__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
}

// Waits (bounded) for use u of a barrier that completes one phase per use.
__device__ __forceinline__ bool mbar_wait_use(uint64_t* b, int64_t u) { return mbar_wait(smem_u32(b), (uint32_t)(u & 1)); }

// Barrier slots in shared memory.
enum { kAFull = 0, kMmaDone = 2, kBFull = 4, kDFree = 7, kRed = 8, kBars = 9 };

template <int DO>
__global__ void __launch_bounds__(kThr + 32, 1) posterior_tc_kernel(const __grid_constant__ ScootTcArgs a) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const int KB = a.n_pad / kKB;
    const uint32_t bchunk = (uint32_t)a.n_pad * 64;
    uint8_t* sA = smem;                                              // [2][3][8 KiB]
    uint8_t* sB = sA + 2 * kParts * kAPart;                          // [3][3][bchunk]
    const int npair = (a.n_obs + 1) / 2;
    float* xs = reinterpret_cast<float*>(sB + 3 * kParts * bchunk);  // [M][npair][DO][2] scaled observations
    float* al = xs + (size_t)a.n_obj * npair * DO * 2;               // [M][n_pad] alpha
    float* red = al + (size_t)a.n_obj * a.n_pad;                     // [2][kQt][kTM]: |V|^2 and mu quarters
    float* cat_s = red + 2 * kQt * kTM;                              // staged categorical table
    __shared__ float4 fm[kMaxD];
    __shared__ __align__(8) uint64_t bars[kBars];
    __shared__ uint32_t tslot;
    const int tid = threadIdx.x, warp = tid >> 5;
    const float4* gfmap = reinterpret_cast<const float4*>(a.state + a.off_fmap);
    const float* gxs = reinterpret_cast<const float*>(a.state + a.off_xs);
    const float* gils = reinterpret_cast<const float*>(a.state + a.off_ils);
    const float* galpha = reinterpret_cast<const float*>(a.state + a.off_alpha);
    const float* gscal = reinterpret_cast<const float*>(a.state + a.off_scal);
    const float* gcat = reinterpret_cast<const float*>(a.state + a.off_cat);
    if (tid < kMaxD) fm[tid] = tid < a.d ? gfmap[tid] : make_float4((float)SCOOT_CATEGORICAL, 0.f, 0.f, 0.f);
    for (int e = tid; e < a.cat_smem; e += blockDim.x) cat_s[e] = __ldg(gcat + e);
    // The observations' scaled ordinal coordinates and alpha, every objective,
    // once; coordinates interleaved by pairs of observations (2p, 2p + 1), so
    // one 16-byte load gives two coordinates of both (the last pair of an odd
    // count repeats its observation).
    for (int e = tid; e < a.n_obj * npair * DO * 2; e += blockDim.x) {
        const int s = e & 1, q = (e >> 1) % DO, mp = (e >> 1) / DO;
        const int m = mp / npair, j = min(2 * (mp - m * npair) + s, a.n_obs - 1);
        xs[e] = q < a.n_ord ? gxs[((size_t)m * a.n_obs + j) * a.d + q] : 0.0f;
    }
    for (int e = tid; e < a.n_obj * a.n_pad; e += blockDim.x) {
        const int m = e / a.n_pad, j = e - m * a.n_pad;
        al[e] = j < a.n_obs ? galpha[(size_t)m * a.n_obs + j] : 0.0f;
    }
    if (tid == 0) {
        mbar_init(&bars[kAFull], kThr);
        mbar_init(&bars[kAFull + 1], kThr);
        mbar_init(&bars[kMmaDone], 1);
        mbar_init(&bars[kMmaDone + 1], 1);
        for (int s = 0; s < 3; ++s) mbar_init(&bars[kBFull + s], 1);
        mbar_init(&bars[kDFree], kThr);
        mbar_init(&bars[kRed], kThr);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tslot)),
                     "r"((uint32_t)(2 * kMaxNpadTc)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tslot;
    const int M = a.n_obj, n_ord = a.n_ord;
    const int64_t n_work = a.list ? (int64_t)*a.n_list : a.n;
    const int64_t n_tiles = (n_work + kTM - 1) / kTM;
    const int64_t my_tiles = n_tiles > (int64_t)blockIdx.x ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    const int64_t total_g = my_tiles * M * KB;

    if (warp == kThr / 32) {
        // ---- control warp (one thread): B copies and the MMAs.
        if ((tid & 31) == 0) {
            // B of k-block g (objective (g / KB) mod M, k-block g mod KB) into slot g mod 3:
            // rows >= 32 kb only, one contiguous tail of each part.
            auto issue_b = [&](int64_t g) {
                const int kb = (int)(g % KB), m = (int)((g / KB) % M);
                const uint32_t skip = (uint32_t)(kKB * kb) * 64u, bytes = bchunk - skip;
                uint64_t* bar = &bars[kBFull + (int)(g % 3)];
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                             "r"(kParts * bytes)
                             : "memory");
                const uint8_t* src = a.bsplit + ((size_t)(m * KB + kb) * kParts) * bchunk + skip;
                const uint32_t dst = smem_u32(sB) + (uint32_t)(g % 3) * kParts * bchunk + skip;
                for (int p = 0; p < kParts; ++p)
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                            dst + (uint32_t)p * bchunk),
                        "l"(src + (size_t)p * bchunk), "r"(bytes), "r"(smem_u32(bar))
                        : "memory");
            };
            bool ok = true;
            if (total_g > 0) issue_b(0);
            for (int64_t g = 0; g < total_g && ok; ++g) {
                const int kb = (int)(g % KB);
                if (g + 1 < total_g) {
                    // slot (g + 1) mod 3 was last read by the MMAs of g - 2
                    if (g >= 2) ok &= mbar_wait_use(&bars[kMmaDone + (int)(g & 1)], (g - 2) >> 1);
                    if (ok) issue_b(g + 1);
                }
                ok = ok && mbar_wait_use(&bars[kBFull + (int)(g % 3)], g / 3);  // B of g has landed
                ok = ok && mbar_wait_use(&bars[kAFull + (int)(g & 1)], g >> 1);  // A of g is written
                if (kb == 0 && g > 0) ok = ok && mbar_wait_use(&bars[kDFree], g / KB - 1);  // D was read back
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t r0 = (uint32_t)(kKB * kb);
                const uint32_t a_base = smem_u32(sA) + (uint32_t)(g & 1) * kParts * kAPart;
                const uint32_t b_base = smem_u32(sB) + (uint32_t)(g % 3) * kParts * bchunk + r0 * 64u;
                const uint32_t idesc = instr_desc((uint32_t)a.n_pad - r0);
                // part products (A part, B part): h h into the main accumulator;
                // h m, m h, h l, l h, m m into the corrections
                const uint32_t pa = 0x120100u, pb = 0x102010u;  // nibble q = part of product q
#pragma unroll
                for (int s2 = 0; s2 < kKB / 16; ++s2)
#pragma unroll
                    for (int q = 0; q < 6; ++q) {
                        const uint64_t da = smem_desc(a_base + ((pa >> (4 * q)) & 0xFu) * kAPart + s2 * 256u);
                        const uint64_t db = smem_desc(b_base + ((pb >> (4 * q)) & 0xFu) * bchunk + s2 * 256u);
                        const uint32_t acc = (kb > 0 || s2 > 0 || q > 1) ? 1u : 0u;
                        const uint32_t dcol = tmem + (q == 0 ? 0u : (uint32_t)a.n_pad) + r0;
                        asm volatile(
                            "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(dcol),
                            "l"(da), "l"(db), "r"(idesc), "r"(acc));
                    }
                asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                                 smem_u32(&bars[kMmaDone + (int)(g & 1)]))
                             : "memory");
            }
            if (!ok) atomicOr(a.err, SCOOT_DEVERR_TIMEOUT);
        }
    } else {
        // ---- SIMT warps: thread t serves candidate row t mod 128 and column quarter t / 128.
        const int r = tid & (kTM - 1), qd = tid >> 7;
        int64_t g = 0, t_obj = 0;  // k-blocks and tile-objectives done
        bool ok = true;
        // The list entries are read one tile ahead and the next tile's pool
        // words prefetched into L2, so a tile starts on an L2 read, not on two
        // dependent HBM reads.
        auto index_at = [&](int64_t it2) -> int64_t {
            const int64_t p2 = (blockIdx.x + it2 * gridDim.x) * kTM + r;
            return (it2 < my_tiles && p2 < n_work) ? (a.list ? (int64_t)a.list[p2] : p2) : 0;
        };
        int64_t i_cur = index_at(0), i_nxt = index_at(1);
        for (int64_t it = 0; it < my_tiles && ok; ++it) {
            const int64_t tile = blockIdx.x + it * gridDim.x;
            const int64_t pos = tile * kTM + r;
            const bool live = pos < n_work;
            const int64_t i = i_cur;
            uint32_t wcur[kMaxD];
#pragma unroll
            for (int q = 0; q < kMaxD; ++q) wcur[q] = q < a.d ? __ldg(a.cand + (int64_t)fm[q].w * a.ld + i) : 0u;
            float u[DO];
#pragma unroll
            for (int q = 0; q < DO; ++q) {
                u[q] = 0.0f;
                if (q < n_ord && live) {
                    const float4 f = fm[q];
                    u[q] = feature_of(wcur[q], (int)f.x, f.y, f.z);
                }
            }
            int pid = 0;  // joint category pattern (mixed radix), out-of-range categories clamped and flagged
#pragma unroll
            for (int q = 0; q < kMaxD; ++q) {
                if (q < n_ord || q >= a.d || !live) continue;
                const float4 f = fm[q];
                const int nc = (int)f.y;
                int v = (int)wcur[q];
                if (v < 0 || v >= nc) {
                    if (qd == 0) atomicOr(a.err, SCOOT_DEVERR_INDEX);
                    v = v < 0 ? 0 : nc - 1;
                }
                pid += v * (int)f.z;
            }
            const int64_t i_nn = index_at(it + 2);
            if (qd == 0)
                for (int q = 0; q < a.d; ++q)
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(a.cand + (int64_t)fm[q].w * a.ld + i_nxt));
            for (int m = 0; m < M && ok; ++m) {
                const float* xsm = xs + (size_t)m * npair * DO * 2;
                const float* alm = al + (size_t)m * a.n_pad;
                const float sf2 = gscal[m * 4 + 0];
                const bool warped = gscal[m * 4 + 3] != 0.0f;
                const bool m32 = a.kernel == SCOOT_MATERN32;
                const float kc = m32 ? 1.7320508075688772f : 2.2360679774997896f;
                const float* catrow = (a.cat_smem ? cat_s : gcat) + (size_t)m * a.n_obs * a.n_pat + pid;
                float ut[DO];
#pragma unroll
                for (int q = 0; q < DO; ++q) {
                    float x = u[q];
                    if (warped && q < n_ord) {
                        const float2 ab = __ldg(reinterpret_cast<const float2*>(a.state + a.off_warp) + m * a.d + q);
                        x = kumaraswamy_cdf(x, ab.x, ab.y);
                    }
                    ut[q] = q < n_ord ? x * gils[m * a.d + q] : 0.0f;
                }
                float mu_part = 0.0f;
                // The categorical part of r^2 for this thread's 8 columns of the
                // k-block, loaded one k-block ahead (rows past n_obs clamped).
                float catv[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) catv[e] = catrow[(size_t)min(8 * qd + e, a.n_obs - 1) * a.n_pat];
                for (int kb = 0; kb < KB; ++kb, ++g) {
                    // This thread's 8 covariances: columns 32 kb + 8 qd + [0, 8).
                    const int c0 = kKB * kb + 8 * qd;
                    // Distances two columns at a time (packed fp32 pairs): d = u - x
                    // exactly (an FMA with -1), r^2 accumulated per float4 of coordinates.
                    // In stages over the 8 columns (distances, then square roots,
                    // then the kernel), so that their independent sqrt / exp
                    // chains overlap.
                    float r2v[8];
#pragma unroll
                    for (int e = 0; e < 8; e += 2) {
                        const int c = c0 + e;  // even
                        const float4* xp = reinterpret_cast<const float4*>(xsm + (size_t)min(c >> 1, npair - 1) * DO * 2);
                        float2 rp[DO / 4];
#pragma unroll
                        for (int q4 = 0; q4 < DO / 4; ++q4) {
                            const float4 v01 = xp[2 * q4], v23 = xp[2 * q4 + 1];  // coordinates 4 q4 .. 4 q4 + 3
                            const float2 d0 = __ffma2_rn(make_float2(v01.x, v01.y), make_float2(-1.f, -1.f),
                                                         make_float2(ut[4 * q4], ut[4 * q4]));
                            const float2 d1 = __ffma2_rn(make_float2(v01.z, v01.w), make_float2(-1.f, -1.f),
                                                         make_float2(ut[4 * q4 + 1], ut[4 * q4 + 1]));
                            const float2 d2 = __ffma2_rn(make_float2(v23.x, v23.y), make_float2(-1.f, -1.f),
                                                         make_float2(ut[4 * q4 + 2], ut[4 * q4 + 2]));
                            const float2 d3 = __ffma2_rn(make_float2(v23.z, v23.w), make_float2(-1.f, -1.f),
                                                         make_float2(ut[4 * q4 + 3], ut[4 * q4 + 3]));
                            rp[q4] = __ffma2_rn(d3, d3, __ffma2_rn(d2, d2, __ffma2_rn(d1, d1, __fmul2_rn(d0, d0))));
                        }
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            float r2 = catv[e + h];
#pragma unroll
                            for (int q4 = 0; q4 < DO / 4; ++q4) r2 += h ? rp[q4].y : rp[q4].x;
                            r2v[e + h] = r2;
                        }
                    }
                    float kv[8], ex[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) kv[e] = sqrt_hw(r2v[e]) * kc;  // a = sqrt(2 nu) r
#pragma unroll
                    for (int e = 0; e < 8; ++e) ex[e] = ex2_hw(kv[e] * -kLog2e);  // exp(-a)
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        kv[e] = (live && c0 + e < a.n_obs) ? sf2 * matern_poly(kv[e], m32) * ex[e] : 0.0f;
#pragma unroll
                    for (int e = 0; e < 8; ++e) mu_part = fmaf(kv[e], alm[c0 + e], mu_part);
                    if (kb + 1 < KB) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) catv[e] = catrow[(size_t)min(c0 + kKB + e, a.n_obs - 1) * a.n_pat];
                    }
                    // A slot g & 1 was last read by the MMAs of g - 2.
                    if (g >= 2 && !mbar_wait_use(&bars[kMmaDone + (int)(g & 1)], (g - 2) >> 1)) {
                        ok = false;
                        break;
                    }
                    uint8_t* adst = sA + (size_t)(g & 1) * kParts * kAPart;
                    {
                        uint32_t w[kParts][4];
#pragma unroll
                        for (int u2 = 0; u2 < 8; u2 += 2) split3x2(kv[u2], kv[u2 + 1], w[0][u2 / 2], w[1][u2 / 2], w[2][u2 / 2]);
                        const uint32_t off = canon_off(r, 8 * qd);
#pragma unroll
                        for (int p = 0; p < kParts; ++p)
                            *reinterpret_cast<uint4*>(adst + p * kAPart + off) = make_uint4(w[p][0], w[p][1], w[p][2], w[p][3]);
                    }
                    // visible to the tensor core (async proxy), then announced
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    mbar_arrive(&bars[kAFull + (int)(g & 1)]);
                }
                if (!ok) break;
                // Epilogue: the MMAs of the last k-block (g - 1) are done.
                if (!mbar_wait_use(&bars[kMmaDone + (int)((g - 1) & 1)], (g - 1) >> 1)) {
                    ok = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                float sq = 0.0f;
                float4* dst4 = reinterpret_cast<float4*>(a.vout);
                const int qw = a.n_pad / kQt;  // columns of this thread's quarter (a multiple of 16)
                for (int cc = qd * qw; cc < (qd + 1) * qw; cc += 16) {
                    uint32_t v[16], w[16];
                    const uint32_t taddr = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)cc;
                    asm volatile(
                        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
                        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
                          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]),
                          "=r"(v[15])
                        : "r"(taddr));
                    asm volatile(
                        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
                        : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7]),
                          "=r"(w[8]), "=r"(w[9]), "=r"(w[10]), "=r"(w[11]), "=r"(w[12]), "=r"(w[13]), "=r"(w[14]),
                          "=r"(w[15])
                        : "r"(taddr + (uint32_t)a.n_pad));
                    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                    float vf[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        vf[e] = __uint_as_float(v[e]) + __uint_as_float(w[e]);
                        sq = fmaf(vf[e], vf[e], sq);
                    }
                    if (live && a.vout) {
#pragma unroll
                        for (int g4 = 0; g4 < 4; ++g4) {
                            const int gi = (cc >> 2) + g4;  // float4 group of rows 4 gi .. 4 gi + 3
                            if (4 * gi < a.n_obs)
                                __stcs(dst4 + vtile_index(pos, m, gi, M, a.n_pad / 4),
                                       make_float4(vf[4 * g4], vf[4 * g4 + 1], vf[4 * g4 + 2], vf[4 * g4 + 3]));
                        }
                    }
                }
                // D may be overwritten by the next tile-objective's MMAs.
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                mbar_arrive(&bars[kDFree]);
                red[qd * kTM + r] = sq;
                red[(kQt + qd) * kTM + r] = mu_part;
                // Both halves' sums are in red (a bounded wait, not a hardware barrier, so
                // that a thread that gave up elsewhere cannot hold the others).
                mbar_arrive(&bars[kRed]);
                if (!mbar_wait_use(&bars[kRed], t_obj++)) {
                    ok = false;
                    break;
                }
                if (qd == 0 && live) {
                    const float* rs = red + r;
                    const float mean = (rs[4 * kTM] + rs[5 * kTM]) + (rs[6 * kTM] + rs[7 * kTM]);
                    const float var = fmaxf(sf2 - ((rs[0] + rs[kTM]) + (rs[2 * kTM] + rs[3 * kTM])), 0.0f);
                    if (a.acq_kind == 0) {
                        const int64_t o = (int64_t)m * a.ldo + (a.by_index ? i : pos);
                        a.mean[o] = mean;
                        a.var[o] = var;
                    } else {
                        const float ybest = gscal[2];
                        const float ei = ei_value(mean, var, ybest, a.xi);
                        if (a.acq_kind == 1) {
                            a.acq[i] = ei;
                        } else {
                            a.acq[i] = ucb_value(mean, var, a.kappa);
                            a.acq[a.lda + i] = pi_value(mean, var, ybest, a.xi);
                            a.acq[2 * a.lda + i] = ei;
                        }
                    }
                }
            }
            i_cur = i_nxt;
            i_nxt = i_nn;
        }
        if (!ok) atomicOr(a.err, SCOOT_DEVERR_TIMEOUT);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)(2 * kMaxNpadTc)));
}

size_t tc_smem(const ScootTcArgs& a, int DO) {
    return (size_t)2 * kParts * kAPart + (size_t)3 * kParts * a.n_pad * 64 + (size_t)a.n_obj * ((a.n_obs + 1) / 2) * DO * 8 +
           (size_t)a.n_obj * a.n_pad * 4 + (size_t)2 * kQt * kTM * 4 + (size_t)a.cat_smem * 4;
}

template <int DO>
scoot_status launch_tc(scoot_ctx* ctx, const ScootTcArgs& a, cudaStream_t st) {
    const size_t smem = tc_smem(a, DO);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(posterior_tc_kernel<DO>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    int sms = 0;
    SCOOT_CUDA(ctx, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, ctx->device));
    const int64_t tiles = (a.n + kTM - 1) / kTM;
    const int64_t blocks = std::max<int64_t>(1, std::min<int64_t>(tiles, sms));
    posterior_tc_kernel<DO><<<(unsigned)blocks, kThr + 32, smem, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

}  // namespace

int64_t scoot_tc_bsplit_bytes(int n_pad, int M) { return (int64_t)M * n_pad * n_pad * 2 * kParts; }

bool scoot_tc_supported(scoot_ctx* ctx, const ScootTcArgs& a, int DO) {
    if (a.n_pad < 64 || a.n_pad > kMaxNpadTc || a.n_pad % 64 != 0) return false;
    int optin = 0;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device) != cudaSuccess) return false;
    return tc_smem(a, DO) <= (size_t)optin;
}

scoot_status scoot_posterior_tc(scoot_ctx* ctx, const ScootTcArgs& a, int DO, cudaStream_t st) {
    if (a.n == 0) return SCOOT_OK;
    {
        const int KB = a.n_pad / kKB;
        const int64_t total = (int64_t)a.n_obj * KB * a.n_pad * (kKB / 8);
        int64_t blocks = (total + 255) / 256;
        if (blocks > 4096) blocks = 4096;
        bsplit_kernel<<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<const float*>(a.state + a.off_linv), a.n_tiles,
                                                       a.n_obs, a.n_pad, a.n_obj, a.bsplit);
        SCOOT_LAUNCHED(ctx);
    }
    switch (DO) {
    case 4: return launch_tc<4>(ctx, a, st);
    case 8: return launch_tc<8>(ctx, a, st);
    case 12: return launch_tc<12>(ctx, a, st);
    default: return launch_tc<16>(ctx, a, st);
    }
}
