// GP posterior (Section 4.3) and acquisition values: EI (Eq. 6) and
// Monte-Carlo EHVI over a box decomposition (Eq. 7), fused or separate.
//
// A block of 128 threads (four per candidate: warp w is quarter w of every
// candidate, lane l serves candidate slot l) owns a tile of 32 candidates.
// Per objective:
//  1. the four threads of a candidate evaluate its covariance row k(x, X)
//     against the n observations (staged in shared memory) into Ks[j][c],
//     splitting j by j mod 4, and accumulate mu = k . alpha;
//  2. the block computes V = L^{-1} Ks as a register-tiled SIMT product
//     (4 candidates x 4 rows per thread) over 32 x 64 tiles of L^{-1} that the
//     host laid out transposed and zero-filled; the tiles are double-buffered
//     in shared memory by cp.async, so the next tile streams in while the
//     current one is multiplied; sigma^2 = s_f^2 - sum_i V_ic^2, clamped at 0.
// The epilogue writes mu and sigma^2, or the EI, or the EHVI of the tile.
#include <cstring>

#include "device_common.cuh"
#include "internal.h"

namespace {

using namespace scoot_dev;

constexpr int kTC = 32;     // candidates per tile
constexpr int kThreads = 128;  // four threads per candidate
constexpr int kQ = kThreads / kTC;  // threads per candidate (= warps: warp w is quarter w)
constexpr int kRB = 64;     // rows of L^{-1} per tile
constexpr int kCJ = 32;     // columns of L^{-1} per host tile
constexpr int kCH = 16;     // columns of L^{-1} per staged half tile (4 KiB)
constexpr int kMaxD = SCOOT_MAX_DIM;
constexpr int kMaxM = SCOOT_MAX_OBJ;
constexpr int kAcqThreads = 128;

enum Epilogue { kWriteMoments = 0, kEI = 1, kEHVI = 2, kWriteWhitened = 3, kMACE = 4, kEHVIX = 5 };

struct ScoreArgs {
    const char* state;
    int64_t off_fmap, off_xs, off_ils, off_alpha, off_linv, off_scal, off_cat, off_warp;
    int32_t n_obs, d, dp, n_obj, kernel, n_rb, n_tiles, n_ord, n_pat;
    const uint32_t* cand;
    int64_t n, ld;
    const uint8_t* mask;
    float* mean;
    float* var;
    int64_t ldo;
    float* acq;
    int64_t lda;                  // kMACE: rows UCB, PI, EI of acq, lda apart
    float xi;
    float kappa;                  // kMACE: UCB coefficient
    const float* box_lo;
    const float* box_hi;
    int32_t n_boxes;
    const float* eps;
    int32_t n_mc;
    const float* grid;            // kEHVIX: per-axis box coordinates [M][grid_cap]
    const uint32_t* corner;       // kEHVIX: box corner indices [B][M]
    int32_t grid_cap;
    int32_t n_grid[kMaxM];
    int32_t psi_rows;             // kEHVIX: sum_j (n_grid[j] + 1), rows of the psi table
    const int32_t* list;          // live candidates (NULL: all of 0 .. n-1)
    const unsigned int* n_list;
    int32_t cat_smem;             // floats of the categorical table staged in shared memory (0: read from L1)
    int32_t cat_off;              // where, in floats from the start of shared memory
    int32_t wbuf_off;             // the next tile's pool words [d][kTC], in floats from the start
    float* vout;                  // kWriteWhitened: V = L^{-1} k* by list position, tiled (vtile_index)
    uint32_t* err;                // device error word
};

// Partial EHVI sum of one candidate over the sample chunks first, first +
// stride, ... (chunks of eight samples, padding samples at -inf); boxes as
// staged by stage_boxes.
template <int M>
__device__ __forceinline__ float ehvi_partial(const float* mu, const float* sd, const float4* blo, const float4* bhi,
                                             int n_boxes, const float4* eps, int n_mc, int first, int stride) {
    constexpr int kCh = 8;
    float total = 0.0f;
    for (int s0 = first * kCh; s0 < n_mc; s0 += stride * kCh) {
        float y[kCh][M], acc[kCh];
#pragma unroll
        for (int k = 0; k < kCh; ++k) {
            acc[k] = 0.0f;
            const bool in = s0 + k < n_mc;
            const float4 e = in ? eps[s0 + k] : make_float4(0.f, 0.f, 0.f, 0.f);
            const float ev[4] = {e.x, e.y, e.z, e.w};
#pragma unroll
            for (int j = 0; j < M; ++j) y[k][j] = in ? fmaf(sd[j], ev[j], mu[j]) : -INFINITY;
        }
        for (int b = 0; b < n_boxes; ++b) {
            const float4 lo4 = blo[b], hi4 = bhi[b];
            const float lo[4] = {lo4.x, lo4.y, lo4.z, lo4.w};
            const float hi[4] = {hi4.x, hi4.y, hi4.z, hi4.w};
#pragma unroll
            for (int k = 0; k < kCh; ++k) {
                float p = fmaxf(fminf(y[k][0], hi[0]) - lo[0], 0.0f);
#pragma unroll
                for (int j = 1; j < M; ++j) p *= fmaxf(fminf(y[k][j], hi[j]) - lo[j], 0.0f);
                acc[k] += p;
            }
        }
#pragma unroll
        for (int k = 0; k < kCh; ++k) total += acc[k];
    }
    return total;
}

// Asynchronous copy of one half of a 32 x 64 tile of L^{-1} (16 columns x 64
// rows, 4 KiB, contiguous in the host's transposed tile layout and 16-byte
// aligned at both ends) into shared memory: each of the 128 threads moves two
// 16-byte pieces with cp.async and commits them as one group.
__device__ __forceinline__ void stage_tile_async(float* dst, const float4* src, int tid) {
#pragma unroll
    for (int k = 0; k < kCH * kRB / 4 / kThreads; ++k) {
        const unsigned s = (unsigned)__cvta_generic_to_shared(dst + 4 * (tid + k * kThreads));
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(src + tid + k * kThreads) : "memory");
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}

// Gathers the d words of the candidates of a tile into wbuf[q][slot] (feature
// order) with 4-byte cp.async, four threads per candidate, one group.
__device__ __forceinline__ void prefetch_words(uint32_t* wbuf, const uint32_t* cand, int64_t ld, const int32_t* list,
                                               const float4* fm, int d, int64_t tile, int64_t n_tiles,
                                               int64_t n_work, int tid) {
    const int s = tid & (kTC - 1);
    const int64_t p = tile * kTC + s;
    if (tile < n_tiles && p < n_work) {
        const int64_t i = list ? (int64_t)list[p] : p;
        for (int q = tid / kTC; q < d; q += kQ) {
            const unsigned dst = (unsigned)__cvta_generic_to_shared(wbuf + q * kTC + s);
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst),
                         "l"(cand + (int64_t)fm[q].w * ld + i) : "memory");
        }
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}

// Waits until every cp.async group this thread committed has landed.
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// One block of 128 threads scores a tile of 32 candidates; thread t works on
// candidate slot t % 32 as quarter t / 32 (its warp) of that candidate:
//  1. the quarters compute the candidate's features; for each objective they
//     split the covariance row k(x, X_j) (j mod 4) into Ks[j][slot] and the
//     partial sums of mu = k . alpha;
//  2. all 128 threads compute V = L^{-1} Ks over 32 x 64 tiles of L^{-1} with a
//     4-candidate x 4-row register tile each; a warp whose 16 rows lie wholly
//     above a tile's columns (upper triangle, all zero) skips that tile;
//     sigma^2 = s_f^2 - sum_i V_i^2;
//  3. the epilogue (EI on one quarter, EHVI or exact EHVI with the quarters
//     splitting the sample chunks or boxes, or the moments / whitened rows)
//     writes the tile.
// Features come in feature order (ordinal parameters first).  DO >= n_ord
// bounds the ordinal register arrays; padded ordinal dimensions are zero on
// both sides and add nothing, so the distance loop has no per-dimension
// branch.  The categorical part of r^2 depends only on the candidate's joint
// category pattern and is read from the host-built table (one load).
template <int EPI, int M, int DO>
__global__ void __launch_bounds__(kThreads, (EPI == kEHVI && M == 2 && DO == 8) ? 6 : 4)
score_kernel(const __grid_constant__ ScoreArgs a) {
    // At least four blocks (16 warps) per SM: registers capped at 128 (80 for
    // the 2-objective EHVI of <= 8 parameters, six blocks).  L^{-1} is staged
    // in half tiles of 16 columns, double-buffered: 8 KiB in all.
    constexpr bool kRegCapped = EPI == kEHVI && M == 2 && DO == 8;
    extern __shared__ __align__(16) float sm[];
    const int n_pad = a.n_rb * kRB;
    // Ks, and after the posterior the exact-EHVI psi table [psi_rows][kTC]
    const int ks_rows = EPI == kEHVIX && a.psi_rows > n_pad ? a.psi_rows : n_pad;
    float* Ks = sm;                                                   // [n_pad][kTC]
    float* xs = Ks + (size_t)ks_rows * kTC;                           // [n_obs][DO] ordinal features
    float* al = xs + (size_t)a.n_obs * DO;                            // [n_pad]
    float* Lt = al + n_pad;                                           // [2][kCH][kRB] double buffer
    float* part = Lt + 2 * kCH * kRB;                                 // [16][kTC]
    float4* fm = reinterpret_cast<float4*>(part + 16 * kTC);          // [kMaxD] feature map
    float4* blo = fm + kMaxD;                          // [B] (general boxes) or [2B] (saturated form)
    float4* bhi = blo + (EPI == kEHVI ? a.n_boxes : 0);
    float4* epsv = bhi + (EPI == kEHVI ? a.n_boxes : 0);
    float* grid_s = reinterpret_cast<float*>(fm + kMaxD);             // kEHVIX: [sum n_grid] (padded to 4)
    uint32_t* corner_s = reinterpret_cast<uint32_t*>(grid_s + ((a.psi_rows + 3) & ~3));  // [B][M]

    const int tid = threadIdx.x;
    const int slot = tid & (kTC - 1), qtr = tid / kTC;
    const int warp = tid >> 5;
    const int nobj = (EPI == kEHVI || EPI == kEHVIX) ? M : ((EPI == kEI || EPI == kMACE) ? 1 : a.n_obj);
    const int64_t n_pad64 = n_pad;
    const float4* gfmap = reinterpret_cast<const float4*>(a.state + a.off_fmap);
    const float* gxs = reinterpret_cast<const float*>(a.state + a.off_xs);
    const float* gils = reinterpret_cast<const float*>(a.state + a.off_ils);
    const float* galpha = reinterpret_cast<const float*>(a.state + a.off_alpha);
    const float4* glinv = reinterpret_cast<const float4*>(a.state + a.off_linv);
    const float* gscal = reinterpret_cast<const float*>(a.state + a.off_scal);
    const float* gcat = reinterpret_cast<const float*>(a.state + a.off_cat);

    // The categorical part of r^2 for every objective, observation and
    // pattern, when small: one shared-memory load per pair instead of L1.
    float* cat_s = sm + a.cat_off;
    for (int e = tid; e < a.cat_smem; e += kThreads) cat_s[e] = __ldg(gcat + e);
    if (EPI == kEHVI) stage_boxes(a.box_lo, a.box_hi, a.n_boxes, a.eps, a.n_mc, M, blo, bhi, epsv);
    if (EPI == kEHVIX) stage_box_grid(a.grid, a.grid_cap, a.n_grid, a.corner, a.n_boxes, M, grid_s, corner_s, a.err);
    if (tid < kMaxD) fm[tid] = tid < a.d ? gfmap[tid] : make_float4((float)SCOOT_CATEGORICAL, 0.f, 0.f, 0.f);
    __syncthreads();
    // Boxes open on the last objective (as scoot_boxes_build makes them) are
    // restaged in saturated form over the same storage (2 float4 per box).
    const bool fast = EPI == kEHVI ? boxes_fast(blo, bhi, a.n_boxes, M) : false;
    if (EPI == kEHVI && fast) {
        stage_boxes_sat(a.box_lo, a.box_hi, a.n_boxes, M, blo);
        __syncthreads();
    }
    const int n_ord = a.n_ord;

    const int64_t n_work = a.list ? (int64_t)*a.n_list : a.n;
    const int64_t n_tiles = (n_work + kTC - 1) / kTC;
    // The next tile's pool words stream into wbuf while this tile is scored.
    uint32_t* wbuf = reinterpret_cast<uint32_t*>(sm + a.wbuf_off);  // [d][kTC]
    prefetch_words(wbuf, a.cand, a.ld, a.list, fm, a.d, blockIdx.x, n_tiles, n_work, tid);
    for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int64_t pos = tile * kTC + slot;
        const bool live = pos < n_work;
        const int64_t i = live ? (a.list ? (int64_t)a.list[pos] : pos) : 0;
        cp_async_wait_all();
        __syncthreads();  // this tile's words are in wbuf
        float u[DO];
#pragma unroll
        for (int q = 0; q < DO; ++q) {
            u[q] = 0.0f;
            if (q < n_ord && live) {
                const float4 f = fm[q];
                u[q] = feature_of(wbuf[q * kTC + slot], (int)f.x, f.y, f.z);
            }
        }
        // Joint category pattern (mixed radix); out-of-range categories are
        // clamped and flagged.
        int pid = 0;
        for (int q = n_ord; q < a.d && live; ++q) {
            const float4 f = fm[q];
            const int nc = (int)f.y;
            int v = (int)wbuf[q * kTC + slot];
            if (v < 0 || v >= nc) {
                atomicOr(a.err, SCOOT_DEVERR_INDEX);
                v = v < 0 ? 0 : nc - 1;
            }
            pid += v * (int)f.z;
        }
        __syncthreads();  // every thread has read its words
        prefetch_words(wbuf, a.cand, a.ld, a.list, fm, a.d, tile + gridDim.x, n_tiles, n_work, tid);
        float mu[kMaxM], vr[kMaxM];
        for (int m = 0; m < nobj; ++m) {
            __syncthreads();  // previous users of xs / al / part / Lt are done
            const float4* tiles = glinv + (size_t)m * a.n_tiles * (kCJ * kRB / 4);
            stage_tile_async(Lt, tiles, tid);  // half tile 0 lands while the covariance row is computed
            const float* sx = gxs + (size_t)m * a.n_obs * a.d;
            for (int e = tid; e < a.n_obs * DO; e += kThreads) {
                const int j = e / DO, q = e - j * DO;
                xs[e] = q < n_ord ? sx[j * a.d + q] : 0.0f;
            }
            for (int j = tid; j < n_pad; j += kThreads) al[j] = j < a.n_obs ? galpha[(size_t)m * a.n_obs + j] : 0.0f;
            const float sf2 = gscal[m * 4 + 0];
            // this candidate's column of the categorical table: shared memory when
            // staged, else global (one generic pointer either way)
            const float* catrow = (a.cat_smem ? cat_s : gcat) + (size_t)m * a.n_obs * a.n_pat + pid;
            float ut[DO];
            const bool warped = gscal[m * 4 + 3] != 0.0f;  // the same in every thread
#pragma unroll
            for (int q = 0; q < DO; ++q) {
                float x = u[q];
                if (warped && q < n_ord) {
                    const float2 ab = __ldg(reinterpret_cast<const float2*>(a.state + a.off_warp) + m * a.d + q);
                    x = kumaraswamy_cdf(x, ab.x, ab.y);
                }
                ut[q] = q < n_ord ? x * gils[m * a.d + q] : 0.0f;
            }
            __syncthreads();
            // 1. covariance row (this quarter's j) and the partial mean.
            float acc = 0.0f;
#pragma unroll 2
            for (int j = qtr; j < a.n_obs; j += kQ) {
                const float4* xj4 = reinterpret_cast<const float4*>(xs + j * DO);
                float r2 = catrow[(size_t)j * a.n_pat];  // categorical part
#pragma unroll
                for (int q4 = 0; q4 < DO / 4; ++q4) {
                    const float4 v = xj4[q4];
                    const float t0 = ut[q4 * 4] - v.x, t1 = ut[q4 * 4 + 1] - v.y;
                    const float t2 = ut[q4 * 4 + 2] - v.z, t3 = ut[q4 * 4 + 3] - v.w;
                    r2 = fmaf(t0, t0, r2);
                    r2 = fmaf(t1, t1, r2);
                    r2 = fmaf(t2, t2, r2);
                    r2 = fmaf(t3, t3, r2);
                }
                const float k = sf2 * matern(sqrtf(r2), a.kernel);
                Ks[j * kTC + slot] = k;
                acc = fmaf(k, al[j], acc);
            }
            for (int j = a.n_obs + qtr; j < n_pad; j += kQ) Ks[j * kTC + slot] = 0.0f;
            part[qtr * kTC + slot] = acc;
            __syncthreads();
            mu[m] = (part[slot] + part[kTC + slot]) + (part[2 * kTC + slot] + part[3 * kTC + slot]);
            // 2. V = L^{-1} Ks and the sum of squares per candidate: thread
            // (cg, rg) holds candidates 4 cg .. 4 cg + 3 and rows 4 rg .. 4 rg + 3
            // of each 64-row block; a warp's rows are 16 consecutive ones.
            const int cg = tid & 7, rg = tid >> 3;
            float sq[4] = {0.f, 0.f, 0.f, 0.f};
            const float4* Ks4 = reinterpret_cast<const float4*>(Ks);
            int t = 0;
            for (int rb = 0; rb < a.n_rb; ++rb) {
                // accumulators in column pairs: acc2[r][cp] = (V[r][2 cp], V[r][2 cp + 1]),
                // updated by packed fp32 FMAs (two per instruction, each lane
                // rounded as fmaf): the k loads give the candidate pairs, the
                // row's L^{-1} value is broadcast to both lanes.
                float2 acc2[4][2];
#pragma unroll
                for (int r = 0; r < 4; ++r) acc2[r][0] = acc2[r][1] = make_float2(0.0f, 0.0f);
                for (int ch = 0; ch < 4 * (rb + 1); ++ch, ++t) {
                    // Half tile t (columns 16 ch .. 16 ch + 15 of this row
                    // block's tiles) has landed in buffer t&1 and every thread
                    // is done with half tile t-1, so half tile t+1 may
                    // overwrite buffer (t+1)&1 while t is multiplied.
                    cp_async_wait_all();
                    __syncthreads();
                    if (t + 1 < 2 * a.n_tiles)
                        stage_tile_async(Lt + ((t + 1) & 1) * (kCH * kRB), tiles + (size_t)(t + 1) * (kCH * kRB / 4), tid);
                    const float4* Lt4 = reinterpret_cast<const float4*>(Lt + (t & 1) * (kCH * kRB));
                    // rows of this warp: rb*64 + 16*warp .. +15; columns ch*16 .. +15;
                    // L^{-1} is zero right of the diagonal, so a warp stops at its
                    // last row.
                    const int j0 = ch * kCH;
                    const int last_row = rb * kRB + 16 * warp + 15;
                    if (j0 > last_row) continue;
#pragma unroll 8
                    for (int jj = 0; jj < kCH; ++jj) {
                        const float4 k4 = Ks4[(j0 + jj) * (kTC / 4) + cg];
                        const float4 l4 = Lt4[jj * (kRB / 4) + rg];
                        const float2 k01 = make_float2(k4.x, k4.y), k23 = make_float2(k4.z, k4.w);
                        const float lv[4] = {l4.x, l4.y, l4.z, l4.w};
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            if (kRegCapped) {  // scalar FMAs in the register-capped variant
                                acc2[r][0].x = fmaf(lv[r], k4.x, acc2[r][0].x);
                                acc2[r][0].y = fmaf(lv[r], k4.y, acc2[r][0].y);
                                acc2[r][1].x = fmaf(lv[r], k4.z, acc2[r][1].x);
                                acc2[r][1].y = fmaf(lv[r], k4.w, acc2[r][1].y);
                            } else {
                                const float2 lb = make_float2(lv[r], lv[r]);
                                acc2[r][0] = __ffma2_rn(lb, k01, acc2[r][0]);
                                acc2[r][1] = __ffma2_rn(lb, k23, acc2[r][1]);
                            }
                        }
                    }
                }
                float accm[4][4];
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    accm[r][0] = acc2[r][0].x;
                    accm[r][1] = acc2[r][0].y;
                    accm[r][2] = acc2[r][1].x;
                    accm[r][3] = acc2[r][1].y;
                }
#pragma unroll
                for (int r = 0; r < 4; ++r)
#pragma unroll
                    for (int c = 0; c < 4; ++c) sq[c] = fmaf(accm[r][c], accm[r][c], sq[c]);
                if (EPI == kWriteWhitened) {
                    // Rows of V for the fantasy downdates, indexed by list
                    // position, in float4 groups of four rows (this thread's
                    // rows are one group), tiled by 32 candidates
                    // (vtile_index).  Rows past n_obs hold zeros (L^{-1} is
                    // zero-filled there).
                    float4* dst4 = reinterpret_cast<float4*>(a.vout);
                    const int g = rb * (kRB / 4) + rg;
                    if (4 * g < a.n_obs) {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const int64_t p = tile * kTC + cg * 4 + c;
                            if (p < n_work)
                                dst4[vtile_index(p, m, g, a.n_obj, (int)(n_pad64 / 4))] =
                                    make_float4(accm[0][c], accm[1][c], accm[2][c], accm[3][c]);
                        }
                    }
                }
            }
            __syncthreads();  // every thread has read its mean quarters from part
#pragma unroll
            for (int c = 0; c < 4; ++c) part[rg * kTC + cg * 4 + c] = sq[c];
            __syncthreads();
            float ss = 0.0f;
#pragma unroll
            for (int g = 0; g < kRB / 4; ++g) ss += part[g * kTC + slot];
            vr[m] = fmaxf(sf2 - ss, 0.0f);
        }
        // 3. epilogue.
        if (EPI == kWriteMoments) {
            if (live && qtr == 0)
                for (int m = 0; m < nobj; ++m) {
                    a.mean[(int64_t)m * a.ldo + i] = mu[m];
                    a.var[(int64_t)m * a.ldo + i] = vr[m];
                }
        } else if (EPI == kWriteWhitened) {
            if (live && qtr == 0)
                for (int m = 0; m < nobj; ++m) {
                    a.mean[(int64_t)m * a.ldo + pos] = mu[m];
                    a.var[(int64_t)m * a.ldo + pos] = vr[m];
                }
        } else if (EPI == kEI) {
            if (live && qtr == 0) a.acq[i] = ei_value(mu[0], vr[0], gscal[2], a.xi);
        } else if (EPI == kEHVIX) {
            // psi table: row poff_j + g holds psi_j(grid_j[g]) (the row past
            // the last grid coordinate, +inf, holds 0).  Every thread read its
            // last Ks value before the barriers that ended the posterior.
            float sd[kMaxM];
#pragma unroll
            for (int m = 0; m < M; ++m) sd[m] = sqrtf(vr[m]);
            int goff = 0, poff = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                for (int g = qtr; g < a.n_grid[m]; g += kQ)
                    Ks[(poff + g) * kTC + slot] = expected_excess(mu[m], sd[m], grid_s[goff + g]);
                if (qtr == 0) Ks[(poff + a.n_grid[m]) * kTC + slot] = 0.0f;
                goff += a.n_grid[m];
                poff += a.n_grid[m] + 1;
            }
            __syncthreads();
            float v = 0.0f;
            for (int b = qtr; b < a.n_boxes; b += kQ) {
                float p = 1.0f;
                int po = 0;
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    const uint32_t c = corner_s[b * M + m];
                    p *= Ks[(po + (int)(c & 0xFFFFu)) * kTC + slot] - Ks[(po + (int)(c >> 16)) * kTC + slot];
                    po += a.n_grid[m] + 1;
                }
                v += p;
            }
            __syncthreads();  // part is free again; the psi table is read
            part[qtr * kTC + slot] = v;
            __syncthreads();
            if (live && qtr == 0) a.acq[i] = (part[slot] + part[kTC + slot]) + (part[2 * kTC + slot] + part[3 * kTC + slot]);
        } else if (EPI == kMACE) {
            if (live && qtr == 0) {
                a.acq[i] = ucb_value(mu[0], vr[0], a.kappa);
                a.acq[a.lda + i] = pi_value(mu[0], vr[0], gscal[2], a.xi);
                a.acq[2 * a.lda + i] = ei_value(mu[0], vr[0], gscal[2], a.xi);
            }
        } else {
            float sd[kMaxM];
#pragma unroll
            for (int m = 0; m < M; ++m) sd[m] = sqrtf(vr[m]);
            float v;
            if constexpr (M >= 2 && M <= 3)  // (the saturated form takes two or three objectives)
                v = fast ? ehvi_partial_sat<M>(mu, sd, blo, a.n_boxes, epsv, a.n_mc, qtr, kQ)
                         : ehvi_partial<M>(mu, sd, blo, bhi, a.n_boxes, epsv, a.n_mc, qtr, kQ);
            else
                v = ehvi_partial<M>(mu, sd, blo, bhi, a.n_boxes, epsv, a.n_mc, qtr, kQ);
            __syncthreads();  // part is free again
            part[qtr * kTC + slot] = v;
            __syncthreads();
            if (live && qtr == 0)
                a.acq[i] = ((part[slot] + part[kTC + slot]) + (part[2 * kTC + slot] + part[3 * kTC + slot])) *
                           (1.0f / (float)a.n_mc);
        }
    }
}

__global__ void __launch_bounds__(kAcqThreads)
mace_kernel(const float* __restrict__ mean, const float* __restrict__ var, const uint8_t* __restrict__ mask,
            int64_t n, float ybest, float xi, float kappa, float* __restrict__ acq, int64_t lda) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const bool live = mask == nullptr || mask[i] != 0;
        const float mu = live ? mean[i] : 0.0f, vr = live ? var[i] : 0.0f;
        acq[i] = live ? ucb_value(mu, vr, kappa) : -INFINITY;
        acq[lda + i] = live ? pi_value(mu, vr, ybest, xi) : -INFINITY;
        acq[2 * lda + i] = live ? ei_value(mu, vr, ybest, xi) : -INFINITY;
    }
}

__global__ void __launch_bounds__(kAcqThreads)
ei_kernel(const float* __restrict__ mean, const float* __restrict__ var, const uint8_t* __restrict__ mask,
          int64_t n, float ybest, float xi, float* __restrict__ acq) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const bool live = mask == nullptr || mask[i] != 0;
        acq[i] = live ? ei_value(mean[i], var[i], ybest, xi) : -INFINITY;
    }
}

template <int M>
__global__ void __launch_bounds__(kAcqThreads)
ehvi_kernel(const __grid_constant__ ScoreArgs a) {
    extern __shared__ __align__(16) float sm[];
    float4* blo = reinterpret_cast<float4*>(sm);
    float4* bhi = blo + a.n_boxes;
    float4* epsv = bhi + a.n_boxes;
    stage_boxes(a.box_lo, a.box_hi, a.n_boxes, a.eps, a.n_mc, M, blo, bhi, epsv);
    __syncthreads();
    const int64_t n_work = a.list ? (int64_t)*a.n_list : a.n;
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; pos < n_work;
         pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
        float mu[kMaxM], sd[kMaxM];
#pragma unroll
        for (int m = 0; m < M; ++m) {
            mu[m] = a.mean[(int64_t)m * a.ldo + i];
            sd[m] = sqrtf(fmaxf(a.var[(int64_t)m * a.ldo + i], 0.0f));
        }
        a.acq[i] = ehvi_value<M>(mu, sd, blo, bhi, a.n_boxes, epsv, a.n_mc);
    }
}

// Exact EHVI on given moments: one thread per candidate with its own column
// of the psi table in shared memory.
template <int M>
__global__ void __launch_bounds__(kAcqThreads)
ehvix_kernel(const __grid_constant__ ScoreArgs a) {
    extern __shared__ __align__(16) float sm[];
    float* psi = sm;                                                    // [psi_rows][kAcqThreads]
    float* grid_s = psi + (size_t)a.psi_rows * kAcqThreads;
    uint32_t* corner_s = reinterpret_cast<uint32_t*>(grid_s + ((a.psi_rows + 3) & ~3));
    stage_box_grid(a.grid, a.grid_cap, a.n_grid, a.corner, a.n_boxes, M, grid_s, corner_s, a.err);
    __syncthreads();
    const int t = threadIdx.x;
    const int64_t n_work = a.list ? (int64_t)*a.n_list : a.n;
    for (int64_t pos = (int64_t)blockIdx.x * blockDim.x + t; pos < n_work; pos += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = a.list ? (int64_t)a.list[pos] : pos;
        int goff = 0, poff = 0;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const float mu = a.mean[(int64_t)m * a.ldo + i];
            const float sd = sqrtf(fmaxf(a.var[(int64_t)m * a.ldo + i], 0.0f));
            for (int g = 0; g < a.n_grid[m]; ++g)
                psi[(poff + g) * kAcqThreads + t] = expected_excess(mu, sd, grid_s[goff + g]);
            psi[(poff + a.n_grid[m]) * kAcqThreads + t] = 0.0f;
            goff += a.n_grid[m];
            poff += a.n_grid[m] + 1;
        }
        float v = 0.0f;
        for (int b = 0; b < a.n_boxes; ++b) {
            float p = 1.0f;
            int po = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const uint32_t c = corner_s[b * M + m];
                p *= psi[(po + (int)(c & 0xFFFFu)) * kAcqThreads + t] - psi[(po + (int)(c >> 16)) * kAcqThreads + t];
                po += a.n_grid[m] + 1;
            }
            v += p;
        }
        a.acq[i] = v;
    }
}

int sm_count(int device) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device);
    return v > 0 ? v : 1;
}

// Arguments of the exact-EHVI calls: the box grid and the psi-table height.
scoot_status fill_box_grid(scoot_ctx* ctx, int M, const float* grid, int32_t grid_cap, const int32_t* h_n_grid,
                           const uint32_t* corner, int32_t n_boxes, ScoreArgs& a) {
    if (M < 2 || M > kMaxM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "EHVI needs 2 <= M <= %d objectives, got %d", kMaxM, M);
    if (n_boxes < 1 || !corner || !h_n_grid || !grid)
        return scoot_fail(ctx, SCOOT_EINVAL, "boxes: B = %d, grid / n_grid / corner must be non-NULL", n_boxes);
    int rows = 0;
    for (int j = 0; j < M; ++j) {
        if (h_n_grid[j] < 0 || h_n_grid[j] > grid_cap || h_n_grid[j] > 65535)
            return scoot_fail(ctx, SCOOT_EINVAL, "n_grid[%d] = %d outside 0..min(grid_cap, 65535)", j, h_n_grid[j]);
        a.n_grid[j] = h_n_grid[j];
        rows += h_n_grid[j] + 1;
    }
    if (rows > 320) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "%d grid rows exceed the psi table (320)", rows);
    if ((size_t)n_boxes * M * 4 > 64 * 1024)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "%d boxes exceed the shared-memory budget", n_boxes);
    a.grid = grid;
    a.grid_cap = grid_cap;
    a.corner = corner;
    a.n_boxes = n_boxes;
    a.psi_rows = rows;
    return SCOOT_OK;
}

scoot_status fill_state_args(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state, ScoreArgs& a) {
    if (!L || !state) return scoot_fail(ctx, SCOOT_EINVAL, "layout or state is NULL");
    if (!scoot_gp_layout_valid(L))
        return scoot_fail(ctx, SCOOT_EINVAL, "GP layout is not one made by scoot_gp_layout_init");
    if (!scoot_aligned16(state)) return scoot_fail(ctx, SCOOT_EINVAL, "state blob is not 16-byte aligned");
    std::memset(&a, 0, sizeof(a));
    a.state = static_cast<const char*>(state);
    a.off_fmap = L->off_fmap;
    a.off_xs = L->off_xs;
    a.off_ils = L->off_ils;
    a.off_alpha = L->off_alpha;
    a.off_linv = L->off_linv;
    a.off_scal = L->off_scal;
    a.off_cat = L->off_cat;
    a.off_warp = L->off_warp;
    a.n_ord = L->n_ord;
    a.n_pat = L->n_pat;
    a.n_obs = L->n;
    a.d = L->d;
    a.dp = (L->d + 3) & ~3;
    a.n_obj = L->n_obj;
    a.kernel = L->kernel;
    a.n_rb = L->n_rb;
    a.n_tiles = L->n_tiles;
    return SCOOT_OK;
}

constexpr int kCatSmemMax = 1024;  // floats of categorical table worth staging per block

size_t score_smem(const ScoreArgs& a, int epi, int DO) {
    const size_t n_pad = (size_t)a.n_rb * kRB;
    const size_t ks_rows = epi == kEHVIX && (size_t)a.psi_rows > n_pad ? (size_t)a.psi_rows : n_pad;
    size_t f = ks_rows * kTC + (size_t)a.n_obs * DO + n_pad + 2 * kCH * kRB + 16 * kTC + 4 * kMaxD;
    if (epi == kEHVI) f += (size_t)(2 * a.n_boxes + a.n_mc) * 4;
    if (epi == kEHVIX) f += (size_t)((a.psi_rows + 3) & ~3) + (size_t)a.n_boxes * kMaxM;
    return f * 4;
}

template <int EPI, int M, int DO>
scoot_status launch_score_dm(scoot_ctx* ctx, ScoreArgs a, cudaStream_t st) {
    // the categorical table of the objectives this epilogue reads, staged when small
    const int nobj = (EPI == kEHVI || EPI == kEHVIX) ? M : ((EPI == kEI || EPI == kMACE) ? 1 : a.n_obj);
    const int64_t cat = (int64_t)nobj * a.n_obs * a.n_pat;
    auto kern = score_kernel<EPI, M, DO>;
    int optin = 0;
    SCOOT_CUDA(ctx, cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device));
    a.cat_off = (int32_t)(score_smem(a, EPI, DO) / 4);
    a.cat_smem = (a.n_ord < a.d && cat <= kCatSmemMax) ? (int32_t)cat : 0;
    a.wbuf_off = a.cat_off + ((a.cat_smem + 3) & ~3);
    const size_t smem = (size_t)(a.wbuf_off + a.d * kTC) * 4;
    if (smem > (size_t)optin)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED,
                          "score kernel needs %zu bytes of shared memory (n = %d observations, %d boxes), the "
                          "device allows %d", smem, a.n_obs, a.n_boxes, optin);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    int per_sm = 0;
    SCOOT_CUDA(ctx, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem));
    if (per_sm < 1) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "score kernel needs %zu bytes of shared memory", smem);
    const int64_t tiles = (a.n + kTC - 1) / kTC;
    int64_t blocks = (int64_t)sm_count(ctx->device) * per_sm;
    if (blocks > tiles) blocks = tiles;
    kern<<<(unsigned)blocks, kThreads, smem, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

template <int EPI, int M>
scoot_status launch_score(scoot_ctx* ctx, ScoreArgs a, cudaStream_t st) {
    if (a.mask) {
        // Score only the candidates still in play; the acquisition of the
        // others is -inf (their moments are left untouched).
        ScootList lst;
        scoot_status s = scoot_compact(ctx, a.mask, a.n, EPI == kWriteMoments ? nullptr : reinterpret_cast<uint32_t*>(a.acq),
                                       0xFF800000u, st, &lst, EPI == kMACE ? 3 : 1, a.lda);
        if (s != SCOOT_OK) return s;
        a.list = lst.list;
        a.n_list = lst.count;
    }
    a.err = ctx->d_err;
    if (a.n_ord <= 4) return launch_score_dm<EPI, M, 4>(ctx, a, st);
    if (a.n_ord <= 8) return launch_score_dm<EPI, M, 8>(ctx, a, st);
    if (a.n_ord <= 12) return launch_score_dm<EPI, M, 12>(ctx, a, st);
    return launch_score_dm<EPI, M, 16>(ctx, a, st);
}

scoot_status check_boxes(scoot_ctx* ctx, int M, const float* lo, const float* hi, int32_t B, const float* eps, int32_t S) {
    if (M < 2 || M > kMaxM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "EHVI needs 2 <= M <= %d objectives, got %d", kMaxM, M);
    if (B < 1 || !lo || !hi) return scoot_fail(ctx, SCOOT_EINVAL, "boxes: B = %d, lo/hi must be non-NULL", B);
    if (S < 1 || !eps) return scoot_fail(ctx, SCOOT_EINVAL, "base samples: S = %d, eps must be non-NULL", S);
    if ((size_t)(2 * B + S) * 16 > 160 * 1024)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "%d boxes and %d samples exceed the shared-memory budget", B, S);
    return SCOOT_OK;
}

template <int EPI>
scoot_status dispatch_m(scoot_ctx* ctx, const ScoreArgs& a, int M, cudaStream_t st) {
    switch (M) {
    case 2: return launch_score<EPI, 2>(ctx, a, st);
    case 3: return launch_score<EPI, 3>(ctx, a, st);
    case 4: return launch_score<EPI, 4>(ctx, a, st);
    default: return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "M = %d", M);
    }
}

// The state part of the tensor-core posterior's arguments, for the first
// nobj objectives.
ScootTcArgs tc_args(scoot_ctx* ctx, const ScoreArgs& a, int nobj) {
    ScootTcArgs t;
    std::memset(&t, 0, sizeof(t));
    t.state = a.state;
    t.off_fmap = a.off_fmap;
    t.off_xs = a.off_xs;
    t.off_ils = a.off_ils;
    t.off_alpha = a.off_alpha;
    t.off_scal = a.off_scal;
    t.off_cat = a.off_cat;
    t.off_warp = a.off_warp;
    t.off_linv = a.off_linv;
    t.n_obs = a.n_obs;
    t.d = a.d;
    t.n_obj = nobj;
    t.kernel = a.kernel;
    t.n_pad = a.n_rb * kRB;
    t.n_ord = a.n_ord;
    t.n_pat = a.n_pat;
    t.n_tiles = a.n_tiles;
    const int64_t cat = (int64_t)nobj * a.n_obs * a.n_pat;
    t.cat_smem = (a.n_ord < a.d && cat <= kCatSmemMax) ? (int32_t)cat : 0;
    t.err = ctx->d_err;
    return t;
}

// Padded ordinal feature count of the kernels (DO).
int tc_do(const ScoreArgs& a) { return a.n_ord <= 4 ? 4 : a.n_ord <= 8 ? 8 : a.n_ord <= 12 ? 12 : 16; }

// The tensor-core route of the entry points that take moments or an
// acquisition straight from the posterior, without V: t carries the outputs
// (mean / var, or the acquisition epilogue) and a.cand / n / ld the pool.
// Workspace: the compacted list (when masked), then the split copy of
// L^{-1}, reserved whole before the compaction writes the list; where the
// mask is 0 the compaction writes -inf into the fill_rows rows of the
// acquisition.  *used is false (nothing launched) when the context has the
// tensor cores off or the model does not fit the tensor-core kernel.
scoot_status tc_direct(scoot_ctx* ctx, const ScoreArgs& a, const uint8_t* mask, ScootTcArgs t, int fill_rows,
                       cudaStream_t st, bool* used) {
    *used = false;
    if (!ctx->tensor_cores || a.n_rb * kRB > kMaxNpadTc) return SCOOT_OK;
    const int DO = tc_do(a);
    if (!scoot_tc_supported(ctx, t, DO)) return SCOOT_OK;
    *used = true;
    const size_t list_bytes = mask ? ((256 + (size_t)a.n * 4 + 255) & ~(size_t)255) : 0;
    scoot_status s = scoot_workspace(ctx, list_bytes + (size_t)scoot_tc_bsplit_bytes(t.n_pad, t.n_obj));
    if (s != SCOOT_OK) return s;
    if (mask) {
        ScootList lst;
        uint32_t* fill = t.acq_kind ? reinterpret_cast<uint32_t*>(t.acq) : nullptr;
        if ((s = scoot_compact(ctx, mask, a.n, fill, 0xFF800000u, st, &lst, fill_rows, t.lda)) != SCOOT_OK) return s;
        t.list = lst.list;
        t.n_list = lst.count;
    }
    t.cand = a.cand;
    t.n = a.n;
    t.ld = a.ld;
    t.vout = nullptr;
    t.by_index = 1;
    t.bsplit = static_cast<uint8_t*>(ctx->ws) + list_bytes;
    return scoot_posterior_tc(ctx, t, DO, st);
}

}  // namespace

scoot_status scoot_posterior_whitened(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                      const uint32_t* cand, int64_t n, int64_t ld, const int32_t* list,
                                      const unsigned int* n_list, float* mean, float* var, float* V, int64_t ldc,
                                      void* tc_work, cudaStream_t st) {
    ScoreArgs a;
    scoot_status s = fill_state_args(ctx, L, state, a);
    if (s != SCOOT_OK) return s;
    if (tc_work && ctx->tensor_cores) {
        ScootTcArgs t = tc_args(ctx, a, a.n_obj);
        t.cand = cand;
        t.n = n;
        t.ld = ld;
        t.list = list;
        t.n_list = n_list;
        t.mean = mean;
        t.var = var;
        t.ldo = ldc;
        t.vout = V;
        t.by_index = 0;
        t.bsplit = static_cast<uint8_t*>(tc_work);
        const int DO = tc_do(a);
        if (scoot_tc_supported(ctx, t, DO)) return scoot_posterior_tc(ctx, t, DO, st);
    }
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.list = list;
    a.n_list = n_list;
    a.mean = mean;
    a.var = var;
    a.ldo = ldc;
    a.vout = V;
    return launch_score<kWriteWhitened, 1>(ctx, a, st);
}

extern "C" {

scoot_status scoot_gp_posterior(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                                float* mean, float* var, int64_t ldo, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ScoreArgs a;
    if ((s = fill_state_args(ctx, L, state, a)) != SCOOT_OK) return s;
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!mean || !var || ldo < n) return scoot_fail(ctx, SCOOT_EINVAL, "mean/var NULL or ldo < n");
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.mask = mask;
    a.mean = mean;
    a.var = var;
    a.ldo = ldo;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    ScootTcArgs t = tc_args(ctx, a, a.n_obj);
    t.mean = mean;
    t.var = var;
    t.ldo = ldo;
    bool used = false;
    s = tc_direct(ctx, a, mask, t, 0, st, &used);
    if (used || s != SCOOT_OK) return s;
    return launch_score<kWriteMoments, 1>(ctx, a, st);
}

scoot_status scoot_acq_ei(scoot_ctx* ctx, const float* mean, const float* var, const uint8_t* mask,
                          int64_t n, float y_best, float xi, float* acq, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n < 0");
    if (n == 0) return SCOOT_OK;
    if (!mean || !var || !acq) return scoot_fail(ctx, SCOOT_EINVAL, "mean, var or acq is NULL");
    int64_t blocks = (n + kAcqThreads - 1) / kAcqThreads;
    const int64_t cap = (int64_t)sm_count(ctx->device) * 16;
    if (blocks > cap) blocks = cap;
    ei_kernel<<<(unsigned)blocks, kAcqThreads, 0, static_cast<cudaStream_t>(stream)>>>(mean, var, mask, n, y_best, xi, acq);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_acq_mace(scoot_ctx* ctx, const float* mean, const float* var, const uint8_t* mask,
                            int64_t n, float y_best, float xi, float kappa, float* acq, int64_t lda, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n < 0");
    if (n == 0) return SCOOT_OK;
    if (!mean || !var || !acq) return scoot_fail(ctx, SCOOT_EINVAL, "mean, var or acq is NULL");
    if (lda < n) return scoot_fail(ctx, SCOOT_EINVAL, "lda = %lld < n", (long long)lda);
    int64_t blocks = (n + kAcqThreads - 1) / kAcqThreads;
    const int64_t cap = (int64_t)sm_count(ctx->device) * 16;
    if (blocks > cap) blocks = cap;
    mace_kernel<<<(unsigned)blocks, kAcqThreads, 0, static_cast<cudaStream_t>(stream)>>>(mean, var, mask, n, y_best,
                                                                                          xi, kappa, acq, lda);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_acq_ehvi(scoot_ctx* ctx, const float* mean, const float* var, int64_t ldm, int32_t n_obj,
                            const uint8_t* mask, int64_t n, const float* box_lo, const float* box_hi,
                            int32_t n_boxes, const float* eps, int32_t n_mc, float* acq, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n < 0");
    if ((s = check_boxes(ctx, n_obj, box_lo, box_hi, n_boxes, eps, n_mc)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!mean || !var || !acq || ldm < n) return scoot_fail(ctx, SCOOT_EINVAL, "mean/var/acq NULL or ldm < n");
    ScoreArgs a;
    std::memset(&a, 0, sizeof(a));
    a.mean = const_cast<float*>(mean);
    a.var = const_cast<float*>(var);
    a.ldo = ldm;
    a.mask = mask;
    a.n = n;
    a.acq = acq;
    a.box_lo = box_lo;
    a.box_hi = box_hi;
    a.n_boxes = n_boxes;
    a.eps = eps;
    a.n_mc = n_mc;
    const size_t smem = (size_t)(2 * n_boxes + n_mc) * 16;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (mask) {
        ScootList lst;
        if ((s = scoot_compact(ctx, mask, n, reinterpret_cast<uint32_t*>(acq), 0xFF800000u, st, &lst)) != SCOOT_OK)
            return s;
        a.list = lst.list;
        a.n_list = lst.count;
    }
    int64_t blocks = (n + kAcqThreads - 1) / kAcqThreads;
    auto go = [&](auto kern) -> scoot_status {
        SCOOT_CUDA(ctx, cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        int per_sm = 0;
        SCOOT_CUDA(ctx, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kAcqThreads, smem));
        if (per_sm < 1) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "EHVI kernel does not fit");
        const int64_t cap = (int64_t)sm_count(ctx->device) * per_sm;
        if (blocks > cap) blocks = cap;
        kern<<<(unsigned)blocks, kAcqThreads, smem, st>>>(a);
        SCOOT_LAUNCHED(ctx);
        return SCOOT_OK;
    };
    switch (n_obj) {
    case 2: return go(ehvi_kernel<2>);
    case 3: return go(ehvi_kernel<3>);
    default: return go(ehvi_kernel<4>);
    }
}

scoot_status scoot_acq_ehvi_exact(scoot_ctx* ctx, const float* mean, const float* var, int64_t ldm, int32_t n_obj,
                                  const uint8_t* mask, int64_t n, const float* grid, int32_t grid_cap,
                                  const int32_t* h_n_grid, const uint32_t* corner, int32_t n_boxes, float* acq,
                                  void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (n < 0) return scoot_fail(ctx, SCOOT_EINVAL, "n < 0");
    ScoreArgs a;
    std::memset(&a, 0, sizeof(a));
    if ((s = fill_box_grid(ctx, n_obj, grid, grid_cap, h_n_grid, corner, n_boxes, a)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!mean || !var || !acq || ldm < n) return scoot_fail(ctx, SCOOT_EINVAL, "mean/var/acq NULL or ldm < n");
    a.mean = const_cast<float*>(mean);
    a.var = const_cast<float*>(var);
    a.ldo = ldm;
    a.mask = mask;
    a.n = n;
    a.acq = acq;
    a.err = ctx->d_err;
    const size_t smem = ((size_t)a.psi_rows * kAcqThreads + ((a.psi_rows + 3) & ~3) + (size_t)n_boxes * n_obj) * 4;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (mask) {
        ScootList lst;
        if ((s = scoot_compact(ctx, mask, n, reinterpret_cast<uint32_t*>(acq), 0xFF800000u, st, &lst)) != SCOOT_OK)
            return s;
        a.list = lst.list;
        a.n_list = lst.count;
    }
    int64_t blocks = (n + kAcqThreads - 1) / kAcqThreads;
    auto go = [&](auto kern) -> scoot_status {
        SCOOT_CUDA(ctx, cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        int per_sm = 0;
        SCOOT_CUDA(ctx, cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kAcqThreads, smem));
        if (per_sm < 1) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "exact EHVI kernel does not fit");
        const int64_t cap = (int64_t)sm_count(ctx->device) * per_sm;
        if (blocks > cap) blocks = cap;
        kern<<<(unsigned)blocks, kAcqThreads, smem, st>>>(a);
        SCOOT_LAUNCHED(ctx);
        return SCOOT_OK;
    };
    switch (n_obj) {
    case 2: return go(ehvix_kernel<2>);
    case 3: return go(ehvix_kernel<3>);
    default: return go(ehvix_kernel<4>);
    }
}

scoot_status scoot_score_ehvi_exact(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                    const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                                    const float* grid, int32_t grid_cap, const int32_t* h_n_grid,
                                    const uint32_t* corner, int32_t n_boxes, float* acq, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ScoreArgs a;
    if ((s = fill_state_args(ctx, L, state, a)) != SCOOT_OK) return s;
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if ((s = fill_box_grid(ctx, L->n_obj, grid, grid_cap, h_n_grid, corner, n_boxes, a)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!acq) return scoot_fail(ctx, SCOOT_EINVAL, "acq is NULL");
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.mask = mask;
    a.acq = acq;
    return dispatch_m<kEHVIX>(ctx, a, L->n_obj, static_cast<cudaStream_t>(stream));
}

scoot_status scoot_score_ei(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                            const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                            float xi, float* acq, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ScoreArgs a;
    if ((s = fill_state_args(ctx, L, state, a)) != SCOOT_OK) return s;
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!acq) return scoot_fail(ctx, SCOOT_EINVAL, "acq is NULL");
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.mask = mask;
    a.acq = acq;
    a.xi = xi;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    ScootTcArgs t = tc_args(ctx, a, 1);
    t.acq_kind = 1;
    t.acq = acq;
    t.lda = n;
    t.xi = xi;
    bool used = false;
    s = tc_direct(ctx, a, mask, t, 1, st, &used);
    if (used || s != SCOOT_OK) return s;
    return launch_score<kEI, 1>(ctx, a, st);
}

scoot_status scoot_score_mace(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                              const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                              float xi, float kappa, float* acq, int64_t lda, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ScoreArgs a;
    if ((s = fill_state_args(ctx, L, state, a)) != SCOOT_OK) return s;
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!acq) return scoot_fail(ctx, SCOOT_EINVAL, "acq is NULL");
    if (lda < n) return scoot_fail(ctx, SCOOT_EINVAL, "lda = %lld < n", (long long)lda);
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.mask = mask;
    a.acq = acq;
    a.lda = lda;
    a.xi = xi;
    a.kappa = kappa;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    ScootTcArgs t = tc_args(ctx, a, 1);
    t.acq_kind = 2;
    t.acq = acq;
    t.lda = lda;
    t.xi = xi;
    t.kappa = kappa;
    bool used = false;
    s = tc_direct(ctx, a, mask, t, 3, st, &used);
    if (used || s != SCOOT_OK) return s;
    return launch_score<kMACE, 1>(ctx, a, st);
}

scoot_status scoot_score_ehvi(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                              const uint32_t* cand, int64_t n, int64_t ld, const uint8_t* mask,
                              const float* box_lo, const float* box_hi, int32_t n_boxes,
                              const float* eps, int32_t n_mc, float* acq, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    ScoreArgs a;
    if ((s = fill_state_args(ctx, L, state, a)) != SCOOT_OK) return s;
    if ((s = scoot_check_pool(ctx, cand, n, ld, L->d)) != SCOOT_OK) return s;
    if ((s = check_boxes(ctx, L->n_obj, box_lo, box_hi, n_boxes, eps, n_mc)) != SCOOT_OK) return s;
    if (n == 0) return SCOOT_OK;
    if (!acq) return scoot_fail(ctx, SCOOT_EINVAL, "acq is NULL");
    a.cand = cand;
    a.n = n;
    a.ld = ld;
    a.mask = mask;
    a.acq = acq;
    a.box_lo = box_lo;
    a.box_hi = box_hi;
    a.n_boxes = n_boxes;
    a.eps = eps;
    a.n_mc = n_mc;
    return dispatch_m<kEHVI>(ctx, a, L->n_obj, static_cast<cudaStream_t>(stream));
}

}  // extern "C"
