// The per-round GP state (Section 4.3) built on the device: features of the
// observations, K + tau^2 I in fp64, its Cholesky factor, L^{-1} and
// alpha = (K + tau^2 I)^{-1} y, written into the same blob layout that the
// host preparation produces and the posterior and scoring kernels read.
//
// L^{-1} comes out of the factorisation itself: the elimination that turns
// K into L^T, applied to the identity, gives L^{-1}.  At step j, with pivot
// p_j = sqrt(A_jj) and l_ij = A_ij / p_j, every row i > j takes
//   A_ik -= l_ij l_kj   (j < k <= i)   and   W_ic -= l_ij W_jc / p_j   (c <= j),
// and row i of L^{-1} is W_i / p_i once the steps before i are done.  The
// rows of one step are independent, so a step is one barrier.  fp64 runs at
// a small fraction of the fp32 rate on this GPU; the n^3/3 multiply-adds of
// a factorisation are its cost.
#include <cmath>
#include <cstring>
#include <vector>

#include <cooperative_groups.h>

#include "internal.h"

namespace {

constexpr int kFeatThreads = 128;
constexpr int kKmatThreads = 128;
constexpr int kCholThreads = 1024;
constexpr int kRowBlockDev = 64;   // rows of L^{-1} per tile (the layout's)
constexpr int kColChunkDev = 32;   // columns of L^{-1} per tile
constexpr int kSmemCholMaxN = 160; // A and W (packed lower triangles, fp64) in shared memory up to this n

struct GpPrepArgs {
    int32_t n, d, M, kernel, n_ord, n_pat, n_rb, n_tiles;
    int64_t tri;                        // n (n + 1) / 2
    int32_t order[SCOOT_MAX_DIM];       // feature f -> source parameter
    int32_t kind[SCOOT_MAX_DIM];        // per source parameter
    int32_t n_choices[SCOOT_MAX_DIM];
    double lo[SCOOT_MAX_DIM], span[SCOOT_MAX_DIM];  // ordinal: (v - lo) / span; log: (ln v - lo) / span
    float fmap[SCOOT_MAX_DIM][4];       // the blob's feature map, computed on the host
    const uint32_t* obs;
    int64_t ld_obs;
    const float* y;                     // [M][n]
    const float* ls;                    // [M][d], source order
    const float* sf2;                   // [M]
    const float* tau2;                  // [M]
    const float* warp;                  // [M][d][2] or nullptr
    char* blob;
    int64_t off_fmap, off_xs, off_ils, off_alpha, off_linv, off_scal, off_cat, off_warp;
    double* U;                          // [M][n][d] scaled features, source order
    double* K;                          // [M][tri] packed lower triangle of K + tau^2 I (factorised in place when n is large)
    double* W;                          // [M][tri] elimination of the identity (n large)
    uint32_t* err;
};

__device__ __forceinline__ int64_t tri_idx(int i, int k) { return (int64_t)i * (i + 1) / 2 + k; }

// 1 / sqrt(v) for v > 0 by Newton-Raphson on f(y) = 1 / y^2 - v from an
// fp32 estimate, y <- y + y (1 - v y^2) / 2: each step doubles the correct
// bits (24 -> 48 -> beyond fp64), in fused multiply-adds only, which keeps
// the pivot off the slow fp64 division and square root.  Outside the fp32
// range of the estimate the library's division and square root are used.
__device__ __forceinline__ double rsqrt_newton(double v) {
    if (!(v > 1e-30 && v < 1e30)) return 1.0 / sqrt(v);
    double y = (double)rsqrtf((float)v);
    const double h = 0.5 * v;
    for (int it = 0; it < 3; ++it) {
        const double e = fma(-h * y, y, 0.5);  // (1 - v y^2) / 2
        y = fma(y, e, y);
    }
    return y;
}

__device__ __forceinline__ double matern_dev(double r, int kernel) {
    if (kernel == SCOOT_MATERN32) {
        const double a = 1.7320508075688772 * r;  // sqrt(3) r
        return (1.0 + a) * exp(-a);
    }
    const double a = 2.23606797749979 * r;  // sqrt(5) r
    return (1.0 + a + a * a / 3.0) * exp(-a);
}

// One thread per (observation j, feature f) of objective m: the feature,
// warped and scaled (fp64 logarithms and powers are slow here, so they are
// spread over n d threads).
__global__ void __launch_bounds__(kFeatThreads) gp_feat_kernel(const __grid_constant__ GpPrepArgs a) {
    const int t = blockIdx.x * kFeatThreads + threadIdx.x, m = blockIdx.y;
    const int d = a.d, j = t / d, f = t - j * d;
    bool bad = false;
    if (j < a.n) {
        float* xs = reinterpret_cast<float*>(a.blob + a.off_xs) + ((int64_t)m * a.n + j) * d;
        double* U = a.U + ((int64_t)m * a.n + j) * d;
        const int c = a.order[f];
        const uint32_t w = a.obs[(int64_t)c * a.ld_obs + j];
        const double l = (double)a.ls[m * d + c];
        bad |= !(l > 0.0) || !isfinite(l);
        if (a.kind[c] == SCOOT_CATEGORICAL) {
            const double u = (double)(int32_t)w;
            U[c] = u;
            xs[f] = (float)u;
        } else {
            const double v = a.kind[c] == SCOOT_CONTINUOUS ? (double)__uint_as_float(w) : (double)(int32_t)w;
            bad |= !isfinite(v) || (a.kind[c] == SCOOT_INT_LOG && !(v > 0.0));
            double u;
            if (a.kind[c] == SCOOT_INT_LOG) u = (log(v) - a.lo[c]) / a.span[c];
            else u = a.span[c] > 0.0 ? (v - a.lo[c]) / a.span[c] : 0.0;
            if (a.warp) {
                const double wa = (double)a.warp[((int64_t)m * d + c) * 2];
                const double wb = (double)a.warp[((int64_t)m * d + c) * 2 + 1];
                bad |= !(wa > 0.0) || !isfinite(wa) || !(wb > 0.0) || !isfinite(wb);
                const double x = fmin(fmax(u, 0.0), 1.0);
                u = 1.0 - pow(1.0 - pow(x, wa), wb);
            }
            U[c] = u / l;
            xs[f] = (float)(u / l);
        }
        if (f == 0) bad |= !isfinite(a.y[(int64_t)m * a.n + j]);
    }
    if (t == 0) {  // per-objective scalars (thread 0 of the objective's first block)
        const float sf2 = a.sf2[m], tau2 = a.tau2[m];
        bad |= !(sf2 > 0.0f) || !isfinite(sf2) || !(tau2 >= 0.0f) || !isfinite(tau2);
        float* ils = reinterpret_cast<float*>(a.blob + a.off_ils) + m * d;
        float* wo = reinterpret_cast<float*>(a.blob + a.off_warp) + (int64_t)m * d * 2;
        for (int g = 0; g < d; ++g) {
            const int c = a.order[g];
            const double l = (double)a.ls[m * d + c];
            const bool cat = a.kind[c] == SCOOT_CATEGORICAL;
            ils[g] = cat ? (float)(1.0 / (l * l)) : (float)(1.0 / l);
            wo[2 * g] = (a.warp && !cat) ? a.warp[((int64_t)m * d + c) * 2] : 1.0f;
            wo[2 * g + 1] = (a.warp && !cat) ? a.warp[((int64_t)m * d + c) * 2 + 1] : 1.0f;
        }
        float* scal = reinterpret_cast<float*>(a.blob + a.off_scal) + m * 4;
        scal[0] = sf2;
        scal[1] = tau2;
        scal[3] = a.warp ? 1.0f : 0.0f;  // scal[2] (best observed y) is written by the factorisation
        if (m == 0) {
            float* fm = reinterpret_cast<float*>(a.blob + a.off_fmap);
            for (int g = 0; g < d; ++g)
                for (int q = 0; q < 4; ++q) fm[g * 4 + q] = a.fmap[g][q];
        }
    }
    if (bad) atomicOr(a.err, SCOOT_DEVERR_VALUE);
}

// Categorical part of r^2 for every (observation, category pattern).
__global__ void __launch_bounds__(kKmatThreads) gp_cat_kernel(const __grid_constant__ GpPrepArgs a) {
    const int64_t t = (int64_t)blockIdx.x * kKmatThreads + threadIdx.x;
    const int m = blockIdx.y;
    if (t >= (int64_t)a.n * a.n_pat) return;
    const int j = (int)(t / a.n_pat), pat = (int)(t - (int64_t)j * a.n_pat);
    double r2 = 0.0;
    int rest = pat;
    for (int f = a.n_ord; f < a.d; ++f) {
        const int c = a.order[f];
        const int v = rest % a.n_choices[c];
        rest /= a.n_choices[c];
        const double l = (double)a.ls[m * a.d + c];
        if (v != (int32_t)a.obs[(int64_t)c * a.ld_obs + j]) r2 += 1.0 / (l * l);
    }
    reinterpret_cast<float*>(a.blob + a.off_cat)[((int64_t)m * a.n + j) * a.n_pat + pat] = (float)r2;
}

// K + tau^2 I, one thread per entry of the lower triangle.
__global__ void __launch_bounds__(kKmatThreads) gp_kmat_kernel(const __grid_constant__ GpPrepArgs a) {
    const int64_t t = (int64_t)blockIdx.x * kKmatThreads + threadIdx.x;
    const int m = blockIdx.y;
    if (t >= a.tri) return;
    int i = (int)((sqrt(8.0 * (double)t + 1.0) - 1.0) * 0.5);
    while ((int64_t)i * (i + 1) / 2 > t) --i;
    while ((int64_t)(i + 1) * (i + 2) / 2 <= t) ++i;
    const int k = (int)(t - (int64_t)i * (i + 1) / 2);
    const double* ui = a.U + ((int64_t)m * a.n + i) * a.d;
    const double* uk = a.U + ((int64_t)m * a.n + k) * a.d;
    double r2 = 0.0;
    for (int c = 0; c < a.d; ++c) {
        const double diff = ui[c] - uk[c];
        if (a.kind[c] == SCOOT_CATEGORICAL) {
            const double l = (double)a.ls[m * a.d + c];
            r2 += diff != 0.0 ? 1.0 / (l * l) : 0.0;
        } else {
            r2 += diff * diff;
        }
    }
    double v = (double)a.sf2[m] * matern_dev(sqrt(r2), a.kernel);
    if (i == k) v += (double)a.tau2[m];
    a.K[(int64_t)m * a.tri + t] = v;
}

// The factorisation of the packed lower triangle A (n x n, K + tau^2 I on
// entry) with the elimination applied to the identity in W, by the whole
// block.  On return, row i of L^{-1} is W_i * rinv[i];
// rinv2[i] = rinv[i]^2; A holds the eliminated values.  col: [2][n] scratch.
// Returns false (in every thread) if a pivot is not positive and finite.
//
// Step j in a single multiply-add per entry: with g_i = A_ij / A_jj,
//   A_ik -= g_i A_kj (j < k <= i)   and   W_ic -= g_i W_jc (c <= j),
// one loop over t = 0 .. i per row (t <= j: W, t > j: A) so that the lanes
// of a warp stay busy.  Column j is read from a contiguous copy (col), which
// the threads that finish its entries in step j - 1 write (two buffers by
// step parity).
__device__ bool eliminate(double* A, double* W, double* col, double* rinv, double* rinv2, int n) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = blockDim.x >> 5;
    // s_bad_at: the first step whose pivot is not positive (n if none).  It is
    // written during step j - 1 with the value j, so a thread still reading it
    // for step j - 1 does not stop early; every thread stops at step j.  The
    // pivot's reciprocals are computed once, by the thread that finishes the
    // diagonal entry (fp64 square roots and divisions are slow here), and
    // read after the step's barrier.
    __shared__ int s_bad_at;
    __syncthreads();  // A is complete; s_bad_at of an earlier call is read by no one
    for (int i = warp; i < n; i += nwarps)
        for (int c = lane; c <= i; c += 32) W[tri_idx(i, c)] = c == i ? 1.0 : 0.0;
    for (int i = tid; i < n; i += (int)blockDim.x) col[i] = A[tri_idx(i, 0)];
    if (tid == 0) {
        const double s0 = A[0];
        const bool bad = !(s0 > 0.0) || !isfinite(s0);
        s_bad_at = bad ? 0 : n;
        rinv[0] = bad ? 0.0 : rsqrt_newton(s0);
        rinv2[0] = rinv[0] * rinv[0];
    }
    __syncthreads();
    for (int j = 0; j < n; ++j) {
        if (s_bad_at <= j) break;  // the same in every thread
        const double r2 = rinv2[j];
        const double* cj = col + (j & 1) * n;
        double* cn = col + ((j + 1) & 1) * n;
        const double* Wj = W + tri_idx(j, 0);
        for (int i = j + 1 + warp; i < n; i += nwarps) {
            double* Ai = A + tri_idx(i, 0);
            double* Wi = W + tri_idx(i, 0);
            const double g = cj[i] * r2;
            for (int t = lane; t <= i; t += 32) {
                double* dst = t <= j ? Wi + t : Ai + t;
                const double src = t <= j ? Wj[t] : cj[t];
                const double v = *dst - g * src;
                *dst = v;
                if (t == j + 1) {  // A[i][j+1] is final: column j + 1 of the next step
                    cn[i] = v;
                    if (i == j + 1) {
                        if (!(v > 0.0) || !isfinite(v)) {
                            s_bad_at = j + 1;
                        } else {
                            const double y = rsqrt_newton(v);
                            rinv[j + 1] = y;
                            rinv2[j + 1] = y * y;
                        }
                    }
                }
            }
        }
        __syncthreads();
    }
    const bool ok = s_bad_at >= n;  // read after the loop's last barrier: the same in every thread
    __syncthreads();                // before a later call rewrites s_bad_at
    return ok;
}

// One block per objective: the factorisation with L^{-1} alongside, then
// alpha, the best observed y and the fp32 tiles of L^{-1}.
__global__ void __launch_bounds__(kCholThreads) gp_chol_kernel(const __grid_constant__ GpPrepArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int n = a.n, m = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = kCholThreads / 32;
    double* rinv = reinterpret_cast<double*>(smem_raw);  // [n] 1 / pivot
    double* rinv2 = rinv + n;                            // [n] 1 / pivot^2
    double* z = rinv2 + n;                               // [n] L^{-1} y
    double* col = z + n;                                 // [2][n] column j of A
    double* A;
    double* W;
    if (n <= kSmemCholMaxN) {
        A = col + 2 * n;
        W = A + a.tri;
        for (int64_t t = tid; t < a.tri; t += kCholThreads) A[t] = a.K[(int64_t)m * a.tri + t];
    } else {
        A = a.K + (int64_t)m * a.tri;
        W = a.W + (int64_t)m * a.tri;
    }
    if (!eliminate(A, W, col, rinv, rinv2, n)) {
        if (tid == 0) atomicOr(a.err, SCOOT_DEVERR_VALUE);
        return;
    }
    const float* y = a.y + (int64_t)m * n;
    // z = L^{-1} y, a warp per row
    for (int i = warp; i < n; i += nwarps) {
        const double* Wi = W + tri_idx(i, 0);
        double t = 0.0;
        for (int c = lane; c <= i; c += 32) t += Wi[c] * (double)y[c];
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) z[i] = t * rinv[i];
    }
    __syncthreads();
    // alpha = L^{-T} z, a thread per column
    float* alpha = reinterpret_cast<float*>(a.blob + a.off_alpha) + (int64_t)m * n;
    for (int c = tid; c < n; c += kCholThreads) {
        double t = 0.0;
        for (int i = c; i < n; ++i) t += W[tri_idx(i, c)] * rinv[i] * z[i];
        alpha[c] = (float)t;
    }
    if (warp == 0) {
        float best = -INFINITY;
        for (int j = lane; j < n; j += 32) best = fmaxf(best, y[j]);
        for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, o));
        if (lane == 0) reinterpret_cast<float*>(a.blob + a.off_scal)[m * 4 + 2] = best;
    }
    // tiles: row block rb, column chunk cj; tile[jj][ii] = L^{-1}[64 rb + ii][32 cj + jj]
    float* tiles = reinterpret_cast<float*>(a.blob + a.off_linv) + (int64_t)m * a.n_tiles * kColChunkDev * kRowBlockDev;
    const int64_t total = (int64_t)a.n_tiles * kColChunkDev * kRowBlockDev;
    for (int64_t e = tid; e < total; e += kCholThreads) {
        const int t = (int)(e / (kColChunkDev * kRowBlockDev));
        const int jj = (int)(e / kRowBlockDev % kColChunkDev), ii = (int)(e % kRowBlockDev);
        int rb = 0;
        while ((rb + 1) * (rb + 2) <= t) ++rb;  // tiles of row blocks before rb: rb (rb + 1)
        const int cj = t - rb * (rb + 1);
        const int row = rb * kRowBlockDev + ii, c = cj * kColChunkDev + jj;
        float v = 0.0f;
        if (row < n && c <= row) v = (float)(W[tri_idx(row, c)] * rinv[row]);
        tiles[e] = v;
    }
}

constexpr int kClusterCTAs = 8;          // CTAs sharing one factorisation (portable cluster size)
constexpr int kClusterThreads = 256;
constexpr int kClusterMaxN = 384;        // rows of A and W split over the cluster's shared memory

// Offset of local row li (global row rank + C li) in a CTA's packed rows:
// row i holds i + 1 entries.
__device__ __forceinline__ int64_t local_row_off(int li, int rank) {
    return (int64_t)li * (rank + 1) + (int64_t)kClusterCTAs * li * (li - 1) / 2;
}

// The factorisation of gp_chol_kernel spread over a cluster of kClusterCTAs
// CTAs (one cluster per objective): CTA r owns rows i = r (mod C) of A and
// W in its shared memory.  What a step needs from other rows travels through
// distributed shared memory before the step's cluster barrier: the thread
// that finishes A_i,j+1 stores it into every CTA's copy of the next pivot
// column, the row j+1 of W is stored the same way as its entries become
// final, and the thread that finishes the next diagonal entry stores its
// reciprocals (or the failure) everywhere.  Then z = L^{-1} y per owned row
// (broadcast), per-CTA partial sums of alpha = L^{-T} z over owned rows
// (added in rank order by CTA 0), and each CTA writes its rows' tiles.
__global__ void __cluster_dims__(kClusterCTAs, 1, 1) __launch_bounds__(kClusterThreads)
gp_chol_cluster_kernel(const __grid_constant__ GpPrepArgs a) {
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int n = a.n, C = kClusterCTAs;
    const int rank = (int)cluster.block_rank(), m = blockIdx.x / C;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = kClusterThreads / 32;
    double* rinv = reinterpret_cast<double*>(smem_raw);  // [n]
    double* rinv2 = rinv + n;                            // [n]
    double* col = rinv2 + n;                             // [2][n] pivot column
    double* wrow = col + 2 * n;                          // [2][n] row j of W
    double* z = wrow + 2 * n;                            // [n]
    double* part = z + n;                                // [n] this CTA's share of alpha
    const int nl = (n - rank + C - 1) / C;               // rows owned
    double* A = part + n;                                // owned rows, packed
    double* W = A + local_row_off(nl, rank);
    __shared__ int s_bad_at;
    const double* K = a.K + (int64_t)m * a.tri;
    // load owned rows; W = I
    for (int li = warp; li < nl; li += nwarps) {
        const int i = rank + C * li;
        const int64_t o = local_row_off(li, rank);
        for (int t = lane; t <= i; t += 32) {
            A[o + t] = K[tri_idx(i, t)];
            W[o + t] = t == i ? 1.0 : 0.0;
        }
    }
    // the first pivot column, row 0 of W and the first pivot, everywhere
    for (int li = tid; li < nl; li += kClusterThreads) {
        const int i = rank + C * li;
        const double v = K[tri_idx(i, 0)];
        for (int r = 0; r < C; ++r) cluster.map_shared_rank(col, r)[i] = v;
    }
    if (tid == 0) {
        const double s0 = K[0];
        const bool bad = !(s0 > 0.0) || !isfinite(s0);
        s_bad_at = bad ? 0 : n;
        rinv[0] = bad ? 0.0 : rsqrt_newton(s0);
        rinv2[0] = rinv[0] * rinv[0];
        wrow[0] = 1.0;
    }
    cluster.sync();
    for (int j = 0; j < n; ++j) {
        if (s_bad_at <= j) break;  // the same in every thread of the cluster
        const double r2 = rinv2[j];
        const double* cj = col + (j & 1) * n;
        const double* wj = wrow + (j & 1) * n;
        const int nb = (j + 1) & 1;
        // owned rows i > j
        int li0 = (j + 1 - rank + C - 1) / C;
        if (li0 < 0) li0 = 0;
        for (int li = li0 + warp; li < nl; li += nwarps) {
            const int i = rank + C * li;
            const int64_t o = local_row_off(li, rank);
            const double g = cj[i] * r2;
            for (int t = lane; t <= i; t += 32) {
                double* dst = t <= j ? W + o + t : A + o + t;
                const double src = t <= j ? wj[t] : cj[t];
                const double v = *dst - g * src;
                *dst = v;
                if (t == j + 1) {  // A_i,j+1 is final: the next pivot column, everywhere
                    for (int r = 0; r < C; ++r) cluster.map_shared_rank(col + nb * n, r)[i] = v;
                    if (i == j + 1) {
                        if (!(v > 0.0) || !isfinite(v)) {
                            for (int r = 0; r < C; ++r) *cluster.map_shared_rank(&s_bad_at, r) = j + 1;
                        } else {
                            const double y = rsqrt_newton(v);
                            for (int r = 0; r < C; ++r) {
                                cluster.map_shared_rank(rinv, r)[j + 1] = y;
                                cluster.map_shared_rank(rinv2, r)[j + 1] = y * y;
                            }
                        }
                    }
                }
                if (i == j + 1 && t <= j)  // W_j+1,t is final: row j + 1 of W, everywhere
                    for (int r = 0; r < C; ++r) cluster.map_shared_rank(wrow + nb * n, r)[t] = v;
            }
            if (i == j + 1 && lane == 0)
                for (int r = 0; r < C; ++r) cluster.map_shared_rank(wrow + nb * n, r)[j + 1] = 1.0;
        }
        cluster.sync();
    }
    if (s_bad_at < n) {  // the same everywhere; no shared memory of another CTA is touched after this
        if (tid == 0 && rank == 0) atomicOr(a.err, SCOOT_DEVERR_VALUE);
        return;
    }
    const float* y = a.y + (int64_t)m * n;
    // z_i for owned rows, everywhere
    for (int li = warp; li < nl; li += nwarps) {
        const int i = rank + C * li;
        const int64_t o = local_row_off(li, rank);
        double t = 0.0;
        for (int c = lane; c <= i; c += 32) t += W[o + c] * (double)y[c];
        for (int sh = 16; sh > 0; sh >>= 1) t += __shfl_xor_sync(0xffffffffu, t, sh);
        if (lane == 0) {
            const double zi = t * rinv[i];
            for (int r = 0; r < C; ++r) cluster.map_shared_rank(z, r)[i] = zi;
        }
    }
    cluster.sync();
    // this CTA's share of alpha_c = sum over owned rows i >= c of L^{-1}_ic z_i
    for (int c = tid; c < n; c += kClusterThreads) {
        double t = 0.0;
        int li = (c - rank + C - 1) / C;
        if (li < 0) li = 0;
        for (; li < nl; ++li) {
            const int i = rank + C * li;
            t += W[local_row_off(li, rank) + c] * rinv[i] * z[i];
        }
        part[c] = t;
    }
    cluster.sync();
    if (rank == 0) {
        float* alpha = reinterpret_cast<float*>(a.blob + a.off_alpha) + (int64_t)m * n;
        for (int c = tid; c < n; c += kClusterThreads) {
            double t = 0.0;
            for (int r = 0; r < C; ++r) t += cluster.map_shared_rank(part, r)[c];
            alpha[c] = (float)t;
        }
        if (warp == 0) {
            float best = -INFINITY;
            for (int j = lane; j < n; j += 32) best = fmaxf(best, y[j]);
            for (int sh = 16; sh > 0; sh >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, sh));
            if (lane == 0) reinterpret_cast<float*>(a.blob + a.off_scal)[m * 4 + 2] = best;
        }
    }
    // tiles: the owner of a row writes its entries (CTA 0 the padding rows)
    float* tiles = reinterpret_cast<float*>(a.blob + a.off_linv) + (int64_t)m * a.n_tiles * kColChunkDev * kRowBlockDev;
    const int64_t total = (int64_t)a.n_tiles * kColChunkDev * kRowBlockDev;
    for (int64_t e = tid; e < total; e += kClusterThreads) {
        const int t = (int)(e / (kColChunkDev * kRowBlockDev));
        const int jj = (int)(e / kRowBlockDev % kColChunkDev), ii = (int)(e % kRowBlockDev);
        int rb = 0;
        while ((rb + 1) * (rb + 2) <= t) ++rb;
        const int cj = t - rb * (rb + 1);
        const int row = rb * kRowBlockDev + ii, c = cj * kColChunkDev + jj;
        if (row < n ? row % C != rank : rank != 0) continue;
        float v = 0.0f;
        if (row < n && c <= row) v = (float)(W[local_row_off(row / C, rank) + c] * rinv[row]);
        tiles[e] = v;
    }
    cluster.sync();  // CTA 0 has read every CTA's part before any CTA exits
}

constexpr int kMleMaxP = SCOOT_MAX_DIM + 2;  // ln l_1 .. ln l_d, ln s_f^2, ln tau^2
constexpr int kSmemMleMaxN = 128;             // A and W in shared memory up to this n
constexpr int kMleThreads = 512;

struct MleArgs {
    int32_t n, d, M, P, kernel, S, steps;
    int64_t tri;
    uint32_t free_mask;                      // bit p: parameter p is fitted
    uint32_t cat_mask;                       // bit c: parameter c is categorical
    double lr;
    double lo[kMleMaxP], hi[kMleMaxP];
    const double* U;                         // [n][d] features (unscaled, unwarped)
    const float* y;                          // [M][n]
    const double* theta0;                    // [S][M][P]
    double* theta;                           // [S][M][P]
    double* lml;                             // [S][M]
    double* grad;                            // [S][M][P] or nullptr
    double* scratch;                         // [S M][2][tri] when n > kSmemMleMaxN
};

// Features of the observations, once per call: one thread per (j, c).
__global__ void __launch_bounds__(kFeatThreads) mle_feat_kernel(const __grid_constant__ GpPrepArgs a) {
    const int t = blockIdx.x * kFeatThreads + threadIdx.x;
    const int j = t / a.d, c = t - j * a.d;
    if (j >= a.n) return;
    const uint32_t w = a.obs[(int64_t)c * a.ld_obs + j];
    double u;
    bool bad = false;
    if (a.kind[c] == SCOOT_CATEGORICAL) {
        u = (double)(int32_t)w;
    } else {
        const double v = a.kind[c] == SCOOT_CONTINUOUS ? (double)__uint_as_float(w) : (double)(int32_t)w;
        bad = !isfinite(v) || (a.kind[c] == SCOOT_INT_LOG && !(v > 0.0));
        if (a.kind[c] == SCOOT_INT_LOG) u = (log(v) - a.lo[c]) / a.span[c];
        else u = a.span[c] > 0.0 ? (v - a.lo[c]) / a.span[c] : 0.0;
    }
    a.U[(int64_t)j * a.d + c] = u;
    if (c == 0)
        for (int m = 0; m < a.M; ++m) bad |= !isfinite(a.y[(int64_t)m * a.n + j]);
    if (bad) atomicOr(a.err, SCOOT_DEVERR_VALUE);
}

// k(r) / s_f^2 and its derivative in r^2 for r^2 = r2.
__device__ __forceinline__ void matern_slope(double r2, int kernel, double* k, double* dk) {
    const double r = sqrt(r2);
    if (kernel == SCOOT_MATERN32) {
        const double a = 1.7320508075688772 * r, e = exp(-a);
        *k = (1.0 + a) * e;
        *dk = -1.5 * e;
    } else {
        const double a = 2.23606797749979 * r, e = exp(-a);
        *k = (1.0 + a + a * a / 3.0) * e;
        *dk = -(5.0 / 6.0) * (1.0 + a) * e;
    }
}

// One block per (start s, objective m): `steps` projected Adam steps on the
// log marginal likelihood (beta1 0.9, beta2 0.999, eps 1e-8, step size
// lr (1 - t / steps)), then the likelihood and gradient at the result.  Each
// evaluation: K + tau^2 I from the features, the factorisation with L^{-1},
// alpha = K^{-1} y, K^{-1} = L^{-T} L^{-1} (into A), and
// d lml / d theta_p = sum_{i >= j} w_ij (alpha_i alpha_j - K^{-1}_ij) dK_ij / dtheta_p
// with w = 1 off the diagonal and 1/2 on it.
__global__ void __launch_bounds__(kMleThreads) gp_mle_kernel(const __grid_constant__ MleArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int n = a.n, d = a.d, P = a.P;
    const int sm = blockIdx.x, m = sm % a.M;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = kMleThreads / 32;
    double* rinv = reinterpret_cast<double*>(smem_raw);  // [n]
    double* rinv2 = rinv + n;                            // [n]
    double* yv = rinv2 + n;                              // [n]
    double* z = yv + n;                                  // [n] L^{-1} y
    double* al = z + n;                                  // [n] alpha
    double* col = al + n;                                // [2][n]
    double* U = col + 2 * n;                             // [d][n]: feature c of observation j at c n + j
    double* A;
    double* W;
    if (n <= kSmemMleMaxN) {
        A = U + (size_t)n * d;
        W = A + a.tri;
    } else {
        A = a.scratch + (size_t)sm * 2 * a.tri;
        W = A + a.tri;
    }
    __shared__ double th[kMleMaxP], m1[kMleMaxP], m2[kMleMaxP], g[kMleMaxP];
    __shared__ double il2[SCOOT_MAX_DIM];  // 1 / l_c^2
    __shared__ double s_sf2, s_tau2;
    __shared__ double red[kMleThreads / 32][kMleMaxP + 1];
    __shared__ double s_total;  // y^T alpha + log det K
    __shared__ int s_fail;
    for (int i = tid; i < n; i += kMleThreads) yv[i] = (double)a.y[(int64_t)m * n + i];
    for (int t = tid; t < n * d; t += kMleThreads) {  // transposed, so that lanes on consecutive
        const int j = t / d, c = t - j * d;           // observations read consecutive words
        U[c * n + j] = a.U[t];
    }
    if (tid < P) {
        th[tid] = a.theta0[(int64_t)sm * P + tid];
        m1[tid] = 0.0;
        m2[tid] = 0.0;
    }
    if (tid == 0) s_fail = 0;
    double lml = 0.0;
    for (int it = 0; it <= a.steps; ++it) {
        __syncthreads();
        if (tid < d) il2[tid] = exp(-2.0 * th[tid]);
        if (tid == 0) {
            s_sf2 = exp(th[d]);
            s_tau2 = exp(th[d + 1]);
        }
        __syncthreads();
        const double sf2 = s_sf2, tau2 = s_tau2;
        // K + tau^2 I
        for (int64_t t = tid; t < a.tri; t += kMleThreads) {
            int i = (int)((sqrt(8.0 * (double)t + 1.0) - 1.0) * 0.5);
            while ((int64_t)i * (i + 1) / 2 > t) --i;
            while ((int64_t)(i + 1) * (i + 2) / 2 <= t) ++i;
            const int k = (int)(t - (int64_t)i * (i + 1) / 2);
            double r2 = 0.0;
            for (int c = 0; c < d; ++c) {
                const double df = U[c * n + i] - U[c * n + k];
                r2 += ((a.cat_mask >> c) & 1u) ? (df != 0.0 ? il2[c] : 0.0) : df * df * il2[c];
            }
            double kv, dk;
            matern_slope(r2, a.kernel, &kv, &dk);
            A[t] = sf2 * kv + (i == k ? tau2 : 0.0);
        }
        if (!eliminate(A, W, col, rinv, rinv2, n)) {
            if (tid == 0) s_fail = 1;
            __syncthreads();
            break;
        }
        // z = L^{-1} y (a warp per row), then alpha = L^{-T} z (a thread per column)
        for (int i = warp; i < n; i += nwarps) {
            const double* Wi = W + tri_idx(i, 0);
            double t = 0.0;
            for (int c = lane; c <= i; c += 32) t += Wi[c] * yv[c];
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            if (lane == 0) z[i] = t * rinv[i];
        }
        __syncthreads();
        for (int c = tid; c < n; c += kMleThreads) {
            double t = 0.0;
            for (int i = c; i < n; ++i) t += W[tri_idx(i, c)] * rinv[i] * z[i];
            al[c] = t;
        }
        // K^{-1} into A: (i, j <= i) = sum_{k >= i} L^{-1}_ki L^{-1}_kj
        for (int64_t t = tid; t < a.tri; t += kMleThreads) {
            int i = (int)((sqrt(8.0 * (double)t + 1.0) - 1.0) * 0.5);
            while ((int64_t)i * (i + 1) / 2 > t) --i;
            while ((int64_t)(i + 1) * (i + 2) / 2 <= t) ++i;
            const int j = (int)(t - (int64_t)i * (i + 1) / 2);
            double v = 0.0;
            for (int k = i; k < n; ++k) v += W[tri_idx(k, i)] * W[tri_idx(k, j)] * rinv2[k];
            A[t] = v;
        }
        __syncthreads();
        // gradient terms and the likelihood's two sums, per thread
        double acc[kMleMaxP + 1];
#pragma unroll
        for (int p = 0; p <= kMleMaxP; ++p) acc[p] = 0.0;
        for (int64_t t = tid; t < a.tri; t += kMleThreads) {
            int i = (int)((sqrt(8.0 * (double)t + 1.0) - 1.0) * 0.5);
            while ((int64_t)i * (i + 1) / 2 > t) --i;
            while ((int64_t)(i + 1) * (i + 2) / 2 <= t) ++i;
            const int k = (int)(t - (int64_t)i * (i + 1) / 2);
            const double w = (al[i] * al[k] - A[t]) * (i == k ? 0.5 : 1.0);
            if (i == k) {
                acc[kMleMaxP - 1] += w * tau2;
                acc[kMleMaxP - 2] += w * sf2;  // k(0) = 1
                continue;
            }
            double r2 = 0.0;
            for (int c = 0; c < d; ++c) {
                const double df = U[c * n + i] - U[c * n + k];
                r2 += ((a.cat_mask >> c) & 1u) ? (df != 0.0 ? il2[c] : 0.0) : df * df * il2[c];
            }
            double kv, dk;
            matern_slope(r2, a.kernel, &kv, &dk);
            const double f = -2.0 * sf2 * dk * w;
#pragma unroll
            for (int c = 0; c < SCOOT_MAX_DIM; ++c) {  // the feature's term of r^2 again (unrolled:
                if (c < d) {                           // acc stays in registers)
                    const double df = U[c * n + i] - U[c * n + k];
                    acc[c] += f * (((a.cat_mask >> c) & 1u) ? (df != 0.0 ? il2[c] : 0.0) : df * df * il2[c]);
                }
            }
            acc[kMleMaxP - 2] += w * sf2 * kv;
        }
        for (int i = tid; i < n; i += kMleThreads) acc[kMleMaxP] += yv[i] * al[i] - 2.0 * log(rinv[i]);
        // acc: lengthscales in 0 .. d-1, s_f^2 and tau^2 at kMleMaxP - 2 and - 1, and
        // y^T alpha + log det K at kMleMaxP; block reduction of the sums
#pragma unroll
        for (int p = 0; p <= kMleMaxP; ++p) {
            double v = acc[p];
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) red[warp][p] = v;
        }
        __syncthreads();
        if (tid <= kMleMaxP) {
            double v = 0.0;
            for (int w2 = 0; w2 < nwarps; ++w2) v += red[w2][tid];
            if (tid < d) g[tid] = v;
            else if (tid == kMleMaxP - 2) g[d] = v;
            else if (tid == kMleMaxP - 1) g[d + 1] = v;
            else if (tid == kMleMaxP) s_total = v;
        }
        __syncthreads();
        lml = -0.5 * s_total - 0.5 * n * 1.8378770664093453;  // log(2 pi)
        if (it == a.steps) break;
        if (tid == 0) {  // projected Adam step on the free parameters
            const double step = a.lr * (1.0 - (double)it / a.steps);
            const double c1 = 1.0 - pow(0.9, it + 1), c2 = 1.0 - pow(0.999, it + 1);
            for (int p = 0; p < P; ++p) {
                if (!((a.free_mask >> p) & 1u)) continue;
                const double gp = g[p];
                m1[p] = 0.9 * m1[p] + 0.1 * gp;
                m2[p] = 0.999 * m2[p] + 0.001 * gp * gp;
                const double upd = step * (m1[p] / c1) / (sqrt(m2[p] / c2) + 1e-8);
                th[p] = fmin(fmax(th[p] + upd, a.lo[p]), a.hi[p]);
            }
        }
    }
    if (tid < P) {
        a.theta[(int64_t)sm * P + tid] = th[tid];
        if (a.grad) a.grad[(int64_t)sm * P + tid] = s_fail ? 0.0 : g[tid];
    }
    if (tid == 0) a.lml[sm] = s_fail ? -INFINITY : lml;
}

}  // namespace

extern "C" {

scoot_status scoot_gp_device_work_bytes(const scoot_gp_layout* L, int64_t* bytes) {
    if (!L || !bytes || !scoot_gp_layout_valid(L)) return SCOOT_EINVAL;
    const int64_t n = L->n, tri = n * (n + 1) / 2;
    *bytes = 8 * (int64_t)L->n_obj * (n * L->d + tri * (n <= kSmemCholMaxN ? 1 : 2));
    return SCOOT_OK;
}

scoot_status scoot_gp_prepare_device(scoot_ctx* ctx, const scoot_param* h_space, const scoot_gp_layout* L,
                                     const uint32_t* obs, int64_t ld_obs, const float* y, const float* lengthscale,
                                     const float* signal_var, const float* noise_var, const float* warp, void* blob,
                                     void* work, int64_t work_bytes, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!h_space || !L) return scoot_fail(ctx, SCOOT_EINVAL, "h_space or layout is NULL");
    scoot_gp_layout chk;
    if (scoot_gp_layout_init(h_space, L->n, L->d, L->n_obj, L->kernel, &chk) != SCOOT_OK ||
        std::memcmp(&chk, L, sizeof(chk)) != 0)
        return scoot_fail(ctx, SCOOT_EINVAL, "layout does not match h_space");
    if (!obs || !y || !lengthscale || !signal_var || !noise_var || !blob)
        return scoot_fail(ctx, SCOOT_EINVAL, "obs, y, lengthscale, signal_var, noise_var or blob is NULL");
    if (ld_obs < L->n) return scoot_fail(ctx, SCOOT_EINVAL, "ld_obs = %lld < n = %d", (long long)ld_obs, L->n);
    if (!scoot_aligned16(blob)) return scoot_fail(ctx, SCOOT_EINVAL, "blob is not 16-byte aligned");
    int64_t need = 0;
    scoot_gp_device_work_bytes(L, &need);
    if (!work || work_bytes < need || !scoot_aligned16(work))
        return scoot_fail(ctx, SCOOT_EINVAL, "work needs %lld bytes, 16-byte aligned", (long long)need);
    GpPrepArgs a;
    std::memset(&a, 0, sizeof(a));
    const int n = L->n, d = L->d, M = L->n_obj;
    a.n = n;
    a.d = d;
    a.M = M;
    a.kernel = L->kernel;
    a.n_ord = L->n_ord;
    a.n_pat = L->n_pat;
    a.n_rb = L->n_rb;
    a.n_tiles = L->n_tiles;
    a.tri = (int64_t)n * (n + 1) / 2;
    int f = 0;
    for (int pass = 0; pass < 2; ++pass)  // ordinal parameters first, then categorical ones
        for (int c = 0; c < d; ++c)
            if ((h_space[c].kind == SCOOT_CATEGORICAL) == (pass == 1)) a.order[f++] = c;
    int stride = 1;
    for (int g = 0; g < d; ++g) {
        const int c = a.order[g];
        const scoot_param& p = h_space[c];
        a.kind[c] = p.kind;
        a.n_choices[c] = p.n_choices;
        float fa = 0.f, fb = 0.f;
        if (p.kind == SCOOT_INT_LOG) {
            a.lo[c] = std::log((double)p.lo);
            a.span[c] = std::log((double)p.hi) - std::log((double)p.lo);
            fa = (float)a.lo[c];
            fb = (float)(1.0 / a.span[c]);
        } else if (p.kind != SCOOT_CATEGORICAL) {
            a.lo[c] = p.lo;
            a.span[c] = (double)p.hi - (double)p.lo;
            fa = p.lo;
            fb = p.hi > p.lo ? (float)(1.0 / ((double)p.hi - (double)p.lo)) : 0.0f;
        } else {
            fa = (float)p.n_choices;
            fb = (float)stride;
            stride *= p.n_choices;
        }
        a.fmap[g][0] = (float)p.kind;
        a.fmap[g][1] = fa;
        a.fmap[g][2] = fb;
        a.fmap[g][3] = (float)c;
    }
    a.obs = obs;
    a.ld_obs = ld_obs;
    a.y = y;
    a.ls = lengthscale;
    a.sf2 = signal_var;
    a.tau2 = noise_var;
    a.warp = warp;
    a.blob = static_cast<char*>(blob);
    a.off_fmap = L->off_fmap;
    a.off_xs = L->off_xs;
    a.off_ils = L->off_ils;
    a.off_alpha = L->off_alpha;
    a.off_linv = L->off_linv;
    a.off_scal = L->off_scal;
    a.off_cat = L->off_cat;
    a.off_warp = L->off_warp;
    const bool in_smem = n <= kSmemCholMaxN;
    const size_t u_bytes = (size_t)M * n * d * sizeof(double);
    const size_t k_bytes = (size_t)M * a.tri * sizeof(double);
    char* ws = static_cast<char*>(work);
    a.U = reinterpret_cast<double*>(ws);
    a.K = reinterpret_cast<double*>(ws + u_bytes);
    a.W = in_smem ? nullptr : reinterpret_cast<double*>(ws + u_bytes + k_bytes);
    a.err = ctx->d_err;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    gp_feat_kernel<<<dim3((n * d + kFeatThreads - 1) / kFeatThreads, M), kFeatThreads, 0, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    if (L->n_ord < d) {
        const int64_t cells = (int64_t)n * L->n_pat;
        gp_cat_kernel<<<dim3((unsigned)((cells + kKmatThreads - 1) / kKmatThreads), M), kKmatThreads, 0, st>>>(a);
        SCOOT_LAUNCHED(ctx);
    } else {
        // no categorical parameter: one pattern, zero distance
        SCOOT_CUDA(ctx, cudaMemsetAsync(static_cast<char*>(blob) + L->off_cat, 0, (size_t)M * n * sizeof(float), st));
    }
    gp_kmat_kernel<<<dim3((unsigned)((a.tri + kKmatThreads - 1) / kKmatThreads), M), kKmatThreads, 0, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    if (n <= kClusterMaxN) {
        // rows split over a cluster; shared memory for the CTA with the most entries
        int64_t own = 0;
        for (int r = 0; r < kClusterCTAs; ++r) {
            const int64_t nl = (n - r + kClusterCTAs - 1) / kClusterCTAs;
            const int64_t e = nl * (r + 1) + (int64_t)kClusterCTAs * nl * (nl - 1) / 2;  // local_row_off(nl, r)
            if (e > own) own = e;
        }
        const size_t csmem = (size_t)8 * n * sizeof(double) + (size_t)2 * own * sizeof(double);
        SCOOT_CUDA(ctx, cudaFuncSetAttribute(gp_chol_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)csmem));
        gp_chol_cluster_kernel<<<M * kClusterCTAs, kClusterThreads, csmem, st>>>(a);
        SCOOT_LAUNCHED(ctx);
        return SCOOT_OK;
    }
    const size_t smem = (size_t)5 * n * sizeof(double) + (in_smem ? (size_t)2 * a.tri * sizeof(double) : 0);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(gp_chol_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    gp_chol_kernel<<<M, kCholThreads, smem, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

scoot_status scoot_gp_mle_work_bytes(int32_t n, int32_t d, int32_t n_obj, int32_t n_starts, int64_t* bytes) {
    if (!bytes || n < 1 || d < 1 || n_obj < 1 || n_starts < 1) return SCOOT_EINVAL;
    const int64_t tri = (int64_t)n * (n + 1) / 2;
    int64_t b = ((int64_t)n * d * 8 + 255) / 256 * 256;
    if (n > kSmemMleMaxN) b += (int64_t)n_starts * n_obj * 2 * tri * 8;
    *bytes = b;
    return SCOOT_OK;
}

scoot_status scoot_gp_mle(scoot_ctx* ctx, const scoot_param* h_space, int32_t d, const uint32_t* obs, int64_t ld_obs,
                          int32_t n, const float* y, int32_t n_obj, int32_t kernel, const double* theta0,
                          int32_t n_starts, const double* h_lo, const double* h_hi, uint32_t free_mask, int32_t steps,
                          double lr, double* theta, double* lml, double* grad, void* work, int64_t work_bytes,
                          void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    if (!h_space || !h_lo || !h_hi) return scoot_fail(ctx, SCOOT_EINVAL, "h_space, h_lo or h_hi is NULL");
    if (d < 1 || d > SCOOT_MAX_DIM) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "d = %d outside 1..%d", d, SCOOT_MAX_DIM);
    if (n < 1 || n > SCOOT_MAX_OBS) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n = %d outside 1..%d", n, SCOOT_MAX_OBS);
    if (n_obj < 1 || n_obj > SCOOT_MAX_OBJ) return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n_obj = %d", n_obj);
    if (kernel != SCOOT_MATERN52 && kernel != SCOOT_MATERN32) return scoot_fail(ctx, SCOOT_EINVAL, "kernel %d", kernel);
    if (n_starts < 1 || (int64_t)n_starts * n_obj > 65535)
        return scoot_fail(ctx, SCOOT_EUNSUPPORTED, "n_starts = %d", n_starts);
    if (steps < 0 || !(lr >= 0.0) || !std::isfinite(lr)) return scoot_fail(ctx, SCOOT_EINVAL, "steps or lr");
    if (ld_obs < n) return scoot_fail(ctx, SCOOT_EINVAL, "ld_obs = %lld < n", (long long)ld_obs);
    if (!obs || !y || !theta0 || !theta || !lml) return scoot_fail(ctx, SCOOT_EINVAL, "a device array is NULL");
    const int P = d + 2;
    MleArgs a;
    std::memset(&a, 0, sizeof(a));
    for (int p = 0; p < P; ++p) {
        if (!std::isfinite(h_lo[p]) || !std::isfinite(h_hi[p]) || h_lo[p] > h_hi[p])
            return scoot_fail(ctx, SCOOT_EINVAL, "bounds of parameter %d", p);
        a.lo[p] = h_lo[p];
        a.hi[p] = h_hi[p];
    }
    GpPrepArgs f;
    std::memset(&f, 0, sizeof(f));
    for (int c = 0; c < d; ++c) {
        const scoot_param& p = h_space[c];
        f.kind[c] = p.kind;
        if (p.kind == SCOOT_CATEGORICAL) {
            if (p.n_choices < 1) return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: n_choices", c);
            a.cat_mask |= 1u << c;
        } else if (p.kind == SCOOT_INT_LOG) {
            if (!(p.lo > 0.0f) || !(p.hi > p.lo)) return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: log range", c);
            f.lo[c] = std::log((double)p.lo);
            f.span[c] = std::log((double)p.hi) - std::log((double)p.lo);
        } else if (p.kind == SCOOT_INT_UNIFORM || p.kind == SCOOT_CONTINUOUS) {
            f.lo[c] = p.lo;
            f.span[c] = (double)p.hi - (double)p.lo;
        } else {
            return scoot_fail(ctx, SCOOT_EINVAL, "parameter %d: kind %d", c, p.kind);
        }
    }
    int64_t need = 0;
    scoot_gp_mle_work_bytes(n, d, n_obj, n_starts, &need);
    if (!work || work_bytes < need || !scoot_aligned16(work))
        return scoot_fail(ctx, SCOOT_EINVAL, "work needs %lld bytes, 16-byte aligned", (long long)need);
    char* ws = static_cast<char*>(work);
    f.n = n;
    f.d = d;
    f.obs = obs;
    f.ld_obs = ld_obs;
    f.U = reinterpret_cast<double*>(ws);
    f.M = n_obj;
    f.y = y;
    f.err = ctx->d_err;
    a.n = n;
    a.d = d;
    a.M = n_obj;
    a.P = P;
    a.kernel = kernel;
    a.S = n_starts;
    a.steps = steps;
    a.tri = (int64_t)n * (n + 1) / 2;
    a.free_mask = free_mask & ((1u << P) - 1u);
    a.lr = lr;
    a.U = f.U;
    a.y = y;
    a.theta0 = theta0;
    a.theta = theta;
    a.lml = lml;
    a.grad = grad;
    a.scratch = n > kSmemMleMaxN ? reinterpret_cast<double*>(ws + ((int64_t)n * d * 8 + 255) / 256 * 256) : nullptr;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    mle_feat_kernel<<<(n * d + kFeatThreads - 1) / kFeatThreads, kFeatThreads, 0, st>>>(f);
    SCOOT_LAUNCHED(ctx);
    const size_t smem = (size_t)(7 * n + (size_t)n * d) * sizeof(double) +
                        (n <= kSmemMleMaxN ? (size_t)2 * a.tri * sizeof(double) : 0);
    SCOOT_CUDA(ctx, cudaFuncSetAttribute(gp_mle_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    gp_mle_kernel<<<n_starts * n_obj, kMleThreads, smem, st>>>(a);
    SCOOT_LAUNCHED(ctx);
    return SCOOT_OK;
}

static int64_t slot256(int64_t b) { return (b + 255) / 256 * 256; }

scoot_status scoot_gp_device_buffer_layout(const scoot_gp_layout* L, int32_t warped, int64_t* upload_bytes,
                                           int64_t* blob_off, int64_t* work_off, int64_t* total_bytes) {
    if (!L || !upload_bytes || !blob_off || !work_off || !total_bytes || !scoot_gp_layout_valid(L)) return SCOOT_EINVAL;
    const int64_t n = L->n, d = L->d, M = L->n_obj;
    int64_t off = slot256(4 * d * n) + slot256(4 * M * n) + slot256(4 * M * d) + 2 * slot256(4 * M);
    if (warped) off += slot256(8 * M * d);
    *upload_bytes = off;
    *blob_off = off;
    off += slot256(L->bytes);
    *work_off = off;
    int64_t wb = 0;
    scoot_gp_device_work_bytes(L, &wb);
    *total_bytes = off + slot256(wb);
    return SCOOT_OK;
}

scoot_status scoot_gp_prepare_device_from_host(scoot_ctx* ctx, const scoot_param* h_space, const scoot_gp_layout* L,
                                               const uint32_t* h_x_obs, int64_t ld_obs, const float* h_y,
                                               const float* h_lengthscale, const float* h_signal_var,
                                               const float* h_noise_var, const float* h_warp, void* h_stage,
                                               void* buf, int64_t buf_bytes, void* stream) {
    scoot_status s = scoot_enter(ctx);
    if (s != SCOOT_OK) return s;
    int64_t up = 0, blob_off = 0, work_off = 0, total = 0;
    if (scoot_gp_device_buffer_layout(L, h_warp != nullptr, &up, &blob_off, &work_off, &total) != SCOOT_OK)
        return scoot_fail(ctx, SCOOT_EINVAL, "invalid layout");
    if (!h_space || !h_x_obs || !h_y || !h_lengthscale || !h_signal_var || !h_noise_var || !h_stage || !buf)
        return scoot_fail(ctx, SCOOT_EINVAL, "a pointer is NULL");
    if (buf_bytes < total || !scoot_aligned16(buf))
        return scoot_fail(ctx, SCOOT_EINVAL, "buf needs %lld bytes, 16-byte aligned", (long long)total);
    if (ld_obs < L->n) return scoot_fail(ctx, SCOOT_EINVAL, "ld_obs < n");
    const int64_t n = L->n, d = L->d, M = L->n_obj;
    char* hs = static_cast<char*>(h_stage);
    int64_t off = 0, o_obs, o_y, o_ls, o_sf, o_tau, o_warp = -1;
    o_obs = off;
    for (int64_t c = 0; c < d; ++c) std::memcpy(hs + off + 4 * c * n, h_x_obs + c * ld_obs, 4 * n);
    off += slot256(4 * d * n);
    o_y = off;
    std::memcpy(hs + off, h_y, 4 * M * n);
    off += slot256(4 * M * n);
    o_ls = off;
    std::memcpy(hs + off, h_lengthscale, 4 * M * d);
    off += slot256(4 * M * d);
    o_sf = off;
    std::memcpy(hs + off, h_signal_var, 4 * M);
    off += slot256(4 * M);
    o_tau = off;
    std::memcpy(hs + off, h_noise_var, 4 * M);
    off += slot256(4 * M);
    if (h_warp) {
        o_warp = off;
        std::memcpy(hs + off, h_warp, 8 * M * d);
        off += slot256(8 * M * d);
    }
    char* db = static_cast<char*>(buf);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    SCOOT_CUDA(ctx, cudaMemcpyAsync(db, hs, (size_t)up, cudaMemcpyHostToDevice, st));
    return scoot_gp_prepare_device(ctx, h_space, L, reinterpret_cast<const uint32_t*>(db + o_obs), n,
                                   reinterpret_cast<const float*>(db + o_y), reinterpret_cast<const float*>(db + o_ls),
                                   reinterpret_cast<const float*>(db + o_sf), reinterpret_cast<const float*>(db + o_tau),
                                   o_warp >= 0 ? reinterpret_cast<const float*>(db + o_warp) : nullptr, db + blob_off,
                                   db + work_off, total - work_off, stream);
}

}  // extern "C"
