// Internal definitions shared by the host and CUDA translation units of libscoot.
#pragma once

#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <functional>
#include <string>
#include <vector>

#include "../../include/scoot.h"

#ifdef __CUDACC__
#include <cuda_runtime.h>
#endif

// Bits of the device error word.
#define SCOOT_DEVERR_INDEX   1u   // a node, feature or box index out of range
#define SCOOT_DEVERR_TIMEOUT 2u   // a bounded wait gave up
#define SCOOT_DEVERR_CAPACITY 4u  // a Pareto filter had more survivors than it can hold
#define SCOOT_DEVERR_VALUE   8u   // a non-finite feature or a label other than 0/1

struct scoot_ctx {
    int32_t device = 0;
    std::string err;
    void* ws = nullptr;          // device workspace (grown on demand)
    size_t ws_bytes = 0;
    uint32_t* d_err = nullptr;   // device error word
};

scoot_status scoot_fail(scoot_ctx* ctx, scoot_status s, const char* fmt, ...);
// fn(0 .. count-1) on the library's persistent host threads and the calling
// thread; returns when all are done.  Safe to nest.
void scoot_host_parallel(int count, const std::function<void(int)>& fn);
// Make ctx->device current; sets an error on failure.
scoot_status scoot_enter(scoot_ctx* ctx);
// Ensure at least `bytes` of workspace (synchronising the device if it grows).
scoot_status scoot_workspace(scoot_ctx* ctx, size_t bytes);

static inline bool scoot_aligned16(const void* p) {
    return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// fp64 GP of one objective over the observations (Section 4.3), host side:
// K + tau^2 I = C C^T, alpha = (K + tau^2 I)^{-1} y.
struct HostGP {
    int n = 0, d = 0, kernel = SCOOT_MATERN52;
    double sf2 = 1.0, tau2 = 0.0;
    std::vector<double> u;        // [n][d] features of the observations
    std::vector<uint8_t> cat;     // [d] 1 for categorical dimensions
    std::vector<double> ell;      // [d] lengthscales
    std::vector<double> chol;     // [n][n], lower triangle
    std::vector<double> alpha;    // [n]
    std::vector<double> warp;     // [d][2] Kumaraswamy (a, b) per parameter; empty: no warping
    double cov(const double* ua, const double* ub) const;       // k(a, b) of (warped) features
    void warp_features(double* u) const;                        // in place; no-op without warping
    void kstar(const double* ux, double* k) const;              // k(x, X_j), j < n; ux unwarped
    void solve_lower(const double* b, double* x) const;         // C x = b
};
// Features of configuration j of a SoA word array (ld = leading dimension).
bool scoot_host_features(const scoot_param* sp, int d, const uint32_t* words, int64_t ld, int64_t j, double* u);
// Factor objective m; SCOOT_EINVAL on bad inputs or a matrix that is not
// numerically positive definite.  cond (optional) receives (max/min pivot)^2.
// warp: [d][2] Kumaraswamy (a, b) per parameter, or NULL; g->u holds the
// warped features of the observations.
scoot_status scoot_host_gp(const scoot_param* sp, int d, const uint32_t* x_obs, int64_t ld_obs, int n,
                           const float* y, const float* lengthscale, float signal_var, float noise_var,
                           int kernel, HostGP* out, double* cond, const float* warp = nullptr);

// Consistency of a GP layout's offsets with its own sizes.
bool scoot_gp_layout_valid(const scoot_gp_layout* L);

// Checks shared by the device entry points.
scoot_status scoot_check_pool(scoot_ctx* ctx, const uint32_t* cand, int64_t n, int64_t ld, int32_t d);

#ifdef __CUDACC__
// Index list of live candidates built by scoot_compact in the context workspace.
struct ScootList {
    int32_t* list;
    unsigned int* count;
};
// Compacts the indices i < n with mask[i] != 0 into out->list (count on the
// device); where mask[i] == 0, fill[r * fill_ld + i] = fill_bits for the
// fill_rows rows of fill, if fill is not NULL.
scoot_status scoot_compact(scoot_ctx* ctx, const uint8_t* mask, int64_t n, uint32_t* fill, uint32_t fill_bits,
                           cudaStream_t st, ScootList* out, int fill_rows = 1, int64_t fill_ld = 0);

// Posterior of the listed candidates into list-position order: mean and var
// [M][ldc], and the whitened rows V = L^{-1} k(X, x) [M][n_rb * 64][ldc]
// (rows >= n left unwritten).  ldc >= the list length.
scoot_status scoot_posterior_whitened(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                      const uint32_t* cand, int64_t n, int64_t ld, const int32_t* list,
                                      const unsigned int* n_list, float* mean, float* var, float* V, int64_t ldc,
                                      cudaStream_t st);

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
