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
    // Phase timing (scoot_ctx_set_timing): events recorded between the
    // launches of the last timed call, and the kind of each launch.
    int32_t timing = 0;
    std::vector<void*> events;   // cudaEvent_t, created on first use
    std::vector<int32_t> mark_kind;
    // The open session of sequential fantasised picks (scoot_fantasy_begin
    // .. scoot_fantasy_end), opaque to everything but fantasy.cu.
    std::vector<char> fant_session;
    // scoot_ctx_set_tensor_cores: the whitened posterior may run its L^{-1} k
    // product on the tensor cores (posterior_tc.cu) where the state fits.
    int32_t tensor_cores = 1;
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

// Layout of the fp64 state of the sequential fantasised picks: built on the
// host (scoot_fantasy_prepare, or scoot_round_state_build with fantasy_q >
// 0) and read by the fantasy kernels.  Offsets count from the start of the
// state and are 256-byte aligned; parameters are in their original order.
struct FantHeader {
    int32_t magic;                 // kFantMagic
    int32_t n, d, M, kernel, q;    // observations, parameters, objectives, covariance, picks
    int32_t front0;                // size of the observations' Pareto front
    int32_t front_cap;             // front0 + q: the front can only grow by one point per pick
    int32_t box_cap;               // cells of the box decomposition the picks may need
    int32_t pad[7];
    double ref[4], sf2[4], tau2[4];
    int64_t off_space;             // double [d][4]: kind, lo, hi, n_choices
    int64_t off_u;                 // double [n][d]: features of the observations
    int64_t off_ell;               // double [M][d]: lengthscales
    int64_t off_alpha;             // double [M][n]: (K + tau^2 I)^{-1} y
    int64_t off_linv;              // double [M][n][n]: L^{-1}, column-major (entry (i, c) at c n + i)
    int64_t off_front;             // double [n][M]: the observations' front (first front0 rows)
    int64_t bytes;
};
constexpr int32_t kFantMagic = 0x544e4146;
// Largest box count the fantasy kernels stage (2 float4 per box in shared memory).
constexpr int32_t kFantBoxMax = 6144;
// Offsets and size of a fantasy state for n observations, d parameters, M
// objectives and q picks (front0, front_cap, box_cap and the values are left 0).
void scoot_fant_layout(int32_t n, int32_t d, int32_t M, int32_t q, FantHeader* h);

// The GP blob (h_blob, may be NULL) and/or the fp64 arrays of a fantasy state
// whose header is already laid out (h_fant, may be NULL) from one
// factorisation per objective; scoot_gp_prepare_warped is this call with
// h_fant = NULL.  Fantasy states take no warping (SCOOT_EUNSUPPORTED).
scoot_status scoot_gp_build(const scoot_param* h_space, const uint32_t* h_x_obs, int64_t ld_obs, const float* h_y,
                            const float* h_lengthscale, const float* h_signal_var, const float* h_noise_var,
                            const float* h_warp, const scoot_gp_layout* L, void* h_blob, double* h_cond,
                            void* h_fant);
// The header, space, front and scalars of a fantasy state (everything but the
// factorisation's arrays, which scoot_gp_build writes).
scoot_status scoot_fant_header(const scoot_param* h_space, const scoot_gp_layout* L, const float* h_y,
                               const float* h_signal_var, const float* h_noise_var, const float* h_ref, int32_t q,
                               void* h_fant, int64_t cap);

// Consistency of a GP layout's offsets with its own sizes.
bool scoot_gp_layout_valid(const scoot_gp_layout* L);

// Phase timing: scoot_marks_begin records the first event of a call on
// stream st, scoot_mark one event after each launch of kind `kind` (no-ops
// unless timing is enabled).  Kinds are listed in include/scoot.h.
scoot_status scoot_marks_begin(scoot_ctx* ctx, void* st);
scoot_status scoot_mark(scoot_ctx* ctx, void* st, int32_t kind);

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
// [M][ldc], and the whitened rows V = L^{-1} k(X, x) in float4 groups of four
// rows, tiled by 32 list positions (scoot_dev::vtile_index), ceil(list
// length / 32) tiles of M * n_rb * 16 * 32 float4 (16-byte aligned; groups
// wholly past row n left unwritten, rows past n inside a written group zero).
// ldc >= the list length.
// tc_work (may be NULL: the SIMT product) is device scratch of at least
// scoot_tc_bsplit_bytes(n_pad, M) bytes, 16-byte aligned, for the split copy
// of L^{-1} that the tensor-core product reads.
scoot_status scoot_posterior_whitened(scoot_ctx* ctx, const scoot_gp_layout* L, const void* state,
                                      const uint32_t* cand, int64_t n, int64_t ld, const int32_t* list,
                                      const unsigned int* n_list, float* mean, float* var, float* V, int64_t ldc,
                                      void* tc_work, cudaStream_t st);

// The tensor-core whitened posterior (posterior_tc.cu): the arguments of the
// SIMT kernel's whitened epilogue plus the split copy of L^{-1}.
constexpr int kMaxNpadTc = 256;  // output rows held in tensor memory (fp32 columns)
struct ScootTcArgs {
    const char* state;
    int64_t off_fmap, off_xs, off_ils, off_alpha, off_scal, off_cat, off_warp, off_linv;
    int32_t n_obs, d, n_obj, kernel, n_pad, n_ord, n_pat, n_tiles, cat_smem;
    const uint32_t* cand;
    int64_t n, ld;
    const int32_t* list;
    const unsigned int* n_list;
    float* mean;
    float* var;
    int64_t ldo;
    float* vout;      // NULL: moments only
    int32_t by_index; // mean / var at the candidate's index (else at its list position)
    uint8_t* bsplit;  // [M][n_pad / 32][3][n_pad * 64 bytes]
    uint32_t* err;
    // Acquisition epilogue (objective 0 only, acq at the candidate's index;
    // mean / var then unused): 0 none, 1 EI (Eq. 6) into acq[i], 2 MACE's
    // UCB, PI and EI (Section 4.5) into acq[i], acq[lda + i], acq[2 lda + i].
    int32_t acq_kind;
    float* acq;
    int64_t lda;
    float xi, kappa;
};
int64_t scoot_tc_bsplit_bytes(int n_pad, int M);
bool scoot_tc_supported(scoot_ctx* ctx, const ScootTcArgs& a, int DO);
scoot_status scoot_posterior_tc(scoot_ctx* ctx, const ScootTcArgs& a, int DO, cudaStream_t st);

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
